"""Pins of the oracle backbone (forward and hand-derived reverse mode) to things other
than itself: central finite differences, torch's own library routines (layer_norm,
rms_norm, scaled_dot_product_attention, gelu, silu) differentiated by torch autograd,
closed forms and special cases."""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import synth
from oracle import dit

TINY_DIT = synth.WORKLOADS["tiny_dit_f32"]
TINY_MMDIT = synth.small_variant(
    synth.WORKLOADS["mmdit_flux512_bf16"], name="tiny_mmdit_f32", dtype="f32", hidden=64,
    heads=4, mlp=256, depth=1, depth_double=1, in_channels=4, latent_h=6, latent_w=4,
    patch=2, txt_len=5, txt_dim=48, G=2, T=4, W=4)


def _inputs(wl, B, seed):
    rng = np.random.Generator(np.random.PCG64(seed))
    z = rng.standard_normal((B, wl.in_channels, wl.latent_h, wl.latent_w))
    t = rng.uniform(0.05, 1.0, size=B)
    txt = rng.standard_normal((B, wl.txt_len, wl.txt_dim))
    cot = rng.standard_normal((B, wl.in_channels, wl.latent_h, wl.latent_w))
    return z, t, txt, cot


# ----------------------------------------------------------------------------- FD
@pytest.mark.parametrize("wl", [TINY_DIT, TINY_MMDIT], ids=lambda w: w.name)
def test_vjp_matches_central_differences(wl):
    """<grad_theta, u> equals d/dh <v(theta + h u), cot> (central, h = 1e-6) for a random
    direction u in every parameter tensor separately."""
    params = synth.make_params(wl, seed=3, bias_scale=0.1)
    z, t, txt, cot = _inputs(wl, 3, 11)
    model = dit.Backbone(wl, params)
    _, cache = model.forward(z, t, txt)
    grads = model.vjp(cache, cot)
    rng = np.random.Generator(np.random.PCG64(5))
    h = 1e-6
    for name in params:
        u = rng.standard_normal(params[name].shape)
        pp = dict(params); pp[name] = params[name] + h * u
        pm = dict(params); pm[name] = params[name] - h * u
        fp = (dit.Backbone(wl, pp).forward(z, t, txt)[0] * cot).sum()
        fm = (dit.Backbone(wl, pm).forward(z, t, txt)[0] * cot).sum()
        fd = (fp - fm) / (2 * h)
        an = (grads[name] * u).sum()
        assert abs(fd - an) <= 1e-7 * max(1.0, abs(an)), (name, fd, an)


# ------------------------------------------------------------------ torch library pin
def _torch_backbone(wl, P, z, t, txt):
    """The same architecture assembled from torch.nn.functional library routines
    (layer_norm, rms_norm, scaled_dot_product_attention, gelu(tanh), silu, linear) and
    RoPE as a complex rotation; torch autograd supplies the reverse mode."""
    d, h, dh, p = wl.hidden, wl.heads, wl.head_dim, wl.patch
    B = z.shape[0]
    gh, gw = wl.latent_h // p, wl.latent_w // p
    xp = z.unfold(2, p, p).unfold(3, p, p)            # B C gh gw p p
    xp = xp.permute(0, 2, 3, 1, 4, 5).reshape(B, gh * gw, -1)
    ximg = F.linear(xp, P["x_embed.w"], P["x_embed.b"])
    if wl.pos_embed:
        q = d // 4
        w = torch.tensor([10000.0 ** (-k / q) for k in range(q)], dtype=torch.float64)
        r = torch.arange(gh, dtype=torch.float64).repeat_interleave(gw)
        c = torch.arange(gw, dtype=torch.float64).repeat(gh)
        ar, ac = r[:, None] * w, c[:, None] * w
        ximg = ximg + torch.cat([ar.sin(), ar.cos(), ac.sin(), ac.cos()], 1)
    xtxt = F.linear(txt, P["txt_embed.w"], P["txt_embed.b"])
    half = wl.freq_dim // 2
    fr = torch.exp(-math.log(10000.0) * torch.arange(half, dtype=torch.float64) / half)
    arg = 1000.0 * t[:, None] * fr[None]
    phi = torch.cat([arg.cos(), arg.sin()], 1)
    cvec = F.linear(F.silu(F.linear(phi, P["t_embed.w1"], P["t_embed.b1"])), P["t_embed.w2"], P["t_embed.b2"])
    sc_ = F.silu(cvec)
    ln = lambda x: F.layer_norm(x, (d,), eps=1e-6)
    modl = lambda x, sh, sc: x * (1 + sc[:, None]) + sh[:, None]
    gelu = lambda x: F.gelu(x, approximate="tanh")
    nt = wl.txt_len
    if wl.rope:
        hd = dh // 2
        th = 10000.0 ** (-2.0 * torch.arange(hd // 2, dtype=torch.float64) / hd)
        rr = torch.cat([torch.zeros(nt), torch.arange(gh, dtype=torch.float64).repeat_interleave(gw)])
        cc = torch.cat([torch.zeros(nt), torch.arange(gw, dtype=torch.float64).repeat(gh)])
        ang = torch.cat([rr[:, None] * th, cc[:, None] * th], 1)      # N x dh/2
        rot = torch.polar(torch.ones_like(ang), ang)

        def rope(x):        # B N h dh -> pairs as complex numbers times e^{i ang}
            xc = torch.view_as_complex(x.reshape(*x.shape[:-1], -1, 2).contiguous())
            return torch.view_as_real(xc * rot[None, :, None, :]).reshape(x.shape)

    def attn(qkv, qn=None, kn=None, ntxt=None):
        N = qkv.shape[1]
        q, k, v = (qkv[..., i * d:(i + 1) * d].reshape(B, N, h, dh) for i in range(3))
        if qn is not None:
            q = torch.cat([F.rms_norm(q[:, :ntxt], (dh,), qn[0], eps=1e-6),
                           F.rms_norm(q[:, ntxt:], (dh,), qn[1], eps=1e-6)], 1)
            k = torch.cat([F.rms_norm(k[:, :ntxt], (dh,), kn[0], eps=1e-6),
                           F.rms_norm(k[:, ntxt:], (dh,), kn[1], eps=1e-6)], 1)
        if wl.rope:
            q, k = rope(q), rope(k)
        o = F.scaled_dot_product_attention(q.transpose(1, 2), k.transpose(1, 2), v.transpose(1, 2))
        return o.transpose(1, 2).reshape(B, N, d)

    L = lambda x, n: F.linear(x, P[n + ".w"], P[n + ".b"])
    if wl.arch == "dit":
        hh = torch.cat([xtxt, ximg], 1)
        for i in range(wl.depth):
            pre = f"blocks.{i}."
            m6 = L(sc_, pre + "mod").chunk(6, dim=1)
            hh = hh + m6[2][:, None] * L(attn(L(modl(ln(hh), m6[0], m6[1]), pre + "qkv")), pre + "proj")
            hh = hh + m6[5][:, None] * L(gelu(L(modl(ln(hh), m6[3], m6[4]), pre + "fc1")), pre + "fc2")
    else:
        ht, hi = xtxt, ximg
        for i in range(wl.depth_double):
            pre = f"double.{i}."
            mt = L(sc_, pre + "txt.mod").chunk(6, dim=1)
            mi = L(sc_, pre + "img.mod").chunk(6, dim=1)
            qkv = torch.cat([L(modl(ln(ht), mt[0], mt[1]), pre + "txt.qkv"),
                             L(modl(ln(hi), mi[0], mi[1]), pre + "img.qkv")], 1)
            o = attn(qkv, (P[pre + "txt.q_norm"], P[pre + "img.q_norm"]),
                     (P[pre + "txt.k_norm"], P[pre + "img.k_norm"]), nt)
            ht = ht + mt[2][:, None] * L(o[:, :nt], pre + "txt.proj")
            hi = hi + mi[2][:, None] * L(o[:, nt:], pre + "img.proj")
            ht = ht + mt[5][:, None] * L(gelu(L(modl(ln(ht), mt[3], mt[4]), pre + "txt.fc1")), pre + "txt.fc2")
            hi = hi + mi[5][:, None] * L(gelu(L(modl(ln(hi), mi[3], mi[4]), pre + "img.fc1")), pre + "img.fc2")
        hh = torch.cat([ht, hi], 1)
        for i in range(wl.depth):
            pre = f"single.{i}."
            m3 = L(sc_, pre + "mod").chunk(3, dim=1)
            l1 = L(modl(ln(hh), m3[0], m3[1]), pre + "lin1")
            qn = (P[pre + "q_norm"], P[pre + "q_norm"])
            kn = (P[pre + "k_norm"], P[pre + "k_norm"])
            o = attn(l1[..., :3 * d], qn, kn, nt)
            hh = hh + m3[2][:, None] * L(torch.cat([o, gelu(l1[..., 3 * d:])], -1), pre + "lin2")
    fm = L(sc_, "final.mod").chunk(2, dim=1)
    vt = L(modl(ln(hh[:, nt:]), fm[0], fm[1]), "final.out")
    C = wl.in_channels
    v = vt.reshape(B, gh, gw, C, p, p).permute(0, 3, 1, 4, 2, 5).reshape(B, C, wl.latent_h, wl.latent_w)
    return v


@pytest.mark.parametrize("wl", [TINY_DIT, TINY_MMDIT], ids=lambda w: w.name)
def test_forward_and_vjp_match_torch_library(wl):
    params = synth.make_params(wl, seed=7, bias_scale=0.1)
    z, t, txt, cot = _inputs(wl, 3, 13)
    model = dit.Backbone(wl, params)
    v, cache = model.forward(z, t, txt)
    grads = model.vjp(cache, cot)
    P = {k: torch.tensor(a, dtype=torch.float64, requires_grad=True) for k, a in params.items()}
    vt = _torch_backbone(wl, P, torch.tensor(z), torch.tensor(t), torch.tensor(txt))
    np.testing.assert_allclose(v, vt.detach().numpy(), rtol=1e-11, atol=1e-11)
    (vt * torch.tensor(cot)).sum().backward()
    for k in params:
        np.testing.assert_allclose(grads[k], P[k].grad.numpy(), rtol=1e-9, atol=1e-11, err_msg=k)


# ---------------------------------------------------------------- special cases
def test_patchify_roundtrip_and_order():
    z = np.arange(2 * 3 * 4 * 6, dtype=np.float64).reshape(2, 3, 4, 6)
    x = dit.patchify(z, 2)
    assert x.shape == (2, 6, 12)
    # token 4 = patch row 1, col 1; feature 7 = channel 1, py 1, px 1
    assert x[1, 4, 7] == z[1, 1, 2 + 1, 2 + 1]
    np.testing.assert_array_equal(dit.unpatchify(x, 3, 4, 6, 2), z)


def test_timestep_embedding_closed_forms():
    phi = dit.timestep_embedding(np.array([0.0, 0.5]), 256)
    np.testing.assert_array_equal(phi[0, :128], 1.0)
    np.testing.assert_array_equal(phi[0, 128:], 0.0)
    assert phi[1, 0] == pytest.approx(math.cos(500.0))          # w_0 = 1
    assert phi[1, 128 + 64] == pytest.approx(math.sin(500.0 * 10000.0 ** -0.5))


def test_attention_uniform_when_scores_vanish():
    rng = np.random.Generator(np.random.PCG64(1))
    v = rng.standard_normal((1, 5, 2, 3))
    o, P = dit.attention(np.zeros_like(v), np.zeros_like(v), v)
    np.testing.assert_allclose(P, 0.2)
    np.testing.assert_allclose(o, np.broadcast_to(v.mean(1, keepdims=True), o.shape))


def test_zero_gates_make_blocks_identity():
    """adaLN-zero special case: with every modulation weight and bias zero the gates vanish,
    each block is the identity, and v depends on the blocks not at all."""
    wl = TINY_DIT
    params = synth.make_params(wl, seed=2)
    z, t, txt, _ = _inputs(wl, 2, 3)
    for k in params:
        if ".mod." in k and k.startswith("blocks"):
            params[k] = np.zeros_like(params[k])
    v1, _ = dit.Backbone(wl, params).forward(z, t, txt)
    for k in params:
        if k.startswith("blocks") and (".qkv." in k or ".fc" in k or ".proj." in k):
            params[k] = params[k] + 1.0
    v2, _ = dit.Backbone(wl, params).forward(z, t, txt)
    np.testing.assert_array_equal(v1, v2)


def test_rope_is_a_rotation_and_text_is_unrotated():
    ang = dit.rope_angles(3, 4, 2, 16)
    assert ang.shape == (14, 8)
    np.testing.assert_array_equal(ang[:2], 0.0)
    rng = np.random.Generator(np.random.PCG64(4))
    x = rng.standard_normal((1, 14, 2, 16))
    y = dit.rope_apply(x, ang)
    np.testing.assert_allclose((y ** 2).sum(-1), (x ** 2).sum(-1))
    np.testing.assert_allclose(dit.rope_apply(y, ang, inverse=True), x, atol=1e-14)
    # token 2 + 1*4 + 2 = patch row 1, col 2: first-half pair 0 turns by 1 rad, second-half by 2
    assert ang[2 + 4 + 2, 0] == 1.0 and ang[2 + 4 + 2, 4] == 2.0


@pytest.mark.parametrize("wl", [TINY_DIT, TINY_MMDIT], ids=lambda w: w.name)
def test_batched_vjp_is_sum_of_single_row_vjps(wl):
    """Linearity of the VJP over rows: the batched full-W VJP equals the sum of the
    single-row VJPs (the batching identity), to 1e-12."""
    params = synth.make_params(wl, seed=9)
    z, t, txt, cot = _inputs(wl, 4, 21)
    model = dit.Backbone(wl, params)
    _, cache = model.forward(z, t, txt)
    g = model.vjp(cache, cot)
    acc = {k: np.zeros_like(a) for k, a in params.items()}
    for b in range(4):
        _, cb = model.forward(z[b:b + 1], t[b:b + 1], txt[b:b + 1])
        gb = model.vjp(cb, cot[b:b + 1])
        for k in acc:
            acc[k] += gb[k]
    for k in acc:
        np.testing.assert_allclose(g[k], acc[k], rtol=1e-12, atol=1e-12 * (1 + np.abs(acc[k]).max()))
