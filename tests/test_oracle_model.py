"""Pins of the oracle backbone (forward and hand-derived reverse mode) to things other
than itself: central finite differences, torch's own library routines (layer_norm,
rms_norm, scaled_dot_product_attention, gelu, silu) differentiated by torch autograd,
closed forms and special cases."""
import math

import numpy as np
import pytest
import torch

import synth
from oracle import dit
from torch_backbone import torch_backbone

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
@pytest.mark.parametrize("wl", [TINY_DIT, TINY_MMDIT], ids=lambda w: w.name)
def test_forward_and_vjp_match_torch_library(wl):
    params = synth.make_params(wl, seed=7, bias_scale=0.1)
    z, t, txt, cot = _inputs(wl, 3, 13)
    model = dit.Backbone(wl, params)
    v, cache = model.forward(z, t, txt)
    grads = model.vjp(cache, cot)
    P = {k: torch.tensor(a, dtype=torch.float64, requires_grad=True) for k, a in params.items()}
    vt = torch_backbone(wl, P, torch.tensor(z), torch.tensor(t), torch.tensor(txt))
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
    o, P = dit.attention(np.zeros_like(v), np.zeros_like(v), v, keep_probs=True)
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
