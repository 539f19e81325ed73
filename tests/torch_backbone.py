"""The backbone assembled from torch.nn.functional library routines (layer_norm, rms_norm,
scaled_dot_product_attention, gelu(tanh), silu, linear) and RoPE as a complex rotation;
torch autograd supplies the reverse mode.  Test infrastructure: a second, independent
statement of the architecture, used to pin the oracle (float64, CPU) and as the reference
of the full-size GPU parity tests (float32, CUDA).  Tables (positions, frequencies,
rotation angles) are computed in float64 and cast to the inputs' dtype."""
import math

import torch
import torch.nn.functional as F


def torch_backbone(wl, P, z, t, txt):
    """The same architecture assembled from torch.nn.functional library routines
    (layer_norm, rms_norm, scaled_dot_product_attention, gelu(tanh), silu, linear) and
    RoPE as a complex rotation; torch autograd supplies the reverse mode."""
    d, h, dh, p = wl.hidden, wl.heads, wl.head_dim, wl.patch
    f64 = dict(dtype=torch.float64, device=z.device)
    cast = lambda x: x.to(z.dtype)
    B = z.shape[0]
    gh, gw = wl.latent_h // p, wl.latent_w // p
    xp = z.unfold(2, p, p).unfold(3, p, p)            # B C gh gw p p
    xp = xp.permute(0, 2, 3, 1, 4, 5).reshape(B, gh * gw, -1)
    ximg = F.linear(xp, P["x_embed.w"], P["x_embed.b"])
    if wl.pos_embed:
        q = d // 4
        w = torch.tensor([10000.0 ** (-k / q) for k in range(q)], **f64)
        r = torch.arange(gh, **f64).repeat_interleave(gw)
        c = torch.arange(gw, **f64).repeat(gh)
        ar, ac = r[:, None] * w, c[:, None] * w
        ximg = ximg + cast(torch.cat([ar.sin(), ar.cos(), ac.sin(), ac.cos()], 1))
    xtxt = F.linear(txt, P["txt_embed.w"], P["txt_embed.b"])
    half = wl.freq_dim // 2
    fr = torch.exp(-math.log(10000.0) * torch.arange(half, **f64) / half)
    arg = 1000.0 * t.to(torch.float64)[:, None] * fr[None]
    phi = cast(torch.cat([arg.cos(), arg.sin()], 1))
    cvec = F.linear(F.silu(F.linear(phi, P["t_embed.w1"], P["t_embed.b1"])), P["t_embed.w2"], P["t_embed.b2"])
    sc_ = F.silu(cvec)
    ln = lambda x: F.layer_norm(x, (d,), eps=1e-6)
    modl = lambda x, sh, sc: x * (1 + sc[:, None]) + sh[:, None]
    gelu = lambda x: F.gelu(x, approximate="tanh")
    nt = wl.txt_len
    if wl.rope:
        hd = dh // 2
        th = 10000.0 ** (-2.0 * torch.arange(hd // 2, **f64) / hd)
        rr = torch.cat([torch.zeros(nt, **f64), torch.arange(gh, **f64).repeat_interleave(gw)])
        cc = torch.cat([torch.zeros(nt, **f64), torch.arange(gw, **f64).repeat(gh)])
        ang = torch.cat([rr[:, None] * th, cc[:, None] * th], 1)      # N x dh/2
        rot = torch.polar(torch.ones_like(ang), ang)
        rot = rot if z.dtype == torch.float64 else rot.to(torch.complex64)

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
