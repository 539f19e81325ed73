"""Float64 DiT / MMDiT backbone: forward and hand-derived reverse mode.

TEST INFRASTRUCTURE ONLY (see oracle/__init__.py).

The paper trains Flux and Qwen-Image off the shelf and never writes their architecture
down (Sec. 4, "Setup").  Phase 4 (Sec. 3.3, Algorithm 1) needs the vector-Jacobian
product J(z,t)^T s of the velocity network with respect to its parameters, so the
backbone is fixed here as a stated reading, written out from its definition:

  patchify      token n = r*(W/p) + c (row-major over the patch grid); feature
                f = ch*p*p + py*p + px
  embeddings    x_img = patch W_in^T + b_in (+ fixed 2D sin-cos table, single-stream
                DiT only); x_txt = txt W_txt^T + b_txt
  t-embedding   phi(t) = [cos(1000 t w_k), sin(1000 t w_k)], w_k = 10000^(-k/128), k<128;
                c = W_t2 SiLU(W_t1 phi + b_t1) + b_t2
  modulation    SiLU(c) W_mod^T + b_mod
  LayerNorm     no affine, biased variance, eps 1e-6
  GELU          tanh approximation
  attention     softmax(q k^T / sqrt(dh)) v over the joint [txt; img] sequence, no mask
  DiT block     (sh1,sc1,g1,sh2,sc2,g2) = mod;
                a = LN(h)(1+sc1)+sh1; h += g1 * proj(attn(qkv(a)));
                m = LN(h)(1+sc2)+sh2; h += g2 * fc2(GELU(fc1(m)))
  MMDiT double  the DiT block with separate weights per stream (txt, img), per-head
                RMSNorm (learned scale, eps 1e-6) on q and k, 2D RoPE, joint attention
  MMDiT single  (sh,sc,g) = mod; a = LN(h)(1+sc)+sh; [qkv|u] = lin1(a);
                h += g * lin2([attn(qkv) | GELU(u)])
  RoPE          head dim split in halves: first half rotated by the patch row r, second
                by the column c; pairs (2i, 2i+1); theta_i = 10000^(-2i/(dh/2));
                text tokens sit at (0, 0) (not rotated)
  final layer   (sh,sc) = mod; v_tok = (LN(h_img)(1+sc)+sh) W_out^T + b_out; unpatchify
"""
from __future__ import annotations

import numpy as np

LN_EPS = 1e-6
RMS_EPS = 1e-6
GELU_C = np.sqrt(2.0 / np.pi)
GELU_A = 0.044715


# --------------------------------------------------------------------------- helpers
def patchify(z, p):
    """[B, C, H, W] -> [B, (H/p)(W/p), C p p], token-major over the patch grid."""
    B, C, H, W = z.shape
    x = z.reshape(B, C, H // p, p, W // p, p).transpose(0, 2, 4, 1, 3, 5)
    return x.reshape(B, (H // p) * (W // p), C * p * p)


def unpatchify(x, C, H, W, p):
    """Inverse of patchify."""
    B = x.shape[0]
    y = x.reshape(B, H // p, W // p, C, p, p).transpose(0, 3, 1, 4, 2, 5)
    return y.reshape(B, C, H, W)


def timestep_embedding(t, dim=256):
    """phi(t) = [cos(1000 t w_k), sin(1000 t w_k)], w_k = 10000^(-k/(dim/2))."""
    half = dim // 2
    w = 10000.0 ** (-np.arange(half, dtype=np.float64) / half)
    arg = 1000.0 * np.asarray(t, dtype=np.float64)[:, None] * w[None, :]
    return np.concatenate([np.cos(arg), np.sin(arg)], axis=1)


def pos_embed_2d(gh, gw, d):
    """Fixed 2D sin-cos table [gh*gw, d]: dims [0,d/2) encode the row, [d/2,d) the column;
    each half is [sin(pos w_k), cos(pos w_k)] with w_k = 10000^(-k/(d/4)), k < d/4."""
    q = d // 4
    w = 10000.0 ** (-np.arange(q, dtype=np.float64) / q)
    rows = np.repeat(np.arange(gh, dtype=np.float64), gw)
    cols = np.tile(np.arange(gw, dtype=np.float64), gh)

    def one(pos):
        a = pos[:, None] * w[None, :]
        return np.concatenate([np.sin(a), np.cos(a)], axis=1)
    return np.concatenate([one(rows), one(cols)], axis=1)


def rope_angles(gh, gw, n_txt, dh):
    """Rotation angles [N, dh/2] (one per rotated pair) for the joint [txt; img] sequence."""
    hd = dh // 2                       # each axis rotates hd dims = hd/2 pairs
    theta = 10000.0 ** (-2.0 * np.arange(hd // 2, dtype=np.float64) / hd)
    rows = np.concatenate([np.zeros(n_txt), np.repeat(np.arange(gh, dtype=np.float64), gw)])
    cols = np.concatenate([np.zeros(n_txt), np.tile(np.arange(gw, dtype=np.float64), gh)])
    return np.concatenate([rows[:, None] * theta[None, :], cols[:, None] * theta[None, :]], axis=1)


def rope_apply(x, ang, inverse=False):
    """Rotate pairs (2i, 2i+1) of x [..., N, h, dh] by ang [N, dh/2] (or by -ang)."""
    c = np.cos(ang)[:, None, :]
    s = np.sin(ang)[:, None, :]
    if inverse:
        s = -s
    x0 = x[..., 0::2]
    x1 = x[..., 1::2]
    out = np.empty_like(x)
    out[..., 0::2] = x0 * c - x1 * s
    out[..., 1::2] = x0 * s + x1 * c
    return out


def silu(x):
    return x / (1.0 + np.exp(-x))


def silu_grad(x):
    sg = 1.0 / (1.0 + np.exp(-x))
    return sg * (1.0 + x * (1.0 - sg))


def gelu(u):
    return 0.5 * u * (1.0 + np.tanh(GELU_C * (u + GELU_A * u ** 3)))


def gelu_grad(u):
    th = np.tanh(GELU_C * (u + GELU_A * u ** 3))
    return 0.5 * (1.0 + th) + 0.5 * u * (1.0 - th ** 2) * GELU_C * (1.0 + 3.0 * GELU_A * u ** 2)


def ln_fwd(x):
    mu = x.mean(-1, keepdims=True)
    xc = x - mu
    rstd = 1.0 / np.sqrt((xc ** 2).mean(-1, keepdims=True) + LN_EPS)
    return xc * rstd, rstd


def ln_bwd(dxh, xh, rstd):
    """d/dx of LayerNorm(x) (no affine) applied to the upstream gradient dxh."""
    return rstd * (dxh - dxh.mean(-1, keepdims=True) - xh * (dxh * xh).mean(-1, keepdims=True))


def rms_fwd(x, g):
    r = 1.0 / np.sqrt((x ** 2).mean(-1, keepdims=True) + RMS_EPS)
    return x * r * g, r


def rms_bwd(dy, x, r, g):
    """Returns (dx, dg summed over all leading axes)."""
    u = dy * g
    n = x.shape[-1]
    dx = r * u - x * r ** 3 * (x * u).sum(-1, keepdims=True) / n
    dg = (dy * x * r).reshape(-1, n).sum(0)
    return dx, dg


def softmax_probs(qh, kh):
    """P = softmax(qh kh^T / sqrt(dh)) row by row, for one (sequence, head): qh, kh [N, dh]
    -> P [N, N] (row n: the weights query n gives the keys)."""
    S = qh @ kh.T / np.sqrt(qh.shape[-1])
    S = S - S.max(-1, keepdims=True)
    P = np.exp(S)
    P /= P.sum(-1, keepdims=True)
    return P


def attention(q, k, v, keep_probs=False):
    """q, k, v: [B, N, h, dh] -> o [B, N, h, dh] (and the probabilities P [B, h, N, N] if
    keep_probs), one (sequence, head) at a time: o = P v."""
    B, N, h, _ = q.shape
    o = np.empty(v.shape)
    P_all = np.empty((B, h, N, N)) if keep_probs else None
    for b in range(B):
        for j in range(h):
            P = softmax_probs(q[b, :, j], k[b, :, j])
            o[b, :, j] = P @ v[b, :, j]
            if keep_probs:
                P_all[b, j] = P
    return o, P_all


def attention_bwd(do, q, k, v):
    """dV = P^T dO, dP = dO V^T, dS = P*(dP - rowsum(dP*P)), dQ = dS K/sqrt(dh),
    dK = dS^T Q/sqrt(dh)  (appendix, Eqs. bwd_V .. bwd_QK), one (sequence, head) at a time;
    P is formed again from q and k exactly as the forward formed it."""
    B, N, h, dh = q.shape
    dq, dk, dv = np.empty(q.shape), np.empty(k.shape), np.empty(v.shape)
    for b in range(B):
        for j in range(h):
            qh, kh, vh, doh = q[b, :, j], k[b, :, j], v[b, :, j], do[b, :, j]
            P = softmax_probs(qh, kh)
            dv[b, :, j] = P.T @ doh
            dP = doh @ vh.T
            dS = P * (dP - (dP * P).sum(-1, keepdims=True))
            dq[b, :, j] = dS @ kh / np.sqrt(dh)
            dk[b, :, j] = dS.T @ qh / np.sqrt(dh)
    return dq, dk, dv


def lin(x, W, b):
    return x @ W.T + b


def lin_bwd(dy, x, W, grads, wname, bname):
    """Accumulate dW = dy^T x and db = sum dy over all rows; return dx = dy W."""
    d2 = dy.reshape(-1, dy.shape[-1])
    x2 = x.reshape(-1, x.shape[-1])
    grads[wname] += d2.T @ x2
    grads[bname] += d2.sum(0)
    return dy @ W


def modulate(xh, sh, sc):
    return xh * (1.0 + sc[:, None, :]) + sh[:, None, :]


def modulate_bwd(dm, xh, sc):
    """Returns (dxh, dsh [B,d], dsc [B,d])."""
    return dm * (1.0 + sc[:, None, :]), dm.sum(1), (dm * xh).sum(1)


# --------------------------------------------------------------------------- model
class Backbone:
    """The pinned velocity network v_theta(z, t, txt) with parameters `params` (float64)."""

    def __init__(self, wl, params):
        self.wl = wl
        self.p = params
        self.gh = wl.latent_h // wl.patch
        self.gw = wl.latent_w // wl.patch
        if wl.pos_embed:
            self.pos = pos_embed_2d(self.gh, self.gw, wl.hidden)
        if wl.rope:
            self.ang = rope_angles(self.gh, self.gw, wl.txt_len, wl.head_dim)

    # ---- attention core shared by all block types: [B,N,3d] -> [B,N,d]
    def _attn_fwd(self, qkv, qn=None, kn=None):
        wl = self.wl
        B, N, _ = qkv.shape
        h, dh, d = wl.heads, wl.head_dim, wl.hidden
        q = qkv[..., :d].reshape(B, N, h, dh)
        k = qkv[..., d:2 * d].reshape(B, N, h, dh)
        v = qkv[..., 2 * d:].reshape(B, N, h, dh)
        cache = {"q_raw": q, "k_raw": k}
        if qn is not None:
            # qn / kn: per-token scale arrays [N, dh] (each stream has its own scale)
            q, cache["rq"] = rms_fwd(q, qn[None, :, None, :])
            k, cache["rk"] = rms_fwd(k, kn[None, :, None, :])
        if wl.rope:
            q = rope_apply(q, self.ang)
            k = rope_apply(k, self.ang)
        o, _ = attention(q, k, v)
        cache.update(q=q, k=k, v=v)
        return o.reshape(B, N, d), cache

    def _attn_bwd(self, do, cache, qn=None, kn=None):
        """Returns (dqkv, dqn_tok [N,dh] or None, dkn_tok)."""
        wl = self.wl
        B, N, d = do.shape
        h, dh = wl.heads, wl.head_dim
        dq, dk, dv = attention_bwd(do.reshape(B, N, h, dh), cache["q"], cache["k"], cache["v"])
        if wl.rope:
            dq = rope_apply(dq, self.ang, inverse=True)
            dk = rope_apply(dk, self.ang, inverse=True)
        dqn = dkn = None
        if qn is not None:
            gq = qn[None, :, None, :]
            gk = kn[None, :, None, :]
            rq, rk = cache["rq"], cache["rk"]
            xq, xk = cache["q_raw"], cache["k_raw"]
            dqn = (dq * xq * rq).sum(axis=(0, 2))       # [N, dh]
            dkn = (dk * xk * rk).sum(axis=(0, 2))
            uq = dq * gq
            uk = dk * gk
            dq = rq * uq - xq * rq ** 3 * (xq * uq).sum(-1, keepdims=True) / dh
            dk = rk * uk - xk * rk ** 3 * (xk * uk).sum(-1, keepdims=True) / dh
        dqkv = np.concatenate([dq.reshape(B, N, d), dk.reshape(B, N, d), dv.reshape(B, N, d)], -1)
        return dqkv, dqn, dkn

    # ---- forward
    def forward(self, z, t, txt):
        """z [B,C,H,W], t [B], txt [B,Ntxt,Dtxt] -> v [B,C,H,W], cache."""
        wl, p = self.wl, self.p
        d = wl.hidden
        B = z.shape[0]
        cache = {}
        xp = patchify(np.asarray(z, np.float64), wl.patch)
        ximg = lin(xp, p["x_embed.w"], p["x_embed.b"])
        if wl.pos_embed:
            ximg = ximg + self.pos[None]
        xtxt = lin(txt, p["txt_embed.w"], p["txt_embed.b"])
        phi = timestep_embedding(t, wl.freq_dim)
        e1 = lin(phi, p["t_embed.w1"], p["t_embed.b1"])
        c = lin(silu(e1), p["t_embed.w2"], p["t_embed.b2"])
        sc_ = silu(c)
        cache.update(xp=xp, txt=txt, phi=phi, e1=e1, c=c, sc_=sc_)
        blocks = []
        nt = wl.txt_len
        if wl.arch == "dit":
            hcur = np.concatenate([xtxt, ximg], axis=1)
            for i in range(wl.depth):
                hcur, bc = self._dit_block_fwd(hcur, sc_, f"blocks.{i}.")
                blocks.append(bc)
        else:
            ht, hi = xtxt, ximg
            for i in range(wl.depth_double):
                ht, hi, bc = self._double_fwd(ht, hi, sc_, f"double.{i}.")
                blocks.append(bc)
            hcur = np.concatenate([ht, hi], axis=1)
            for i in range(wl.depth):
                hcur, bc = self._single_fwd(hcur, sc_, f"single.{i}.")
                blocks.append(bc)
        cache["blocks"] = blocks
        fm = lin(sc_, p["final.mod.w"], p["final.mod.b"])
        sh, scl = fm[:, :d], fm[:, d:]
        xf, rf = ln_fwd(hcur[:, nt:])
        mf = modulate(xf, sh, scl)
        vt = lin(mf, p["final.out.w"], p["final.out.b"])
        cache.update(xf=xf, rf=rf, scl=scl, mf=mf)
        v = unpatchify(vt, wl.in_channels, wl.latent_h, wl.latent_w, wl.patch)
        return v, cache

    def _dit_block_fwd(self, h, sc_, pre):
        p, d = self.p, self.wl.hidden
        mod = lin(sc_, p[pre + "mod.w"], p[pre + "mod.b"])
        sh1, sc1, g1, sh2, sc2, g2 = (mod[:, k * d:(k + 1) * d] for k in range(6))
        x1, r1 = ln_fwd(h)
        a = modulate(x1, sh1, sc1)
        qkv = lin(a, p[pre + "qkv.w"], p[pre + "qkv.b"])
        o, ac = self._attn_fwd(qkv)
        y1 = lin(o, p[pre + "proj.w"], p[pre + "proj.b"])
        h2 = h + g1[:, None, :] * y1
        x2, r2 = ln_fwd(h2)
        m = modulate(x2, sh2, sc2)
        u = lin(m, p[pre + "fc1.w"], p[pre + "fc1.b"])
        gu = gelu(u)
        y2 = lin(gu, p[pre + "fc2.w"], p[pre + "fc2.b"])
        h3 = h2 + g2[:, None, :] * y2
        return h3, dict(pre=pre, mod=mod, x1=x1, r1=r1, a=a, ac=ac, o=o, y1=y1,
                        x2=x2, r2=r2, m=m, u=u, gu=gu, y2=y2)

    def _double_fwd(self, ht, hi, sc_, pre):
        """Double-stream block: per-stream weights, joint attention over [txt; img]."""
        p, wl = self.p, self.wl
        d, nt = wl.hidden, wl.txt_len
        st = {}
        qkvs = []
        for s, hs in (("txt", ht), ("img", hi)):
            q = pre + s + "."
            mod = lin(sc_, p[q + "mod.w"], p[q + "mod.b"])
            x1, r1 = ln_fwd(hs)
            a = modulate(x1, mod[:, :d], mod[:, d:2 * d])
            qkv = lin(a, p[q + "qkv.w"], p[q + "qkv.b"])
            st[s] = dict(mod=mod, x1=x1, r1=r1, a=a)
            qkvs.append(qkv)
        qkv = np.concatenate(qkvs, axis=1)
        N = qkv.shape[1]
        qn = np.concatenate([np.broadcast_to(p[pre + "txt.q_norm"], (nt, wl.head_dim)),
                             np.broadcast_to(p[pre + "img.q_norm"], (N - nt, wl.head_dim))])
        kn = np.concatenate([np.broadcast_to(p[pre + "txt.k_norm"], (nt, wl.head_dim)),
                             np.broadcast_to(p[pre + "img.k_norm"], (N - nt, wl.head_dim))])
        o, ac = self._attn_fwd(qkv, qn, kn)
        outs = {}
        for s, hs, sl in (("txt", ht, slice(0, nt)), ("img", hi, slice(nt, N))):
            q = pre + s + "."
            c = st[s]
            mod = c["mod"]
            g1, sh2, sc2, g2 = (mod[:, k * d:(k + 1) * d] for k in range(2, 6))
            os_ = o[:, sl]
            y1 = lin(os_, p[q + "proj.w"], p[q + "proj.b"])
            h2 = hs + g1[:, None, :] * y1
            x2, r2 = ln_fwd(h2)
            m = modulate(x2, sh2, sc2)
            u = lin(m, p[q + "fc1.w"], p[q + "fc1.b"])
            gu = gelu(u)
            y2 = lin(gu, p[q + "fc2.w"], p[q + "fc2.b"])
            outs[s] = h2 + g2[:, None, :] * y2
            c.update(o=os_, y1=y1, x2=x2, r2=r2, m=m, u=u, gu=gu, y2=y2)
        return outs["txt"], outs["img"], dict(pre=pre, st=st, ac=ac, qn=qn, kn=kn)

    def _single_fwd(self, h, sc_, pre):
        """Flux-style single block: one lin1 producing [qkv | u], lin2 on [o | GELU(u)]."""
        p, wl = self.p, self.wl
        d = wl.hidden
        N = h.shape[1]
        mod = lin(sc_, p[pre + "mod.w"], p[pre + "mod.b"])
        sh, sc, g = mod[:, :d], mod[:, d:2 * d], mod[:, 2 * d:]
        x1, r1 = ln_fwd(h)
        a = modulate(x1, sh, sc)
        l1 = lin(a, p[pre + "lin1.w"], p[pre + "lin1.b"])
        qkv, u = l1[..., :3 * d], l1[..., 3 * d:]
        qn = np.broadcast_to(p[pre + "q_norm"], (N, wl.head_dim))
        kn = np.broadcast_to(p[pre + "k_norm"], (N, wl.head_dim))
        o, ac = self._attn_fwd(qkv, qn, kn)
        cat = np.concatenate([o, gelu(u)], axis=-1)
        y = lin(cat, p[pre + "lin2.w"], p[pre + "lin2.b"])
        return h + g[:, None, :] * y, dict(pre=pre, mod=mod, x1=x1, r1=r1, a=a, u=u,
                                             ac=ac, cat=cat, y=y, qn=qn, kn=kn)

    # ---- reverse mode
    def vjp(self, cache, cot):
        """Parameter gradient sum_rows J(row)^T cot[row] for cot [B,C,H,W] (Phase 4).

        z and txt are fixed samples (Sec. 3.3, Phase 2): no gradient flows to them."""
        wl, p = self.wl, self.p
        d, nt = wl.hidden, wl.txt_len
        grads = {k: np.zeros_like(v) for k, v in p.items()}
        dvt = patchify(np.asarray(cot, np.float64), wl.patch)
        dmf = lin_bwd(dvt, cache["mf"], p["final.out.w"], grads, "final.out.w", "final.out.b")
        dxf, dsh, dscl = modulate_bwd(dmf, cache["xf"], cache["scl"])
        dhimg = ln_bwd(dxf, cache["xf"], cache["rf"])
        sc_ = cache["sc_"]
        dsc_ = lin_bwd(np.concatenate([dsh, dscl], 1), sc_, p["final.mod.w"], grads,
                       "final.mod.w", "final.mod.b")
        B = dvt.shape[0]
        blocks = cache["blocks"]
        if wl.arch == "dit":
            dh = np.concatenate([np.zeros((B, nt, d)), dhimg], axis=1)
            for bc in reversed(blocks):
                dh, dmod = self._dit_block_bwd(dh, bc, grads)
                pre = bc["pre"]
                dsc_ += lin_bwd(dmod, sc_, p[pre + "mod.w"], grads, pre + "mod.w", pre + "mod.b")
            dxtxt, dximg = dh[:, :nt], dh[:, nt:]
        else:
            dh = np.concatenate([np.zeros((B, nt, d)), dhimg], axis=1)
            for bc in reversed(blocks[wl.depth_double:]):
                dh, dmod = self._single_bwd(dh, bc, grads)
                pre = bc["pre"]
                dsc_ += lin_bwd(dmod, sc_, p[pre + "mod.w"], grads, pre + "mod.w", pre + "mod.b")
            dht, dhi = dh[:, :nt], dh[:, nt:]
            for bc in reversed(blocks[:wl.depth_double]):
                dht, dhi, dmods = self._double_bwd(dht, dhi, bc, grads)
                for s in ("txt", "img"):
                    q = bc["pre"] + s + "."
                    dsc_ += lin_bwd(dmods[s], sc_, p[q + "mod.w"], grads, q + "mod.w", q + "mod.b")
            dxtxt, dximg = dht, dhi
        dc = dsc_ * silu_grad(cache["c"])
        dse1 = lin_bwd(dc, silu(cache["e1"]), p["t_embed.w2"], grads, "t_embed.w2", "t_embed.b2")
        de1 = dse1 * silu_grad(cache["e1"])
        lin_bwd(de1, cache["phi"], p["t_embed.w1"], grads, "t_embed.w1", "t_embed.b1")
        lin_bwd(dximg, cache["xp"], p["x_embed.w"], grads, "x_embed.w", "x_embed.b")
        lin_bwd(dxtxt, cache["txt"], p["txt_embed.w"], grads, "txt_embed.w", "txt_embed.b")
        return grads

    def _dit_block_bwd(self, dh3, c, grads):
        p, d = self.p, self.wl.hidden
        pre, mod = c["pre"], c["mod"]
        sh1, sc1, g1, sh2, sc2, g2 = (mod[:, k * d:(k + 1) * d] for k in range(6))
        dg2 = (dh3 * c["y2"]).sum(1)
        dy2 = g2[:, None, :] * dh3
        dgu = lin_bwd(dy2, c["gu"], p[pre + "fc2.w"], grads, pre + "fc2.w", pre + "fc2.b")
        du = dgu * gelu_grad(c["u"])
        dm = lin_bwd(du, c["m"], p[pre + "fc1.w"], grads, pre + "fc1.w", pre + "fc1.b")
        dx2, dsh2, dsc2 = modulate_bwd(dm, c["x2"], sc2)
        dh2 = dh3 + ln_bwd(dx2, c["x2"], c["r2"])
        dg1 = (dh2 * c["y1"]).sum(1)
        dy1 = g1[:, None, :] * dh2
        do = lin_bwd(dy1, c["o"], p[pre + "proj.w"], grads, pre + "proj.w", pre + "proj.b")
        dqkv, _, _ = self._attn_bwd(do, c["ac"])
        da = lin_bwd(dqkv, c["a"], p[pre + "qkv.w"], grads, pre + "qkv.w", pre + "qkv.b")
        dx1, dsh1, dsc1 = modulate_bwd(da, c["x1"], sc1)
        dh = dh2 + ln_bwd(dx1, c["x1"], c["r1"])
        return dh, np.concatenate([dsh1, dsc1, dg1, dsh2, dsc2, dg2], axis=1)

    def _double_bwd(self, dht, dhi, bc, grads):
        p, wl = self.p, self.wl
        d, nt = wl.hidden, wl.txt_len
        pre, st = bc["pre"], bc["st"]
        dos, dh2s, dmods = [], {}, {}
        for s, dh3 in (("txt", dht), ("img", dhi)):
            q = pre + s + "."
            c = st[s]
            mod = c["mod"]
            g1, sh2, sc2, g2 = (mod[:, k * d:(k + 1) * d] for k in range(2, 6))
            dg2 = (dh3 * c["y2"]).sum(1)
            dy2 = g2[:, None, :] * dh3
            dgu = lin_bwd(dy2, c["gu"], p[q + "fc2.w"], grads, q + "fc2.w", q + "fc2.b")
            du = dgu * gelu_grad(c["u"])
            dm = lin_bwd(du, c["m"], p[q + "fc1.w"], grads, q + "fc1.w", q + "fc1.b")
            dx2, dsh2, dsc2 = modulate_bwd(dm, c["x2"], sc2)
            dh2 = dh3 + ln_bwd(dx2, c["x2"], c["r2"])
            dg1 = (dh2 * c["y1"]).sum(1)
            dy1 = g1[:, None, :] * dh2
            dos.append(lin_bwd(dy1, c["o"], p[q + "proj.w"], grads, q + "proj.w", q + "proj.b"))
            dh2s[s] = dh2
            dmods[s] = [None, None, dg1, dsh2, dsc2, dg2]
        do = np.concatenate(dos, axis=1)
        dqkv, dqn, dkn = self._attn_bwd(do, bc["ac"], bc["qn"], bc["kn"])
        grads[pre + "txt.q_norm"] += dqn[:nt].sum(0)
        grads[pre + "img.q_norm"] += dqn[nt:].sum(0)
        grads[pre + "txt.k_norm"] += dkn[:nt].sum(0)
        grads[pre + "img.k_norm"] += dkn[nt:].sum(0)
        out = {}
        for s, sl in (("txt", slice(0, nt)), ("img", slice(nt, None))):
            q = pre + s + "."
            c = st[s]
            sc1 = c["mod"][:, d:2 * d]
            da = lin_bwd(dqkv[:, sl], c["a"], p[q + "qkv.w"], grads, q + "qkv.w", q + "qkv.b")
            dx1, dsh1, dsc1 = modulate_bwd(da, c["x1"], sc1)
            out[s] = dh2s[s] + ln_bwd(dx1, c["x1"], c["r1"])
            dmods[s][0], dmods[s][1] = dsh1, dsc1
            dmods[s] = np.concatenate(dmods[s], axis=1)
        return out["txt"], out["img"], dmods

    def _single_bwd(self, dh, c, grads):
        p, wl = self.p, self.wl
        d = wl.hidden
        pre, mod = c["pre"], c["mod"]
        sc, g = mod[:, d:2 * d], mod[:, 2 * d:]
        dg = (dh * c["y"]).sum(1)
        dy = g[:, None, :] * dh
        dcat = lin_bwd(dy, c["cat"], p[pre + "lin2.w"], grads, pre + "lin2.w", pre + "lin2.b")
        do, dgu = dcat[..., :d], dcat[..., d:]
        du = dgu * gelu_grad(c["u"])
        dqkv, dqn, dkn = self._attn_bwd(do, c["ac"], c["qn"], c["kn"])
        grads[pre + "q_norm"] += dqn.sum(0)
        grads[pre + "k_norm"] += dkn.sum(0)
        da = lin_bwd(np.concatenate([dqkv, du], axis=-1), c["a"], p[pre + "lin1.w"], grads,
                     pre + "lin1.w", pre + "lin1.b")
        dx1, dsh, dsc = modulate_bwd(da, c["x1"], sc)
        return dh + ln_bwd(dx1, c["x1"], c["r1"]), np.concatenate([dsh, dsc, dg], axis=1)
