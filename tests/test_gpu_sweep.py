"""The routing and window sweep of the Qwen-width configuration (dual-stream blocks only) at a
reduced size: for W in {2, 4, 8} and jagg_frac in {0, 0.5, 1}, a whole group's update stage
through the library -- per-window step signals, the jagg_frac routing, the aggregated
endpoint cotangents of the JAGG windows and the per-step signals of the others, one joint
VJP over every window's rows -- against the oracle's sum of window gradients (JAGG for the
routed windows, exact for the rest).  Then the per-window cosine between the JAGG and the
exact gradients, the quantity the calibration rule routes on (grad_reduce on the GPU
against the oracle's grad_stats), and the routes it gives.

Each stage gets identical inputs on both sides: the oracle's rollout (model outputs rounded
to float32, states stored in float32) feeds the signals, and the network-input times are
the float32 values the library's forward takes."""
import numpy as np
import pytest
import torch

import synth
from gpu_cases import GpuModel, cosine, flat, rel_l2
from oracle import dit, grpo, path
from oracle.rollout import rollout

pytestmark = pytest.mark.gpu

jg = pytest.importorskip("paper_2607_17572_gb300")

QWEN = synth.WORKLOADS["mmdit_qwen_sweep_bf16"]
WL = synth.small_variant(QWEN, name="qwen_tiny_f32", dtype="f32", hidden=64, heads=4, mlp=256, depth=0,
                         depth_double=2, in_channels=4, latent_h=4, latent_w=4, patch=1, txt_len=8, txt_dim=64,
                         G=4, T=8, clip_eps=1e-4)


def _group(W, seed=3):
    wl = synth.small_variant(WL, W=W)
    params = synth.make_params(wl)
    draws = synth.draw_group(wl, seed=seed)
    t = synth.time_grid(wl.T, wl.shift)
    sig = synth.sigma_schedule(t, wl.eta)
    model_o = dit.Backbone(wl, params)
    z, v, lp = rollout(model_o, wl, draws, t, sig)
    v = v.astype(np.float32).astype(np.float64)
    logp_old = lp + draws.delta
    rewards = draws.rewards.astype(np.float32).astype(np.float64)
    return wl, params, draws, t, sig, model_o, z, v, logp_old, rewards


def _signals(wl, w, z, v, t, sig, logp_old, rewards, jagg):
    """The library's Phase 2 (+3) for window w: cotangent rows in the window's row order."""
    G, W, D = wl.G, wl.W, wl.D
    dev = "cuda"
    f64 = dict(dtype=torch.float64, device=dev)
    sl = slice(w * W, (w + 1) * W)
    vw = torch.tensor(v[:, sl].reshape(G, W, D), dtype=torch.float32, device=dev)
    zw = torch.tensor(z[:, w * W:w * W + W + 1].reshape(G, W + 1, D), dtype=torch.float32, device=dev)
    out = dict(logp_new=torch.empty(G, W, **f64), ratio=torch.empty(G, W, **f64),
               clipped=torch.empty(G, W, dtype=torch.uint8, device=dev), adv_out=torch.empty(G, **f64))
    ws = jg.alloc_bytes(jg.signals_workspace_bytes(G, W, D))
    kw = dict(cot_out=torch.empty(2 * G, D, device=dev)) if jagg else dict(s_out=torch.empty(G, W, D, device=dev))
    jg.grpo_step_signals(vw, zw, torch.tensor(t[w * W:w * W + W + 1], **f64), torch.tensor(sig[sl], **f64),
                         torch.tensor(logp_old[:, sl], **f64), torch.tensor(rewards, dtype=torch.float32, device=dev),
                         wl.clip_eps, wl.adv_clip, wl.adv_eps, 1.0 / (G * wl.T), ws=ws, **kw, **out)
    return (kw["cot_out"] if jagg else kw["s_out"].reshape(G * W, D)).cpu().numpy(), out["clipped"].cpu().numpy()


def _rows(wl, w, z, t32, jagg):
    """The window's VJP rows in the order of _signals' cotangents (JAGG: endpoint 0 of every
    sample, then endpoint W-1; exact: sample-major, row i W + j)."""
    G, W = wl.G, wl.W
    zw = z[:, w * W:(w + 1) * W]
    tw = t32[w * W:(w + 1) * W]
    if jagg:
        return (np.concatenate([zw[:, 0], zw[:, W - 1]]), np.concatenate([np.full(G, tw[0]), np.full(G, tw[-1])]))
    return zw.reshape((G * W,) + zw.shape[2:]), np.tile(tw, G)


def _oracle_signals(wl, w, z, v, t, sig, logp_old, rewards):
    G, W, D = wl.G, wl.W, wl.D
    sl = slice(w * W, (w + 1) * W)
    s, _, _, clipped = grpo.step_signals(v[:, sl].reshape(G, W, D), z[:, w * W:w * W + W + 1].reshape(G, W + 1, D),
                                         t[w * W:w * W + W + 1], sig[sl], logp_old[:, sl], grpo.advantages(rewards),
                                         wl.clip_eps, 1.0 / (G * wl.T))
    return s.reshape((G, W) + z.shape[2:]), clipped


@pytest.mark.parametrize("jagg_frac", [0.0, 0.5, 1.0])
@pytest.mark.parametrize("W", [2, 4, 8])
def test_routed_group_update_matches_oracle(W, jagg_frac):
    wl, params, draws, t, sig, model_o, z, v, logp_old, rewards = _group(W)
    nw = wl.T // W
    t32 = t.astype(np.float32).astype(np.float64)
    routes, frac = jg.jagg_route(nw, jagg_frac)
    assert routes == grpo.route_schedule(nw, jagg_frac).tolist()
    gm = GpuModel(jg, wl, params)
    zs, ts, cots = [], [], []
    g_o = None
    for w in range(nw):
        cot, clipped = _signals(wl, w, z, v, t, sig, logp_old, rewards, routes[w])
        s_o, clipped_o = _oracle_signals(wl, w, z, v, t, sig, logp_old, rewards)
        np.testing.assert_array_equal(clipped, clipped_o)
        zr, tr = _rows(wl, w, z, t32, routes[w])
        zs.append(zr)
        ts.append(tr)
        cots.append(cot)
        gw = path.window_gradient(model_o, z[:, w * W:(w + 1) * W], t32[w * W:(w + 1) * W], draws.txt, s_o,
                                  jagg=bool(routes[w]))
        g_o = gw if g_o is None else {k: g_o[k] + gw[k] for k in g_o}
    zr, tr, cot = np.concatenate(zs), np.concatenate(ts), np.concatenate(cots)
    B = zr.shape[0]
    _, saved, ws = gm.forward(zr, tr, np.broadcast_to(draws.txt, (B,) + draws.txt.shape))
    grad = gm.vjp(saved, ws, B, cot.reshape(zr.shape))
    torch.cuda.synchronize()
    assert jg.device_status() == 0
    g_gpu = jg.unpack_grads(gm.cfg, grad)
    names = list(g_o)
    err, cs = rel_l2(flat(g_gpu, names), flat(g_o, names)), cosine(flat(g_gpu, names), flat(g_o, names))
    print(f"W={W} jagg_frac={jagg_frac}: routes {routes}, gradient rel L2 {err:.2e}, cos {cs:.8f}")
    assert err <= 1e-4 and cs >= 0.999


@pytest.mark.parametrize("W", [2, 4, 8])
def test_window_cosines_and_calibrated_routes_match_oracle(W):
    """Per window: cos(g_JAGG, g_exact) from the library's two VJPs and grad_reduce, against
    the oracle's; the calibration rule's routes agree except within 1e-3 of the threshold."""
    wl, params, draws, t, sig, model_o, z, v, logp_old, rewards = _group(W, seed=4)
    nw = wl.T // W
    t32 = t.astype(np.float32).astype(np.float64)
    gm = GpuModel(jg, wl, params)
    P = jg.param_count(gm.cfg)
    out3 = torch.empty(3, dtype=torch.float64, device="cuda")
    gws = jg.alloc_bytes(jg.grad_reduce_workspace_bytes(P))
    cos_gpu, cos_o = [], []
    for w in range(nw):
        grads = []
        for jagg in (True, False):
            cot, _ = _signals(wl, w, z, v, t, sig, logp_old, rewards, jagg)
            zr, tr = _rows(wl, w, z, t32, jagg)
            B = zr.shape[0]
            _, saved, ws = gm.forward(zr, tr, np.broadcast_to(draws.txt, (B,) + draws.txt.shape))
            grads.append(gm.vjp(saved, ws, B, cot.reshape(zr.shape)))
        jg.grad_reduce(grads[0], grads[1], out3=out3, ws=gws)
        torch.cuda.synchronize()
        ab, aa, bb = out3.cpu().numpy()
        cos_gpu.append(ab / np.sqrt(aa * bb))
        s_o, _ = _oracle_signals(wl, w, z, v, t, sig, logp_old, rewards)
        zw, tw = z[:, w * W:(w + 1) * W], t32[w * W:(w + 1) * W]
        gj = path.window_gradient(model_o, zw, tw, draws.txt, s_o, jagg=True)
        ge = path.window_gradient(model_o, zw, tw, draws.txt, s_o, jagg=False)
        names = list(gj)
        cos_o.append(grpo.grad_stats(flat(gj, names), flat(ge, names))[3])
    assert jg.device_status() == 0
    print(f"W={W}: cos gpu {np.round(cos_gpu, 6)}, oracle {np.round(cos_o, 6)}")
    np.testing.assert_allclose(cos_gpu, cos_o, atol=1e-5)
    if W == 2:
        np.testing.assert_allclose(cos_o, 1.0, atol=1e-12)   # W = 2: JAGG is the exact gradient
    routes, frac = jg.jagg_route(nw, cos=cos_gpu, tau=0.5)
    ro, fo = grpo.route_calibrate(np.array(cos_o), 0.5)
    near = np.abs(np.array(cos_o) - 0.5) < 1e-3
    assert all(a == b for a, b, n in zip(routes, ro.tolist(), near) if not n)
