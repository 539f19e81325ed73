"""GPU parity of Phase 1 (forward with saved activations) and Phase 4 (the joint VJP)
with the float64 oracle on the same seeded weights, inputs and cotangents."""
import numpy as np
import pytest
import torch

import synth
from gpu_cases import GpuModel, cosine, flat, model_inputs, oracle_vjp, rel_l2
from oracle import dit, path

pytestmark = pytest.mark.gpu

jg = pytest.importorskip("paper_2607_17572_gb300")

TINY = synth.WORKLOADS["tiny_dit_f32"]
DITB = synth.WORKLOADS["dit_b_bf16"]

FLUX = synth.WORKLOADS["mmdit_flux512_bf16"]
TINY_MM = synth.small_variant(TINY, name="tiny_mmdit", arch="mmdit", depth=2, depth_double=2, shift=3.0)

CASES = [
    # (workload, rows B, forward tol, gradient tol)
    (TINY, 8, 1e-5, 1e-4),                                                    # 2G rows of the tiny config
    (synth.small_variant(TINY, name="tiny_odd", latent_h=6, latent_w=5, txt_len=3, txt_dim=40), 3, 1e-5, 1e-4),
    (synth.small_variant(DITB, name="ditb_2blocks", depth=2), 4, 2e-2, 1e-2),  # DiT-B width, 2 blocks
    (synth.small_variant(DITB, name="ditb_ragged", depth=1, latent_h=18, latent_w=22, txt_len=29), 3, 2e-2, 1e-2),
    # MMDiT: double blocks (per-stream weights, QK RMSNorm, 2D RoPE, joint attention)
    # followed by Flux-style single blocks
    (TINY_MM, 8, 1e-5, 1e-4),
    (synth.small_variant(TINY_MM, name="tiny_mmdit_odd", latent_h=6, latent_w=5, txt_len=3, txt_dim=40), 3,
     1e-5, 1e-4),
    (synth.small_variant(TINY_MM, name="tiny_mmdit_doubles_only", depth=0, depth_double=3), 4, 1e-5, 1e-4),
    (synth.small_variant(TINY_MM, name="tiny_mmdit_singles_only", depth=3, depth_double=0), 4, 1e-5, 1e-4),
    (synth.small_variant(TINY_MM, name="tiny_mmdit_dh32", hidden=128, heads=4, mlp=256), 2, 1e-5, 1e-4),
    # bf16 at the Flux head dim (128) and at 64, reduced width and depth
    (synth.small_variant(FLUX, name="mmdit_dh128_1d1s", hidden=512, heads=4, mlp=2048, depth=1, depth_double=1,
                         latent_h=16, latent_w=20, txt_len=24, txt_dim=256), 2, 2e-2, 1e-2),
    (synth.small_variant(FLUX, name="mmdit_dh64_2d1s", hidden=384, heads=6, mlp=1536, depth=1, depth_double=2,
                         latent_h=14, latent_w=14, txt_len=37, txt_dim=128), 3, 2e-2, 1e-2),
]


def _check(wl, B, ftol, gtol, seed=5):
    params = synth.make_params(wl)
    z, t, txt = model_inputs(wl, B, seed)
    rng = np.random.Generator(np.random.PCG64(seed + 1))
    cot = synth.storage_round(rng.standard_normal(z.shape), wl.dtype)
    gm = GpuModel(jg, wl, params)
    v, saved, ws = gm.forward(z, t, txt)
    grad = gm.vjp(saved, ws, B, cot)
    torch.cuda.synchronize()
    assert jg.device_status() == 0
    v_o, g_o = oracle_vjp(wl, params, z, t, txt, cot)
    fv = rel_l2(v.float().cpu().numpy(), v_o)
    assert fv <= ftol, f"forward rel L2 {fv:.3e}"
    g_gpu = jg.unpack_grads(gm.cfg, grad)
    names = list(g_o)
    tot = rel_l2(flat(g_gpu, names), flat(g_o, names))
    cs = cosine(flat(g_gpu, names), flat(g_o, names))
    per = {k: rel_l2(g_gpu[k], g_o[k]) for k in names}
    worst = max(per, key=per.get)
    print(f"{wl.name}: forward {fv:.2e}, grad rel L2 {tot:.2e}, cos {cs:.6f}, worst {worst} {per[worst]:.2e}")
    assert tot <= gtol, f"gradient rel L2 {tot:.3e} (worst {worst}: {per[worst]:.3e})"
    assert cs >= 0.999
    # every tensor on its own, so that a wrong gradient of a small tensor (a bias, a norm
    # scale, the final layer) cannot hide under the norm of the large ones
    bad = {k: e for k, e in per.items() if e > 5 * gtol}
    assert not bad, f"tensors beyond {5 * gtol:.0e}: {bad}"
    return grad, gm, saved, ws, cot


@pytest.mark.parametrize("wl,B,ftol,gtol", CASES, ids=[c[0].name for c in CASES])
def test_forward_and_joint_vjp_match_oracle(wl, B, ftol, gtol):
    _check(wl, B, ftol, gtol)


def test_vjp_accumulates_and_is_linear_in_the_cotangent():
    wl = TINY
    grad, gm, saved, ws, cot = _check(wl, 8, 1e-5, 1e-4)
    g1 = grad.clone()
    gm.vjp(saved, ws, 8, 2.0 * cot, grad=grad)      # grad += J^T (2 cot)
    torch.cuda.synchronize()
    assert rel_l2(grad.cpu().numpy(), 3.0 * g1.cpu().numpy()) < 1e-5


@pytest.mark.parametrize("wl", [synth.small_variant(DITB, name="ditb_2blocks", depth=2),
                                synth.small_variant(FLUX, name="mmdit_dh128_2d3s", hidden=512, heads=4, mlp=2048,
                                                    depth=3, depth_double=2, latent_h=16, latent_w=16, txt_len=40,
                                                    txt_dim=256)],
                         ids=lambda w: w.name)
def test_forward_without_saves_matches_saved_forward(wl):
    params = synth.make_params(wl)
    z, t, txt = model_inputs(wl, 4, 9)
    gm = GpuModel(jg, wl, params)
    v1, _, _ = gm.forward(z, t, txt, save=True)
    v2, _, _ = gm.forward(z, t, txt, save=False)
    torch.cuda.synchronize()
    assert torch.equal(v1, v2)


@pytest.mark.slow
def test_dit_b_full_depth_joint_vjp():
    """DiT-B (12 blocks, 333 tokens) at its JAGG batch of 2G = 16 rows."""
    _check(DITB, 2 * DITB.G, 2e-2, 1e-2, seed=11)


@pytest.mark.parametrize("wl,G,tol", [(TINY, 4, 1e-5), (synth.small_variant(DITB, name="ditb_2blocks", depth=2), 4,
                                                        5e-3)], ids=["tiny_f32", "ditb_2blocks_bf16"])
def test_sequential_graph_variant_matches_the_joint_vjp(wl, G, tol):
    """Algorithm 2: forward of endpoint 0 into one G-row arena, VJP with s_base, forward of
    endpoint W-1 into the same arena, VJP with s_corr -- the same gradient as one joint VJP
    over 2G rows, with half the saved activations.  (bf16: a G-row and a 2G-row product may
    pick different tile widths and round differently, a few 1e-3 relative.)"""
    params = synth.make_params(wl)
    z, t, txt = model_inputs(wl, 2 * G, 21)
    t[:G], t[G:] = 0.8, 0.55
    rng = np.random.Generator(np.random.PCG64(22))
    cot = rng.standard_normal(z.shape)
    gm = GpuModel(jg, wl, params)
    v, saved, ws = gm.forward(z, t, txt)
    g_joint = gm.vjp(saved, ws, 2 * G, cot)
    assert gm.model.saved_bytes(G) <= 0.51 * gm.model.saved_bytes(2 * G)
    g_seq = torch.zeros_like(g_joint)
    arena = jg.alloc_bytes(gm.model.saved_bytes(G))      # the one arena of both endpoints
    ws1 = jg.alloc_bytes(gm.model.workspace_bytes(G))
    for part in (slice(0, G), slice(G, 2 * G)):
        zt = gm.tensor(z[part])
        jg.dit_forward_save(gm.model, zt, torch.tensor(t[part], dtype=torch.float32, device="cuda"),
                            gm.tensor(txt[part]), torch.empty_like(zt), saved=arena, ws=ws1)
        gm.vjp(arena, ws1, G, cot[part], grad=g_seq)
    torch.cuda.synchronize()
    r = rel_l2(g_seq.cpu().numpy(), g_joint.cpu().numpy())
    print(f"{wl.name}: sequential vs joint rel L2 {r:.2e}")
    assert r <= tol


@pytest.mark.parametrize("wl,G,tol", [(TINY, 4, 1e-4), (synth.small_variant(DITB, name="ditb_2blocks", depth=2), 4,
                                                        1e-2)], ids=["tiny_f32", "ditb_2blocks_bf16"])
def test_sequential_graph_variant_matches_oracle(wl, G, tol):
    """Algorithm 2 against the oracle's JAGG window gradient.  In the variant's order: the
    signals of steps 0..W-2 are aggregated (jagg_aggregate_span against the window's endpoint
    times) into both rows; endpoint 0 is forwarded into the one G-row arena and its VJP
    takes s_base; the last step's signal is added to s_corr; endpoint W-1 is forwarded into
    the same arena and its VJP takes s_corr.  The oracle: path.window_gradient (Eq.
    s_base_corr, one joint VJP over both endpoints) on the same signals."""
    W = wl.W
    params = synth.make_params(wl)
    rng = np.random.Generator(np.random.PCG64(31))
    z_win = synth.storage_round(rng.standard_normal((G, W, wl.in_channels, wl.latent_h, wl.latent_w)), wl.dtype)
    txt = synth.storage_round(rng.standard_normal((wl.txt_len, wl.txt_dim)), wl.dtype)
    t = synth.time_grid(8, 3.0)[1:W + 1].astype(np.float32).astype(np.float64)    # shifted: alpha != j/(W-1)
    s = rng.standard_normal((G, W) + z_win.shape[2:]).astype(np.float32).astype(np.float64)
    gm = GpuModel(jg, wl, params)
    dev = "cuda"
    f64 = dict(dtype=torch.float64, device=dev)
    st = torch.tensor(s.reshape(G, W, -1), dtype=torch.float32, device=dev)
    cot = torch.empty(2 * G, st.shape[-1], dtype=torch.float32, device=dev)
    arena = jg.alloc_bytes(gm.model.saved_bytes(G))
    ws = jg.alloc_bytes(gm.model.workspace_bytes(G))
    grad = torch.zeros(jg.param_count(gm.cfg), dtype=torch.float32, device=dev)
    txt_g = gm.tensor(np.broadcast_to(txt, (G,) + txt.shape))
    jg.jagg_aggregate_span(st, torch.tensor(t[:W - 1], **f64), t[0], t[W - 1], cot, steps=(0, W - 1))
    for e, j in enumerate((0, W - 1)):
        if e == 1:
            jg.jagg_aggregate_span(st, torch.tensor(t[W - 1:], **f64), t[0], t[W - 1], cot, accumulate=True,
                                   steps=(W - 1, 1))
        zt = gm.tensor(z_win[:, j])
        jg.dit_forward_save(gm.model, zt, torch.full((G,), float(t[j]), dtype=torch.float32, device=dev), txt_g,
                            torch.empty_like(zt), saved=arena, ws=ws)
        jg.dit_joint_vjp(gm.model, arena, G, cot[e * G:(e + 1) * G].reshape(G, *z_win.shape[2:]).contiguous(),
                         grad, ws)
    torch.cuda.synchronize()
    assert jg.device_status() == 0
    g_o = path.window_gradient(dit.Backbone(wl, params), z_win, t, txt, s, jagg=True)
    g_gpu = jg.unpack_grads(gm.cfg, grad)
    names = list(g_o)
    err, cs = rel_l2(flat(g_gpu, names), flat(g_o, names)), cosine(flat(g_gpu, names), flat(g_o, names))
    per = {k: rel_l2(g_gpu[k], g_o[k]) for k in names}
    worst = max(per, key=per.get)
    print(f"{wl.name}: sequential graph vs oracle rel L2 {err:.2e}, cos {cs:.7f}, worst {worst} {per[worst]:.2e}")
    assert err <= tol and cs >= 0.999
    bad = {k: e for k, e in per.items() if e > 5 * tol}
    assert not bad, f"tensors beyond {5 * tol:.0e}: {bad}"
