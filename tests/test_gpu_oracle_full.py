"""Oracle parity of the bf16 path at the full sizes of the Flux-width (512^2 and 1024^2) and
Qwen-width workloads: full width, depth and token count, the launch configurations the
bench times.

One JAGG window of one sample, in the staged protocol of the clip discontinuity: the
library's sampler rolls the group out over the first window's W steps (no-save forwards
and the fused sampler step); the library's step signals run on its own velocities; one
sample's two endpoint rows (z_0 and z_{W-1}) go through dit_forward_save and dit_joint_vjp
with that sample's two cotangent rows.  The float64 oracle takes the same per-step
signals and computes the window's JAGG gradient (Eq. s_base_corr aggregation, forward,
reverse mode; Algorithm 1, Phase 4) on the same bf16 weights and inputs.  Compared: the
step signals of the whole group (clip mask, log-probs, s), the forward, the cotangent rows,
the whole parameter gradient (relative L2, cosine) and every parameter tensor on its own.

The weights are drawn on the device by synth.device_params (seconds at 2.5 B parameters)
and handed to both sides."""
import time

import numpy as np
import pytest
import torch

import synth
from gpu_cases import rel_l2
from oracle import dit, grpo, path

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

jg = pytest.importorskip("paper_2607_17572_gb300")

# Gradient bars of the bf16 path (relative L2 and cosine over the whole gradient), and a
# bound for every parameter tensor on its own, so that a wrong gradient of a small tensor
# (a bias, a norm scale) cannot hide under the norm of the large ones.
TOL_TOTAL, TOL_COS, TOL_TENSOR = 1e-2, 0.999, 5e-2

CASES = ["mmdit_flux512_bf16", "mmdit_flux1024_bf16", "mmdit_qwen_sweep_bf16"]


def rollout_window(wl, model, draws, t, sig, dev):
    """The group's first window on the device: per step the no-save forward of the G
    current samples and the fused sampler step.  Returns z [G, W+1, D] f32, v [G, W, D]
    bf16 (the velocities the signals score) and the rollout's log-probs [G, W] f64."""
    G, W, D = wl.G, wl.W, wl.D
    shape = (wl.in_channels, wl.latent_h, wl.latent_w)
    z = torch.zeros(G, W + 1, D, dtype=torch.float32, device=dev)
    z[:, 0] = torch.tensor(draws.z0.reshape(-1), dtype=torch.float32, device=dev)
    zin = z[:, 0].reshape(G, *shape).to(torch.bfloat16).contiguous()
    v = torch.empty(G, W, D, dtype=torch.bfloat16, device=dev)
    lp = torch.empty(G, W, dtype=torch.float64, device=dev)
    txt = torch.tensor(draws.txt, dtype=torch.bfloat16, device=dev).unsqueeze(0).expand(G, -1, -1).contiguous()
    ws = jg.alloc_bytes(model.workspace_bytes(G))
    rws = jg.alloc_bytes(jg.rollout_workspace_bytes(G, D))
    for j in range(W):
        vj = torch.empty(G, *shape, dtype=torch.bfloat16, device=dev)
        tj = torch.full((G,), float(t[j]), dtype=torch.float32, device=dev)
        jg.dit_forward_save(model, zin, tj, txt, vj, ws=ws)
        v[:, j] = vj.reshape(G, D)
        xi = torch.tensor(draws.xi[:, j].reshape(G, D), dtype=torch.float32, device=dev)
        jg.jagg_rollout_step(vj, z, j, xi, float(t[j]), float(t[j + 1]), float(sig[j]), lp, rws, z_model=zin)
    torch.cuda.synchronize()
    return z, v, lp


def sums(a, b):
    """(sum (a-b)^2, sum b^2, sum a b, sum a^2) in float64."""
    a = np.asarray(a, np.float64).ravel()
    b = np.asarray(b, np.float64).ravel()
    d = a - b
    return np.array([d @ d, b @ b, a @ b, a @ a])


@pytest.mark.parametrize("name", CASES)
def test_full_size_jagg_window_matches_oracle(name):
    wl = synth.WORKLOADS[name]
    dev = torch.device("cuda")
    G, W, D = wl.G, wl.W, wl.D
    shape = (wl.in_channels, wl.latent_h, wl.latent_w)
    cfg = jg.Config.from_workload(wl)
    pd = synth.device_params(wl, synth.WEIGHT_SEED, dev)
    weights = jg.pack_params(cfg, pd, dev)
    model = jg.Model(cfg, weights)
    draws = synth.draw_group(wl)
    t = synth.time_grid(wl.T, wl.shift)
    sig = synth.sigma_schedule(t, wl.eta)
    t32 = t.astype(np.float32).astype(np.float64)

    # ---- Phases 1-3 on the device: rollout of the window, step signals, aggregation
    z, v, lp = rollout_window(wl, model, draws, t, sig, dev)
    logp_old = lp + torch.tensor(draws.delta[:, :W], dtype=torch.float64, device=dev)
    rewards = torch.tensor(draws.rewards, dtype=torch.float32, device=dev)
    f64 = dict(dtype=torch.float64, device=dev)
    out = dict(logp_new=torch.empty(G, W, **f64), ratio=torch.empty(G, W, **f64),
               clipped=torch.empty(G, W, dtype=torch.uint8, device=dev), adv_out=torch.empty(G, **f64))
    sws = jg.alloc_bytes(jg.signals_workspace_bytes(G, W, D))
    s = torch.empty(G, W, D, dtype=torch.float32, device=dev)
    cot = torch.empty(2 * G, D, dtype=torch.float32, device=dev)
    scale = 1.0 / (G * wl.T)
    args = (v.view(G, W, D), z, torch.tensor(t[:W + 1], **f64), torch.tensor(sig[:W], **f64), logp_old, rewards,
            wl.clip_eps, wl.adv_clip, wl.adv_eps, scale)
    jg.grpo_step_signals(*args, ws=sws, s_out=s, **out)
    jg.grpo_step_signals(*args, ws=sws, cot_out=cot, **out)

    # ---- Phase 4 on the device for sample 0: endpoint rows with saves, the joint VJP
    zr = torch.stack([z[0, 0], z[0, W - 1]]).reshape(2, *shape).to(torch.bfloat16).contiguous()
    tr = torch.tensor([t[0], t[W - 1]], dtype=torch.float32, device=dev)
    txt2 = torch.tensor(draws.txt, dtype=torch.bfloat16, device=dev).unsqueeze(0).expand(2, -1, -1).contiguous()
    saved = jg.alloc_bytes(model.saved_bytes(2))
    ws = jg.alloc_bytes(model.workspace_bytes(2))
    v_end = torch.empty_like(zr)
    jg.dit_forward_save(model, zr, tr, txt2, v_end, saved=saved, ws=ws)
    grad = torch.zeros(jg.param_count(cfg), dtype=torch.float32, device=dev)
    jg.dit_joint_vjp(model, saved, 2, cot[[0, G]].contiguous(), grad, ws)
    torch.cuda.synchronize()
    assert jg.device_status() == 0
    z_h, v_h, s_h = z.double().cpu().numpy(), v.double().cpu().numpy(), s.double().cpu().numpy()
    cot_h, zr_h, v_end_h = cot.double().cpu().numpy(), zr.double().cpu().numpy(), v_end.double().cpu().numpy()
    clipped, logp_new = out["clipped"].cpu().numpy(), out["logp_new"].cpu().numpy()
    g_gpu = jg.unpack_grads(cfg, grad)
    params = {k: x.double().cpu().numpy() for k, x in pd.items()}
    del saved, ws, grad, weights, model, pd, z, v, s, cot
    torch.cuda.empty_cache()

    # ---- the oracle on the same inputs
    t0 = time.time()
    A = grpo.advantages(draws.rewards.astype(np.float32).astype(np.float64), wl.adv_eps, wl.adv_clip)
    s_o, lp_o, _, clip_o = grpo.step_signals(v_h, z_h, t[:W + 1], sig[:W], logp_old.cpu().numpy(), A, wl.clip_eps,
                                             scale)
    assert np.array_equal(clipped, clip_o), "clip decisions differ from the oracle"
    assert np.max(np.abs(logp_new - lp_o)) <= 1e-6 * max(10.0, D / 50.0)
    e_s = rel_l2(s_h, s_o)
    assert e_s <= 1e-4, f"step signals rel L2 {e_s:.2e}"
    cot_o = grpo.aggregate(s_h[:1], t[:W])                    # sample 0: [s_base; s_corr]
    e_c = rel_l2(cot_h[[0, G]], cot_o)
    assert e_c <= 1e-5, f"cotangent rows rel L2 {e_c:.2e}"
    # the window's JAGG gradient of sample 0 (path.window_gradient, with the forward's v kept)
    model_o = dit.Backbone(wl, params)
    z_win = np.stack([zr_h[0]] + [zr_h[0]] * (W - 2) + [zr_h[1]])[None]   # only the endpoints enter
    z_rows, t_rows = path.window_rows(z_win, t32[:W], jagg=True)
    cot_rows = path.window_cotangent(s_h[:1].reshape((1, W) + shape), t32[:W], jagg=True)
    v_o, cache = model_o.forward(z_rows, t_rows, np.broadcast_to(draws.txt, (2,) + draws.txt.shape))
    g_o = model_o.vjp(cache, cot_rows)
    del cache
    e_v = rel_l2(v_end_h, v_o)
    t_oracle = time.time() - t0

    tot = np.zeros(4)
    per = {}
    for k in g_o:
        q = sums(g_gpu[k], g_o[k])
        tot += q
        per[k] = np.sqrt(q[0] / q[1]) if q[1] > 0 else np.sqrt(q[0])
    err, cs = np.sqrt(tot[0] / tot[1]), tot[2] / np.sqrt(tot[1] * tot[3])
    worst = sorted(per, key=per.get, reverse=True)[:4]
    print(f"{name}: oracle {t_oracle:.0f} s; signals rel L2 {e_s:.2e}; forward {e_v:.2e}; gradient rel L2 "
          f"{err:.2e}, cos {cs:.6f}; worst tensors " + ", ".join(f"{k} {per[k]:.2e}" for k in worst))
    assert e_v <= 2e-2, f"forward rel L2 {e_v:.2e}"
    assert err <= TOL_TOTAL and cs >= TOL_COS, f"gradient rel L2 {err:.2e}, cos {cs:.6f}"
    bad = {k: e for k, e in per.items() if e > TOL_TENSOR}
    assert not bad, f"tensors beyond {TOL_TENSOR}: {bad}"
