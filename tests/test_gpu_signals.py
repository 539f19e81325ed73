"""GPU parity of the GRPO step signals, the JAGG aggregation and the gradient reductions
with the float64 oracle on the same seeded inputs (Phase 2 and Phase 3 of Algorithm 1)."""
import numpy as np
import pytest
import torch

import synth
from oracle import grpo

pytestmark = pytest.mark.gpu

jg = pytest.importorskip("paper_2607_17572_gb300")


def _rel(a, b):
    a = np.asarray(a, np.float64).ravel()
    b = np.asarray(b, np.float64).ravel()
    nb = np.linalg.norm(b)
    return np.linalg.norm(a - b) / (nb if nb > 0 else 1.0)


def _case(G, W, D, v_dtype, clip_eps, shift, seed):
    """A window with v-hat drawn from N(0,1), a trajectory z_{j+1} = z_j + v dt + sigma xi,
    and old log-probs set a margin away from the clip boundaries."""
    rng = np.random.Generator(np.random.PCG64(seed))
    t = synth.time_grid(4 * W, shift)[W:2 * W + 1]
    sig = synth.sigma_schedule(t, 0.7)
    v = synth.storage_round(rng.standard_normal((G, W, D)), v_dtype)
    z = np.zeros((G, W + 1, D))
    z[:, 0] = rng.standard_normal((G, D))
    for j in range(W):
        z[:, j + 1] = z[:, j] + v[:, j] * (t[j + 1] - t[j]) + sig[j] * rng.standard_normal((G, D))
    z = z.astype(np.float32).astype(np.float64)
    lp = np.array([[grpo.step_logprob(z[i, j + 1], z[i, j], v[i, j], t[j], t[j + 1], sig[j]) for j in range(W)]
                   for i in range(G)])
    e = clip_eps
    inside = rng.uniform(-0.3 * e, 0.3 * e, (G, W))
    outside = rng.uniform(2 * e, 3 * e, (G, W)) * rng.choice([-1.0, 1.0], (G, W))
    delta = np.where(rng.uniform(size=(G, W)) < 0.5, inside, outside)
    rewards = synth.storage_round(rng.standard_normal(G), "f32")
    return v, z, t, sig, lp + delta, rewards


@pytest.mark.parametrize("G,W,D,v_dtype,eps,shift", [
    (4, 4, 64, "f32", 1e-4, 1.0),            # tiny configuration
    (8, 4, 16384, "bf16", 0.1, 1.0),         # DiT-B latent
    (8, 4, 65536, "bf16", 0.1, 3.0),         # Flux-width 512^2 latent, shifted grid
    (3, 2, 12345, "bf16", 0.1, 3.0),         # ragged D, W = 2
    (1, 8, 1000, "f32", 0.2, 1.0),           # single sample: std = 0, A = 0
    (5, 3, 8193, "f32", 0.05, 3.0),          # D one past a CTA chunk
])
def test_step_signals_and_aggregation_match_oracle(G, W, D, v_dtype, eps, shift):
    v, z, t, sig, lpo, rewards = _case(G, W, D, v_dtype, eps, shift, seed=G * 1000 + D)
    scale = 1.0 / (G * 16)
    A = grpo.advantages(rewards)
    s_o, lp_o, ratio_o, clip_o = grpo.step_signals(v, z, t, sig, lpo, A, eps, scale)
    dev = "cuda"
    f64 = dict(dtype=torch.float64, device=dev)
    tv = torch.tensor(v, dtype=torch.bfloat16 if v_dtype == "bf16" else torch.float32, device=dev)
    out = dict(logp_new=torch.empty(G, W, **f64), ratio=torch.empty(G, W, **f64),
               clipped=torch.empty(G, W, dtype=torch.uint8, device=dev), adv_out=torch.empty(G, **f64))
    s = torch.full((G, W, D), float("nan"), device=dev)
    cot = torch.full((2 * G, D), float("nan"), device=dev) if W >= 2 else None
    ws = jg.alloc_bytes(jg.signals_workspace_bytes(G, W, D))
    jg.grpo_step_signals(tv, torch.tensor(z, dtype=torch.float32, device=dev), torch.tensor(t, **f64),
                         torch.tensor(sig, **f64), torch.tensor(lpo, **f64),
                         torch.tensor(rewards, dtype=torch.float32, device=dev), eps, 5.0, 1e-8, scale, ws=ws,
                         s_out=s, cot_out=cot, **out)
    torch.cuda.synchronize()
    assert jg.device_status() == 0
    np.testing.assert_allclose(out["adv_out"].cpu().numpy(), A, rtol=1e-12, atol=1e-12)
    # log-probs: f32 residuals, f64 sums -> absolute error far below the clip margins
    lp_tol = 1e-6 * max(10.0, D / 50)
    assert np.max(np.abs(out["logp_new"].cpu().numpy() - lp_o)) < lp_tol
    np.testing.assert_allclose(out["ratio"].cpu().numpy(), ratio_o, rtol=2 * lp_tol)
    np.testing.assert_array_equal(out["clipped"].cpu().numpy(), clip_o)
    # s = c_ij r_ij: r is formed in f32 (about 1e-7 relative per element), so log-prob carries
    # an absolute error near 1e-7 sqrt(D) and rho the same relative error; the f32 bar 1e-4
    # covers it with a wide margin at every D here.
    assert _rel(s.cpu().numpy(), s_o) < 1e-4
    if cot is not None:
        assert _rel(cot.cpu().numpy(), grpo.aggregate(s_o, t[:W])) < 1e-4
        # the standalone aggregation on the GPU's own signals
        cot2 = torch.empty_like(cot)
        jg.jagg_aggregate(s, torch.tensor(t[:W], **f64), cot2)
        torch.cuda.synchronize()
        assert _rel(cot2.cpu().numpy(), grpo.aggregate(s.cpu().numpy(), t[:W])) < 1e-6


def test_aggregate_rejects_degenerate_window():
    dev = "cuda"
    s = torch.ones(2, 3, 10, device=dev)
    cot = torch.empty(4, 10, device=dev)
    jg.device_status(clear=True)
    jg.jagg_aggregate(s, torch.tensor([0.5, 0.4, 0.5], dtype=torch.float64, device=dev), cot)
    torch.cuda.synchronize()
    assert jg.device_status() & 2
    assert torch.all(cot == 0)
    with pytest.raises(jg.JaggError):
        jg.jagg_aggregate(s[:, :1].contiguous(), torch.tensor([0.5], dtype=torch.float64, device=dev), cot)


@pytest.mark.parametrize("P", [1, 7, 1000, 4096 * 1000 + 3, 130_000_000])
def test_grad_reduce_matches_numpy(P):
    dev = "cuda"
    g = torch.Generator(device=dev).manual_seed(P % 1000)
    a = torch.randn(P, device=dev, generator=g)
    b = 0.5 * a + torch.randn(P, device=dev, generator=g)
    acc = torch.randn(P, device=dev, generator=g)
    acc0 = acc.clone()
    out3 = torch.empty(3, dtype=torch.float64, device=dev)
    ws = jg.alloc_bytes(jg.grad_reduce_workspace_bytes(P))
    jg.grad_reduce(a, b, alpha=0.25, acc=acc, out3=out3, ws=ws)
    torch.cuda.synchronize()
    ad, bd = a.double(), b.double()
    ref = torch.stack([ad @ bd, ad @ ad, bd @ bd]).cpu().numpy()
    np.testing.assert_allclose(out3.cpu().numpy(), ref, rtol=1e-6)
    assert torch.allclose(acc, acc0 + 0.25 * a, rtol=0, atol=1e-6)
    ab, aa, bb = out3.cpu().numpy()
    ro = grpo.grad_stats(a.cpu().numpy(), b.cpu().numpy())
    assert abs(ab / np.sqrt(aa * bb) - ro[3]) < 1e-6
