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


def _eps_case(G, W, D, e_dtype, clip_eps, seed):
    """An epsilon-prediction window on the variance-preserving cosine schedule: eps-hat from
    N(0,1), z_{j+1} = (DDIM mean of z_j, eps_j) + sigma_j xi, old log-probs as in _case."""
    rng = np.random.Generator(np.random.PCG64(seed))
    t = synth.time_grid(4 * W, 3.0)[W:2 * W + 1] * 0.9 + 0.05
    al, sg = synth.vp_schedule(t)
    sig = synth.sigma_schedule(t, 0.5)
    e = synth.storage_round(rng.standard_normal((G, W, D)), e_dtype)
    z = np.zeros((G, W + 1, D))
    z[:, 0] = rng.standard_normal((G, D))
    for j in range(W):
        mu = grpo.ddim_mean(z[:, j], e[:, j], al[j], al[j + 1], sg[j], sg[j + 1])
        z[:, j + 1] = mu + sig[j] * rng.standard_normal((G, D))
    z = z.astype(np.float32).astype(np.float64)
    lp = np.array([[grpo.step_logprob_eps(z[i, j + 1], z[i, j], e[i, j], al[j], al[j + 1], sg[j], sg[j + 1], sig[j])
                    for j in range(W)] for i in range(G)])
    inside = rng.uniform(-0.3 * clip_eps, 0.3 * clip_eps, (G, W))
    outside = rng.uniform(2 * clip_eps, 3 * clip_eps, (G, W)) * rng.choice([-1.0, 1.0], (G, W))
    delta = np.where(rng.uniform(size=(G, W)) < 0.5, inside, outside)
    rewards = synth.storage_round(rng.standard_normal(G), "f32")
    return e, z, t, al, sg, sig, lp + delta, rewards


def _run_eps(e, z, t, al, sg, sig, lpo, rewards, eps, scale, e_dtype, with_cot=True):
    dev = "cuda"
    G, W, D = e.shape
    f64 = dict(dtype=torch.float64, device=dev)
    out = dict(logp_new=torch.empty(G, W, **f64), ratio=torch.empty(G, W, **f64),
               clipped=torch.empty(G, W, dtype=torch.uint8, device=dev), adv_out=torch.empty(G, **f64))
    s = torch.full((G, W, D), float("nan"), device=dev)
    cot = torch.full((2 * G, D), float("nan"), device=dev) if with_cot else None
    ws = jg.alloc_bytes(jg.signals_workspace_bytes(G, W, D))
    te = torch.tensor(e, dtype=torch.bfloat16 if e_dtype == "bf16" else torch.float32, device=dev)
    jg.grpo_step_signals_eps(te, torch.tensor(z, dtype=torch.float32, device=dev), torch.tensor(t, **f64),
                             torch.tensor(al, **f64), torch.tensor(sg, **f64), torch.tensor(sig, **f64),
                             torch.tensor(lpo, **f64), torch.tensor(rewards, dtype=torch.float32, device=dev), eps,
                             5.0, 1e-8, scale, ws=ws, s_out=s, cot_out=cot, **out)
    torch.cuda.synchronize()
    return s, cot, out


@pytest.mark.parametrize("G,W,D,e_dtype,eps", [
    (4, 4, 64, "f32", 1e-4),
    (8, 4, 16384, "bf16", 0.1),
    (3, 2, 12345, "bf16", 0.1),       # ragged D, W = 2
    (5, 3, 8193, "f32", 0.05),        # D one past a CTA chunk
])
def test_eps_prediction_signals_match_oracle(G, W, D, e_dtype, eps):
    """grpo_step_signals_eps (the DDIM mean of Eq. logprob) against the oracle, element by
    element, with the same bars as the velocity path."""
    e, z, t, al, sg, sig, lpo, rewards = _eps_case(G, W, D, e_dtype, eps, seed=7 * G + D)
    scale = 1.0 / (G * 16)
    A = grpo.advantages(rewards)
    s_o, lp_o, ratio_o, clip_o = grpo.step_signals_eps(e, z, al, sg, sig, lpo, A, eps, scale)
    jg.device_status(clear=True)
    s, cot, out = _run_eps(e, z, t, al, sg, sig, lpo, rewards, eps, scale, e_dtype)
    assert jg.device_status() == 0
    lp_tol = 1e-6 * max(10.0, D / 50)
    assert np.max(np.abs(out["logp_new"].cpu().numpy() - lp_o)) < lp_tol
    np.testing.assert_allclose(out["ratio"].cpu().numpy(), ratio_o, rtol=2 * lp_tol)
    np.testing.assert_array_equal(out["clipped"].cpu().numpy(), clip_o)
    assert _rel(s.cpu().numpy(), s_o) < 1e-4
    assert _rel(cot.cpu().numpy(), grpo.aggregate(s_o, t[:W])) < 1e-4


def test_eps_prediction_rejects_a_nonpositive_alpha():
    """alpha_t <= 0 makes the DDIM mean undefined: the device status reports it."""
    e, z, t, al, sg, sig, lpo, rewards = _eps_case(2, 3, 100, "f32", 0.1, seed=5)
    al = al.copy()
    al[3] = 0.0
    jg.device_status(clear=True)
    _run_eps(e, z, t, al, sg, sig, lpo, rewards, 0.1, 0.1, "f32", with_cot=False)
    assert jg.device_status() & 2
    jg.device_status(clear=True)


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


@pytest.mark.parametrize("G,W,D", [(4, 4, 64), (8, 5, 3000), (3, 8, 1 << 16)])
def test_span_aggregation_and_ablation_match_oracle(G, W, D):
    """The sequential-graph split (steps 0..W-2, then the last step accumulated) and the
    endpoint-only ablation (span over {0, W-1}) against the oracle's definitions."""
    dev = "cuda"
    rng = np.random.Generator(np.random.PCG64(G * 100 + W))
    s = rng.standard_normal((G, W, D)).astype(np.float32)
    t = synth.time_grid(16, 3.0)[2:2 + W]
    f64 = dict(dtype=torch.float64, device=dev)
    st = torch.tensor(s, device=dev)
    cot = torch.full((2 * G, D), float("nan"), device=dev)
    jg.jagg_aggregate_span(st, torch.tensor(t[:-1], **f64), t[0], t[-1], cot, steps=(0, W - 1))
    jg.jagg_aggregate_span(st, torch.tensor(t[-1:], **f64), t[0], t[-1], cot, accumulate=True, steps=(W - 1, 1))
    ref = grpo.aggregate(s.astype(np.float64), t)
    torch.cuda.synchronize()
    assert np.abs(cot.cpu().numpy() - ref).max() <= 1e-5 * max(1.0, np.abs(ref).max())
    # ablation: step 0 and step W-1 read in place, each over its own span (bit-exact pair)
    ab = torch.empty(2 * G, D, device=dev)
    jg.jagg_aggregate_span(st, torch.tensor(t[:1], **f64), t[0], t[-1], ab, steps=(0, 1))
    jg.jagg_aggregate_span(st, torch.tensor(t[-1:], **f64), t[0], t[-1], ab, accumulate=True, steps=(W - 1, 1))
    torch.cuda.synchronize()
    np.testing.assert_array_equal(ab.cpu().numpy(), grpo.aggregate_ablate(s).astype(np.float32))
    # a contiguous [G, 2, D] pair over the span {t_0, t_{W-1}} gives the same rows
    ends = torch.stack([st[:, 0], st[:, -1]], 1).contiguous()
    ab2 = torch.empty(2 * G, D, device=dev)
    jg.jagg_aggregate_span(ends, torch.tensor([t[0], t[-1]], **f64), t[0], t[-1], ab2)
    torch.cuda.synchronize()
    assert torch.equal(ab, ab2)
    with pytest.raises(jg.JaggError):
        jg.jagg_aggregate_span(ends, torch.tensor([t[0], t[0]], **f64), t[0], t[0], ab)


# ------------------------------------------------------------------ rollout sampler step
from oracle import rollout as oracle_rollout  # noqa: E402


def _sched(eps_model, t):
    if not eps_model:
        return None
    al, sg = synth.vp_schedule(np.asarray(t))
    return al, sg


@pytest.mark.parametrize("G,T,D,y_dtype,eps_model", [
    (4, 3, 64, "f32", False),
    (8, 4, 16384, "bf16", False),      # DiT-B latent
    (3, 2, 12345, "bf16", True),       # ragged D, noise prediction
    (5, 3, 8193, "f32", True),         # D one past a CTA chunk
])
def test_rollout_step_matches_oracle(G, T, D, y_dtype, eps_model):
    """jagg_rollout_step against the oracle's sampler step, writing step j -> j+1 of a
    [G, T+1, D] trajectory buffer in place: the stored sample to float32 rounding of the
    f32 mean, the log-prob with the signals' bar."""
    dev = "cuda"
    rng = np.random.Generator(np.random.PCG64(G * 31 + D))
    t = synth.time_grid(4 * T, 3.0)[T:2 * T + 1] * 0.9 + 0.05
    sig = synth.sigma_schedule(t, 0.7)
    sch = _sched(eps_model, t)
    z = torch.zeros(G, T + 1, D, device=dev)
    z[:, 0] = torch.tensor(rng.standard_normal((G, D)), dtype=torch.float32, device=dev)
    logp = torch.full((G, T), float("nan"), dtype=torch.float64, device=dev)
    ws = jg.alloc_bytes(jg.rollout_workspace_bytes(G, D))
    jg.device_status(clear=True)
    for j in range(T):
        y = synth.storage_round(rng.standard_normal((G, D)), y_dtype)
        xi = rng.standard_normal((G, D)).astype(np.float32)
        sched_j = None if sch is None else (sch[0][j], sch[0][j + 1], sch[1][j], sch[1][j + 1])
        z_cur = z[:, j].cpu().numpy().astype(np.float64)
        yt = torch.tensor(y, dtype=torch.bfloat16 if y_dtype == "bf16" else torch.float32, device=dev)
        zm = torch.empty(G, D, dtype=torch.bfloat16, device=dev)
        jg.jagg_rollout_step(yt, z, j, torch.tensor(xi, device=dev), t[j], t[j + 1], sig[j], logp, ws, sched=sched_j,
                             z_model=zm)
        torch.cuda.synchronize()
        assert torch.equal(zm, z[:, j + 1].bfloat16())      # the next forward's input, RNE-rounded
        zn_o, lp_o = oracle_rollout.sampler_step(z_cur, y, xi, t[j], t[j + 1], sig[j], sched_j)
        zn = z[:, j + 1].cpu().numpy().astype(np.float64)
        assert np.max(np.abs(zn - zn_o)) <= 4e-7 * max(1.0, np.abs(zn_o).max())
        # the log-prob of the sample the GPU stored, by the oracle's Eq. logprob
        if sched_j is None:
            lp_ref = [grpo.step_logprob(zn[i], z_cur[i], y[i], t[j], t[j + 1], sig[j]) for i in range(G)]
        else:
            lp_ref = [grpo.step_logprob_eps(zn[i], z_cur[i], y[i], *sched_j, sig[j]) for i in range(G)]
        lp_tol = 1e-6 * max(10.0, D / 50)
        lp = logp[:, j].cpu().numpy()
        assert np.max(np.abs(lp - np.array(lp_ref))) < lp_tol
        # and the oracle's own sample scores alike (the two samples differ by f32 roundings)
        assert np.max(np.abs(lp - lp_o)) < lp_tol + 1e-3
    assert jg.device_status() == 0


@pytest.mark.parametrize("eps_model", [False, True])
def test_rollout_logprobs_are_reproduced_exactly_by_the_step_signals(eps_model):
    """theta = theta_old: scoring the stored rollout with the same model outputs gives the
    rollout's own log-probs bit for bit, so every ratio is exactly 1 and no step is clipped."""
    dev = "cuda"
    G, W, D = 6, 4, 20000
    rng = np.random.Generator(np.random.PCG64(11 + eps_model))
    t = synth.time_grid(4 * W, 3.0)[W:2 * W + 1] * 0.9 + 0.05
    sig = synth.sigma_schedule(t, 0.7)
    sch = _sched(eps_model, t)
    f64 = dict(dtype=torch.float64, device=dev)
    z = torch.zeros(G, W + 1, D, device=dev)
    z[:, 0] = torch.tensor(rng.standard_normal((G, D)), dtype=torch.float32, device=dev)
    y = torch.tensor(rng.standard_normal((G, W, D)), dtype=torch.bfloat16, device=dev)
    xi = torch.tensor(rng.standard_normal((G, W, D)), dtype=torch.float32, device=dev)
    logp = torch.empty(G, W, **f64)
    ws = jg.alloc_bytes(jg.rollout_workspace_bytes(G, D))
    for j in range(W):
        sched_j = None if sch is None else (sch[0][j], sch[0][j + 1], sch[1][j], sch[1][j + 1])
        jg.jagg_rollout_step(y[:, j].contiguous(), z, j, xi[:, j].contiguous(), t[j], t[j + 1], sig[j], logp, ws,
                             sched=sched_j)
    out = dict(logp_new=torch.empty(G, W, **f64), ratio=torch.empty(G, W, **f64),
               clipped=torch.empty(G, W, dtype=torch.uint8, device=dev), adv_out=torch.empty(G, **f64))
    sws = jg.alloc_bytes(jg.signals_workspace_bytes(G, W, D))
    rewards = torch.tensor(rng.standard_normal(G), dtype=torch.float32, device=dev)
    args = (torch.tensor(sig[:W], **f64), logp, rewards, 0.1, 5.0, 1e-8, 1.0)
    if eps_model:
        jg.grpo_step_signals_eps(y, z, torch.tensor(t, **f64), torch.tensor(sch[0], **f64),
                                 torch.tensor(sch[1], **f64), *args, ws=sws, **out)
    else:
        jg.grpo_step_signals(y, z, torch.tensor(t, **f64), *args, ws=sws, **out)
    torch.cuda.synchronize()
    assert jg.device_status() == 0
    assert torch.equal(out["logp_new"], logp)
    assert torch.all(out["ratio"] == 1.0)
    assert not out["clipped"].any()


def test_rollout_step_rejects_bad_arguments():
    dev = "cuda"
    z = torch.zeros(2, 3, 10, device=dev)
    y = torch.zeros(2, 10, device=dev)
    logp = torch.empty(2, 2, dtype=torch.float64, device=dev)
    ws = jg.alloc_bytes(jg.rollout_workspace_bytes(2, 10))
    with pytest.raises(jg.JaggError):
        jg.jagg_rollout_step(y, z, 0, y, 0.5, 0.4, 0.0, logp, ws)     # sigma must be positive
    with pytest.raises(jg.JaggError):
        jg.jagg_rollout_step(y, z, 0, y, 0.5, 0.4, 0.1, logp, jg.alloc_bytes(8))   # workspace too small


# ------------------------------------------------------------------ clip decisions at the boundary
def _dyadic_case(G, W, D, v_dtype, seed):
    """A window whose residuals r = z_{j+1} - z_j - v_j dt_j are computed exactly by both
    sides: a uniform grid (dt = -1/8), v multiples of 2^-4 in [-4, 4] (exact in bf16), noise
    multiples of 2^-8 in [-1/2, 1/2].  Every partial sum of r^2 is then exact in float32, so
    the library's log-prob equals the oracle's to the rounding of the f64 normaliser."""
    rng = np.random.Generator(np.random.PCG64(seed))
    q = lambda x, step, lim: np.clip(np.round(x / step) * step, -lim, lim)
    t = synth.time_grid(2 * W, 1.0)[:W + 1]
    sig = synth.sigma_schedule(t, 0.7)
    v = q(rng.standard_normal((G, W, D)), 2.0 ** -4, 4.0)
    z = np.zeros((G, W + 1, D))
    z[:, 0] = q(rng.standard_normal((G, D)), 2.0 ** -8, 4.0)
    for j in range(W):
        z[:, j + 1] = z[:, j] + v[:, j] * (t[j + 1] - t[j]) + q(sig[j] * rng.standard_normal((G, D)), 2.0 ** -8, 0.5)
    assert np.array_equal(z.astype(np.float32), z)
    lp = np.array([[grpo.step_logprob(z[i, j + 1], z[i, j], v[i, j], t[j], t[j + 1], sig[j]) for j in range(W)]
                   for i in range(G)])
    rewards = synth.storage_round(rng.standard_normal(G), "f32")
    return v, z, t, sig, lp, rewards, rng


def _signals_call(v, z, t, sig, lpo, rewards, eps, scale, v_dtype):
    dev = "cuda"
    G, W, D = v.shape
    f64 = dict(dtype=torch.float64, device=dev)
    out = dict(logp_new=torch.empty(G, W, **f64), ratio=torch.empty(G, W, **f64),
               clipped=torch.empty(G, W, dtype=torch.uint8, device=dev), adv_out=torch.empty(G, **f64))
    s = torch.full((G, W, D), float("nan"), device=dev)
    ws = jg.alloc_bytes(jg.signals_workspace_bytes(G, W, D))
    jg.grpo_step_signals(torch.tensor(v, dtype=torch.bfloat16 if v_dtype == "bf16" else torch.float32, device=dev),
                         torch.tensor(z, dtype=torch.float32, device=dev), torch.tensor(t, **f64),
                         torch.tensor(sig, **f64), torch.tensor(lpo, **f64),
                         torch.tensor(rewards, dtype=torch.float32, device=dev), eps, 5.0, 1e-8, scale, ws=ws,
                         s_out=s, **out)
    torch.cuda.synchronize()
    assert jg.device_status() == 0
    return s.cpu().numpy(), {k: x.cpu().numpy() for k, x in out.items()}


@pytest.mark.parametrize("D,v_dtype", [(4096, "f32"), (65536, "bf16")])
def test_clip_mask_near_the_boundary_matches_oracle(D, v_dtype):
    """log rho placed within (1e-6, 1e-3) of log(1 + eps) or log(1 - eps), on either side
    (log-uniform distances): the clip decisions agree with the oracle bit for bit."""
    G, W, eps = 8, 4, 0.1
    v, z, t, sig, lp, rewards, rng = _dyadic_case(G, W, D, v_dtype, seed=D + 1)
    bound = np.where(rng.uniform(size=(G, W)) < 0.5, np.log1p(eps), np.log1p(-eps))
    margin = 10.0 ** rng.uniform(-6, -3, (G, W)) * rng.choice([-1.0, 1.0], (G, W))
    lpo = lp - (bound + margin)
    scale = 1.0 / (G * 16)
    A = grpo.advantages(rewards)
    s_o, lp_o, ratio_o, clip_o = grpo.step_signals(v, z, t, sig, lpo, A, eps, scale)
    s, out = _signals_call(v, z, t, sig, lpo, rewards, eps, scale, v_dtype)
    assert np.max(np.abs(out["logp_new"] - lp_o)) <= 1e-9 * max(1.0, np.abs(lp_o).max())
    np.testing.assert_array_equal(out["clipped"], clip_o)
    assert 0 < clip_o.sum() < G * W            # both outcomes occur
    assert _rel(s, s_o) < 1e-6


def test_clip_tie_counts_as_unclipped_on_the_device():
    """rho = 1 + eps with A > 0 (and rho = 1 - eps with A < 0) exactly, eps formed in float64
    from the library's own ratio: the step keeps its gradient, bit-equal to the one it gets
    under a wide clip range; one ulp of rho past the tie it is clipped."""
    G, W, D = 6, 4, 4096
    v, z, t, sig, lp, rewards, rng = _dyadic_case(G, W, D, "f32", seed=77)
    lpo = lp - rng.uniform(-0.08, 0.08, (G, W))
    scale = 1.0 / (G * 16)
    A = grpo.advantages(rewards)
    s_wide, out = _signals_call(v, z, t, sig, lpo, rewards, 0.5, scale, "f32")
    assert not out["clipped"].any()
    rho = out["ratio"]
    for sign in (1.0, -1.0):
        cand = [(i, j) for i in range(G) for j in range(W) if A[i] * sign > 0 and (rho[i, j] - 1.0) * sign > 0]
        i, j = cand[0]
        eps_tie = (rho[i, j] - 1.0) * sign                   # exact: 1 +- eps_tie == rho[i, j]
        assert 1.0 + sign * eps_tie == rho[i, j]
        s_tie, o_tie = _signals_call(v, z, t, sig, lpo, rewards, eps_tie, scale, "f32")
        assert o_tie["clipped"][i, j] == 0 and o_tie["ratio"][i, j] == rho[i, j]
        np.testing.assert_array_equal(s_tie[i, j], s_wide[i, j])
        assert np.abs(s_tie[i, j]).sum() > 0
        _, o_past = _signals_call(v, z, t, sig, lpo, rewards, eps_tie - np.spacing(rho[i, j]), scale, "f32")
        assert o_past["clipped"][i, j] == 1
