"""Pins of the oracle's GRPO signals, aggregation, routing and reductions: scipy's Gaussian
log-density, numpy's std, central finite differences of Eq. grpo_loss, closed forms of
Eq. alpha / Eq. s_base_corr, and the routing values printed in the paper."""
import json
import math
import os

import numpy as np
import pytest
from scipy import stats

import synth
from oracle import grpo

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_logprob_is_the_isotropic_gaussian_density():
    rng = np.random.Generator(np.random.PCG64(0))
    D = 37
    z, zn, v = rng.standard_normal((3, D))
    t0, t1, sig = 0.8, 0.7375, 0.31
    mu = z + v * (t1 - t0)
    ref = stats.norm.logpdf(zn, loc=mu, scale=sig).sum()
    assert grpo.step_logprob(zn, z, v, t0, t1, sig) == pytest.approx(ref, rel=1e-13)


def test_advantages_match_numpy_and_clamp_bound():
    r = np.array([0.3, -1.2, 2.5, 0.0, 0.7])
    A = grpo.advantages(r)
    np.testing.assert_allclose(A, (r - r.mean()) / (np.std(r, ddof=1) + 1e-8), rtol=1e-14)
    # unbiased std bounds |A| by (G-1)/sqrt(G); with one outlier it is attained
    G = 8
    r = np.zeros(G); r[0] = 1.0
    assert abs(grpo.advantages(r)[0]) == pytest.approx((G - 1) / math.sqrt(G), rel=1e-7)
    assert np.all(grpo.advantages(np.array([1.0, 100.0, 2.0]), adv_clip=0.5) <= 0.5)
    np.testing.assert_array_equal(grpo.advantages(np.full(4, 3.0)), 0.0)


def _signals_case(seed, D=6, W=3, G=3, rho_shift=None, eps=0.1):
    rng = np.random.Generator(np.random.PCG64(seed))
    t = synth.time_grid(W, shift=3.0)
    sig = synth.sigma_schedule(t, 0.7)
    z = rng.standard_normal((G, W + 1, D))
    v = rng.standard_normal((G, W, D))
    lp = np.array([[grpo.step_logprob(z[i, j + 1], z[i, j], v[i, j], t[j], t[j + 1], sig[j])
                    for j in range(W)] for i in range(G)])
    shift = rng.uniform(-3 * eps, 3 * eps, size=(G, W)) if rho_shift is None else rho_shift
    A = np.array([1.3, -0.7, 0.4])[:G]
    return v, z, t, sig, lp + shift, A


@pytest.mark.parametrize("seed", [1, 2, 3])
def test_signals_are_the_gradient_of_the_window_loss(seed):
    """s_ij equals the central difference of scale * sum_j L_ij (Eq. grpo_loss) in v_ij."""
    eps, scale = 0.1, 0.37
    v, z, t, sig, lpo, A = _signals_case(seed, eps=eps)
    s, _, ratio, clipped = grpo.step_signals(v, z, t, sig, lpo, A, eps, scale)
    h = 1e-6
    G, W, D = v.shape
    for i in range(G):
        for j in range(W):
            if abs(abs(ratio[i, j] - 1.0) - eps) < 1e-4:
                continue   # at the kink the loss is not differentiable
            for k in range(D):
                vp = v[i].copy(); vp[j, k] += h
                vm = v[i].copy(); vm[j, k] -= h
                fd = (grpo.window_loss(vp, z[i], t, sig, lpo[i], A[i], eps, scale)
                      - grpo.window_loss(vm, z[i], t, sig, lpo[i], A[i], eps, scale)) / (2 * h)
                assert fd == pytest.approx(s[i, j, k], rel=1e-6, abs=1e-9)
    assert clipped.any() and not clipped.all()


def test_clip_follows_the_max_of_the_surrogate():
    """Zero gradient exactly when the clipped branch is strictly larger: (A>0, rho>1+eps)
    or (A<0, rho<1-eps); the other two out-of-range cases keep their gradient."""
    eps = 0.1
    W, G = 1, 2
    v, z, t, sig, lp, _ = _signals_case(4, W=W, G=G, rho_shift=np.zeros((G, W)), eps=eps)
    for A, log_rho, expect_clipped in [(1.0, 0.2, 1), (1.0, -0.2, 0), (-1.0, -0.2, 1),
                                        (-1.0, 0.2, 0), (1.0, 0.05, 0), (-1.0, -0.05, 0)]:
        lpo = lp - log_rho
        s, _, ratio, clipped = grpo.step_signals(v, z, t, sig, lpo, np.array([A, A]), eps, 1.0)
        np.testing.assert_allclose(ratio, math.exp(log_rho), rtol=1e-12)
        assert clipped[0, 0] == expect_clipped, (A, log_rho)
        assert (np.abs(s[0]).sum() == 0) == bool(expect_clipped)


def test_zero_advantage_and_unit_ratio():
    v, z, t, sig, lp, _ = _signals_case(5, rho_shift=np.zeros((3, 3)))
    s, _, ratio, clipped = grpo.step_signals(v, z, t, sig, lp, np.zeros(3), 0.1, 1.0)
    np.testing.assert_array_equal(s, 0.0)
    np.testing.assert_allclose(ratio, 1.0, rtol=1e-12)
    assert not clipped.any()


def test_alpha_closed_forms():
    t = synth.time_grid(16, 1.0)[4:8]
    np.testing.assert_allclose(grpo.alpha_weights(t), np.arange(4) / 3, atol=1e-15)
    ts = synth.time_grid(16, 3.0)[4:8]
    al = grpo.alpha_weights(ts)
    assert al[0] == 0.0 and al[-1] == 1.0
    assert np.all(np.diff(al) > 0)
    # shifted grid: alpha is the affine coordinate of t, not j/(W-1)
    assert abs(al[1] - 1 / 3) > 1e-3
    np.testing.assert_allclose(ts[0] + al * (ts[-1] - ts[0]), ts, atol=1e-15)


def test_aggregation_partition_of_unity_and_endpoints():
    rng = np.random.Generator(np.random.PCG64(8))
    s = rng.standard_normal((3, 4, 10))
    t = synth.time_grid(16, 3.0)[8:12]
    cot = grpo.aggregate(s, t)
    np.testing.assert_allclose(cot[:3] + cot[3:], s.sum(1), atol=1e-14)
    al = grpo.alpha_weights(t)
    np.testing.assert_allclose(cot[3:], np.einsum("j,gjd->gd", al, s), atol=1e-14)
    # s_0 only in the base row, s_{W-1} only in the correction row
    e = np.zeros_like(s); e[:, 0] = s[:, 0]
    np.testing.assert_array_equal(grpo.aggregate(e, t)[3:], 0.0)
    e = np.zeros_like(s); e[:, 3] = s[:, 3]
    np.testing.assert_array_equal(grpo.aggregate(e, t)[:3], 0.0)
    # W = 2: the cotangents are s_0 and s_1 themselves (JAGG is exact)
    np.testing.assert_array_equal(grpo.aggregate(s[:, :2], t[:2]), np.concatenate([s[:, 0], s[:, 1]]))


def test_routing_reproduces_the_papers_table():
    with open(os.path.join(GOLDEN, "routing_table.json")) as f:
        g = json.load(f)
    for model, row in g["calibration"].items():
        route, frac = grpo.route_calibrate(row["cos"], g["tau"])
        assert route.tolist() == row["route"], model
        assert frac == pytest.approx(row["derived_frac"])
    for case in g["schedule"]:
        assert grpo.route_schedule(case["n_windows"], case["jagg_frac"]).tolist() == case["route"]


def test_grad_stats_against_numpy():
    rng = np.random.Generator(np.random.PCG64(2))
    a, b = rng.standard_normal((2, 1000))
    ab, aa, bb, cos, rho = grpo.grad_stats(a, b)
    assert ab == pytest.approx(np.dot(a, b)) and aa == pytest.approx(np.dot(a, a))
    assert cos == pytest.approx(np.dot(a, b) / np.linalg.norm(a) / np.linalg.norm(b))
    assert rho == pytest.approx(np.linalg.norm(a) / np.linalg.norm(b))
    assert grpo.grad_stats(a, 2 * a)[3] == pytest.approx(1.0)


def test_span_aggregation_reassembles_the_window():
    """Spans of a window's steps, each with alpha against the window's endpoint times, add up
    to the whole-window aggregation; the sequential-graph split (steps 0..W-2 before the
    last step is known, then the last step alone) in particular."""
    rng = np.random.Generator(np.random.PCG64(81))
    G, W, D = 3, 5, 7
    s = rng.standard_normal((G, W, D))
    t = synth.time_grid(20, 3.0)[6:6 + W]
    full = grpo.aggregate(s, t)
    np.testing.assert_allclose(grpo.aggregate_span(s, t, t[0], t[-1]), full, atol=1e-14)
    first = grpo.aggregate_span(s[:, :-1], t[:-1], t[0], t[-1])
    last = grpo.aggregate_span(s[:, -1:], t[-1:], t[0], t[-1])
    np.testing.assert_allclose(first + last, full, atol=1e-14)
    # the last step adds only to the correction rows, the first only to the base rows
    np.testing.assert_array_equal(last[:G], 0.0)
    np.testing.assert_array_equal(grpo.aggregate_span(s[:, :1], t[:1], t[0], t[-1])[G:], 0.0)
    # any partition of the steps works
    parts = [grpo.aggregate_span(s[:, a:b], t[a:b], t[0], t[-1]) for a, b in ((0, 2), (2, 3), (3, 5))]
    np.testing.assert_allclose(sum(parts), full, atol=1e-14)


def test_ablation_keeps_the_endpoint_signals():
    """The endpoint-only ablation: s_0 and s_{W-1} unweighted; it coincides with JAGG exactly
    when the window has no middle steps (W = 2), and equals the span aggregation over the
    two endpoint steps."""
    rng = np.random.Generator(np.random.PCG64(82))
    G, W, D = 2, 4, 6
    s = rng.standard_normal((G, W, D))
    t = synth.time_grid(16, 3.0)[:W]
    ab = grpo.aggregate_ablate(s)
    np.testing.assert_array_equal(ab[:G], s[:, 0])
    np.testing.assert_array_equal(ab[G:], s[:, -1])
    np.testing.assert_array_equal(grpo.aggregate_ablate(s[:, :2]), grpo.aggregate(s[:, :2], t[:2]))
    ends = np.stack([s[:, 0], s[:, -1]], axis=1)
    np.testing.assert_allclose(grpo.aggregate_span(ends, [t[0], t[-1]], t[0], t[-1]), ab, atol=1e-15)
    # with middle steps the two differ (the ablation discards s_1 .. s_{W-2})
    assert np.abs(ab - grpo.aggregate(s, t)).max() > 1e-3


# ------------------------------------------------------------------ epsilon-prediction mean
def _eps_case(seed, G=3, W=3, D=6):
    rng = np.random.Generator(np.random.PCG64(seed))
    t = synth.time_grid(W, shift=3.0) * 0.9 + 0.05     # keep alpha_t, sigma_t away from 0
    al, sg = synth.vp_schedule(t)
    sig = synth.sigma_schedule(t, 0.7)
    z = rng.standard_normal((G, W + 1, D))
    e = rng.standard_normal((G, W, D))
    return t, al, sg, sig, z, e


def test_ddim_mean_on_the_flow_schedule_is_the_euler_step():
    """With alpha_t = 1 - t, sigma_t = t (the rectified-flow interpolation) the epsilon
    model eps_hat is the velocity model v_hat = (eps_hat - z) / (1 - t): the DDIM mean then
    equals the Euler step z + v_hat (t_{j+1} - t_j), and the step log-probs agree."""
    rng = np.random.Generator(np.random.PCG64(90))
    D = 23
    z, zn, e = rng.standard_normal((3, D))
    t0, t1, sig = 0.8, 0.7375, 0.31
    v = (e - z) / (1.0 - t0)
    np.testing.assert_allclose(grpo.ddim_mean(z, e, 1 - t0, 1 - t1, t0, t1), z + v * (t1 - t0), rtol=1e-12,
                               atol=1e-14)
    assert grpo.step_logprob_eps(zn, z, e, 1 - t0, 1 - t1, t0, t1, sig) == pytest.approx(
        grpo.step_logprob(zn, z, v, t0, t1, sig), rel=1e-13)


def test_eps_signals_follow_the_chain_rule_through_the_flow_signals():
    """On the rectified-flow schedule d v_hat / d eps_hat = 1 / (1 - t_j), so the epsilon
    signals are the (independently pinned) velocity signals divided by 1 - t_j, with the
    same log-probs, ratios and clip decisions."""
    rng = np.random.Generator(np.random.PCG64(91))
    G, W, D = 3, 4, 9
    t = synth.time_grid(W, shift=3.0) * 0.9 + 0.05
    sig = synth.sigma_schedule(t, 0.7)
    z = rng.standard_normal((G, W + 1, D))
    e = rng.standard_normal((G, W, D))
    v = (e - z[:, :W]) / (1.0 - t[:W])[None, :, None]
    lp = np.array([[grpo.step_logprob(z[i, j + 1], z[i, j], v[i, j], t[j], t[j + 1], sig[j]) for j in range(W)]
                   for i in range(G)])
    lpo = lp + rng.uniform(-0.3, 0.3, size=(G, W))
    A = np.array([1.3, -0.7, 0.4])
    sv, lv, rv, cv = grpo.step_signals(v, z, t, sig, lpo, A, 0.1, 0.37)
    se, le, re_, ce = grpo.step_signals_eps(e, z, 1.0 - t, t, sig, lpo, A, 0.1, 0.37)
    np.testing.assert_allclose(le, lv, rtol=1e-12)
    np.testing.assert_allclose(re_, rv, rtol=1e-10)
    np.testing.assert_array_equal(ce, cv)
    np.testing.assert_allclose(se, sv / (1.0 - t[:W])[None, :, None], rtol=1e-9, atol=1e-15)
    assert ce.any() and not ce.all()


def test_ddim_mean_recovers_the_noised_sample():
    """For z_j = alpha_j x + sigma_j eps and the true noise eps_hat = eps, the DDIM mean is the
    same sample noised to the next time: alpha_{j+1} x + sigma_{j+1} eps (variance-preserving
    and variance-exploding schedules)."""
    rng = np.random.Generator(np.random.PCG64(92))
    x, eps = rng.standard_normal((2, 31))
    t = np.array([0.9, 0.55])
    al, sg = synth.vp_schedule(t)
    for a, s in ((al, sg), (np.ones(2), np.array([4.0, 1.5]))):
        z = a[0] * x + s[0] * eps
        np.testing.assert_allclose(grpo.ddim_mean(z, eps, a[0], a[1], s[0], s[1]), a[1] * x + s[1] * eps,
                                   rtol=1e-12, atol=1e-13)


@pytest.mark.parametrize("seed", [93, 94])
def test_eps_signals_are_the_gradient_of_the_window_loss(seed):
    """s_ij equals the central difference of the epsilon window loss in eps_hat_ij."""
    clip, scale = 0.1, 0.37
    t, al, sg, sig, z, e = _eps_case(seed)
    G, W, D = e.shape
    lp = np.array([[grpo.step_logprob_eps(z[i, j + 1], z[i, j], e[i, j], al[j], al[j + 1], sg[j], sg[j + 1], sig[j])
                    for j in range(W)] for i in range(G)])
    rng = np.random.Generator(np.random.PCG64(seed + 100))
    lpo = lp + rng.uniform(-0.3, 0.3, size=(G, W))
    A = np.array([1.3, -0.7, 0.4])
    s, _, ratio, clipped = grpo.step_signals_eps(e, z, al, sg, sig, lpo, A, clip, scale)
    h = 1e-6
    for i in range(G):
        for j in range(W):
            if abs(abs(ratio[i, j] - 1.0) - clip) < 1e-4:
                continue
            for k in range(D):
                ep = e[i].copy(); ep[j, k] += h
                em = e[i].copy(); em[j, k] -= h
                fd = (grpo.window_loss_eps(ep, z[i], al, sg, sig, lpo[i], A[i], clip, scale)
                      - grpo.window_loss_eps(em, z[i], al, sg, sig, lpo[i], A[i], clip, scale)) / (2 * h)
                assert fd == pytest.approx(s[i, j, k], rel=1e-6, abs=1e-9)
    assert clipped.any() and not clipped.all()


# ------------------------------------------------------------------ sampler step (rollout)
from oracle import rollout as oracle_rollout  # noqa: E402


@pytest.mark.parametrize("eps_model", [False, True])
def test_sampler_step_logprob_is_the_density_of_its_noise(eps_model):
    """z_{j+1} - mu = sigma xi up to the float32 storage of z_{j+1}, so the log-prob of the
    drawn sample is the standard-normal density of xi rescaled: -||xi||^2 / 2 - D log(sqrt(2 pi)
    sigma) (scipy), within the storage rounding."""
    rng = np.random.Generator(np.random.PCG64(95))
    G, D = 3, 40
    z, y, xi = rng.standard_normal((3, G, D))
    t0, t1, sig = 0.7, 0.62, 0.2
    sched = tuple(np.concatenate(synth.vp_schedule([t0, t1]))[[0, 1, 2, 3]]) if eps_model else None
    zn, lp = oracle_rollout.sampler_step(z, y, xi, t0, t1, sig, sched)
    ref = stats.norm.logpdf(xi, scale=1.0).sum(axis=1) - D * math.log(sig)
    np.testing.assert_allclose(lp, ref, rtol=0, atol=1e-4)
    assert zn.dtype == np.float64 and np.array_equal(zn, zn.astype(np.float32).astype(np.float64))


def test_sampler_step_without_noise_follows_the_flow():
    """sigma -> 0: the flow step is the Euler step of dz/dt = v (exact for a constant field:
    z moves by v (t_{j+1} - t_j)); the epsilon step on the rectified-flow schedule with
    eps = z + (1 - t) v is the same step."""
    rng = np.random.Generator(np.random.PCG64(96))
    D = 17
    z, v, xi = rng.standard_normal((3, D))
    t0, t1 = 0.9, 0.75
    zn, _ = oracle_rollout.sampler_step(z, v, xi, t0, t1, 1e-12)
    np.testing.assert_allclose(zn, z + v * (t1 - t0), atol=1e-6)
    e = z + (1 - t0) * v
    zn2, _ = oracle_rollout.sampler_step(z, e, xi, t0, t1, 1e-12, sched=(1 - t0, 1 - t1, t0, t1))
    np.testing.assert_allclose(zn2, zn, atol=1e-6)


def test_clip_tie_counts_as_unclipped():
    """At rho = 1 + eps (A > 0) or rho = 1 - eps (A < 0) exactly, both branches of the max()
    in Eq. grpo_loss have the same value; the step keeps its gradient, which equals the one
    it has under a wider clip range."""
    G, W = 2, 1
    v, z, t, sig, lp, _ = _signals_case(6, W=W, G=G, rho_shift=np.zeros((G, W)), eps=0.1)
    for A, log_rho in [(1.0, 0.07), (-1.0, -0.07)]:
        lpo = lp - log_rho
        _, _, ratio, _ = grpo.step_signals(v, z, t, sig, lpo, np.array([A, A]), 0.5, 1.0)
        rho = ratio[0, 0]
        eps_tie = rho - 1.0 if A > 0 else 1.0 - rho     # exact (Sterbenz): 1 +- eps_tie == rho
        assert (1.0 + eps_tie == rho) if A > 0 else (1.0 - eps_tie == rho)
        s_tie, _, _, clipped = grpo.step_signals(v, z, t, sig, lpo, np.array([A, A]), eps_tie, 1.0)
        s_wide, _, _, _ = grpo.step_signals(v, z, t, sig, lpo, np.array([A, A]), 0.5, 1.0)
        assert clipped[0, 0] == 0
        np.testing.assert_array_equal(s_tie[0], s_wide[0])
        assert np.abs(s_tie[0]).sum() > 0
        # one ulp of rho past the tie the clipped branch is strictly larger
        past = eps_tie - np.spacing(rho)
        _, _, _, clipped = grpo.step_signals(v, z, t, sig, lpo, np.array([A, A]), past, 1.0)
        assert clipped[0, 0] == 1
