"""The paper's exactness theorem and corollary as pins of the oracle's JAGG path.

Theorem (Exact Jacobian Interpolation, Sec. 3.4) and its corollary: for a velocity model
linear in (z, t) and window inputs on the affine path between the endpoints with the
same alpha_j as Eq. alpha, J_0^T s_base + J_{W-1}^T s_corr equals sum_j J_j^T s_j."""
import numpy as np
import pytest

import synth
from oracle import dit, grpo, path
from oracle.linear_velocity import LinearVelocity


def _affine_window(rng, t_win, D, G):
    al = grpo.alpha_weights(t_win)
    z0 = rng.standard_normal((G, D))
    z1 = rng.standard_normal((G, D))
    return np.stack([(1 - a) * z0 + a * z1 for a in al], axis=1)      # [G, W, D]


@pytest.mark.parametrize("shift,W", [(1.0, 4), (3.0, 4), (3.0, 8), (1.0, 2)])
def test_jagg_equals_exact_for_linear_velocity(shift, W):
    rng = np.random.Generator(np.random.PCG64(17))
    D, k, G = 12, 5, 3
    model = LinearVelocity(D, k, rng)
    t_all = synth.time_grid(16, shift)
    t_win = t_all[4:4 + W]
    z = _affine_window(rng, t_win, D, G)
    s = rng.standard_normal((G, W, D))
    exact = sum(model.vjp(z[:, j], np.full(G, t_win[j]), s[:, j]) for j in range(W))
    zr, tr = path.window_rows(z, t_win, jagg=True)
    jagg = model.vjp(zr, tr, grpo.aggregate(s, t_win))
    assert np.linalg.norm(jagg - exact) <= 1e-10 * np.linalg.norm(exact)


def test_the_theorem_has_teeth():
    """On a shifted grid, alpha = j/(W-1) (or an off-path middle point) breaks exactness, so
    the pin above would catch an aggregation that ignored the network-input time."""
    rng = np.random.Generator(np.random.PCG64(18))
    D, k, G, W = 12, 5, 3, 4
    model = LinearVelocity(D, k, rng)
    t_win = synth.time_grid(16, 3.0)[4:8]
    z = _affine_window(rng, t_win, D, G)
    s = rng.standard_normal((G, W, D))
    exact = sum(model.vjp(z[:, j], np.full(G, t_win[j]), s[:, j]) for j in range(W))
    zr, tr = path.window_rows(z, t_win, jagg=True)
    uniform = np.linspace(0.0, 1.0, W)
    wrong = np.concatenate([np.einsum("j,gjd->gd", 1 - uniform, s), np.einsum("j,gjd->gd", uniform, s)])
    assert np.linalg.norm(model.vjp(zr, tr, wrong) - exact) > 1e-3 * np.linalg.norm(exact)
    z_off = z.copy(); z_off[:, 1] += 0.1 * rng.standard_normal((G, D))
    exact_off = sum(model.vjp(z_off[:, j], np.full(G, t_win[j]), s[:, j]) for j in range(W))
    jagg = model.vjp(zr, tr, grpo.aggregate(s, t_win))
    assert np.linalg.norm(jagg - exact_off) > 1e-3 * np.linalg.norm(exact_off)


def test_linear_velocity_vjp_matches_central_differences():
    rng = np.random.Generator(np.random.PCG64(19))
    D, k, B = 7, 3, 4
    m = LinearVelocity(D, k, rng)
    z = rng.standard_normal((B, D)); t = rng.uniform(size=B); cot = rng.standard_normal((B, D))
    g = m.vjp(z, t, cot)
    th = m.flat_params()
    u = rng.standard_normal(th.shape)
    h = 1e-6
    m.set_flat(th + h * u); fp = (m.forward(z, t) * cot).sum()
    m.set_flat(th - h * u); fm = (m.forward(z, t) * cot).sum()
    assert (fp - fm) / (2 * h) == pytest.approx(g @ u, rel=1e-8)


def test_w2_jagg_is_exact_for_the_dit():
    """With W = 2, alpha in {0, 1}: JAGG's two rows carry s_0 and s_1 unchanged, so the
    JAGG window gradient equals the exact one for any backbone."""
    wl = synth.WORKLOADS["tiny_dit_f32"]
    params = synth.make_params(wl)
    model = dit.Backbone(wl, params)
    rng = np.random.Generator(np.random.PCG64(20))
    G, W = 2, 2
    zw = rng.standard_normal((G, W, wl.in_channels, wl.latent_h, wl.latent_w))
    t_win = synth.time_grid(8, 1.0)[2:4]
    txt = rng.standard_normal((wl.txt_len, wl.txt_dim))
    s = rng.standard_normal(zw.shape)
    gj = path.window_gradient(model, zw, t_win, txt, s, jagg=True)
    ge = path.window_gradient(model, zw, t_win, txt, s, jagg=False)
    for k in gj:
        np.testing.assert_allclose(gj[k], ge[k], rtol=1e-12, atol=1e-14)


def test_sequential_graph_variant_equals_the_joint_backward():
    """Algorithm 2 (Sec. 3.4): two VJPs of G rows, the first with s_base formed from steps
    0..W-2 only, the second with s_corr completed by the last step, give the same
    gradient as the joint backward over 2G rows (the VJP is linear in the rows)."""
    rng = np.random.Generator(np.random.PCG64(19))
    D, k, G, W = 12, 5, 3, 4
    model = LinearVelocity(D, k, rng)
    t_win = synth.time_grid(16, 3.0)[4:4 + W]
    z = _affine_window(rng, t_win, D, G)
    s = rng.standard_normal((G, W, D))
    zr, tr = path.window_rows(z, t_win, jagg=True)
    joint = model.vjp(zr, tr, grpo.aggregate(s, t_win))
    part = grpo.aggregate_span(s[:, :-1], t_win[:-1], t_win[0], t_win[-1])
    g0 = model.vjp(z[:, 0], np.full(G, t_win[0]), part[:G])
    corr = part[G:] + grpo.aggregate_span(s[:, -1:], t_win[-1:], t_win[0], t_win[-1])[G:]
    g1 = model.vjp(z[:, -1], np.full(G, t_win[-1]), corr)
    assert np.linalg.norm(g0 + g1 - joint) <= 1e-12 * np.linalg.norm(joint)


def test_ablation_is_not_exact_where_jagg_is():
    """On the theorem's linear model with W > 2 the endpoint-only ablation misses the middle
    steps' contribution (JAGG recovers it exactly); with W = 2 both are exact."""
    rng = np.random.Generator(np.random.PCG64(20))
    D, k, G = 12, 5, 3
    model = LinearVelocity(D, k, rng)
    for W, exact_expected in ((4, False), (2, True)):
        t_win = synth.time_grid(16, 3.0)[4:4 + W]
        z = _affine_window(rng, t_win, D, G)
        s = rng.standard_normal((G, W, D))
        exact = sum(model.vjp(z[:, j], np.full(G, t_win[j]), s[:, j]) for j in range(W))
        zr, tr = path.window_rows(z, t_win, jagg=True)
        ab = model.vjp(zr, tr, grpo.aggregate_ablate(s))
        err = np.linalg.norm(ab - exact) / np.linalg.norm(exact)
        assert (err <= 1e-10) == exact_expected, (W, err)
