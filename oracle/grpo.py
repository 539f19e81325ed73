"""Float64 GRPO signals, JAGG aggregation, routing and gradient reductions.

TEST INFRASTRUCTURE ONLY (see oracle/__init__.py).

Readings of passages the paper leaves open:
  * advantage: eps = 1e-8, unbiased (Bessel) group std, clamp to +-adv_clip (5.0 in the
    hyper-parameter table);
  * log-prob: the isotropic Gaussian density of the whole latent, i.e. the normalising
    term is D * log(sqrt(2 pi) sigma_j) (it cancels in the ratio); the mean is the
    rectified-flow Euler step mu = z_j + v_j (t_{j+1} - t_j) exactly as Eq. logprob states;
  * epsilon-prediction mean: Eq. logprob writes sigma_{t_j} both for the step's noise scale
    and for the diffusion schedule inside the DDIM mean; the oracle keeps them apart (the
    schedule (alpha_t, sigma_t) of z_t = alpha_t x + sigma_t eps enters the mean only, the
    step's scale the density only), and takes the mean exactly as printed (the deterministic
    DDIM step) whatever the step's noise scale;
  * PPO clip: the gradient follows the max() of Eq. grpo_loss: a step contributes zero
    only when the clipped branch is strictly larger (A > 0 and rho > 1 + eps, or A < 0 and
    rho < 1 - eps); at a tie the step counts as unclipped.  The remark after Phase 2
    states the stronger "zero whenever rho leaves the interval", which the equation does
    not give;
  * loss scale: the per-step surrogate is multiplied by `scale` (1/(G T) averages over
    the group and the trajectory, Eq. grpo_loss averaging over the W steps of a window);
  * routing: n_jagg = floor(jagg_frac * n_windows + 1e-9) leading windows; in calibration
    mode a window qualifies when cos >= tau and the derived jagg_frac is the longest
    qualifying prefix divided by n_windows.
"""
from __future__ import annotations

import math

import numpy as np


def advantages(rewards, eps=1e-8, adv_clip=5.0):
    """Eq. advantage: A_i = (r_i - mean) / (std + eps), clamped to [-adv_clip, adv_clip]."""
    r = np.asarray(rewards, dtype=np.float64)
    G = r.shape[0]
    mu = r.sum() / G
    sd = math.sqrt(((r - mu) ** 2).sum() / (G - 1)) if G > 1 else 0.0
    return np.clip((r - mu) / (sd + eps), -adv_clip, adv_clip)


def step_logprob(z_next, z_cur, v_hat, t_cur, t_next, sigma):
    """Eq. logprob for one step of one sample (arrays of D elements):
    -||z_{j+1} - mu||^2 / (2 sigma^2) - D log(sqrt(2 pi) sigma), mu = z_j + v_j (t_{j+1} - t_j)."""
    z_next = np.asarray(z_next, np.float64).ravel()
    mu = np.asarray(z_cur, np.float64).ravel() + np.asarray(v_hat, np.float64).ravel() * (t_next - t_cur)
    D = z_next.size
    return -((z_next - mu) ** 2).sum() / (2.0 * sigma ** 2) - D * math.log(math.sqrt(2.0 * math.pi) * sigma)


def ppo_step_loss(A, rho, clip_eps):
    """One summand of Eq. grpo_loss: max(-A rho, -A clip(rho, 1-eps, 1+eps))."""
    return max(-A * rho, -A * min(max(rho, 1.0 - clip_eps), 1.0 + clip_eps))


def window_loss(v_hat, z, t, sigma, logp_old, A, clip_eps, scale):
    """scale * sum_j L_j for one sample over one window (Eq. grpo_loss up to the 1/W,
    which `scale` carries).  v_hat [W, D], z [W+1, D], t [W+1], sigma [W], logp_old [W]."""
    total = 0.0
    for j in range(v_hat.shape[0]):
        lp = step_logprob(z[j + 1], z[j], v_hat[j], t[j], t[j + 1], sigma[j])
        total += ppo_step_loss(A, math.exp(lp - logp_old[j]), clip_eps)
    return scale * total


def step_signals(v_hat, z, t, sigma, logp_old, A, clip_eps, scale):
    """Phase 2: s_ij = dL_ij / d v_ij through the SDE log-prob and the PPO clip only,
    with z_j a fixed sample (Sec. 3.3, Phase 2; Eq. logprob; Eq. grpo_loss).

    v_hat [G, W, D], z [G, W+1, D], t [W+1], sigma [W], logp_old [G, W], A [G].
    Returns s [G, W, D], logp_new [G, W], ratio [G, W], clipped [G, W] (uint8: 1 when the
    clipped branch of the max() is strictly larger, so the step's gradient is zero).

    d logp / d v_j = (z_{j+1} - z_j - v_j dt_j) dt_j / sigma_j^2 and d rho = rho d logp, so
    the unclipped branch -A rho has gradient -A rho (z_{j+1} - z_j - v_j dt_j) dt_j / sigma_j^2.
    """
    v_hat = np.asarray(v_hat, np.float64)
    z = np.asarray(z, np.float64)
    G, W, D = v_hat.shape
    s = np.zeros((G, W, D))
    logp = np.zeros((G, W))
    ratio = np.zeros((G, W))
    clipped = np.zeros((G, W), np.uint8)
    for i in range(G):
        for j in range(W):
            dt = t[j + 1] - t[j]
            r = z[i, j + 1] - z[i, j] - v_hat[i, j] * dt
            logp[i, j] = step_logprob(z[i, j + 1], z[i, j], v_hat[i, j], t[j], t[j + 1], sigma[j])
            rho = math.exp(logp[i, j] - logp_old[i, j])
            ratio[i, j] = rho
            a = A[i]
            if (a > 0 and rho > 1.0 + clip_eps) or (a < 0 and rho < 1.0 - clip_eps):
                clipped[i, j] = 1
                continue
            s[i, j] = scale * (-a) * rho * r * dt / sigma[j] ** 2
    return s, logp, ratio, clipped


def ddim_mean(z_cur, eps_hat, a_cur, a_next, s_cur, s_next):
    """Eq. logprob, epsilon-prediction case: the mean of the transition is the deterministic
    DDIM step of the schedule (alpha_t, sigma_t) of z_t = alpha_t x + sigma_t eps,
        mu = alpha_{t_{j+1}} (z_j / alpha_{t_j} - (sigma_{t_j} / alpha_{t_j}
                                                   - sigma_{t_{j+1}} / alpha_{t_{j+1}}) eps_hat_j).
    a_cur, a_next, s_cur, s_next are alpha_{t_j}, alpha_{t_{j+1}}, sigma_{t_j}, sigma_{t_{j+1}}
    (schedule values, not the step's noise scale)."""
    z_cur = np.asarray(z_cur, np.float64)
    eps_hat = np.asarray(eps_hat, np.float64)
    return a_next * (z_cur / a_cur - (s_cur / a_cur - s_next / a_next) * eps_hat)


def step_logprob_eps(z_next, z_cur, eps_hat, a_cur, a_next, s_cur, s_next, sigma):
    """Eq. logprob with the epsilon-prediction mean (ddim_mean); sigma is the step's noise
    scale, as in step_logprob."""
    z_next = np.asarray(z_next, np.float64).ravel()
    mu = ddim_mean(z_cur, eps_hat, a_cur, a_next, s_cur, s_next).ravel()
    D = z_next.size
    return -((z_next - mu) ** 2).sum() / (2.0 * sigma ** 2) - D * math.log(math.sqrt(2.0 * math.pi) * sigma)


def window_loss_eps(eps_hat, z, sched_alpha, sched_sigma, sigma, logp_old, A, clip_eps, scale):
    """window_loss for an epsilon-prediction backbone.  eps_hat [W, D], z [W+1, D],
    sched_alpha / sched_sigma [W+1] = alpha_{t_j}, sigma_{t_j} at the window's times."""
    al, sg = sched_alpha, sched_sigma
    total = 0.0
    for j in range(eps_hat.shape[0]):
        lp = step_logprob_eps(z[j + 1], z[j], eps_hat[j], al[j], al[j + 1], sg[j], sg[j + 1], sigma[j])
        total += ppo_step_loss(A, math.exp(lp - logp_old[j]), clip_eps)
    return scale * total


def step_signals_eps(eps_hat, z, sched_alpha, sched_sigma, sigma, logp_old, A, clip_eps, scale):
    """Phase 2 for an epsilon-prediction backbone: s_ij = dL_ij / d eps_hat_ij (Sec. 3.3,
    Phase 2; Eq. logprob, epsilon case; Eq. grpo_loss).  Shapes as step_signals, with
    sched_alpha / sched_sigma [W+1] in place of t.

    mu is affine in eps_hat with slope c_j = -alpha_{t_{j+1}} (sigma_{t_j} / alpha_{t_j}
    - sigma_{t_{j+1}} / alpha_{t_{j+1}}), so d logp / d eps_hat = (z_{j+1} - mu) c_j / sigma_j^2
    and the unclipped branch -A rho has gradient -A rho (z_{j+1} - mu) c_j / sigma_j^2."""
    eps_hat = np.asarray(eps_hat, np.float64)
    z = np.asarray(z, np.float64)
    al = np.asarray(sched_alpha, np.float64)
    sg = np.asarray(sched_sigma, np.float64)
    G, W, D = eps_hat.shape
    s = np.zeros((G, W, D))
    logp = np.zeros((G, W))
    ratio = np.zeros((G, W))
    clipped = np.zeros((G, W), np.uint8)
    for i in range(G):
        for j in range(W):
            mu = ddim_mean(z[i, j], eps_hat[i, j], al[j], al[j + 1], sg[j], sg[j + 1])
            c = -al[j + 1] * (sg[j] / al[j] - sg[j + 1] / al[j + 1])
            logp[i, j] = step_logprob_eps(z[i, j + 1], z[i, j], eps_hat[i, j], al[j], al[j + 1], sg[j], sg[j + 1],
                                          sigma[j])
            rho = math.exp(logp[i, j] - logp_old[i, j])
            ratio[i, j] = rho
            a = A[i]
            if (a > 0 and rho > 1.0 + clip_eps) or (a < 0 and rho < 1.0 - clip_eps):
                clipped[i, j] = 1
                continue
            s[i, j] = scale * (-a) * rho * (z[i, j + 1] - mu) * c / sigma[j] ** 2
    return s, logp, ratio, clipped


def alpha_weights(t_window):
    """Eq. alpha: alpha_j = (t_0 - t_j) / (t_0 - t_{W-1}) over the window's network-input times."""
    t = np.asarray(t_window, np.float64)
    return (t[0] - t) / (t[0] - t[-1])


def aggregate(s, t_window):
    """Eq. s_base_corr: s_base = sum_j (1 - alpha_j) s_j, s_corr = sum_j alpha_j s_j.

    s [G, W, D] -> cotangent rows [2G, D]: rows 0..G-1 are s_base (endpoint j = 0),
    rows G..2G-1 are s_corr (endpoint j = W-1)."""
    s = np.asarray(s, np.float64)
    G, W, D = s.shape
    al = alpha_weights(t_window)
    base = np.zeros((G, D))
    corr = np.zeros((G, D))
    for j in range(W):
        base += (1.0 - al[j]) * s[:, j]
        corr += al[j] * s[:, j]
    return np.concatenate([base, corr], axis=0)


def aggregate_span(s, t_steps, t_first, t_last):
    """Eq. s_base_corr restricted to some of a window's steps, with alpha taken against the
    window's own endpoint times (Eq. alpha): alpha_j = (t_first - t_j) / (t_first - t_last).

    The sequential-graph variant (Sec. 3.4, Algorithm 2) forms s_base from steps 0 .. W-2
    before step W-1 is computed (alpha_{W-1} = 1 contributes nothing to s_base) and adds
    the last step to s_corr later (alpha_0 = 0 contributes nothing to s_corr).
    s [G, n, D] -> [2G, D] partial sums (rows 0..G-1 base, G..2G-1 corr)."""
    s = np.asarray(s, np.float64)
    G, n, D = s.shape
    t = np.asarray(t_steps, np.float64)
    al = (t_first - t) / (t_first - t_last)
    base = np.zeros((G, D))
    corr = np.zeros((G, D))
    for j in range(n):
        base += (1.0 - al[j]) * s[:, j]
        corr += al[j] * s[:, j]
    return np.concatenate([base, corr], axis=0)


def aggregate_ablate(s):
    """The endpoint-only ablation of Sec. 4: only s_0 and s_{W-1} are kept and each is
    back-propagated through its own endpoint with weight 1 (the intermediate steps are
    discarded and no t-weighting is applied).  s [G, W, D] -> [2G, D]: rows 0..G-1 = s_0,
    rows G..2G-1 = s_{W-1}."""
    s = np.asarray(s, np.float64)
    return np.concatenate([s[:, 0], s[:, -1]], axis=0)


def route_schedule(n_windows, jagg_frac):
    """jagg_frac routing (Sec. 3.3, "High-noise vs. low-noise scheduling"): the first
    floor(jagg_frac n + 1e-9) windows (highest noise first) take JAGG."""
    n_jagg = int(math.floor(jagg_frac * n_windows + 1e-9))
    n_jagg = max(0, min(n_windows, n_jagg))
    return np.array([1 if w < n_jagg else 0 for w in range(n_windows)], np.uint8)


def route_calibrate(cos, tau=0.5):
    """Calibration rule of the gradient-quality appendix: a window qualifies for JAGG when
    cos(g_JAGG, g_exact) >= tau.  Returns (per-window decision, derived jagg_frac =
    longest qualifying prefix / n_windows)."""
    cos = np.asarray(cos, np.float64)
    route = (cos >= tau).astype(np.uint8)
    prefix = 0
    for r in route:
        if not r:
            break
        prefix += 1
    return route, prefix / len(cos)


def grad_stats(a, b):
    """<a,b>, ||a||^2, ||b||^2 and the derived cosine and norm ratio rho = ||a|| / ||b||
    (the two quantities of the gradient-quality table)."""
    a = np.asarray(a, np.float64).ravel()
    b = np.asarray(b, np.float64).ravel()
    ab, aa, bb = float(a @ b), float(a @ a), float(b @ b)
    cos = ab / math.sqrt(aa * bb) if aa > 0 and bb > 0 else 0.0
    return ab, aa, bb, cos, math.sqrt(aa / bb) if bb > 0 else float("inf")
