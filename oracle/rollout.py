"""Stochastic sampler steps and the flow-SDE rollout producing trajectories and old
log-probs for synthetic workloads.

TEST INFRASTRUCTURE ONLY (see oracle/__init__.py).

The paper's rollout samples G trajectories per prompt from shared initial noise with a
stochastic sampler (Sec. 3.2; appendix "Sampling and rollout").  Here each step is the
Euler-Maruyama step whose Gaussian transition Eq. logprob scores:
z_{j+1} = z_j + v_theta(z_j, t_j) (t_{j+1} - t_j) + sigma_j xi_j, with xi drawn by `synth`.
Trajectories are stored in float32 (the precision the GPU path reads them in); the
network sees them rounded to its storage type.
"""
from __future__ import annotations

import numpy as np

from .grpo import ddim_mean, step_logprob, step_logprob_eps


def sampler_step(z_cur, y_hat, xi, t_cur, t_next, sigma, sched=None):
    """One step of the stochastic sampler whose Gaussian transition Eq. logprob scores, and
    the log-probability of the sample it draws (the rollout's old log-prob):
        z_{j+1} = mu_theta(z_j, t_j) + sigma_j xi_j,   xi_j ~ N(0, I) (passed in),
    with mu the rectified-flow Euler step z_j + v_j (t_{j+1} - t_j) when sched is None, else
    the DDIM mean of an epsilon-prediction model (ddim_mean) with
    sched = (alpha_{t_j}, alpha_{t_{j+1}}, sigma_{t_j}, sigma_{t_{j+1}}).

    z_next is rounded to float32, the precision trajectories are stored in, before its
    log-probability is taken (the update stage scores the stored sample).  Arrays of D
    elements (or [G, D] with the log-prob per row)."""
    z_cur = np.asarray(z_cur, np.float64)
    y_hat = np.asarray(y_hat, np.float64)
    if sched is None:
        mu = z_cur + y_hat * (t_next - t_cur)
    else:
        mu = ddim_mean(z_cur, y_hat, *sched)
    z_next = (mu + sigma * np.asarray(xi, np.float64)).astype(np.float32).astype(np.float64)
    rows = z_next.reshape(-1, z_next.shape[-1]) if z_next.ndim > 1 else z_next[None]
    zc = z_cur.reshape(rows.shape)
    yh = y_hat.reshape(rows.shape)
    if sched is None:
        lp = [step_logprob(rows[i], zc[i], yh[i], t_cur, t_next, sigma) for i in range(rows.shape[0])]
    else:
        lp = [step_logprob_eps(rows[i], zc[i], yh[i], *sched, sigma) for i in range(rows.shape[0])]
    return z_next, (np.array(lp) if z_next.ndim > 1 else lp[0])


def rollout(model, wl, draws, t, sigma, n_steps=None, storage_round=None):
    """Returns z [G, n+1, C, H, W] (float32 values), v [G, n, C, H, W], logp [G, n]."""
    G = wl.G
    n = wl.T if n_steps is None else n_steps
    shape = (wl.in_channels, wl.latent_h, wl.latent_w)
    z = np.zeros((G, n + 1) + shape)
    v = np.zeros((G, n) + shape)
    logp = np.zeros((G, n))
    z[:, 0] = draws.z0[None]
    txt = np.broadcast_to(draws.txt, (G,) + draws.txt.shape)
    for j in range(n):
        zin = z[:, j] if storage_round is None else storage_round(z[:, j])
        vj, _ = model.forward(zin, np.full(G, t[j]), txt)
        if storage_round is not None:
            vj = storage_round(vj)
        v[:, j] = vj
        xi = draws.xi[:, j].reshape(G, -1)
        zn, lp = sampler_step(z[:, j].reshape(G, -1), vj.reshape(G, -1), xi, t[j], t[j + 1], sigma[j])
        z[:, j + 1] = zn.reshape((G,) + shape)
        logp[:, j] = lp
    return z, v, logp
