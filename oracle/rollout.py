"""Flow-SDE rollout producing trajectories and old log-probs for synthetic workloads.

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

from .grpo import step_logprob


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
        znext = z[:, j] + vj * (t[j + 1] - t[j]) + sigma[j] * draws.xi[:, j]
        z[:, j + 1] = znext.astype(np.float32).astype(np.float64)
        for i in range(G):
            logp[i, j] = step_logprob(z[i, j + 1], z[i, j], v[i, j], t[j], t[j + 1], sigma[j])
    return z, v, logp
