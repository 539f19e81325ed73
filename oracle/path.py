"""JAGG and exact per-step window gradients (Algorithm 1 and its per-step baseline).

TEST INFRASTRUCTURE ONLY (see oracle/__init__.py).
"""
from __future__ import annotations

import numpy as np

from .grpo import aggregate


def window_rows(z_win, t_win, jagg):
    """Rows of the window's VJP batch.

    z_win [G, W, ...] are the window's network inputs z_0..z_{W-1}, t_win [W] their times.
    JAGG (Phase 4): 2G rows, endpoint 0 for every sample then endpoint W-1.
    Exact per-step baseline: W*G rows ordered step-major (row j*G + i)."""
    G, W = z_win.shape[:2]
    if jagg:
        z = np.concatenate([z_win[:, 0], z_win[:, W - 1]], axis=0)
        t = np.concatenate([np.full(G, t_win[0]), np.full(G, t_win[W - 1])])
    else:
        z = np.concatenate([z_win[:, j] for j in range(W)], axis=0)
        t = np.concatenate([np.full(G, t_win[j]) for j in range(W)])
    return z, t


def window_cotangent(s, t_win, jagg):
    """Cotangent rows matching window_rows: Eq. s_base_corr for JAGG, s itself otherwise."""
    G, W = s.shape[:2]
    if jagg:
        return aggregate(s.reshape(G, W, -1), t_win).reshape((2 * G,) + s.shape[2:])
    return np.concatenate([s[:, j] for j in range(W)], axis=0)


def window_gradient(model, z_win, t_win, txt, s, jagg):
    """Phase 4: the parameter gradient of one window, JAGG (2 endpoint rows with the
    aggregated cotangents) or exact (W rows per sample with their own s_j)."""
    z, t = window_rows(z_win, t_win, jagg)
    cot = window_cotangent(s, t_win, jagg)
    B = z.shape[0]
    txtb = np.broadcast_to(txt, (B,) + txt.shape)
    _, cache = model.forward(z, t, txtb)
    return model.vjp(cache, cot)
