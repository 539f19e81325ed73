"""A velocity model that is linear in (z, t), for the exactness theorem.

TEST INFRASTRUCTURE ONLY (see oracle/__init__.py).

Theorem (Exact Jacobian Interpolation, Sec. 3.4) assumes v_theta(z, t) linear in the
inputs (z, t).  The model here is v = U (V z + t a + b) + c with theta = (U, V, a, b, c):
linear in (z, t) for fixed theta, bilinear in theta, so its parameter Jacobian J(z, t)
genuinely depends on (z, t) and the theorem is not vacuous.
"""
from __future__ import annotations

import numpy as np


class LinearVelocity:
    def __init__(self, D, k, rng):
        self.U = rng.standard_normal((D, k))
        self.V = rng.standard_normal((k, D)) / np.sqrt(D)
        self.a = rng.standard_normal(k)
        self.b = rng.standard_normal(k)
        self.c = rng.standard_normal(D)

    def forward(self, z, t):
        """z [B, D], t [B] -> v [B, D]."""
        hid = z @ self.V.T + t[:, None] * self.a[None] + self.b[None]
        return hid @ self.U.T + self.c[None]

    def vjp(self, z, t, cot):
        """sum_rows J(z_row, t_row)^T cot_row as a flat vector over (U, V, a, b, c)."""
        hid = z @ self.V.T + t[:, None] * self.a[None] + self.b[None]
        dU = cot.T @ hid
        dc = cot.sum(0)
        dhid = cot @ self.U
        dV = dhid.T @ z
        da = (dhid * t[:, None]).sum(0)
        db = dhid.sum(0)
        return np.concatenate([dU.ravel(), dV.ravel(), da, db, dc])

    def flat_params(self):
        return np.concatenate([self.U.ravel(), self.V.ravel(), self.a, self.b, self.c])

    def set_flat(self, th):
        D, k = self.U.shape
        o = 0
        self.U = th[o:o + D * k].reshape(D, k); o += D * k
        self.V = th[o:o + k * D].reshape(k, D); o += k * D
        self.a = th[o:o + k]; o += k
        self.b = th[o:o + k]; o += k
        self.c = th[o:o + D]
