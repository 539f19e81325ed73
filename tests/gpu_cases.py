"""Shared set-up of the GPU parity tests: seeded inputs from `synth`, the CUDA path through
the C ABI, and the oracle on the same inputs.  Imported by tests only."""
from __future__ import annotations

import numpy as np
import torch

import synth
from oracle import dit


def rel_l2(a, b) -> float:
    a = np.asarray(a, np.float64).ravel()
    b = np.asarray(b, np.float64).ravel()
    nb = np.linalg.norm(b)
    return float(np.linalg.norm(a - b) / (nb if nb > 0 else 1.0))


def cosine(a, b) -> float:
    a = np.asarray(a, np.float64).ravel()
    b = np.asarray(b, np.float64).ravel()
    return float(a @ b / (np.linalg.norm(a) * np.linalg.norm(b)))


def flat(grads: dict, names) -> np.ndarray:
    return np.concatenate([np.asarray(grads[k], np.float64).ravel() for k in names])


def model_inputs(wl, B, seed):
    """Latents, per-row times (f32 values) and text embeddings for B sequences."""
    rng = np.random.Generator(np.random.PCG64(seed))
    z = synth.storage_round(rng.standard_normal((B, wl.in_channels, wl.latent_h, wl.latent_w)), wl.dtype)
    t = rng.uniform(0.05, 1.0, size=B).astype(np.float32).astype(np.float64)
    txt = synth.storage_round(rng.standard_normal((B, wl.txt_len, wl.txt_dim)), wl.dtype)
    return z, t, txt


class GpuModel:
    """The library's model on cuda over the workload's seeded weights."""

    def __init__(self, jg, wl, params):
        self.jg = jg
        self.wl = wl
        self.cfg = jg.Config.from_workload(wl)
        self.weights = jg.pack_params(self.cfg, params)
        self.model = jg.Model(self.cfg, self.weights)
        self.tdt = self.cfg.torch_dtype

    def tensor(self, x):
        return torch.tensor(np.ascontiguousarray(x), dtype=self.tdt, device="cuda")

    def forward(self, z, t, txt, save=True):
        jg = self.jg
        B = z.shape[0]
        zt, tt, xt = self.tensor(z), torch.tensor(t, dtype=torch.float32, device="cuda"), self.tensor(txt)
        v = torch.empty_like(zt)
        ws = jg.alloc_bytes(self.model.workspace_bytes(B))
        saved = jg.alloc_bytes(self.model.saved_bytes(B)) if save else None
        jg.dit_forward_save(self.model, zt, tt, xt, v, saved=saved, ws=ws)
        return v, saved, ws

    def vjp(self, saved, ws, B, cot, grad=None):
        jg = self.jg
        if grad is None:
            grad = torch.zeros(jg.param_count(self.cfg), dtype=torch.float32, device="cuda")
        jg.dit_joint_vjp(self.model, saved, B, torch.tensor(np.ascontiguousarray(cot), dtype=torch.float32,
                                                             device="cuda"), grad, ws)
        return grad


def oracle_vjp(wl, params, z, t, txt, cot):
    model = dit.Backbone(wl, params)
    v, cache = model.forward(z, t, txt)
    return v, model.vjp(cache, cot)
