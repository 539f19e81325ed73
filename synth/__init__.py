"""Seeded synthetic inputs for the JAGG backward path.

This module is the one piece shared by the CUDA path's tests/bench and the float64
oracle.  It holds none of the method's arithmetic: it defines the workloads as plain
data, draws random numbers (numpy PCG64), initialises weights (Xavier-uniform), builds
the sampler's time schedule that the method takes as an input, and rounds drawn values
to bf16 so that both sides receive identical numbers.

Workloads follow the paper's text-to-image settings (rectified-flow DiT/MMDiT backbones,
groups of G samples of one prompt, T sampling steps split into windows of W steps,
Sec. 4 and the hyper-parameter table of the appendix), shrunk or truncated so that a
single GPU holds them.  The paper's seeds are kept: weights 42, sampler noise 12627.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field, replace

import numpy as np

WEIGHT_SEED = 42      # appendix "Common GRPO and optimization settings": seed 42
NOISE_SEED = 12627    # same passage: sampler seed 12627


@dataclass(frozen=True)
class Workload:
    """One synthetic workload: the backbone shape plus the GRPO trajectory setup."""
    name: str
    arch: str                 # "dit" (single-stream blocks) or "mmdit" (double + single)
    dtype: str                # "f32" or "bf16": storage/compute type of the GPU path
    hidden: int               # d
    heads: int                # h (head dim = d / h)
    mlp: int                  # MLP width
    depth: int                # single-stream blocks (dit) / Flux-style single blocks (mmdit)
    depth_double: int         # double-stream blocks (mmdit only)
    in_channels: int          # latent channels C
    latent_h: int
    latent_w: int
    patch: int
    txt_len: int
    txt_dim: int
    G: int                    # group size (samples of one prompt)
    T: int                    # sampling steps
    W: int                    # JAGG window
    shift: float              # timestep shift of the network-input time (1 = none)
    eta: float                # SDE noise level (sigma_j = eta * sqrt(|dt_j|))
    clip_eps: float           # PPO clip range
    jagg_frac: float = 1.0
    adv_clip: float = 5.0
    adv_eps: float = 1e-8
    freq_dim: int = 256

    @property
    def head_dim(self) -> int:
        return self.hidden // self.heads

    @property
    def n_img(self) -> int:
        return (self.latent_h // self.patch) * (self.latent_w // self.patch)

    @property
    def n_tok(self) -> int:
        return self.n_img + self.txt_len

    @property
    def D(self) -> int:
        """Latent elements per sample (the dimension of v-hat and z)."""
        return self.in_channels * self.latent_h * self.latent_w

    @property
    def n_windows(self) -> int:
        return self.T // self.W

    @property
    def patch_dim(self) -> int:
        return self.in_channels * self.patch * self.patch

    @property
    def rope(self) -> bool:
        return self.arch == "mmdit"

    @property
    def pos_embed(self) -> bool:
        return self.arch == "dit"


WORKLOADS = {
    # 2 single-stream blocks, d=64, fp32; 4x4x4 latent, patch 1; G=4, T=8, W=4.
    "tiny_dit_f32": Workload(
        name="tiny_dit_f32", arch="dit", dtype="f32", hidden=64, heads=4, mlp=256,
        depth=2, depth_double=0, in_channels=4, latent_h=4, latent_w=4, patch=1,
        txt_len=8, txt_dim=64, G=4, T=8, W=4, shift=1.0, eta=0.7, clip_eps=1e-4),
    # DiT-B shape: 12 single-stream blocks, d=768, 12 heads, MLP 3072; 32x32x16 latent,
    # patch 2 (256 image tokens) + 77 text tokens; G=8, T=16, W=4, jagg_frac=1.
    "dit_b_bf16": Workload(
        name="dit_b_bf16", arch="dit", dtype="bf16", hidden=768, heads=12, mlp=3072,
        depth=12, depth_double=0, in_channels=16, latent_h=32, latent_w=32, patch=2,
        txt_len=77, txt_dim=768, G=8, T=16, W=4, shift=1.0, eta=0.7, clip_eps=0.1),
    # Flux-width MMDiT, 4 double + 8 single blocks, 512^2 (1024 img + 512 txt tokens).
    "mmdit_flux512_bf16": Workload(
        name="mmdit_flux512_bf16", arch="mmdit", dtype="bf16", hidden=3072, heads=24,
        mlp=12288, depth=8, depth_double=4, in_channels=16, latent_h=64, latent_w=64,
        patch=2, txt_len=512, txt_dim=4096, G=8, T=16, W=4, shift=3.0, eta=0.7,
        clip_eps=0.1),
    # Same model at 1024^2 (4096 img + 512 txt tokens), G=4.
    "mmdit_flux1024_bf16": Workload(
        name="mmdit_flux1024_bf16", arch="mmdit", dtype="bf16", hidden=3072, heads=24,
        mlp=12288, depth=8, depth_double=4, in_channels=16, latent_h=128, latent_w=128,
        patch=2, txt_len=512, txt_dim=4096, G=4, T=16, W=4, shift=3.0, eta=0.7,
        clip_eps=0.1),
    # Qwen-Image-width dual-stream sweep model: 8 double blocks, 1024 img + 256 txt.
    "mmdit_qwen_sweep_bf16": Workload(
        name="mmdit_qwen_sweep_bf16", arch="mmdit", dtype="bf16", hidden=3072, heads=24,
        mlp=12288, depth=0, depth_double=8, in_channels=16, latent_h=64, latent_w=64,
        patch=2, txt_len=256, txt_dim=3072, G=8, T=16, W=4, shift=3.0, eta=0.7,
        clip_eps=0.1),
}


def small_variant(wl: Workload, **over) -> Workload:
    """A reshaped copy of a workload (tests use it for odd sizes and ragged tails)."""
    return replace(wl, **over)


# ----------------------------------------------------------------------------------
# bf16 rounding (round-to-nearest-even of the float32 value), so both sides get the
# same representable numbers.
# ----------------------------------------------------------------------------------
def bf16_bits(x) -> np.ndarray:
    """Bit patterns of the nearest bf16 values (ties to even) of finite inputs.  The sum
    stays below 2^32 for every finite or infinite float32 (NaN is never rounded here)."""
    f = np.ascontiguousarray(np.asarray(x, dtype=np.float32))
    u = f.view(np.uint32)
    rounded = (u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)
    return rounded.astype(np.uint16)


def bf16_round(x) -> np.ndarray:
    """float64 array holding the bf16-representable values nearest to x."""
    bits = bf16_bits(x).astype(np.uint32) << 16
    return bits.view(np.float32).astype(np.float64)


def storage_round(x, dtype: str) -> np.ndarray:
    """Round to the storage precision of a workload ("f32" or "bf16"), as float64."""
    if dtype == "bf16":
        return bf16_round(x)
    return np.asarray(x, dtype=np.float32).astype(np.float64)


# ----------------------------------------------------------------------------------
# Weights: names and shapes of the parameter tensors (nn.Linear convention, [out, in]).
# ----------------------------------------------------------------------------------
def param_shapes(wl: Workload):
    """Ordered (name, shape) list of every parameter tensor of the backbone."""
    d, dm, pd = wl.hidden, wl.mlp, wl.patch_dim
    dh = wl.head_dim
    out = [
        ("x_embed.w", (d, pd)), ("x_embed.b", (d,)),
        ("txt_embed.w", (d, wl.txt_dim)), ("txt_embed.b", (d,)),
        ("t_embed.w1", (d, wl.freq_dim)), ("t_embed.b1", (d,)),
        ("t_embed.w2", (d, d)), ("t_embed.b2", (d,)),
    ]
    if wl.arch == "dit":
        for i in range(wl.depth):
            p = f"blocks.{i}."
            out += [(p + "mod.w", (6 * d, d)), (p + "mod.b", (6 * d,)),
                    (p + "qkv.w", (3 * d, d)), (p + "qkv.b", (3 * d,)),
                    (p + "proj.w", (d, d)), (p + "proj.b", (d,)),
                    (p + "fc1.w", (dm, d)), (p + "fc1.b", (dm,)),
                    (p + "fc2.w", (d, dm)), (p + "fc2.b", (d,))]
    else:
        for i in range(wl.depth_double):
            for s in ("img", "txt"):
                p = f"double.{i}.{s}."
                out += [(p + "mod.w", (6 * d, d)), (p + "mod.b", (6 * d,)),
                        (p + "qkv.w", (3 * d, d)), (p + "qkv.b", (3 * d,)),
                        (p + "q_norm", (dh,)), (p + "k_norm", (dh,)),
                        (p + "proj.w", (d, d)), (p + "proj.b", (d,)),
                        (p + "fc1.w", (dm, d)), (p + "fc1.b", (dm,)),
                        (p + "fc2.w", (d, dm)), (p + "fc2.b", (d,))]
        for i in range(wl.depth):
            p = f"single.{i}."
            out += [(p + "mod.w", (3 * d, d)), (p + "mod.b", (3 * d,)),
                    (p + "lin1.w", (3 * d + dm, d)), (p + "lin1.b", (3 * d + dm,)),
                    (p + "q_norm", (dh,)), (p + "k_norm", (dh,)),
                    (p + "lin2.w", (d, d + dm)), (p + "lin2.b", (d,))]
    out += [("final.mod.w", (2 * d, d)), ("final.mod.b", (2 * d,)),
            ("final.out.w", (pd, d)), ("final.out.b", (pd,))]
    return out


def make_params(wl: Workload, seed: int = WEIGHT_SEED, bias_scale: float = 0.02):
    """Xavier-uniform matrices, small uniform biases, RMSNorm scales near 1.

    Every matrix (modulation and final layer included) is Xavier-initialised: an
    adaLN-zero initialisation would zero the gates and with them every gradient but the
    last layer's.  Biases are drawn from U(-bias_scale, bias_scale) rather than zero so
    that a misplaced bias shows up in parity tests.  Values are rounded to the
    workload's storage type.
    """
    rng = np.random.Generator(np.random.PCG64(seed))
    params = {}
    for name, shape in param_shapes(wl):
        if len(shape) == 2:
            bound = math.sqrt(6.0 / (shape[0] + shape[1]))
            v = rng.uniform(-bound, bound, size=shape)
        elif name.endswith("_norm"):
            v = 1.0 + rng.uniform(-0.1, 0.1, size=shape)
        else:
            v = rng.uniform(-bias_scale, bias_scale, size=shape)
        params[name] = storage_round(v, wl.dtype)
    return params


def device_params(wl: Workload, seed: int = WEIGHT_SEED, device="cuda", bias_scale: float = 0.02):
    """The draws of make_params (Xavier-uniform matrices, small uniform biases, RMSNorm
    scales near 1, rounded to the storage type) made by torch's generator on a device:
    seconds for the 2.5 B parameters of the Flux-width models, where the host generator
    takes minutes.  Returns {name: float32 device tensor}.  A different stream of numbers
    from make_params with the same seed; both sides of a comparison take the one dict."""
    import torch
    gen = torch.Generator(device=device).manual_seed(seed)
    params = {}
    for name, shape in param_shapes(wl):
        v = torch.empty(shape, dtype=torch.float32, device=device)
        if len(shape) == 2:
            bound = math.sqrt(6.0 / (shape[0] + shape[1]))
            v.uniform_(-bound, bound, generator=gen)
        elif name.endswith("_norm"):
            v.uniform_(0.9, 1.1, generator=gen)
        else:
            v.uniform_(-bias_scale, bias_scale, generator=gen)
        params[name] = v.bfloat16().float() if wl.dtype == "bf16" else v
    return params


# ----------------------------------------------------------------------------------
# Sampler schedule (an input of the method: the network-input times t_j and the
# per-step noise scale sigma_j).
# ----------------------------------------------------------------------------------
def time_grid(T: int, shift: float = 1.0) -> np.ndarray:
    """t_k = 1 - k/T for k = 0..T, then the flow-matching shift t' = s t / (1 + (s-1) t)."""
    t = 1.0 - np.arange(T + 1, dtype=np.float64) / T
    if shift != 1.0:
        t = shift * t / (1.0 + (shift - 1.0) * t)
    return t


def sigma_schedule(t: np.ndarray, eta: float) -> np.ndarray:
    """sigma_j = eta * sqrt(|t_{j+1} - t_j|): Euler-Maruyama step of a constant-eta SDE."""
    return eta * np.sqrt(np.abs(np.diff(t)))


def vp_schedule(t: np.ndarray):
    """A variance-preserving diffusion schedule (alpha_t, sigma_t) = (cos(pi t / 2),
    sin(pi t / 2)) at the times t, for epsilon-prediction inputs."""
    t = np.asarray(t, np.float64)
    return np.cos(0.5 * np.pi * t), np.sin(0.5 * np.pi * t)


# ----------------------------------------------------------------------------------
# Random draws.
# ----------------------------------------------------------------------------------
@dataclass
class GroupDraws:
    z0: np.ndarray          # [C, H, W]  shared initial noise of the group
    txt: np.ndarray         # [txt_len, txt_dim] prompt embedding shared by the group
    xi: np.ndarray          # [G, T, C, H, W] per-sample SDE noise
    rewards: np.ndarray     # [G]
    delta: np.ndarray       # [G, T] perturbation of the old log-probs
    extra: dict = field(default_factory=dict)


def draw_group(wl: Workload, seed: int = NOISE_SEED, clip_margin: bool = True) -> GroupDraws:
    """Draw one group's noise, prompt embedding, rewards and old-log-prob offsets.

    delta sets log(rho) = -delta for a policy equal to the rollout policy.  With
    clip_margin the draws stay away from the clip boundaries +-eps: half of them lie in
    (-0.3 eps, 0.3 eps) (inside the trust region) and half in +-(2 eps, 3 eps) (outside),
    so both branches of the PPO clip occur and small rounding differences between two
    implementations cannot flip a decision.
    """
    rng = np.random.Generator(np.random.PCG64(seed))
    C, H, Wd = wl.in_channels, wl.latent_h, wl.latent_w
    z0 = storage_round(rng.standard_normal((C, H, Wd)), wl.dtype)
    txt = storage_round(rng.standard_normal((wl.txt_len, wl.txt_dim)), wl.dtype)
    xi = rng.standard_normal((wl.G, wl.T, C, H, Wd))
    rewards = rng.standard_normal(wl.G)
    e = wl.clip_eps
    if clip_margin:
        inside = rng.uniform(-0.3 * e, 0.3 * e, size=(wl.G, wl.T))
        outside = rng.uniform(2.0 * e, 3.0 * e, size=(wl.G, wl.T)) * rng.choice([-1.0, 1.0], size=(wl.G, wl.T))
        pick = rng.uniform(size=(wl.G, wl.T)) < 0.5
        delta = np.where(pick, inside, outside)
    else:
        delta = rng.uniform(-2.0 * e, 2.0 * e, size=(wl.G, wl.T))
    return GroupDraws(z0=z0, txt=txt, xi=xi, rewards=rewards, delta=delta)


def random_like(shape, seed: int, scale: float = 1.0, dtype: str = "f32") -> np.ndarray:
    """N(0, scale^2) draws rounded to a storage type (cotangents, signals, velocities)."""
    rng = np.random.Generator(np.random.PCG64(seed))
    return storage_round(scale * rng.standard_normal(shape), dtype)


def uniform_like(shape, seed: int, lo: float, hi: float) -> np.ndarray:
    rng = np.random.Generator(np.random.PCG64(seed))
    return rng.uniform(lo, hi, size=shape)
