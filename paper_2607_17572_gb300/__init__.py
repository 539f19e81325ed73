"""Python binding of the JAGG backward library (libjagg.so, sm_103a).

Argument marshalling only: every function here passes device pointers, sizes and the
current CUDA stream to the C ABI of include/jagg.h and raises JaggError on a non-zero
status.  PyTorch provides device memory and streams.  There is no fallback: if the
library has not been built, or no CUDA device is present, the calls fail.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import torch

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "_lib", "libjagg.so")

DTYPE_F32 = 0
DTYPE_BF16 = 1
ARCH_DIT = 0
ARCH_MMDIT = 1

_TORCH_DTYPE = {DTYPE_F32: torch.float32, DTYPE_BF16: torch.bfloat16}


class JaggError(RuntimeError):
    pass


class Config(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "arch", "dtype", "hidden", "heads", "mlp", "depth", "depth_double", "in_channels",
        "latent_h", "latent_w", "patch", "txt_len", "txt_dim", "freq_dim")]

    @classmethod
    def from_workload(cls, wl) -> "Config":
        return cls(arch=ARCH_DIT if wl.arch == "dit" else ARCH_MMDIT,
                   dtype=DTYPE_BF16 if wl.dtype == "bf16" else DTYPE_F32,
                   hidden=wl.hidden, heads=wl.heads, mlp=wl.mlp, depth=wl.depth,
                   depth_double=wl.depth_double, in_channels=wl.in_channels,
                   latent_h=wl.latent_h, latent_w=wl.latent_w, patch=wl.patch,
                   txt_len=wl.txt_len, txt_dim=wl.txt_dim, freq_dim=wl.freq_dim)

    @property
    def torch_dtype(self):
        return _TORCH_DTYPE[self.dtype]


class GemmDesc(ctypes.Structure):
    _fields_ = [("M", ctypes.c_int32), ("N", ctypes.c_int32), ("K", ctypes.c_int32),
                ("A", ctypes.c_void_p), ("lda", ctypes.c_int64), ("a_mn", ctypes.c_int32),
                ("a_dtype", ctypes.c_int32), ("B", ctypes.c_void_p), ("ldb", ctypes.c_int64),
                ("b_mn", ctypes.c_int32), ("b_dtype", ctypes.c_int32), ("epi", ctypes.c_int32),
                ("bias", ctypes.c_void_p), ("bias_dtype", ctypes.c_int32), ("C", ctypes.c_void_p),
                ("ldc", ctypes.c_int64), ("c_dtype", ctypes.c_int32), ("C2", ctypes.c_void_p),
                ("ldc2", ctypes.c_int64), ("aux", ctypes.c_void_p), ("ld_aux", ctypes.c_int64),
                ("gate", ctypes.c_void_p), ("gate_stride", ctypes.c_int64),
                ("rows_per_seq", ctypes.c_int32), ("split_k", ctypes.c_int32),
                ("force_simt", ctypes.c_int32), ("c_trans", ctypes.c_int32), ("bias_m", ctypes.c_int32),
                ("tile_n", ctypes.c_int32)]


class ProfileStat(ctypes.Structure):
    _fields_ = [("family", ctypes.c_char * 32), ("launches", ctypes.c_int64), ("ms", ctypes.c_double),
                ("flops", ctypes.c_double), ("bytes", ctypes.c_double)]


class ProfileLaunch(ctypes.Structure):
    _fields_ = [("family", ctypes.c_char * 32), ("m", ctypes.c_int32), ("n", ctypes.c_int32),
                ("k", ctypes.c_int32), ("ms", ctypes.c_double), ("flops", ctypes.c_double),
                ("bytes", ctypes.c_double)]


_lib = None
_P = ctypes.c_void_p
_I = ctypes.c_int
_I64 = ctypes.c_int64
_SZ = ctypes.c_size_t
_D = ctypes.c_double

_SIGNATURES = {
    "jagg_last_error": (ctypes.c_char_p, []),
    "jagg_device_status": (_I, [ctypes.POINTER(ctypes.c_uint), _I]),
    "jagg_launch_count": (_I64, []),
    "jagg_profile_enable": (_I, [_I]),
    "jagg_profile_read": (_I, [ctypes.POINTER(ProfileStat), _I, ctypes.POINTER(_I)]),
    "jagg_profile_launches": (_I, [ctypes.POINTER(ProfileLaunch), _I, ctypes.POINTER(_I)]),
    "jagg_param_count": (_I64, [ctypes.POINTER(Config)]),
    "jagg_param_tensor_count": (_I, [ctypes.POINTER(Config)]),
    "jagg_param_info": (_I, [ctypes.POINTER(Config), _I, ctypes.c_char_p, _SZ, ctypes.POINTER(_I64),
                             ctypes.POINTER(_I64), ctypes.POINTER(_I64)]),
    "jagg_model_create": (_I, [ctypes.POINTER(Config), _P, ctypes.POINTER(_P)]),
    "jagg_model_destroy": (_I, [_P]),
    "jagg_saved_bytes": (_I64, [_P, _I]),
    "jagg_workspace_bytes": (_I64, [_P, _I]),
    "dit_forward_save": (_I, [_P, _P, _P, _P, _I, _P, _P, _SZ, _P, _SZ, _P]),
    "dit_joint_vjp": (_I, [_P, _P, _SZ, _I, _P, _P, _P, _SZ, _P]),
    "jagg_signals_workspace_bytes": (_I64, [_I, _I, _I64]),
    "grpo_step_signals": (_I, [_P, _I, _P, _P, _P, _P, _P, _I, _I, _I64, _D, _D, _D, _D, _P, _P, _P, _P,
                               _P, _P, _P, _SZ, _P]),
    "grpo_step_signals_eps": (_I, [_P, _I, _P, _P, _P, _P, _P, _P, _P, _I, _I, _I64, _D, _D, _D, _D, _P, _P, _P,
                                   _P, _P, _P, _P, _SZ, _P]),
    "jagg_rollout_workspace_bytes": (_I64, [_I, _I64]),
    "jagg_rollout_step": (_I, [_P, _I, _I64, _P, _P, _I64, _P, _I64, _I, _I64, _D, _D, _D, _P, _P, _I64, _P, _I,
                               _P, _SZ, _P]),
    "grpo_step_signals_static": (_I, [_P, _I, _P, _P, _P, _P, _P, _I, _I, _I64, _D, _D, _D, _D, _P, _P, _P, _P,
                                      _P, _P, _P]),
    "jagg_aggregate": (_I, [_P, _P, _I, _I, _I64, _P, _P]),
    "jagg_aggregate_span": (_I, [_P, _I64, _P, _D, _D, _I, _I, _I64, _P, _I, _P]),
    "jagg_route": (_I, [_I, _D, _P, _D, _P, _P]),
    "jagg_grad_reduce_workspace_bytes": (_I64, [_I64]),
    "grad_reduce": (_I, [_P, _P, _I64, ctypes.c_float, _P, _P, _P, _SZ, _P]),
    "jagg_test_gemm": (_I, [ctypes.POINTER(GemmDesc), _P]),
    "jagg_test_wait_timeout": (_I, [ctypes.c_ulonglong, _P, _P]),
    "jagg_test_attention_fwd": (_I, [_P, _I, _I, _I, _I, _I, _P, _P, _P]),
    "jagg_test_attention_scratch_bytes": (_I64, [_I, _I, _I, _I]),
    "jagg_test_attention_bwd": (_I, [_P, _P, _P, _P, _I, _I, _I, _I, _I, _P, _P, _P]),
    "jagg_test_attention_fwd_streams": (_I, [_P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _I, _P]),
    "jagg_test_ln_gate_bwd": (_I, [_I, _I, _I, _I, _I, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P,
                                   _I, _P]),
    "jagg_test_qk_norm_rope_fwd": (_I, [_P, _I64, _I, _I, _I, _I, _I, _I, _P, _P, _I, _P, _P, _P, _I, _P]),
    "jagg_test_qk_norm_rope_bwd": (_I, [_P, _I64, _I, _I, _I, _I, _I, _I, _P, _P, _I, _P, _P, _P, _I64, _P, _P, _I,
                                        _P]),
    "jagg_test_colsum": (_I, [_P, _I, _I, _I, _I64, _P, _P]),
    "jagg_test_attention_bwd_streams": (_I, [_P, _P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _P, _P, _P, _I,
                                             _P]),
}


def lib():
    """Loads libjagg.so (built by __graft_entry__.build()); raises if it is missing."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise JaggError(f"{LIB_PATH} is missing: build it with __graft_entry__.build()")
        L = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGNATURES.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def _check(status: int, what: str):
    if status != 0:
        msg = lib().jagg_last_error().decode(errors="replace")
        raise JaggError(f"{what} failed with status {status}: {msg}")


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


def _need_cuda(*ts):
    for t in ts:
        if t is not None and not isinstance(t, int) and (not t.is_cuda or not t.is_contiguous()):
            raise JaggError("device tensors must be contiguous CUDA tensors")


# ----------------------------------------------------------------------------- tables
@dataclass(frozen=True)
class ParamInfo:
    name: str
    offset: int
    rows: int
    cols: int

    @property
    def numel(self) -> int:
        return self.rows * self.cols


def param_table(cfg: Config):
    """The library's parameter layout: one ParamInfo per tensor, in buffer order."""
    n = lib().jagg_param_tensor_count(ctypes.byref(cfg))
    if n < 0:
        _check(-1, "jagg_param_tensor_count")
    out = []
    buf = ctypes.create_string_buffer(128)
    off, r, c = _I64(), _I64(), _I64()
    for i in range(n):
        _check(lib().jagg_param_info(ctypes.byref(cfg), i, buf, 128, ctypes.byref(off), ctypes.byref(r),
                                     ctypes.byref(c)), "jagg_param_info")
        out.append(ParamInfo(buf.value.decode(), off.value, r.value, c.value))
    return out


def param_count(cfg: Config) -> int:
    n = lib().jagg_param_count(ctypes.byref(cfg))
    if n < 0:
        _check(-1, "jagg_param_count")
    return n


def pack_params(cfg: Config, arrays: dict, device="cuda") -> torch.Tensor:
    """Places named parameter arrays (host arrays or device tensors) into one flat buffer in
    the library's layout on `device`."""
    flat = torch.zeros(param_count(cfg), dtype=cfg.torch_dtype, device=device)
    for p in param_table(cfg):
        a = torch.as_tensor(arrays[p.name]).reshape(-1)
        flat[p.offset:p.offset + p.numel] = a.to(device=device, dtype=cfg.torch_dtype)
    return flat


def unpack_grads(cfg: Config, grad: torch.Tensor) -> dict:
    """Splits a flat gradient buffer into named arrays (host float64 numpy)."""
    g = grad.detach().to("cpu", torch.float64)
    out = {}
    for p in param_table(cfg):
        v = g[p.offset:p.offset + p.numel]
        out[p.name] = (v.reshape(p.rows, p.cols) if p.cols > 1 else v.reshape(p.rows)).numpy()
    return out


# ----------------------------------------------------------------------------- model
class Model:
    """A jagg_model_t over a flat device weight buffer."""

    def __init__(self, cfg: Config, weights: torch.Tensor):
        _need_cuda(weights)
        self.cfg = cfg
        self.weights = weights
        h = _P()
        _check(lib().jagg_model_create(ctypes.byref(cfg), _ptr(weights), ctypes.byref(h)), "jagg_model_create")
        self.handle = h

    def __del__(self):
        if getattr(self, "handle", None) and _lib is not None:
            _lib.jagg_model_destroy(self.handle)
            self.handle = None

    def saved_bytes(self, B: int) -> int:
        return lib().jagg_saved_bytes(self.handle, B)

    def workspace_bytes(self, B: int) -> int:
        return lib().jagg_workspace_bytes(self.handle, B)

    @property
    def n_img(self) -> int:
        return (self.cfg.latent_h // self.cfg.patch) * (self.cfg.latent_w // self.cfg.patch)


def alloc_bytes(n: int, device="cuda") -> torch.Tensor:
    return torch.empty(max(int(n), 16), dtype=torch.uint8, device=device)


def dit_forward_save(model: Model, z, t, txt, v_out, saved=None, ws=None, stream=None):
    _need_cuda(z, t, txt, v_out, saved, ws)
    B = z.shape[0]
    _check(lib().dit_forward_save(model.handle, _ptr(z), _ptr(t), _ptr(txt), B, _ptr(v_out), _ptr(saved),
                                  0 if saved is None else saved.numel(), _ptr(ws), ws.numel(), _stream(stream)),
           "dit_forward_save")


def dit_joint_vjp(model: Model, saved, B: int, cot, grad, ws, stream=None):
    _need_cuda(saved, cot, grad, ws)
    _check(lib().dit_joint_vjp(model.handle, _ptr(saved), saved.numel(), B, _ptr(cot), _ptr(grad), _ptr(ws),
                               ws.numel(), _stream(stream)), "dit_joint_vjp")


def signals_workspace_bytes(G: int, W: int, D: int) -> int:
    return lib().jagg_signals_workspace_bytes(G, W, D)


def grpo_step_signals(v_hat, z, t, sigma, logp_old, rewards, clip_eps, adv_clip, adv_eps, scale,
                      logp_new, ratio, clipped, adv_out, ws, s_out=None, cot_out=None, stream=None):
    _need_cuda(v_hat, z, t, sigma, logp_old, rewards, logp_new, ratio, clipped, adv_out, ws, s_out, cot_out)
    G, W = v_hat.shape[0], v_hat.shape[1]
    D = v_hat[0, 0].numel()
    vd = DTYPE_BF16 if v_hat.dtype == torch.bfloat16 else DTYPE_F32
    _check(lib().grpo_step_signals(_ptr(v_hat), vd, _ptr(z), _ptr(t), _ptr(sigma), _ptr(logp_old), _ptr(rewards),
                                   G, W, D, clip_eps, adv_clip, adv_eps, scale, _ptr(s_out), _ptr(cot_out),
                                   _ptr(logp_new), _ptr(ratio), _ptr(clipped), _ptr(adv_out), _ptr(ws), ws.numel(),
                                   _stream(stream)), "grpo_step_signals")


def grpo_step_signals_eps(eps_hat, z, t, sched_alpha, sched_sigma, sigma, logp_old, rewards, clip_eps, adv_clip,
                          adv_eps, scale, logp_new, ratio, clipped, adv_out, ws, s_out=None, cot_out=None,
                          stream=None):
    """Phase 2 for an epsilon-prediction backbone: the DDIM mean of the schedule
    (sched_alpha, sched_sigma) [W+1] f64 (device) replaces the flow Euler step."""
    _need_cuda(eps_hat, z, t, sched_alpha, sched_sigma, sigma, logp_old, rewards, logp_new, ratio, clipped, adv_out,
               ws, s_out, cot_out)
    G, W = eps_hat.shape[0], eps_hat.shape[1]
    D = eps_hat[0, 0].numel()
    vd = DTYPE_BF16 if eps_hat.dtype == torch.bfloat16 else DTYPE_F32
    _check(lib().grpo_step_signals_eps(_ptr(eps_hat), vd, _ptr(z), _ptr(t), _ptr(sched_alpha), _ptr(sched_sigma),
                                       _ptr(sigma), _ptr(logp_old), _ptr(rewards), G, W, D, clip_eps, adv_clip,
                                       adv_eps, scale, _ptr(s_out), _ptr(cot_out), _ptr(logp_new), _ptr(ratio),
                                       _ptr(clipped), _ptr(adv_out), _ptr(ws), ws.numel(), _stream(stream)),
           "grpo_step_signals_eps")


def grpo_step_signals_static(v_hat, z, t, sigma, logp_old, rewards, clip_eps, adv_clip, adv_eps, scale,
                             logp_new, ratio, clipped, adv_out, s_out=None, cot_out=None, stream=None):
    """grpo_step_signals without a workspace: scratch comes from an array compiled into the
    library, for callers that cannot allocate device memory."""
    _need_cuda(v_hat, z, t, sigma, logp_old, rewards, logp_new, ratio, clipped, adv_out, s_out, cot_out)
    G, W = v_hat.shape[0], v_hat.shape[1]
    D = v_hat[0, 0].numel()
    vd = DTYPE_BF16 if v_hat.dtype == torch.bfloat16 else DTYPE_F32
    _check(lib().grpo_step_signals_static(_ptr(v_hat), vd, _ptr(z), _ptr(t), _ptr(sigma), _ptr(logp_old),
                                          _ptr(rewards), G, W, D, clip_eps, adv_clip, adv_eps, scale, _ptr(s_out),
                                          _ptr(cot_out), _ptr(logp_new), _ptr(ratio), _ptr(clipped), _ptr(adv_out),
                                          _stream(stream)), "grpo_step_signals_static")


def rollout_workspace_bytes(G: int, D: int) -> int:
    return lib().jagg_rollout_workspace_bytes(G, D)


def jagg_rollout_step(y_hat, z, j: int, xi, t_cur: float, t_next: float, sigma: float, logp, ws, sched=None,
                      z_model=None, stream=None):
    """One sampler step of G trajectories in place: z [G, T+1, ...] f32 (step j -> j+1),
    y_hat [G, ...] model outputs at z[:, j], xi [G, ...] f32 noise, logp [G, T] f64 (column j
    written).  sched = (alpha_cur, alpha_next, sigma_cur, sigma_next) for a noise-prediction
    model, None for a velocity model.  z_model [G, ...] (bf16 or f32), if given, receives
    z[:, j+1] in its dtype (the next forward's input)."""
    _need_cuda(y_hat, z, xi, logp, ws, z_model)
    G = z.shape[0]
    D = z[0, 0].numel()
    assert z.is_contiguous() and y_hat.is_contiguous() and xi.is_contiguous() and logp.is_contiguous()
    assert y_hat[0].numel() == D and xi[0].numel() == D and 0 <= j < z.shape[1] - 1
    es = z.element_size()
    zc = z.data_ptr() + j * D * es
    yd = DTYPE_BF16 if y_hat.dtype == torch.bfloat16 else DTYPE_F32
    sch = (_D * 4)(*[float(x) for x in sched]) if sched is not None else None
    _check(lib().jagg_rollout_step(_ptr(y_hat), yd, D, zc, zc + D * es, z.shape[1] * D, _ptr(xi), D, G, D,
                                   float(t_cur), float(t_next), float(sigma), sch, logp.data_ptr() + j * 8,
                                   logp.shape[1], _ptr(z_model),
                                   DTYPE_BF16 if z_model is not None and z_model.dtype == torch.bfloat16
                                   else DTYPE_F32, _ptr(ws), ws.numel(), _stream(stream)), "jagg_rollout_step")


def jagg_aggregate(s, t_window, cot, stream=None):
    _need_cuda(s, t_window, cot)
    G, W = s.shape[0], s.shape[1]
    D = s[0, 0].numel()
    _check(lib().jagg_aggregate(_ptr(s), _ptr(t_window), G, W, D, _ptr(cot), _stream(stream)), "jagg_aggregate")


def jagg_aggregate_span(s, t_steps, t_first: float, t_last: float, cot, accumulate: bool = False, steps=None,
                        stream=None):
    """Phase 3 over a span of steps.  s [G, W, ...] f32 window signals; `steps` = (first, n)
    selects n consecutive steps (default: all), read in place; t_steps [n] f64 (device);
    cot [2G, ...] f32."""
    _need_cuda(s, t_steps, cot)
    G, W = s.shape[0], s.shape[1]
    D = s[0, 0].numel()
    j0, n = steps if steps is not None else (0, W)
    assert s.is_contiguous() and 0 <= j0 and j0 + n <= W
    ptr = s.data_ptr() + j0 * D * s.element_size()
    _check(lib().jagg_aggregate_span(ptr, W * D, _ptr(t_steps), float(t_first), float(t_last), G, n, D, _ptr(cot),
                                     1 if accumulate else 0, _stream(stream)), "jagg_aggregate_span")


def jagg_route(n_windows: int, jagg_frac: float = 1.0, cos=None, tau: float = 0.5):
    """Host routing; returns (route list of 0/1, derived jagg_frac)."""
    route = (ctypes.c_uint8 * n_windows)()
    frac = _D()
    cos_arr = None
    if cos is not None:
        cos_arr = (_D * n_windows)(*[float(c) for c in cos])
    _check(lib().jagg_route(n_windows, float(jagg_frac), cos_arr, float(tau), route, ctypes.byref(frac)),
           "jagg_route")
    return list(route), frac.value


def grad_reduce_workspace_bytes(P: int) -> int:
    return lib().jagg_grad_reduce_workspace_bytes(P)


def grad_reduce(a, b=None, alpha: float = 1.0, acc=None, out3=None, ws=None, stream=None):
    _need_cuda(a, b, acc, out3, ws)
    _check(lib().grad_reduce(_ptr(a), _ptr(b), a.numel(), float(alpha), _ptr(acc), _ptr(out3), _ptr(ws),
                             0 if ws is None else ws.numel(), _stream(stream)), "grad_reduce")


def launch_count() -> int:
    return lib().jagg_launch_count()


def profile_enable(on: bool):
    _check(lib().jagg_profile_enable(1 if on else 0), "jagg_profile_enable")


def profile_read() -> dict:
    """{family: {"launches", "ms", "flops", "bytes"}} (synchronises the device)."""
    arr = (ProfileStat * 16)()
    n = _I()
    _check(lib().jagg_profile_read(arr, 16, ctypes.byref(n)), "jagg_profile_read")
    return {arr[i].family.decode(): dict(launches=arr[i].launches, ms=arr[i].ms, flops=arr[i].flops,
                                         bytes=arr[i].bytes) for i in range(n.value)}


def profile_launches(cap: int = 200000) -> list:
    """Recorded launches in order: (family, m, n, k, ms, flops, bytes)."""
    arr = (ProfileLaunch * cap)()
    n = _I()
    _check(lib().jagg_profile_launches(arr, cap, ctypes.byref(n)), "jagg_profile_launches")
    return [(arr[i].family.decode(), arr[i].m, arr[i].n, arr[i].k, arr[i].ms, arr[i].flops, arr[i].bytes)
            for i in range(n.value)]


def device_status(clear: bool = True) -> int:
    v = ctypes.c_uint()
    _check(lib().jagg_device_status(ctypes.byref(v), 1 if clear else 0), "jagg_device_status")
    return v.value


# ----------------------------------------------------------------------------- kernel tests
def test_gemm(desc: GemmDesc, stream=None):
    _check(lib().jagg_test_gemm(ctypes.byref(desc), _stream(stream)), "jagg_test_gemm")


def test_attention_fwd(qkv, B, N, heads, dh, o, lse, stream=None):
    dt = DTYPE_BF16 if qkv.dtype == torch.bfloat16 else DTYPE_F32
    _check(lib().jagg_test_attention_fwd(_ptr(qkv), B, N, heads, dh, dt, _ptr(o), _ptr(lse), _stream(stream)),
           "jagg_test_attention_fwd")


def test_attention_bwd(qkv, o, lse, dO, B, N, heads, dh, dqkv, stream=None):
    dt = DTYPE_BF16 if qkv.dtype == torch.bfloat16 else DTYPE_F32
    scratch = alloc_bytes(lib().jagg_test_attention_scratch_bytes(B, N, heads, dh), qkv.device)
    _check(lib().jagg_test_attention_bwd(_ptr(qkv), _ptr(o), _ptr(lse), _ptr(dO), B, N, heads, dh, dt, _ptr(dqkv),
                                         _ptr(scratch), _stream(stream)), "jagg_test_attention_bwd")


def test_attention_fwd_streams(qkv, o, lse, B, N, n0, heads, dh, impl=0, stream=None):
    """Forward over two-stream views: qkv and o given as pairs (first n0 tokens of every
    sequence, the rest), contiguous; n0 = N uses the first only."""
    dt = DTYPE_BF16 if qkv[0].dtype == torch.bfloat16 else DTYPE_F32
    second = lambda pair: _ptr(pair[1]) if n0 < N else None
    _check(lib().jagg_test_attention_fwd_streams(_ptr(qkv[0]), second(qkv), _ptr(o[0]), second(o), _ptr(lse), B, N,
                                                 n0, heads, dh, dt, impl, _stream(stream)),
           "jagg_test_attention_fwd_streams")


def test_attention_bwd_streams(qkv, o, lse, dO, B, N, n0, heads, dh, dqkv, impl=0, stream=None):
    """Backward over two-stream views: each [B, N, *] tensor argument is given as a pair
    (first n0 tokens of every sequence, the rest), contiguous; n0 = N uses the first only."""
    dt = DTYPE_BF16 if qkv[0].dtype == torch.bfloat16 else DTYPE_F32
    scratch = alloc_bytes(lib().jagg_test_attention_scratch_bytes(B, N, heads, dh), qkv[0].device)
    second = lambda pair: _ptr(pair[1]) if n0 < N else None
    _check(lib().jagg_test_attention_bwd_streams(
        _ptr(qkv[0]), second(qkv), _ptr(o[0]), second(o), _ptr(lse), _ptr(dO[0]), second(dO), B, N, n0, heads, dh,
        dt, _ptr(dqkv[0]), second(dqkv), _ptr(scratch), impl, _stream(stream)), "jagg_test_attention_bwd_streams")


def test_ln_gate_bwd(M, d, rows_per_seq, dh_in, dh_out, dm=None, h=None, mean=None, rstd=None, scale=None,
                     dshift=None, dscale=None, y=None, gate=None, dgate=None, dy=None, dbias=None, stream=None):
    """LayerNorm + modulation and gate backward on contiguous rows (jagg_test_ln_gate_bwd);
    the LayerNorm part runs when dm is given, the gate part when y is given."""
    do_ln, do_gate = dm is not None, y is not None
    dt = DTYPE_BF16 if (y is not None and y.dtype == torch.bfloat16) else DTYPE_F32
    _check(lib().jagg_test_ln_gate_bwd(M, d, rows_per_seq, int(do_ln), int(do_gate), _ptr(dm), _ptr(h), _ptr(mean),
                                       _ptr(rstd), _ptr(scale), _ptr(dshift), _ptr(dscale), _ptr(dh_in),
                                       _ptr(dh_out), _ptr(y), _ptr(gate), _ptr(dgate), _ptr(dy), _ptr(dbias), dt,
                                       _stream(stream)), "jagg_test_ln_gate_bwd")


def test_qk_norm_rope_fwd(qkv, M, N, heads, n_txt, gw, qscale, kscale, qk_out, rq, rk, rope=True, stream=None):
    """Per-head RMSNorm + 2D RoPE of q, k (jagg_test_qk_norm_rope_fwd); qkv [M, >= 2d]."""
    d = qk_out.shape[-1] // 2
    dt = DTYPE_BF16 if qkv.dtype == torch.bfloat16 else DTYPE_F32
    _check(lib().jagg_test_qk_norm_rope_fwd(_ptr(qkv), qkv.stride(0), M, N, d, heads, n_txt, gw, _ptr(qscale),
                                            _ptr(kscale), int(rope), _ptr(qk_out), _ptr(rq), _ptr(rk), dt,
                                            _stream(stream)), "jagg_test_qk_norm_rope_fwd")


def test_qk_norm_rope_bwd(qkv, M, N, heads, n_txt, gw, qscale, kscale, rq, rk, dqk, dqscale, dkscale, rope=True,
                          stream=None):
    """Its backward in place on dqk [M, >= 2d] (jagg_test_qk_norm_rope_bwd)."""
    d = qscale.numel() * heads
    dt = DTYPE_BF16 if qkv.dtype == torch.bfloat16 else DTYPE_F32
    _check(lib().jagg_test_qk_norm_rope_bwd(_ptr(qkv), qkv.stride(0), M, N, d, heads, n_txt, gw, _ptr(qscale),
                                            _ptr(kscale), int(rope), _ptr(rq), _ptr(rk), _ptr(dqk), dqk.stride(0),
                                            _ptr(dqscale), _ptr(dkscale), dt, _stream(stream)),
           "jagg_test_qk_norm_rope_bwd")


def test_colsum(X, db, stream=None):
    """db += column sums of X [rows, cols] (f32 or bf16) (jagg_test_colsum)."""
    _check(lib().jagg_test_colsum(_ptr(X), int(X.dtype == torch.float32), X.shape[0], X.shape[1], X.stride(0),
                                  _ptr(db), _stream(stream)), "jagg_test_colsum")


def test_wait_timeout(limit_ns: int, out, stream=None):
    """A bounded mbarrier wait that nothing satisfies, with the given limit: out [2] u64 device
    (int64 tensor) receives (gave up, nanoseconds waited)."""
    _need_cuda(out)
    _check(lib().jagg_test_wait_timeout(int(limit_ns), _ptr(out), _stream(stream)), "jagg_test_wait_timeout")
