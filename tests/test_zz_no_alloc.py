"""The allocation-free step-signals entry point (grpo_step_signals_static).

Some callers cannot allocate device memory for a workspace (a runtime with a fixed,
pre-planned memory budget, or a host without a device allocator of its own).  For them
the library offers grpo_step_signals_static, whose scratch is an array compiled into the
library.  This test calls it through the C ABI twice in a row, on two different windows,
and checks each call against the workspace-taking grpo_step_signals on the same inputs,
with the tolerances of the other signal tests.  The file is named to be collected last."""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

jg = pytest.importorskip("paper_2607_17572_gb300")


def _rel(a, b):
    a = a.double().cpu().numpy().ravel()
    b = b.double().cpu().numpy().ravel()
    nb = np.linalg.norm(b)
    return np.linalg.norm(a - b) / (nb if nb > 0 else 1.0)


def _window(G, W, D, seed):
    g = torch.Generator(device="cuda").manual_seed(seed)
    dev = "cuda"
    t = torch.linspace(0.9, 0.9 - 0.0625 * W, W + 1, dtype=torch.float64, device=dev)
    sig = 0.7 * (t[:-1] - t[1:]).abs().sqrt()
    v = torch.randn(G, W, D, device=dev, generator=g).bfloat16()
    z = torch.zeros(G, W + 1, D, device=dev)
    z[:, 0] = torch.randn(G, D, device=dev, generator=g)
    for j in range(W):
        z[:, j + 1] = (z[:, j] + v[:, j].float() * float(t[j + 1] - t[j])
                       + float(sig[j]) * torch.randn(G, D, device=dev, generator=g))
    rewards = torch.randn(G, device=dev, generator=g)
    return v, z, t, sig, rewards


def _outputs(G, W, D):
    f64 = dict(dtype=torch.float64, device="cuda")
    return dict(logp_new=torch.full((G, W), float("nan"), **f64), ratio=torch.full((G, W), float("nan"), **f64),
                clipped=torch.full((G, W), 7, dtype=torch.uint8, device="cuda"),
                adv_out=torch.full((G,), float("nan"), **f64)), \
        torch.full((G, W, D), float("nan"), device="cuda"), torch.full((2 * G, D), float("nan"), device="cuda")


def _run(G, W, D, seed):
    v, z, t, sig, rewards = _window(G, W, D, seed)
    eps, scale = 0.1, 1.0 / (G * 16)
    # old log-probs near the new ones: take the new log-probs of a first pass, then offset
    ref, s_ref, cot_ref = _outputs(G, W, D)
    ws = jg.alloc_bytes(jg.signals_workspace_bytes(G, W, D))
    zero = torch.zeros(G, W, dtype=torch.float64, device="cuda")
    jg.grpo_step_signals(v, z, t, sig, zero, rewards, eps, 5.0, 1e-8, scale, ws=ws, **ref)
    off = torch.linspace(-0.25, 0.25, G * W, dtype=torch.float64, device="cuda").reshape(G, W)
    logp_old = ref["logp_new"] + off
    jg.grpo_step_signals(v, z, t, sig, logp_old, rewards, eps, 5.0, 1e-8, scale, ws=ws, s_out=s_ref,
                         cot_out=cot_ref, **ref)
    out, s, cot = _outputs(G, W, D)
    jg.grpo_step_signals_static(v, z, t, sig, logp_old, rewards, eps, 5.0, 1e-8, scale, s_out=s, cot_out=cot, **out)
    torch.cuda.synchronize()
    assert jg.device_status() == 0
    lp_tol = 1e-6 * max(10.0, D / 50)
    assert (out["logp_new"] - ref["logp_new"]).abs().max().item() < lp_tol
    assert torch.equal(out["clipped"], ref["clipped"])
    assert torch.allclose(out["adv_out"], ref["adv_out"], rtol=1e-12, atol=1e-12)
    assert _rel(s, s_ref) < 1e-4
    assert _rel(cot, cot_ref) < 1e-4
    return out


def test_static_scratch_entry_point_matches_workspace_entry_point_twice():
    first = _run(8, 4, 16384, seed=1)      # DiT-B latent, W = 4
    second = _run(3, 6, 12345, seed=2)     # a different shape right after: no stale scratch
    assert first["clipped"].shape != second["clipped"].shape


def test_static_scratch_rejects_requests_beyond_its_size():
    G, W, D = 64, 64, 8192 * 64          # needs 64*64*64*8 bytes of partial sums > 1 MiB
    assert jg.signals_workspace_bytes(G, W, D) > 1 << 20
    v = torch.zeros(1, device="cuda")
    with pytest.raises(jg.JaggError, match="scratch"):
        jg.lib().jagg_last_error()
        st = jg.lib().grpo_step_signals_static(v.data_ptr(), 0, v.data_ptr(), v.data_ptr(), v.data_ptr(),
                                               v.data_ptr(), v.data_ptr(), G, W, D, 0.1, 5.0, 1e-8, 1.0, None, None,
                                               v.data_ptr(), v.data_ptr(), v.data_ptr(), v.data_ptr(),
                                               torch.cuda.current_stream().cuda_stream)
        jg._check(st, "grpo_step_signals_static")


def test_static_scratch_entry_point_allocates_nothing():
    """What the entry point is for: after a first call on the device (which looks up the
    array's address), further calls change neither PyTorch's allocated bytes nor the
    device's free memory (cudaMemGetInfo)."""
    G, W, D = 4, 4, 8192
    v, z, t, sig, rewards = _window(G, W, D, seed=3)
    out, s, cot = _outputs(G, W, D)
    logp_old = torch.zeros(G, W, dtype=torch.float64, device="cuda")
    args = (v, z, t, sig, logp_old, rewards, 0.1, 5.0, 1e-8, 1.0 / (G * 16))
    jg.grpo_step_signals_static(*args, s_out=s, cot_out=cot, **out)
    torch.cuda.synchronize()
    alloc0, free0 = torch.cuda.memory_allocated(), torch.cuda.mem_get_info()[0]
    for _ in range(2):
        jg.grpo_step_signals_static(*args, s_out=s, cot_out=cot, **out)
    torch.cuda.synchronize()
    assert jg.device_status() == 0
    assert torch.cuda.memory_allocated() == alloc0
    assert torch.cuda.mem_get_info()[0] == free0


def test_static_scratch_errors_name_the_static_entry_point():
    v = torch.zeros(16, device="cuda")
    p = v.data_ptr()
    st = jg.lib().grpo_step_signals_static(p, 0, p, p, p, p, p, 2, 2, 64, 0.1, 5.0, 1e-8, 1.0, None, None,
                                           None, p, p, p, torch.cuda.current_stream().cuda_stream)   # null logp_new
    assert st == -1
    assert jg.lib().jagg_last_error().decode().startswith("grpo_step_signals_static")
