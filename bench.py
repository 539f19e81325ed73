#!/usr/bin/env python3
"""Throughput of the JAGG backward path on GB300.

One step = the whole update-stage backward of one GRPO group.  Default workload: the
Flux-width MMDiT at 1024^2 (4 double-stream + 8 single-stream blocks, d = 3072, 24 heads
of 128, MLP 12288; 4096 image + 512 text tokens; G = 4 samples, T = 16 sampling steps,
windows of W = 4, jagg_frac = 1).  Per window: the step signals with the fused t-weighted
aggregation (Phases 2-3), then the joint VJP over the window's 2G endpoint rows,
accumulating the fp32 parameter gradient (Phase 4, Algorithm 1); after the last window the
gradient's squared norm.  When the whole group's saved activations fit in HBM at once the
step is one timed region; smaller models batch every window's endpoint rows into one
joint VJP (the window gradients add).  The forward passes of Phase 1 (endpoints saved,
middle steps without saves) run before the timed region: their saved activations are
inputs resident in HBM.  The metric is trajectory-steps of gradient per second: G * T
(sample, step) pairs per step.

Also timed: the exact per-step path (jagg_frac = 0: the VJP over all W*G step inputs of
every window with their own s_j), the sequential-graph variant and the endpoint-only
ablation, the update stage (forwards on the stored experience + backward, JAGG against
the exact path), the rollout sampler, and `e2e`, the update stage through the public API
from pinned host buffers (Phase 1 forwards included).  `--sweep` times the routing and
window sweep (W in {2, 4, 8} x jagg_frac in {0, 0.5, 1}) on the Qwen-width MMDiT with the
per-window gradient cosines behind each routing decision.  `--impl reference` times the
float64 CPU oracle.
"""
from __future__ import annotations

import argparse
import json
import os
import subprocess
import sys
import tempfile
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import synth  # noqa: E402

METRIC = "JAGG backward trajectory-steps/s on 1 GB300; tensor-pipe % of BF16 peak"
UNIT = "trajectory-steps/s"


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=10)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", choices=["jagg", "reference"], default="jagg")
    p.add_argument("--workload", default=None,
                   help="default mmdit_flux1024_bf16 (mmdit_qwen_sweep_bf16 with --sweep)")
    p.add_argument("--sweep", action="store_true",
                   help="the routing and window sweep: W in {2, 4, 8} x jagg_frac in {0, 0.5, 1}")
    p.add_argument("--no-graph", action="store_true", help="launch eagerly instead of replaying a CUDA graph")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--quick", action="store_true", help="skip the full-W, e2e and CPU legs")
    p.add_argument("--G", type=int, default=0,
                   help="override the workload's group size (small cases for profiler captures)")
    p.add_argument("--kernel", choices=["attention_bwd", "attention_fwd", "gemm", "hbm"], default=None,
                   help="time one kernel family alone on the workload's shapes instead of the step")
    p.add_argument("--product", default="all",
                   help="for --kernel gemm: one of the block's backward products (gemm_products: DiT fc2_dx, "
                        "fc1_dx, qkv_dx, proj_dx, fc2_dw, fc1_dw, qkv_dw, proj_dw; MMDiT lin2_dx_o, lin2_dx_u, "
                        "lin1_dx, lin2_dw, lin1_dw and the img_ products of a double block) or all")
    p.add_argument("--rows", type=int, default=0, help="sequences per call for --kernel (default 2G)")
    p.add_argument("--vjp-rows", choices=["auto", "group", "window"], default="auto",
                   help="one joint VJP per group (all windows' rows) or per window; auto picks the group "
                        "when its saved activations fit in half of the free device memory")
    return p.parse_args()


def workload(args):
    name = args.workload or ("mmdit_qwen_sweep_bf16" if getattr(args, "sweep", False) else "mmdit_flux1024_bf16")
    wl = synth.WORKLOADS[name]
    if args.G:
        wl = synth.small_variant(wl, name=f"{wl.name}_G{args.G}", G=args.G)
    return wl


def describe(wl) -> str:
    if wl.arch == "dit":
        blocks = f"DiT {wl.depth} blocks"
    else:
        blocks = f"MMDiT {wl.depth_double} double + {wl.depth} single blocks"
    return (f"{wl.name}: {blocks} d={wl.hidden} h={wl.heads} mlp={wl.mlp}, {wl.n_img} img + {wl.txt_len} txt "
            f"tokens, G={wl.G}, T={wl.T}, W={wl.W}, jagg_frac={wl.jagg_frac}")


# DRAM bytes (read + write) per launch of the dense-product kernel over its algorithmic
# bytes, from one ncu capture of the kernel alone (`--kernel gemm`) on the workload's
# backward products at the step's rows; the roofline's `traffic` is this ratio times the
# step's algorithmic bytes per launch.  Absent: no capture of the current kernel.
TRAFFIC_RATIO = {"mmdit_flux1024_bf16": 3.01}


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return d.get("bf16_tflops", 1914.6), d.get("bf16_tflops_sustained", 1710.6), d.get("hbm_gbs", 6771.1), "measured"
    return 1900.0, 1700.0, 6800.0, "fallback"


# ----------------------------------------------------------------------------- distributed
def dist_setup(need_gpu: bool = True):
    """One rank per GPU (NCCL).  The reference arm (the float64 oracle on the host cores)
    needs no GPU: without one its ranks meet over gloo."""
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    gpu = need_gpu or torch.cuda.is_available()
    if ws > 1:
        import torch.distributed as dist
        if gpu:
            torch.cuda.set_device(local)
            dist.init_process_group("nccl", device_id=torch.device("cuda", local))
        else:
            dist.init_process_group("gloo")
    elif gpu:
        torch.cuda.set_device(0)
    return ws, rank


def barrier(ws):
    if ws > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, ws: int) -> float:
    """The slowest rank's time (the whole job's step time); host tensors under gloo."""
    if ws == 1:
        return x
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(units_per_rank: float, ms_per_step: float, ws: int) -> float:
    """Whole-job throughput: every rank's units over the slowest rank's step time."""
    return ws * units_per_rank / (ms_per_step / 1000.0)


# ----------------------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi samples (every 200 ms) of SM clock and throttle reasons during a region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.idx), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"], stdout=self.f,
                                         stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        self.f.flush()
        self.f.seek(0)
        rows = [r.split(",") for r in self.f.read().strip().splitlines() if r.strip()]
        os.unlink(self.f.name)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        sm = [float(r[1]) for r in rows if r[1].strip().replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].strip().replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = set()
        for r in rows:
            for k, name in enumerate(names):
                if len(r) > 5 + k and r[5 + k].strip().lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": float(np.median(sm)) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(rows)}


# ----------------------------------------------------------------------------- workload
def device_params(jg, cfg, seed, dev):
    """Seeded random weights of the architecture, drawn on the device from the library's
    parameter table (Xavier-uniform matrices, biases U(-0.02, 0.02), RMSNorm scales
    U(0.9, 1.1)), rounded to bf16 values; seconds even for the 2.5 B parameters of the
    Flux-width MMDiT, where the host generator of the oracle's inputs takes minutes."""
    gen = torch.Generator(device=dev).manual_seed(seed)
    w = torch.zeros(jg.param_count(cfg), dtype=torch.float32, device=dev)
    for p in jg.param_table(cfg):
        view = w[p.offset:p.offset + p.numel]
        if p.name.endswith("q_norm") or p.name.endswith("k_norm"):
            view.uniform_(0.9, 1.1, generator=gen)
        elif p.cols == 1:
            view.uniform_(-0.02, 0.02, generator=gen)
        else:
            a = (6.0 / (p.rows + p.cols)) ** 0.5
            view.uniform_(-a, a, generator=gen)
    return w.bfloat16().float()


class Bench:
    def __init__(self, wl, dev):
        import paper_2607_17572_gb300 as jg
        self.jg = jg
        self.wl = wl
        self.dev = dev
        self.cfg = jg.Config.from_workload(wl)
        self.tdt = self.cfg.torch_dtype
        self.weights = device_params(jg, self.cfg, synth.WEIGHT_SEED, dev).to(self.tdt)
        self.model = jg.Model(self.cfg, self.weights)
        self.P = jg.param_count(self.cfg)
        G, T, W = wl.G, wl.T, wl.W
        self.nw = T // W
        self.D = wl.D
        self.shape = (wl.in_channels, wl.latent_h, wl.latent_w)
        self.draws = synth.draw_group(wl)
        self.t = synth.time_grid(T, wl.shift)
        self.sig = synth.sigma_schedule(self.t, wl.eta)
        self.scale = 1.0 / (G * T)
        f64 = dict(dtype=torch.float64, device=dev)
        self.t_dev = torch.tensor(self.t, **f64)
        self.sig_dev = torch.tensor(self.sig, **f64)
        self.rewards = torch.tensor(self.draws.rewards, dtype=torch.float32, device=dev)
        self.txt1 = torch.tensor(self.draws.txt, dtype=self.tdt, device=dev)
        # workspace for the largest single call: one window's W*G rows, or the batched calls
        # over every window (2G endpoint rows each, or W*G step rows each) when their saved
        # activations take at most half of the device (the test `fits` applies, against
        # free memory)
        total = torch.cuda.get_device_properties(dev).total_memory
        cands = [W * G] + [r for r in (2 * G * self.nw, W * G * self.nw) if self.model.saved_bytes(r) < 0.5 * total]
        self.ws_rows = max(cands)
        self.ws = jg.alloc_bytes(self.model.workspace_bytes(self.ws_rows), dev)
        self.sws = jg.alloc_bytes(jg.signals_workspace_bytes(G, W, self.D), dev)
        self.rws = jg.alloc_bytes(jg.rollout_workspace_bytes(G, self.D), dev)
        self.gws = jg.alloc_bytes(jg.grad_reduce_workspace_bytes(self.P), dev)
        self.grad = torch.zeros(self.P, dtype=torch.float32, device=dev)
        self.out3 = torch.zeros(3, **f64)
        self.sig_out = dict(logp_new=torch.empty(G, W, **f64), ratio=torch.empty(G, W, **f64),
                            clipped=torch.empty(G, W, dtype=torch.uint8, device=dev), adv_out=torch.empty(G, **f64))
        self.cot_all = torch.empty(self.nw * W * G, self.D, dtype=torch.float32, device=dev)

    # rows of a window's forward: JAGG = [z_0 of each sample; z_{W-1} of each sample],
    # exact = (sample, step) pairs in sample-major order, matching s [G, W, D]
    def rows(self, z_win, w, jagg):
        G, W = self.wl.G, self.wl.W
        tw = self.t[w * W:(w + 1) * W]
        if jagg:
            z = torch.cat([z_win[:, 0], z_win[:, W - 1]], 0)
            t = np.concatenate([np.full(G, tw[0]), np.full(G, tw[W - 1])])
        else:
            z = z_win.reshape(G * W, *self.shape)
            t = np.tile(tw, G)
        return z.to(self.tdt).contiguous(), torch.tensor(t, dtype=torch.float32, device=self.dev)

    def txt_rows(self, B):
        return self.txt1.unsqueeze(0).expand(B, -1, -1).contiguous()

    def sampler(self):
        """The group's rollout on the device (theta_old = theta): per step, the forward without
        saves on the G current samples, then the fused sampler step (Euler-Maruyama draw with
        the passed-in noise, f32 trajectory store, the next forward's bf16 input and the old
        log-prob).  Returns the closure and its buffers."""
        jg, wl, dev = self.jg, self.wl, self.dev
        G, T = wl.G, wl.T
        z = torch.zeros(G, T + 1, self.D, dtype=torch.float32, device=dev)
        z0 = torch.tensor(self.draws.z0.reshape(-1), dtype=torch.float32, device=dev)
        xi = torch.tensor(np.ascontiguousarray(self.draws.xi.reshape(G, T, -1).transpose(1, 0, 2)),
                          dtype=torch.float32, device=dev)            # [T, G, D]: xi[j] contiguous
        v_all = torch.empty(T, G, *self.shape, dtype=self.tdt, device=dev)
        zin = torch.empty(G, *self.shape, dtype=self.tdt, device=dev)
        lp = torch.empty(G, T, dtype=torch.float64, device=dev)
        txt = self.txt_rows(G)
        tin = [torch.full((G,), float(self.t[j]), dtype=torch.float32, device=dev) for j in range(T)]

        def run():
            z[:, 0].copy_(z0.unsqueeze(0).expand(G, -1))
            zin.copy_(z[:, 0].reshape(G, *self.shape))
            for j in range(T):
                jg.dit_forward_save(self.model, zin, tin[j], txt, v_all[j], ws=self.ws)
                jg.jagg_rollout_step(v_all[j], z, j, xi[j], self.t[j], self.t[j + 1], self.sig[j], lp, self.rws,
                                     z_model=zin)
        return run, z, v_all, lp

    def rollout(self):
        """Synthetic trajectories from the model itself: the device sampler; old log-probs =
        the rollout's log-probs + delta."""
        wl, dev = self.wl, self.dev
        G, T, W = wl.G, wl.T, wl.W
        run, z, v_all, lp = self.sampler()
        run()
        self.z = z
        self.v_all = v_all.transpose(0, 1).reshape(G, T, -1).contiguous()
        self.v_win = [self.v_all[:, w * W:(w + 1) * W].contiguous() for w in range(self.nw)]
        self.z_win = [self.z[:, w * W:w * W + W + 1].contiguous() for w in range(self.nw)]
        self.logp_rollout = lp.clone()
        self.logp_old = lp + torch.tensor(self.draws.delta, dtype=torch.float64, device=dev)
        self.lpo_win = [self.logp_old[:, w * W:(w + 1) * W].contiguous() for w in range(self.nw)]
        torch.cuda.synchronize()

    def signals(self, w, logp_old, cot_out=None, s_out=None):
        W = self.wl.W
        self.jg.grpo_step_signals(self.v_win[w], self.z_win[w], self.t_dev[w * W:w * W + W + 1],
                                  self.sig_dev[w * W:(w + 1) * W], logp_old, self.rewards, self.wl.clip_eps,
                                  self.wl.adv_clip, self.wl.adv_eps, self.scale, ws=self.sws, cot_out=cot_out,
                                  s_out=s_out, **self.sig_out)

    def plan(self, routes):
        """Rows of the group's Phase 4: (window, is_jagg, first_row, rows) per window --
        the 2G endpoint rows of a JAGG window, the W*G step rows of an exact window."""
        G, W = self.wl.G, self.wl.W
        out, r = [], 0
        for w in range(self.nw):
            n = 2 * G if routes[w] else W * G
            out.append((w, bool(routes[w]), r, n))
            r += n
        return out, r

    def batch_group(self, routes, mode) -> bool:
        """True: one saved arena (and one joint VJP) for every window of the group."""
        if mode != "auto":
            return mode == "group"
        return self.fits(routes, batched=True)

    def fits(self, routes, batched) -> bool:
        """Every window's saved activations can be resident at once.  batched (one arena,
        one joint VJP over the group): the workspace covers the group's rows and the arena
        takes at most half of the free memory; otherwise (one arena per window) the arenas
        together take at most 90 % of it."""
        plan, rows = self.plan(routes)
        torch.cuda.empty_cache()
        free, _ = torch.cuda.mem_get_info(self.dev)
        self.last_fit = {"free_gb": free / 1e9, "saved_gb_needed": (self.model.saved_bytes(rows) if batched else sum(
            self.model.saved_bytes(n) for (_, _, _, n) in plan)) / 1e9}
        if batched:
            return rows <= self.ws_rows and self.model.saved_bytes(rows) < 0.5 * free
        return sum(self.model.saved_bytes(n) for (_, _, _, n) in plan) < 0.9 * free

    def forward_saves(self, routes, batched, windows=None):
        """Phase 1 with saves for the rows of the plan (or of the listed windows only).
        batched: one arena holding every window's rows (one joint VJP per group); otherwise
        one arena per window."""
        wl = self.wl
        G, W = wl.G, wl.W
        plan, _ = self.plan(routes)
        if windows is not None:
            plan = [p for p in plan if p[0] in windows]
        rows = [self.rows(self.z[:, w * W:(w + 1) * W].reshape(G, W, *self.shape), w, jagg)
                for (w, jagg, _, _) in plan]
        if batched:
            groups = [(torch.cat([r[0] for r in rows]), torch.cat([r[1] for r in rows]), plan)]
        else:
            groups = [(rows[i][0], rows[i][1], [plan[i]]) for i in range(len(plan))]
        arenas = []
        for z, t, pl in groups:
            B = z.shape[0]
            saved = self.jg.alloc_bytes(self.model.saved_bytes(B), self.dev)
            v = torch.empty_like(z)
            self.jg.dit_forward_save(self.model, z, t, self.txt_rows(B), v, saved=saved, ws=self.ws)
            arenas.append((saved, B, pl))
        torch.cuda.synchronize()
        return arenas

    def step(self, arenas, reduce=True):
        """Phases 2-4 for the windows of the arenas, then the gradient's squared norm."""
        jg, G, W, D = self.jg, self.wl.G, self.wl.W, self.D
        for saved, B, pl in arenas:
            row0 = pl[0][2]
            for (w, jagg, r, n) in pl:
                dst = self.cot_all[r:r + n]
                if jagg:
                    self.signals(w, self.lpo_win[w], cot_out=dst)
                else:
                    self.signals(w, self.lpo_win[w], s_out=dst.view(G, W, D))
            jg.dit_joint_vjp(self.model, saved, B, self.cot_all[row0:row0 + B], self.grad, self.ws)
        if reduce:
            jg.grad_reduce(self.grad, None, out3=self.out3, ws=self.gws)


def time_steps(fn, steps, warmup, ws, use_graph):
    """W warm-up calls, then K calls timed with CUDA events on the launching stream."""
    stream = torch.cuda.current_stream()
    graph = None
    if use_graph:
        side = torch.cuda.Stream()
        side.wait_stream(stream)
        with torch.cuda.stream(side):
            fn()
        stream.wait_stream(side)
        torch.cuda.synchronize()
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            fn()
        run = graph.replay
    else:
        run = fn
    for _ in range(warmup):
        run()
    torch.cuda.synchronize()
    barrier(ws)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    # the timed steps are the profiled range of `ncu --profile-from-start off`
    torch.cuda.profiler.start()
    e0.record(stream)
    for _ in range(steps):
        run()
    e1.record(stream)
    torch.cuda.synchronize()
    torch.cuda.profiler.stop()
    barrier(ws)
    return e0.elapsed_time(e1) / steps, graph


# ----------------------------------------------------------------------------- oracle legs
def oracle_sample_plan(wl):
    """What the float64 oracle runs as a bounded sample of the workload, and what it stands
    for.  DiT widths: one JAGG window of 2 samples through the whole model (4 endpoint
    rows).  MMDiT widths, where the whole model takes the oracle minutes per sequence: one
    endpoint row through one block at the workload's full width and token count (a Flux-style
    single block when the model has them, else one double-stream block) with the model's
    embeddings and final layer, its time scaled to one sample's JAGG window (2 endpoint rows
    through the whole model) by the algorithmic FLOPs of flops_per_sequence.
    Returns (sample workload, rows, samples the run stands for, scale)."""
    if wl.arch == "dit":
        return wl, 4, 2, 1.0
    sub = synth.small_variant(wl, depth=min(wl.depth, 1), depth_double=0 if wl.depth else 1)
    full = sum(flops_per_sequence(wl)) * 2
    part = sum(flops_per_sequence(sub))
    return sub, 1, 1, full / part


_ORACLE_MODEL = {}   # the sample's backbone, built once per process


def oracle_sample(wl):
    """One bounded sample of the workload on the float64 oracle (oracle_sample_plan): the step
    signals of one window on synthetic v-hat, the t-weighted aggregation, the forward of the
    sample's rows with caches and the VJP.  Returns (seconds measured, trajectory-steps the
    sample stands for, seconds scaled to them, description)."""
    from oracle import dit, grpo
    sub, rows, n_samples, scale = oracle_sample_plan(wl)
    if _ORACLE_MODEL.get("name") != sub.name:
        _ORACLE_MODEL.update(name=sub.name, model=dit.Backbone(sub, synth.make_params(sub)))
    model = _ORACLE_MODEL["model"]
    rng = np.random.Generator(np.random.PCG64(5))
    W = wl.W
    shape = (wl.in_channels, wl.latent_h, wl.latent_w)
    t = synth.time_grid(wl.T, wl.shift)[:W + 1]
    sig = synth.sigma_schedule(t, wl.eta)
    z = synth.storage_round(rng.standard_normal((n_samples, W + 1) + shape), wl.dtype)
    v = synth.storage_round(rng.standard_normal((n_samples, W) + shape), wl.dtype)
    lpo = np.zeros((n_samples, W))
    txt = np.broadcast_to(synth.draw_group(wl).txt, (rows, wl.txt_len, wl.txt_dim))
    t0 = time.perf_counter()
    s, _, _, _ = grpo.step_signals(v.reshape(n_samples, W, -1), z.reshape(n_samples, W + 1, -1), t, sig, lpo,
                                   grpo.advantages(rng.standard_normal(n_samples)), wl.clip_eps,
                                   1.0 / (wl.G * wl.T))
    cot = grpo.aggregate(s, t[:W]).reshape((2 * n_samples,) + shape)[:rows]
    zr = np.concatenate([z[:, 0], z[:, W - 1]])[:rows]
    tr = np.concatenate([np.full(n_samples, t[0]), np.full(n_samples, t[W - 1])])[:rows]
    _, cache = model.forward(zr, tr, txt)
    model.vjp(cache, cot)
    sec = time.perf_counter() - t0
    if scale == 1.0:
        desc = (f"one JAGG window (W={W}) of {wl.name} for {n_samples} of the G={wl.G} samples: step signals, "
                f"aggregation, endpoint forwards with caches and the joint VJP over {rows} rows")
    else:
        kind = "Flux-style single block" if sub.depth else "double-stream block"
        desc = (f"{rows} endpoint row of {wl.name} through one {kind} at full width and {wl.n_tok} tokens "
                f"(+ embeddings, final layer, one window's step signals and aggregation): forward with caches "
                f"and VJP, {sec:.1f} s measured, scaled by algorithmic FLOPs x{scale:.1f} to one sample's JAGG "
                f"window (2 endpoint rows through all {wl.depth_double} double + {wl.depth} single blocks)")
    return sec, n_samples * W, sec * scale, desc


def threads_used():
    try:
        from threadpoolctl import threadpool_info
        n = [i.get("num_threads") for i in threadpool_info() if i.get("internal_api") in ("openblas", "mkl", "blis")]
        if n:
            return int(max(n))
    except Exception:
        pass
    return os.cpu_count() or 1


def run_reference(args, ws, rank):
    """The reference arm: the float64 oracle on the host cores, each step one bounded sample
    of the workload (oracle_sample), rank 0 only."""
    if rank != 0:
        return
    wl = workload(args)
    for _ in range(args.warmup):
        oracle_sample(wl)
    tot, units, measured = 0.0, 0, 0.0
    for _ in range(args.steps):
        sec, u, scaled, desc = oracle_sample(wl)
        measured += sec
        tot += scaled
        units += u
    value = units / tot
    cores = threads_used()
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * tot / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": describe(wl)},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": desc,
                             "measured_s_per_step": measured / args.steps},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ----------------------------------------------------------------------------- main leg
def measure(b, routes, batched, args, ws, use_graph, profile=False):
    """Device time of Phases 2-4 of one group step.

    batched: one saved arena holding every window's rows and one joint VJP per group;
    otherwise one arena and one joint VJP per window.  When every window's arena fits in
    device memory at once, the whole step is one timed region; otherwise (MMDiT widths,
    full-W) each window is timed with its own arena resident and the window times add,
    the gradient norm counted once."""
    jg = b.jg
    res = {"ms": 0.0, "launches": 0, "prof": {}, "rows": 0, "vjps": 0, "saved_gb": 0.0, "resident": True}

    def run_part(arenas, reduce):
        n0 = jg.launch_count()
        b.step(arenas, reduce)
        torch.cuda.synchronize()
        res["launches"] += jg.launch_count() - n0
        assert jg.device_status() == 0, "device status set during the step"
        ms, graph = time_steps(lambda: b.step(arenas, reduce), args.steps, args.warmup, ws, use_graph)
        del graph
        res["ms"] += ms
        res["rows"] = max(res["rows"], max(a[1] for a in arenas))
        res["vjps"] += len(arenas)
        res["saved_gb"] = max(res["saved_gb"], sum(a[0].numel() for a in arenas) / 1e9)
        if profile:  # per-family device time of the same work (events around each launch, eager)
            jg.profile_enable(True)
            for _ in range(args.steps):
                b.step(arenas, reduce)
            for k, v in jg.profile_read().items():
                acc = res["prof"].setdefault(k, {"launches": 0.0, "ms": 0.0, "flops": 0.0, "bytes": 0.0})
                for q in acc:
                    acc[q] += v[q] / args.steps
            jg.profile_enable(False)

    if batched or b.fits(routes, batched=False):
        run_part(b.forward_saves(routes, batched=batched), True)
    else:
        res["resident"] = False
        for w in range(b.nw):
            arenas = b.forward_saves(routes, batched=False, windows=[w])
            run_part(arenas, w == b.nw - 1)
            del arenas
            torch.cuda.empty_cache()
    res["ms"] = max_over_ranks(res["ms"], ws)
    return res


def graph_variants(b, args, ws, use_graph):
    """The sequential-graph variant (Algorithm 2: per window, endpoint 0 forward into one
    G-row arena, its VJP, endpoint W-1 forward into the same arena, its VJP) against the
    joint variant (one 2G-row forward and VJP per window), same scope: the endpoint forwards
    with saves and the VJPs, on the cotangents of the JAGG step (signals excluded, they are
    the same for both)."""
    jg, wl, dev = b.jg, b.wl, b.dev
    G, W = wl.G, wl.W
    rows = [b.rows(b.z[:, w * W:(w + 1) * W].reshape(G, W, *b.shape), w, True) for w in range(b.nw)]
    txt1, txt2 = b.txt_rows(G), b.txt_rows(2 * G)
    arena = jg.alloc_bytes(b.model.saved_bytes(G), dev)
    v1 = torch.empty(G, *b.shape, dtype=b.tdt, device=dev)

    def sequential():
        for w, (z, t) in enumerate(rows):
            for e in range(2):
                sl = slice(e * G, (e + 1) * G)
                jg.dit_forward_save(b.model, z[sl], t[sl], txt1, v1, saved=arena, ws=b.ws)
                jg.dit_joint_vjp(b.model, arena, G, b.cot_all[w * 2 * G + e * G:w * 2 * G + (e + 1) * G], b.grad,
                                 b.ws)
    ms_s, graph = time_steps(sequential, args.steps, args.warmup, ws, use_graph)
    del graph
    seq_gb = arena.numel() / 1e9
    del arena
    torch.cuda.empty_cache()
    arena2 = jg.alloc_bytes(b.model.saved_bytes(2 * G), dev)
    v2 = torch.empty(2 * G, *b.shape, dtype=b.tdt, device=dev)

    def joint():
        for w, (z, t) in enumerate(rows):
            jg.dit_forward_save(b.model, z, t, txt2, v2, saved=arena2, ws=b.ws)
            jg.dit_joint_vjp(b.model, arena2, 2 * G, b.cot_all[w * 2 * G:(w + 1) * 2 * G], b.grad, b.ws)
    ms_j, graph = time_steps(joint, args.steps, args.warmup, ws, use_graph)
    del graph
    joint_gb = arena2.numel() / 1e9
    del arena2
    torch.cuda.empty_cache()
    units = wl.G * wl.T
    return {"sequential": {"value": ws * units / (ms_s / 1000.0), "unit": UNIT, "ms_per_step": max_over_ranks(ms_s, ws),
                           "saved_gb": seq_gb},
            "joint": {"value": ws * units / (ms_j / 1000.0), "unit": UNIT, "ms_per_step": max_over_ranks(ms_j, ws),
                      "saved_gb": joint_gb},
            "scope": "per window: endpoint forwards with saves + VJPs on the JAGG cotangents (signals excluded)"}


def ablate_step(b, args, ws, use_graph, batched, steps, warmup):
    """The endpoint-only ablation (Sec. 4): per window the step signals, then s_0 and s_{W-1}
    read in place as the two cotangent rows (no t-weighting), then the joint VJP(s) over the
    endpoint rows, batched like the headline -- the headline step with the aggregation
    swapped.  None when the endpoint arenas do not fit at once."""
    jg, wl, dev = b.jg, b.wl, b.dev
    G, W, D = wl.G, wl.W, b.D
    routes = [1] * b.nw
    if not (batched or b.fits(routes, batched=False)):
        return None
    arenas = b.forward_saves(routes, batched=batched)
    s_win = torch.empty(G, W, D, dtype=torch.float32, device=dev)

    def step():
        for saved, B, pl in arenas:
            row0 = pl[0][2]
            for (w, _, r, _) in pl:
                b.signals(w, b.lpo_win[w], s_out=s_win)
                tw = b.t_dev[w * W:(w + 1) * W]
                cot = b.cot_all[r:r + 2 * G]
                t0, t1 = float(b.t[w * W]), float(b.t[w * W + W - 1])
                jg.jagg_aggregate_span(s_win, tw[:1], t0, t1, cot, steps=(0, 1))
                jg.jagg_aggregate_span(s_win, tw[W - 1:], t0, t1, cot, accumulate=True, steps=(W - 1, 1))
            jg.dit_joint_vjp(b.model, saved, B, b.cot_all[row0:row0 + B], b.grad, b.ws)
        jg.grad_reduce(b.grad, None, out3=b.out3, ws=b.gws)
    ms, graph = time_steps(step, steps, warmup, ws, use_graph)
    del graph, arenas
    torch.cuda.empty_cache()
    return {"value": ws * wl.G * wl.T / (ms / 1000.0), "unit": UNIT, "ms_per_step": max_over_ranks(ms, ws),
            "steps": steps, "warmup": warmup}


def flops_per_sequence(wl):
    """Algorithmic FLOPs (2 per multiply-add) of one sequence through the backbone:
    (forward, backward).  Per block the four dense products of every token (4 d^2 + 2 d dm
    multiply-adds: qkv, proj, fc1, fc2 -- or lin1, lin2 of a single block), attention
    4 N^2 d, the modulation product; embeddings and final layer.  Backward: the input and
    weight gradients of every product (2x, weight gradient only for the input embeddings,
    which pass no gradient to z or the text), 8 N^2 d for attention (recomputing S is not
    counted)."""
    d, dm, N = wl.hidden, wl.mlp, wl.n_tok
    blocks = wl.depth + wl.depth_double
    lin = 2.0 * N * (4 * d * d + 2 * d * dm)
    att = 4.0 * N * N * d
    mod_rows = (6 * d * wl.depth if wl.arch == "dit" else 12 * d * wl.depth_double + 3 * d * wl.depth) + 2 * d
    mod = 2.0 * d * mod_rows + 2.0 * (wl.freq_dim * d + d * d)
    emb_in = 2.0 * d * (wl.n_img * wl.patch_dim + wl.txt_len * wl.txt_dim)
    emb_out = 2.0 * d * wl.n_img * wl.patch_dim
    fwd = blocks * (lin + att) + mod + emb_in + emb_out
    bwd = blocks * (2 * lin + 2 * att) + 2 * mod + emb_in + 2 * emb_out
    return fwd, bwd


def family_roofline(fam, name, peak, src, label):
    """Roofline object of one kernel family over the step's launches: algorithmic FLOPs
    per launch over its average launch duration (events around each launch)."""
    f = fam.get(name, {"launches": 0, "ms": 0.0, "flops": 0.0, "bytes": 0.0})
    n = max(f["launches"], 1)
    achieved = f["flops"] / (f["ms"] / 1000.0) / 1e12 if f["ms"] > 0 else 0.0
    return {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s", "frac": achieved / peak,
            "kernel": label, "peak_source": src, "launches_per_step": f["launches"],
            "flops_per_launch": f["flops"] / n, "algorithmic_bytes_per_launch": f.get("bytes", 0.0) / n,
            "ms_per_launch": f["ms"] / n}


def run_gpu(args, ws, rank):
    import paper_2607_17572_gb300 as jg
    dev = torch.device("cuda", torch.cuda.current_device())
    wl = workload(args)
    b = Bench(wl, dev)
    b.rollout()
    routes, _ = jg.jagg_route(b.nw, wl.jagg_frac)
    batched = b.batch_group(routes, args.vjp_rows)
    use_graph = not args.no_graph
    units = wl.G * wl.T
    # the legs beside the headline: at most 5 timed steps on the MMDiT widths (seconds each)
    leg_steps = args.steps if wl.arch == "dit" else min(args.steps, 5)
    leg_warm = max(3, args.warmup) if wl.arch == "dit" else 3
    lg = argparse.Namespace(steps=leg_steps, warmup=leg_warm)

    # ---- JAGG path: timed region, then the per-family breakdown of the same work
    with ClockSampler(torch.cuda.current_device()) as clk:
        r = measure(b, routes, batched, args, ws, use_graph, profile=True)
    clocks = clk.summary()
    ms = r["ms"]
    value = job_rate(units, ms, ws)
    burst, sustained, hbm, src = peaks()
    fam = {k: v for k, v in r["prof"].items() if v["launches"]}
    # the products and attention run back to back for the seconds of a step: sustained peak
    psrc = f"bf16_tflops_sustained of {src} peaks"
    roofline = family_roofline(fam, "gemm_tcgen05", sustained, psrc,
                               "gemm_tc_kernel (all dense products of the joint VJP)")
    ratio = TRAFFIC_RATIO.get(wl.name)
    roofline["traffic"] = ratio * roofline["algorithmic_bytes_per_launch"] if ratio else None
    roofline["frac_of_burst"] = roofline["achieved"] / burst
    att = family_roofline(fam, "attention_bwd", sustained, psrc,
                          f"fa_bwd_tc{wl.head_dim}_kernel (attention backward)")
    att["frac_of_burst"] = att["achieved"] / burst
    step_flops = sum(v["flops"] for k, v in fam.items() if k != "gemm_simt")
    families = {k: {"launches_per_step": v["launches"], "ms_per_step": v["ms"],
                    "tflops": (v["flops"] / (v["ms"] / 1000.0) / 1e12) if v["ms"] > 0 else None,
                    "algorithmic_gb_per_step": v["bytes"] / 1e9,
                    "gbs": (v["bytes"] / (v["ms"] / 1000.0) / 1e9) if v["ms"] > 0 else None}
                for k, v in fam.items()}
    if batched:
        batching = f"one joint VJP per group over all {b.nw} windows' endpoint rows"
    else:
        batching = f"one joint VJP per window ({b.nw} per step)" + (
            ", every window's saved activations resident" if r["resident"] else
            ", each window timed with its own saved activations resident, the window times added")
    out = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
           "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
           "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
           "config": {"workload": describe(wl), "rows_per_vjp": r["rows"], "windows": b.nw,
                      "cuda_graph": use_graph, "vjp_batching": batching,
                      "l2": "inputs larger than L2 (saved activations %.1f GB resident)" % r["saved_gb"],
                      "memory_plan": getattr(b, "last_fit", None),
                      "parallelism": f"replicas x{ws}" if ws > 1 else "single GPU"},
           "roofline": roofline, "roofline_attention_bwd": att,
           "algorithmic_tflops_per_step": step_flops / 1e12,
           "step_tflops_per_s": step_flops / (ms / 1000.0) / 1e12, "families": families,
           "gpu_launches": r["launches"] * args.steps, "clocks": clocks}
    torch.cuda.empty_cache()

    if not args.quick:
        # ---- the same JAGG step with one joint VJP per window (Algorithm 1 as written)
        if batched:
            rw = measure(b, routes, False, lg, ws, use_graph)
            out["per_window_vjp"] = {"value": ws * units / (rw["ms"] / 1000.0), "unit": UNIT,
                                     "ms_per_step": rw["ms"], "rows_per_vjp": rw["rows"], "vjps_per_step": rw["vjps"]}
        # ---- exact per-step path (jagg_frac = 0), batched like the headline when it fits
        full = [0] * b.nw
        rf = measure(b, full, b.batch_group(full, args.vjp_rows), lg, ws, use_graph)
        out["full_w"] = {"value": ws * units / (rf["ms"] / 1000.0), "unit": UNIT, "ms_per_step": rf["ms"],
                         "rows_per_vjp": rf["rows"], "vjps_per_step": rf["vjps"], "steps": lg.steps,
                         "resident": ("every window" if rf["resident"] else
                                      "one window at a time, the window times added")}
        out["jagg_speedup_vs_full_w"] = rf["ms"] / ms
        out["ideal_speedup"] = wl.W / 2
        torch.cuda.empty_cache()
        out["graph_variants"] = graph_variants(b, lg, ws, use_graph)
        ab = ablate_step(b, args, ws, use_graph, batched, lg.steps, lg.warmup)
        if ab is not None:
            out["ablate"] = ab
        out["update_stage"] = update_stage(b, args, ws, use_graph, lg.steps, lg.warmup)
        out["rollout"] = rollout_leg(b, lg, ws, use_graph)
    if not args.no_e2e:
        out["e2e"] = run_e2e(b, args, ws, routes, steps=lg.steps, warmup=lg.warmup)
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        sec, u, scaled, desc = oracle_sample(wl)
        out["cpu_baseline"] = {"value": u / scaled, "unit": UNIT, "cores": threads_used(), "kind": "oracle",
                               "sample": desc, "measured_s": sec}
    if rank == 0:
        print(json.dumps(out), flush=True)


def update_chunks(b, routes):
    """Windows per Phase-4 call of the update stage: every window at once when the group's
    saved activations fit (one arena, one joint VJP over the group), else one window at a
    time through one arena (Algorithm 1's loop over windows)."""
    G, W = b.wl.G, b.wl.W
    mid = sum((W - 2) * G for w in range(b.nw) if routes[w])
    if b.fits(routes, batched=True) and mid <= b.ws_rows:
        return [list(range(b.nw))]
    return [[w] for w in range(b.nw)]


def update_step(b, routes, host):
    """The update stage of one group (the paper's "update": forwards on the stored
    experience, then the backward).  Per window routed to JAGG: the endpoint forwards with
    saves, the middle steps' forwards without, the step signals with the aggregation, the
    joint VJP over the 2G endpoint rows; per exact window: every step's forward with saves,
    each step's own signal, the VJP over its W*G rows.  Windows share one VJP call when the
    group's saved activations fit (update_chunks).  After the last window, the gradient's
    squared norm.  host=True: the step starts by copying the group's trajectory, old
    log-probs and rewards from pinned host buffers and ends by reading the new log-probs
    and the gradient norm back.  Returns (step, h2d bytes, d2h bytes)."""
    jg, wl, dev = b.jg, b.wl, b.dev
    G, W, D = wl.G, wl.W, b.D
    h_z = b.z.cpu().pin_memory()
    h_lpo = b.logp_old.cpu().pin_memory()
    h_rw = b.rewards.cpu().pin_memory()
    h_lpn = torch.empty(G, wl.T, dtype=torch.float64).pin_memory()
    h_out3 = torch.empty(3, dtype=torch.float64).pin_memory()
    chunks = update_chunks(b, routes)

    def rows_of(c):
        sv = sum(2 * G if routes[w] else W * G for w in c)
        mid = sum((W - 2) * G for w in c if routes[w])
        return sv, mid
    n_sv = max(rows_of(c)[0] for c in chunks)
    n_mid = max(max(rows_of(c)[1] for c in chunks), 1)
    saved = jg.alloc_bytes(b.model.saved_bytes(n_sv), dev)
    z_sv = torch.empty(n_sv, *b.shape, dtype=b.tdt, device=dev)
    v_sv = torch.empty_like(z_sv)
    z_mid = torch.empty(n_mid, *b.shape, dtype=b.tdt, device=dev)
    v_mid = torch.empty_like(z_mid)
    txt_sv, txt_mid = b.txt_rows(n_sv), b.txt_rows(n_mid)
    t_sv, t_mid = [], []
    for c in chunks:
        ts, tm = [], []
        for w in c:
            tw = b.t[w * W:(w + 1) * W]
            if routes[w]:
                ts.append(np.repeat([tw[0], tw[W - 1]], G))
                tm.append(np.tile(tw[1:W - 1], G))
            else:
                ts.append(np.tile(tw, G))       # sample-major, matching s [G, W, D]
        t_sv.append(torch.tensor(np.concatenate(ts), dtype=torch.float32, device=dev))
        t_mid.append(torch.tensor(np.concatenate(tm), dtype=torch.float32, device=dev) if tm else None)

    def step():
        if host:
            b.z.copy_(h_z, non_blocking=True)
            b.logp_old.copy_(h_lpo, non_blocking=True)
            b.rewards.copy_(h_rw, non_blocking=True)
        for ci, c in enumerate(chunks):
            r = m = 0
            for w in c:
                zw = b.z[:, w * W:(w + 1) * W].reshape(G, W, *b.shape)
                if routes[w]:
                    z_sv[r:r + G].copy_(zw[:, 0])
                    z_sv[r + G:r + 2 * G].copy_(zw[:, W - 1])
                    r += 2 * G
                    if W > 2:
                        z_mid[m:m + (W - 2) * G].copy_(zw[:, 1:W - 1].reshape(-1, *b.shape))
                        m += (W - 2) * G
                else:
                    z_sv[r:r + W * G].copy_(zw.reshape(G * W, *b.shape))
                    r += W * G
            # Phase 1: saved rows (endpoints, or every step of an exact window), middle steps without saves
            jg.dit_forward_save(b.model, z_sv[:r], t_sv[ci], txt_sv[:r], v_sv[:r], saved=saved, ws=b.ws)
            if m:
                jg.dit_forward_save(b.model, z_mid[:m], t_mid[ci], txt_mid[:m], v_mid[:m], ws=b.ws)
            r = m = 0
            for w in c:
                b.z_win[w].copy_(b.z[:, w * W:w * W + W + 1])
                b.lpo_win[w].copy_(b.logp_old[:, w * W:(w + 1) * W])
                vw = b.v_win[w]
                if routes[w]:
                    vw[:, 0].copy_(v_sv[r:r + G].reshape(G, -1))
                    vw[:, W - 1].copy_(v_sv[r + G:r + 2 * G].reshape(G, -1))
                    if W > 2:
                        vw[:, 1:W - 1].copy_(v_mid[m:m + (W - 2) * G].reshape(G, W - 2, -1))
                        m += (W - 2) * G
                    # Phases 2-3
                    b.signals(w, b.lpo_win[w], cot_out=b.cot_all[r:r + 2 * G])
                    r += 2 * G
                else:
                    vw.copy_(v_sv[r:r + W * G].reshape(G, W, D))
                    b.signals(w, b.lpo_win[w], s_out=b.cot_all[r:r + W * G].view(G, W, D))
                    r += W * G
                if host:
                    h_lpn[:, w * W:(w + 1) * W].copy_(b.sig_out["logp_new"], non_blocking=True)
            # Phase 4
            jg.dit_joint_vjp(b.model, saved, r, b.cot_all[:r], b.grad, b.ws)
        jg.grad_reduce(b.grad, None, out3=b.out3, ws=b.gws)
        if host:
            h_out3.copy_(b.out3, non_blocking=True)
            torch.cuda.current_stream().synchronize()

    h2d = h_z.numel() * 4 + h_lpo.numel() * 8 + h_rw.numel() * 4
    d2h = h_lpn.numel() * 8 + h_out3.numel() * 8
    return step, h2d, d2h, len(chunks) == 1


def update_stage(b, args, ws, use_graph, steps, warmup):
    """The update time the paper reports for its efficiency analysis (forwards on the stored
    experience + backward), device-resident, JAGG against the exact per-step path."""
    wl = b.wl
    units = wl.G * wl.T
    lg = argparse.Namespace(steps=steps, warmup=warmup)
    step, _, _, one = update_step(b, [1] * b.nw, host=False)
    ms_j, graph = time_steps(step, lg.steps, lg.warmup, ws, use_graph)
    del graph, step
    torch.cuda.empty_cache()
    out = {"jagg": {"value": ws * units / (ms_j / 1000.0), "unit": UNIT, "ms_per_step": max_over_ranks(ms_j, ws),
                    "vjp_calls": 1 if one else b.nw}}
    fstep, _, _, one = update_step(b, [0] * b.nw, host=False)
    ms_f, graph = time_steps(fstep, lg.steps, lg.warmup, ws, use_graph)
    del graph, fstep
    torch.cuda.empty_cache()
    out["full_w"] = {"value": ws * units / (ms_f / 1000.0), "unit": UNIT, "ms_per_step": max_over_ranks(ms_f, ws),
                     "vjp_calls": 1 if one else b.nw}
    out["speedup"] = ms_f / ms_j
    # forward = 1 unit, backward = 2: W * 3 units exact against W + 2 * 2 with JAGG
    out["ideal_speedup"] = 3.0 * wl.W / (wl.W + 4.0)
    out["steps"], out["warmup"] = steps, warmup
    out["scope"] = ("per group: the forwards on the stored trajectories (JAGG: endpoints saved, middle steps "
                    "without; exact: every step saved), the step signals, the VJP(s), the gradient norm")
    return out


def rollout_leg(b, args, ws, use_graph):
    """The rollout sampler on the device: per step the G forwards without saves and the fused
    sampler step; G * T trajectory-steps per run."""
    wl = b.wl
    run, _, _, _ = b.sampler()
    ms, graph = time_steps(run, args.steps, args.warmup, ws, use_graph)
    del graph
    return {"value": ws * wl.G * wl.T / (ms / 1000.0), "unit": "trajectory-steps/s (sampled)",
            "ms_per_step": max_over_ranks(ms, ws)}


def run_e2e(b, args, ws, routes, steps, warmup):
    """The JAGG update stage through the public API from pinned host buffers (update_step
    with host=True), timed on the host clock."""
    wl = b.wl
    step, h2d, d2h, one = update_step(b, routes, host=True)
    for _ in range(warmup):
        step()
    barrier(ws)
    t0 = time.perf_counter()
    for _ in range(steps):
        step()
    sec = max_over_ranks((time.perf_counter() - t0) / steps, ws)
    del step
    torch.cuda.empty_cache()
    return {"value": ws * wl.G * wl.T / sec, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "ms_per_step": 1000 * sec, "steps": steps, "warmup": warmup,
            "includes": ("H2D of the group's trajectory, old log-probs and rewards; per window the Phase 1 "
                         "forwards (2G endpoint rows saved, (W-2)G middle rows unsaved), signals with aggregation; "
                         + ("one joint VJP over the group" if one else "one joint VJP per window") +
                         "; gradient norm; D2H of the new log-probs and the norm")}


def window_cosines(b):
    """Per window, the cosine between its JAGG gradient (the 2G endpoint rows with the
    aggregated cotangents) and its exact per-step gradient (all W*G rows with their own
    s_j), each accumulated into its own zeroed buffer and compared by grad_reduce: the
    quantity the gradient-quality appendix routes on (cos >= 0.5)."""
    jg, wl, dev = b.jg, b.wl, b.dev
    G, W, D = wl.G, wl.W, b.D
    g_j = torch.empty(b.P, dtype=torch.float32, device=dev)
    g_e = torch.empty(b.P, dtype=torch.float32, device=dev)
    out3 = torch.empty(3, dtype=torch.float64, device=dev)
    cos = []
    for w in range(b.nw):
        g_j.zero_()
        g_e.zero_()
        zw = b.z[:, w * W:(w + 1) * W].reshape(G, W, *b.shape)
        for jagg, g in ((True, g_j), (False, g_e)):
            z, t = b.rows(zw, w, jagg)
            B = z.shape[0]
            saved = jg.alloc_bytes(b.model.saved_bytes(B), dev)
            v = torch.empty_like(z)
            jg.dit_forward_save(b.model, z, t, b.txt_rows(B), v, saved=saved, ws=b.ws)
            cot = b.cot_all[:B]
            if jagg:
                b.signals(w, b.lpo_win[w], cot_out=cot)
            else:
                b.signals(w, b.lpo_win[w], s_out=cot.view(G, W, D))
            jg.dit_joint_vjp(b.model, saved, B, cot, g, b.ws)
            torch.cuda.synchronize()
            del saved, v
        jg.grad_reduce(g_j, g_e, out3=out3, ws=b.gws)
        ab, aa, bb = out3.tolist()
        cos.append(ab / (aa * bb) ** 0.5 if aa > 0 and bb > 0 else 0.0)
    del g_j, g_e
    torch.cuda.empty_cache()
    return cos


def run_sweep(args, ws, rank):
    """The routing and window sweep on the Qwen-width MMDiT (8 double-stream blocks, d = 3072,
    1024 image + 256 text tokens, G = 8, T = 16): for W in {2, 4, 8} and jagg_frac in
    {0, 0.5, 1} (schedule routing, n_jagg = floor(jagg_frac n_w)), the group step of
    Phases 2-4 with one joint VJP per window (Algorithm 1), every window's saved activations
    resident; the speed-up over jagg_frac = 0 against the ideal ratio of VJP rows (W/2 when
    every window is routed); per window the cosine between the JAGG and exact gradients
    and the routes the calibration rule (cos >= 0.5) derives from them."""
    import paper_2607_17572_gb300 as jg
    dev = torch.device("cuda", torch.cuda.current_device())
    base = workload(args)
    use_graph = not args.no_graph
    burst, sustained, hbm, src = peaks()
    table, t_start = {}, time.perf_counter()
    with ClockSampler(torch.cuda.current_device()) as clk:
        for W in (2, 4, 8):
            wl = synth.small_variant(base, W=W)
            b = Bench(wl, dev)
            b.rollout()
            cells = {}
            for frac in (0.0, 0.5, 1.0):
                routes, _ = jg.jagg_route(b.nw, frac)
                r = measure(b, routes, False, args, ws, use_graph)
                rows = sum(2 * wl.G if x else W * wl.G for x in routes)
                cells[str(frac)] = {"value": job_rate(wl.G * wl.T, r["ms"], ws), "ms_per_step": r["ms"],
                                    "routes": routes, "vjp_rows_per_step": rows,
                                    "resident": r["resident"]}
                torch.cuda.empty_cache()
            full_rows = cells["0.0"]["vjp_rows_per_step"]
            for c in cells.values():
                c["speedup_vs_full_w"] = cells["0.0"]["ms_per_step"] / c["ms_per_step"]
                c["ideal_speedup"] = full_rows / c["vjp_rows_per_step"]
            cos = window_cosines(b)
            calib, derived = jg.jagg_route(b.nw, 1.0, cos=cos, tau=0.5)
            table[f"W={W}"] = {"windows": b.nw, "cells": cells, "window_cos": cos, "calibrated_routes": calib,
                               "derived_jagg_frac": derived}
            del b
            torch.cuda.empty_cache()
    if rank == 0:
        print(json.dumps({"metric": METRIC, "unit": UNIT, "sweep": "W x jagg_frac", "workload": describe(base),
                          "steps": args.steps, "warmup": args.warmup, "cuda_graph": use_graph, "table": table,
                          "clocks": clk.summary(), "wall_s": time.perf_counter() - t_start}), flush=True)


def run_kernel_attention_bwd(args):
    """The attention backward (or forward) alone on the workload's joint attention (B sequences, the
    text and image streams in their own buffers as in the MMDiT double blocks), timed with
    CUDA events over the timed calls; the kernel's own device time comes from the
    library's per-launch events."""
    import paper_2607_17572_gb300 as jg
    wl = workload(args)
    dev = torch.device("cuda", torch.cuda.current_device())
    B = args.rows or 2 * wl.G
    N, H, dh = wl.n_tok, wl.heads, wl.head_dim
    n0 = wl.txt_len if wl.arch == "mmdit" else N
    d = H * dh
    gen = torch.Generator(device=dev).manual_seed(synth.NOISE_SEED)
    qkv = (torch.randn(B * N, 3 * d, device=dev, generator=gen) * 1.5).bfloat16()
    o = torch.empty(B * N, d, device=dev, dtype=torch.bfloat16)
    lse = torch.empty(B, H, N, device=dev)
    jg.test_attention_fwd(qkv, B, N, H, dh, o, lse)
    dO = torch.randn(B * N, d, device=dev, generator=gen).bfloat16()

    def split(x):
        x = x.view(B, N, -1)
        return x[:, :n0].contiguous(), x[:, n0:].contiguous()
    views = (split(qkv), split(o), split(dO))
    dq = (torch.empty(B, n0, 3 * d, device=dev, dtype=torch.bfloat16),
          torch.empty(B, N - n0, 3 * d, device=dev, dtype=torch.bfloat16))
    fwd = args.kernel == "attention_fwd"
    family = "attention_fwd" if fwd else "attention_bwd"
    if fwd:  # the forward on the same views: o and lse rewritten each call
        call = lambda: jg.test_attention_fwd_streams(views[0], views[1], lse, B, N, n0, H, dh)
    else:
        call = lambda: jg.test_attention_bwd_streams(views[0], views[1], lse, views[2], B, N, n0, H, dh, dq)
    for _ in range(args.warmup):
        call()
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.profiler.start()
    e0.record(stream)
    for _ in range(args.steps):
        call()
    e1.record(stream)
    torch.cuda.synchronize()
    torch.cuda.profiler.stop()
    ms = e0.elapsed_time(e1) / args.steps
    jg.profile_enable(True)
    for _ in range(args.steps):
        call()
    prof = jg.profile_read()
    jg.profile_enable(False)
    fam = prof[family]
    flops = (4.0 if fwd else 8.0) * B * H * N * N * dh
    kms = fam["ms"] / max(fam["launches"], 1)
    burst, sustained, hbm, src = peaks()
    tf = flops / (kms / 1000.0) / 1e12
    print(json.dumps({"kernel": family, "workload": describe(wl), "rows": B, "heads": H, "head_dim": dh,
                      "tokens": N, "text_tokens": n0 if n0 < N else 0, "steps": args.steps,
                      "ms_per_call": ms, "kernel_ms": kms, "algorithmic_tflop": flops / 1e12,
                      "roofline": {"bound": "tensor", "achieved": tf, "peak": burst, "unit": "TFLOP/s",
                                   "frac": tf / burst, "peak_source": f"bf16_tflops (burst) of {src} peaks"},
                      "aux_ms_per_call": 0.0 if fwd else prof["attention_bwd_aux"]["ms"] / args.steps}), flush=True)


def gemm_products(wl, rows):
    """The dense products of one block's backward at `rows` token rows, in the operand layouts
    of the joint VJP: name -> (M, N, K, a_mn, b_mn, epilogue).  Input gradients dX = dY W
    (K-major dY, MN-major W; the ones into GELU's input times GELU'(u), the multiplier
    epilogue), weight gradients dW += dY^T X (both MN-major, f32 accumulation).  DiT: one
    block.  MMDiT: a Flux-style single block at the joint rows (lin2's two input-gradient
    parts, [o] and [GELU(u)]; lin1 over [qkv | u]) and a double block's image-stream
    products at its image rows."""
    d, f = wl.hidden, wl.mlp

    def block(r, pre=""):
        return {pre + "fc2_dx": (r, f, d, False, True, "mul_aux"), pre + "fc1_dx": (r, d, f, False, True, "store"),
                pre + "qkv_dx": (r, d, 3 * d, False, True, "store"), pre + "proj_dx": (r, d, d, False, True, "store"),
                pre + "fc2_dw": (d, f, r, True, True, "accum"), pre + "fc1_dw": (f, d, r, True, True, "accum"),
                pre + "qkv_dw": (3 * d, d, r, True, True, "accum"), pre + "proj_dw": (d, d, r, True, True, "accum")}
    if wl.arch == "dit":
        return block(rows)
    out = {}
    if wl.depth:
        out.update({"lin2_dx_o": (rows, d, d, False, True, "store"),
                    "lin2_dx_u": (rows, f, d, False, True, "mul_aux"),
                    "lin1_dx": (rows, d, 3 * d + f, False, True, "store"),
                    "lin2_dw": (d, d + f, rows, True, True, "accum"),
                    "lin1_dw": (3 * d + f, d, rows, True, True, "accum")})
    if wl.depth_double:
        out.update(block(rows * wl.n_img // wl.n_tok, "img_"))
    return out


def run_kernel_gemm(args):
    """The block's backward products alone at the step's VJP rows (2G rows per window, every
    window: the joint VJP's token rows), each timed with CUDA events over the timed calls and
    by the library's per-launch events, on random bf16 operands (a few hundred MB at most)."""
    import paper_2607_17572_gb300 as jg
    wl = workload(args)
    dev = torch.device("cuda", torch.cuda.current_device())
    rows = (args.rows or 2 * wl.G * (wl.T // wl.W)) * wl.n_tok
    prods = gemm_products(wl, rows)
    names = list(prods) if args.product == "all" else [args.product]
    gen = torch.Generator(device=dev).manual_seed(synth.NOISE_SEED)
    burst, sustained, hbm, src = peaks()
    out = {}
    for name in names:
        M, N, K, a_mn, b_mn, epi = prods[name]
        A = torch.randn(K, M, device=dev, generator=gen).bfloat16() if a_mn else \
            torch.randn(M, K, device=dev, generator=gen).bfloat16()
        B = (torch.randn(K, N, device=dev, generator=gen) if b_mn else
             torch.randn(N, K, device=dev, generator=gen)).mul_(K ** -0.5).bfloat16()
        d = jg.GemmDesc()
        d.M, d.N, d.K = M, N, K
        d.A, d.lda, d.a_mn, d.a_dtype = A.data_ptr(), M if a_mn else K, int(a_mn), jg.DTYPE_BF16
        d.B, d.ldb, d.b_mn, d.b_dtype = B.data_ptr(), N if b_mn else K, int(b_mn), jg.DTYPE_BF16
        d.rows_per_seq = 1
        keep = [A, B]
        if epi == "accum":
            C = torch.zeros(M, N, device=dev)
            d.epi, d.C, d.ldc, d.c_dtype = 4, C.data_ptr(), N, jg.DTYPE_F32
        else:
            C = torch.empty(M, N, device=dev, dtype=torch.bfloat16)
            d.epi, d.C, d.ldc, d.c_dtype = (3 if epi == "mul_aux" else 0), C.data_ptr(), N, jg.DTYPE_BF16
            if epi == "mul_aux":
                X = torch.rand(M, N, device=dev, generator=gen).bfloat16()
                d.aux, d.ld_aux = X.data_ptr(), N
                keep.append(X)
        keep.append(C)
        call = lambda: jg.test_gemm(d)
        for _ in range(args.warmup):
            call()
        torch.cuda.synchronize()
        stream = torch.cuda.current_stream()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.profiler.start()
        e0.record(stream)
        for _ in range(args.steps):
            call()
        e1.record(stream)
        torch.cuda.synchronize()
        torch.cuda.profiler.stop()
        ms = e0.elapsed_time(e1) / args.steps
        jg.profile_enable(True)
        for _ in range(args.steps):
            call()
        fam = jg.profile_read()["gemm_tcgen05"]
        jg.profile_enable(False)
        kms = fam["ms"] / max(fam["launches"], 1)
        tf = 2.0 * M * N * K / (kms / 1000.0) / 1e12
        out[name] = {"M": M, "N": N, "K": K, "epilogue": epi, "ms_per_call": ms, "kernel_ms": kms, "tflops": tf,
                     "frac_of_burst": tf / burst}
        del keep, C
        torch.cuda.empty_cache()
    print(json.dumps({"kernel": "gemm", "workload": describe(wl), "rows": rows, "steps": args.steps,
                      "peak": {"tflops": burst, "source": f"bf16_tflops (burst) of {src} peaks"},
                      "products": out}), flush=True)


def run_kernel_hbm(args):
    """The bandwidth-bound kernels of the joint VJP alone at the workload's per-window shapes
    (rows = 2G sequences of one window by default) on random operands, each timed by the
    library's per-launch events over the timed calls and reported against the measured HBM
    copy bandwidth: the LayerNorm + modulation and gate backward (a single block's rows), the
    QK-norm + RoPE forward and backward, the bias column sums (a single block's lin1 output
    gradient), the step signals with the fused aggregation, grad_reduce (a 256 M-parameter
    slice: the norm and a dot with a second gradient).  Every operand a few hundred MB."""
    import paper_2607_17572_gb300 as jg
    wl = workload(args)
    dev = torch.device("cuda", torch.cuda.current_device())
    seqs = args.rows or 2 * wl.G
    N, d, dm, H = wl.n_tok, wl.hidden, wl.mlp, wl.heads
    M = seqs * N
    gen = torch.Generator(device=dev).manual_seed(synth.NOISE_SEED)
    bf = torch.bfloat16
    f = dict(device=dev, dtype=torch.float32)
    burst, sustained, hbm, src = peaks()
    out = {}

    def run(name, family, fn):
        for _ in range(args.warmup):
            fn()
        torch.cuda.synchronize()
        torch.cuda.profiler.start()
        jg.profile_enable(True)
        for _ in range(args.steps):
            fn()
        prof = jg.profile_read()
        jg.profile_enable(False)
        torch.cuda.profiler.stop()
        fam = prof[family]
        ms = fam["ms"] / max(fam["launches"], 1)
        gbs = fam["bytes"] / max(fam["launches"], 1) / (ms / 1000.0) / 1e9
        out[name] = {"family": family, "ms_per_launch": ms, "algorithmic_mb_per_launch": fam["bytes"] / max(fam["launches"], 1) / 1e6,
                     "gbs": gbs, "frac_of_hbm": gbs / hbm}

    # LayerNorm + modulation and gate backward over a single block's rows
    h = torch.randn(M, d, **f, generator=gen)
    mean, rstd = h.mean(1), torch.rsqrt(h.var(1, unbiased=False) + 1e-6)
    dmv = torch.randn(M, d, **f, generator=gen)
    dh = torch.randn(M, d, **f, generator=gen)
    y = torch.randn(M, d, **f, generator=gen).to(bf)
    dy = torch.empty(M, d, device=dev, dtype=bf)
    scale, gate = torch.randn(seqs, d, **f, generator=gen), torch.randn(seqs, d, **f, generator=gen)
    acc3 = [torch.zeros(seqs, d, **f) for _ in range(3)]
    dbias = torch.zeros(d, **f)
    run("ln_gate_bwd", "ln_gate_bwd",
        lambda: jg.test_ln_gate_bwd(M, d, N, dh, dh, dm=dmv, h=h, mean=mean, rstd=rstd, scale=scale, dshift=acc3[0],
                                    dscale=acc3[1], y=y, gate=gate, dgate=acc3[2], dy=dy, dbias=dbias))
    del h, mean, rstd, dmv, dh, y, dy
    torch.cuda.empty_cache()
    if wl.arch == "mmdit":
        dh_ = wl.head_dim
        qkv = (torch.randn(M, 3 * d, **f, generator=gen) * 2).to(bf)
        qs, ks = torch.ones(dh_, device=dev, dtype=bf), torch.ones(dh_, device=dev, dtype=bf)
        qk = torch.empty(M, 2 * d, device=dev, dtype=bf)
        rq, rk = torch.empty(M, H, **f), torch.empty(M, H, **f)
        gw = wl.latent_w // wl.patch
        run("qk_norm_rope_fwd", "qk_norm_rope_fwd",
            lambda: jg.test_qk_norm_rope_fwd(qkv, M, N, H, wl.txt_len, gw, qs, ks, qk, rq, rk))
        dqk = torch.randn(M, 3 * d + dm, **f, generator=gen).to(bf)
        dqs, dks = torch.zeros(dh_, **f), torch.zeros(dh_, **f)
        run("qk_norm_rope_bwd", "qk_norm_rope_bwd",
            lambda: jg.test_qk_norm_rope_bwd(qkv, M, N, H, wl.txt_len, gw, qs, ks, rq, rk, dqk, dqs, dks))
        del qkv, qk, rq, rk
        X = dqk
    else:
        X = torch.randn(M, 3 * d, **f, generator=gen).to(bf)
    db = torch.zeros(X.shape[1], **f)
    run("colsum", "colsum", lambda: jg.test_colsum(X, db))
    del X
    torch.cuda.empty_cache()
    # the step signals of one window with the fused aggregation (Phases 2-3)
    G, W, D = wl.G, wl.W, wl.D
    v = torch.randn(G, W, D, **f, generator=gen).to(bf)
    z = torch.randn(G, W + 1, D, **f, generator=gen)
    t = synth.time_grid(wl.T, wl.shift)
    sig = synth.sigma_schedule(t, wl.eta)
    f64 = dict(dtype=torch.float64, device=dev)
    so = dict(logp_new=torch.empty(G, W, **f64), ratio=torch.empty(G, W, **f64),
              clipped=torch.empty(G, W, dtype=torch.uint8, device=dev), adv_out=torch.empty(G, **f64))
    cot = torch.empty(2 * G, D, **f)
    sws = jg.alloc_bytes(jg.signals_workspace_bytes(G, W, D), dev)
    targs = (v, z, torch.tensor(t[:W + 1], **f64), torch.tensor(sig[:W], **f64), torch.zeros(G, W, **f64),
             torch.randn(G, **f, generator=gen), wl.clip_eps, wl.adv_clip, wl.adv_eps, 1.0 / (G * wl.T))
    run("step_signals", "step_signals", lambda: jg.grpo_step_signals(*targs, ws=sws, cot_out=cot, **so))
    # grad_reduce on a 256 M-parameter slice: |a|^2 and <a, b>
    P = 256 * 1024 * 1024
    ga, gb = torch.randn(P, **f, generator=gen), torch.randn(P, **f, generator=gen)
    out3 = torch.zeros(3, **f64)
    gws = jg.alloc_bytes(jg.grad_reduce_workspace_bytes(P), dev)
    run("grad_reduce_dot", "grad_reduce", lambda: jg.grad_reduce(ga, gb, out3=out3, ws=gws))
    print(json.dumps({"kernel": "hbm", "workload": describe(wl), "rows": M, "sequences": seqs, "steps": args.steps,
                      "peak": {"hbm_gbs": hbm, "source": f"hbm_gbs of {src} peaks"}, "kernels": out}), flush=True)


def main():
    args = parse()
    ws, rank = dist_setup(need_gpu=args.impl != "reference" or args.kernel is not None)
    if args.kernel in ("attention_bwd", "attention_fwd"):
        if rank == 0:
            run_kernel_attention_bwd(args)
    elif args.kernel == "gemm":
        if rank == 0:
            run_kernel_gemm(args)
    elif args.kernel == "hbm":
        if rank == 0:
            run_kernel_hbm(args)
    elif args.impl == "reference":
        run_reference(args, ws, rank)
    elif args.sweep:
        run_sweep(args, ws, rank)
    else:
        run_gpu(args, ws, rank)
    if ws > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
