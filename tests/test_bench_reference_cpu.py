"""bench.py's reference arm (the float64 oracle timed on the host cores) on CPU: one JSON
line with the contract's keys, `"impl": "reference"`, a cpu_baseline describing the run
and an e2e block with no host-device traffic."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_prints_one_contract_line():
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload",
                        "tiny_dit_f32", "--steps", "1", "--warmup", "1"], capture_output=True, text=True,
                       cwd=ROOT, env=env, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["value"] > 0 and d["higher_is_better"] is True
    for k in ("metric", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "scaling", "dtype", "data", "config"):
        assert k in d, k
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"] and cb["sample"]
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["d2h_bytes_per_step"] == 0
    assert d["e2e"]["value"] == d["value"] and d["e2e"]["unit"] == d["unit"]


def test_oracle_sample_of_an_mmdit_scales_by_the_flop_model():
    """At MMDiT widths the CPU baseline times one endpoint row through one block and scales
    the time by the FLOP model to one sample's JAGG window; the model's forward matches the
    workloads' per-sequence forward FLOPs (DiT-B 60.9 GFLOP, Flux-width 4.54 / 15.7 TFLOP)."""
    sys.path.insert(0, ROOT)
    import bench
    import synth
    fwd = {n: bench.flops_per_sequence(synth.WORKLOADS[n])[0] for n in
           ("dit_b_bf16", "mmdit_flux512_bf16", "mmdit_flux1024_bf16")}
    assert abs(fwd["dit_b_bf16"] / 60.9e9 - 1) < 5e-3
    assert abs(fwd["mmdit_flux512_bf16"] / 4.54e12 - 1) < 5e-3
    assert abs(fwd["mmdit_flux1024_bf16"] / 15.7e12 - 1) < 5e-3
    wl = synth.small_variant(synth.WORKLOADS["mmdit_flux512_bf16"], name="tiny_mmdit", hidden=64, heads=4, mlp=256,
                             latent_h=8, latent_w=8, txt_len=8, txt_dim=32)
    sub, rows, n, scale = bench.oracle_sample_plan(wl)
    assert (sub.depth, sub.depth_double, rows, n) == (1, 0, 1, 1)
    full = 2 * sum(bench.flops_per_sequence(wl))
    assert abs(scale * sum(bench.flops_per_sequence(sub)) / full - 1) < 1e-12
    sec, units, scaled, desc = bench.oracle_sample(wl)
    assert units == wl.W and abs(scaled / (sec * scale) - 1) < 1e-12 and "scaled" in desc
