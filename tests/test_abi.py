"""The C ABI library loads on the host, exports every entry point the headers declare, and
its host-only calls (parameter table, routing) agree with their definitions.  No kernel is
launched."""
import ctypes
import os
import re

import numpy as np
import pytest

import synth
from oracle import grpo

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def jg():
    from paper_2607_17572_gb300 import _build
    _build.build()
    import paper_2607_17572_gb300 as jg
    jg.lib()
    return jg


def _declared(header):
    src = open(os.path.join(ROOT, "include", header)).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    names = re.findall(r"^\s*(?:const\s+)?[A-Za-z_][A-Za-z0-9_]*\s*\**\s*([A-Za-z_][A-Za-z0-9_]*)\s*\(", src, re.M)
    return sorted(set(n for n in names if n not in ("if", "while", "for", "return", "sizeof")))


@pytest.mark.parametrize("header", ["jagg.h", "jagg_testing.h"])
def test_every_declared_symbol_is_exported(jg, header):
    names = _declared(header)
    assert len(names) >= 4
    L = ctypes.CDLL(jg.LIB_PATH)
    for n in names:
        assert hasattr(L, n), f"{n} declared in {header} but not exported"


def test_main_entry_points_are_declared():
    names = _declared("jagg.h")
    for n in ["dit_forward_save", "grpo_step_signals", "jagg_route", "jagg_aggregate", "dit_joint_vjp",
              "grad_reduce"]:
        assert n in names


@pytest.mark.parametrize("name", sorted(synth.WORKLOADS))
def test_param_table_matches_the_workload_shapes(jg, name):
    wl = synth.WORKLOADS[name]
    cfg = jg.Config.from_workload(wl)
    table = jg.param_table(cfg)
    shapes = dict(synth.param_shapes(wl))
    assert sorted(p.name for p in table) == sorted(shapes)
    end = 0
    for p in sorted(table, key=lambda p: p.offset):
        shp = shapes[p.name]
        assert (p.rows, p.cols) == (shp[0], shp[1] if len(shp) == 2 else 1)
        assert p.offset >= end and p.offset % 64 == 0
        end = p.offset + p.numel
    assert jg.param_count(cfg) >= end


def test_unsupported_and_bad_configs_are_rejected(jg):
    wl = synth.WORKLOADS["tiny_dit_f32"]
    cfg = jg.Config.from_workload(wl)
    cfg.heads = 3
    assert jg.lib().jagg_param_count(ctypes.byref(cfg)) < 0
    assert "heads" in jg.lib().jagg_last_error().decode()


def test_routing_is_bit_exact_with_the_oracle(jg):
    rng = np.random.Generator(np.random.PCG64(3))
    for n in [1, 2, 4, 5, 8, 13]:
        for frac in [0.0, 0.25, 0.4, 0.5, 0.6, 0.75, 1.0, 1.0 / 3, 2.0 / 3]:
            r, f = jg.jagg_route(n, frac)
            assert r == grpo.route_schedule(n, frac).tolist(), (n, frac)
        cos = rng.uniform(0.0, 1.0, size=n)
        cos[rng.uniform(size=n) < 0.3] = 0.5          # ties at the threshold count as JAGG
        r, f = jg.jagg_route(n, cos=cos, tau=0.5)
        ro, fo = grpo.route_calibrate(cos, 0.5)
        assert r == ro.tolist() and f == fo


def test_route_argument_errors(jg):
    route = (ctypes.c_uint8 * 4)()
    assert jg.lib().jagg_route(4, 1.5, None, 0.5, route, None) == -1
    assert jg.lib().jagg_route(0, 0.5, None, 0.5, route, None) == -1


def test_host_argument_checks_of_the_signal_and_sampler_entry_points(jg):
    """Argument errors are caught on the host before any launch (so these calls run without a
    device): a missing schedule, a non-positive noise scale, too small a workspace, strides
    below the row length, a span whose endpoint times coincide."""
    L = jg.lib()
    fake = 1 << 20                                   # never dereferenced: every call fails first
    ws = 256
    # grpo_step_signals_eps without a schedule
    st = L.grpo_step_signals_eps(fake, 0, fake, fake, None, None, fake, fake, fake, 2, 3, 100, 0.1, 5.0, 1e-8,
                                 1.0, None, None, fake, fake, fake, fake, fake, ws, None)
    assert st < 0 and "schedule" in L.jagg_last_error().decode()
    # jagg_rollout_step: sigma must be positive; workspace size; strides
    args = lambda sigma, zs, wsb: (fake, 0, 0, fake, fake, zs, fake, 0, 2, 100, 0.9, 0.8, sigma, None, fake, 1, None,
                                   0, fake, wsb, None)
    assert L.jagg_rollout_step(*args(0.0, 0, 1 << 20)) < 0
    assert "sigma" in L.jagg_last_error().decode()
    assert L.jagg_rollout_step(*args(0.1, 0, 8)) == -5        # JAGG_ERR_WORKSPACE
    assert "workspace" in L.jagg_last_error().decode()
    assert L.jagg_rollout_step(*args(0.1, 50, 1 << 20)) < 0
    assert "stride" in L.jagg_last_error().decode()
    assert L.jagg_rollout_workspace_bytes(2, 100) >= 2 * 8
    # jagg_aggregate_span with equal endpoint times
    assert L.jagg_aggregate_span(fake, 0, fake, 0.5, 0.5, 2, 3, 100, fake, 0, None) < 0
    assert "endpoints" in L.jagg_last_error().decode()


def test_static_signals_argument_errors_name_the_static_entry_point(jg):
    """grpo_step_signals_static reports its argument errors under its own name (checked
    before any device call)."""
    L = jg.lib()
    st = L.grpo_step_signals_static(None, 0, None, None, None, None, None, 0, 4, 64, 0.1, 5.0, 1e-8, 1.0, None, None,
                                    None, None, None, None, None)
    assert st == -1
    assert L.jagg_last_error().decode().startswith("grpo_step_signals_static")


def test_wait_timeout_rejects_limits_outside_its_range(jg):
    """The bounded-wait test entry point takes a limit in (0, 2 s]; others are argument
    errors returned before any launch."""
    L = jg.lib()
    for bad in (0, 2_000_000_001):
        assert L.jagg_test_wait_timeout(bad, ctypes.c_void_p(16), None) == -1
        assert "limit" in L.jagg_last_error().decode()
