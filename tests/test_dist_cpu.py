"""The multi-rank host logic of bench.py on CPU: two gloo ranks (the GPU runs use one NCCL
rank per GPU and replicate the step, with no collective on the data path).  Each rank
reports a different step time; the job's time is the slowest rank's and the job's rate
counts every rank's units."""
import os
import socket
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, ws, port, out):
    sys.path.insert(0, ROOT)
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=ws)
    try:
        bench.barrier(ws)
        ms = 10.0 + 5.0 * rank                      # rank 1 is the slower one
        job_ms = bench.max_over_ranks(ms, ws)
        out.put((rank, job_ms, bench.job_rate(128, job_ms, ws)))
        bench.barrier(ws)
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("ws", [2])
def test_job_time_is_the_slowest_rank_and_rate_counts_all_ranks(ws):
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, ws, port, out)) for r in range(ws)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    got = sorted(out.get(timeout=10) for _ in range(ws))
    for rank, job_ms, rate in got:
        assert job_ms == 15.0                        # max over the ranks, seen by every rank
        assert rate == pytest.approx(ws * 128 / 0.015)
