"""The benchmark's multi-process path on the CPU (gloo, world size 2): every rank
runs its own replica, the timed region's length is the maximum over ranks, the
whole-job rate counts every rank's steps, and the reference arm's non-zero
ranks exit without work.  (The GPU runs use NCCL for the same calls.)"""
from __future__ import annotations

import io
import os
import socket
import sys
from contextlib import redirect_stdout

import pytest

torch = pytest.importorskip("torch")

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank: int, world: int, port: int, out):
    import argparse

    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    os.environ.update({"MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port), "RANK": str(rank),
                       "WORLD_SIZE": str(world)})
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        elapsed = 10.0 + 5.0 * rank                      # rank 1 is the slow one
        worst = bench.max_over_ranks(elapsed, "cpu")
        bench.barrier()
        rate = bench.whole_job_rate(world, 128, worst)
        buf = io.StringIO()
        args = argparse.Namespace(gpus=world, steps=2, warmup=1)
        with redirect_stdout(buf):
            if rank != 0:
                bench.run_reference(args)             # non-zero ranks return at once, silent
        out.put((rank, worst, rate, buf.getvalue()))
    finally:
        dist.destroy_process_group()


def test_two_ranks_max_time_and_whole_job_rate():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    res = [out.get(timeout=120) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    res.sort()
    for rank, worst, rate, printed in res:
        assert worst == 15.0                           # the slowest rank's time
        assert rate == pytest.approx(2 * 128 / 0.015)  # both ranks' steps over that time
        if rank == 1:
            assert printed == ""


def test_single_process_is_unchanged():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(12.5, "cpu") == 12.5
    assert bench.whole_job_rate(1, 128, 25.6) == pytest.approx(5000.0)
