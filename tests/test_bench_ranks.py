"""The multi-rank side of bench.py on CPU (gloo, two ranks): the job's time is the slowest rank's,
its rate counts every replica's work, and the reference arm runs on rank 0 only.  The path does not
shard (one independent replica per GPU), so these host rules are all there is to the N > 1 path."""

import io
import os
import socket
import sys
from contextlib import redirect_stdout

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    sys.path.insert(0, ROOT)
    import bench
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        ms = [1.5, 4.25][rank]  # the second rank is the slow one
        job_ms = bench.max_over_ranks(ms, "cpu")
        rate = bench.job_rate(world, 1000.0, job_ms)
        out[rank] = (job_ms, rate)
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_time_and_count_every_replica():
    world, port = 2, _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_rank_main, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    for rank in range(world):
        job_ms, rate = res[rank]
        assert job_ms == 4.25
        assert rate == pytest.approx(2 * 1000.0 / 4.25e-3)


def test_one_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(2.0, "cpu") == 2.0
    assert bench.job_rate(1, 10.0, 5.0) == pytest.approx(2000.0)


def test_reference_arm_runs_on_rank_zero_only(monkeypatch):
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setenv("LOCAL_RANK", "1")
    args = bench.parse(["--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "3"])
    buf = io.StringIO()
    with redirect_stdout(buf):
        assert bench.run_reference(args) is None
    assert buf.getvalue() == ""
