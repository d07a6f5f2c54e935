"""The multi-GPU bench path on the CPU: world size 2 over gloo (127.0.0.1).

Sequences are independent, so N GPUs run N replicas with no data-path
collective; what the ranks share is the timing: a barrier around the timed
region, the slowest rank's time, and the whole-job rate computed from it.
The reference arm runs on rank 0 only.  These tests run that host logic in two
CPU processes (no GPU).
"""
import os
import socket
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def free_port():
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world_size, port, queue):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world_size), LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world_size)
    try:
        ws, r, _ = bench.dist_env()
        dist.barrier()
        local_ms = 10.0 * (rank + 1)            # rank 1 is the slow one
        ms = bench.max_over_ranks(local_ms, dist, "cpu")
        rate = bench.whole_job_rate(ws, 8, 100, ms)
        dist.barrier()
        queue.put((r, ws, ms, rate))
    finally:
        dist.destroy_process_group()


def test_two_ranks_take_the_slowest_time_and_the_whole_job_rate():
    ctx = mp.get_context("spawn")
    queue = ctx.SimpleQueue()
    port = free_port()
    mp.start_processes(_rank_main, args=(2, port, queue), nprocs=2, join=True, start_method="spawn")
    got = sorted(queue.get() for _ in range(2))
    for r, ws, ms, rate in got:
        assert ws == 2
        assert ms == pytest.approx(20.0)            # max over ranks, seen by both
        assert rate == pytest.approx(2 * 8 * 100 / 0.020)   # weak scaling: both ranks' tokens
    assert [g[0] for g in got] == [0, 1]


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    import bench
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setattr(sys, "argv", ["bench.py", "--impl", "reference", "--gpus", "2"])
    args = bench.parse()
    assert bench.run_reference(args) == 0
    assert capsys.readouterr().out == ""        # rank 1 prints nothing and does no work


def test_single_process_needs_no_process_group():
    import bench
    assert bench.max_over_ranks(12.5, None, "cpu") == 12.5
    assert bench.whole_job_rate(1, 8, 10, 1.0) == pytest.approx(80000.0)
