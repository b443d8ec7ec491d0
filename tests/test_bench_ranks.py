"""The multi-rank logic of bench.py on CPU: two gloo ranks, one process each.

On N GPUs the benchmark runs one replica per rank (the MoE layer has no
exchange step); the job's time is the largest rank's time and its value the
work of all ranks over that time. Only rank 0 reports; the reference arm runs
on rank 0 alone.
"""
import io
import os
import socket
import sys
from contextlib import redirect_stdout

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, times, out):
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    t = bench.max_over_ranks(times[rank], world, "cpu")
    out[rank] = (t, bench.job_rate(100, world, t))
    dist.barrier()
    dist.destroy_process_group()


def test_job_time_is_the_slowest_rank_and_value_aggregates_all_ranks():
    world, port = 2, _free_port()
    mgr = mp.get_context("spawn").Manager()
    out = mgr.dict()
    times = [0.25, 0.5]
    mp.start_processes(_rank_main, args=(world, port, times, out), nprocs=world, start_method="spawn")
    assert out[0][0] == out[1][0] == 0.5
    assert out[0][1] == out[1][1] == 100 * 2 / 0.5


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(0.3, 1, "cpu") == 0.3
    assert bench.job_rate(64, 1, 2.0) == 32.0


def test_reference_arm_prints_only_on_rank_zero(monkeypatch):
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setattr(sys, "argv", ["bench.py", "--impl", "reference", "--steps", "1", "--warmup", "1"])
    buf = io.StringIO()
    with redirect_stdout(buf):
        bench.main()
    assert buf.getvalue() == ""
