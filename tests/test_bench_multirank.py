"""The multi-rank path of bench.py on CPU: two `gloo` ranks.

The attention shards with no exchange step, so the only cross-rank logic is
the timing: every rank times its own replica, the job's time is the slowest
rank's, and the value counts the work of all ranks.  The reference arm runs
on rank 0 alone; the other ranks leave without work.
"""
import argparse
import io
import os
import socket
import sys
from contextlib import redirect_stdout

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402

WORLD = 2


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, port, times, ops, out):
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}",
                            rank=rank, world_size=WORLD)
    try:
        dist.barrier()
        t = bench.slowest(dist, times[rank])
        v = bench.job_tops(ops, WORLD, t)
        out[rank] = (t, v)
    finally:
        dist.destroy_process_group()


def test_slowest_rank_and_whole_job_value():
    port = _free_port()
    times = [0.25, 0.40]            # rank 1 is the slow one
    ops = 3.0e12
    with mp.Manager() as mgr:
        out = mgr.dict()
        mp.spawn(_rank_main, args=(port, times, ops, out), nprocs=WORLD, join=True)
        got = dict(out)
    for r in range(WORLD):
        t, v = got[r]
        assert t == max(times)
        assert v == pytest.approx(ops * WORLD / max(times) / 1e12)


def test_single_process_needs_no_group():
    assert bench.slowest(None, 0.5) == 0.5
    assert bench.job_tops(2e12, 1, 2.0) == pytest.approx(1.0)


def test_reference_arm_runs_on_rank_zero_only(monkeypatch):
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("LOCAL_RANK", "1")
    args = argparse.Namespace(gpus=2, steps=1, warmup=0, impl="reference")
    buf = io.StringIO()
    with redirect_stdout(buf):
        rc = bench.run_reference(args)
    assert rc == 0
    assert buf.getvalue() == ""
