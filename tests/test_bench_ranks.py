"""The multi-rank path of bench.py on CPU (gloo, world size 2): the step time every rank reports is
the slowest rank's, the whole-job rate counts every rank's tokens over that time, and the
reference arm does its work on rank 0 only.  No GPU: the path only exchanges host values."""
import os
import socket

import pytest


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, port, out):
    import sys
    import torch
    import torch.distributed as dist
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import bench
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=2)
    try:
        local_ms = [10.0, 12.5][rank]
        ms = bench.max_over_ranks(torch, local_ms, torch.device("cpu"))
        out[rank] = (ms, bench.job_rate(256, ms, 2))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_and_job_rate_gloo():
    import torch.multiprocessing as mp
    port = _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_rank_main, args=(port, out), nprocs=2, join=True)
        res = dict(out)
    assert res[0] == res[1]
    ms, rate = res[0]
    assert ms == 12.5
    assert rate == pytest.approx(2 * 256 / 12.5e-3)


def test_single_rank_is_identity():
    import torch
    import bench
    assert bench.max_over_ranks(torch, 3.25, torch.device("cpu")) == 3.25
    assert bench.job_rate(256, 50.0, 1) == pytest.approx(256 / 0.05)


def test_reference_arm_other_ranks_do_no_work(monkeypatch, capsys):
    import argparse
    import bench
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("LOCAL_RANK", "1")
    args = argparse.Namespace(steps=1, warmup=0, cpu_tokens=1)
    assert bench.run_reference(args) is None
    assert capsys.readouterr().out == ""
