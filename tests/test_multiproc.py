"""The bench's multi-replica bookkeeping on CPU: two gloo ranks on 127.0.0.1.  With N
replicas each rank decodes its own batch (weak scaling, no collective on the data path);
the reported step time is the slowest rank's, and the value counts every rank's tokens.
The reference arm runs on rank 0 only."""
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    import bench

    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # rank r "measured" a step of (r + 1) ms and an end-to-end step of (10 - r) ms
        got = bench.max_over_ranks([rank + 1.0, 10.0 - rank], device="cpu")
        out[rank] = got
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_two_gloo_ranks():
    world = 2
    ctx = mp.get_context("spawn")
    with ctx.Manager() as mgr:
        out = mgr.dict()
        mp.start_processes(_rank_main, args=(world, _free_port(), out), nprocs=world, join=True, start_method="spawn")
        res = dict(out)
    assert res[0] == res[1] == [2.0, 10.0]


def test_single_process_values_pass_through():
    sys.path.insert(0, ROOT)
    import bench

    assert bench.max_over_ranks([3.5, 1.25]) == [3.5, 1.25]


def test_whole_job_throughput_counts_every_replica():
    sys.path.insert(0, ROOT)
    import bench

    assert bench.whole_job_tok_s(1, 1, 2.0) == pytest.approx(500.0)
    assert bench.whole_job_tok_s(4, 1, 2.0) == pytest.approx(2000.0)
    assert bench.whole_job_tok_s(2, 16, 4.0) == pytest.approx(8000.0)


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    sys.path.insert(0, ROOT)
    import bench

    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    import argparse

    ns = argparse.Namespace(m=1, pct=70, steps=1, warmup=0, gpus=2)
    assert bench.run_reference(ns) is None
    assert capsys.readouterr().out == ""  # no JSON line and no oracle work on rank 1
