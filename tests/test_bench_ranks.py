"""Host logic of bench.py's multi-GPU mode on CPU (gloo, world size 2): the
path has no data-path exchange, every rank decodes its own sequences, and the
whole-job numbers are the slowest rank's time and the sum of the ranks'
committed tokens.  Under torchrun the CPU reference arm runs on rank 0 only."""
import argparse
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms, committed = bench.rank_aggregate(dist, "cpu", 10.0 + rank, 100 * (rank + 1))
        q.put((rank, ms, committed))
    finally:
        dist.destroy_process_group()


def test_rank_aggregate_gloo_world2():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=5) for _ in range(2))
    for rank, ms, committed in got:
        assert ms == 11.0           # the slowest rank's time
        assert committed == 300.0   # every rank's tokens


def test_rank_aggregate_single_process():
    assert bench.rank_aggregate(None, "cpu", 3.5, 7) == (3.5, 7.0)


def test_reference_arm_runs_on_rank_zero_only(capsys):
    args = argparse.Namespace(workload="llama7b-n16", steps=3, warmup=3, cpu_layers=2, gpus=2)
    assert bench.run_reference(args, 1) == 0
    assert capsys.readouterr().out == ""
