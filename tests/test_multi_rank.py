"""bench.py's multi-GPU path on CPU: replicas only, one process per rank, the job's time is the max
over ranks of the timed region and the value counts every rank's units.  Two gloo ranks on
127.0.0.1 stand in for the GPUs."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank: int, world: int, port: int, q):
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        ms = [120.0, 150.0][rank]  # rank 1 is the slower one
        dist.barrier()
        t = bench.max_over_ranks(ms, world, torch.device("cpu"))
        q.put((rank, t, bench.job_throughput(8, 1000, 10, world, t)))
    finally:
        dist.destroy_process_group()


def test_two_ranks_take_the_max_and_count_both_replicas():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [r for r, _, _ in got] == [0, 1]
    assert all(t == 150.0 for _, t, _ in got)                      # both ranks see the slowest rank's time
    assert all(v == pytest.approx(8 * 1000 * 10 * 2 / 0.150) for _, _, v in got)


def test_single_rank_is_the_identity():
    assert bench.max_over_ranks(42.0, 1, torch.device("cpu")) == 42.0
    assert bench.job_throughput(8, 1000, 10, 1, 100.0) == pytest.approx(8e5)
