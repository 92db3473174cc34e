"""The multi-rank bookkeeping of bench.py on CPU: two gloo ranks, each with
its own batch (weak scaling); the job time is the slowest rank's and the
throughput counts every rank's tokens."""
import os
import socket

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    local_ms = 10.0 * (rank + 1)            # rank 1 is the slower one
    value, ms = bench.combine_ranks(local_ms, tokens_per_rank=8192, dist=dist, device="cpu")
    q.put((rank, value, ms))
    dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_rank():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=10) for _ in range(world))
    for rank, value, ms in got:
        assert ms == pytest.approx(20.0)
        assert value == pytest.approx(2 * 8192 / 0.020)


def test_single_rank_without_process_group():
    value, ms = bench.combine_ranks(4.0, tokens_per_rank=1000)
    assert ms == 4.0 and value == pytest.approx(1000 / 0.004)
