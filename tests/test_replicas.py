"""The N > 1 path of bench.py is replicas only (one independent sequence per
rank, no collective on the data path).  Its rank logic — the slowest rank's
time and the sum of all ranks' tokens — is checked here with two gloo ranks
on the CPU."""
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


def _rank(rank, world, port, out):
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    ms, tok = bench.reduce_over_ranks(10.0 + 5.0 * rank, 100 + rank, dist, "cpu")
    out[rank] = (ms, tok)
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_replicas_reduce_time_and_tokens():
    world = 2
    port = _free_port()
    ctx = mp.get_context("spawn")
    out = ctx.Manager().dict()
    procs = [ctx.Process(target=_rank, args=(r, world, port, out)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    assert dict(out) == {0: (15.0, 201.0), 1: (15.0, 201.0)}


def test_single_rank_reduction_is_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.reduce_over_ranks(3.5, 7) == (3.5, 7.0)
