"""The N-process benchmark path on the CPU: two gloo ranks run independent replicas and
the whole-job figures are the sum of units over ranks and the maximum time over ranks."""

import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      LOCAL_RANK=str(rank), WORLD_SIZE=str(world))
    import bench

    r, lr, w = bench.dist_env()
    assert (r, lr, w) == (rank, rank, world)
    bench.init_dist(w, "gloo")
    units, secs = bench.aggregate(100.0 * (rank + 1), 1.5 + rank, w, "cpu")
    bench.barrier(w)
    out[rank] = (units, secs)
    dist.destroy_process_group()


def test_two_rank_aggregation():
    world = 2
    port = _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_worker, args=(world, port, out), nprocs=world, join=True)
        got = dict(out)
    for rank in range(world):
        assert got[rank] == (300.0, 2.5)


def test_single_rank_is_identity():
    import bench

    assert bench.aggregate(5.0, 2.0, 1, "cpu") == (5.0, 2.0)
