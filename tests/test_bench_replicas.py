"""The multi-GPU path of bench.py is N independent replicas: check its
host-side aggregation (sum of ratings over the slowest rank's time) with
world_size 2 over gloo on CPU."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    import torch.distributed as dist

    import bench

    dist.init_process_group("gloo", rank=rank, world_size=world)
    ratings = 1000.0 * (rank + 1)
    ms = 10.0 * (rank + 1)
    got = bench.replica_throughput(world, ratings, ms)
    mx = bench._max_over_ranks(world, ms)
    sm = bench._sum_over_ranks(world, ratings)
    bench._barrier(world)
    dist.destroy_process_group()
    q.put((rank, got, mx, sm))


def test_replica_aggregation_two_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = [q.get(timeout=120) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, got, mx, sm in out:
        assert mx == 20.0 and sm == 3000.0
        assert got == pytest.approx(3000.0 / 0.020)
