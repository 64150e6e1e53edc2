"""Replica aggregation of bench.py with world size 2 on CPU (gloo): value is
the units all ranks processed over the slowest rank's time, with no
collective in the data path (each rank runs its own replica)."""
import os
import socket

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", init_method="env://")
    import bench
    units = 1000.0 * (rank + 1)           # ranks may process different amounts
    secs = 0.5 + 0.25 * rank              # and take different times
    assert bench.dist_env() == (world, rank, rank)
    value, tmax = bench.aggregate(units, secs, world, True)
    dist.barrier()
    q.put((rank, value, tmax))
    dist.destroy_process_group()


@pytest.mark.timeout(120)
def test_two_rank_replica_aggregation():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(100)
        assert p.exitcode == 0
    res = sorted(q.get() for _ in range(2))
    for rank, value, tmax in res:
        assert tmax == pytest.approx(0.75)
        assert value == pytest.approx(3000.0 / 0.75)


def test_single_rank_aggregation():
    import bench
    assert bench.aggregate(100.0, 2.0, 1, False) == (50.0, 2.0)
