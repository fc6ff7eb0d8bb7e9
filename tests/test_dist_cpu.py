"""Multi-rank host logic of the benchmark on CPU (gloo, world size 2).

The quantizer shards by rows with no exchange step, so the only cross-rank
operations are the barrier and the max-over-ranks reduction of the timed
region; these run here on two gloo ranks.
"""

import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, results):
    import torch
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    import bench
    r, w, lr = bench.dist_env()
    assert (r, w, lr) == (rank, world, rank)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    # rank 1 is the slow one: its time must be what every rank reports
    t = 1.5 if rank == 1 else 1.0
    dist.barrier()
    tmax = bench.max_over_ranks(t, world)
    v = bench.weak_scaling_value(1000, 10, world, tmax)
    results[rank] = (tmax, v)
    dist.destroy_process_group()


@pytest.mark.timeout(120)
def test_two_rank_max_time_and_weak_scaling_value():
    world = 2
    port = _free_port()
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    results = mgr.dict()
    procs = [ctx.Process(target=_worker, args=(r, world, port, results)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(90)
        assert p.exitcode == 0
    assert results[0] == results[1]
    tmax, v = results[0]
    assert tmax == 1.5
    assert v == pytest.approx(1000 * 10 * 2 / 1.5)


def test_single_rank_defaults():
    import bench
    assert bench.max_over_ranks(3.0, 1) == 3.0
    assert bench.weak_scaling_value(58720256, 4, 1, 2.0) == 58720256 * 4 / 2.0

