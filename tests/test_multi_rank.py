"""The N > 1 benchmark path on CPU: two ranks over gloo (127.0.0.1) reduce
their timings with max_over_ranks and the weak-scaling rate counts every
replica's work against the slowest rank's time."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        # rank-dependent "timings": the reduction must return the slowest
        got = bench.max_over_ranks([10.0 + rank, 50.0 - rank, 3.5 * (rank + 1)])
        rate = bench.weak_rate(2.0e12, steps=4, world=world, ms=got[0], scale=1e12)
        q.put((rank, got, rate))
    finally:
        dist.destroy_process_group()


def test_two_rank_timing_reduction():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = [q.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, got, rate in res:
        assert got == [11.0, 50.0, 7.0]
        # 2 replicas x 4 steps x 2e12 flops in 11 ms
        assert rate == pytest.approx(2 * 4 * 2.0 / 11e-3)


def test_single_process_is_identity():
    import bench
    assert bench.max_over_ranks([1.5, 2.5]) == [1.5, 2.5]
    assert bench.weak_rate(1e9, 2, 1, 1.0, 1e9) == pytest.approx(2000.0)
