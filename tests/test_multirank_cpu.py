"""The multi-rank path of the benchmark on CPU (gloo, world size 2).

The fake-quantizer shards by tensors or rows with no data-path collective:
each rank runs its own replica and the only exchange is the MAX of the step
time over ranks.  Two gloo processes check that reduction and the weak-scaling
aggregate built on it, plus the per-rank barrier around a timed region.
"""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as tmp


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
        dist.barrier()
        ms = [3.0, 5.5][rank]                       # rank 1 is the slower replica
        m = bench.max_over_ranks(ms, world)
        gbs = bench.aggregate_gbs(1.0e9, world, m)  # 1 GB per rank per step
        dist.barrier()
        q.put((rank, m, gbs))
    finally:
        dist.destroy_process_group()


def test_two_rank_max_and_weak_scaling():
    world, port = 2, _free_port()
    ctx = tmp.get_context("spawn")
    q = ctx.SimpleQueue()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    res = sorted(q.get() for _ in range(world))
    for rank, m, gbs in res:
        assert m == 5.5                              # every rank sees the slowest time
        assert gbs == pytest.approx(2 * 1.0e9 / 5.5e-3 / 1e9)


def test_single_rank_is_identity():
    import bench
    assert bench.max_over_ranks(4.25, 1) == 4.25
    assert bench.aggregate_gbs(2.0e9, 1, 4.0) == pytest.approx(500.0)
