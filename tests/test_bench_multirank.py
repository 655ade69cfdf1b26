"""The multi-rank path of bench.py on CPU: two gloo ranks (weak scaling, no data-path collective).

Each rank runs its own replica; the only exchange is the timing reduction: tokens are summed over
ranks and the elapsed time is the maximum over ranks."""
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


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    import bench

    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # rank r processed 16 tokens in (r + 1) seconds
        tokens, elapsed = bench.aggregate(16, float(rank + 1))
        r, w, _ = bench.dist_setup(world)
        q.put((rank, tokens, elapsed, r, w))
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 3])
def test_aggregate_over_gloo_ranks(world):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, tokens, elapsed, r, w in res:
        assert tokens == 16 * world and elapsed == float(world)
        assert r == rank and w == world


def test_aggregate_single_process_is_identity():
    import bench

    assert not dist.is_initialized()
    assert bench.aggregate(16, 0.5) == (16, 0.5)
