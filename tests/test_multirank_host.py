"""The benchmark's multi-rank host logic on CPU with gloo, world size 2:
barrier, max-over-ranks timing and the whole-job throughput (replicas, no
data-path collective)."""
import os
import socket

import pytest
import torch
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
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    ws, r, local = bench.dist_setup()
    assert (ws, r, local) == (world, rank, rank)
    elapsed = [120.0, 200.0][rank]
    dist.barrier()
    m = bench.max_over_ranks(elapsed, dist, "cpu")
    q.put((rank, m, bench.job_throughput(100, ws, m)))
    dist.barrier()
    dist.destroy_process_group()


def test_max_over_ranks_gloo_world2():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=10) for _ in range(2))
    for rank, m, v in res:
        assert m == 200.0
        assert v == pytest.approx(100 * 2 / 0.2)


def test_single_rank_defaults():
    import bench
    assert bench.max_over_ranks(3.5, None) == 3.5
    assert bench.job_throughput(10, 1, 1000.0) == 10.0
