"""Host-side logic of the multi-GPU benchmark path, run as two gloo ranks on
the CPU: replicas report the slowest rank's time and the sum of their units."""
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


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        assert bench.dist_env() == (rank, world, rank)
        max_ms, units = bench.aggregate_over_ranks(10.0 * (rank + 1), 1000.0 + rank, world)
        q.put((rank, max_ms, units))
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2])
def test_replicas_take_max_time_and_sum_units(world):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=10) for _ in range(world))
    for rank, max_ms, units in got:
        assert max_ms == 10.0 * world
        assert units == sum(1000.0 + r for r in range(world))


def test_single_rank_is_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.aggregate_over_ranks(3.5, 7.0, 1) == (3.5, 7.0)


def test_induced_subgraph_renumbers_and_drops_outside_edges():
    import numpy as np
    sys.path.insert(0, ROOT)
    import bench
    rowptr = np.array([0, 2, 4, 6, 8], np.int64)      # 4-cycle 0-1-2-3-0
    colidx = np.array([1, 3, 0, 2, 1, 3, 0, 2], np.int32)
    rp, ci = bench.induced_subgraph(rowptr, colidx, 1, 4)   # nodes 1, 2, 3
    assert rp.tolist() == [0, 1, 3, 4]
    assert ci.tolist() == [1, 0, 2, 1]
