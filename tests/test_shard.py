"""The sharded layer's host logic on the CPU: the row partition, each rank's
renumbered CSR and halo, and the halo exchange over two (and three) gloo
ranks. The products are the oracle's (no GPU here): each rank takes the
oracle's product of its own rows with 1/sqrt(dhat) applied, exchanges rows
with exchange_rows, and aggregates its block by the plain definition of
Eq. 13 over its table; the blocks, put back together, must equal the oracle's
whole-graph layer."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import oracle
from paper_2010_07565_gb300 import inputs, shard


def free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def case():
    return inputs.layer_case(600, 150, 12, seed=77, mean_degree=6.0, hub_degree=250)


def test_partition_balances_work_and_covers_every_row():
    c = case()
    rp = c["rowptr"]
    cost = np.diff(rp) + 1
    for world in (1, 2, 3, 5, 8):
        b = shard.partition_rows(rp, world)
        assert b[0] == 0 and b[-1] == len(rp) - 1 and np.all(np.diff(b) >= 0)
        work = [int(cost[b[r]:b[r + 1]].sum()) for r in range(world)]
        assert sum(work) == int(cost.sum())
        assert max(work) <= cost.sum() / world + cost.max()      # within one row of even


def test_local_plan_renumbers_and_lists_the_halo():
    c = case()
    rp, ci = c["rowptr"], c["colidx"]
    b = shard.partition_rows(rp, 3)
    for rank in range(3):
        lrp, lci, halo, recv = shard.local_plan(rp, ci, b, rank)
        lo, hi = b[rank], b[rank + 1]
        n_own = hi - lo
        assert np.array_equal(np.diff(lrp), np.diff(rp)[lo:hi])        # full degrees kept
        assert np.all(np.diff(halo) > 0) and np.all((halo < lo) | (halo >= hi))
        assert recv.sum() == halo.size and recv[rank] == 0
        table = np.concatenate([np.arange(lo, hi), halo])             # local id -> global id
        assert np.array_equal(table[lci], ci[rp[lo]:rp[hi]])


def _rank_main(rank, world, port, result_path):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        c = case()
        rp, ci = c["rowptr"], c["colidx"]
        b = shard.partition_rows(rp, world)
        plan = shard.build_plan(rp, ci, b, rank)
        lo, hi = plan.lo, plan.hi
        # This rank's product rows (the oracle's), with 1/sqrt(dhat_j) applied.
        Y = oracle.centre(c["X"][lo:hi], c["s"], c["t"])
        SB, beta = oracle.weight_binarize(c["W"])
        z = oracle.zeta(oracle.binary_dot(oracle.sign(Y), SB), oracle.row_scale(Y), beta)
        dhat = np.diff(plan.rowptr) + 1.0
        zp = torch.from_numpy(z / np.sqrt(dhat)[:, None])
        table = shard.exchange_rows(zp, plan).numpy()
        # Eq. 13 on the block: H_i = dhat_i^-1/2 (Z'_i + sum over the row's entries of Z'_q).
        H = np.empty((plan.n_own, z.shape[1]))
        for i in range(plan.n_own):
            q = plan.colidx[plan.rowptr[i]:plan.rowptr[i + 1]]
            H[i] = (table[i] + table[q].sum(axis=0)) / np.sqrt(dhat[i])
        np.save(f"{result_path}.{rank}.npy", H)
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 3])
def test_sharded_layer_equals_the_whole_graph_layer(tmp_path, world):
    path = str(tmp_path / "H")
    mp.start_processes(_rank_main, args=(world, free_port(), path), nprocs=world,
                       start_method="spawn")
    c = case()
    ref = oracle.layer_forward(c["X"], c["W"], c["rowptr"], c["colidx"], c["s"], c["t"])["H"]
    H = np.concatenate([np.load(f"{path}.{r}.npy") for r in range(world)])
    assert H.shape == ref.shape
    assert np.allclose(H, ref, rtol=1e-12, atol=1e-12)
