"""The sharded layer's host logic on the CPU: the row partition, each rank's
renumbered CSR and halo, and the halo exchange over two (and three) gloo
ranks, in both forms. The products are the oracle's (no GPU here): each rank
takes the oracle's product of its own rows with 1/sqrt(dhat) applied and
either exchanges those rows (exchange_rows) or exchanges the packed signs and
row scales of its rows (exchange_packed_rows) and computes the halo's product
itself, with the halo degrees the plan carries; it then aggregates its block
by the plain definition of Eq. 13 over its table. The blocks, put back
together, must equal the oracle's whole-graph layer -- also with more ranks
than rows (empty blocks) and on a graph without edges (no halo)."""
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


# Graphs: a hub of degree 250 (most rows' halos cross ranks), three rows on
# more ranks than rows (an empty block), and no edges at all (no halo).
CASES = {"hub": dict(N=600, K=150, F=12, seed=77, mean_degree=6.0, hub_degree=250),
         "tiny": dict(N=3, K=70, F=5, seed=5, mean_degree=2.0),
         "edgeless": dict(N=50, K=40, F=7, seed=9, mean_degree=0.0)}


def case(name="hub"):
    return inputs.layer_case(**CASES[name])


def test_partition_of_fewer_rows_than_ranks_leaves_empty_blocks():
    rp = case("tiny")["rowptr"]
    b = shard.partition_rows(rp, 5)
    assert b.tolist()[0] == 0 and b.tolist()[-1] == 3 and np.all(np.diff(b) >= 0)
    assert int((np.diff(b) == 0).sum()) == 2          # five ranks, three rows
    empty = int(np.flatnonzero(np.diff(b) == 0)[0])
    lrp, lci, halo, recv = shard.local_plan(rp, case("tiny")["colidx"], b, empty)
    assert lrp.tolist() == [0] and lci.size == 0 and halo.size == 0 and recv.sum() == 0
    assert shard.partition_rows(np.zeros(1, np.int64), 3).tolist() == [0, 0, 0, 0]


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


def unpack_signs(bits, K):
    """Signs (+-1, int8) of packed rows (bit k of a row at word k / 64,
    position k % 64)."""
    w = np.ascontiguousarray(bits).view(np.uint64)
    k = np.arange(K)
    b = (w[:, k // 64] >> (k % 64).astype(np.uint64)) & np.uint64(1)
    return np.where(b == 1, 1, -1).astype(np.int8)


def _rank_main(rank, world, port, result_path, packed=False, name="hub"):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        c = case(name)
        rp, ci = c["rowptr"], c["colidx"]
        b = shard.partition_rows(rp, world)
        plan = shard.build_plan(rp, ci, b, rank)
        lo, hi = plan.lo, plan.hi
        assert np.array_equal(np.diff(plan.halo_rowptr), np.diff(rp)[plan.halo])
        # This rank's product rows (the oracle's), with 1/sqrt(dhat_j) applied.
        Y = oracle.centre(c["X"][lo:hi], c["s"], c["t"])
        SF, alpha = oracle.sign(Y), oracle.row_scale(Y)
        SB, beta = oracle.weight_binarize(c["W"])
        z = oracle.zeta(oracle.binary_dot(SF, SB), alpha, beta)
        dhat = np.diff(plan.rowptr) + 1.0
        zp = z / np.sqrt(dhat)[:, None]
        if packed:
            K = c["X"].shape[1]
            bits = torch.from_numpy(np.ascontiguousarray(oracle.pack(SF)).view(np.int64))
            hb, ha = shard.exchange_packed_rows(bits, torch.from_numpy(alpha), plan)
            zh = oracle.zeta(oracle.binary_dot(unpack_signs(hb.numpy(), K), SB), ha.numpy(), beta)
            zh = zh / np.sqrt(np.diff(plan.halo_rowptr) + 1.0)[:, None]
            table = np.concatenate([zp, zh])
        else:
            table = shard.exchange_rows(torch.from_numpy(zp), plan).numpy()
        # Eq. 13 on the block: H_i = dhat_i^-1/2 (Z'_i + sum over the row's entries of Z'_q).
        H = np.empty((plan.n_own, z.shape[1]))
        for i in range(plan.n_own):
            q = plan.colidx[plan.rowptr[i]:plan.rowptr[i + 1]]
            H[i] = (table[i] + table[q].sum(axis=0)) / np.sqrt(dhat[i])
        np.save(f"{result_path}.{rank}.npy", H)
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world,packed,name", [(2, False, "hub"), (3, False, "hub"),
                                               (2, True, "hub"), (3, True, "hub"),
                                               (4, False, "tiny"), (4, True, "tiny"),
                                               (3, True, "edgeless")])
def test_sharded_layer_equals_the_whole_graph_layer(tmp_path, world, packed, name):
    path = str(tmp_path / "H")
    mp.start_processes(_rank_main, args=(world, free_port(), path, packed, name), nprocs=world,
                       start_method="spawn")
    c = case(name)
    ref = oracle.layer_forward(c["X"], c["W"], c["rowptr"], c["colidx"], c["s"], c["t"])["H"]
    H = np.concatenate([np.load(f"{path}.{r}.npy") for r in range(world)])
    assert H.shape == ref.shape
    assert np.allclose(H, ref, rtol=1e-12, atol=1e-12)


def test_exchange_bytes_choose_the_smaller_form():
    # C1's widths: packed signs (23 words) + scale, 188 B a row, against 256 B
    assert shard.exchange_bytes_per_row(1433, 64, True) == 188
    assert shard.exchange_bytes_per_row(1433, 64, False) == 256
    # C4's layer 1: 84 B against 512 B; layer 2 (K = 128, F = 41): 20 against 164
    assert shard.exchange_bytes_per_row(602, 128, True) == 84
    assert shard.exchange_bytes_per_row(128, 41, True) < shard.exchange_bytes_per_row(128, 41, False)
    # wide rows of few features: the product rows are smaller
    assert shard.exchange_bytes_per_row(8192, 16, True) > shard.exchange_bytes_per_row(8192, 16, False)
