"""Pins of the oracle's inductive aggregators (Sec. 6.3's inductive models,
Table 3, read with GraphSAGE's definitions) to facts that do not come from
the oracle's own loops:

* the dense operators built from the CSR and applied with a BLAS matmul:
  D^-1 (A + I) for the mean aggregator, and I (on zself) plus D^-1 A (on
  zneigh, zero rows for isolated nodes) for GraphSAGE-mean;
* on a regular graph D^-1 (A + I) equals Eq. 1's D^-1/2 (A + I) D^-1/2, so the
  mean aggregator equals the pinned symmetric one;
* the mean operators' rows sum to one: constant columns are kept;
* relabelling the nodes permutes the result the same way;
* no edges: the mean aggregator is the identity, GraphSAGE-mean returns zself;
* Table 3's GraphSAGE figures (tests/test_cost_model.py) reproduce only with
  two products per layer and an aggregation of d_out-wide rows, the structure
  layer_forward_inductive("sage") computes.
"""
import numpy as np
import pytest

import oracle
from paper_2010_07565_gb300 import inputs


def rng(seed):
    return np.random.Generator(np.random.PCG64(seed))


def random_csr(N, p, seed, isolated=0):
    g = rng(seed)
    A = g.random((N, N)) < p
    np.fill_diagonal(A, False)
    A[:isolated, :] = False                              # the first `isolated` nodes
    A[:, :isolated] = False
    rows, cols = np.nonzero(np.triu(A | A.T, 1))      # each undirected edge once
    return inputs.edges_to_csr(rows, cols, N)


def dense(rowptr, colidx, N):
    A = np.zeros((N, N))
    for i in range(N):
        A[i, colidx[rowptr[i]:rowptr[i + 1]]] = 1.0
    return A


def test_mean_aggregator_is_the_dense_row_normalised_operator():
    N, F = 40, 5
    rowptr, colidx = random_csr(N, 0.1, seed=1)
    z = rng(2).standard_normal((N, F))
    Ahat = dense(rowptr, colidx, N) + np.eye(N)
    M = Ahat / Ahat.sum(axis=1, keepdims=True)
    np.testing.assert_allclose(oracle.aggregate_mean(rowptr, colidx, z), M @ z,
                               rtol=1e-12, atol=1e-14)


def test_sage_aggregator_is_self_plus_the_dense_neighbour_mean():
    N, F = 45, 4
    rowptr, colidx = random_csr(N, 0.06, seed=3, isolated=4)
    deg = np.diff(rowptr)
    assert (deg == 0).any() and (deg > 0).any()          # isolated nodes are covered
    g = rng(4)
    zs, zn = g.standard_normal((N, F)), g.standard_normal((N, F))
    A = dense(rowptr, colidx, N)
    M = A / np.maximum(deg, 1)[:, None]
    np.testing.assert_allclose(oracle.aggregate_sage(rowptr, colidx, zs, zn), zs + M @ zn,
                               rtol=1e-12, atol=1e-14)


def test_mean_equals_the_symmetric_operator_on_a_regular_graph():
    N, F = 30, 3
    ring = np.arange(N)
    rows = np.concatenate([ring, ring])                  # each undirected edge once
    cols = np.concatenate([(ring + 1) % N, (ring + 5) % N])
    rowptr, colidx = inputs.edges_to_csr(rows, cols, N)
    assert np.all(np.diff(rowptr) == 4)
    z = rng(5).standard_normal((N, F))
    np.testing.assert_allclose(oracle.aggregate_mean(rowptr, colidx, z),
                               oracle.aggregate(rowptr, colidx, z), rtol=1e-12, atol=1e-14)


def test_mean_operators_keep_constant_columns():
    N = 50
    rowptr, colidx = random_csr(N, 0.08, seed=6, isolated=3)
    c = np.tile(np.array([[2.5, -1.0, 0.0]]), (N, 1))
    np.testing.assert_allclose(oracle.aggregate_mean(rowptr, colidx, c), c, rtol=1e-14)
    has = (np.diff(rowptr) > 0)[:, None]
    zs = rng(7).standard_normal((N, 3))
    np.testing.assert_allclose(oracle.aggregate_sage(rowptr, colidx, zs, c), zs + c * has,
                               rtol=1e-13, atol=1e-14)


@pytest.mark.parametrize("which", ["mean", "sage"])
def test_relabelling_the_nodes_permutes_the_result(which):
    N, F = 35, 4
    rowptr, colidx = random_csr(N, 0.12, seed=8)
    g = rng(9)
    zs, zn = g.standard_normal((N, F)), g.standard_normal((N, F))
    perm = g.permutation(N)                      # new label of old node v is perm[v]
    r, c = np.repeat(np.arange(N), np.diff(rowptr)), colidx
    once = r < c
    rp2, ci2 = inputs.edges_to_csr(perm[r[once]], perm[c[once]], N)
    zs2, zn2 = np.empty_like(zs), np.empty_like(zn)
    zs2[perm], zn2[perm] = zs, zn
    if which == "mean":
        a, b = oracle.aggregate_mean(rowptr, colidx, zs), oracle.aggregate_mean(rp2, ci2, zs2)
    else:
        a = oracle.aggregate_sage(rowptr, colidx, zs, zn)
        b = oracle.aggregate_sage(rp2, ci2, zs2, zn2)
    np.testing.assert_allclose(b[perm], a, rtol=1e-12, atol=1e-14)


def test_without_edges():
    N, F = 8, 3
    rowptr, colidx = np.zeros(N + 1, np.int64), np.zeros(0, np.int32)
    g = rng(10)
    zs, zn = g.standard_normal((N, F)), g.standard_normal((N, F))
    np.testing.assert_array_equal(oracle.aggregate_mean(rowptr, colidx, zs), zs)
    np.testing.assert_array_equal(oracle.aggregate_sage(rowptr, colidx, zs, zn), zs)


def test_inductive_layer_composes_the_products():
    case = inputs.layer_case(60, 50, 6, seed=11)
    Wn = inputs.weights(50, 6, seed=12)
    r = oracle.layer_forward_inductive(case["X"], case["W"], case["rowptr"], case["colidx"],
                                       "sage", case["s"], case["t"], W_neigh=Wn)
    ref = oracle.layer_forward(case["X"], case["W"], case["rowptr"], case["colidx"],
                               case["s"], case["t"])
    np.testing.assert_array_equal(r["zeta"], ref["zeta"])
    refn = oracle.layer_forward(case["X"], Wn, case["rowptr"], case["colidx"], case["s"],
                                case["t"])
    np.testing.assert_array_equal(r["zeta_n"], refn["zeta"])
    g = oracle.layer_forward_inductive(case["X"], case["W"], case["rowptr"], case["colidx"],
                                       "gcn", case["s"], case["t"])
    np.testing.assert_array_equal(g["H"], ref["H"])
    assert np.all(np.abs(r["H"]) <= r["absterm"] * (1 + 1e-12))
