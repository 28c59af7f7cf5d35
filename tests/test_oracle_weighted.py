"""Pins of the oracle's weighted-adjacency aggregation (Sec. 3's A = [a_ij]
with general entries, D^_ii = sum_j (A + I)_ij, Eq. 1's operator) to things
other than itself: a weight of m equals m copies of the edge in the 0/1
oracle, a dense D^-1/2 (A + I) D^-1/2 built with numpy, the operator's fixed
vector sqrt(dhat), its symmetry for symmetric weights, and the limits of unit
and zero weights. A dropped self-loop, a transposed weight, the unweighted
degree or a weight applied twice fails one of them.
"""
import numpy as np
import pytest

import oracle
from paper_2010_07565_gb300 import inputs


def rng(seed):
    return np.random.Generator(np.random.PCG64(seed))


def csr_rows(rowptr):
    return np.repeat(np.arange(len(rowptr) - 1), np.diff(rowptr))


def dense_operator(rowptr, colidx, values):
    """D^-1/2 (A + I) D^-1/2 as a dense matrix, A[i, colidx[e]] = values[e]."""
    N = len(rowptr) - 1
    A = np.zeros((N, N))
    np.add.at(A, (csr_rows(rowptr), colidx), values)
    Ahat = A + np.eye(N)
    d = Ahat.sum(axis=1)
    Dm = np.diag(1.0 / np.sqrt(d))
    return Dm @ Ahat @ Dm


def test_integer_weights_equal_repeated_edges():
    """A weight of m on (i, j) is m parallel unit edges: the 0/1 oracle on the
    multigraph CSR (each entry repeated m times) gives the same degrees and H."""
    rp, ci = inputs.random_graph(60, 5.0, 11, hub_degree=20)
    row = csr_rows(rp)
    g = rng(4)
    lo, hi = np.minimum(row, ci), np.maximum(row, ci)
    m = 1 + (lo * 7 + hi * 13) % 3          # 1..3, the same on (i, j) and (j, i)
    rep_ci = np.repeat(ci, m).astype(np.int32)
    rep_rp = np.concatenate([[0], np.cumsum(np.bincount(row, weights=m, minlength=60))])
    rep_rp = rep_rp.astype(np.int64)
    assert rep_rp[-1] == rep_ci.size
    z = g.standard_normal((60, 5))
    np.testing.assert_allclose(oracle.degree_weighted(rp, m.astype(np.float64)),
                               oracle.degree(rep_rp), rtol=0, atol=1e-12)
    H = oracle.aggregate_weighted(rp, ci, m.astype(np.float32), z)
    np.testing.assert_allclose(H, oracle.aggregate(rep_rp, rep_ci, z), rtol=1e-13, atol=1e-13)


@pytest.mark.parametrize("seed", [1, 2, 3])
def test_aggregate_weighted_equals_dense_operator(seed):
    """Against numpy's dense D^-1/2 (A + I) D^-1/2 zeta, with weights that are
    not symmetric (a transposed a_ij would show) and some zero."""
    rp, ci = inputs.random_graph(9, 3.0, seed)
    g = rng(seed + 50)
    w = g.uniform(0.0, 3.0, ci.size)
    w[g.random(ci.size) < 0.2] = 0.0
    z = g.standard_normal((9, 4))
    H, A = oracle.aggregate_weighted(rp, ci, w, z, with_absterm=True)
    Op = dense_operator(rp, ci, w)
    np.testing.assert_allclose(H, Op @ z, rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(A, np.abs(Op) @ np.abs(z), rtol=1e-12, atol=1e-13)
    rows = np.array([8, 0, 3])
    np.testing.assert_allclose(oracle.aggregate_weighted(rp, ci, w, z, rows=rows), H[rows],
                               rtol=0, atol=0)


def test_sqrt_degree_is_a_fixed_vector():
    """A~ v = v for v_i = sqrt(dhat_i): sum_j a^_ij sqrt(dhat_j) / sqrt(dhat_i
    dhat_j) = dhat_i / sqrt(dhat_i), whatever the weights."""
    rp, ci = inputs.random_graph(500, 8.0, 5, hub_degree=200)
    w = inputs.edge_weights(rp, ci, 9)
    v = np.sqrt(oracle.degree_weighted(rp, w))[:, None]
    np.testing.assert_allclose(oracle.aggregate_weighted(rp, ci, w, v), v, rtol=1e-12)


def test_symmetric_weights_give_a_symmetric_operator():
    rp, ci = inputs.random_graph(40, 6.0, 8)
    w = inputs.edge_weights(rp, ci, 2)
    Op = oracle.aggregate_weighted(rp, ci, w, np.eye(40))     # column k = A~ e_k
    np.testing.assert_allclose(Op, Op.T, rtol=0, atol=1e-15)


def test_unit_weights_reduce_to_eq1_and_zero_weights_to_the_self_loop():
    rp, ci = inputs.random_graph(300, 6.0, 3, hub_degree=100)
    z = rng(7).standard_normal((300, 6))
    np.testing.assert_allclose(oracle.aggregate_weighted(rp, ci, np.ones(ci.size), z),
                               oracle.aggregate(rp, ci, z), rtol=1e-14, atol=1e-15)
    np.testing.assert_allclose(oracle.aggregate_weighted(rp, ci, np.zeros(ci.size), z), z,
                               rtol=0, atol=0)


def test_weights_scale_the_edges_not_the_self_loop():
    """Doubling every weight changes dhat_i from 1 + s_i to 1 + 2 s_i: an
    isolated node is unchanged, and a two-node graph follows the closed form."""
    rp = np.array([0, 1, 2, 2], np.int64)            # 0 - 1, node 2 isolated
    ci = np.array([1, 0], np.int32)
    z = np.array([[1.0], [3.0], [5.0]])
    for a in (0.5, 2.0, 7.0):
        H = oracle.aggregate_weighted(rp, ci, np.array([a, a]), z)
        d = 1.0 + a
        np.testing.assert_allclose(H[:, 0], [(1.0 + a * 3.0) / d, (3.0 + a * 1.0) / d, 5.0],
                                   rtol=1e-15)


def test_bad_weights_and_empty_graphs():
    rp, ci = inputs.random_graph(20, 4.0, 1)
    z = np.ones((20, 2))
    w = np.ones(ci.size)
    w[3] = -1.0
    with pytest.raises(ValueError):
        oracle.aggregate_weighted(rp, ci, w, z)
    w[3] = np.nan
    with pytest.raises(ValueError):
        oracle.aggregate_weighted(rp, ci, w, z)
    empty_rp = np.zeros(6, np.int64)
    zz = rng(3).standard_normal((5, 3))
    np.testing.assert_array_equal(
        oracle.aggregate_weighted(empty_rp, np.zeros(0, np.int32), np.zeros(0), zz), zz)


def test_layer_forward_weighted_composes_the_steps():
    c = inputs.layer_case(120, 70, 9, seed=4, mean_degree=5.0)
    rp, ci = c["rowptr"], c["colidx"]
    w = inputs.edge_weights(rp, ci, 3)
    out = oracle.layer_forward_weighted(c["X"], c["W"], rp, ci, w, c["s"], c["t"])
    ref = oracle.layer_forward(c["X"], c["W"], rp, ci, c["s"], c["t"])
    np.testing.assert_array_equal(out["dot"], ref["dot"])
    Op = dense_operator(rp, ci, w.astype(np.float64))
    np.testing.assert_allclose(out["H"], Op @ ref["zeta"], rtol=1e-12, atol=1e-13)
    ones = oracle.layer_forward_weighted(c["X"], c["W"], rp, ci, np.ones(ci.size),
                                         c["s"], c["t"])
    np.testing.assert_allclose(ones["H"], ref["H"], rtol=1e-14, atol=1e-15)


def test_edge_weights_are_symmetric_positive_and_seeded():
    rp, ci = inputs.random_graph(200, 7.0, 6, hub_degree=50)
    w = inputs.edge_weights(rp, ci, 12)
    assert w.dtype == np.float32 and w.shape == ci.shape
    assert w.min() >= 0.5 and w.max() < 2.0
    row = csr_rows(rp)
    lookup = {(int(i), int(j)): float(x) for i, j, x in zip(row, ci, w)}
    assert all(lookup[(j, i)] == x for (i, j), x in lookup.items())
    np.testing.assert_array_equal(w, inputs.edge_weights(rp, ci, 12))
    assert not np.array_equal(w, inputs.edge_weights(rp, ci, 13))
