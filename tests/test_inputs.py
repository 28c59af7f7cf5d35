"""The seeded workload generators against the input recipe they implement
(feature distributions, graph sizes and structure, CSR validity, seeds), on
the CPU. C1-C3 are generated in full; the Chung-Lu and Erdos-Renyi
generators of C4 and C5 are checked at reduced sizes."""
import math

import numpy as np
import pytest

from paper_2010_07565_gb300 import inputs


def check_csr(rowptr, colidx, N):
    assert rowptr.dtype == np.int64 and colidx.dtype == np.int32
    assert rowptr.shape == (N + 1,) and rowptr[0] == 0 and rowptr[-1] == colidx.size
    assert np.all(np.diff(rowptr) >= 0)
    assert colidx.size == 0 or (colidx.min() >= 0 and colidx.max() < N)
    rows = np.repeat(np.arange(N, dtype=np.int64), np.diff(rowptr))
    cols = colidx.astype(np.int64)
    assert not np.any(rows == cols), "self-loop in the CSR"
    # strictly ascending columns within each row: no duplicates
    same_row = rows[1:] == rows[:-1]
    assert np.all(cols[1:][same_row] > cols[:-1][same_row])
    # symmetric: the sorted (row, col) keys equal the sorted (col, row) keys
    assert np.array_equal(np.sort(rows * N + cols), np.sort(cols * N + rows))
    return np.diff(rowptr)


@pytest.fixture(scope="module")
def graphs():
    return {name: inputs.graph(inputs.get_workload(name)) for name in ("C1", "C2", "C3")}


def test_c1_cora_shaped(graphs):
    w = inputs.get_workload("C1")
    assert (w.N, w.K, w.hidden, w.out) == (2708, 1433, 64, 7)
    X = inputs.features(w)
    assert X.shape == (2708, 1433) and X.dtype == np.float32
    assert set(np.unique(X)) <= {0.0, 1.0}
    assert abs(X.mean() - 0.0127) < 5e-4
    deg = check_csr(*graphs["C1"], w.N)
    # preferential attachment with m = 2: node 1 adds one edge, every later node two
    assert deg.sum() == 2 * (1 + 2 * (w.N - 2))
    assert deg.min() >= 1 and deg.max() >= 10 * deg.mean()          # heavy tail


def test_c2_citeseer_shaped(graphs):
    w = inputs.get_workload("C2")
    assert (w.N, w.K, w.hidden, w.out) == (3327, 3703, 64, 6)
    X = inputs.features(w)
    assert set(np.unique(X)) <= {0.0, 1.0} and abs(X.mean() - 0.0085) < 4e-4
    deg = check_csr(*graphs["C2"], w.N)
    assert int(np.sum(deg == 0)) == 33                                # ~1% isolated
    expected = (w.N - 33 - 1) * (0.58 * 1 + 0.42 * 2)                 # undirected edges
    assert abs(deg.sum() / 2 - expected) < 0.03 * expected


def test_c3_pubmed_shaped(graphs):
    w = inputs.get_workload("C3")
    assert (w.N, w.K, w.hidden, w.out) == (19717, 500, 64, 3)
    X = inputs.features(w)
    assert X.min() >= 0.0
    assert abs(np.mean(X != 0) - 0.10) < 2e-3
    norms = np.sqrt((X.astype(np.float64) ** 2).sum(axis=1))
    assert np.all((norms == 0.0) | (np.abs(norms - 1.0) < 1e-5))   # rows L2-normalised
    deg = check_csr(*graphs["C3"], w.N)
    expected = (w.N - 1) * (0.75 * 2 + 0.25 * 3)
    assert abs(deg.sum() / 2 - expected) < 0.02 * expected
    assert deg.min() >= 1                                             # no isolated node


def test_node_ids_are_permuted(graphs):
    # Unpermuted preferential attachment puts the hubs at the lowest ids.
    for name in ("C1", "C3"):
        rowptr, _ = graphs[name]
        deg = np.diff(rowptr)
        head = deg[: deg.size // 20]
        assert head.mean() < 1.5 * deg.mean(), name


def test_chung_lu_at_reduced_size():
    rng = np.random.Generator(np.random.PCG64(7))
    N, edges, cap = 20000, 500_000, 2000
    u, v = inputs.chung_lu(N, edges, 2.0 * edges / N, cap, rng)
    assert u.size == edges and np.all(u < v)
    deg = check_csr(*inputs.edges_to_csr(u, v, N), N)
    assert deg.mean() == 2.0 * edges / N                              # exactly the target
    assert deg.max() >= 10 * deg.mean() and deg.max() <= 1.3 * cap   # truncated power law


def test_erdos_renyi_at_reduced_size():
    rng = np.random.Generator(np.random.PCG64(8))
    N = 4096
    u, v = inputs.erdos_renyi(N, 8 * N, rng)
    deg = check_csr(*inputs.edges_to_csr(u, v, N), N)
    assert deg.sum() == 16 * N                                        # mean CSR degree 16
    assert deg.max() < 16 + 8 * math.sqrt(16)                         # no heavy tail


def test_sweep_points_and_names():
    w = inputs.get_workload("C5_K4096_F256")
    assert (w.N, w.K, w.hidden, w.layers, w.undirected_edges) == (1 << 20, 4096, 256, 1, 8 << 20)
    with pytest.raises(KeyError):
        inputs.get_workload("C6")
    with pytest.raises(AssertionError):
        inputs.get_workload("C5_K100_F64")


def test_seeds_make_inputs_reproducible(graphs):
    w = inputs.get_workload("C1")
    assert np.array_equal(inputs.features(w), inputs.features(w))
    rp, ci = inputs.graph(w)
    assert np.array_equal(rp, graphs["C1"][0]) and np.array_equal(ci, graphs["C1"][1])
    assert not np.array_equal(inputs.features(w, seed=5), inputs.features(w))
    W1, W2 = inputs.layer_weights(w)
    assert np.array_equal(W1, inputs.weights(w.K, w.hidden, 3001))
    assert W2.shape == (w.hidden, w.out)


def test_weights_are_normal_with_variance_one_over_k():
    K, F = 1433, 256
    W = inputs.weights(K, F, seed=3).astype(np.float64)
    assert abs(W.mean()) < 3.0 / math.sqrt(K * F) / math.sqrt(K)
    assert abs(W.std() * math.sqrt(K) - 1.0) < 0.01
