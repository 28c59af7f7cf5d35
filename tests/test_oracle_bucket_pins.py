"""Pins of the oracle's sub-row bucketing (Sec. 4.1: buckets of B consecutive
values, each with its own scale) to facts outside the oracle's own formulas:

* B = 1: every entry is its own bucket, the scales are |y_ik| and |W_kj|, so
  alpha_ik sign(y_ik) = y_ik exactly and zeta must be the textbook Y W
  (numpy); non-square shapes catch a transposed operand;
* B >= K: one bucket per row / column, i.e. Bi-GCN's own product (pinned by
  the existing tests through the integer dots);
* additivity: zeta with buckets equals the sum over buckets of Bi-GCN's
  product restricted to each bucket's columns;
* rows and columns that are +-c_b within each bucket lose nothing: zeta = Y W;
* each bucket's scale is the least-squares optimum of || v - a sign(v) ||
  over that bucket (the derivative vanishes, perturbations are worse).
"""
import numpy as np
import pytest

import oracle


def rng(seed):
    return np.random.Generator(np.random.PCG64(seed))


def bucketed(Y, Wt, B):
    SF, SB = oracle.sign(Y), oracle.sign(np.ascontiguousarray(Wt.T))
    return oracle.zeta_bucketed(SF, oracle.row_scale_bucketed(Y, B), SB,
                                oracle.weight_scale_bucketed(Wt, B), B, with_absterm=True)


def test_one_entry_per_bucket_is_the_exact_product():
    g = rng(1)
    Y = g.standard_normal((9, 37)).astype(np.float32)
    Wt = g.standard_normal((37, 5)).astype(np.float32)
    z, mag = bucketed(Y, Wt, 1)
    ref = Y.astype(np.float64) @ Wt.astype(np.float64)
    np.testing.assert_allclose(z, ref, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(mag, np.abs(Y).astype(np.float64) @ np.abs(Wt).astype(np.float64),
                               rtol=1e-12)


@pytest.mark.parametrize("B", [70, 71, 500])
def test_one_bucket_is_the_bi_gcn_product(B):
    g = rng(2)
    Y = g.standard_normal((11, 70)).astype(np.float32)
    Wt = g.standard_normal((70, 6)).astype(np.float32)
    SF, (SB, beta) = oracle.sign(Y), oracle.weight_binarize(Wt)
    ref = oracle.zeta(oracle.binary_dot(SF, SB), oracle.row_scale(Y), beta)
    z, _ = bucketed(Y, Wt, B)
    np.testing.assert_allclose(z, ref, rtol=1e-13, atol=1e-13)


@pytest.mark.parametrize("B", [2, 16, 64, 100])
def test_buckets_add_up_bi_gcn_products_of_their_columns(B):
    g = rng(3)
    K = 250
    Y = g.standard_normal((13, K)).astype(np.float32)
    Wt = g.standard_normal((K, 7)).astype(np.float32)
    total = np.zeros((13, 7))
    for k0 in range(0, K, B):
        Yb, Wb = np.ascontiguousarray(Y[:, k0:k0 + B]), np.ascontiguousarray(Wt[k0:k0 + B])
        SB, beta = oracle.weight_binarize(Wb)
        total += oracle.zeta(oracle.binary_dot(oracle.sign(Yb), SB), oracle.row_scale(Yb), beta)
    z, _ = bucketed(Y, Wt, B)
    np.testing.assert_allclose(z, total, rtol=1e-12, atol=1e-12)


def test_plus_minus_c_per_bucket_loses_nothing():
    g = rng(4)
    N, K, F, B = 6, 200, 4, 64
    nb = oracle.buckets(K, B)
    cy = g.uniform(0.5, 2.0, (N, nb))
    cw = g.uniform(0.5, 2.0, (F, nb))
    kb = np.arange(K) // B
    Y = (np.where(g.random((N, K)) < 0.5, -1.0, 1.0) * cy[:, kb]).astype(np.float32)
    Wt = (np.where(g.random((K, F)) < 0.5, -1.0, 1.0) * cw[:, kb].T).astype(np.float32)
    z, _ = bucketed(Y, Wt, B)
    np.testing.assert_allclose(z, Y.astype(np.float64) @ Wt.astype(np.float64), rtol=1e-12,
                               atol=1e-12)


def test_each_bucket_scale_is_the_least_squares_optimum():
    g = rng(5)
    Y = g.standard_normal((3, 130)).astype(np.float32)
    B = 64
    a = oracle.row_scale_bucketed(Y, B)
    S = oracle.sign(Y).astype(np.float64)
    for i in range(3):
        for b in range(oracle.buckets(130, B)):
            v, sgn = Y[i, b * B:(b + 1) * B].astype(np.float64), S[i, b * B:(b + 1) * B]
            err = lambda s: np.sum((v - s * sgn) ** 2)
            assert np.sum((v - a[i, b] * sgn) * sgn) == pytest.approx(0.0, abs=1e-9)
            assert err(a[i, b]) < err(a[i, b] * 1.001) and err(a[i, b]) < err(a[i, b] * 0.999)
    bw = oracle.weight_scale_bucketed(np.ascontiguousarray(Y.T), B)
    np.testing.assert_allclose(bw, a, rtol=1e-15)          # the same definition on columns
