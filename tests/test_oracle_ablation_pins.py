"""Pins of the oracle's ablation products (Sec. 6.3's "binarize features only"
and "binarize weights only" rows) to facts that do not come from the
oracle's own formulas:

* where binarization is the identity -- every column of W is +-c_j (then
  W~ = W) or every centred row is +-c_i (then H~ = Y) -- the product is the
  textbook matrix product, computed here by numpy; the shapes are not square,
  so a transposed operand or a wrong index fails;
* binarizing the other operand as well gives Bi-GCN's own Eq. 11-12 product,
  whose integer form the existing pins check: Y W~ with Y = H~ and H~ W with
  W = W~ both equal alpha_i beta_j dot_ij;
* the weights-only product is linear in Y; the features-only one is odd and
  positively homogeneous in Y (sign and the mean-|y| scale commute with
  positive scaling and flip with negation of a row without zeros);
* |terms|: absterm equals the product of |Y| with |W~| (resp. |H~| with |W|),
  and bounds |zeta|.
"""
import numpy as np
import pytest

import oracle
from paper_2010_07565_gb300 import inputs


def rng(seed):
    return np.random.Generator(np.random.PCG64(seed))


def pm(g, shape):
    return np.where(g.random(shape) < 0.5, -1.0, 1.0)


def test_weights_only_equals_the_matrix_product_when_columns_are_plus_minus_c():
    g = rng(1)
    N, K, F = 13, 37, 5
    Y = g.standard_normal((N, K)).astype(np.float32)
    c = np.array([0.5, 2.0, 0.125, 1.0, 3.0])
    Wt = (pm(g, (K, F)) * c[None, :]).astype(np.float32)          # W~ = W exactly
    SB, beta = oracle.weight_binarize(Wt)
    np.testing.assert_array_equal(beta, c)
    z = oracle.real_binary_product(Y, SB, beta)
    np.testing.assert_allclose(z, Y.astype(np.float64) @ Wt.astype(np.float64),
                               rtol=1e-12, atol=1e-12)


def test_features_only_equals_the_matrix_product_when_rows_are_plus_minus_c():
    g = rng(2)
    N, K, F = 11, 29, 7
    c = g.uniform(0.25, 4.0, N).astype(np.float32)
    Y = (pm(g, (N, K)) * c[:, None]).astype(np.float32)           # H~ = Y exactly
    Wt = g.standard_normal((K, F)).astype(np.float32)
    SF = oracle.sign(Y)
    alpha = oracle.row_scale(Y)
    np.testing.assert_allclose(alpha, c.astype(np.float64), rtol=1e-15)
    z = oracle.binary_real_product(SF, alpha, Wt)
    np.testing.assert_allclose(z, Y.astype(np.float64) @ Wt.astype(np.float64),
                               rtol=1e-12, atol=1e-12)


def test_binarizing_the_other_operand_gives_the_bi_gcn_product():
    g = rng(3)
    N, K, F = 9, 70, 6
    Y = g.standard_normal((N, K)).astype(np.float32)
    Wt = g.standard_normal((K, F)).astype(np.float32)
    SF, alpha = oracle.sign(Y), oracle.row_scale(Y)
    SB, beta = oracle.weight_binarize(Wt)
    dot = oracle.binary_dot(SF, SB)
    # Y W~ with Y := H~ (alpha rounded to fp32, the real operand's type).
    a32 = alpha.astype(np.float32)
    Htilde = (a32[:, None] * SF).astype(np.float32)
    tol = 1e-13 * K * alpha.max() * beta.max()      # rounding of the double sums where dot = 0
    np.testing.assert_allclose(oracle.real_binary_product(Htilde, SB, beta),
                               oracle.zeta(dot, a32.astype(np.float64), beta), rtol=1e-12,
                               atol=tol)
    # H~ W with W := W~ (beta rounded to fp32).
    b32 = beta.astype(np.float32)
    Wtilde = (SB.T * b32[None, :]).astype(np.float32)
    np.testing.assert_allclose(oracle.binary_real_product(SF, alpha, Wtilde),
                               oracle.zeta(dot, alpha, b32.astype(np.float64)), rtol=1e-12,
                               atol=tol)


def test_weights_only_is_linear_in_the_features():
    g = rng(4)
    N, K, F = 8, 40, 3
    Y1 = g.standard_normal((N, K)).astype(np.float32)
    Y2 = g.standard_normal((N, K)).astype(np.float32)
    SB, beta = oracle.weight_binarize(g.standard_normal((K, F)).astype(np.float32))
    a, b = 0.75, -2.5          # Y1 a + Y2 b is exact in fp32 only approximately: use float64 sums
    lhs = oracle.real_binary_product((a * Y1 + b * Y2).astype(np.float32), SB, beta)
    rhs = a * oracle.real_binary_product(Y1, SB, beta) + b * oracle.real_binary_product(Y2, SB, beta)
    _, mag = oracle.real_binary_product(np.abs(a * Y1) + np.abs(b * Y2), SB, beta,
                                        with_absterm=True)
    assert np.all(np.abs(lhs - rhs) <= 1e-6 * mag)


def test_features_only_is_odd_and_positively_homogeneous():
    g = rng(5)
    N, K, F = 8, 40, 4
    Y = g.standard_normal((N, K)).astype(np.float32)
    assert np.all(Y != 0)
    Wt = g.standard_normal((K, F)).astype(np.float32)

    def prod(V):
        return oracle.binary_real_product(oracle.sign(V), oracle.row_scale(V), Wt)

    z = prod(Y)
    np.testing.assert_allclose(prod(-Y), -z, rtol=1e-13, atol=1e-13)
    np.testing.assert_allclose(prod(4.0 * Y), 4.0 * z, rtol=1e-13, atol=1e-13)


def test_absterm_is_the_product_of_magnitudes_and_bounds_zeta():
    g = rng(6)
    N, K, F = 7, 33, 5
    Y = g.standard_normal((N, K)).astype(np.float32)
    Wt = g.standard_normal((K, F)).astype(np.float32)
    SB, beta = oracle.weight_binarize(Wt)
    z, a = oracle.real_binary_product(Y, SB, beta, with_absterm=True)
    np.testing.assert_allclose(a, np.abs(Y).astype(np.float64).sum(1)[:, None] * beta[None, :],
                               rtol=1e-12)
    assert np.all(np.abs(z) <= a * (1 + 1e-12))
    SF, alpha = oracle.sign(Y), oracle.row_scale(Y)
    z, a = oracle.binary_real_product(SF, alpha, Wt, with_absterm=True)
    np.testing.assert_allclose(a, alpha[:, None] * np.abs(Wt).astype(np.float64).sum(0)[None, :],
                               rtol=1e-12)
    assert np.all(np.abs(z) <= a * (1 + 1e-12))


@pytest.mark.parametrize("binarize", ["weights", "features"])
def test_ablation_layer_without_edges_is_the_product(binarize):
    case = inputs.layer_case(20, 50, 4, seed=7, mean_degree=0.0)
    assert case["rowptr"][-1] == 0
    r = oracle.layer_forward_ablation(case["X"], case["W"], case["rowptr"], case["colidx"],
                                      binarize, case["s"], case["t"])
    np.testing.assert_array_equal(r["H"], r["zeta"])
    np.testing.assert_array_equal(r["scale"], r["zeta_abs"])


def test_ablation_both_is_the_bi_gcn_layer():
    case = inputs.layer_case(30, 64, 5, seed=8)
    r = oracle.layer_forward_ablation(case["X"], case["W"], case["rowptr"], case["colidx"],
                                      "both", case["s"], case["t"])
    ref = oracle.layer_forward(case["X"], case["W"], case["rowptr"], case["colidx"],
                               case["s"], case["t"])
    np.testing.assert_array_equal(r["H"], ref["H"])
    assert np.all(np.abs(r["H"]) <= r["scale"] * (1 + 1e-12))
