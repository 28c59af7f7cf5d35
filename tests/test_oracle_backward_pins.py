"""Pins of the oracle's back-propagation (Algorithm 1, Eqs. bp-H and bp-W)
to mathematics that does not come from the oracle's own formulas:

* adjoint identities -- the gradients of Algorithm 1 are the transposes of
  the forward's linear maps, so <A~^T dH, Z> = <dH, A~ Z> (with the forward's
  separately written gather), <dL/dW~, V> = <G, H~ V> and
  <dL/dH~, U> = <G, U W~^T> for random dH, Z, V, U: a transposed operand or
  a wrong index fails them;
* special cases: no edges (A~ = I), one node (an outer product);
* Eq. bp-H's indicator at and around |g| = 1 (strict inequality);
* Eq. bp-W by finite differences: its first term is the exact derivative of
  sum g * W~ through the column scale beta_j = mean |W_:,j| with the signs
  held, and its second the derivative of sum g * beta_j * htanh(W) with beta
  held -- the straight-through estimator 1(|r| < 1) is htanh's derivative.
"""
import numpy as np
import pytest

import oracle
from paper_2010_07565_gb300 import inputs


def rng(seed):
    return np.random.Generator(np.random.PCG64(seed))


def random_csr(N, p, seed, symmetric=True):
    g = rng(seed)
    A = g.random((N, N)) < p
    np.fill_diagonal(A, False)
    if symmetric:
        A = A | A.T
    rows, cols = np.nonzero(A)
    return inputs.edges_to_csr(rows, cols, N)


@pytest.mark.parametrize("symmetric", [True, False])
def test_transpose_aggregation_is_the_adjoint_of_the_forward_one(symmetric):
    N, F = 40, 5
    rowptr, colidx = random_csr(N, 0.15, seed=3 + symmetric, symmetric=symmetric)
    g = rng(11)
    dH, Z = g.standard_normal((N, F)), g.standard_normal((N, F))
    lhs = np.sum(oracle.aggregate_t(rowptr, colidx, dH) * Z)
    rhs = np.sum(dH * oracle.aggregate(rowptr, colidx, Z))
    assert lhs == pytest.approx(rhs, rel=1e-12)


def test_transpose_aggregation_equals_the_forward_one_on_a_symmetric_graph():
    N, F = 60, 3
    rowptr, colidx = random_csr(N, 0.1, seed=5)
    dH = rng(12).standard_normal((N, F))
    np.testing.assert_allclose(oracle.aggregate_t(rowptr, colidx, dH),
                               oracle.aggregate(rowptr, colidx, dH), rtol=1e-12, atol=1e-14)


def test_transpose_aggregation_without_edges_is_the_identity():
    N, F = 9, 4
    rowptr = np.zeros(N + 1, np.int64)
    dH = rng(13).standard_normal((N, F))
    assert np.array_equal(oracle.aggregate_t(rowptr, np.zeros(0, np.int32), dH), dH)


def layer_state(N, K, F, seed):
    g = rng(seed)
    Y = g.standard_normal((N, K)).astype(np.float32)
    Wt = g.standard_normal((K, F)).astype(np.float32)   # |W| > 1 occurs
    SF = oracle.sign(Y)
    alpha = oracle.row_scale(Y)
    SB, beta = oracle.weight_binarize(Wt)
    G = g.standard_normal((N, F))
    return g, Y, Wt, SF, alpha, SB, beta, G


def test_weight_gradient_is_the_adjoint_of_the_product_in_w():
    g, Y, Wt, SF, alpha, SB, beta, G = layer_state(30, 70, 6, seed=21)
    Wg = oracle.grad_wtilde(SF, alpha, G)
    V = g.standard_normal((70, 6))
    Htilde = alpha[:, None] * SF.astype(np.float64)            # H~ = diag(alpha) sign(Y)
    assert np.sum(Wg * V) == pytest.approx(np.sum(G * (Htilde @ V)), rel=1e-11)


def test_input_gradient_is_the_adjoint_of_the_product_in_h():
    g, Y, Wt, SF, alpha, SB, beta, G = layer_state(30, 70, 6, seed=22)
    Ht = oracle.grad_htilde(G, beta, SB)
    U = g.standard_normal((30, 70))
    Wtilde = (beta[:, None] * SB.astype(np.float64)).T          # W~[k,j] = beta_j sign(W_kj)
    assert np.sum(Ht * U) == pytest.approx(np.sum(G * (U @ Wtilde)), rel=1e-11)


def test_weight_gradient_of_one_node_is_an_outer_product():
    g, Y, Wt, SF, alpha, SB, beta, G = layer_state(1, 10, 3, seed=23)
    Wg, absterm = oracle.grad_wtilde(SF, alpha, G, with_absterm=True)
    for k in range(10):
        for j in range(3):
            assert Wg[k, j] == alpha[0] * SF[0, k] * G[0, j]
    np.testing.assert_array_equal(absterm, np.abs(alpha[0] * G[0]))


def test_input_gradient_clipping_is_strict_at_one():
    Ht = np.array([[-1.5, -1.0, -0.999999, 0.0, 0.5, 0.9999999, 1.0, 1.0000001, 7.0]])
    np.testing.assert_array_equal(oracle.grad_input(Ht),
                                  [[0.0, 0.0, -0.999999, 0.0, 0.5, 0.9999999, 0.0, 0.0, 0.0]])


def test_weight_gradient_matches_finite_differences():
    """Eq. bp-W = d/dW [sum g * beta(W) * B] (signs held)
                + d/dW [sum g * beta * htanh(W)] (scale held), per entry."""
    K, F = 12, 4
    g = rng(31)
    Wt = (1.3 * g.standard_normal((K, F))).astype(np.float32)
    Wg = g.standard_normal((K, F))
    SB, beta = oracle.weight_binarize(Wt)
    dW = oracle.grad_weight(Wg, SB, beta, Wt)
    W = Wt.astype(np.float64)
    Bk = SB.T.astype(np.float64)                                 # K x F signs, held

    def f_scale(Wv):                                             # through beta_j = mean |W_:,j|
        return np.sum(Wg * (np.abs(Wv).mean(axis=0)[None, :] * Bk))

    def f_ste(Wv):                                               # sign replaced by htanh
        return np.sum(Wg * (beta[None, :] * np.clip(Wv, -1.0, 1.0)))

    h = 1e-6
    checked = 0
    for k in range(K):
        for j in range(F):
            w = W[k, j]
            if abs(w) < 1e-3 or abs(abs(w) - 1.0) < 1e-3:
                continue                                         # kinks of |.| and htanh
            E = np.zeros_like(W)
            E[k, j] = h
            fd = ((f_scale(W + E) - f_scale(W - E)) + (f_ste(W + E) - f_ste(W - E))) / (2 * h)
            assert dW[k, j] == pytest.approx(fd, rel=1e-6, abs=1e-8), (k, j)
            checked += 1
    assert checked > 40
    assert np.any(np.abs(W) > 1.0) and np.any(np.abs(W) < 1.0)   # both STE branches seen


def test_layer_backward_composes_the_steps():
    case = inputs.layer_case(25, 40, 5, seed=41)
    dH = rng(42).standard_normal((25, 5))
    r = oracle.layer_backward(case["X"], case["W"], case["rowptr"], case["colidx"], dH,
                              case["s"], case["t"])
    np.testing.assert_array_equal(r["dX"], np.where(np.abs(r["Ht"]) < 1.0, r["Ht"], 0.0))
    assert r["Wg"].shape == (40, 5) and r["dW"].shape == (40, 5) and r["dX"].shape == (25, 40)
