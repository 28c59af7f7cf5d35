"""Pins of the CPU oracle to the paper and to mathematics (no GPU).

Every oracle routine is checked here against something other than itself:
brute force on tiny inputs, an independent popcount evaluation of the packed
words, the least-squares optimality that defines the scales, exact special
cases where the binarized layer reduces to a dense matrix product, and
invariants of the normalised adjacency operator. A plausible slip in the
oracle (a dropped self-loop, a transposed operand, a wrong divisor, sign(0)
taken as -1, a mis-ordered bit) fails at least one test below.
"""
import numpy as np
import pytest

import oracle
from paper_2010_07565_gb300 import inputs


def rng(seed):
    return np.random.Generator(np.random.PCG64(seed))


# ------------------------------------------------------------ sign, Eq. 8 ----
def test_sign_of_zero_and_negative_zero_is_plus_one():
    v = np.array([0.0, -0.0, 1e-45, -1e-45, 3.0, -3.0, np.inf, -np.inf], np.float32)
    assert oracle.sign(v).tolist() == [1, 1, 1, -1, 1, -1, 1, -1]


# ------------------------------------------------------ packed layout -------
@pytest.mark.parametrize("K", [1, 2, 31, 32, 33, 63, 64, 65, 127, 128, 129, 200])
def test_pack_layout_decodes_bit_by_bit(K):
    S = np.where(rng(K).random((5, K)) < 0.5, 1, -1).astype(np.int8)
    bits = oracle.pack(S)
    W = oracle.words_for(K)
    assert bits.shape == (5, W)
    for r in range(5):
        word_ints = [int(x) for x in bits[r]]
        for k in range(64 * W):
            b = (word_ints[k // 64] >> (k % 64)) & 1
            if k < K:
                assert b == (1 if S[r, k] > 0 else 0)
            else:
                assert b == 0, "pad bits must be zero"


def test_pack_extra_words_are_zero():
    S = np.ones((3, 70), np.int8)
    bits = oracle.pack(S, words=4)
    assert [int(x) for x in bits[0]] == [2**64 - 1, 2**6 - 1, 0, 0]


# ---------------------------------------- Eq. 11 == Eq. 12 (XNOR, popcount) --
@pytest.mark.parametrize("K", list(range(1, 201)))
def test_xnor_popcount_identity_on_packed_words(K):
    """Eq. 12 evaluates Eq. 11's +-1 inner product with XNOR and a bit count.
    With pad bits 0 in both operands: dot = K - 2 popc(a ^ b)
    = 2 popc(~(a ^ b) restricted to K bits) - K."""
    g = rng(1000 + K)
    SF = np.where(g.random((3, K)) < 0.5, 1, -1).astype(np.int8)
    SB = np.where(g.random((4, K)) < 0.5, 1, -1).astype(np.int8)
    dot = oracle.binary_dot(SF, SB)
    A, B = oracle.pack(SF), oracle.pack(SB)
    mask = (1 << K) - 1
    for i in range(3):
        a = sum(int(w) << (64 * q) for q, w in enumerate(A[i]))
        for j in range(4):
            b = sum(int(w) << (64 * q) for q, w in enumerate(B[j]))
            assert dot[i, j] == K - 2 * bin(a ^ b).count("1")
            assert dot[i, j] == 2 * bin(~(a ^ b) & mask).count("1") - K


def test_binary_dot_matches_float_matmul_of_signs():
    g = rng(7)
    SF = np.where(g.random((37, 301)) < 0.5, 1, -1).astype(np.int8)
    SB = np.where(g.random((11, 301)) < 0.5, 1, -1).astype(np.int8)
    ref = SF.astype(np.float64) @ SB.astype(np.float64).T
    assert np.array_equal(oracle.binary_dot(SF, SB), ref.astype(np.int32))


def test_binary_dot_extremes():
    K = 97
    plus = np.ones((1, K), np.int8)
    assert oracle.binary_dot(plus, plus)[0, 0] == K
    assert oracle.binary_dot(plus, -plus)[0, 0] == -K


# --------------------------------------------------------- scales, Eq. 4/7 --
def _ls_err(y, a):
    s = np.where(y >= 0, 1.0, -1.0)
    return float(((y - a * s) ** 2).sum())


def test_row_scale_is_the_least_squares_optimum():
    """Eq. 7's scale (read as mean |y|) minimises ||y - a sign(y)||^2."""
    Y = rng(3).standard_normal((6, 129)).astype(np.float32)
    alpha = oracle.row_scale(Y)
    y64 = Y.astype(np.float64)
    for i in range(6):
        e0 = _ls_err(y64[i], alpha[i])
        for f in (1 - 1e-3, 1 + 1e-3):
            assert _ls_err(y64[i], alpha[i] * f) > e0
        # the optimum of a quadratic in a is where its derivative vanishes
        s = np.where(y64[i] >= 0, 1.0, -1.0)
        assert abs(float((s * (y64[i] - alpha[i] * s)).sum())) < 1e-9


def test_row_scale_closed_forms():
    c = 0.375
    pattern = np.where(rng(5).random(77) < 0.5, 1.0, -1.0)
    Y = np.stack([c * pattern, np.abs(np.linspace(0.5, 2.0, 77)),
                  np.zeros(77)]).astype(np.float32)
    alpha = oracle.row_scale(Y)
    assert alpha[0] == c
    S = oracle.sign(Y)
    assert np.array_equal(alpha[0] * S[0], Y[0])   # the approximation of Eq. 9 is exact
    assert np.all(S[1] == 1)
    assert alpha[1] == pytest.approx(float(np.abs(Y[1].astype(np.float64)).mean()), rel=1e-15)
    assert alpha[2] == 0.0 and np.all(S[2] == 1)


def test_weight_scale_and_sign_per_column():
    """Eq. 3/4 act on columns of W (K x F): constant columns give |c|, and the
    scale is the least-squares optimum of Eq. 5's approximation."""
    K, F = 50, 3
    W = np.empty((K, F), np.float32)
    W[:, 0] = -0.25
    W[:, 1] = 2.0
    W[:, 2] = rng(9).standard_normal(K)
    SB, beta = oracle.weight_binarize(W)
    assert SB.shape == (F, K)
    assert np.all(SB[0] == -1) and np.all(SB[1] == 1)
    assert beta[0] == 0.25 and beta[1] == 2.0
    w = W[:, 2].astype(np.float64)
    assert np.array_equal(SB[2], np.where(w >= 0, 1, -1))
    for f in (1 - 1e-3, 1 + 1e-3):
        assert _ls_err(w, beta[2] * f) > _ls_err(w, beta[2])


# --------------------------------------------- special case: dense matmul ---
def test_binarized_product_equals_dense_product_on_binary_inputs():
    """If every row of H is +-c_i and every column of W is +-d_j, binarization
    loses nothing (Eq. 5 and Eq. 9 hold with equality) and Eq. 11's zeta is
    exactly the full-precision product H W of Eq. 1."""
    g = rng(11)
    N, K, F = 23, 70, 9
    c = 2.0 ** g.integers(-4, 4, N)
    d = 2.0 ** g.integers(-6, 2, F)
    H = (np.where(g.random((N, K)) < 0.5, 1.0, -1.0) * c[:, None]).astype(np.float32)
    W = (np.where(g.random((K, F)) < 0.5, 1.0, -1.0) * d[None, :]).astype(np.float32)
    Y = oracle.centre(H)
    SF, alpha = oracle.sign(Y), oracle.row_scale(Y)
    SB, beta = oracle.weight_binarize(W)
    z = oracle.zeta(oracle.binary_dot(SF, SB), alpha, beta)
    assert np.array_equal(z, H.astype(np.float64) @ W.astype(np.float64))


# ------------------------------------------------- aggregation, Eq. 1 / 13 --
def dense_operator(rowptr, colidx):
    """A~ = D^-1/2 (A + I) D^-1/2 built densely from the CSR (Eq. 1)."""
    N = rowptr.shape[0] - 1
    A = np.zeros((N, N))
    for i in range(N):
        A[i, colidx[rowptr[i]:rowptr[i + 1]]] = 1.0
    Ahat = A + np.eye(N)
    dhat = Ahat.sum(axis=1)
    Dm = np.diag(1.0 / np.sqrt(dhat))
    return Dm @ Ahat @ Dm


def test_aggregate_equals_dense_normalised_adjacency():
    rowptr, colidx = inputs.random_graph(40, 5.0, seed=21, hub_degree=25)
    z = rng(2).standard_normal((40, 3))
    H = oracle.aggregate(rowptr, colidx, z)
    np.testing.assert_allclose(H, dense_operator(rowptr, colidx) @ z, rtol=1e-13, atol=1e-14)


def test_aggregate_operator_is_symmetric():
    rowptr, colidx = inputs.random_graph(30, 4.0, seed=22)
    Op = oracle.aggregate(rowptr, colidx, np.eye(30))   # column j = A~ e_j
    np.testing.assert_allclose(Op, Op.T, rtol=0, atol=1e-15)


def test_aggregate_fixes_sqrt_degree_vector():
    """(A~ v)_i = dhat_i^-1/2 sum_j ahat_ij = dhat_i^1/2 for v = dhat^1/2."""
    rowptr, colidx = inputs.random_graph(300, 6.0, seed=23, hub_degree=120)
    v = np.sqrt(oracle.degree(rowptr))[:, None]
    np.testing.assert_allclose(oracle.aggregate(rowptr, colidx, v), v, rtol=1e-13)


def test_degree_counts_the_self_loop():
    rowptr = np.array([0, 2, 3, 4, 4], np.int64)
    assert oracle.degree(rowptr).tolist() == [3.0, 2.0, 2.0, 1.0]


def test_isolated_node_is_the_identity_and_rows_subset():
    rowptr = np.array([0, 1, 2, 2], np.int64)
    colidx = np.array([1, 0], np.int32)
    z = np.array([[1.0, -2.0], [3.0, 4.0], [5.0, 6.0]])
    H = oracle.aggregate(rowptr, colidx, z)
    assert H[2].tolist() == [5.0, 6.0]
    np.testing.assert_allclose(H[0], (z[0] + z[1]) / 2.0)
    Hs, A = oracle.aggregate(rowptr, colidx, z, rows=[2, 0], with_absterm=True)
    assert np.array_equal(Hs, H[[2, 0]])
    np.testing.assert_allclose(A[1], (np.abs(z[0]) + np.abs(z[1])) / 2.0)


def test_empty_graph_is_the_identity():
    rowptr = np.zeros(5, np.int64)
    z = rng(4).standard_normal((4, 2))
    assert np.array_equal(oracle.aggregate(rowptr, np.empty(0, np.int32), z), z)


@pytest.mark.parametrize("rowptr,colidx", [
    ([1, 1, 2], [0, 1]),          # rowptr[0] != 0
    ([0, 2, 1], [1, 0]),          # not monotone
    ([0, 1, 2], [1, 2]),          # column out of range
    ([0, 1, 2], [-1, 0]),         # negative column
])
def test_aggregate_rejects_malformed_csr(rowptr, colidx):
    with pytest.raises(ValueError):
        oracle.aggregate(np.array(rowptr, np.int64), np.array(colidx, np.int32),
                         np.zeros((2, 1)))


# ------------------------------------------------------- centring, Sec. 6.2 --
def test_centring_gives_zero_mean_unit_variance():
    g = rng(31)
    X = (g.standard_normal((4000, 17)) * g.uniform(0.5, 3.0, 17) + g.uniform(-2, 2, 17))
    X = X.astype(np.float32)
    s, t = inputs.bn_stats(X)
    Y = oracle.centre(X, s, t).astype(np.float64)
    np.testing.assert_allclose(Y.mean(axis=0), 0.0, atol=1e-5)
    np.testing.assert_allclose(Y.var(axis=0), 1.0, atol=1e-4)


def test_centring_is_one_fp32_fma():
    X = np.array([[1.0000001, -3.5, 0.0]], np.float32)
    s = np.array([3.0, 0.5, 2.0], np.float32)
    t = np.array([-3.0000002, 1.75, -0.0], np.float32)
    Y = oracle.centre(X, s, t)
    exact = X.astype(np.float64) * s + t          # exact in double here
    assert np.array_equal(Y, exact.astype(np.float32))
    assert Y[0, 1] == 0.0 and oracle.sign(Y)[0, 1] == 1


def test_identity_centring_keeps_values_bit_for_bit():
    X = rng(6).standard_normal((3, 9)).astype(np.float32)
    X[0, 0] = -0.0
    Y = oracle.centre(X)
    assert np.array_equal(Y.view(np.uint32), X.view(np.uint32))


# -------------------------------------------------------------- composition --
def test_layer_forward_composes_the_steps():
    case = inputs.layer_case(50, 130, 5, seed=41)
    r = oracle.layer_forward(case["X"], case["W"], case["rowptr"], case["colidx"],
                             case["s"], case["t"])
    dense = dense_operator(case["rowptr"], case["colidx"])
    np.testing.assert_allclose(r["H"], dense @ r["zeta"], rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(r["absterm"], np.abs(dense) @ np.abs(r["zeta"]),
                               rtol=1e-12, atol=1e-14)
    assert r["bits"].shape == (50, 3) and r["wbits"].shape == (5, 3)
