"""Kernel-by-kernel parity of the CUDA path (through the C ABI) with the CPU
oracle, on seeded inputs whose sizes span several tiles with ragged tails,
plus the edge cases of the method (empty graphs, isolated nodes, a high-degree
hub, K not a multiple of 32 or 64, sign of zero, padded strides).

Packed bits and integer dots must be bit-exact; fp32 results must satisfy
|gpu - oracle| <= 1e-6 + 1e-4 |oracle| element by element.
"""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import assert_bits_equal, assert_close, bits_np, padded, to_dev
from paper_2010_07565_gb300 import binding as B
from paper_2010_07565_gb300 import inputs

pytestmark = pytest.mark.gpu


def rng(seed):
    return np.random.Generator(np.random.PCG64(seed))


# ------------------------------------------------------ steps 1+2: pack rows --
PACK_CASES = [(1, 1), (2, 31), (17, 32), (33, 33), (5, 63), (40, 64), (7, 65), (300, 127),
              (129, 128), (64, 129), (1000, 500), (777, 602), (513, 1433), (97, 3703),
              (3, 8192)]


@pytest.mark.parametrize("N,K", PACK_CASES)
@pytest.mark.parametrize("affine", [True, False])
def test_pack_rows(cuda_device, N, K, affine):
    g = rng(N * 7919 + K)
    X = (g.standard_normal((N, K)) * 2.0 + 0.3).astype(np.float32)
    X[0, 0] = 0.0
    if K > 1:
        X[0, 1] = -0.0
    s, t = inputs.bn_stats(X) if affine else (None, None)
    bits, alpha = B.pack_rows(to_dev(X), to_dev(s), to_dev(t))
    Y = oracle.centre(X, s, t)
    assert_bits_equal(bits, oracle.pack(oracle.sign(Y)), "packed rows")
    assert_close(alpha, oracle.row_scale(Y), "alpha")


def test_pack_rows_strided_input_and_extra_words(cuda_device):
    N, K, ldx, words = 333, 150, 161, 5
    g = rng(3)
    X = g.standard_normal((N, K)).astype(np.float32)
    s, t = inputs.bn_stats(X)
    Xd, _ = padded(to_dev(X), N, K, ldx, fill=float("nan"))
    bits = torch.full((N, words), -1, dtype=torch.int64, device=cuda_device)
    alpha = torch.empty(N, dtype=torch.float32, device=cuda_device)
    B.bigcn_pack_rows(Xd, to_dev(s), to_dev(t), bits, alpha)
    Y = oracle.centre(X, s, t)
    assert_bits_equal(bits, oracle.pack(oracle.sign(Y), words=words), "packed rows, 5 words")
    assert_close(alpha, oracle.row_scale(Y), "alpha")


def test_pack_rows_zero_features_and_exact_zeros(cuda_device):
    """All-zero rows, constant columns (variance 0) and -0.0 all pack to +1."""
    N, K = 50, 100
    X = np.zeros((N, K), np.float32)
    X[:, 10] = 3.0                      # constant column: centred to (near) zero
    X[5, :] = -0.0
    X[7, 20:40] = -1.0
    s, t = inputs.bn_stats(X)
    bits, alpha = B.pack_rows(to_dev(X), to_dev(s), to_dev(t))
    Y = oracle.centre(X, s, t)
    assert_bits_equal(bits, oracle.pack(oracle.sign(Y)), "packed rows")
    assert_close(alpha, oracle.row_scale(Y), "alpha")
    bits0, alpha0 = B.pack_rows(to_dev(np.zeros((3, 70), np.float32)))
    assert [int(x) for x in bits_np(bits0)[0]] == [2**64 - 1, 2**6 - 1]
    assert alpha0.cpu().tolist() == [0.0, 0.0, 0.0]


def test_pack_rows_bernoulli_features(cuda_device):
    """{0,1} features as in the citation workloads, centred by their own BN stats."""
    g = rng(11)
    X = inputs.draw_features(g, 2000, 1433, "bernoulli", 0.0127)
    s, t = inputs.bn_stats(X)
    bits, alpha = B.pack_rows(to_dev(X), to_dev(s), to_dev(t))
    Y = oracle.centre(X, s, t)
    assert_bits_equal(bits, oracle.pack(oracle.sign(Y)), "packed rows")
    assert_close(alpha, oracle.row_scale(Y), "alpha")


# --------------------------------------------------- step 3: pack weights ----
@pytest.mark.parametrize("K,F", [(1, 1), (64, 3), (65, 7), (128, 41), (500, 64), (602, 128),
                                 (1433, 64), (3703, 6), (8192, 256), (33, 300)])
def test_pack_weights(cuda_device, K, F):
    W = inputs.weights(K, F, seed=K * 31 + F)
    W[0, 0] = 0.0
    bits, beta = B.pack_weights(to_dev(W))
    SB, ref_beta = oracle.weight_binarize(W)
    assert_bits_equal(bits, oracle.pack(SB), "packed weight columns")
    assert_close(beta, ref_beta, "beta")


def test_pack_weights_strided(cuda_device):
    K, F, ldw = 200, 37, 45
    W = inputs.weights(K, F, seed=1)
    Wd, _ = padded(to_dev(W), K, F, ldw, fill=float("nan"))
    bits = torch.full((F, 6), -1, dtype=torch.int64, device=cuda_device)
    beta = torch.empty(F, dtype=torch.float32, device=cuda_device)
    B.bigcn_pack_weights(Wd, bits, beta)
    SB, ref_beta = oracle.weight_binarize(W)
    assert_bits_equal(bits, oracle.pack(SB, words=6), "packed weight columns, 6 words")
    assert_close(beta, ref_beta, "beta")


# ------------------------------------------------------- step 4: the GEMM ----
GEMM_CASES = [(1, 1, 1), (17, 3, 64), (129, 7, 65), (300, 41, 128), (257, 64, 602),
              (130, 128, 1433), (64, 256, 500), (200, 6, 3703), (5, 300, 8192),
              (1000, 64, 64), (131, 17, 129), (33, 33, 31)]


def random_signs(g, n, K):
    return np.where(g.random((n, K)) < 0.5, 1, -1).astype(np.int8)


@pytest.mark.parametrize("N,F,K", GEMM_CASES)
def test_xnor_gemm(cuda_device, N, F, K):
    g = rng(N * 1009 + F * 13 + K)
    SF, SB = random_signs(g, N, K), random_signs(g, F, K)
    alpha = g.uniform(0.1, 2.0, N).astype(np.float32)
    beta = g.uniform(0.001, 0.1, F).astype(np.float32)
    Z, dots = B.xnor_gemm(to_dev(oracle.pack(SF)), to_dev(alpha), to_dev(oracle.pack(SB)),
                          to_dev(beta), K, with_dots=True)
    ref_dot = oracle.binary_dot(SF, SB)
    assert np.array_equal(dots.cpu().numpy(), ref_dot)
    assert_close(Z, oracle.zeta(ref_dot, alpha.astype(np.float64), beta.astype(np.float64)),
                 "Z")


def test_xnor_gemm_extreme_dots_and_strided_output(cuda_device):
    """Rows equal / opposite to the columns give dot = +-K; Z written with ldz > F."""
    K, F, N, ldz = 8192, 5, 70, 9
    g = rng(5)
    SB = random_signs(g, F, K)
    SF = np.concatenate([SB, -SB, random_signs(g, N - 2 * F, K)])
    alpha = np.ones(N, np.float32)
    beta = np.full(F, 0.5, np.float32)
    Zd, Zbuf = padded(torch.zeros((N, F), device=cuda_device), N, F, ldz, fill=7.0)
    dots = torch.empty((N, F), dtype=torch.int32, device=cuda_device)
    B.bigcn_xnor_gemm(to_dev(oracle.pack(SF)), to_dev(alpha), to_dev(oracle.pack(SB)),
                      to_dev(beta), K, Zd, dots)
    d = dots.cpu().numpy()
    assert np.all(np.diag(d[:F]) == K) and np.all(np.diag(d[F:2 * F]) == -K)
    assert np.array_equal(d, oracle.binary_dot(SF, SB))
    assert_close(Zd, oracle.zeta(d, alpha.astype(np.float64), beta.astype(np.float64)), "Z")
    assert torch.all(Zbuf[:, F:] == 7.0), "padding of Z was overwritten"


# -------------------------------------------------------- step 5: the SpMM ---
SPMM_CASES = [
    # (N, mean degree, hub degree, F)
    (1, 0.0, 0, 1), (2, 1.0, 0, 3), (50, 0.0, 0, 7), (333, 4.0, 0, 6), (1000, 8.0, 200, 41),
    (2048, 16.0, 0, 64), (777, 3.0, 500, 128), (500, 5.0, 0, 256), (301, 4.0, 0, 300),
    (129, 2.8, 0, 2), (4096, 2.0, 0, 5), (200, 6.0, 150, 1)]


@pytest.mark.parametrize("N,deg,hub,F", SPMM_CASES)
def test_spmm_norm(cuda_device, N, deg, hub, F):
    rowptr, colidx = inputs.random_graph(N, deg, seed=N + F, hub_degree=hub)
    Z = rng(N * 3 + F).standard_normal((N, F)).astype(np.float32)
    H = B.spmm_norm(to_dev(rowptr), to_dev(colidx), to_dev(Z))
    assert_close(H, oracle.aggregate(rowptr, colidx, Z.astype(np.float64)), "H")


def test_spmm_star_hub_of_degree_20000(cuda_device):
    N, F = 20001, 41
    leaves = np.arange(1, N, dtype=np.int64)
    rowptr, colidx = inputs.edges_to_csr(np.zeros_like(leaves), leaves, N)
    assert rowptr[1] == 20000
    Z = rng(8).standard_normal((N, F)).astype(np.float32)
    H = B.spmm_norm(to_dev(rowptr), to_dev(colidx), to_dev(Z))
    assert_close(H, oracle.aggregate(rowptr, colidx, Z.astype(np.float64)), "H")


def test_spmm_strided_and_sqrt_degree_fixed_point(cuda_device):
    """A~ v = v for v_i = sqrt(dhat_i), through the GPU path with ldz, ldh > F."""
    rowptr, colidx = inputs.random_graph(3000, 6.0, seed=4, hub_degree=1000)
    v = np.sqrt(oracle.degree(rowptr)).astype(np.float32)[:, None]
    Zd, _ = padded(to_dev(v), 3000, 1, 3, fill=float("nan"))
    Hd, Hbuf = padded(torch.zeros((3000, 1), device=cuda_device), 3000, 1, 5, fill=9.0)
    B.bigcn_spmm_norm(to_dev(rowptr), to_dev(colidx), Zd, Hd)
    assert_close(Hd, v.astype(np.float64), "A~ sqrt(dhat)")
    assert torch.all(Hbuf[:, 1:] == 9.0)


def test_spmm_empty_graph_is_identity(cuda_device):
    N, F = 1000, 64
    Z = rng(2).standard_normal((N, F)).astype(np.float32)
    rowptr = np.zeros(N + 1, np.int64)
    H = B.spmm_norm(to_dev(rowptr), to_dev(np.empty(0, np.int32)), to_dev(Z))
    assert np.array_equal(H.cpu().numpy(), Z)


def test_spmm_malformed_csr_stays_in_bounds(cuda_device):
    """Out-of-range column indices are skipped and row ranges clamped: the
    result is defined by those rules and nothing is read out of bounds."""
    N, F = 6, 4
    rowptr = np.array([0, 2, 3, 3, 9, 9, 12], np.int64)    # row 3 runs past nnz = 10
    colidx = np.array([1, 99, 0, 4, -5, 2, 1, 0, 5, 3], np.int32)
    Z = rng(3).standard_normal((N, F)).astype(np.float32)
    H = B.spmm_norm(to_dev(rowptr), to_dev(colidx), to_dev(Z)).cpu().numpy()
    assert np.all(np.isfinite(H[:4]))
    # row 0: self + neighbour 1 (99 skipped); its dhat counts both entries
    d = lambda r: 1.0 + (rowptr[r + 1] - rowptr[r])
    expect0 = (Z[0] / d(0) + Z[1] / np.sqrt(d(0) * d(1)))
    np.testing.assert_allclose(H[0], expect0, rtol=1e-5, atol=1e-6)


# ------------------------------------------------------------- fused layer ---
@pytest.mark.parametrize("N,K,F,deg,hub", [(1, 1, 1, 0.0, 0), (301, 203, 19, 4.0, 40),
                                           (1000, 602, 128, 8.0, 300), (2708, 1433, 64, 4.0, 0),
                                           (517, 64, 7, 3.0, 0), (129, 128, 41, 10.0, 100)])
def test_layer_forward_matches_oracle(cuda_device, N, K, F, deg, hub):
    case = inputs.layer_case(N, K, F, seed=N + K + F, mean_degree=deg, hub_degree=hub)
    H = B.layer_forward(to_dev(case["X"]), to_dev(case["W"]), to_dev(case["rowptr"]),
                        to_dev(case["colidx"]), to_dev(case["s"]), to_dev(case["t"]))
    ref = oracle.layer_forward(case["X"], case["W"], case["rowptr"], case["colidx"],
                               case["s"], case["t"])
    assert_close(H, ref["H"], "fused layer H")


def test_layer_forward_equals_step_by_step(cuda_device):
    case = inputs.layer_case(1500, 300, 64, seed=77, mean_degree=6.0, hub_degree=700)
    d = {k: to_dev(v) for k, v in case.items()}
    bits, alpha = B.pack_rows(d["X"], d["s"], d["t"])
    wbits, beta = B.pack_weights(d["W"])
    Z = B.xnor_gemm(bits, alpha, wbits, beta, 300)
    H_steps = B.spmm_norm(d["rowptr"], d["colidx"], Z).cpu().numpy()
    H_fused = B.layer_forward(d["X"], d["W"], d["rowptr"], d["colidx"], d["s"], d["t"])
    # The fused layer keeps Z factored (integer dots, row scale, column scale)
    # and so adds the same fp32 terms in another order: equal to the steps
    # within the parity tolerance, not bit for bit.
    assert_close(H_fused, H_steps.astype(np.float64), "fused vs steps")


def test_layer_forward_strided_and_workspace_reuse(cuda_device):
    N, K, F = 400, 130, 10
    case = inputs.layer_case(N, K, F, seed=9)
    Xd, _ = padded(to_dev(case["X"]), N, K, 140, fill=float("nan"))
    Wd, _ = padded(to_dev(case["W"]), K, F, 12, fill=float("nan"))
    Hd, Hbuf = padded(torch.zeros((N, F), device=cuda_device), N, F, 16, fill=5.0)
    ws = torch.full((B.bigcn_layer_workspace_bytes(N, K, F),), 0xAB, dtype=torch.uint8,
                    device=cuda_device)
    ref = oracle.layer_forward(case["X"], case["W"], case["rowptr"], case["colidx"],
                               case["s"], case["t"])
    for _ in range(2):
        B.bigcn_layer_forward(Xd, to_dev(case["s"]), to_dev(case["t"]), Wd,
                              to_dev(case["rowptr"]), to_dev(case["colidx"]), ws, Hd)
        assert_close(Hd, ref["H"], "H (strided)")
    assert torch.all(Hbuf[:, F:] == 5.0)


# ---------------------------------------------------------- argument errors --
def test_invalid_arguments_return_status_and_leave_outputs(cuda_device):
    X = torch.ones((10, 70), device=cuda_device)
    bits = torch.full((10, 2), 123, dtype=torch.int64, device=cuda_device)
    alpha = torch.full((10,), 4.0, device=cuda_device)
    short_bits = torch.full((10, 1), 123, dtype=torch.int64, device=cuda_device)
    with pytest.raises(B.BigcnError) as e:
        B.bigcn_pack_rows(X, None, None, short_bits, alpha)      # words < ceil(K/64)
    assert e.value.status == 1
    with pytest.raises(B.BigcnError) as e:
        B.bigcn_pack_rows(X, torch.ones(70, device=cuda_device), None, bits, alpha)
    assert e.value.status == 1
    misaligned = torch.empty(10 * 70 + 1, device=cuda_device)[1:].view(10, 70)
    raw = torch.empty(2 * 10 * 2 + 1, dtype=torch.int32, device=cuda_device)
    st = B.lib().bigcn_pack_rows(misaligned.data_ptr(), 10, 70, 70, None, None,
                                 raw.data_ptr() + 4, 2, alpha.data_ptr(), None)
    assert st == 2
    torch.cuda.synchronize()
    assert torch.all(bits == 123) and torch.all(alpha == 4.0)
    Z = torch.zeros((10, 4), device=cuda_device)
    rowptr = torch.zeros(11, dtype=torch.int64, device=cuda_device)
    with pytest.raises(B.BigcnError):
        B.bigcn_spmm_norm(rowptr, torch.empty(0, dtype=torch.int32, device=cuda_device), Z, Z)
    ws = torch.empty(16, dtype=torch.uint8, device=cuda_device)
    with pytest.raises(B.BigcnError):                              # workspace too small
        B.bigcn_layer_forward(X, None, None, torch.ones((70, 4), device=cuda_device), rowptr,
                              torch.empty(0, dtype=torch.int32, device=cuda_device), ws, Z)


# ------------------------------------------------- fused two-layer forward ---
@pytest.mark.parametrize("N,K,Fh,Fo,deg,hub", [
    (1, 1, 4, 1, 0.0, 0),             # a single isolated node
    (301, 203, 64, 7, 4.0, 40),        # fused path (Fh % 4 == 0, Fo <= 64)
    (1000, 602, 128, 41, 8.0, 300),    # fused, two packed words per hidden row
    (517, 130, 16, 3, 3.0, 0),         # fused, narrowest lane groups
    (400, 150, 30, 5, 4.0, 0),         # Fh not a multiple of 4: unfused path
    (300, 100, 64, 80, 4.0, 0),        # Fo > 64: unfused path
    (257, 70, 200, 9, 5.0, 0),         # Fh > 128: unfused path
])
def test_forward_2layer_matches_oracle(cuda_device, N, K, Fh, Fo, deg, hub):
    case = inputs.layer_case(N, K, Fh, seed=N + K + Fh + Fo, mean_degree=deg, hub_degree=hub)
    W2 = inputs.weights(Fh, Fo, seed=N + 99)
    d = {k: to_dev(v) for k, v in case.items()}
    ws = torch.empty(B.bigcn_forward_2layer_workspace_bytes(N, K, Fh, Fo), dtype=torch.uint8,
                     device=cuda_device)
    H1 = torch.full((N, Fh), float("nan"), device=cuda_device)
    out = torch.full((N, Fo), float("nan"), device=cuda_device)
    B.bigcn_forward_2layer(d["X"], d["s"], d["t"], d["W"], to_dev(W2), d["rowptr"],
                           d["colidx"], ws, out, H1=H1)
    ref1 = oracle.layer_forward(case["X"], case["W"], case["rowptr"], case["colidx"],
                                case["s"], case["t"])
    assert_close(H1, ref1["H"], "H1")
    ref2 = oracle.layer_forward(H1.cpu().numpy(), W2, case["rowptr"], case["colidx"])
    assert_close(out, ref2["H"], "logits")
    # without H1 requested: the same logits
    out2 = torch.full((N, Fo), float("nan"), device=cuda_device)
    B.bigcn_forward_2layer(d["X"], d["s"], d["t"], d["W"], to_dev(W2), d["rowptr"],
                           d["colidx"], ws, out2)
    assert torch.equal(out, out2)


# Rows of X whose starts sit off every vector alignment (odd row strides, a
# base 4 or 12 bytes past a 16-byte boundary), rows shorter than one 32-wide
# chunk or than 16 bytes, Citeseer-shaped rows on the split front (several
# warps per row), more row groups than resident CTAs, and rows too long for
# the fused front (80 KB: packing and product as separate kernels).
@pytest.mark.parametrize("N,K,ldx,offset,Fh,centred", [
    (333, 1, 1, 0, 8, True),          # one feature per row
    (333, 3, 5, 1, 8, False),         # rows shorter than 16 bytes, odd stride
    (200, 9, 9, 1, 33, True),         # one partial chunk, 33 hidden columns
    (700, 3703, 3703, 0, 64, True),   # Citeseer-shaped rows (stride 14812 bytes)
    (700, 3703, 3705, 3, 64, True),   # same rows, odd stride, base 12 bytes past
    (5000, 1433, 1437, 1, 16, True),  # more row groups than resident CTAs
    (64, 20000, 20001, 1, 128, True), # rows of 80 KB: packing, then the product
])
def test_forward_2layer_front_unaligned_rows(cuda_device, N, K, ldx, offset, Fh, centred):
    Fo = 5
    case = inputs.layer_case(N, K, Fh, seed=N + K + ldx, mean_degree=3.0, centred=centred)
    W2 = inputs.weights(Fh, Fo, seed=K + 5)
    d = {k: to_dev(v) for k, v in case.items()}
    buf = torch.full((N * ldx + offset + 8,), float("nan"), device=cuda_device)
    X = buf[offset:offset + N * ldx].view(N, ldx)[:, :K]
    X.copy_(d["X"])
    ws = torch.empty(B.bigcn_forward_2layer_workspace_bytes(N, K, Fh, Fo), dtype=torch.uint8,
                     device=cuda_device)
    H1 = torch.full((N, Fh), float("nan"), device=cuda_device)
    out = torch.full((N, Fo), float("nan"), device=cuda_device)
    B.bigcn_forward_2layer(X, d["s"], d["t"], d["W"], to_dev(W2), d["rowptr"], d["colidx"],
                           ws, out, H1=H1)
    ref1 = oracle.layer_forward(case["X"], case["W"], case["rowptr"], case["colidx"],
                                case["s"], case["t"])
    assert_close(H1, ref1["H"], "H1")
    ref2 = oracle.layer_forward(H1.cpu().numpy(), W2, case["rowptr"], case["colidx"])
    assert_close(out, ref2["H"], "logits")
    assert B.device_timeouts() == 0


# Above K = 32767 the dots no longer fit 16 bits: layer 1's Z' stays fp32.
@pytest.mark.parametrize("N,K,Fh,Fo", [(40, 33000, 16, 3), (300, 32767, 8, 5)])
def test_forward_2layer_k_at_and_past_the_16_bit_limit(cuda_device, N, K, Fh, Fo):
    case = inputs.layer_case(N, K, Fh, seed=N + K, mean_degree=3.0)
    W2 = inputs.weights(Fh, Fo, seed=K)
    d = {k: to_dev(v) for k, v in case.items()}
    ws = torch.empty(B.bigcn_forward_2layer_workspace_bytes(N, K, Fh, Fo), dtype=torch.uint8,
                     device=cuda_device)
    H1 = torch.full((N, Fh), float("nan"), device=cuda_device)
    out = torch.full((N, Fo), float("nan"), device=cuda_device)
    B.bigcn_forward_2layer(d["X"], d["s"], d["t"], d["W"], to_dev(W2), d["rowptr"], d["colidx"],
                           ws, out, H1=H1)
    ref1 = oracle.layer_forward(case["X"], case["W"], case["rowptr"], case["colidx"],
                                case["s"], case["t"])
    assert_close(H1, ref1["H"], "H1")
    ref2 = oracle.layer_forward(H1.cpu().numpy(), W2, case["rowptr"], case["colidx"])
    assert_close(out, ref2["H"], "logits")
    H = B.layer_forward(d["X"], d["W"], d["rowptr"], d["colidx"], d["s"], d["t"])
    assert_close(H, ref1["H"], "one layer")


# Predicted classes: the argmax of each logits row, lowest index on ties
# (numpy's rule), computed in the last aggregation's epilogue, or by a separate
# kernel when the rows span more than one column slab (Fo > 256).
@pytest.mark.parametrize("N,K,Fh,Fo,dup", [
    (2708, 1433, 64, 7, False),     # Cora-shaped
    (1000, 602, 128, 41, True),      # ties: W2 columns 3 and 7 equal 0 and 5
    (300, 100, 64, 80, False),       # unfused layer 2, one slab
    (257, 70, 32, 300, True),        # two slabs: the separate argmax kernel
])
def test_forward_2layer_predictions(cuda_device, N, K, Fh, Fo, dup):
    case = inputs.layer_case(N, K, Fh, seed=N + Fo, mean_degree=4.0)
    W2 = inputs.weights(Fh, Fo, seed=Fo)
    if dup:
        W2[:, 3], W2[:, 7] = W2[:, 0], W2[:, 5]
    d = {k: to_dev(v) for k, v in case.items()}
    ws = torch.empty(B.bigcn_forward_2layer_workspace_bytes(N, K, Fh, Fo), dtype=torch.uint8,
                     device=cuda_device)
    H1 = torch.empty((N, Fh), device=cuda_device)
    out = torch.empty((N, Fo), device=cuda_device)
    pred = torch.full((N,), -7, dtype=torch.int32, device=cuda_device)
    B.bigcn_forward_2layer(d["X"], d["s"], d["t"], d["W"], to_dev(W2), d["rowptr"], d["colidx"],
                           ws, out, H1=H1, pred=pred)
    logits = out.cpu().numpy()
    p = pred.cpu().numpy()
    assert np.array_equal(p, np.argmax(logits, axis=1)), "argmax of the GPU's own logits"
    if dup:
        assert not np.any((p == 3) | (p == 7)), "a tie goes to the lower index"
    ref2 = oracle.layer_forward(H1.cpu().numpy(), W2, case["rowptr"], case["colidx"])["H"]
    top2 = np.sort(ref2, axis=1)[:, -2:]
    clear = (top2[:, 1] - top2[:, 0]) > 2 * (1e-6 + 1e-4 * np.abs(top2[:, 1]))
    assert np.array_equal(p[clear], np.argmax(ref2, axis=1)[clear]), "oracle argmax"
    assert clear.mean() > 0.5


def test_forward_2layer_records_one_event_per_kernel_boundary(cuda_device):
    N, K, Fh, Fo = 500, 300, 64, 7
    case = inputs.layer_case(N, K, Fh, seed=3)
    d = {k: to_dev(v) for k, v in case.items()}
    W2 = to_dev(inputs.weights(Fh, Fo, seed=4))
    n = B.bigcn_forward_2layer_launches(N, K, Fh, Fo)
    # K <= 2048: both aggregations on the tensor cores, any Fh <= 128 fused
    assert n == 4 and B.bigcn_forward_2layer_launches(N, K, 30, 7) == 4
    # longer rows keep the CUDA-core aggregation, fused only for Fh % 4 == 0
    assert B.bigcn_forward_2layer_launches(N, 3000, 30, 7) == 6
    assert B.bigcn_forward_2layer_launches(N, 3000, 64, 7) == 4
    assert B.bigcn_forward_2layer_launches(N, 3000, 200, 7) == 7
    assert B.bigcn_forward_2layer_launches(N, 8192, 256, 7) == 7
    events = [torch.cuda.Event(enable_timing=True) for _ in range(n + 1)]
    for e in events:
        e.record()
    torch.cuda.synchronize()
    ws = torch.empty(B.bigcn_forward_2layer_workspace_bytes(N, K, Fh, Fo), dtype=torch.uint8,
                     device=cuda_device)
    out = torch.empty((N, Fo), device=cuda_device)
    B.bigcn_forward_2layer(d["X"], d["s"], d["t"], d["W"], W2, d["rowptr"], d["colidx"], ws,
                           out, events=events)
    torch.cuda.synchronize()
    spans = [events[q].elapsed_time(events[q + 1]) for q in range(n)]
    assert all(t >= 0.0 for t in spans)
    assert events[0].elapsed_time(events[n]) > 0.0


def hub_graph(N, hubs, seed, mean_degree=4.0):
    """Random graph plus hub rows: (node, degree) pairs joined to random others.
    Rows far above the mean degree (here 2049 to 8190 neighbours) take the
    kernels' whole-block path."""
    g = rng(seed)
    rowptr, colidx = inputs.random_graph(N, mean_degree, seed=seed)
    rows = np.repeat(np.arange(N), np.diff(rowptr))
    keys = [np.minimum(rows, colidx) * N + np.maximum(rows, colidx)]
    for node, deg in hubs:
        others = g.choice(np.delete(np.arange(N), node), size=deg, replace=False)
        keys.append(np.minimum(node, others) * N + np.maximum(node, others))
    keys = np.unique(np.concatenate(keys).astype(np.int64))
    return inputs.edges_to_csr(keys // N, keys % N, N)


HUBS = [(3, 2049), (7, 2500), (250, 5000), (256, 2100), (4000, 8190), (8999, 3000)]


@pytest.mark.parametrize("F", [1, 6, 41, 128, 300])
@pytest.mark.parametrize("prescaled", [False, True])
def test_spmm_many_heavy_rows(cuda_device, F, prescaled):
    N = 9000
    rowptr, colidx = hub_graph(N, HUBS, seed=F)
    deg = np.diff(rowptr)
    assert (deg > 2048).sum() >= len(HUBS)
    Z = rng(F + 1).standard_normal((N, F)).astype(np.float32)
    Zd, H = to_dev(Z), torch.empty((N, F), device=cuda_device)
    if prescaled:
        B.bigcn_spmm_prescaled(to_dev(rowptr), to_dev(colidx), Zd, H)
        dinv = 1.0 / np.sqrt(oracle.degree(rowptr))
        ref = oracle.aggregate(rowptr, colidx, Z.astype(np.float64) / dinv[:, None])
    else:
        B.bigcn_spmm_norm(to_dev(rowptr), to_dev(colidx), Zd, H)
        ref = oracle.aggregate(rowptr, colidx, Z.astype(np.float64))
    assert_close(H, ref, f"H (F={F}, heavy rows)")


@pytest.mark.parametrize("Fh,Fo", [(128, 41), (64, 7), (16, 3)])
def test_forward_2layer_heavy_rows(cuda_device, Fh, Fo):
    N, K = 9000, 300
    rowptr, colidx = hub_graph(N, HUBS, seed=Fh + Fo)
    g = rng(Fo)
    X = g.standard_normal((N, K)).astype(np.float32)
    s, t = inputs.bn_stats(X)
    W1, W2 = inputs.weights(K, Fh, seed=5), inputs.weights(Fh, Fo, seed=6)
    ws = torch.empty(B.bigcn_forward_2layer_workspace_bytes(N, K, Fh, Fo), dtype=torch.uint8,
                     device=cuda_device)
    H1 = torch.empty((N, Fh), device=cuda_device)
    out = torch.empty((N, Fo), device=cuda_device)
    B.bigcn_forward_2layer(to_dev(X), to_dev(s), to_dev(t), to_dev(W1), to_dev(W2),
                           to_dev(rowptr), to_dev(colidx), ws, out, H1=H1)
    ref1 = oracle.layer_forward(X, W1, rowptr, colidx, s, t)
    assert_close(H1, ref1["H"], "H1 with heavy rows")
    ref2 = oracle.layer_forward(H1.cpu().numpy(), W2, rowptr, colidx)
    assert_close(out, ref2["H"], "logits with heavy rows")


# ------------------------------------------- tensor-core path of step 4 ------
TC_CASES = [(128, 32, 128), (129, 33, 129), (300, 64, 200), (1000, 128, 1000),
            (257, 256, 8192), (77, 257, 300), (512, 100, 3703), (1, 40, 602), (384, 41, 64 * 40)]


@pytest.mark.parametrize("N,F,K", TC_CASES)
def test_xnor_gemm_tensor_core_path(cuda_device, N, F, K):
    """Shapes at and around the tensor-core product's K and F thresholds with
    fewer 128-row tiles than SMs, which the POPC kernel takes: dots exact at
    +-K. The tcgen05 kernels themselves, at the row counts that select them:
    test_gpu_tc_product.py."""
    g = rng(N + 7 * F + 13 * K)
    SF, SB = random_signs(g, N, K), random_signs(g, F, K)
    if N >= 2 and F >= 2:
        SF[0] = SB[0]            # dot = +K
        SF[1] = -SB[1]           # dot = -K
    alpha = g.uniform(0.1, 2.0, N).astype(np.float32)
    beta = g.uniform(0.001, 0.1, F).astype(np.float32)
    Z, dots = B.xnor_gemm(to_dev(oracle.pack(SF)), to_dev(alpha), to_dev(oracle.pack(SB)),
                          to_dev(beta), K, with_dots=True)
    ref_dot = oracle.binary_dot(SF, SB)
    got = dots.cpu().numpy()
    assert np.array_equal(got, ref_dot), f"{int((got != ref_dot).sum())} dots differ"
    assert_close(Z, oracle.zeta(ref_dot, alpha.astype(np.float64), beta.astype(np.float64)), "Z")
    assert B.device_timeouts() == 0


def test_xnor_gemm_tensor_core_degree_scaled(cuda_device):
    N, F, K = 700, 128, 602
    g = rng(99)
    SF, SB = random_signs(g, N, K), random_signs(g, F, K)
    alpha = g.uniform(0.1, 2.0, N).astype(np.float32)
    beta = g.uniform(0.001, 0.1, F).astype(np.float32)
    rowptr, _ = inputs.random_graph(N, 6.0, seed=3, hub_degree=200)
    Z = torch.empty((N, F), device=cuda_device)
    B.bigcn_xnor_gemm_degscaled(to_dev(oracle.pack(SF)), to_dev(alpha), to_dev(oracle.pack(SB)),
                                to_dev(beta), K, to_dev(rowptr), Z)
    dinv = 1.0 / np.sqrt(oracle.degree(rowptr))
    ref = oracle.zeta(oracle.binary_dot(SF, SB), alpha.astype(np.float64),
                      beta.astype(np.float64)) * dinv[:, None]
    assert_close(Z, ref, "Z'")
    assert B.device_timeouts() == 0


# The tensor-core aggregations on long rows: one-row windows (mean degree at
# least 24), hub rows split over a whole block, widths that are not multiples
# of 16 (padding tiles), and K at the fp16 limit of the dots (2048).
@pytest.mark.parametrize("N,K,Fh,Fo,deg,hub", [
    (3000, 602, 128, 41, 40.0, 2500),    # Reddit-like widths, hubs on the block path
    (2000, 2048, 64, 7, 30.0, 0),        # largest K of the fp16 dots
    (1500, 300, 40, 17, 60.0, 1200),     # widths not multiples of 16
    (800, 100, 16, 3, 24.0, 700),        # one tile each side
])
def test_forward_2layer_long_rows(cuda_device, N, K, Fh, Fo, deg, hub):
    case = inputs.layer_case(N, K, Fh, seed=N + K + Fh, mean_degree=deg, hub_degree=hub)
    W2 = inputs.weights(Fh, Fo, seed=N + Fo)
    d = {k: to_dev(v) for k, v in case.items()}
    ws = torch.empty(B.bigcn_forward_2layer_workspace_bytes(N, K, Fh, Fo), dtype=torch.uint8,
                     device=cuda_device)
    H1 = torch.full((N, Fh), float("nan"), device=cuda_device)
    out = torch.full((N, Fo), float("nan"), device=cuda_device)
    pred = torch.full((N,), -7, dtype=torch.int32, device=cuda_device)
    B.bigcn_forward_2layer(d["X"], d["s"], d["t"], d["W"], to_dev(W2), d["rowptr"],
                           d["colidx"], ws, out, H1=H1, pred=pred)
    torch.cuda.synchronize()
    assert B.device_timeouts() == 0
    ref1 = oracle.layer_forward(case["X"], case["W"], case["rowptr"], case["colidx"],
                                case["s"], case["t"])
    assert_close(H1, ref1["H"], "H1")
    ref2 = oracle.layer_forward(H1.cpu().numpy(), W2, case["rowptr"], case["colidx"])
    assert_close(out, ref2["H"], "logits")
    assert np.array_equal(pred.cpu().numpy(), np.argmax(out.cpu().numpy(), axis=1))
