"""Parity of the variant entry points at the Reddit-shaped workload's full size
(C4: N = 232,965, K = 602, F = 128, 114.6M CSR entries, mean degree 492), in
the configuration the benchmark times them: layer 1's back-propagation
(Algorithm 1 with Eqs. bp-H, bp-W), both ablation layers of Sec. 6.3 (one
operand of Eq. 11 kept real), the inductive mean and GraphSAGE-mean layers
(Sec. 6.3, Table 3), sub-row bucketing with buckets of 128 and 512
features (Sec. 4.1) and the layer over a weighted adjacency (Sec. 3's
general a_ij).

The oracle computes what it can one by one at this size:
  - products (Eq. 11 and its variants) on 2048 seeded sampled rows, from the
    oracle's own centring, signs and scales of those rows;
  - layer outputs H on 2048 sampled rows, from the oracle's aggregation over
    every neighbour's product, where the neighbours' products come from the
    GPU's product entry point (checked on the sampled rows; per-step parity);
  - the backward's dL/dH on 2048 sampled rows (the oracle aggregates dH for
    those rows itself) and dL/dW on all K rows of 8 seeded columns, each entry
    summed over all N nodes by the oracle.
These runs take the C4-only paths: hundreds of 128-row tiles per product,
node chunks of the dW reduction, heavy-row blocks and column slabs of the
aggregations.
"""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import (ATOL, RTOL, assert_bits_equal, assert_close, bits_np, check_sum,
                         to_dev)
from paper_2010_07565_gb300 import binding as B
from paper_2010_07565_gb300 import inputs

pytestmark = pytest.mark.gpu

NSAMPLE = 2048


def sample(N, n, seed):
    g = np.random.Generator(np.random.PCG64(seed))
    return np.sort(g.choice(N, size=min(n, N), replace=False))


@pytest.fixture(scope="module")
def c4dev(c4, cuda_device):
    w, d = c4
    g = {k: to_dev(d[k]) for k in ("X", "s", "t", "W1", "rowptr", "colidx")}
    # the oracle's centring, signs and scales of every node (cheap: N x K)
    Y = oracle.centre(d["X"], d["s"], d["t"])
    yield w, d, g, Y
    del g
    torch.cuda.empty_cache()


def nterms_of(rowptr, rows):
    return int(np.diff(rowptr)[rows].max()) + 1


def check_layer_rows(H, rows, rowptr, colidx, zeta, zabs, what, K, agg="gcn", zeta_n=None,
                     zabs_n=None):
    """H[rows] against the oracle's aggregator over the given products; the
    error scale is the aggregator applied to ``zabs`` (the products' |terms|
    where the layer recomputes a real product, else |zeta|), and the sums have
    K product terms and up to the largest sampled degree + 1 aggregation terms."""
    if agg == "gcn":
        ref = oracle.aggregate(rowptr, colidx, zeta, rows=rows)
        scale = oracle.aggregate(rowptr, colidx, zabs, rows=rows)
    elif agg == "mean":
        ref = oracle.aggregate_mean(rowptr, colidx, zeta, rows=rows)
        scale = oracle.aggregate_mean(rowptr, colidx, zabs, rows=rows)
    else:
        ref = oracle.aggregate_sage(rowptr, colidx, zeta, zeta_n, rows=rows)
        scale = oracle.aggregate_sage(rowptr, colidx, zabs, zabs_n, rows=rows)
    Hh = H.cpu().numpy()[rows] if isinstance(H, torch.Tensor) else H
    check_sum(Hh, ref, scale, what, nterms=K + nterms_of(rowptr, rows))


# ------------------------------------------------------------ ablation rows --
@pytest.mark.parametrize("mode", ["weights", "features"])
def test_c4_ablation_layer(cuda_device, c4dev, mode):
    w, d, g, Y = c4dev
    N, K, F = w.N, w.K, w.hidden
    rows = sample(N, NSAMPLE, 61)
    words = (K + 63) // 64
    Z = torch.empty((N, F), device=cuda_device)
    if mode == "weights":
        bits = torch.empty((F, words), dtype=torch.int64, device=cuda_device)
        scl = torch.empty(F, device=cuda_device)
        B.bigcn_pack_weights(g["W1"], bits, scl)
        B.bigcn_real_binary_gemm(g["X"], g["s"], g["t"], bits, scl, Z)
        SB, beta = oracle.weight_binarize(d["W1"])
        ref_rows, abs_rows = oracle.real_binary_product(Y[rows], SB, beta, with_absterm=True)
        # |terms| of every row: beta_j sum_k |y_ik|
        zabs = np.abs(Y).astype(np.float64).sum(axis=1)[:, None] * beta[None, :]
    else:
        bits = torch.empty((N, words), dtype=torch.int64, device=cuda_device)
        scl = torch.empty(N, device=cuda_device)
        B.bigcn_pack_rows(g["X"], g["s"], g["t"], bits, scl)
        pws = torch.empty(B.bigcn_binary_real_gemm_workspace_bytes(K, F), dtype=torch.uint8,
                          device=cuda_device)
        B.bigcn_binary_real_gemm(bits, scl, K, g["W1"], pws, Z)
        SF = oracle.sign(Y[rows])
        alpha_rows = oracle.row_scale(Y[rows])
        ref_rows, abs_rows = oracle.binary_real_product(SF, alpha_rows, d["W1"],
                                                        with_absterm=True)
        alpha = oracle.row_scale(Y)
        zabs = alpha[:, None] * np.abs(d["W1"].astype(np.float64)).sum(axis=0)[None, :]
    ws = torch.empty(B.bigcn_layer_ablation_workspace_bytes(mode, N, K, F), dtype=torch.uint8,
                     device=cuda_device)
    H = torch.empty((N, F), device=cuda_device)
    B.bigcn_layer_forward_ablation(mode, g["X"], g["s"], g["t"], g["W1"], g["rowptr"],
                                   g["colidx"], ws, H)
    torch.cuda.synchronize()
    assert B.device_timeouts() == 0
    Zh = Z.cpu().numpy().astype(np.float64)
    check_sum(Zh[rows], ref_rows, abs_rows, f"C4 {mode}-only product (sampled)", nterms=K)
    check_layer_rows(H, rows, d["rowptr"], d["colidx"], Zh, zabs,
                     f"C4 {mode}-only layer H (sampled)", K)


# ------------------------------------------------------- inductive layers ---
@pytest.mark.parametrize("agg", ["mean", "sage"])
def test_c4_inductive_layer(cuda_device, c4dev, agg):
    w, d, g, Y = c4dev
    N, K, F = w.N, w.K, w.hidden
    rows = sample(N, NSAMPLE, 62)
    Wn = inputs.weights(K, F, 3200 + w.index) if agg == "sage" else None
    Wn_d = to_dev(Wn) if Wn is not None else None
    ws = torch.empty(B.bigcn_inductive_layer_workspace_bytes(agg, N, K, F), dtype=torch.uint8,
                     device=cuda_device)
    H = torch.empty((N, F), device=cuda_device)
    B.bigcn_inductive_layer_forward(agg, g["X"], g["s"], g["t"], g["W1"], g["rowptr"],
                                    g["colidx"], ws, H, W_neigh=Wn_d)
    # the products of every node, with their exact dots, through the product entry point
    bits, alpha = B.pack_rows(g["X"], g["s"], g["t"])

    def product(Wt_d):
        wbits, beta = B.pack_weights(Wt_d)
        _, dots = B.xnor_gemm(bits, alpha, wbits, beta, K, with_dots=True)
        return dots, beta

    dots, beta = product(g["W1"])
    dots_n, beta_n = product(Wn_d) if agg == "sage" else (None, None)
    torch.cuda.synchronize()
    assert B.device_timeouts() == 0
    SF = oracle.sign(Y[rows])
    assert_bits_equal(bits_np(bits)[rows], oracle.pack(SF), "packed rows (sampled)")
    a_h = alpha.cpu().numpy()
    assert_close(a_h[rows], oracle.row_scale(Y[rows]), "alpha (sampled)")
    SB, ref_beta = oracle.weight_binarize(d["W1"])
    assert_close(beta, ref_beta, "beta")
    dh = dots.cpu().numpy()
    assert np.array_equal(dh[rows], oracle.binary_dot(SF, SB))
    z = oracle.zeta(dh, a_h, beta.cpu().numpy())
    if agg == "mean":
        check_layer_rows(H, rows, d["rowptr"], d["colidx"], z, np.abs(z),
                         "C4 mean layer H (sampled)", K, agg="mean")
    else:
        SBn, ref_beta_n = oracle.weight_binarize(Wn)
        assert_close(beta_n, ref_beta_n, "beta (neighbour weights)")
        dnh = dots_n.cpu().numpy()
        assert np.array_equal(dnh[rows], oracle.binary_dot(SF, SBn))
        zn = oracle.zeta(dnh, a_h, beta_n.cpu().numpy())
        check_layer_rows(H, rows, d["rowptr"], d["colidx"], z, np.abs(z),
                         "C4 sage layer H (sampled)", K, agg="sage", zeta_n=zn,
                         zabs_n=np.abs(zn))


# ------------------------------------------------------ weighted adjacency ---
def test_c4_weighted_layer(cuda_device, c4dev):
    """Layer 1 over seeded symmetric edge weights (Sec. 3's general a_ij), as
    the benchmark's --weighted line times it: the weighted degrees of every
    node, the product's dots and H on the sampled rows."""
    w, d, g, Y = c4dev
    N, K, F = w.N, w.K, w.hidden
    rows = sample(N, NSAMPLE, 64)
    vals = inputs.edge_weights(d["rowptr"], d["colidx"], 4100 + w.index)
    v_d = to_dev(vals)
    ws = torch.empty(B.bigcn_weighted_layer_workspace_bytes(N, K, F), dtype=torch.uint8,
                     device=cuda_device)
    H = torch.empty((N, F), device=cuda_device)
    B.bigcn_weighted_layer_forward(g["X"], g["s"], g["t"], g["W1"], g["rowptr"], g["colidx"],
                                   v_d, ws, H)
    dinv = torch.empty(N, device=cuda_device)
    B.bigcn_weighted_dinv(g["rowptr"], v_d, dinv)
    bits, alpha = B.pack_rows(g["X"], g["s"], g["t"])
    wbits, beta = B.pack_weights(g["W1"])
    _, dots = B.xnor_gemm(bits, alpha, wbits, beta, K, with_dots=True)
    torch.cuda.synchronize()
    assert B.device_timeouts() == 0
    del v_d, ws
    assert_close(dinv, 1.0 / np.sqrt(oracle.degree_weighted(d["rowptr"], vals)),
                 "C4 weighted dinv", rtol=1e-6, atol=0.0)
    SF = oracle.sign(Y[rows])
    SB, _ = oracle.weight_binarize(d["W1"])
    dh = dots.cpu().numpy()
    assert np.array_equal(dh[rows], oracle.binary_dot(SF, SB))
    z = oracle.zeta(dh, alpha.cpu().numpy(), beta.cpu().numpy())
    ref = oracle.aggregate_weighted(d["rowptr"], d["colidx"], vals, z, rows=rows)
    scale = oracle.aggregate_weighted(d["rowptr"], d["colidx"], vals, np.abs(z), rows=rows)
    check_sum(H.cpu().numpy()[rows], ref, scale, "C4 weighted layer H (sampled)",
              nterms=K + nterms_of(d["rowptr"], rows))


# ------------------------------------------------------- sub-row bucketing ---
@pytest.mark.parametrize("Bk", [128, 512])
def test_c4_bucketed_layer(cuda_device, c4dev, Bk):
    w, d, g, Y = c4dev
    N, K, F = w.N, w.K, w.hidden
    rows = sample(N, NSAMPLE, 63)
    words, nb = (K + 63) // 64, (K + Bk - 1) // Bk
    a_bits = torch.empty((N, words), dtype=torch.int64, device=cuda_device)
    alpha = torch.empty((N, nb), device=cuda_device)
    b_bits = torch.empty((F, words), dtype=torch.int64, device=cuda_device)
    beta = torch.empty((F, nb), device=cuda_device)
    Z = torch.empty((N, F), device=cuda_device)
    B.bigcn_pack_rows_bucketed(g["X"], g["s"], g["t"], Bk, a_bits, alpha)
    B.bigcn_pack_weights_bucketed(g["W1"], Bk, b_bits, beta)
    B.bigcn_xnor_gemm_bucketed(a_bits, alpha, b_bits, beta, K, Bk, Z)
    ws = torch.empty(B.bigcn_layer_bucketed_workspace_bytes(N, K, F, Bk), dtype=torch.uint8,
                     device=cuda_device)
    H = torch.empty((N, F), device=cuda_device)
    B.bigcn_layer_forward_bucketed(Bk, g["X"], g["s"], g["t"], g["W1"], g["rowptr"],
                                   g["colidx"], ws, H)
    torch.cuda.synchronize()
    Yr = Y[rows]
    SF = oracle.sign(Yr)
    assert_bits_equal(bits_np(a_bits)[rows], oracle.pack(SF), f"B={Bk} packed rows (sampled)")
    ab_rows = oracle.row_scale_bucketed(Yr, Bk)
    assert_close(alpha.cpu().numpy()[rows], ab_rows, f"B={Bk} alpha (sampled)")
    SB = oracle.sign(np.ascontiguousarray(d["W1"].T))
    assert_bits_equal(b_bits, oracle.pack(SB), f"B={Bk} packed weights")
    bb = oracle.weight_scale_bucketed(d["W1"], Bk)
    assert_close(beta, bb, f"B={Bk} beta")
    ref_rows, abs_rows = oracle.zeta_bucketed(SF, ab_rows, SB, bb, Bk, with_absterm=True)
    Zh = Z.cpu().numpy().astype(np.float64)
    check_sum(Zh[rows], ref_rows, abs_rows, f"C4 bucketed product B={Bk} (sampled)", nterms=K)
    # |terms| of every row: sum over buckets of alpha_ib beta_jb (bucket size)
    sizes = np.minimum(Bk, K - Bk * np.arange(nb)).astype(np.float64)
    zabs = (alpha.cpu().numpy().astype(np.float64) * sizes[None, :]) @ \
        np.abs(beta.cpu().numpy().astype(np.float64)).T
    check_layer_rows(H, rows, d["rowptr"], d["colidx"], Zh, zabs,
                     f"C4 bucketed layer B={Bk} H (sampled)", K)


# --------------------------------------------------------------- backward ---
def test_c4_layer_backward(cuda_device, c4dev):
    w, d, g, Y = c4dev
    N, K, F = w.N, w.K, w.hidden
    rows = sample(N, NSAMPLE, 64)
    cols = sample(F, 8, 65)
    # dL/dH1, scaled so that some |dL/dH~| reach the clip of Eq. bp-H
    dH = (60.0 * np.random.Generator(np.random.PCG64(4004)).standard_normal((N, F))
          ).astype(np.float32)
    ws = torch.empty(B.bigcn_layer_backward_workspace_bytes(N, K, F), dtype=torch.uint8,
                     device=cuda_device)
    dW = torch.full((K, F), float("nan"), device=cuda_device)
    dX = torch.full((N, K), float("nan"), device=cuda_device)
    B.bigcn_layer_backward(g["X"], g["s"], g["t"], g["W1"], g["rowptr"], g["colidx"],
                           to_dev(dH), ws, dW, dX=dX)
    torch.cuda.synchronize()
    assert B.device_timeouts() == 0
    SF = oracle.sign(Y)
    alpha = oracle.row_scale(Y)
    SB, beta = oracle.weight_binarize(d["W1"])
    # dW on 8 columns: G's columns summed over all N by the oracle.
    G_cols = oracle.aggregate_t(d["rowptr"], d["colidx"], dH[:, cols].astype(np.float64))
    Wg, wg_abs = oracle.grad_wtilde(SF, alpha, G_cols, with_absterm=True)
    ref_dW = oracle.grad_weight(Wg, SB[cols], beta[cols], np.ascontiguousarray(d["W1"][:, cols]))
    scale_w = np.broadcast_to(wg_abs * (1.0 + beta[cols]), ref_dW.shape)
    check_sum(dW.cpu().numpy()[:, cols], ref_dW, scale_w, "C4 backward dW (8 columns)",
              nterms=N + K)
    # dX on sampled rows (A~^T = A~ for the symmetric CSR).
    G_rows = oracle.aggregate(d["rowptr"], d["colidx"], dH.astype(np.float64), rows=rows)
    Ht, ht_abs = oracle.grad_htilde(G_rows, beta, SB, with_absterm=True)
    ref_dX = oracle.grad_input(Ht)
    dXr = dX.cpu().numpy()[rows].astype(np.float64)
    scale_x = np.broadcast_to(ht_abs[:, None], dXr.shape)
    tol = ATOL + RTOL * np.maximum(np.abs(Ht), scale_x)
    edge = np.abs(np.abs(Ht) - 1.0) <= tol          # either side of the clip is right here
    check_sum(dXr[~edge], ref_dX[~edge], scale_x[~edge], "C4 backward dX (sampled)", nterms=F)
    assert np.all((dXr[edge] == 0.0) | (np.abs(dXr[edge] - Ht[edge]) <= tol[edge]))
    assert 0 < np.count_nonzero(np.abs(Ht) >= 1.0) < Ht.size   # the clip is exercised
