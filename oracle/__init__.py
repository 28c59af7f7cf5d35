"""Plain CPU oracle of the Bi-GCN layer forward (Wang et al., CVPR 2021).

TEST INFRASTRUCTURE. Only the tests, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg import this package; the product path never does,
and the two share no code. The arithmetic lives in ``bigcn_oracle.c``; this
module marshals numpy arrays into it and composes the steps in the paper's
order:

    step 1  centring (Sec. 6.2)            oracle_centre
    step 2  F = sign(Y), row scale (Eq. 8, Eq. 7)       oracle_sign, oracle_row_scale
    step 3  B = sign(W), column scale (Eq. 3, Eq. 4)    oracle_weight_binarize
    step 4  zeta = alpha beta (F . B) (Eq. 11, Eq. 12)  oracle_binary_dot, oracle_zeta
    step 5  H = A~ zeta (Eq. 13, Eq. 1)                 oracle_aggregate
            ... with a weighted A (Sec. 3)              oracle_degree_weighted,
                                                        oracle_aggregate_weighted

the ablation variants of step 4 (Sec. 6.3, one operand kept real):

    zeta = Y W~   (weights binarized only)              oracle_real_binary_product
    zeta = H~ W   (features binarized only)             oracle_binary_real_product

sub-row bucketing (Sec. 4.1, buckets of B consecutive values):

    per-bucket alpha, beta; zeta = sum_b alpha_ib beta_jb dot_b
        oracle_row_scale_bucketed, oracle_weight_scale_bucketed, oracle_zeta_bucketed

the inductive aggregators (Sec. 6.3, Table 3, GraphSAGE's definitions):

    H_i = mean over N(i) u {i} of zeta_j            oracle_aggregate_mean
    H_i = zself_i + mean over N(i) of zneigh_j      oracle_aggregate_sage

and the layer's back-propagation (Algorithm 1, Eqs. bp-H, bp-W):

    G = A~^T dH                      oracle_aggregate_t
    dL/dW~ = H~^T G, dL/dH~ = G W~^T oracle_grad_wtilde, oracle_grad_htilde
    dL/dH (clipped), dL/dW (STE)     oracle_grad_input, oracle_grad_weight

Naming follows the layer's C interface: ``alpha`` is the per-node scale (the
paper's beta, Eq. 7) and ``beta`` the per-weight-column scale (the paper's
alpha, Eq. 4). Floating-point results are float64; the only fp32 arithmetic is
the centring, whose result decides the sign bits and so must round exactly as
the kernel's does.
"""
from __future__ import annotations

import ctypes
import threading

import numpy as np

from . import build as _build

_lib = None
_lock = threading.Lock()

_f32p = np.ctypeslib.ndpointer(np.float32, flags="C_CONTIGUOUS")
_f64p = np.ctypeslib.ndpointer(np.float64, flags="C_CONTIGUOUS")
_i8p = np.ctypeslib.ndpointer(np.int8, flags="C_CONTIGUOUS")
_i32p = np.ctypeslib.ndpointer(np.int32, flags="C_CONTIGUOUS")
_i64p = np.ctypeslib.ndpointer(np.int64, flags="C_CONTIGUOUS")
_u64p = np.ctypeslib.ndpointer(np.uint64, flags="C_CONTIGUOUS")
_vp = ctypes.c_void_p
_i32 = ctypes.c_int32
_i64 = ctypes.c_int64


def lib() -> ctypes.CDLL:
    """Load (building first if needed) the oracle's shared library."""
    global _lib
    with _lock:
        if _lib is None:
            h = ctypes.CDLL(_build.build())
            h.oracle_centre.argtypes = [_f32p, _i64, _i32, _i64, _vp, _vp, _f32p]
            h.oracle_centre.restype = None
            h.oracle_sign.argtypes = [_f32p, _i64, _i8p]
            h.oracle_sign.restype = None
            h.oracle_row_scale.argtypes = [_f32p, _i64, _i32, _f64p]
            h.oracle_row_scale.restype = None
            h.oracle_weight_binarize.argtypes = [_f32p, _i32, _i32, _i64, _i8p, _f64p]
            h.oracle_weight_binarize.restype = None
            h.oracle_pack.argtypes = [_i8p, _i64, _i32, _i32, _u64p]
            h.oracle_pack.restype = None
            h.oracle_binary_dot.argtypes = [_i8p, _i64, _i8p, _i32, _i32, _i32p]
            h.oracle_binary_dot.restype = None
            h.oracle_zeta.argtypes = [_i32p, _f64p, _f64p, _i64, _i32, _f64p]
            h.oracle_zeta.restype = None
            h.oracle_degree.argtypes = [_i64p, _i64, _f64p]
            h.oracle_degree.restype = None
            h.oracle_aggregate.argtypes = [_i64p, _i32p, _i64, _f64p, _i32, _vp, _i64,
                                           _f64p, _vp]
            h.oracle_aggregate.restype = ctypes.c_int
            h.oracle_aggregate_t.argtypes = [_i64p, _i32p, _i64, _f64p, _i32, _f64p]
            h.oracle_aggregate_t.restype = ctypes.c_int
            h.oracle_grad_wtilde.argtypes = [_i8p, _f64p, _f64p, _i64, _i32, _i32, _f64p, _vp]
            h.oracle_grad_wtilde.restype = None
            h.oracle_grad_htilde.argtypes = [_f64p, _f64p, _i8p, _i64, _i32, _i32, _f64p, _vp]
            h.oracle_grad_htilde.restype = None
            h.oracle_grad_input.argtypes = [_f64p, _i64, _f64p]
            h.oracle_grad_input.restype = None
            h.oracle_real_binary_product.argtypes = [_f32p, _i64, _i32, _i8p, _f64p, _i32,
                                                     _f64p, _vp]
            h.oracle_real_binary_product.restype = None
            h.oracle_binary_real_product.argtypes = [_i8p, _f64p, _i64, _i32, _f32p, _i32,
                                                     _i64, _f64p, _vp]
            h.oracle_binary_real_product.restype = None
            h.oracle_aggregate_mean.argtypes = [_i64p, _i32p, _i64, _f64p, _i32, _vp, _i64,
                                                _f64p, _vp]
            h.oracle_aggregate_mean.restype = ctypes.c_int
            h.oracle_aggregate_sage.argtypes = [_i64p, _i32p, _i64, _f64p, _f64p, _i32, _vp,
                                                _i64, _f64p, _vp]
            h.oracle_aggregate_sage.restype = ctypes.c_int
            h.oracle_row_scale_bucketed.argtypes = [_f32p, _i64, _i32, _i32, _f64p]
            h.oracle_row_scale_bucketed.restype = None
            h.oracle_weight_scale_bucketed.argtypes = [_f32p, _i32, _i32, _i64, _i32, _f64p]
            h.oracle_weight_scale_bucketed.restype = None
            h.oracle_zeta_bucketed.argtypes = [_i8p, _f64p, _i64, _i8p, _f64p, _i32, _i32, _i32,
                                               _f64p, _vp]
            h.oracle_zeta_bucketed.restype = None
            h.oracle_grad_weight.argtypes = [_f64p, _i8p, _f64p, _f32p, _i32, _i32, _i64, _f64p]
            h.oracle_grad_weight.restype = None
            h.oracle_degree_weighted.argtypes = [_i64p, _f64p, _i64, _f64p]
            h.oracle_degree_weighted.restype = None
            h.oracle_aggregate_weighted.argtypes = [_i64p, _i32p, _f64p, _i64, _f64p, _i32,
                                                    _vp, _i64, _f64p, _vp]
            h.oracle_aggregate_weighted.restype = ctypes.c_int
            _lib = h
    return _lib


def words_for(K: int) -> int:
    """Number of 64-bit words that hold K packed signs."""
    return (int(K) + 63) // 64


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


# ---------------------------------------------------------------- step 1 ----
def centre(X, s=None, t=None) -> np.ndarray:
    """Sec. 6.2: Y = fmaf(X, s, t) per feature, fp32; identity when s is None."""
    X = _c(X, np.float32)
    N, K = X.shape
    Y = np.empty((N, K), np.float32)
    if s is None:
        lib().oracle_centre(X, N, K, K, None, None, Y)
    else:
        s = _c(s, np.float32)
        t = _c(t, np.float32)
        assert s.shape == (K,) and t.shape == (K,)
        lib().oracle_centre(X, N, K, K, s.ctypes.data, t.ctypes.data, Y)
    return Y


# ------------------------------------------------------------ steps 2, 3 ----
def sign(V) -> np.ndarray:
    """Eq. 3 / Eq. 8: +1 where v >= 0 (sign(0) = +1), else -1, as int8."""
    V = _c(V, np.float32)
    S = np.empty(V.shape, np.int8)
    lib().oracle_sign(V.reshape(-1), V.size, S.reshape(-1))
    return S


def row_scale(Y) -> np.ndarray:
    """Eq. 7 read as the mean |y| over the row's d_in entries (float64)."""
    Y = _c(Y, np.float32)
    N, K = Y.shape
    alpha = np.empty(N, np.float64)
    lib().oracle_row_scale(Y, N, K, alpha)
    return alpha


def weight_binarize(Wt):
    """Eq. 3 and Eq. 4 on W (K x F): returns (SB as F x K int8, beta float64)."""
    Wt = _c(Wt, np.float32)
    K, F = Wt.shape
    SB = np.empty((F, K), np.int8)
    beta = np.empty(F, np.float64)
    lib().oracle_weight_binarize(Wt, K, F, F, SB, beta)
    return SB, beta


def pack(S, words=None) -> np.ndarray:
    """Store a +-1 matrix (n x K) in the interface's packed layout (n x words)."""
    S = _c(S, np.int8)
    n, K = S.shape
    words = words_for(K) if words is None else int(words)
    bits = np.empty((n, words), np.uint64)
    lib().oracle_pack(S, n, K, words, bits)
    return bits


# ---------------------------------------------------------------- step 4 ----
def binary_dot(SF, SB) -> np.ndarray:
    """Eq. 11's inner products F_i . B_j of +-1 vectors (int32, N x F)."""
    SF = _c(SF, np.int8)
    SB = _c(SB, np.int8)
    N, K = SF.shape
    F, K2 = SB.shape
    assert K == K2
    dot = np.empty((N, F), np.int32)
    lib().oracle_binary_dot(SF, N, SB, F, K, dot)
    return dot


def zeta(dot, alpha, beta) -> np.ndarray:
    """Eq. 11/12: zeta_ij = alpha_i beta_j dot_ij (float64)."""
    dot = _c(dot, np.int32)
    N, F = dot.shape
    out = np.empty((N, F), np.float64)
    lib().oracle_zeta(dot, _c(alpha, np.float64), _c(beta, np.float64), N, F, out)
    return out


# ---------------------------------------------------------------- step 5 ----
def degree(rowptr) -> np.ndarray:
    """Sec. 3.1: dhat_i = 1 + |N(i)| (the self-loop of A + I included)."""
    rowptr = _c(rowptr, np.int64)
    N = rowptr.shape[0] - 1
    d = np.empty(N, np.float64)
    lib().oracle_degree(rowptr, N, d)
    return d


def aggregate(rowptr, colidx, zeta_, rows=None, with_absterm=False):
    """Eq. 13: H = A~ zeta with A~ = D^-1/2 (A + I) D^-1/2 (Eq. 1), float64.

    ``rows`` restricts the output to those rows (in that order). With
    ``with_absterm`` also returns the per-element sum of |terms|.
    """
    rowptr = _c(rowptr, np.int64)
    colidx = _c(colidx, np.int32)
    z = _c(zeta_, np.float64)
    N = rowptr.shape[0] - 1
    assert z.shape[0] == N
    F = z.shape[1]
    if rows is None:
        rows_arr, nrows, rows_ptr = None, N, None
    else:
        rows_arr = _c(rows, np.int64)
        nrows = rows_arr.shape[0]
        rows_ptr = rows_arr.ctypes.data
    H = np.empty((nrows, F), np.float64)
    A = np.empty((nrows, F), np.float64) if with_absterm else None
    if colidx.size == 0:
        colidx = np.zeros(1, np.int32)  # a valid pointer; never read when nnz == 0
    rc = lib().oracle_aggregate(rowptr, colidx, N, z, F, rows_ptr, nrows, H,
                                None if A is None else A.ctypes.data)
    if rc != 0:
        raise ValueError("malformed CSR or row index")
    return (H, A) if with_absterm else H


# ----------------------------------------------------------- composition ----
def layer_forward(X, Wt, rowptr, colidx, s=None, t=None, rows=None) -> dict:
    """One binarized graph-convolution layer, Eq. 10-13, every step kept.

    With ``rows`` only the aggregation is restricted to those rows; every
    other step runs on all N rows (the aggregation reads zeta of neighbours).
    """
    Y = centre(X, s, t)
    SF = sign(Y)
    alpha = row_scale(Y)
    SB, beta = weight_binarize(Wt)
    dot = binary_dot(SF, SB)
    z = zeta(dot, alpha, beta)
    H, absterm = aggregate(rowptr, colidx, z, rows=rows, with_absterm=True)
    return dict(Y=Y, SF=SF, alpha=alpha, bits=pack(SF), SB=SB, beta=beta,
                wbits=pack(SB), dot=dot, zeta=z, H=H, absterm=absterm)


def forward_2layer(X, s, t, W1, W2, rowptr, colidx) -> dict:
    """The 2-layer Bi-GCN of Sec. 6.2: layer 1 centred, layer 2 on H1 raw.

    The layer interface carries fp32, so H1 is rounded to fp32 before it
    becomes layer 2's input (no activation between layers, Sec. 4.1.2).
    """
    l1 = layer_forward(X, W1, rowptr, colidx, s, t)
    H1 = l1["H"].astype(np.float32)
    l2 = layer_forward(H1, W2, rowptr, colidx)
    return dict(layer1=l1, layer2=l2, H1=H1, logits=l2["H"])


# ---------------------------------------------------- weighted adjacency ----
def degree_weighted(rowptr, values) -> np.ndarray:
    """Sec. 3 with a weighted A: dhat_i = sum_j (A + I)_ij = 1 + the sum of
    row i's CSR values (float64)."""
    rowptr, v = _c(rowptr, np.int64), _c(values, np.float64)
    N = rowptr.shape[0] - 1
    d = np.empty(N, np.float64)
    lib().oracle_degree_weighted(rowptr, v if v.size else np.zeros(1), N, d)
    return d


def aggregate_weighted(rowptr, colidx, values, zeta_, rows=None, with_absterm=False):
    """Eq. 13 with Eq. 1's operator on a weighted A (values[e] = a_ij of CSR
    entry e): H_i = zeta_i / dhat_i + sum_e a_ij zeta_j / sqrt(dhat_i dhat_j),
    float64. Weights must be finite and >= 0."""
    rowptr, colidx = _c(rowptr, np.int64), _c(colidx, np.int32)
    v, z = _c(values, np.float64), _c(zeta_, np.float64)
    N, F = z.shape
    assert rowptr.shape[0] == N + 1 and v.shape == colidx.shape
    keep, nrows, rp = _rows_arg(rows, N)
    H = np.empty((nrows, F), np.float64)
    A = np.empty((nrows, F), np.float64) if with_absterm else None
    if colidx.size == 0:
        colidx, v = np.zeros(1, np.int32), np.zeros(1, np.float64)
    if lib().oracle_aggregate_weighted(rowptr, colidx, v, N, z, F, rp, nrows, H,
                                       None if A is None else A.ctypes.data) != 0:
        raise ValueError("malformed CSR, row index or weight")
    return (H, A) if with_absterm else H


def layer_forward_weighted(X, Wt, rowptr, colidx, values, s=None, t=None, rows=None) -> dict:
    """One binarized layer (Eqs. 10-13) over a weighted adjacency: the steps
    of ``layer_forward`` with ``aggregate_weighted`` as step 5."""
    Y = centre(X, s, t)
    SF = sign(Y)
    alpha = row_scale(Y)
    SB, beta = weight_binarize(Wt)
    dot = binary_dot(SF, SB)
    z = zeta(dot, alpha, beta)
    H, absterm = aggregate_weighted(rowptr, colidx, values, z, rows=rows, with_absterm=True)
    return dict(Y=Y, SF=SF, alpha=alpha, SB=SB, beta=beta, dot=dot, zeta=z,
                dhat=degree_weighted(rowptr, values), H=H, absterm=absterm)


# ------------------------------------------------------ ablation variants ----
BINARIZE = ("both", "weights", "features")


def real_binary_product(Y, SB, beta, with_absterm=False):
    """Weights binarized, features real: zeta = Y W~, W~[k,j] = beta_j SB[j,k]
    (the "binarize weights only" row of Sec. 6.3's transductive table)."""
    Y = _c(Y, np.float32)
    SB = _c(SB, np.int8)
    N, K = Y.shape
    F = SB.shape[0]
    assert SB.shape[1] == K
    z = np.empty((N, F), np.float64)
    a = np.empty((N, F), np.float64) if with_absterm else None
    lib().oracle_real_binary_product(Y, N, K, SB, _c(beta, np.float64), F, z,
                                     None if a is None else a.ctypes.data)
    return (z, a) if with_absterm else z


def binary_real_product(SF, alpha, Wt, with_absterm=False):
    """Features binarized, weights real: zeta = H~ W, H~[i,k] = alpha_i SF[i,k]
    (the "binarize features only" row of Sec. 6.3's transductive table)."""
    SF = _c(SF, np.int8)
    Wt = _c(Wt, np.float32)
    N, K = SF.shape
    F = Wt.shape[1]
    assert Wt.shape[0] == K
    z = np.empty((N, F), np.float64)
    a = np.empty((N, F), np.float64) if with_absterm else None
    lib().oracle_binary_real_product(SF, _c(alpha, np.float64), N, K, Wt, F, F, z,
                                     None if a is None else a.ctypes.data)
    return (z, a) if with_absterm else z


def layer_forward_ablation(X, Wt, rowptr, colidx, binarize, s=None, t=None, rows=None) -> dict:
    """One graph-convolution layer with the operands of Eq. 11 binarized as
    ``binarize`` says: "both" (Bi-GCN, Eqs. 10-13), "weights" (features kept
    real) or "features" (weights kept real), then Eq. 13's aggregation.

    Besides H and the aggregation's own |terms|, returns ``scale``: A~ applied
    to the product's |terms|, the error scale of any evaluation order of the
    whole layer (A~ has no negative entries).
    """
    if binarize == "both":
        r = layer_forward(X, Wt, rowptr, colidx, s, t, rows)
        za = np.abs(r["alpha"])[:, None] * np.abs(r["beta"])[None, :] * Wt.shape[0]
        r["scale"] = aggregate(rowptr, colidx, za, rows=rows)
        return r
    assert binarize in ("weights", "features")
    Y = centre(X, s, t)
    out = dict(Y=Y)
    if binarize == "weights":
        SB, beta = weight_binarize(Wt)
        z, za = real_binary_product(Y, SB, beta, with_absterm=True)
        out.update(SB=SB, beta=beta, wbits=pack(SB))
    else:
        SF = sign(Y)
        alpha = row_scale(Y)
        z, za = binary_real_product(SF, alpha, Wt, with_absterm=True)
        out.update(SF=SF, alpha=alpha, bits=pack(SF))
    H, absterm = aggregate(rowptr, colidx, z, rows=rows, with_absterm=True)
    out.update(zeta=z, zeta_abs=za, H=H, absterm=absterm,
               scale=aggregate(rowptr, colidx, za, rows=rows))
    return out


# ------------------------------------------------------ sub-row bucketing ----
def buckets(K: int, B: int) -> int:
    return (K + B - 1) // B


def row_scale_bucketed(Y, B):
    """Eq. 7 per bucket of B consecutive features: alpha (N x nb)."""
    Y = _c(Y, np.float32)
    N, K = Y.shape
    a = np.empty((N, buckets(K, B)), np.float64)
    lib().oracle_row_scale_bucketed(Y, N, K, B, a)
    return a


def weight_scale_bucketed(Wt, B):
    """Eq. 4 per bucket of B consecutive entries of each column: beta (F x nb)."""
    Wt = _c(Wt, np.float32)
    K, F = Wt.shape
    b = np.empty((F, buckets(K, B)), np.float64)
    lib().oracle_weight_scale_bucketed(Wt, K, F, F, B, b)
    return b


def zeta_bucketed(SF, alpha_b, SB, beta_b, B, with_absterm=False):
    """Eqs. 11-12 with one scale pair per bucket: sum_b alpha_ib beta_jb dot_b."""
    SF, SB = _c(SF, np.int8), _c(SB, np.int8)
    N, K = SF.shape
    F = SB.shape[0]
    z = np.empty((N, F), np.float64)
    a = np.empty((N, F), np.float64) if with_absterm else None
    lib().oracle_zeta_bucketed(SF, _c(alpha_b, np.float64), N, SB, _c(beta_b, np.float64), F,
                               K, B, z, None if a is None else a.ctypes.data)
    return (z, a) if with_absterm else z


def layer_forward_bucketed(X, Wt, rowptr, colidx, B, s=None, t=None, rows=None) -> dict:
    """The Bi-GCN layer with buckets of B consecutive features (Sec. 4.1) in
    place of whole rows / columns, then Eq. 13's aggregation. ``scale`` is
    A~ applied to the product's |terms| (A~ has no negative entries)."""
    Y = centre(X, s, t)
    SF = sign(Y)
    SB = sign(np.ascontiguousarray(np.asarray(Wt, np.float32).T))
    alpha_b = row_scale_bucketed(Y, B)
    beta_b = weight_scale_bucketed(Wt, B)
    z, za = zeta_bucketed(SF, alpha_b, SB, beta_b, B, with_absterm=True)
    H, absterm = aggregate(rowptr, colidx, z, rows=rows, with_absterm=True)
    return dict(Y=Y, SF=SF, SB=SB, alpha_b=alpha_b, beta_b=beta_b, bits=pack(SF),
                wbits=pack(SB), zeta=z, zeta_abs=za, H=H, absterm=absterm,
                scale=aggregate(rowptr, colidx, za, rows=rows))


# ---------------------------------------------------- inductive aggregators ----
AGGREGATORS = ("gcn", "mean", "sage")


def _rows_arg(rows, N):
    if rows is None:
        return None, N, None
    r = _c(rows, np.int64)
    return r, r.shape[0], r.ctypes.data


def aggregate_mean(rowptr, colidx, zeta_, rows=None, with_absterm=False):
    """Inductive GCN's mean aggregator: H_i = mean of zeta over N(i) u {i}."""
    rowptr, colidx, z = _c(rowptr, np.int64), _c(colidx, np.int32), _c(zeta_, np.float64)
    N, F = z.shape
    keep, nrows, rp = _rows_arg(rows, N)
    H = np.empty((nrows, F), np.float64)
    A = np.empty((nrows, F), np.float64) if with_absterm else None
    if colidx.size == 0:
        colidx = np.zeros(1, np.int32)
    if lib().oracle_aggregate_mean(rowptr, colidx, N, z, F, rp, nrows, H,
                                   None if A is None else A.ctypes.data) != 0:
        raise ValueError("malformed CSR or row index")
    return (H, A) if with_absterm else H


def aggregate_sage(rowptr, colidx, zself, zneigh, rows=None, with_absterm=False):
    """GraphSAGE's mean aggregator with concatenation on the products:
    H_i = zself_i + mean over N(i) of zneigh (0 without neighbours)."""
    rowptr, colidx = _c(rowptr, np.int64), _c(colidx, np.int32)
    zs, zn = _c(zself, np.float64), _c(zneigh, np.float64)
    assert zs.shape == zn.shape
    N, F = zs.shape
    keep, nrows, rp = _rows_arg(rows, N)
    H = np.empty((nrows, F), np.float64)
    A = np.empty((nrows, F), np.float64) if with_absterm else None
    if colidx.size == 0:
        colidx = np.zeros(1, np.int32)
    if lib().oracle_aggregate_sage(rowptr, colidx, N, zs, zn, F, rp, nrows, H,
                                   None if A is None else A.ctypes.data) != 0:
        raise ValueError("malformed CSR or row index")
    return (H, A) if with_absterm else H


def layer_forward_inductive(X, Wt, rowptr, colidx, aggregator, s=None, t=None, W_neigh=None,
                            rows=None) -> dict:
    """One binarized layer of an inductive GNN (Sec. 6.3, Table 3): the
    product of Eqs. 10-12 on every node's own features, then the aggregator:
    "gcn" (Eq. 13), "mean" (inductive GCN) or "sage" (GraphSAGE-mean, with a
    second weight matrix W_neigh binarized column by column like Wt)."""
    Y = centre(X, s, t)
    SF = sign(Y)
    alpha = row_scale(Y)
    SB, beta = weight_binarize(Wt)
    z = zeta(binary_dot(SF, SB), alpha, beta)
    out = dict(Y=Y, SF=SF, alpha=alpha, SB=SB, beta=beta, zeta=z)
    if aggregator == "gcn":
        H, a = aggregate(rowptr, colidx, z, rows=rows, with_absterm=True)
    elif aggregator == "mean":
        H, a = aggregate_mean(rowptr, colidx, z, rows=rows, with_absterm=True)
    elif aggregator == "sage":
        SBn, beta_n = weight_binarize(W_neigh)
        zn = zeta(binary_dot(SF, SBn), alpha, beta_n)
        out.update(SBn=SBn, beta_n=beta_n, zeta_n=zn)
        H, a = aggregate_sage(rowptr, colidx, z, zn, rows=rows, with_absterm=True)
    else:
        raise ValueError(aggregator)
    out.update(H=H, absterm=a)
    return out


# ------------------------------------------------------- back-propagation ----
def aggregate_t(rowptr, colidx, dH) -> np.ndarray:
    """Algorithm 1: G = A~^T dH, scattering each row's gradient to its
    neighbours and itself (float64)."""
    rowptr = _c(rowptr, np.int64)
    colidx = _c(colidx, np.int32)
    dH = _c(dH, np.float64)
    N, F = dH.shape
    assert rowptr.shape[0] == N + 1
    G = np.empty((N, F), np.float64)
    if colidx.size == 0:
        colidx = np.zeros(1, np.int32)
    if lib().oracle_aggregate_t(rowptr, colidx, N, dH, F, G) != 0:
        raise ValueError("malformed CSR")
    return G


def grad_wtilde(SF, alpha, G, with_absterm=False):
    """Algorithm 1: dL/dW~ = H~^T G with H~ = diag(alpha) SF (K x F)."""
    SF = _c(SF, np.int8)
    G = _c(G, np.float64)
    N, K = SF.shape
    F = G.shape[1]
    out = np.empty((K, F), np.float64)
    a = np.empty(F, np.float64) if with_absterm else None
    lib().oracle_grad_wtilde(SF, _c(alpha, np.float64), G, N, K, F, out,
                             None if a is None else a.ctypes.data)
    return (out, a) if with_absterm else out


def grad_htilde(G, beta, SB, with_absterm=False):
    """Algorithm 1: dL/dH~ = G W~^T with W~[k,j] = beta_j SB[j,k] (N x K)."""
    G = _c(G, np.float64)
    SB = _c(SB, np.int8)
    N, F = G.shape
    K = SB.shape[1]
    out = np.empty((N, K), np.float64)
    a = np.empty(N, np.float64) if with_absterm else None
    lib().oracle_grad_htilde(G, _c(beta, np.float64), SB, N, K, F, out,
                             None if a is None else a.ctypes.data)
    return (out, a) if with_absterm else out


def grad_input(Ht) -> np.ndarray:
    """Eq. bp-H: dL/dH = dL/dH~ where |dL/dH~| < 1, else 0."""
    Ht = _c(Ht, np.float64)
    out = np.empty(Ht.shape, np.float64)
    lib().oracle_grad_input(Ht.reshape(-1), Ht.size, out.reshape(-1))
    return out


def grad_weight(Wg, SB, beta, Wt) -> np.ndarray:
    """Eq. bp-W (d_in = K): the gradient of W through the column scale plus
    the straight-through estimator 1(|W| < 1) of sign()."""
    Wg = _c(Wg, np.float64)
    Wt = _c(Wt, np.float32)
    K, F = Wt.shape
    out = np.empty((K, F), np.float64)
    lib().oracle_grad_weight(Wg, _c(SB, np.int8), _c(beta, np.float64), Wt, K, F, F, out)
    return out


def layer_backward(X, Wt, rowptr, colidx, dH, s=None, t=None) -> dict:
    """Algorithm 1 for one layer: from dL/dH^(l+1) (dH, N x F) to dL/dH^(l)
    (Eq. bp-H, w.r.t. the layer's binarized input, i.e. the centred X for
    layer 1) and dL/dW (Eq. bp-W), every intermediate kept."""
    Y = centre(X, s, t)
    SF = sign(Y)
    alpha = row_scale(Y)
    SB, beta = weight_binarize(Wt)
    G = aggregate_t(rowptr, colidx, dH)
    Wg, wg_abs = grad_wtilde(SF, alpha, G, with_absterm=True)
    Ht, ht_abs = grad_htilde(G, beta, SB, with_absterm=True)
    return dict(Y=Y, SF=SF, alpha=alpha, SB=SB, beta=beta, G=G, Wg=Wg, Wg_abs=wg_abs,
                Ht=Ht, Ht_abs=ht_abs, dX=grad_input(Ht), dW=grad_weight(Wg, SB, beta, Wt))
