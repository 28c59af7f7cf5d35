"""Python binding of libbigcn.so (include/bigcn.h): argument marshalling only.

The ``bigcn_*`` functions mirror the C entry points one to one and take torch
CUDA tensors for every array; they read pointers, sizes and row strides off
the tensors, pass the current torch stream (or ``stream``), and raise
:class:`BigcnError` on a non-OK status. Every step of the computation runs in
the library's kernels; there is no Python or CPU fallback, and the library
must have been built (``__graft_entry__.build()``) before first use.

The lower-case helpers (``pack_rows``, ``layer_forward``, ...) only allocate
the outputs with torch and call the matching ``bigcn_*`` function.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

from . import build as _build

_lib = None
_lock = threading.Lock()

BIGCN_OK = 0
STATUS_NAMES = {0: "BIGCN_OK", 1: "BIGCN_ERR_INVALID_ARG", 2: "BIGCN_ERR_MISALIGNED",
                3: "BIGCN_ERR_CUDA", 4: "BIGCN_ERR_UNSUPPORTED", 5: "BIGCN_ERR_SCRATCH_LIMIT"}
STATIC_SCRATCH_BYTES = 32 << 20   # BIGCN_STATIC_SCRATCH_BYTES

_p = ctypes.c_void_p
_i32 = ctypes.c_int32
_i64 = ctypes.c_int64
_sz = ctypes.c_size_t

SIGNATURES = {
    "bigcn_status_string": ([ctypes.c_int], ctypes.c_char_p),
    "bigcn_words": ([_i32], _i32),
    "bigcn_pack_rows": ([_p, _i64, _i32, _i64, _p, _p, _p, _i32, _p, _p], ctypes.c_int),
    "bigcn_pack_weights": ([_p, _i32, _i32, _i64, _p, _i32, _p, _p], ctypes.c_int),
    "bigcn_xnor_gemm": ([_p, _p, _i64, _p, _p, _i32, _i32, _i32, _p, _i64, _p, _p],
                        ctypes.c_int),
    "bigcn_xnor_gemm_degscaled": ([_p, _p, _i64, _p, _p, _i32, _i32, _i32, _p, _p, _i64, _p],
                                  ctypes.c_int),
    "bigcn_spmm_norm": ([_p, _p, _i64, _i64, _p, _i64, _i32, _p, _i64, _p], ctypes.c_int),
    "bigcn_spmm_prescaled": ([_p, _p, _i64, _i64, _p, _i64, _i32, _p, _i64, _p], ctypes.c_int),
    "bigcn_device_timeouts": ([], _i32),
    "bigcn_layer_workspace_bytes": ([_i64, _i32, _i32], _sz),
    "bigcn_layer_forward": ([_p, _i64, _i32, _i64, _p, _p, _p, _i32, _i64, _p, _p, _i64, _p,
                             _sz, _p, _i64, _p], ctypes.c_int),
    "bigcn_layer_forward_timed": ([_p, _i64, _i32, _i64, _p, _p, _p, _i32, _i64, _p, _p, _i64,
                                   _p, _sz, _p, _i64, _p, _i32, _p], ctypes.c_int),
    "bigcn_layer_backward_workspace_bytes": ([_i64, _i32, _i32], _sz),
    "bigcn_layer_backward": ([_p, _i64, _i32, _i64, _p, _p, _p, _i32, _i64, _p, _p, _i64, _p,
                              _i64, _p, _i64, _p, _i64, _p, _sz, _p], ctypes.c_int),
    "bigcn_forward_2layer_workspace_bytes": ([_i64, _i32, _i32, _i32], _sz),
    "bigcn_forward_2layer_launches": ([_i64, _i32, _i32, _i32], _i32),
    "bigcn_forward_2layer_aggregation": ([_i32, _i32, _i32], _i32),
    "bigcn_spmm_prescaled_rows": ([_p, _p, _i64, _i64, _i64, _p, _i64, _i32, _p, _i64, _p],
                                  ctypes.c_int),
    "bigcn_forward_2layer": ([_p, _i64, _i32, _i64, _p, _p, _p, _i32, _i64, _p, _i32, _i64, _p,
                              _p, _i64, _p, _sz, _p, _i64, _p, _i64, _p, _p, _i32, _p],
                             ctypes.c_int),
    "bigcn_real_binary_gemm": ([_p, _i64, _i32, _i64, _p, _p, _p, _p, _i32, _i32, _p, _i64,
                                _p], ctypes.c_int),
    "bigcn_binary_real_gemm_workspace_bytes": ([_i32, _i32], _sz),
    "bigcn_binary_real_gemm": ([_p, _p, _i64, _i32, _i32, _p, _i32, _i64, _p, _sz, _p, _i64,
                                _p], ctypes.c_int),
    "bigcn_layer_ablation_workspace_bytes": ([_i32, _i64, _i32, _i32], _sz),
    "bigcn_layer_forward_ablation": ([_i32, _p, _i64, _i32, _i64, _p, _p, _p, _i32, _i64, _p,
                                      _p, _i64, _p, _sz, _p, _i64, _p], ctypes.c_int),
    "bigcn_inductive_layer_workspace_bytes": ([_i32, _i64, _i32, _i32], _sz),
    "bigcn_inductive_layer_forward": ([_i32, _p, _i64, _i32, _i64, _p, _p, _p, _i32, _i64, _p,
                                       _i64, _p, _p, _i64, _p, _sz, _p, _i64, _p], ctypes.c_int),
    "bigcn_pack_rows_bucketed": ([_p, _i64, _i32, _i64, _p, _p, _i32, _p, _i32, _p, _p],
                                 ctypes.c_int),
    "bigcn_pack_weights_bucketed": ([_p, _i32, _i32, _i64, _i32, _p, _i32, _p, _p], ctypes.c_int),
    "bigcn_xnor_gemm_bucketed": ([_p, _p, _i64, _p, _p, _i32, _i32, _i32, _i32, _p, _i64, _p],
                                 ctypes.c_int),
    "bigcn_layer_bucketed_workspace_bytes": ([_i64, _i32, _i32, _i32], _sz),
    "bigcn_layer_forward_bucketed": ([_i32, _p, _i64, _i32, _i64, _p, _p, _p, _i32, _i64, _p,
                                      _p, _i64, _p, _sz, _p, _i64, _p], ctypes.c_int),
    "bigcn_layer_forward_static": ([_p, _i64, _i32, _i64, _p, _p, _p, _i32, _i64, _p, _p, _i64,
                                    _p, _i64, _p], ctypes.c_int),
    "bigcn_weighted_dinv": ([_p, _p, _i64, _i64, _p, _p], ctypes.c_int),
    "bigcn_spmm_norm_weighted": ([_p, _p, _p, _p, _i64, _i64, _p, _i64, _i32, _p, _i64, _p],
                                 ctypes.c_int),
    "bigcn_weighted_layer_workspace_bytes": ([_i64, _i32, _i32], _sz),
    "bigcn_weighted_layer_forward": ([_p, _i64, _i32, _i64, _p, _p, _p, _i32, _i64, _p, _p, _p,
                                      _i64, _p, _sz, _p, _i64, _p], ctypes.c_int),
}


class BigcnError(RuntimeError):
    def __init__(self, fn: str, status: int):
        super().__init__(f"{fn} returned {STATUS_NAMES.get(status, status)}")
        self.status = status


def library_path() -> str:
    return _build.LIB


def lib() -> ctypes.CDLL:
    """The loaded libbigcn.so. Raises if it has not been built."""
    global _lib
    with _lock:
        if _lib is None:
            path = _build.LIB
            if not os.path.exists(path):
                raise RuntimeError(
                    f"{path} is missing: build the CUDA library first "
                    "(python -c 'import __graft_entry__ as g; g.build()')")
            h = ctypes.CDLL(path)
            for name, (args, res) in SIGNATURES.items():
                fn = getattr(h, name)
                fn.argtypes = args
                fn.restype = res
            _lib = h
    return _lib


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, torch.cuda.Stream):
        return ctypes.c_void_p(stream.cuda_stream)
    return ctypes.c_void_p(int(stream))


def _ld(t):
    """Row stride in elements of a 2-D tensor whose rows are contiguous."""
    if t.dim() != 2 or t.stride(1) != 1:
        raise ValueError("expected a 2-D tensor with unit column stride")
    return t.stride(0)


def _check(fn: str, status: int):
    if status != BIGCN_OK:
        raise BigcnError(fn, status)


def status_string(status: int) -> str:
    return lib().bigcn_status_string(status).decode()


def device_timeouts() -> int:
    """Bounded device waits that ran out since the last call (synchronizes)."""
    return int(lib().bigcn_device_timeouts())


def words_for(K: int) -> int:
    return int(lib().bigcn_words(K))


# ------------------------------------------------------ one-to-one entries ---
def bigcn_pack_rows(X, scale, shift, bits, alpha, stream=None, K=None):
    """Steps 1+2 (Sec. 6.2, Eqs. 7-8): bits, alpha <- X (N x K fp32)."""
    N, Kx = X.shape
    K = Kx if K is None else K
    _check("bigcn_pack_rows", lib().bigcn_pack_rows(
        _ptr(X), N, K, _ld(X), _ptr(scale), _ptr(shift), _ptr(bits), _ld(bits),
        _ptr(alpha), _stream(stream)))


def bigcn_pack_weights(Wt, bits, beta, stream=None):
    """Step 3 (Eqs. 3-4): bits (F x words), beta <- Wt (K x F fp32)."""
    K, F = Wt.shape
    _check("bigcn_pack_weights", lib().bigcn_pack_weights(
        _ptr(Wt), K, F, _ld(Wt), _ptr(bits), _ld(bits), _ptr(beta), _stream(stream)))


def bigcn_xnor_gemm(a_bits, alpha, b_bits, beta, K, Z, dots=None, stream=None):
    """Step 4 (Eqs. 11-12): Z = alpha_i beta_j (K - 2 popc(a_i ^ b_j))."""
    N, words = a_bits.shape
    F = b_bits.shape[0]
    if b_bits.shape[1] != words:
        raise ValueError("a_bits and b_bits must have the same row width")
    _check("bigcn_xnor_gemm", lib().bigcn_xnor_gemm(
        _ptr(a_bits), _ptr(alpha), N, _ptr(b_bits), _ptr(beta), F, K, words, _ptr(Z), _ld(Z),
        _ptr(dots), _stream(stream)))


def bigcn_spmm_norm(rowptr, colidx, Z, H, stream=None):
    """Step 5 (Eqs. 1, 13): H = D^-1/2 (A + I) D^-1/2 Z."""
    N = rowptr.shape[0] - 1
    F = Z.shape[1]
    _check("bigcn_spmm_norm", lib().bigcn_spmm_norm(
        _ptr(rowptr), _ptr(colidx) if colidx.numel() else None, N, colidx.numel(), _ptr(Z),
        _ld(Z), F, _ptr(H), _ld(H), _stream(stream)))


def bigcn_xnor_gemm_degscaled(a_bits, alpha, b_bits, beta, K, rowptr, Z, stream=None):
    """Step 4 with row i also scaled by 1/sqrt(dhat_i) (the source-side factor
    of Eq. 1's normalisation)."""
    N, words = a_bits.shape
    F = b_bits.shape[0]
    if b_bits.shape[1] != words:
        raise ValueError("a_bits and b_bits must have the same row width")
    _check("bigcn_xnor_gemm_degscaled", lib().bigcn_xnor_gemm_degscaled(
        _ptr(a_bits), _ptr(alpha), N, _ptr(b_bits), _ptr(beta), F, K, words, _ptr(rowptr),
        _ptr(Z), _ld(Z), _stream(stream)))


def bigcn_spmm_prescaled(rowptr, colidx, Z, H, stream=None):
    """Step 5 over rows that already carry their 1/sqrt(dhat_j)."""
    N = rowptr.shape[0] - 1
    F = Z.shape[1]
    _check("bigcn_spmm_prescaled", lib().bigcn_spmm_prescaled(
        _ptr(rowptr), _ptr(colidx) if colidx.numel() else None, N, colidx.numel(), _ptr(Z),
        _ld(Z), F, _ptr(H), _ld(H), _stream(stream)))


def bigcn_spmm_prescaled_rows(rowptr, colidx, Z, H, stream=None):
    """A block of output rows (H: n_rows x F) aggregated over a table of
    pre-scaled rows (Z: n_cols x F, the block's own rows first)."""
    n_rows, n_cols = H.shape[0], Z.shape[0]
    _check("bigcn_spmm_prescaled_rows", lib().bigcn_spmm_prescaled_rows(
        _ptr(rowptr), _ptr(colidx) if colidx.numel() else None, n_rows, n_cols, colidx.numel(),
        _ptr(Z), _ld(Z), Z.shape[1], _ptr(H), _ld(H), _stream(stream)))


def bigcn_layer_workspace_bytes(N: int, K: int, F: int) -> int:
    return int(lib().bigcn_layer_workspace_bytes(N, K, F))


def bigcn_layer_forward(X, scale, shift, Wt, rowptr, colidx, workspace, H, stream=None):
    """One fused layer (Eq. 13 with zeta of Eqs. 11-12)."""
    N, K = X.shape
    F = Wt.shape[1]
    _check("bigcn_layer_forward", lib().bigcn_layer_forward(
        _ptr(X), N, K, _ld(X), _ptr(scale), _ptr(shift), _ptr(Wt), F, _ld(Wt), _ptr(rowptr),
        _ptr(colidx) if colidx.numel() else None, colidx.numel(), _ptr(workspace),
        workspace.numel() * workspace.element_size(), _ptr(H), _ld(H), _stream(stream)))


def bigcn_layer_forward_timed(X, scale, shift, Wt, rowptr, colidx, workspace, H, events,
                              stream=None):
    """bigcn_layer_forward recording ``events`` (torch.cuda.Event objects
    created with enable_timing=True and recorded once, so that the CUDA event
    exists) before each of its four kernels and after the last."""
    N, K = X.shape
    F = Wt.shape[1]
    ev = (ctypes.c_void_p * len(events))(*[e.cuda_event for e in events])
    _check("bigcn_layer_forward_timed", lib().bigcn_layer_forward_timed(
        _ptr(X), N, K, _ld(X), _ptr(scale), _ptr(shift), _ptr(Wt), F, _ld(Wt), _ptr(rowptr),
        _ptr(colidx) if colidx.numel() else None, colidx.numel(), _ptr(workspace),
        workspace.numel() * workspace.element_size(), _ptr(H), _ld(H), ev, len(events),
        _stream(stream)))


# Which operands of Eq. 11 are binarized (enum bigcn_binarize).
BINARIZE = {"both": 0, "weights": 1, "features": 2}


def bigcn_real_binary_gemm(X, scale, shift, b_bits, beta, Z, stream=None):
    """Weights binarized, features real: Z = Y W~ (Y = X centred by
    scale/shift)."""
    N, K = X.shape
    F = beta.shape[0]
    _check("bigcn_real_binary_gemm", lib().bigcn_real_binary_gemm(
        _ptr(X), N, K, _ld(X), _ptr(scale), _ptr(shift), _ptr(b_bits), _ptr(beta), F,
        _ld(b_bits), _ptr(Z), _ld(Z), _stream(stream)))


def bigcn_binary_real_gemm_workspace_bytes(K: int, F: int) -> int:
    return int(lib().bigcn_binary_real_gemm_workspace_bytes(K, F))


def bigcn_binary_real_gemm(a_bits, alpha, K, Wt, workspace, Z, stream=None):
    """Features binarized, weights real: Z = H~ W (H~ = diag(alpha) signs)."""
    N = alpha.shape[0]
    F = Wt.shape[1]
    _check("bigcn_binary_real_gemm", lib().bigcn_binary_real_gemm(
        _ptr(a_bits), _ptr(alpha), N, K, _ld(a_bits), _ptr(Wt), F, _ld(Wt), _ptr(workspace),
        workspace.numel() * workspace.element_size(), _ptr(Z), _ld(Z), _stream(stream)))


def bigcn_layer_ablation_workspace_bytes(binarize, N: int, K: int, F: int) -> int:
    return int(lib().bigcn_layer_ablation_workspace_bytes(BINARIZE.get(binarize, binarize),
                                                          N, K, F))


def bigcn_layer_forward_ablation(binarize, X, scale, shift, Wt, rowptr, colidx, workspace, H,
                                 stream=None):
    """One layer with the operands of Eq. 11 binarized as ``binarize`` says
    ("both", "weights", "features" or the enum's value)."""
    N, K = X.shape
    F = Wt.shape[1]
    _check("bigcn_layer_forward_ablation", lib().bigcn_layer_forward_ablation(
        BINARIZE.get(binarize, binarize), _ptr(X), N, K, _ld(X), _ptr(scale), _ptr(shift),
        _ptr(Wt), F, _ld(Wt), _ptr(rowptr), _ptr(colidx) if colidx.numel() else None,
        colidx.numel(), _ptr(workspace), workspace.numel() * workspace.element_size(), _ptr(H),
        _ld(H), _stream(stream)))


def bigcn_pack_rows_bucketed(X, scale, shift, B, bits, alpha, stream=None):
    """Sub-row bucketing (Sec. 4.1): packed signs and alpha (N x nb) per
    bucket of B features (a multiple of 64)."""
    N, K = X.shape
    _check("bigcn_pack_rows_bucketed", lib().bigcn_pack_rows_bucketed(
        _ptr(X), N, K, _ld(X), _ptr(scale), _ptr(shift), B, _ptr(bits), _ld(bits), _ptr(alpha),
        _stream(stream)))


def bigcn_pack_weights_bucketed(Wt, B, bits, beta, stream=None):
    """Packed weight columns and beta (F x nb) per bucket of B entries."""
    K, F = Wt.shape
    _check("bigcn_pack_weights_bucketed", lib().bigcn_pack_weights_bucketed(
        _ptr(Wt), K, F, _ld(Wt), B, _ptr(bits), _ld(bits), _ptr(beta), _stream(stream)))


def bigcn_xnor_gemm_bucketed(a_bits, alpha, b_bits, beta, K, B, Z, stream=None):
    """Z = sum over buckets of alpha_ib beta_jb dot_b."""
    N = a_bits.shape[0]
    F = b_bits.shape[0]
    _check("bigcn_xnor_gemm_bucketed", lib().bigcn_xnor_gemm_bucketed(
        _ptr(a_bits), _ptr(alpha), N, _ptr(b_bits), _ptr(beta), F, K, _ld(a_bits), B, _ptr(Z),
        _ld(Z), _stream(stream)))


def bigcn_layer_bucketed_workspace_bytes(N: int, K: int, F: int, B: int) -> int:
    return int(lib().bigcn_layer_bucketed_workspace_bytes(N, K, F, B))


def bigcn_layer_forward_bucketed(B, X, scale, shift, Wt, rowptr, colidx, workspace, H,
                                 stream=None):
    """One layer with bucketed binarization (buckets of B features)."""
    N, K = X.shape
    F = Wt.shape[1]
    _check("bigcn_layer_forward_bucketed", lib().bigcn_layer_forward_bucketed(
        B, _ptr(X), N, K, _ld(X), _ptr(scale), _ptr(shift), _ptr(Wt), F, _ld(Wt), _ptr(rowptr),
        _ptr(colidx) if colidx.numel() else None, colidx.numel(), _ptr(workspace),
        workspace.numel() * workspace.element_size(), _ptr(H), _ld(H), _stream(stream)))


# Aggregators of the inductive layers (enum bigcn_aggregator).
AGGREGATOR = {"gcn": 0, "mean": 1, "sage": 2}


def bigcn_inductive_layer_workspace_bytes(aggregator, N: int, K: int, F: int) -> int:
    return int(lib().bigcn_inductive_layer_workspace_bytes(
        AGGREGATOR.get(aggregator, aggregator), N, K, F))


def bigcn_inductive_layer_forward(aggregator, X, scale, shift, Wt, rowptr, colidx, workspace, H,
                                  W_neigh=None, stream=None):
    """One binarized inductive layer: the product, then the ``aggregator``
    ("gcn", "mean", "sage"; "sage" takes W_neigh)."""
    N, K = X.shape
    F = Wt.shape[1]
    _check("bigcn_inductive_layer_forward", lib().bigcn_inductive_layer_forward(
        AGGREGATOR.get(aggregator, aggregator), _ptr(X), N, K, _ld(X), _ptr(scale), _ptr(shift),
        _ptr(Wt), F, _ld(Wt), _ptr(W_neigh), _ld(W_neigh) if W_neigh is not None else 0,
        _ptr(rowptr), _ptr(colidx) if colidx.numel() else None, colidx.numel(), _ptr(workspace),
        workspace.numel() * workspace.element_size(), _ptr(H), _ld(H), _stream(stream)))


def bigcn_layer_backward_workspace_bytes(N: int, K: int, F: int) -> int:
    return int(lib().bigcn_layer_backward_workspace_bytes(N, K, F))


def bigcn_layer_backward(X, scale, shift, Wt, rowptr, colidx, dH, workspace, dW, dX=None,
                         stream=None):
    """Algorithm 1 for one layer: dW (K x F, Eq. bp-W) and optionally dX
    (N x K, Eq. bp-H) from dH = dL/dH^(l+1) (N x F)."""
    N, K = X.shape
    F = Wt.shape[1]
    _check("bigcn_layer_backward", lib().bigcn_layer_backward(
        _ptr(X), N, K, _ld(X), _ptr(scale), _ptr(shift), _ptr(Wt), F, _ld(Wt), _ptr(rowptr),
        _ptr(colidx) if colidx.numel() else None, colidx.numel(), _ptr(dH), _ld(dH), _ptr(dX),
        _ld(dX) if dX is not None else 0, _ptr(dW), _ld(dW), _ptr(workspace),
        workspace.numel() * workspace.element_size(), _stream(stream)))


def bigcn_forward_2layer_workspace_bytes(N: int, K: int, Fh: int, Fo: int) -> int:
    return int(lib().bigcn_forward_2layer_workspace_bytes(N, K, Fh, Fo))


def bigcn_forward_2layer_launches(N: int, K: int, Fh: int, Fo: int) -> int:
    n = int(lib().bigcn_forward_2layer_launches(N, K, Fh, Fo))
    if n < 0:
        raise BigcnError("bigcn_forward_2layer_launches", 1)
    return n


def bigcn_forward_2layer_aggregation(K: int, Fh: int, Fo: int) -> int:
    """1 when bigcn_forward_2layer aggregates on the tensor cores (fp16 dots),
    0 on the CUDA cores."""
    n = int(lib().bigcn_forward_2layer_aggregation(K, Fh, Fo))
    if n < 0:
        raise BigcnError("bigcn_forward_2layer_aggregation", 1)
    return n


def bigcn_forward_2layer(X, scale, shift, W1, W2, rowptr, colidx, workspace, out, H1=None,
                         events=None, stream=None, pred=None):
    """The two-layer forward of Sec. 6.2 (hidden layer on centred X, output
    layer on H1 raw). ``events``: torch.cuda.Event objects (created with
    enable_timing=True, external=True and recorded once) to be recorded
    before each kernel and after the last. ``pred``: optional int32 tensor of
    N that receives each row's argmax of the logits."""
    N, K = X.shape
    Fh, Fo = W1.shape[1], W2.shape[1]
    if W2.shape[0] != Fh:
        raise ValueError("W2 must have as many rows as W1 has columns")
    if events:
        ev = (ctypes.c_void_p * len(events))(*[e.cuda_event for e in events])
        n_ev = len(events)
    else:
        ev, n_ev = None, 0
    _check("bigcn_forward_2layer", lib().bigcn_forward_2layer(
        _ptr(X), N, K, _ld(X), _ptr(scale), _ptr(shift), _ptr(W1), Fh, _ld(W1), _ptr(W2), Fo,
        _ld(W2), _ptr(rowptr), _ptr(colidx) if colidx.numel() else None, colidx.numel(),
        _ptr(workspace), workspace.numel() * workspace.element_size(), _ptr(H1),
        _ld(H1) if H1 is not None else 0, _ptr(out), _ld(out), _ptr(pred), ev, n_ev,
        _stream(stream)))


def bigcn_layer_forward_static(X, scale, shift, Wt, rowptr, colidx, H, stream=None):
    """The layer on the library's own static device scratch, for callers that
    cannot allocate device memory (no workspace argument; layers whose
    workspace exceeds STATIC_SCRATCH_BYTES are refused)."""
    N, K = X.shape
    F = Wt.shape[1]
    _check("bigcn_layer_forward_static", lib().bigcn_layer_forward_static(
        _ptr(X), N, K, _ld(X), _ptr(scale), _ptr(shift), _ptr(Wt), F, _ld(Wt), _ptr(rowptr),
        _ptr(colidx) if colidx.numel() else None, colidx.numel(), _ptr(H), _ld(H),
        _stream(stream)))


def bigcn_weighted_dinv(rowptr, values, dinv, stream=None):
    """dinv_i = 1/sqrt(1 + sum of row i's edge weights) (Sec. 3, weighted A)."""
    N = rowptr.numel() - 1
    _check("bigcn_weighted_dinv", lib().bigcn_weighted_dinv(
        _ptr(rowptr), _ptr(values) if values.numel() else None, N, values.numel(), _ptr(dinv),
        _stream(stream)))


def bigcn_spmm_norm_weighted(rowptr, colidx, values, dinv, Z, H, stream=None):
    N, F = Z.shape
    _check("bigcn_spmm_norm_weighted", lib().bigcn_spmm_norm_weighted(
        _ptr(rowptr), _ptr(colidx) if colidx.numel() else None,
        _ptr(values) if values.numel() else None, _ptr(dinv), N, colidx.numel(), _ptr(Z), _ld(Z),
        F, _ptr(H), _ld(H), _stream(stream)))


def bigcn_weighted_layer_workspace_bytes(N: int, K: int, F: int) -> int:
    return int(lib().bigcn_weighted_layer_workspace_bytes(N, K, F))


def bigcn_weighted_layer_forward(X, scale, shift, Wt, rowptr, colidx, values, workspace, H,
                                 stream=None):
    N, K = X.shape
    F = Wt.shape[1]
    _check("bigcn_weighted_layer_forward", lib().bigcn_weighted_layer_forward(
        _ptr(X), N, K, _ld(X), _ptr(scale), _ptr(shift), _ptr(Wt), F, _ld(Wt), _ptr(rowptr),
        _ptr(colidx) if colidx.numel() else None, _ptr(values) if values.numel() else None,
        colidx.numel(), _ptr(workspace), workspace.numel() * workspace.element_size(), _ptr(H),
        _ld(H), _stream(stream)))


# ------------------------------------------------- allocating conveniences ---
def pack_rows(X, scale=None, shift=None, stream=None):
    N, K = X.shape
    bits = torch.empty((N, words_for(K)), dtype=torch.int64, device=X.device)
    alpha = torch.empty(N, dtype=torch.float32, device=X.device)
    bigcn_pack_rows(X, scale, shift, bits, alpha, stream)
    return bits, alpha


def pack_weights(Wt, stream=None):
    K, F = Wt.shape
    bits = torch.empty((F, words_for(K)), dtype=torch.int64, device=Wt.device)
    beta = torch.empty(F, dtype=torch.float32, device=Wt.device)
    bigcn_pack_weights(Wt, bits, beta, stream)
    return bits, beta


def xnor_gemm(a_bits, alpha, b_bits, beta, K, with_dots=False, stream=None):
    N, F = a_bits.shape[0], b_bits.shape[0]
    Z = torch.empty((N, F), dtype=torch.float32, device=a_bits.device)
    dots = torch.empty((N, F), dtype=torch.int32, device=a_bits.device) if with_dots else None
    bigcn_xnor_gemm(a_bits, alpha, b_bits, beta, K, Z, dots, stream)
    return (Z, dots) if with_dots else Z


def spmm_norm(rowptr, colidx, Z, stream=None):
    H = torch.empty_like(Z, memory_format=torch.contiguous_format)
    bigcn_spmm_norm(rowptr, colidx, Z, H, stream)
    return H


def layer_workspace(N, K, F, device):
    nbytes = bigcn_layer_workspace_bytes(N, K, F)
    return torch.empty(max(nbytes, 1), dtype=torch.uint8, device=device)


def layer_forward(X, Wt, rowptr, colidx, scale=None, shift=None, workspace=None, stream=None):
    N, K = X.shape
    F = Wt.shape[1]
    if workspace is None:
        workspace = layer_workspace(N, K, F, X.device)
    H = torch.empty((N, F), dtype=torch.float32, device=X.device)
    bigcn_layer_forward(X, scale, shift, Wt, rowptr, colidx, workspace, H, stream)
    return H
