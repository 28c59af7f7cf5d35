"""Two-layer Bi-GCN forward on one GPU: device buffers and the sequence of
C-ABI calls, optionally replayed as a CUDA graph.

This is plumbing around libbigcn.so: torch owns the device memory and the
stream, and every step of the computation is one call of the C interface:

    layer 1:  bigcn_pack_rows (centred)  -> bigcn_pack_weights
              -> bigcn_xnor_gemm_degscaled -> bigcn_spmm_prescaled
    layer 2:  the same four calls on H1, without centring (Sec. 4.1.2)

i.e. two bigcn_layer_forward's worth of kernels, issued one by one so that
callers can put timing events between them. The layer-2 output is the
logits (no softmax: Eq. 2 belongs to training).
"""
from __future__ import annotations

import torch

from . import binding as B

STEP_KERNELS = ("pack_rows", "pack_weights", "xnor_gemm", "spmm")


class GCN2Forward:
    """Buffers and launch sequence of the 2-layer Bi-GCN forward of Sec. 6.2."""

    def __init__(self, N: int, K: int, hidden: int, out: int, nnz: int, device):
        self.N, self.K, self.hidden, self.out, self.nnz = N, K, hidden, out, nnz
        self.device = torch.device(device)
        f32, i64 = torch.float32, torch.int64
        e = lambda *shape, dtype=f32: torch.empty(shape, dtype=dtype, device=self.device)
        w1, w2 = B.words_for(K), B.words_for(hidden)
        # inputs
        self.X, self.s, self.t = e(N, K), e(K), e(K)
        self.W1, self.W2 = e(K, hidden), e(hidden, out)
        self.rowptr, self.colidx = e(N + 1, dtype=i64), e(max(nnz, 1), dtype=torch.int32)[:nnz]
        # layer 1 intermediates and output
        self.bits1, self.alpha1 = e(N, w1, dtype=i64), e(N)
        self.wbits1, self.beta1 = e(hidden, w1, dtype=i64), e(hidden)
        self.Z1, self.H1 = e(N, hidden), e(N, hidden)
        # layer 2
        self.bits2, self.alpha2 = e(N, w2, dtype=i64), e(N)
        self.wbits2, self.beta2 = e(out, w2, dtype=i64), e(out)
        self.Z2, self.logits = e(N, out), e(N, out)
        self.graph = None

    def input_tensors(self):
        return dict(X=self.X, s=self.s, t=self.t, W1=self.W1, W2=self.W2,
                    rowptr=self.rowptr, colidx=self.colidx)

    def load(self, non_blocking: bool = True, **tensors):
        """Copy inputs (host, pinned host or device tensors) into the buffers."""
        dst = self.input_tensors()
        for name, src in tensors.items():
            dst[name].copy_(src, non_blocking=non_blocking)

    def launch(self, events=None):
        """Enqueue the 8 kernels on the current stream. ``events`` (9 or None)
        are recorded before the first, between each, and after the last."""
        rec = (lambda k: events[k].record()) if events is not None else (lambda k: None)
        rec(0)
        B.bigcn_pack_rows(self.X, self.s, self.t, self.bits1, self.alpha1)
        rec(1)
        B.bigcn_pack_weights(self.W1, self.wbits1, self.beta1)
        rec(2)
        B.bigcn_xnor_gemm_degscaled(self.bits1, self.alpha1, self.wbits1, self.beta1, self.K,
                                    self.rowptr, self.Z1)
        rec(3)
        B.bigcn_spmm_prescaled(self.rowptr, self.colidx, self.Z1, self.H1)
        rec(4)
        B.bigcn_pack_rows(self.H1, None, None, self.bits2, self.alpha2)
        rec(5)
        B.bigcn_pack_weights(self.W2, self.wbits2, self.beta2)
        rec(6)
        B.bigcn_xnor_gemm_degscaled(self.bits2, self.alpha2, self.wbits2, self.beta2,
                                    self.hidden, self.rowptr, self.Z2)
        rec(7)
        B.bigcn_spmm_prescaled(self.rowptr, self.colidx, self.Z2, self.logits)
        rec(8)

    def capture(self, events=None):
        """Capture launch(events) into a CUDA graph (replayed by replay())."""
        s = torch.cuda.Stream(device=self.device)
        s.wait_stream(torch.cuda.current_stream(self.device))
        with torch.cuda.stream(s):
            self.launch(events)          # warm-up outside the graph
        torch.cuda.current_stream(self.device).wait_stream(s)
        torch.cuda.synchronize(self.device)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            self.launch(events)
        self.graph = g
        return g

    def replay(self):
        self.graph.replay()
