"""Two-layer Bi-GCN forward on one GPU: device buffers, the C-ABI calls and
their CUDA-graph capture.

Plumbing around libbigcn.so: torch owns the device memory and the stream,
and every step of the computation runs in the library's kernels.

``launch()`` makes the one call ``bigcn_forward_2layer`` (4 kernels for the
usual widths: both weight packs; layer-1 centre + pack + XNOR GEMM; layer-1
aggregation fused with layer 2's pack and GEMM; layer-2 aggregation).
``launch_steps()`` runs the same forward as eight separate step calls
(pack_rows, pack_weights, xnor_gemm_degscaled, spmm_prescaled per layer),
keeping every intermediate in its own buffer, for step-by-step checks.
The output is the logits (no softmax: Eq. 2 belongs to training).
"""
from __future__ import annotations

import torch

from . import binding as B

STEP_KERNELS = ("pack_rows", "pack_weights", "xnor_gemm", "spmm")


FRONT = "L1.pack_rows+L1.xnor_gemm"
FUSED_AGG = "L1.spmm+L2.pack_rows+L2.xnor_gemm"


def fused_kernel_names(N: int, K: int, Fh: int, Fo: int):
    """Names of the kernels bigcn_forward_2layer launches for these sizes, in
    order (4 to 7 of them, depending on which fusions the widths allow)."""
    n = B.bigcn_forward_2layer_launches(N, K, Fh, Fo)
    front_fused = n in (4, 6)
    agg_fused = n in (4, 5)
    names = ["pack_weights(W1,W2)"]
    names += [FRONT] if front_fused else ["L1.pack_rows", "L1.xnor_gemm"]
    names += [FUSED_AGG] if agg_fused else ["L1.spmm", "L2.pack_rows", "L2.xnor_gemm"]
    names += ["L2.spmm"]
    return tuple(names)


class GCN2Forward:
    """Buffers and launch sequence of the 2-layer Bi-GCN forward of Sec. 6.2."""

    def __init__(self, N: int, K: int, hidden: int, out: int, nnz: int, device,
                 keep_h1: bool = False):
        self.N, self.K, self.hidden, self.out, self.nnz = N, K, hidden, out, nnz
        self.device = torch.device(device)
        f32, i64 = torch.float32, torch.int64
        e = lambda *shape, dtype=f32: torch.empty(shape, dtype=dtype, device=self.device)
        # inputs
        self.X, self.s, self.t = e(N, K), e(K), e(K)
        self.W1, self.W2 = e(K, hidden), e(hidden, out)
        self.rowptr, self.colidx = e(N + 1, dtype=i64), e(max(nnz, 1), dtype=torch.int32)[:nnz]
        # fused forward
        nbytes = B.bigcn_forward_2layer_workspace_bytes(N, K, hidden, out)
        self.workspace = torch.empty(max(nbytes, 1), dtype=torch.uint8, device=self.device)
        self.logits = e(N, out)
        self.H1 = e(N, hidden) if keep_h1 else None
        self.kernel_names = fused_kernel_names(N, K, hidden, out)
        self.graph = None
        self._steps = None

    def input_tensors(self):
        return dict(X=self.X, s=self.s, t=self.t, W1=self.W1, W2=self.W2,
                    rowptr=self.rowptr, colidx=self.colidx)

    def load(self, non_blocking: bool = True, **tensors):
        """Copy inputs (host, pinned host or device tensors) into the buffers."""
        dst = self.input_tensors()
        for name, src in tensors.items():
            dst[name].copy_(src, non_blocking=non_blocking)

    def launch(self, events=None):
        """Enqueue the fused forward on the current stream; ``events`` (len =
        launches + 1) are recorded before each kernel and after the last."""
        B.bigcn_forward_2layer(self.X, self.s, self.t, self.W1, self.W2, self.rowptr,
                               self.colidx, self.workspace, self.logits, H1=self.H1,
                               events=events)

    def capture(self, events=None):
        """Capture launch(events) into a CUDA graph (replayed by replay())."""
        if events:
            for ev in events:       # torch creates the CUDA event on first record
                ev.record()
        s = torch.cuda.Stream(device=self.device)
        s.wait_stream(torch.cuda.current_stream(self.device))
        with torch.cuda.stream(s):
            self.launch(events)     # warm-up outside the graph
        torch.cuda.current_stream(self.device).wait_stream(s)
        torch.cuda.synchronize(self.device)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            self.launch(events)
        self.graph = g
        return g

    def replay(self):
        self.graph.replay()

    # ----------------------------------------------------- step by step ----
    def _alloc_steps(self):
        N, K, Fh, Fo = self.N, self.K, self.hidden, self.out
        f32, i64 = torch.float32, torch.int64
        e = lambda *shape, dtype=f32: torch.empty(shape, dtype=dtype, device=self.device)
        w1, w2 = B.words_for(K), B.words_for(Fh)
        self._steps = True
        self.bits1, self.alpha1 = e(N, w1, dtype=i64), e(N)
        self.wbits1, self.beta1 = e(Fh, w1, dtype=i64), e(Fh)
        self.Z1, self.H1s = e(N, Fh), e(N, Fh)
        self.bits2, self.alpha2 = e(N, w2, dtype=i64), e(N)
        self.wbits2, self.beta2 = e(Fo, w2, dtype=i64), e(Fo)
        self.Z2, self.logits_steps = e(N, Fo), e(N, Fo)

    def launch_steps(self):
        """The same forward as eight step calls, every intermediate kept."""
        if self._steps is None:
            self._alloc_steps()
        B.bigcn_pack_rows(self.X, self.s, self.t, self.bits1, self.alpha1)
        B.bigcn_pack_weights(self.W1, self.wbits1, self.beta1)
        B.bigcn_xnor_gemm_degscaled(self.bits1, self.alpha1, self.wbits1, self.beta1, self.K,
                                    self.rowptr, self.Z1)
        B.bigcn_spmm_prescaled(self.rowptr, self.colidx, self.Z1, self.H1s)
        B.bigcn_pack_rows(self.H1s, None, None, self.bits2, self.alpha2)
        B.bigcn_pack_weights(self.W2, self.wbits2, self.beta2)
        B.bigcn_xnor_gemm_degscaled(self.bits2, self.alpha2, self.wbits2, self.beta2,
                                    self.hidden, self.rowptr, self.Z2)
        B.bigcn_spmm_prescaled(self.rowptr, self.colidx, self.Z2, self.logits_steps)
