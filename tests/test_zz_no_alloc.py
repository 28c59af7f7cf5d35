"""The layer entry point that allocates nothing: bigcn_layer_forward_static.

It exists for callers that may not allocate device memory at all — serving
loops that ban cudaMalloc/cudaFree once running because both can stall the
device, plug-ins whose host application owns the whole device memory budget,
deployments that fix their memory footprint at load time. Instead of a
workspace argument it uses a 32 MiB array compiled into the library.

Checked here through the C ABI: its output equals that of
bigcn_layer_forward with a caller-allocated workspace bit for bit (both run
the same kernels on 256-byte aligned scratch, so any difference would be a
stale or misplaced scratch read), with no bounded device wait run out, on
two calls in a row per case and across
cases of different sizes, so a call must not depend on what the previous
call left in the shared array; and a layer whose workspace would not fit is
refused with BIGCN_ERR_SCRATCH_LIMIT before anything runs. The file is named
so that pytest collects it last.
"""
import ctypes

import numpy as np
import pytest
import torch

from gpu_helpers import assert_close, to_dev
from paper_2010_07565_gb300 import binding as B
from paper_2010_07565_gb300 import inputs

pytestmark = pytest.mark.gpu

SCRATCH_LIMIT = 5

CASES = [
    # (N, K, F, mean degree, hub degree, centred)
    (2708, 1433, 64, 4.0, 0, True),      # a Cora-shaped first layer
    (2708, 64, 7, 4.0, 0, False),        # its second layer
    (19717, 500, 64, 4.5, 400, True),    # a PubMed-shaped first layer
    (301, 203, 19, 4.0, 40, True),
]


def call_static(d, H):
    N, K = d["X"].shape
    F = d["W"].shape[1]
    p = lambda t: None if t is None else ctypes.c_void_p(t.data_ptr())
    return B.lib().bigcn_layer_forward_static(
        p(d["X"]), N, K, K, p(d["s"]), p(d["t"]), p(d["W"]), F, F, p(d["rowptr"]),
        p(d["colidx"]), d["colidx"].numel(), p(H), F,
        ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))


def test_static_scratch_layer_matches_workspace_layer(cuda_device):
    for (N, K, F, deg, hub, centred) in CASES:
        case = inputs.layer_case(N, K, F, seed=N + K + F, mean_degree=deg, hub_degree=hub,
                                 centred=centred)
        d = {k: to_dev(v) for k, v in case.items()}
        ws = torch.empty(B.bigcn_layer_workspace_bytes(N, K, F), dtype=torch.uint8,
                         device=cuda_device)
        H_ref = torch.empty((N, F), dtype=torch.float32, device=cuda_device)
        B.bigcn_layer_forward(d["X"], d["s"], d["t"], d["W"], d["rowptr"], d["colidx"], ws,
                              H_ref)
        ref = H_ref.cpu().numpy().astype(np.float64)
        assert B.device_timeouts() == 0
        for call in range(2):
            H = torch.full((N, F), float("nan"), dtype=torch.float32, device=cuda_device)
            assert call_static(d, H) == 0, f"call {call} on N={N}, K={K}, F={F}"
            torch.cuda.synchronize()
            assert B.device_timeouts() == 0, f"call {call} on N={N}, K={K}, F={F}"
            assert_close(H, ref, f"static-scratch layer, call {call}, N={N} K={K} F={F}")
            assert torch.equal(H, H_ref), f"call {call} on N={N}, K={K}, F={F}: not bit-equal"


def test_static_scratch_refuses_a_layer_that_does_not_fit(cuda_device):
    N, K, F = 200_000, 602, 128           # workspace ~118 MB > 32 MiB
    assert B.bigcn_layer_workspace_bytes(N, K, F) > B.STATIC_SCRATCH_BYTES
    d = dict(X=torch.zeros((N, K), device=cuda_device), s=None, t=None,
             W=torch.zeros((K, F), device=cuda_device),
             rowptr=torch.zeros(N + 1, dtype=torch.int64, device=cuda_device),
             colidx=torch.zeros(0, dtype=torch.int32, device=cuda_device))
    H = torch.full((N, F), 3.0, device=cuda_device)
    assert call_static(d, H) == SCRATCH_LIMIT
    torch.cuda.synchronize()
    assert bool(torch.all(H == 3.0))
    assert B.status_string(SCRATCH_LIMIT) == "BIGCN_ERR_SCRATCH_LIMIT"
