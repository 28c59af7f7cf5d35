"""GPU back-propagation of one layer (bigcn_layer_backward) against the
oracle's Algorithm 1 with Eqs. bp-H and bp-W, on the same seeded inputs.

Tolerance. dW and dX come from sums whose terms cancel -- dW over all N
rows, dX over the F columns -- evaluated in fp32 on the GPU and in double in
the oracle. They are compared with |gpu - oracle| <= 1e-6 + 1e-4 * scale,
scale = max(|oracle|, the sum of the |terms| that make the value) (the scale
of any fp32 evaluation order's error); the plain form, scale = |oracle|, is
required wherever 1e-4 |oracle| exceeds sqrt(n) 2^-24 scale, the typical
rounding error of an fp32 sum of n terms (below that the terms have cancelled
to under what fp32 resolves). Where |dL/dH~| lies within that tolerance of 1, Eq. bp-H's clip
may fall either way, and both results are accepted.
"""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import ATOL, RTOL, check_sum as check, to_dev
from paper_2010_07565_gb300 import binding as B
from paper_2010_07565_gb300 import inputs

pytestmark = pytest.mark.gpu


def rng(seed):
    return np.random.Generator(np.random.PCG64(seed))


def run_backward(case, dH, with_dx=True, dev=None):
    d = {k: to_dev(v) for k, v in case.items()}
    N, K = case["X"].shape
    F = case["W"].shape[1]
    ws = torch.empty(max(B.bigcn_layer_backward_workspace_bytes(N, K, F), 1), dtype=torch.uint8,
                     device=dev)
    dW = torch.full((K, F), float("nan"), device=dev)
    dX = torch.full((N, K), float("nan"), device=dev) if with_dx else None
    B.bigcn_layer_backward(d["X"], d["s"], d["t"], d["W"], d["rowptr"], d["colidx"],
                           to_dev(dH.astype(np.float32)), ws, dW, dX=dX)
    torch.cuda.synchronize()
    return dW.cpu().numpy().astype(np.float64), (dX.cpu().numpy().astype(np.float64)
                                                 if with_dx else None)




CASES = [
    # (N, K, F, mean degree, hub degree, centred)
    (300, 70, 6, 4.0, 0, True),
    (517, 130, 16, 3.0, 0, False),
    (1000, 602, 41, 8.0, 300, True),      # K past a 64-multiple, hub rows
    (2708, 1433, 64, 4.0, 0, True),       # Cora-shaped layer 1
    (5000, 200, 33, 5.0, 800, True),      # several row chunks for dW
    (1, 1, 1, 0.0, 0, False),             # a single node and feature
]


@pytest.mark.parametrize("N,K,F,deg,hub,centred", CASES)
def test_layer_backward_matches_oracle(cuda_device, N, K, F, deg, hub, centred):
    case = inputs.layer_case(N, K, F, seed=N + K + F, mean_degree=deg, hub_degree=hub,
                             centred=centred)
    dH = 5.0 * rng(N * 7 + F).standard_normal((N, F))   # some |dL/dH~| >= 1
    dW, dX = run_backward(case, dH, dev=cuda_device)
    ref = oracle.layer_backward(case["X"], case["W"], case["rowptr"], case["colidx"], dH,
                                case["s"], case["t"])
    # dW: error scale through dW~ (sum over rows) and its column sum.
    scale_w = np.broadcast_to(ref["Wg_abs"] * (1.0 + ref["beta"]), dW.shape)
    check(dW, ref["dW"], scale_w, "dW", nterms=N + K)
    # dX: clipped dL/dH~; accept either side of the clip where |dL/dH~| ~ 1.
    scale_x = np.broadcast_to(ref["Ht_abs"][:, None], dX.shape)
    tol = ATOL + RTOL * np.maximum(np.abs(ref["Ht"]), scale_x)
    edge = np.abs(np.abs(ref["Ht"]) - 1.0) <= tol
    inside = ~edge
    check(dX[inside], ref["dX"][inside], scale_x[inside], "dX", nterms=F)
    ok_edge = (dX[edge] == 0.0) | (np.abs(dX[edge] - ref["Ht"][edge]) <= tol[edge])
    assert ok_edge.all()
    assert np.isfinite(dW).all() and np.isfinite(dX).all()
    # Some entries are clipped and some are not (Eq. bp-H is exercised).
    if N * K > 1000:
        assert 0 < np.count_nonzero(np.abs(ref["Ht"]) >= 1.0) < ref["Ht"].size


def test_layer_backward_without_dx_and_zero_gradient(cuda_device):
    case = inputs.layer_case(400, 100, 8, seed=5)
    dW, dX = run_backward(case, np.zeros((400, 8)), with_dx=False, dev=cuda_device)
    assert dX is None and np.array_equal(dW, np.zeros_like(dW))


def test_layer_backward_is_deterministic(cuda_device):
    case = inputs.layer_case(3000, 300, 24, seed=9, hub_degree=500)
    dH = rng(10).standard_normal((3000, 24))
    a = run_backward(case, dH, dev=cuda_device)
    b = run_backward(case, dH, dev=cuda_device)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])


def test_layer_backward_argument_errors(cuda_device):
    X = torch.zeros((10, 8), device=cuda_device)
    W = torch.zeros((8, 3), device=cuda_device)
    rowptr = torch.zeros(11, dtype=torch.int64, device=cuda_device)
    colidx = torch.zeros(0, dtype=torch.int32, device=cuda_device)
    dH = torch.zeros((10, 3), device=cuda_device)
    dW = torch.full((8, 3), 5.0, device=cuda_device)
    small = torch.empty(16, dtype=torch.uint8, device=cuda_device)
    with pytest.raises(B.BigcnError):                              # workspace too small
        B.bigcn_layer_backward(X, None, None, W, rowptr, colidx, dH, small, dW)
    ws = torch.empty(B.bigcn_layer_backward_workspace_bytes(10, 8, 3), dtype=torch.uint8,
                     device=cuda_device)
    with pytest.raises(B.BigcnError):                              # dW overlaps dH
        B.bigcn_layer_backward(X, None, None, W, rowptr, colidx, dH, ws, dH[:8])
    torch.cuda.synchronize()
    assert torch.all(dW == 5.0)
