"""GPU parity of the binarized inductive layers (Sec. 6.3, Table 3:
Bi-inductiveGCN's mean aggregator and Bi-GraphSAGE's self + neighbour-mean
aggregator) against the oracle, through the C ABI.

The products are exact integers scaled by fp32 alpha and beta; the
aggregation's fp32 sums are compared with |gpu - oracle| <= 1e-6 + 1e-4 *
max(|oracle|, scale), scale = the sum of the |terms| of the aggregation, the
plain |oracle|-relative form required wherever 1e-4 |oracle| exceeds
sqrt(n) 2^-24 scale, the typical rounding error of an fp32 sum of n terms.
Graphs: isolated nodes (GraphSAGE's mean is then 0), a hub heavy enough for
the whole-block path, mean degree past 8 (eight dots per lane), no edges; K
past 32767 (the product kept in fp32 instead of 16-bit dots); F not a
multiple of 8 (padded halves of GraphSAGE's concatenated product).
"""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import check_sum as check, padded, to_dev
from paper_2010_07565_gb300 import binding as B
from paper_2010_07565_gb300 import inputs

pytestmark = pytest.mark.gpu




def maxdeg(case):
    return int(np.diff(case["rowptr"]).max(initial=0)) + 1


def run(agg, case, Wn=None, ldh=None, dev=None):
    d = {k: to_dev(v) for k, v in case.items()}
    N, K = case["X"].shape
    F = case["W"].shape[1]
    ws = torch.empty(max(B.bigcn_inductive_layer_workspace_bytes(agg, N, K, F), 1),
                     dtype=torch.uint8, device=dev)
    if ldh is None:
        H = torch.full((N, F), float("nan"), device=dev)
        buf = H
    else:
        H, buf = padded(torch.zeros((N, F), device=dev), N, F, ldh, fill=-3.0)
    B.bigcn_inductive_layer_forward(agg, d["X"], d["s"], d["t"], d["W"], d["rowptr"],
                                    d["colidx"], ws, H, W_neigh=to_dev(Wn))
    torch.cuda.synchronize()
    return H.cpu().numpy(), buf


CASES = [
    # (N, K, F, mean degree, hub degree)
    (300, 70, 6, 4.0, 0),
    (400, 90, 13, 1.0, 0),           # many isolated nodes
    (2708, 1433, 64, 4.0, 0),        # Cora-shaped layer 1
    (3327, 3703, 64, 2.8, 0),        # Citeseer-shaped: GraphSAGE on the split front
    (5000, 300, 33, 6.0, 900),       # a hub on the whole-block path
    (3000, 200, 128, 12.0, 0),       # mean degree past 8: eight dots per lane
    (50, 20, 5, 0.0, 0),             # no edges
]


@pytest.mark.parametrize("N,K,F,deg,hub", CASES)
@pytest.mark.parametrize("agg", ["mean", "sage"])
def test_inductive_layer_matches_oracle(cuda_device, agg, N, K, F, deg, hub):
    case = inputs.layer_case(N, K, F, seed=3 * N + F, mean_degree=deg, hub_degree=hub,
                             features_kind="bernoulli" if K == 1433 else "normal")
    Wn = inputs.weights(K, F, seed=K + 17 * F) if agg == "sage" else None
    H, _ = run(agg, case, Wn, dev=cuda_device)
    ref = oracle.layer_forward_inductive(case["X"], case["W"], case["rowptr"], case["colidx"],
                                         agg, case["s"], case["t"], W_neigh=Wn)
    check(H, ref["H"], ref["absterm"], f"{agg} layer {N}x{K}x{F}", nterms=K + maxdeg(case))
    assert B.device_timeouts() == 0


@pytest.mark.parametrize("agg", ["mean", "sage"])
def test_inductive_layer_past_the_16_bit_dots(cuda_device, agg):
    N, K, F = 150, 33000, 7
    case = inputs.layer_case(N, K, F, seed=5, mean_degree=3.0)
    Wn = inputs.weights(K, F, seed=6) if agg == "sage" else None
    H, _ = run(agg, case, Wn, dev=cuda_device)
    ref = oracle.layer_forward_inductive(case["X"], case["W"], case["rowptr"], case["colidx"],
                                         agg, case["s"], case["t"], W_neigh=Wn)
    check(H, ref["H"], ref["absterm"], f"{agg} layer, K = {K}", nterms=K + maxdeg(case))


def test_inductive_layer_padded_output_and_gcn_mode(cuda_device):
    N, K, F = 1200, 150, 10
    case = inputs.layer_case(N, K, F, seed=7, mean_degree=5.0)
    Wn = inputs.weights(K, F, seed=8)
    H, buf = run("sage", case, Wn, ldh=13, dev=cuda_device)
    assert torch.all(buf[:, F:] == -3.0)
    ref = oracle.layer_forward_inductive(case["X"], case["W"], case["rowptr"], case["colidx"],
                                         "sage", case["s"], case["t"], W_neigh=Wn)
    check(H, ref["H"], ref["absterm"], "sage layer, padded H", nterms=K + maxdeg(case))
    # The "gcn" aggregator is bigcn_layer_forward.
    d = {k: to_dev(v) for k, v in case.items()}
    ws = torch.empty(B.bigcn_inductive_layer_workspace_bytes("gcn", N, K, F), dtype=torch.uint8,
                     device=cuda_device)
    H1, H2 = torch.empty((N, F), device=cuda_device), torch.empty((N, F), device=cuda_device)
    B.bigcn_inductive_layer_forward("gcn", d["X"], d["s"], d["t"], d["W"], d["rowptr"],
                                    d["colidx"], ws, H1)
    B.bigcn_layer_forward(d["X"], d["s"], d["t"], d["W"], d["rowptr"], d["colidx"], ws, H2)
    torch.cuda.synchronize()
    assert torch.equal(H1, H2)


def test_inductive_layer_is_deterministic(cuda_device):
    case = inputs.layer_case(3000, 300, 40, seed=9, hub_degree=700)
    Wn = inputs.weights(300, 40, seed=10)
    a, _ = run("sage", case, Wn, dev=cuda_device)
    b, _ = run("sage", case, Wn, dev=cuda_device)
    assert np.array_equal(a, b)


def test_inductive_argument_errors(cuda_device):
    N, K, F = 10, 8, 3
    X = torch.zeros((N, K), device=cuda_device)
    W = torch.zeros((K, F), device=cuda_device)
    rowptr = torch.zeros(N + 1, dtype=torch.int64, device=cuda_device)
    colidx = torch.zeros(0, dtype=torch.int32, device=cuda_device)
    H = torch.full((N, F), 5.0, device=cuda_device)
    assert B.bigcn_inductive_layer_workspace_bytes(9, N, K, F) == 0
    ws = torch.empty(B.bigcn_inductive_layer_workspace_bytes("sage", N, K, F), dtype=torch.uint8,
                     device=cuda_device)
    with pytest.raises(B.BigcnError):                              # GraphSAGE without W_neigh
        B.bigcn_inductive_layer_forward("sage", X, None, None, W, rowptr, colidx, ws, H)
    with pytest.raises(B.BigcnError):                              # unknown aggregator
        B.bigcn_inductive_layer_forward(9, X, None, None, W, rowptr, colidx, ws, H, W_neigh=W)
    with pytest.raises(B.BigcnError):                              # workspace too small
        B.bigcn_inductive_layer_forward("sage", X, None, None, W, rowptr, colidx, ws[:256], H,
                                        W_neigh=W)
    torch.cuda.synchronize()
    assert torch.all(H == 5.0)
