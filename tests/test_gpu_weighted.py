"""Parity of the weighted-adjacency calls (Sec. 3's A = [a_ij] with general
entries, Eq. 1's operator on A + I) against the oracle: the weighted degrees
(dinv = 1/sqrt(dhat), rows summed by one warp and, past 2048 entries, by a
whole block), the weighted aggregation over fp32 rows (every lane-group
width and column slab, heavy rows, padded row strides) and the weighted
layer, whose product is kept factored (uint16 dots, 4 or 8 a lane) or is
fp32 (K > 32767), and which runs the tensor-core product from 128 rows per
SM. Edge weights are seeded, symmetric, uniform in [0.5, 2); one case has
zero weights."""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import assert_close, check_sum, padded, to_dev
from paper_2010_07565_gb300 import binding as B
from paper_2010_07565_gb300 import inputs

pytestmark = pytest.mark.gpu


def dinv_ref(rowptr, values):
    return 1.0 / np.sqrt(oracle.degree_weighted(rowptr, values))


# (N, mean degree, hub degree, zero weights)
DINV_CASES = [(1, 0.0, 0, False), (7, 2.0, 0, False), (1003, 6.0, 0, False),
              (5003, 6.0, 4500, False), (4000, 12.0, 2049, True)]


@pytest.mark.parametrize("N,deg,hub,zero", DINV_CASES)
def test_weighted_dinv(cuda_device, N, deg, hub, zero):
    rp, ci = inputs.random_graph(N, deg, N + hub, hub_degree=hub)
    vals = np.zeros(ci.size, np.float32) if zero else inputs.edge_weights(rp, ci, N)
    dinv = torch.full((N,), float("nan"), device=cuda_device)
    B.bigcn_weighted_dinv(to_dev(rp), to_dev(vals), dinv)
    again = torch.empty_like(dinv)
    B.bigcn_weighted_dinv(to_dev(rp), to_dev(vals), again)
    torch.cuda.synchronize()
    assert_close(dinv, dinv_ref(rp, vals), f"dinv N={N} hub={hub}", rtol=1e-6, atol=0.0)
    assert torch.equal(dinv, again)             # a fixed summation order


# (N, F, ldz pad, mean degree, hub)
SPMM_CASES = [(500, 1, 0, 4.0, 0), (777, 3, 1, 6.0, 300), (1000, 8, 0, 12.0, 700),
              (2000, 64, 4, 9.0, 1500), (600, 130, 0, 5.0, 0), (900, 300, 2, 10.0, 600)]


@pytest.mark.parametrize("N,F,pad,deg,hub", SPMM_CASES)
def test_spmm_norm_weighted(cuda_device, N, F, pad, deg, hub):
    rp, ci = inputs.random_graph(N, deg, 3 * N + F, hub_degree=hub)
    vals = inputs.edge_weights(rp, ci, F)
    z = np.random.default_rng(N + F).standard_normal((N, F)).astype(np.float32)
    Zv, _ = padded(to_dev(z), N, F, F + pad)
    Hv, _ = padded(torch.zeros((N, F), device=cuda_device), N, F, F + pad, float("nan"))
    dinv = torch.empty(N, device=cuda_device)
    rp_d, ci_d, v_d = to_dev(rp), to_dev(ci), to_dev(vals)
    B.bigcn_weighted_dinv(rp_d, v_d, dinv)
    B.bigcn_spmm_norm_weighted(rp_d, ci_d, v_d, dinv, Zv, Hv)
    torch.cuda.synchronize()
    ref, absterm = oracle.aggregate_weighted(rp, ci, vals, z, with_absterm=True)
    check_sum(Hv.cpu().numpy(), ref, absterm, f"weighted aggregation N={N} F={F}",
              nterms=int(np.diff(rp).max()) + 1)


def run_layer(cuda_device, case, vals):
    d = {k: to_dev(v) for k, v in case.items()}
    N, K = case["X"].shape
    F = case["W"].shape[1]
    ws = torch.empty(B.bigcn_weighted_layer_workspace_bytes(N, K, F), dtype=torch.uint8,
                     device=cuda_device)
    H = torch.full((N, F), float("nan"), device=cuda_device)
    B.bigcn_weighted_layer_forward(d["X"], d["s"], d["t"], d["W"], d["rowptr"], d["colidx"],
                                   to_dev(vals), ws, H)
    torch.cuda.synchronize()
    assert B.device_timeouts() == 0
    return H.cpu().numpy()


# (N, K, F, mean degree, hub): factored uint16 dots 4 a lane (mean degree < 8)
# and 8 a lane, heavy rows, F not a multiple of 4, fp32 product (K > 32767).
LAYER_CASES = [(1000, 300, 64, 6.0, 0), (2000, 602, 128, 12.0, 900), (777, 1433, 7, 4.0, 0),
               (3001, 100, 41, 16.0, 2500), (1, 50, 5, 0.0, 0), (300, 33000, 5, 4.0, 0)]


@pytest.mark.parametrize("N,K,F,deg,hub", LAYER_CASES)
def test_weighted_layer_forward(cuda_device, N, K, F, deg, hub):
    case = inputs.layer_case(N, K, F, seed=N + K + F, mean_degree=deg, hub_degree=hub)
    rp, ci = case["rowptr"], case["colidx"]
    vals = inputs.edge_weights(rp, ci, K)
    H = run_layer(cuda_device, case, vals)
    ref = oracle.layer_forward_weighted(case["X"], case["W"], rp, ci, vals, case["s"], case["t"])
    check_sum(H, ref["H"], ref["absterm"], f"weighted layer N={N} K={K} F={F}",
              nterms=K + (int(np.diff(rp).max()) if N > 1 else 0) + 1)


def test_weighted_layer_with_zero_and_unit_weights(cuda_device):
    """Zero weights leave each node its own product (dhat = 1); unit weights
    give the 0/1 layer."""
    case = inputs.layer_case(1500, 256, 32, seed=77, mean_degree=8.0)
    rp, ci = case["rowptr"], case["colidx"]
    H0 = run_layer(cuda_device, case, np.zeros(ci.size, np.float32))
    ref0 = oracle.layer_forward_weighted(case["X"], case["W"], rp, ci, np.zeros(ci.size),
                                         case["s"], case["t"])
    check_sum(H0, ref0["zeta"], np.abs(ref0["zeta"]), "weighted layer, zero weights", nterms=257)
    H1 = run_layer(cuda_device, case, np.ones(ci.size, np.float32))
    ref1 = oracle.layer_forward(case["X"], case["W"], rp, ci, case["s"], case["t"])
    check_sum(H1, ref1["H"], ref1["absterm"], "weighted layer, unit weights",
              nterms=256 + int(np.diff(rp).max()) + 1)


def test_weighted_layer_on_the_tensor_core_product(cuda_device):
    """Enough rows for the tcgen05 product (128 per SM, a ragged last tile);
    H compared on sampled rows."""
    sms = torch.cuda.get_device_properties(cuda_device).multi_processor_count
    N, K, F = 128 * sms + 77, 602, 128
    case = inputs.layer_case(N, K, F, seed=5, mean_degree=10.0, hub_degree=3000)
    rp, ci = case["rowptr"], case["colidx"]
    vals = inputs.edge_weights(rp, ci, 6)
    H = run_layer(cuda_device, case, vals)
    rows = np.unique(np.concatenate([[0, 1, N - 1],
                                     np.random.default_rng(3).choice(N, 1024, replace=False)]))
    ref = oracle.layer_forward_weighted(case["X"], case["W"], rp, ci, vals, case["s"], case["t"],
                                        rows=rows)
    check_sum(H[rows], ref["H"], ref["absterm"], "weighted layer, tensor-core product (sampled)",
              nterms=K + int(np.diff(rp)[rows].max()) + 1)
