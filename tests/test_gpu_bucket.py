"""GPU parity of sub-row bucketing (Sec. 4.1, buckets of B consecutive values
with their own scales) against the oracle, through the C ABI: packed signs
bit-exact, per-bucket scales and products within |g - o| <= 1e-6 + 1e-4 *
max(|o|, scale) (scale = the sum of the |terms|, the products being sums of
per-bucket terms with both signs); the plain form is required wherever
1e-4 |o| exceeds sqrt(n) 2^-24 scale, the typical rounding error of an fp32
sum of n terms.
Buckets from one word (64) to more than K (one bucket: Bi-GCN), K and F
ragged, a last bucket shorter than B, few tiles (the k-steps split over a
cluster) and many, extra words in the packed rows.
"""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import check_sum as check, assert_bits_equal, assert_close, to_dev
from paper_2010_07565_gb300 import binding as B_
from paper_2010_07565_gb300 import inputs

pytestmark = pytest.mark.gpu


def rng(seed):
    return np.random.Generator(np.random.PCG64(seed))




PACK_CASES = [(1, 1, 64), (37, 63, 64), (20, 64, 64), (19, 65, 64), (300, 200, 128),
              (129, 1433, 192), (64, 1433, 640), (50, 500, 4096)]


@pytest.mark.parametrize("N,K,B", PACK_CASES)
@pytest.mark.parametrize("affine", [True, False])
def test_pack_rows_bucketed(cuda_device, N, K, B, affine):
    g = rng(N + K + B)
    X = (g.standard_normal((N, K)) * 1.5 + 0.2).astype(np.float32)
    X[0, 0] = 0.0
    if K > 1:
        X[0, 1] = -0.0
    s, t = inputs.bn_stats(X) if affine else (None, None)
    words = oracle.words_for(K) + 1                         # one extra word must read zero
    nb = oracle.buckets(K, B)
    bits = torch.full((N, words), -1, dtype=torch.int64, device=cuda_device)
    alpha = torch.empty((N, nb), device=cuda_device)
    B_.bigcn_pack_rows_bucketed(to_dev(X), to_dev(s), to_dev(t), B, bits, alpha)
    Y = oracle.centre(X, s, t)
    assert_bits_equal(bits, oracle.pack(oracle.sign(Y), words=words), "bucketed packed rows")
    assert_close(alpha, oracle.row_scale_bucketed(Y, B), "alpha per bucket")


@pytest.mark.parametrize("K,F,B", [(1, 1, 64), (63, 6, 64), (130, 17, 64), (602, 128, 192),
                                   (1433, 64, 512), (500, 3, 4096)])
def test_pack_weights_bucketed(cuda_device, K, F, B):
    Wt = inputs.weights(K, F, seed=K + F + B)
    Wt[0, 0] = -0.0
    words, nb = oracle.words_for(K), oracle.buckets(K, B)
    bits = torch.full((F, words), -1, dtype=torch.int64, device=cuda_device)
    beta = torch.empty((F, nb), device=cuda_device)
    B_.bigcn_pack_weights_bucketed(to_dev(Wt), B, bits, beta)
    SB = oracle.sign(np.ascontiguousarray(Wt.T))
    assert_bits_equal(bits, oracle.pack(SB), "bucketed packed weights")
    assert_close(beta, oracle.weight_scale_bucketed(Wt, B), "beta per bucket")


GEMM_CASES = [(1, 1, 1, 64), (100, 63, 6, 64), (300, 130, 16, 64), (2708, 1433, 64, 128),
              (1000, 602, 100, 192), (20000, 500, 64, 128), (700, 1024, 33, 1024),
              (513, 700, 20, 2048)]


@pytest.mark.parametrize("N,K,F,B", GEMM_CASES)
def test_xnor_gemm_bucketed(cuda_device, N, K, F, B):
    g = rng(3 * N + K + F + B)
    SF = np.where(g.random((N, K)) < 0.5, -1, 1).astype(np.int8)
    SB = np.where(g.random((F, K)) < 0.5, -1, 1).astype(np.int8)
    nb = oracle.buckets(K, B)
    alpha = g.uniform(0.05, 2.0, (N, nb)).astype(np.float32)
    beta = g.uniform(0.05, 2.0, (F, nb)).astype(np.float32)
    ref, mag = oracle.zeta_bucketed(SF, alpha.astype(np.float64), SB, beta.astype(np.float64), B,
                                    with_absterm=True)
    Z = torch.full((N, F), float("nan"), device=cuda_device)
    B_.bigcn_xnor_gemm_bucketed(to_dev(oracle.pack(SF)), to_dev(alpha), to_dev(oracle.pack(SB)),
                                to_dev(beta), K, B, Z)
    torch.cuda.synchronize()
    check(Z.cpu().numpy(), ref, mag, f"bucketed product {N}x{K}x{F}, B={B}", nterms=K)


LAYER_CASES = [(300, 70, 6, 64, 4.0, 0), (2708, 1433, 64, 256, 4.0, 0),
               (5000, 300, 33, 128, 6.0, 900), (19717, 500, 64, 128, 4.5, 0),
               (400, 200, 8, 4096, 3.0, 0)]


@pytest.mark.parametrize("N,K,F,B,deg,hub", LAYER_CASES)
def test_layer_forward_bucketed(cuda_device, N, K, F, B, deg, hub):
    case = inputs.layer_case(N, K, F, seed=N + F + B, mean_degree=deg, hub_degree=hub,
                             features_kind="bernoulli" if K == 1433 else "normal")
    d = {k: to_dev(v) for k, v in case.items()}
    ws = torch.empty(B_.bigcn_layer_bucketed_workspace_bytes(N, K, F, B), dtype=torch.uint8,
                     device=cuda_device)
    H = torch.full((N, F), float("nan"), device=cuda_device)
    B_.bigcn_layer_forward_bucketed(B, d["X"], d["s"], d["t"], d["W"], d["rowptr"], d["colidx"],
                                    ws, H)
    torch.cuda.synchronize()
    ref = oracle.layer_forward_bucketed(case["X"], case["W"], case["rowptr"], case["colidx"], B,
                                        case["s"], case["t"])
    nt = K + int(np.diff(case["rowptr"]).max(initial=0)) + 1
    check(H.cpu().numpy(), ref["H"], ref["scale"], f"bucketed layer B={B}", nterms=nt)
    if B >= K:       # one bucket: Bi-GCN's layer
        bi = oracle.layer_forward(case["X"], case["W"], case["rowptr"], case["colidx"],
                                  case["s"], case["t"])
        check(H.cpu().numpy(), bi["H"], ref["scale"], "one bucket = Bi-GCN", nterms=nt)


def test_bucketed_argument_errors(cuda_device):
    X = torch.zeros((10, 100), device=cuda_device)
    bits = torch.zeros((10, 2), dtype=torch.int64, device=cuda_device)
    alpha = torch.full((10, 2), 5.0, device=cuda_device)
    for bad_B in (0, 32, 100, -64):
        with pytest.raises(B_.BigcnError):
            B_.bigcn_pack_rows_bucketed(X, None, None, bad_B, bits, alpha)
    assert B_.bigcn_layer_bucketed_workspace_bytes(10, 100, 4, 96) == 0
    Z = torch.zeros((10, 4), device=cuda_device)
    with pytest.raises(B_.BigcnError):                           # words != ceil(K / 64)
        B_.bigcn_xnor_gemm_bucketed(torch.zeros((10, 3), dtype=torch.int64, device=cuda_device),
                                    alpha, torch.zeros((4, 3), dtype=torch.int64,
                                                       device=cuda_device),
                                    torch.ones((4, 2), device=cuda_device), 100, 64, Z)
    torch.cuda.synchronize()
    assert torch.all(alpha == 5.0)
