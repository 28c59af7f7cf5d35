"""GPU parity of the ablation products and layers (Sec. 6.3's "binarize weights
only" and "binarize features only" rows) against the oracle, through the C ABI.

Tolerance. Each product is a sum over K of real terms with both signs, done
in fp32 (the real operand split into three bf16 parts) on the GPU and in
double in the oracle. Values are compared with |gpu - oracle| <= 1e-6 + 1e-4 *
max(|oracle|, scale), scale = the sum of the |terms| that make the value (the
scale of any fp32 evaluation order's error); the plain form, scale = |oracle|,
is required wherever 1e-4 |oracle| exceeds sqrt(n) 2^-24 scale, the typical
rounding error of an fp32 sum of n terms (below that the terms have cancelled
to under what fp32 resolves).

Shapes: few 128-row tiles (the k-blocks then split over a cluster of CTAs),
enough tiles for every SM with a ragged last tile, K not a multiple of 64, F
from 1 to past one column tile, padded row strides.
"""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import check_sum as check, padded, to_dev
from paper_2010_07565_gb300 import binding as B
from paper_2010_07565_gb300 import inputs

pytestmark = pytest.mark.gpu


def rng(seed):
    return np.random.Generator(np.random.PCG64(seed))




def features(N, K, seed, kind="normal"):
    g = rng(seed)
    if kind == "sparse":               # {0,1} bag-of-words rows, as the citation graphs'
        return (g.random((N, K)) < 0.02).astype(np.float32)
    return (1.5 * g.standard_normal((N, K)) + 0.2).astype(np.float32)


# (N, K, F): cluster-split k-blocks (few tiles), one tile per SM and more,
# K and F ragged, F over one column tile.
REAL_BINARY_CASES = [
    (1, 1, 1), (100, 63, 6), (300, 130, 16), (1000, 602, 128), (700, 200, 256),
    (500, 100, 300), (2708, 1433, 64), (3327, 3703, 64), (20000, 500, 64), (19717, 500, 3),
]


@pytest.mark.parametrize("N,K,F", REAL_BINARY_CASES)
@pytest.mark.parametrize("centred", [True, False])
def test_real_binary_gemm(cuda_device, N, K, F, centred):
    X = features(N, K, N + K + F, "sparse" if K in (1433, 3703) else "normal")
    s, t = inputs.bn_stats(X) if centred else (None, None)
    Wt = inputs.weights(K, F, seed=K + 3 * F)
    SB, beta = oracle.weight_binarize(Wt)
    beta32 = beta.astype(np.float32)
    Y = oracle.centre(X, s, t)
    ref, mag = oracle.real_binary_product(Y, SB, beta32.astype(np.float64), with_absterm=True)
    Z = torch.full((N, F), float("nan"), device=cuda_device)
    B.bigcn_real_binary_gemm(to_dev(X), to_dev(s), to_dev(t), to_dev(oracle.pack(SB)),
                             to_dev(beta32), Z)
    torch.cuda.synchronize()
    check(Z.cpu().numpy(), ref, mag, f"Y W~ {N}x{K}x{F}", nterms=K)
    assert B.device_timeouts() == 0


@pytest.mark.parametrize("ldx", [157, 158, 160])   # rows 4-, 8- and 16-byte aligned
def test_real_binary_gemm_padded_strides(cuda_device, ldx):
    N, K, F, ldz = 900, 150, 40, 45
    X = features(N, K, 11)
    s, t = inputs.bn_stats(X)
    Wt = inputs.weights(K, F, seed=12)
    SB, beta = oracle.weight_binarize(Wt)
    beta32 = beta.astype(np.float32)
    Xd, _ = padded(to_dev(X), N, K, ldx, fill=float("nan"))     # padding must never be read
    Zd, zbuf = padded(torch.zeros((N, F), device=cuda_device), N, F, ldz, fill=-7.0)
    B.bigcn_real_binary_gemm(Xd, to_dev(s), to_dev(t), to_dev(oracle.pack(SB)), to_dev(beta32),
                             Zd)
    torch.cuda.synchronize()
    ref, mag = oracle.real_binary_product(oracle.centre(X, s, t), SB,
                                          beta32.astype(np.float64), with_absterm=True)
    check(Zd.cpu().numpy(), ref, mag, "Y W~ strided", nterms=K)
    assert torch.all(zbuf[:, F:] == -7.0)


BINARY_REAL_CASES = [
    (1, 1, 1), (100, 63, 6), (300, 130, 16), (1000, 602, 128), (500, 100, 200),
    (2708, 1433, 64), (20000, 500, 64), (19717, 500, 3),
]


@pytest.mark.parametrize("N,K,F", BINARY_REAL_CASES)
def test_binary_real_gemm(cuda_device, N, K, F):
    X = features(N, K, 2 * N + K + F)
    Y = oracle.centre(X, *inputs.bn_stats(X))
    SF = oracle.sign(Y)
    alpha32 = oracle.row_scale(Y).astype(np.float32)
    Wt = inputs.weights(K, F, seed=K + 5 * F)
    ref, mag = oracle.binary_real_product(SF, alpha32.astype(np.float64), Wt, with_absterm=True)
    ws = torch.empty(B.bigcn_binary_real_gemm_workspace_bytes(K, F), dtype=torch.uint8,
                     device=cuda_device)
    Z = torch.full((N, F), float("nan"), device=cuda_device)
    B.bigcn_binary_real_gemm(to_dev(oracle.pack(SF)), to_dev(alpha32), K, to_dev(Wt), ws, Z)
    torch.cuda.synchronize()
    check(Z.cpu().numpy(), ref, mag, f"H~ W {N}x{K}x{F}", nterms=K)
    assert B.device_timeouts() == 0


def test_binary_real_gemm_strided_weights(cuda_device):
    N, K, F, ldw = 640, 77, 30, 37
    g = rng(21)
    SF = np.where(g.random((N, K)) < 0.5, -1, 1).astype(np.int8)
    alpha32 = g.uniform(0.1, 2.0, N).astype(np.float32)
    Wt = inputs.weights(K, F, seed=22)
    Wd, _ = padded(to_dev(Wt), K, F, ldw, fill=float("nan"))
    ws = torch.empty(B.bigcn_binary_real_gemm_workspace_bytes(K, F), dtype=torch.uint8,
                     device=cuda_device)
    Z = torch.full((N, F), float("nan"), device=cuda_device)
    B.bigcn_binary_real_gemm(to_dev(oracle.pack(SF)), to_dev(alpha32), K, Wd, ws, Z)
    torch.cuda.synchronize()
    ref, mag = oracle.binary_real_product(SF, alpha32.astype(np.float64), Wt, with_absterm=True)
    check(Z.cpu().numpy(), ref, mag, "H~ W strided", nterms=K)


LAYER_CASES = [
    # (N, K, F, mean degree, hub degree)
    (200, 70, 6, 4.0, 0),
    (2708, 1433, 64, 4.0, 0),        # Cora-shaped layer 1 (few tiles: cluster split)
    (5000, 300, 33, 6.0, 900),
    (19717, 500, 64, 4.5, 0),        # PubMed-shaped layer 1 (one tile per SM)
    (50, 20, 5, 0.0, 0),             # no edges
]


@pytest.mark.parametrize("N,K,F,deg,hub", LAYER_CASES)
@pytest.mark.parametrize("binarize", ["weights", "features"])
def test_layer_forward_ablation(cuda_device, N, K, F, deg, hub, binarize):
    case = inputs.layer_case(N, K, F, seed=N + F, mean_degree=deg, hub_degree=hub,
                             features_kind="bernoulli" if K == 1433 else "normal")
    d = {k: to_dev(v) for k, v in case.items()}
    ws = torch.empty(B.bigcn_layer_ablation_workspace_bytes(binarize, N, K, F),
                     dtype=torch.uint8, device=cuda_device)
    H = torch.full((N, F), float("nan"), device=cuda_device)
    B.bigcn_layer_forward_ablation(binarize, d["X"], d["s"], d["t"], d["W"], d["rowptr"],
                                   d["colidx"], ws, H)
    torch.cuda.synchronize()
    ref = oracle.layer_forward_ablation(case["X"], case["W"], case["rowptr"], case["colidx"],
                                        binarize, case["s"], case["t"])
    check(H.cpu().numpy(), ref["H"], ref["scale"], f"layer ({binarize} binarized)",
          nterms=K + int(np.diff(case["rowptr"]).max(initial=0)) + 1)
    assert B.device_timeouts() == 0


def test_layer_forward_ablation_both_is_the_bi_gcn_layer(cuda_device):
    case = inputs.layer_case(1500, 300, 40, seed=31)
    d = {k: to_dev(v) for k, v in case.items()}
    N, K, F = 1500, 300, 40
    H = [torch.empty((N, F), device=cuda_device) for _ in range(2)]
    ws = torch.empty(B.bigcn_layer_ablation_workspace_bytes("both", N, K, F), dtype=torch.uint8,
                     device=cuda_device)
    assert ws.numel() == B.bigcn_layer_workspace_bytes(N, K, F)
    B.bigcn_layer_forward_ablation("both", d["X"], d["s"], d["t"], d["W"], d["rowptr"],
                                   d["colidx"], ws, H[0])
    B.bigcn_layer_forward(d["X"], d["s"], d["t"], d["W"], d["rowptr"], d["colidx"], ws, H[1])
    torch.cuda.synchronize()
    assert torch.equal(H[0], H[1])


@pytest.mark.parametrize("binarize", ["weights", "features"])
def test_layer_forward_ablation_is_deterministic(cuda_device, binarize):
    case = inputs.layer_case(2000, 900, 64, seed=41, hub_degree=300)
    d = {k: to_dev(v) for k, v in case.items()}
    ws = torch.empty(B.bigcn_layer_ablation_workspace_bytes(binarize, 2000, 900, 64),
                     dtype=torch.uint8, device=cuda_device)
    out = []
    for _ in range(2):
        H = torch.empty((2000, 64), device=cuda_device)
        B.bigcn_layer_forward_ablation(binarize, d["X"], d["s"], d["t"], d["W"], d["rowptr"],
                                       d["colidx"], ws, H)
        out.append(H)
    torch.cuda.synchronize()
    assert torch.equal(out[0], out[1])


def test_ablation_argument_errors(cuda_device):
    N, K, F = 10, 8, 3
    X = torch.zeros((N, K), device=cuda_device)
    W = torch.zeros((K, F), device=cuda_device)
    rowptr = torch.zeros(N + 1, dtype=torch.int64, device=cuda_device)
    colidx = torch.zeros(0, dtype=torch.int32, device=cuda_device)
    H = torch.full((N, F), 5.0, device=cuda_device)
    assert B.bigcn_layer_ablation_workspace_bytes(7, N, K, F) == 0
    ws = torch.empty(B.bigcn_layer_ablation_workspace_bytes("features", N, K, F),
                     dtype=torch.uint8, device=cuda_device)
    with pytest.raises(B.BigcnError):                              # unknown variant
        B.bigcn_layer_forward_ablation(7, X, None, None, W, rowptr, colidx, ws, H)
    with pytest.raises(B.BigcnError):                              # workspace too small
        B.bigcn_layer_forward_ablation("features", X, None, None, W, rowptr, colidx, ws[:64], H)
    bits = torch.zeros((F, 2), dtype=torch.int64, device=cuda_device)   # words != ceil(K/64)
    with pytest.raises(B.BigcnError):
        B.bigcn_real_binary_gemm(X, None, None, bits, torch.ones(F, device=cuda_device), H)
    with pytest.raises(B.BigcnError):                              # Z overlaps X
        B.bigcn_real_binary_gemm(X, None, None, bits[:, :1], torch.ones(F, device=cuda_device),
                                 X[:, :F])
    torch.cuda.synchronize()
    assert torch.all(H == 5.0)
