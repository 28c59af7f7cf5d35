"""The tensor-core (tcgen05) XNOR product at the sizes that select it: the
step call takes it once there are at least as many 128-row tiles as SMs, and
the layer entry points additionally hand it the weight signs pre-expanded
into FP8 tiles (256-column tiles then run the warp-specialised kernel with
256-row CTAs). Shapes are ragged on every side -- rows past the last full
tile, columns past the last full tile, K not a multiple of the 128-sign
k-block -- and the dots are compared bit for bit with the oracle's on
sampled rows (plus the first and last rows and rows planted at +-K)."""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import assert_close, check_sum, to_dev
from paper_2010_07565_gb300 import binding as B
from paper_2010_07565_gb300 import inputs

pytestmark = pytest.mark.gpu


def tc_rows(cuda_device):
    """The fewest rows that give every SM a 128-row tile."""
    sms = torch.cuda.get_device_properties(cuda_device).multi_processor_count
    return 128 * sms


def sampled(N, n, seed):
    g = np.random.default_rng(seed)
    rows = np.unique(np.concatenate([np.arange(4), np.arange(N - 4, N),
                                     g.choice(N, size=min(n, N), replace=False)]))
    return rows


# (extra rows past the tile count, F, K)
STEP_CASES = [(77, 32, 128), (1, 33, 129), (255, 100, 1000), (128, 257, 2560), (3, 64, 8192)]


@pytest.mark.parametrize("extra,F,K", STEP_CASES)
def test_xnor_gemm_step_on_the_tensor_cores(cuda_device, extra, F, K):
    N = tc_rows(cuda_device) + extra
    g = np.random.default_rng(N + 7 * F + 13 * K)
    SF = np.where(g.random((N, K)) < 0.5, 1, -1).astype(np.int8)
    SB = np.where(g.random((F, K)) < 0.5, 1, -1).astype(np.int8)
    SF[0] = SB[0]            # dot = +K
    SF[1] = -SB[1]           # dot = -K
    SF[N - 1] = SB[F - 1]    # last row, last column: +K
    alpha = g.uniform(0.1, 2.0, N).astype(np.float32)
    beta = g.uniform(0.001, 0.1, F).astype(np.float32)
    Z, dots = B.xnor_gemm(to_dev(oracle.pack(SF)), to_dev(alpha), to_dev(oracle.pack(SB)),
                          to_dev(beta), K, with_dots=True)
    torch.cuda.synchronize()
    assert B.device_timeouts() == 0
    rows = sampled(N, 1024, N + K)
    ref = oracle.binary_dot(SF[rows], SB)
    got = dots.cpu().numpy()[rows]
    assert np.array_equal(got, ref), f"{int((got != ref).sum())} dots differ"
    assert got[0, 0] == K and got[1, 1] == -K and got[-1, F - 1] == K
    assert_close(Z.cpu().numpy()[rows],
                 oracle.zeta(ref, alpha[rows].astype(np.float64), beta.astype(np.float64)), "Z")


# Layers whose weight tiles are pre-expanded: (extra rows, K, F, mean degree, hub)
LAYER_CASES = [
    (77, 1030, 200, 6.0, 0),       # 256-column tile, warp-specialised kernel, ragged K and F
    (200, 4160, 300, 5.0, 900),    # two 256-column tiles (the second 44 wide), a hub row
    (77, 4100, 100, 6.0, 0),       # 128-column tiles with pre-expanded weights
]


@pytest.mark.parametrize("extra,K,F,deg,hub", LAYER_CASES)
def test_layer_forward_with_pre_expanded_weight_tiles(cuda_device, extra, K, F, deg, hub):
    N = tc_rows(cuda_device) + extra
    case = inputs.layer_case(N, K, F, seed=N + K + F, mean_degree=deg, hub_degree=hub)
    rp, ci = case["rowptr"], case["colidx"]
    d = {k: to_dev(v) for k, v in case.items()}
    ws = torch.empty(B.bigcn_layer_workspace_bytes(N, K, F), dtype=torch.uint8,
                     device=cuda_device)
    H = torch.full((N, F), float("nan"), device=cuda_device)
    B.bigcn_layer_forward(d["X"], d["s"], d["t"], d["W"], d["rowptr"], d["colidx"], ws, H)
    torch.cuda.synchronize()
    assert B.device_timeouts() == 0
    rows = sampled(N, 1024, K + F)
    ref = oracle.layer_forward(case["X"], case["W"], rp, ci, case["s"], case["t"], rows=rows)
    nterms = K + int(np.diff(rp)[rows].max()) + 1
    check_sum(H.cpu().numpy()[rows], ref["H"], ref["absterm"],
              f"pre-expanded weight tiles K={K} F={F} H (sampled)", nterms)
