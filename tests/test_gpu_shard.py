"""The sharded layer's device half on one GPU: each rank's block runs through
the library's kernels (packing, the degree-scaled XNOR product of its rows,
and bigcn_spmm_prescaled_rows over its table of own and halo rows). The ranks
are emulated one after the other in this process, the halo rows taken from the
owning block's product on the host (the exchange itself is the gloo-tested
host logic); the blocks put back together must equal the oracle's layer."""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import assert_close, check_sum, to_dev
from paper_2010_07565_gb300 import binding as B
from paper_2010_07565_gb300 import inputs, shard

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("N,K,F,deg,hub,world", [
    (600, 150, 12, 6.0, 250, 2),
    (3000, 602, 41, 30.0, 2000, 3),      # Reddit-like widths, a hub
    (2708, 1433, 64, 4.0, 0, 4),         # Cora-shaped layer 1
])
def test_sharded_layer_matches_oracle(cuda_device, N, K, F, deg, hub, world):
    c = inputs.layer_case(N, K, F, seed=N + world, mean_degree=deg, hub_degree=hub)
    rp, ci = c["rowptr"], c["colidx"]
    bounds = shard.partition_rows(rp, world)
    W = to_dev(c["W"])
    s, t = to_dev(c["s"]), to_dev(c["t"])
    plans, zp = [], []
    for r in range(world):        # every block's degree-scaled product, on the GPU
        lrp, lci, halo, recv = shard.local_plan(rp, ci, bounds, r)
        lo, hi = bounds[r], bounds[r + 1]
        X = to_dev(np.ascontiguousarray(c["X"][lo:hi]))
        bits, alpha = B.pack_rows(X, s, t)
        wbits, beta = B.pack_weights(W)
        Z = torch.empty((hi - lo, F), device=cuda_device)
        B.bigcn_xnor_gemm_degscaled(bits, alpha, wbits, beta, K, to_dev(lrp), Z)
        plans.append((lrp, lci, halo))
        zp.append(Z)
    Zall = torch.cat(zp)                                   # global numbering
    H = []
    for r in range(world):        # each block's aggregation over its table
        lrp, lci, halo = plans[r]
        table = torch.cat([zp[r], Zall[torch.from_numpy(halo).to(cuda_device)]])
        Hr = torch.full((bounds[r + 1] - bounds[r], F), float("nan"), device=cuda_device)
        B.bigcn_spmm_prescaled_rows(to_dev(lrp), to_dev(lci), table, Hr)
        H.append(Hr)
    torch.cuda.synchronize()
    ref = oracle.layer_forward(c["X"], c["W"], rp, ci, c["s"], c["t"])
    check_sum(torch.cat(H), ref["H"], ref["absterm"], f"sharded layer x{world}",
              nterms=K + int(np.diff(rp).max()) + 1)


def test_prescaled_rows_equals_prescaled_on_the_whole_graph(cuda_device):
    c = inputs.layer_case(1000, 64, 20, seed=3, mean_degree=8.0, hub_degree=300)
    d = {k: to_dev(v) for k, v in c.items()}
    Z = torch.randn((1000, 20), device=cuda_device)
    H1 = torch.empty_like(Z)
    H2 = torch.empty_like(Z)
    B.bigcn_spmm_prescaled(d["rowptr"], d["colidx"], Z, H1)
    B.bigcn_spmm_prescaled_rows(d["rowptr"], d["colidx"], Z, H2)
    torch.cuda.synchronize()
    assert torch.equal(H1, H2)


def test_prescaled_rows_bounds_and_errors(cuda_device):
    # two output rows over a four-row table; entries past the table are skipped
    rowptr = torch.tensor([0, 2, 4], dtype=torch.int64, device=cuda_device)
    colidx = torch.tensor([2, 3, 0, 4], dtype=torch.int32, device=cuda_device)
    Z = torch.arange(8, dtype=torch.float32, device=cuda_device).view(4, 2)
    H = torch.empty((2, 2), device=cuda_device)
    B.bigcn_spmm_prescaled_rows(rowptr, colidx, Z, H)
    torch.cuda.synchronize()
    ref = np.array([Z[0].tolist(), Z[1].tolist()]) + np.array([(Z[2] + Z[3]).tolist(),
                                                              Z[0].tolist()])
    assert_close(H, ref / np.sqrt(3.0), "table rows")
    with pytest.raises(B.BigcnError):        # fewer table rows than output rows
        B.bigcn_spmm_prescaled_rows(rowptr, colidx, Z[:1], H)
