"""The sharded layer's device half on one GPU: each rank's block runs through
the library's kernels (packing, the degree-scaled XNOR product of its rows,
and bigcn_spmm_prescaled_rows over its table of own and halo rows). The ranks
are emulated one after the other in this process, the halo rows taken from the
owning blocks (the exchange itself is the gloo-tested host logic): either
their product rows, or their packed signs and row scales, whose product the
receiving rank then computes with the halo rows' degrees. The blocks put back
together must equal the oracle's layer."""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import assert_close, check_sum, to_dev
from paper_2010_07565_gb300 import binding as B
from paper_2010_07565_gb300 import inputs, shard

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("packed", [False, True])
@pytest.mark.parametrize("N,K,F,deg,hub,world", [
    (600, 150, 12, 6.0, 250, 2),
    (3000, 602, 41, 30.0, 2000, 3),      # Reddit-like widths, a hub
    (2708, 1433, 64, 4.0, 0, 4),         # Cora-shaped layer 1
])
def test_sharded_layer_matches_oracle(cuda_device, N, K, F, deg, hub, world, packed):
    c = inputs.layer_case(N, K, F, seed=N + world, mean_degree=deg, hub_degree=hub)
    rp, ci = c["rowptr"], c["colidx"]
    bounds = shard.partition_rows(rp, world)
    W = to_dev(c["W"])
    s, t = to_dev(c["s"]), to_dev(c["t"])
    plans, zp, bp, ap = [], [], [], []
    wbits, beta = B.pack_weights(W)
    for r in range(world):        # every block's degree-scaled product, on the GPU
        lrp, lci, halo, recv = shard.local_plan(rp, ci, bounds, r)
        lo, hi = bounds[r], bounds[r + 1]
        X = to_dev(np.ascontiguousarray(c["X"][lo:hi]))
        bits, alpha = B.pack_rows(X, s, t)
        Z = torch.empty((hi - lo, F), device=cuda_device)
        B.bigcn_xnor_gemm_degscaled(bits, alpha, wbits, beta, K, to_dev(lrp), Z)
        plans.append((lrp, lci, halo))
        zp.append(Z)
        bp.append(bits)
        ap.append(alpha)
    Zall, bits_all, alpha_all = torch.cat(zp), torch.cat(bp), torch.cat(ap)   # global numbering
    H = []
    for r in range(world):        # each block's aggregation over its table
        lrp, lci, halo = plans[r]
        hidx = torch.from_numpy(halo).to(cuda_device)
        if packed:                # the halo's product from its packed rows and degrees
            halo_rowptr = np.concatenate([[0], np.cumsum(np.diff(rp)[halo])]).astype(np.int64)
            Zh = torch.empty((halo.shape[0], F), device=cuda_device)
            if halo.shape[0] > 0:
                B.bigcn_xnor_gemm_degscaled(bits_all[hidx].contiguous(),
                                            alpha_all[hidx].contiguous(), wbits, beta, K,
                                            to_dev(halo_rowptr), Zh)
            table = torch.cat([zp[r], Zh])
        else:
            table = torch.cat([zp[r], Zall[hidx]])
        Hr = torch.full((bounds[r + 1] - bounds[r], F), float("nan"), device=cuda_device)
        B.bigcn_spmm_prescaled_rows(to_dev(lrp), to_dev(lci), table, Hr)
        H.append(Hr)
    torch.cuda.synchronize()
    ref = oracle.layer_forward(c["X"], c["W"], rp, ci, c["s"], c["t"])
    check_sum(torch.cat(H), ref["H"], ref["absterm"],
              f"sharded layer x{world}" + (" (packed exchange)" if packed else ""),
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


@pytest.mark.parametrize("exchange", ["rows", "packed"])
def test_layer_forward_sharded_one_rank(cuda_device, exchange):
    """layer_forward_sharded end to end through NCCL with a single rank (its
    block is the whole graph, the halo empty), in both exchange forms."""
    import socket
    import torch.distributed as dist
    with socket.socket() as sk:
        sk.bind(("127.0.0.1", 0))
        port = sk.getsockname()[1]
    dist.init_process_group("nccl", init_method=f"tcp://127.0.0.1:{port}", rank=0,
                            world_size=1)
    try:
        c = inputs.layer_case(700, 300, 24, seed=21, mean_degree=6.0, hub_degree=200)
        rp, ci = c["rowptr"], c["colidx"]
        plan = shard.build_plan(rp, ci, shard.partition_rows(rp, 1), 0)
        H = shard.layer_forward_sharded(to_dev(c["X"]), to_dev(c["s"]), to_dev(c["t"]),
                                        to_dev(c["W"]), plan, exchange=exchange)
        torch.cuda.synchronize()
    finally:
        dist.destroy_process_group()
    ref = oracle.layer_forward(c["X"], c["W"], rp, ci, c["s"], c["t"])
    check_sum(H, ref["H"], ref["absterm"], f"sharded layer, one NCCL rank ({exchange})",
              nterms=300 + int(np.diff(rp).max()) + 1)
