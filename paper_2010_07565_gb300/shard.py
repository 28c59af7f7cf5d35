"""The Bi-GCN layer (Eq. 13) on a graph whose rows are partitioned across GPUs.

Steps 1-4 of a layer (centring, packing, the XNOR product) are independent per
row, so each rank computes them for its own contiguous block of rows, with the
packed weights replicated. Step 5 sums, for every row, the products of its
neighbours (Eq. 1): the one exchange of the layer. Each rank needs the rows of
the (degree-scaled) product that its rows reference but other ranks own -- its
halo -- and sends the rows of its own block that other ranks reference.

  partition_rows   contiguous row blocks with about equal work (row length + 1)
  ShardPlan        a rank's block in its own numbering: the block's rows first,
                   then its halo rows; which halo rows come from which rank and
                   which own rows go to which rank
  exchange_rows    the halo exchange, one all-to-all of the requested rows
                   (torch.distributed: NCCL between GPUs, gloo on the CPU)
  exchange_packed_rows
                   the other form of the exchange: the requested rows' packed
                   signs and row scales (8 ceil(K/64) + 4 bytes a row instead
                   of 4 F), from which the receiving rank computes the halo's
                   product itself (the halo rows' degrees come with the plan)
  layer_forward_sharded
                   the layer on one rank: the library's kernels for steps 1-4
                   on its block, the exchange (the smaller of the two forms by
                   default), then bigcn_spmm_prescaled_rows

The degree of every row (dhat = 1 + row length) is known to the rank that
owns the row, which also applies 1/sqrt(dhat_j) to its product rows before
sending them; a row's own degree factor is applied by the aggregation.
"""
from __future__ import annotations

import dataclasses

import numpy as np
import torch


def partition_rows(rowptr: np.ndarray, world: int) -> np.ndarray:
    """Bounds (world + 1) of contiguous row blocks with about equal work:
    each row costs its length + 1 (the self-loop). Block r is rows
    bounds[r] .. bounds[r + 1] - 1."""
    rowptr = np.asarray(rowptr, np.int64)
    n = rowptr.shape[0] - 1
    if world < 1:
        raise ValueError("world must be at least 1")
    cost = np.cumsum(np.diff(rowptr) + 1)                     # work up to and including row i
    total = int(cost[-1]) if n > 0 else 0
    targets = (np.arange(1, world, dtype=np.float64) * total) / world
    cuts = np.searchsorted(cost, targets, side="left") + 1 if n > 0 else np.zeros(world - 1)
    bounds = np.concatenate([[0], np.minimum(cuts, n), [n]]).astype(np.int64)
    return np.maximum.accumulate(bounds)


@dataclasses.dataclass
class ShardPlan:
    """Rank `rank`'s block of rows [lo, hi) of an n-row graph split by `bounds`.

    rowptr, colidx: the block's CSR in its own numbering -- column q < n_own is
    own row lo + q, column n_own + h is halo row halo[h] (global id).
    recv_counts[r]: halo rows that come from rank r (halo is sorted, so they
    are consecutive and in rank order). send_index: the own rows (local
    indices) other ranks need, grouped by destination rank with send_counts.
    halo_rowptr: cumulative degrees of the halo rows (halo_rowptr[h + 1] -
    halo_rowptr[h] = row length of halo[h] in the whole graph), so that the
    degree-scaled product of received packed rows runs as for own rows.
    """
    rank: int
    bounds: np.ndarray
    lo: int
    hi: int
    rowptr: np.ndarray
    colidx: np.ndarray
    halo: np.ndarray
    recv_counts: np.ndarray
    send_index: np.ndarray
    send_counts: np.ndarray
    halo_rowptr: np.ndarray = None

    @property
    def n_own(self) -> int:
        return self.hi - self.lo

    @property
    def n_cols(self) -> int:
        return self.n_own + int(self.halo.shape[0])


def owner_of(bounds: np.ndarray, rows: np.ndarray) -> np.ndarray:
    """The rank whose block holds each of the global row ids."""
    return np.searchsorted(np.asarray(bounds, np.int64), rows, side="right") - 1


def local_plan(rowptr: np.ndarray, colidx: np.ndarray, bounds: np.ndarray, rank: int):
    """The receiving half of a rank's plan, from the whole CSR: its block's CSR
    renumbered and its halo (sorted global ids) with the count per owner.
    Returns (rowptr_local, colidx_local, halo, recv_counts)."""
    rowptr = np.asarray(rowptr, np.int64)
    colidx = np.asarray(colidx, np.int64)
    world = len(bounds) - 1
    lo, hi = int(bounds[rank]), int(bounds[rank + 1])
    cols = colidx[rowptr[lo]:rowptr[hi]]
    rp = (rowptr[lo:hi + 1] - rowptr[lo]).astype(np.int64)
    own = (cols >= lo) & (cols < hi)
    halo = np.unique(cols[~own])
    local = np.empty(cols.shape[0], np.int64)
    local[own] = cols[own] - lo
    local[~own] = (hi - lo) + np.searchsorted(halo, cols[~own])
    recv = np.bincount(owner_of(bounds, halo), minlength=world).astype(np.int64) \
        if halo.size else np.zeros(world, np.int64)
    return rp, local.astype(np.int32), halo, recv


def build_plan(rowptr: np.ndarray, colidx: np.ndarray, bounds: np.ndarray, rank: int,
               group=None) -> ShardPlan:
    """A rank's full plan: its receiving half from the CSR, then the sending
    half from the other ranks' requests (one all-to-all of the requested ids)."""
    import torch.distributed as dist
    world = len(bounds) - 1
    rp, ci, halo, recv = local_plan(rowptr, colidx, bounds, rank)
    lo = int(bounds[rank])
    dev = _collective_device(group)
    req = torch.from_numpy(halo.astype(np.int64)).to(dev)
    recv_t = torch.from_numpy(recv).to(dev)
    send_t = torch.empty_like(recv_t)
    dist.all_to_all_single(send_t, recv_t, group=group)            # how many each asks me for
    send_counts = send_t.cpu().numpy().astype(np.int64)
    asked = torch.empty(int(send_counts.sum()), dtype=torch.int64, device=dev)
    dist.all_to_all_single(asked, req, output_split_sizes=send_counts.tolist(),
                           input_split_sizes=recv.tolist(), group=group)
    send_index = asked.cpu().numpy() - lo
    # The degrees of the rows this rank sends, answered the same way.
    own_deg = np.diff(rp)
    sent_deg = torch.from_numpy(own_deg[send_index].astype(np.int64)).to(dev)
    halo_deg = torch.empty(int(halo.shape[0]), dtype=torch.int64, device=dev)
    dist.all_to_all_single(halo_deg, sent_deg, output_split_sizes=recv.tolist(),
                           input_split_sizes=send_counts.tolist(), group=group)
    halo_rowptr = np.concatenate([[0], np.cumsum(halo_deg.cpu().numpy())]).astype(np.int64)
    return ShardPlan(rank, np.asarray(bounds, np.int64), lo, int(bounds[rank + 1]), rp, ci, halo,
                     recv, send_index.astype(np.int64), send_counts, halo_rowptr)


def _collective_device(group=None):
    import torch.distributed as dist
    backend = dist.get_backend(group)
    if backend == "nccl":
        return torch.device("cuda", torch.cuda.current_device())
    return torch.device("cpu")


def exchange_rows(own: torch.Tensor, plan: ShardPlan, group=None) -> torch.Tensor:
    """The halo exchange: returns the table [own rows; halo rows] (n_cols x F)
    that the block's aggregation reads. `own` is n_own x F on the collective's
    device (CUDA for NCCL, CPU for gloo)."""
    import torch.distributed as dist
    F = own.shape[1]
    send = own[torch.from_numpy(plan.send_index).to(own.device)].contiguous()
    table = torch.empty((plan.n_cols, F), dtype=own.dtype, device=own.device)
    table[:plan.n_own] = own
    halo_rows = table[plan.n_own:]
    dist.all_to_all_single(halo_rows, send, output_split_sizes=plan.recv_counts.tolist(),
                           input_split_sizes=plan.send_counts.tolist(), group=group)
    return table


def exchange_packed_rows(bits: torch.Tensor, alpha: torch.Tensor, plan: ShardPlan, group=None):
    """The packed form of the halo exchange: returns the halo rows' packed
    signs (n_halo x words, int64) and row scales alpha (n_halo), received from
    their owners. ``bits`` / ``alpha`` are this rank's own rows."""
    import torch.distributed as dist
    idx = torch.from_numpy(plan.send_index).to(bits.device)
    n_halo = int(plan.halo.shape[0])
    halo_bits = torch.empty((n_halo, bits.shape[1]), dtype=bits.dtype, device=bits.device)
    halo_alpha = torch.empty(n_halo, dtype=alpha.dtype, device=alpha.device)
    splits = dict(output_split_sizes=plan.recv_counts.tolist(),
                  input_split_sizes=plan.send_counts.tolist(), group=group)
    dist.all_to_all_single(halo_bits, bits[idx].contiguous(), **splits)
    dist.all_to_all_single(halo_alpha, alpha[idx].contiguous(), **splits)
    return halo_bits, halo_alpha


def exchange_bytes_per_row(K: int, F: int, packed: bool) -> int:
    """Bytes a halo row costs in the exchange: the product row (4 F) or the
    packed signs and the row scale (8 ceil(K/64) + 4)."""
    return 8 * ((K + 63) // 64) + 4 if packed else 4 * F


def layer_forward_sharded(X_own, scale, shift, Wt, plan: ShardPlan, group=None,
                          exchange: str = "auto"):
    """One Bi-GCN layer on this rank's block of rows (X_own: n_own x K on this
    rank's GPU): the product of its rows with 1/sqrt(dhat) applied (Eqs. 10-12,
    bigcn_xnor_gemm_degscaled on the block's CSR, whose row lengths are the
    rows' full degrees), the halo exchange (NCCL), and the aggregation of its
    rows (Eq. 13, bigcn_spmm_prescaled_rows). ``exchange``: "rows" sends the
    halo's product rows, "packed" their packed signs and row scales (the
    receiving rank then runs the same degree-scaled product on them, with the
    halo degrees from the plan), "auto" the one with fewer bytes a row.
    Returns H_own (n_own x F)."""
    from . import binding as B
    dev = X_own.device
    K, F = Wt.shape
    if exchange == "auto":
        exchange = "packed" if exchange_bytes_per_row(K, F, True) < \
            exchange_bytes_per_row(K, F, False) else "rows"
    if exchange not in ("rows", "packed"):
        raise ValueError("exchange must be 'rows', 'packed' or 'auto'")
    rowptr = torch.from_numpy(plan.rowptr).to(dev)
    colidx = torch.from_numpy(plan.colidx).to(dev)
    bits, alpha = B.pack_rows(X_own, scale, shift)
    wbits, beta = B.pack_weights(Wt)
    if exchange == "rows":
        Zp = torch.empty((plan.n_own, F), dtype=torch.float32, device=dev)
        B.bigcn_xnor_gemm_degscaled(bits, alpha, wbits, beta, K, rowptr, Zp)
        table = exchange_rows(Zp, plan, group)
    else:
        halo_bits, halo_alpha = exchange_packed_rows(bits, alpha, plan, group)
        table = torch.empty((plan.n_cols, F), dtype=torch.float32, device=dev)
        B.bigcn_xnor_gemm_degscaled(bits, alpha, wbits, beta, K, rowptr, table[:plan.n_own])
        if plan.n_cols > plan.n_own:
            B.bigcn_xnor_gemm_degscaled(halo_bits, halo_alpha, wbits, beta, K,
                                        torch.from_numpy(plan.halo_rowptr).to(dev),
                                        table[plan.n_own:])
    H = torch.empty((plan.n_own, F), dtype=torch.float32, device=dev)
    B.bigcn_spmm_prescaled_rows(rowptr, colidx, table, H)
    return H
