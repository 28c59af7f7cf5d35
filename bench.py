#!/usr/bin/env python3
"""Benchmark: the 2-layer Bi-GCN forward (Wang et al., CVPR 2021) on GB300.

One step = one pass of the whole hot path over the workload: for each of the
two layers, centre + sign-pack the node rows (Sec. 6.2, Eqs. 7-8), sign-pack
the weight columns (Eqs. 3-4), the XNOR-popcount product (Eqs. 11-12) and the
normalised-adjacency aggregation (Eqs. 1, 13) -- one bigcn_forward_2layer
call (5 kernels for the usual widths), replayed as a CUDA graph with timing
events around it. Per-kernel durations come from a second pass of the same
forward with an event between kernels.

Default workload: C4 (the Reddit-shaped 2-layer configuration: N=232965,
K=602, hidden 128, out 41, 114.6M CSR entries), the largest configuration
that runs as a 2-layer forward on one GPU. Smaller workloads (C1..C3) fit in
L2, so L2 is flushed before every step, outside the timed events: a 256 MiB
buffer is written and its first half read back, which leaves L2 holding clean
lines of that buffer (the inputs come from HBM, and the step does not pay for
writing back the flush's dirty lines).

Prints one JSON line (rank 0): nodes/s of the device-resident forward, the
same through host buffers (e2e), per-kernel times and the dominant kernel's
roofline, the CPU oracle timed on the host as a baseline, and SM clocks
sampled during the timed region. ``--impl reference`` times the CPU oracle
itself on the same workload (the reference arm).

Multi-GPU (torchrun): the layer on one graph has no partition without an
exchange step, so N GPUs run N independent replicas ("replicas only"); value
= nodes processed by all ranks / the slowest rank's time.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

METRIC = "Bi-GCN layer fwd nodes/s; XNOR-GEMM bit-ops/s; SpMM GB/s as % of GB300 peak"
DEFAULT_WORKLOAD = "C4"
L2_FLUSH_BYTES = 256 << 20
L2_BYTES = 129 << 20        # the GB300's L2
TOPS_STYLE_NOTE = ("2 N K F / t in 10^12 per second: each bit-MAC counted as a multiply and "
                   "an add, as dense-GEMM TOPS are; the bit-ops/s figure counts one XNOR + "
                   "count per (i, j, k)")
# 32-bit population counts per clock per SM, as measured on GB300 by
# tests/probes/instruction_rates.cu (profiles/xnor_gemm_instruction_rates.txt:
# 151.8 T bit-ops/s over 152 SMs at 2070 MHz); the ALU ceiling of the POPC products.
POPC_PER_CLK_PER_SM = 15.1
FALLBACK_HBM_GBS = 6800.0


# --------------------------------------------------------------- host logic --
def dist_env():
    return (int(os.environ.get("RANK", 0)), int(os.environ.get("WORLD_SIZE", 1)),
            int(os.environ.get("LOCAL_RANK", 0)))


def aggregate_over_ranks(total_ms: float, units: float, world: int):
    """Max of the per-rank timed totals and the sum of units over ranks
    (replicas): returns (max_ms, total_units)."""
    if world == 1:
        return total_ms, units
    import torch
    import torch.distributed as dist
    dev = torch.device("cuda", torch.cuda.current_device()) if dist.get_backend() == "nccl" \
        else torch.device("cpu")
    t = torch.tensor([total_ms], dtype=torch.float64, device=dev)
    u = torch.tensor([units], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    dist.all_reduce(u, op=dist.ReduceOp.SUM)
    return float(t.item()), float(u.item())


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return p, "measured"
    return {"hbm_gbs": FALLBACK_HBM_GBS, "sm_max_mhz": 2070.0}, "fallback"


def induced_subgraph(rowptr, colidx, lo: int, hi: int):
    """CSR of the subgraph induced by nodes [lo, hi), renumbered from 0."""
    rp = rowptr[lo:hi + 1] - rowptr[lo]
    cols = colidx[rowptr[lo]:rowptr[hi]].astype(np.int64)
    rows = np.repeat(np.arange(hi - lo), np.diff(rp))
    keep = (cols >= lo) & (cols < hi)
    counts = np.bincount(rows[keep], minlength=hi - lo)
    out = np.zeros(hi - lo + 1, np.int64)
    np.cumsum(counts, out=out[1:])
    return out, (cols[keep] - lo).astype(np.int32)


# Random row gathers from an L2-resident buffer (63 MB), plain 16-byte loads,
# every SM busy: bytes/s by row size, measured on GB300 by
# tests/probes/l2_gather.cu (profiles/l2_gather_rates.txt).
L2_GATHER_GBS = {16: 900.0, 64: 8867.0, 128: 20304.0, 256: 21238.0, 512: 21334.0}


def l2_gather_peak(row_bytes):
    """The measured L2 gather ceiling for rows of this size (the entry for the
    smallest measured row size at least this large)."""
    for size in sorted(L2_GATHER_GBS):
        if row_bytes <= size:
            return L2_GATHER_GBS[size], size
    return L2_GATHER_GBS[512], 512


def tensor_core_aggregation(w):
    from paper_2010_07565_gb300 import binding as B
    return B.bigcn_forward_2layer_aggregation(w.K, w.hidden, w.out) == 1


def z_rows(w):
    """Bytes per node of layer 1's and layer 2's factored products as the
    forward keeps them (dot rows + row scale): fp16 dots in rows padded to 16
    on the tensor-core path; else uint16 dots (rows padded to 8) or fp32 for
    layer 1 and fp32 rows padded to 4 for layer 2."""
    K, Fh, Fo = w.K, w.hidden, w.out
    if tensor_core_aggregation(w):
        return 2.0 * ((Fh + 15) // 16 * 16) + 4.0, 2.0 * ((Fo + 15) // 16 * 16) + 4.0
    z1 = 2.0 * ((Fh + 7) // 8 * 8) + 4.0 if K <= 32767 else 4.0 * Fh
    return z1, 4.0 * ((Fo + 3) // 4 * 4)


def kernel_work(w, nnz, name):
    """Algorithmic work of one launch of the named kernel of the 2-layer
    forward: (amount, unit, bound)."""
    N, K, Fh, Fo = w.N, w.K, w.hidden, w.out
    W1, W2 = (K + 63) // 64, (Fh + 63) // 64
    csr = 8.0 * (N + 1) + 4.0 * nnz
    r1, r2 = z_rows(w)
    z1, z2 = N * r1, N * r2
    table = {
        "pack_weights(W1,W2)": (4.0 * K * Fh + 8.0 * Fh * W1 + 4.0 * Fh + 4.0 * Fh * Fo
                                + 8.0 * Fo * W2 + 4.0 * Fo, "bytes", "hbm"),
        "L1.pack_rows": (4.0 * N * K + 8.0 * N * W1 + 4.0 * N + 8.0 * K, "bytes", "hbm"),
        "L1.pack_rows+L1.xnor_gemm": (4.0 * N * K + 8.0 * K + z1 + 8.0 * (N + 1),
                                      "bytes", "hbm", float(N) * K * Fh),
        "L1.xnor_gemm": (float(N) * K * Fh, "bit-ops", "alu"),
        "L1.spmm+L2.pack_rows+L2.xnor_gemm": (csr + z1 + z2, "bytes", "hbm"),
        "L1.spmm": (csr + z1 + 4.0 * N * Fh, "bytes", "hbm"),
        "L2.pack_rows": (4.0 * N * Fh + 8.0 * N * W2 + 4.0 * N, "bytes", "hbm"),
        "L2.xnor_gemm": (float(N) * Fh * Fo, "bit-ops", "alu"),
        "L2.spmm": (csr + z2 + 4.0 * N * Fo, "bytes", "hbm"),
    }
    return table[name][:3]


def workload_bytes(w, nnz):
    """Bytes a 2-layer forward touches: the features, the CSR, both weight
    matrices, both layers' factored products (16-bit dots and a row scale)
    and the logits."""
    pad16 = lambda f: (f + 15) // 16 * 16
    return (4.0 * w.N * w.K + 8.0 * (w.N + 1) + 4.0 * nnz + 4.0 * w.K * w.hidden +
            4.0 * w.hidden * w.out + w.N * (2.0 * pad16(w.hidden) + 4.0) +
            w.N * (2.0 * pad16(w.out) + 4.0) + 4.0 * w.N * w.out)


def kernel_bitops(w, name):
    """XNOR-popcount bit-operations a kernel performs (0 for pure data movement)."""
    N, K, Fh, Fo = w.N, w.K, w.hidden, w.out
    return {"L1.pack_rows+L1.xnor_gemm": float(N) * K * Fh, "L1.xnor_gemm": float(N) * K * Fh,
            "L1.spmm+L2.pack_rows+L2.xnor_gemm": float(N) * Fh * Fo,
            "L2.xnor_gemm": float(N) * Fh * Fo}.get(name, 0.0)


KERNEL_FILES = {"pack_rows": "pack.cu", "pack_weights": "pack.cu", "xnor_gemm": "xnor_gemm_tc.cu",
                "spmm": "spmm.cu",
                "pack_weights(W1,W2)": "pack.cu", "L1.pack_rows": "pack.cu",
                "L1.pack_rows+L1.xnor_gemm": "front.cu",
                "L2.pack_rows": "pack.cu", "L1.xnor_gemm": "xnor_gemm.cu",
                "L2.xnor_gemm": "xnor_gemm.cu", "L1.spmm": "spmm.cu", "L2.spmm": "spmm.cu",
                "L1.spmm+L2.pack_rows+L2.xnor_gemm": "spmm.cu"}


def sweep_tensor_core_aggregation(w):
    """The one-layer entry points keep fp16 dots and aggregate on the tensor
    cores for K <= 2048 and F <= 128 (csrc/layer.cu)."""
    return w.K <= 2048 and w.hidden <= 128


def kernel_file(name, w=None):
    if w is not None and name in ("L1.spmm+L2.pack_rows+L2.xnor_gemm", "L2.spmm") and \
            tensor_core_aggregation(w):
        return "spmm_tc.cu"
    if w is not None and name == "spmm" and w.layers == 1 and sweep_tensor_core_aggregation(w):
        return "spmm_tc.cu"
    return KERNEL_FILES[name]


def source_hash(name, w=None):
    path = os.path.join(ROOT, "paper_2010_07565_gb300", "csrc", kernel_file(name, w))
    with open(path, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()[:16]


def profiled_traffic(name, workload, w=None):
    """DRAM bytes per launch from a committed ncu summary, if it was taken on
    the current source of the kernel (profiles/<kernel>_<workload>.txt lines
    'source_sha256_16: ...' and 'dram_bytes_per_launch: ...')."""
    fname = name.replace("(", "_").replace(")", "").replace(",", "_").replace("+", "_")
    path = os.path.join(ROOT, "profiles", f"{fname}_{workload}.txt")
    if not os.path.exists(path):
        return None
    fields = {}
    with open(path) as f:
        for line in f:
            if ":" in line:
                k, v = line.split(":", 1)
                fields[k.strip()] = v.strip()
    if fields.get("source_sha256_16") != source_hash(name, w):
        return None
    try:
        return float(fields["dram_bytes_per_launch"])
    except (KeyError, ValueError):
        return None


def sources_hash(files):
    """sha-256 (16 hex digits) of the listed kernel source files, in order."""
    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(ROOT, "paper_2010_07565_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def profile_file_traffic(fname, files):
    """DRAM bytes per launch from profiles/<fname> if its 'source_sha256_16'
    is the hash of the listed sources as they are now; else None."""
    path = os.path.join(ROOT, "profiles", fname)
    if not os.path.exists(path):
        return None
    fields = {}
    with open(path) as f:
        for line in f:
            if ":" in line:
                k, v = line.split(":", 1)
                fields[k.strip()] = v.strip()
    if fields.get("source_sha256_16", "").split(" ")[0] != sources_hash(files):
        return None
    try:
        return float(fields["dram_bytes_per_launch"].split(" ")[0])
    except (KeyError, ValueError):
        return None


INDUCTIVE_SOURCES = {
    "gcn": ["inductive.cu", "pack.cu", "xnor_gemm.cu", "xnor_gemm_tc.cu", "layer.cu", "spmm_tc.cu"],
    "mean": ["inductive.cu", "pack.cu", "xnor_gemm.cu", "xnor_gemm_tc.cu", "spmm.cu"],
    "sage": ["inductive.cu", "pack.cu", "xnor_gemm.cu", "xnor_gemm_tc.cu", "spmm.cu"]}
BACKWARD_SOURCES = ["backward.cu", "pack.cu", "spmm.cu", "ablation.cu"]
WEIGHTED_SOURCES = ["weighted.cu", "pack.cu", "xnor_gemm.cu", "xnor_gemm_tc.cu", "spmm.cu"]


class ClockSampler:
    """nvidia-smi clock / throttle samples every ``interval_ms`` while running
    (the bench opens it before the warm-up steps, so that short timed regions
    still see samples under load)."""
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int, interval_ms: int = 100):
        self.gpu = gpu_index
        self.interval = interval_ms
        self.proc = None
        self.out = None

    def __enter__(self):
        try:
            self.out = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.QUERY}",
                 "--format=csv,noheader,nounits", "-lms", str(self.interval)],
                stdout=self.out, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        if self.proc is None or self.out is None:
            return None
        self.out.seek(0)
        rows = [r.split(",") for r in self.out.read().strip().splitlines() if r.count(",") >= 8]
        os.unlink(self.out.name)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].strip().replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[5:9]) if "Active" in v
                          and "Not" not in v})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": float(rows[0][2]) if rows[0][2].strip().replace(".", "").isdigit()
                else None,
                "reasons": reasons, "samples": len(rows)}


# ---------------------------------------------------------------- workload --
WORKLOAD_ARRAYS = ("X", "s", "t", "W1", "W2", "rowptr", "colidx")


def build_workload(name):
    """The seeded workload ``name``. With BIGCN_BENCH_CACHE set to a
    directory, the arrays are also saved there (and loaded on later runs)
    under a key made of the name and the sha-256 of the generator's source,
    so that a series of runs on one machine draws the Reddit-shaped graph
    once; the arrays are the same either way."""
    from paper_2010_07565_gb300 import inputs
    w = inputs.get_workload(name)
    cache = os.environ.get("BIGCN_BENCH_CACHE")
    path = None
    if cache:
        with open(inputs.__file__, "rb") as f:
            key = hashlib.sha256(f.read()).hexdigest()[:16]
        path = os.path.join(cache, f"{name}_{key}.npz")
        if os.path.exists(path):
            with np.load(path) as z:
                return w, {k: z[k] for k in WORKLOAD_ARRAYS}
    X = inputs.features(w)
    s, t = inputs.bn_stats(X)
    W1, W2 = inputs.layer_weights(w)
    rowptr, colidx = inputs.graph(w)
    data = dict(X=X, s=s, t=t, W1=W1, W2=W2, rowptr=rowptr, colidx=colidx)
    if path is not None:
        os.makedirs(cache, exist_ok=True)
        tmp = f"{path}.{os.getpid()}.npz"
        np.savez(tmp, **data)
        os.replace(tmp, path)
    return w, data


def oracle_block_nodes(w, data, budget_s):
    """Nodes of a block (the first n nodes, their induced subgraph) whose CPU
    oracle 2-layer forward takes at most about ``budget_s``: the block is
    doubled from 256 nodes while four times the last measured time still fits
    (an induced subgraph's edges grow with the square of its nodes, so a
    per-node rate from a small block would overshoot on dense graphs)."""
    import oracle
    n = min(w.N, 256)
    while True:
        rp, ci = induced_subgraph(data["rowptr"], data["colidx"], 0, n)
        t0 = time.perf_counter()
        oracle.forward_2layer(np.ascontiguousarray(data["X"][:n]), data["s"], data["t"],
                              data["W1"], data["W2"], rp, ci)
        t = time.perf_counter() - t0
        if n >= w.N or 4.0 * t > budget_s:
            return n
        n = min(w.N, 2 * n)


def time_oracle(w, data, budget_s, rows=None):
    """Run the CPU oracle's 2-layer forward on the subgraph induced by the
    first ``rows`` nodes (all if None) repeatedly for about ``budget_s``;
    returns (nodes/s, sample description)."""
    import oracle
    n = w.N if rows is None else int(min(rows, w.N))
    rp, ci = (data["rowptr"], data["colidx"]) if n == w.N else \
        induced_subgraph(data["rowptr"], data["colidx"], 0, n)
    X = np.ascontiguousarray(data["X"][:n])
    reps, t0 = 0, time.perf_counter()
    while True:
        oracle.forward_2layer(X, data["s"], data["t"], data["W1"], data["W2"], rp, ci)
        reps += 1
        el = time.perf_counter() - t0
        if el >= budget_s:
            break
    what = "full" if n == w.N else f"the subgraph induced by nodes [0, {n}) of"
    return n * reps / el, f"{reps} x the oracle's 2-layer forward on {what} {w.name} ({el:.1f} s)"


# ------------------------------------------------------------ reference arm --
def run_reference(args, rank, world):
    """The CPU oracle as the reference arm: each step is one oracle forward
    on a node block of the workload (its induced subgraph), sized so that
    warm-up plus steps take about two and a half minutes."""
    if rank != 0:
        return 0
    import oracle
    w, data = build_workload(args.workload)
    # the largest block (by doubling) whose forward fits a step's share of
    # about two and a half minutes
    n = oracle_block_nodes(w, data, 150.0 / max(args.steps + args.warmup, 1))
    times = []
    for step in range(args.warmup + args.steps):
        lo = (step * n) % max(w.N - n + 1, 1)
        rp, ci = induced_subgraph(data["rowptr"], data["colidx"], lo, lo + n)
        X = np.ascontiguousarray(data["X"][lo:lo + n])
        t0 = time.perf_counter()
        oracle.forward_2layer(X, data["s"], data["t"], data["W1"], data["W2"], rp, ci)
        if step >= args.warmup:
            times.append(time.perf_counter() - t0)
    total = sum(times)
    value = n * len(times) / total
    sample = (f"each step: the oracle's 2-layer forward on the subgraph induced by {n} "
              f"consecutive nodes of {w.name}")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "nodes/s",
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * total / len(times), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32+b1", "data": "synthetic",
            "config": {"workload": w.description, "name": w.name, "nodes_per_step": n},
            "cpu_baseline": {"value": value, "unit": "nodes/s", "cores": 1, "kind": "oracle",
                             "sample": sample, "host_cores": os.cpu_count()},
            "e2e": {"value": value, "unit": "nodes/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# ----------------------------------------------------------------- our arm --
def run_gpu(args, rank, world, local_rank):
    import torch
    import torch.distributed as dist

    from paper_2010_07565_gb300 import cost_model
    from paper_2010_07565_gb300.runner import GCN2Forward

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    w, data = build_workload(args.workload)
    nnz = int(data["colidx"].shape[0])
    host = {k: torch.from_numpy(np.ascontiguousarray(v)).pin_memory() for k, v in data.items()}

    # The timed forward: one CUDA graph of the whole 2-layer forward, with
    # timing events only around it (event nodes inside a graph cost ~5 us each).
    model = GCN2Forward(w.N, w.K, w.hidden, w.out, nnz, dev)
    model.load(non_blocking=False, **host)
    model.capture()
    # The per-kernel pass: the same forward with an event between kernels.
    names = model.kernel_names
    probe = GCN2Forward(w.N, w.K, w.hidden, w.out, nnz, dev)
    probe.load(non_blocking=False, **host)
    kev = [torch.cuda.Event(enable_timing=True, external=True) for _ in range(len(names) + 1)]
    probe.capture(kev)
    torch.cuda.synchronize()

    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    flush_half = flush[: flush.numel() // 2]

    def flush_l2():
        flush.zero_()
        flush_half.sum()

    ea, eb = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    step_ms = []
    # Clocks are sampled from the warm-up on: a short timed region alone may
    # see no sample.
    with ClockSampler(local_rank) as clocks:
        for _ in range(args.warmup):
            flush_l2()
            model.replay()
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        for _ in range(args.steps):
            flush_l2()
            ea.record()
            model.replay()
            eb.record()
            eb.synchronize()
            step_ms.append(ea.elapsed_time(eb))
        torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    total_ms = float(sum(step_ms))
    max_ms, units = aggregate_over_ranks(total_ms, float(w.N) * args.steps, world)
    value = units / (max_ms * 1e-3)

    # Warm L2: workloads whose inputs and intermediates fit L2 also timed with
    # no flush between steps (a reported figure beside the flushed one).
    warm = None
    if workload_bytes(w, nnz) < L2_BYTES:
        warm_ms = []
        for _ in range(args.steps):
            ea.record()
            model.replay()
            eb.record()
            eb.synchronize()
            warm_ms.append(ea.elapsed_time(eb))
        wmax, wunits = aggregate_over_ranks(float(sum(warm_ms)), float(w.N) * args.steps, world)
        warm = {"value": wunits / (wmax * 1e-3), "unit": "nodes/s",
                "ms_per_step": wmax / args.steps,
                "note": "the same graph replayed with no L2 flush between steps: the "
                        "workload's bytes fit the 129 MB L2"}

    # Per-kernel durations (events between kernels, L2 flushed before each pass).
    per_kernel = [[] for _ in names]
    for i in range(min(args.steps, 300) + 3):
        flush_l2()
        probe.replay()
        kev[-1].synchronize()
        if i >= 3:
            for k in range(len(names)):
                per_kernel[k].append(kev[k].elapsed_time(kev[k + 1]))

    # The chain's launch and dependency latency: the same CUDA-graph forward
    # (same widths) on a one-node graph without edges.
    floor = GCN2Forward(1, w.K, w.hidden, w.out, 0, dev)
    floor.load(non_blocking=False, X=host["X"][:1], s=host["s"], t=host["t"], W1=host["W1"],
               W2=host["W2"], rowptr=torch.zeros(2, dtype=torch.int64))
    floor.capture()
    for _ in range(20):
        floor.replay()
    torch.cuda.synchronize()
    floor_ms = []
    for _ in range(200):
        ea.record()
        floor.replay()
        eb.record()
        eb.synchronize()
        floor_ms.append(ea.elapsed_time(eb))

    # End to end through host buffers: pinned inputs -> device, forward, logits -> host.
    logits_host = torch.empty((w.N, w.out), dtype=torch.float32).pin_memory()
    h2d = sum(int(v.numel() * v.element_size()) for v in host.values())
    d2h = int(logits_host.numel() * logits_host.element_size())
    e2e_steps = max(3, min(args.steps, 200))
    e2e_ms = []
    for i in range(e2e_steps + 2):
        ea.record()
        model.load(non_blocking=True, **host)
        model.replay()
        logits_host.copy_(model.logits, non_blocking=True)
        eb.record()
        eb.synchronize()
        if i >= 2:
            e2e_ms.append(ea.elapsed_time(eb))
    e2e_max, e2e_units = aggregate_over_ranks(float(sum(e2e_ms)), float(w.N) * len(e2e_ms), world)

    if rank != 0:
        return 0

    peaks, peak_kind = load_peaks()
    hbm = float(peaks.get("hbm_gbs", FALLBACK_HBM_GBS))
    props = torch.cuda.get_device_properties(dev)
    sm_max = float(peaks.get("sm_max_mhz", 2070.0))
    popc_peak = props.multi_processor_count * POPC_PER_CLK_PER_SM * 32 * sm_max * 1e6
    kernels = []
    for k, name in enumerate(names):
        work, unit, bound = kernel_work(w, nnz, name)
        kernels.append(dict(name=name, mean_us=1e3 * statistics.fmean(per_kernel[k]), work=work,
                            unit=unit, bound=bound))
    for r in kernels:   # a kernel doing both is bound by the larger of its two ideal times
        ops = kernel_bitops(w, r["name"])
        if r["bound"] == "hbm" and ops / popc_peak > r["work"] / (hbm * 1e9):
            r.update(work=ops, unit="bit-ops", bound="alu")
    dom = max(kernels, key=lambda r: r["mean_us"])
    rate = dom["work"] / (dom["mean_us"] * 1e-6)
    if dom["bound"] == "hbm":
        achieved, peak, unit = rate / 1e9, hbm, "GB/s"
    else:
        achieved, peak, unit = rate / 1e12, popc_peak / 1e12, "T bit-ops/s"
    traffic = profiled_traffic(dom["name"], w.name, w)
    by_name = {r["name"]: r for r in kernels}
    gemm1 = by_name.get("L1.xnor_gemm") or by_name["L1.pack_rows+L1.xnor_gemm"]
    agg1 = by_name.get("L1.spmm+L2.pack_rows+L2.xnor_gemm") or by_name["L1.spmm"]
    spmm_gbs = kernel_work(w, nnz, agg1["name"])[0] / (agg1["mean_us"] * 1e-6) / 1e9
    # Bytes an aggregation gathers: one row of the factored product (with its
    # row scale) and one column index per CSR entry and self-loop -- what a
    # graph without reuse moves, served from L2 where rows repeat -- against
    # the measured L2 gather ceiling for rows of that size.
    r1, r2 = z_rows(w)
    gathers = {}
    for label, r, rec in (("layer1", r1, agg1), ("layer2", r2, by_name["L2.spmm"])):
        gb = (float(nnz + w.N) * (r + 4.0) + 8.0 * (w.N + 1)) / (rec["mean_us"] * 1e-6) / 1e9
        peak_g, size = l2_gather_peak(r)
        gathers[label] = {"kernel": rec["name"], "gathered_gbs": gb, "row_bytes": r,
                          "l2_gather_peak_gbs": peak_g, "frac": gb / peak_g,
                          "peak_source": f"measured random {size}-byte row gathers from a "
                                         "63 MB L2-resident buffer (profiles/l2_gather_rates.txt)"}
    gather_gbs = gathers["layer1"]["gathered_gbs"]

    cpu_baseline = None
    if world == 1 and not args.no_cpu_baseline:
        rows = oracle_block_nodes(w, data, args.cpu_seconds)
        v, sample = time_oracle(w, data, budget_s=args.cpu_seconds, rows=rows)
        cpu_baseline = {"value": v, "unit": "nodes/s", "cores": 1, "kind": "oracle",
                        "sample": sample, "host_cores": os.cpu_count(),
                        "note": "the oracle is single-threaded: 1 of the host's cores"}

    dims = [w.K, w.hidden, w.out]
    line = {
        "metric": METRIC, "value": value, "unit": "nodes/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": max_ms / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f32+b1", "data": "synthetic",
        "config": {"workload": w.description, "name": w.name, "N": w.N, "K": w.K,
                   "hidden": w.hidden, "out": w.out, "nnz": nnz,
                   "l2": "flushed before every step outside the timed events (256 MiB written, "
                         "its first half read back)",
                   "launch": f"one CUDA graph per step: bigcn_forward_2layer, {len(names)} kernels",
                   "parallelism": "replicas" if world > 1 else "single GPU"},
        "components": {
            "xnor_gemm_bitops_per_s": kernel_bitops(w, gemm1["name"]) / (gemm1["mean_us"] * 1e-6),
            "xnor_gemm_tops_style": 2.0 * kernel_bitops(w, gemm1["name"]) /
                                    (gemm1["mean_us"] * 1e-6) / 1e12,
            "xnor_gemm_tops_style_note": TOPS_STYLE_NOTE,
            "warm_l2": warm,
            "spmm_gbs": spmm_gbs, "spmm_pct_of_hbm_peak": 100.0 * spmm_gbs / hbm,
            "l1_aggregation_gather_gbs": gather_gbs,
            "l1_aggregation_gather_frac_of_hbm": gather_gbs / hbm,
            "aggregation_gathers": gathers,
            "l1_aggregation_gather_note": "every neighbour row (and row scale) of the factored "
                                          "product an aggregation reads, per second; rows that "
                                          "repeat are served from L2, so this can exceed HBM",
            "per_kernel_us": {r["name"]: round(r["mean_us"], 3) for r in kernels},
            "per_kernel_note": "from a second pass of the same graph with an event node "
                               "between kernels (each node adds a few us)",
            "latency_floor": {"us": 1e3 * statistics.median(floor_ms),
                              "kernels": len(floor.kernel_names),
                              "note": "median step of the same CUDA-graph forward on a one-node "
                                      "graph without edges (same widths): the launch and "
                                      "dependency latency of the kernel chain"}},
        "roofline": {"kernel": dom["name"], "bound": dom["bound"],
                     "achieved": achieved, "peak": peak, "unit": unit, "frac": achieved / peak,
                     "traffic": traffic,
                     "l2_gather": next((g for g in gathers.values() if g["kernel"] == dom["name"]),
                                       None),
                     "peak_source": (f"{peak_kind} MEASURED_PEAKS.json hbm_gbs"
                                     if dom["bound"] == "hbm" else
                                     f"{POPC_PER_CLK_PER_SM} POPC/clk/SM x {props.multi_processor_count}"
                                     f" SMs x 32 bits x {sm_max:.0f} MHz")},
        "cpu_baseline": cpu_baseline,
        "e2e": {"value": e2e_units / (e2e_max * 1e-3), "unit": "nodes/s",
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
        "gpu_launches": len(names) * args.steps,
        "clocks": clocks.summary(),
        "paper_context": {
            "cycle_ops_gcn": cost_model.cycle_ops(w.N, nnz // 2, dims, False),
            "cycle_ops_bigcn": cost_model.cycle_ops(w.N, nnz // 2, dims, True),
            "note": "Sec. 5.3's analytic cycle-operation counts for this shape; the paper "
                    "reports no measured timings"},
    }
    print(json.dumps(line), flush=True)
    return 0


SWEEP_KERNELS = ("pack_rows", "pack_weights", "xnor_gemm", "spmm")


def run_sweep(args, rank, world, local_rank):
    """One Bi-GCN layer on a C5 sweep point (2^20 nodes, K, F): one
    bigcn_layer_forward_timed call per step, with an event before each of the
    layer's four kernels (pack rows, pack weights, XNOR product, aggregation)
    and after the last. The features (up to 34 GB) are drawn on the device by
    torch's seeded generator; the other inputs come from the usual seeds.
    The inputs are larger than L2, so no flush is needed between steps."""
    import torch

    from paper_2010_07565_gb300 import binding as B
    from paper_2010_07565_gb300 import inputs

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    w = inputs.get_workload(args.workload)
    if args.sweep_nodes:    # a smaller case of the same sweep point (profiler captures)
        import dataclasses
        w = dataclasses.replace(w, N=args.sweep_nodes, undirected_edges=8 * args.sweep_nodes,
                                description=w.description.replace("N=2^20",
                                                                  f"N={args.sweep_nodes}"))
    N, K, F = w.N, w.K, w.hidden
    gen = torch.Generator(device=dev)
    gen.manual_seed(1000 + w.index)
    X = torch.randn((N, K), device=dev, generator=gen)
    Wt = torch.from_numpy(inputs.weights(K, F, 3000 + w.index)).to(dev)
    rp, ci = inputs.graph(w)
    rowptr, colidx = torch.from_numpy(rp).to(dev), torch.from_numpy(ci).to(dev)
    nnz = int(ci.shape[0])
    ws = torch.empty(B.bigcn_layer_workspace_bytes(N, K, F), dtype=torch.uint8, device=dev)
    H = torch.empty((N, F), device=dev)
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(5)]
    for e in ev:            # torch creates the CUDA event at its first record
        e.record()

    def step():
        B.bigcn_layer_forward_timed(X, None, None, Wt, rowptr, colidx, ws, H, ev)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    per_kernel = [[] for _ in SWEEP_KERNELS]
    step_ms = []
    with ClockSampler(local_rank) as clocks:
        for _ in range(args.steps):
            step()
            ev[4].synchronize()
            for k in range(4):
                per_kernel[k].append(ev[k].elapsed_time(ev[k + 1]))
            step_ms.append(ev[0].elapsed_time(ev[4]))
    total_ms = float(sum(step_ms))
    max_ms, units = aggregate_over_ranks(total_ms, float(N) * args.steps, world)
    if rank != 0:
        return 0
    peaks, peak_kind = load_peaks()
    hbm = float(peaks.get("hbm_gbs", FALLBACK_HBM_GBS))
    mean_us = [1e3 * statistics.fmean(t) for t in per_kernel]
    words = (K + 63) // 64
    # The layer keeps Z factored when K <= 32767: fp16 dots in rows padded to
    # 16 (K <= 2048, F <= 128) or uint16 dots in rows padded to 8, plus a row scale.
    if sweep_tensor_core_aggregation(w):
        z_bytes = 2.0 * N * ((F + 15) // 16 * 16) + 4.0 * N
    elif K <= 32767:
        z_bytes = 2.0 * N * ((F + 7) // 8 * 8) + 4.0 * N
    else:
        z_bytes = 4.0 * N * F
    work = {"pack_rows": (4.0 * N * K + 8.0 * N * words + 4.0 * N, "bytes", "hbm"),
            "pack_weights": (4.0 * K * F + 8.0 * F * words + 4.0 * F, "bytes", "hbm"),
            "xnor_gemm": (float(N) * K * F, "bit-ops", "tensor"),
            "spmm": (8.0 * (N + 1) + 4.0 * nnz + z_bytes + 4.0 * N * F, "bytes", "hbm")}
    k_dom = max(range(4), key=lambda k: mean_us[k])
    name = SWEEP_KERNELS[k_dom]
    amount, unit, bound = work[name]
    rate = amount / (mean_us[k_dom] * 1e-6)
    if bound == "hbm":
        achieved, peak, runit = rate / 1e9, hbm, "GB/s"
        src = f"{peak_kind} MEASURED_PEAKS.json hbm_gbs"
    else:
        # FP8 dense tensor peak: the measured bf16 burst figure x 2 (fp8 = 2 x bf16 nominal)
        achieved, peak, runit = 2.0 * rate / 1e12, 2.0 * float(peaks.get("bf16_tflops", 1900.0)), \
            "TFLOP/s (fp8, 2 flops per +-1 MAC)"
        src = f"{peak_kind} MEASURED_PEAKS.json bf16_tflops x 2 (fp8/bf16 nominal ratio)"
    line = {
        "metric": METRIC, "value": units / (max_ms * 1e-3), "unit": "nodes/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": max_ms / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32+b1",
        "data": "synthetic",
        "config": {"workload": w.description, "name": w.name, "N": N, "K": K, "F": F, "nnz": nnz,
                   "l2": "inputs larger than L2 (no flush)",
                   "launch": "bigcn_layer_forward_timed: pack rows, pack weights, XNOR "
                             "product, aggregation (4 kernels, an event between each)"},
        "components": {
            "per_kernel_us": {n: round(t, 3) for n, t in zip(SWEEP_KERNELS, mean_us)},
            "pack_rows_gbs": work["pack_rows"][0] / (mean_us[0] * 1e-6) / 1e9,
            "xnor_gemm_bitops_per_s": work["xnor_gemm"][0] / (mean_us[2] * 1e-6),
            "xnor_gemm_tops_style": 2.0 * work["xnor_gemm"][0] / (mean_us[2] * 1e-6) / 1e12,
            "xnor_gemm_tops_style_note": TOPS_STYLE_NOTE,
            "spmm_gbs": work["spmm"][0] / (mean_us[3] * 1e-6) / 1e9},
        "roofline": {"kernel": name, "bound": bound, "achieved": achieved, "peak": peak,
                     "unit": runit, "frac": achieved / peak,
                     "traffic": profiled_traffic(name, w.name, w), "peak_source": src},
        "cpu_baseline": None, "e2e": None,
        "note": "sweep point: one layer, kernel-level timing; no host-buffer run (the features "
                "alone are up to 34 GB)",
        "gpu_launches": 4 * args.steps, "clocks": clocks.summary(),
    }
    print(json.dumps(line), flush=True)
    return 0


def run_backward(args, rank, world, local_rank):
    """Back-propagation of layer 1 of a 2-layer workload (C1..C4): one
    bigcn_layer_backward call per step (Algorithm 1 with Eqs. bp-H and bp-W:
    pack rows and weights, A~ dH, dL/dW~, dL/dH~ clipped, dL/dW), from a
    seeded upstream gradient dH = dL/dH1 (N x hidden, N(0, 1)); inputs resident
    on the device, L2 flushed before every step outside the timed events."""
    import torch

    from paper_2010_07565_gb300 import binding as B

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    w, data = build_workload(args.workload)
    N, K, F = w.N, w.K, w.hidden
    d = {k: torch.from_numpy(np.ascontiguousarray(v)).to(dev)
         for k, v in data.items() if k in ("X", "s", "t", "W1", "rowptr", "colidx")}
    gen = torch.Generator(device=dev)
    gen.manual_seed(4000 + w.index)
    dH = torch.randn((N, F), device=dev, generator=gen)
    ws = torch.empty(B.bigcn_layer_backward_workspace_bytes(N, K, F), dtype=torch.uint8,
                     device=dev)
    dW = torch.empty((K, F), device=dev)
    dX = torch.empty((N, K), device=dev)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    flush_half = flush[: flush.numel() // 2]

    def step():
        B.bigcn_layer_backward(d["X"], d["s"], d["t"], d["W1"], d["rowptr"], d["colidx"], dH,
                               ws, dW, dX=dX)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    times = []
    with ClockSampler(local_rank) as clocks:
        for _ in range(args.steps):
            flush.zero_()
            flush_half.sum()
            e0.record()
            step()
            e1.record()
            e1.synchronize()
            times.append(e0.elapsed_time(e1))
    total_ms = float(sum(times))
    max_ms, units = aggregate_over_ranks(total_ms, float(N) * args.steps, world)
    if rank != 0:
        return 0
    peaks, peak_kind = load_peaks()
    mean_ms = max_ms / args.steps
    # The two +-1 x fp32 products (dL/dW~ and dL/dH~, N K F multiply-adds each)
    # run on the tensor cores, fp32-accurate through three bf16 parts: their
    # ceiling is the measured bf16 peak / 3. The rate is taken over the whole
    # step (pack, aggregation, products, sums), so it is a lower bound.
    flops = 2.0 * 2.0 * N * K * F
    tc_peak = float(peaks.get("bf16_tflops", 1900.0)) / 3.0
    achieved = flops / (mean_ms * 1e-3) / 1e12
    line = {
        "metric": "Bi-GCN layer backward nodes/s (Algorithm 1, Eqs. bp-H, bp-W)",
        "value": units / (max_ms * 1e-3), "unit": "nodes/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": mean_ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32+b1",
        "data": "synthetic",
        "config": {"workload": w.description + " -- layer 1 backward", "name": w.name, "N": N,
                   "K": K, "F": F, "nnz": int(data["colidx"].shape[0]),
                   "l2": "flushed before every step outside the timed events",
                   "launch": "bigcn_layer_backward (9 kernels)"},
        "roofline": {"kernel": "whole backward step (the two products' flops over the step's "
                               "time)", "bound": "tensor", "achieved": achieved,
                     "peak": tc_peak,
                     "unit": "TFLOP/s (2 N K F per product; fp32-accurate = 3 bf16 MMAs)",
                     "frac": achieved / tc_peak,
                     "traffic": profile_file_traffic(f"backward_step_{w.name}.txt",
                                                     BACKWARD_SOURCES),
                     "traffic_note": "DRAM bytes of one whole call (its 9 kernels)",
                     "peak_source": f"{peak_kind} MEASURED_PEAKS.json bf16_tflops / 3"},
        "cpu_baseline": None, "e2e": None, "gpu_launches": 9 * args.steps,
        "clocks": clocks.summary(),
    }
    print(json.dumps(line), flush=True)
    return 0


def run_ablation(args, rank, world, local_rank):
    """Layer 1 of a workload with one operand of Eq. 11 kept real (Sec. 6.3's
    ablation rows): ``--ablation weights`` binarizes only the weights (zeta =
    Y W~, the centred features real), ``--ablation features`` only the
    features (zeta = H~ W). Each step is one bigcn_layer_forward_ablation
    call (pack, product with the degree scale, aggregation); the product is
    also timed alone through its own entry point. C1..C4 use the workload's
    seeded inputs with L2 flushed before every step (outside the events); a
    C5 point draws its features on the device and needs no flush."""
    import torch

    from paper_2010_07565_gb300 import binding as B
    from paper_2010_07565_gb300 import inputs

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    mode = args.ablation
    w = inputs.get_workload(args.workload)
    N, K, F = w.N, w.K, w.hidden
    if w.name.startswith("C5_"):
        gen = torch.Generator(device=dev)
        gen.manual_seed(1000 + w.index)
        X = torch.randn((N, K), device=dev, generator=gen)
        s = t = None
        Wt = torch.from_numpy(inputs.weights(K, F, 3000 + w.index)).to(dev)
        rp, ci = inputs.graph(w)
        flush_needed = False
    else:
        w, data = build_workload(args.workload)
        X = torch.from_numpy(data["X"]).to(dev)
        s, t = torch.from_numpy(data["s"]).to(dev), torch.from_numpy(data["t"]).to(dev)
        Wt = torch.from_numpy(data["W1"]).to(dev)
        rp, ci = data["rowptr"], data["colidx"]
        flush_needed = True
    rowptr, colidx = torch.from_numpy(rp).to(dev), torch.from_numpy(ci).to(dev)
    nnz = int(ci.shape[0])
    words = (K + 63) // 64
    ws = torch.empty(B.bigcn_layer_ablation_workspace_bytes(mode, N, K, F), dtype=torch.uint8,
                     device=dev)
    H = torch.empty((N, F), device=dev)
    Z = torch.empty((N, F), device=dev)
    # Packed operand of the product-alone timing, made once by the library.
    if mode == "weights":
        bits = torch.empty((F, words), dtype=torch.int64, device=dev)
        scl = torch.empty(F, device=dev)
        B.bigcn_pack_weights(Wt, bits, scl)

        def product():
            B.bigcn_real_binary_gemm(X, s, t, bits, scl, Z)
        pbytes = 4.0 * N * K + 8.0 * F * words + 4.0 * F + 8.0 * K + 4.0 * N * F
    else:
        bits = torch.empty((N, words), dtype=torch.int64, device=dev)
        scl = torch.empty(N, device=dev)
        B.bigcn_pack_rows(X, s, t, bits, scl)
        pws = torch.empty(B.bigcn_binary_real_gemm_workspace_bytes(K, F), dtype=torch.uint8,
                          device=dev)

        def product():
            B.bigcn_binary_real_gemm(bits, scl, K, Wt, pws, Z)
        pbytes = 8.0 * N * words + 4.0 * N + 4.0 * K * F + 4.0 * N * F

    def layer():
        B.bigcn_layer_forward_ablation(mode, X, s, t, Wt, rowptr, colidx, ws, H)

    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    flush_half = flush[: flush.numel() // 2]
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    def timed(fn, steps):
        out = []
        for _ in range(steps):
            if flush_needed:
                flush.zero_()
                flush_half.sum()
            e0.record()
            fn()
            e1.record()
            e1.synchronize()
            out.append(e0.elapsed_time(e1))
        return out

    for _ in range(args.warmup):
        layer()
        product()
    torch.cuda.synchronize()
    with ClockSampler(local_rank) as clocks:
        layer_ms = timed(layer, args.steps)
        prod_ms = timed(product, args.steps)
    assert B.device_timeouts() == 0
    total_ms = float(sum(layer_ms))
    max_ms, units = aggregate_over_ranks(total_ms, float(N) * args.steps, world)
    if rank != 0:
        return 0
    peaks, peak_kind = load_peaks()
    hbm = float(peaks.get("hbm_gbs", FALLBACK_HBM_GBS))
    bf16 = float(peaks.get("bf16_tflops", 1900.0))
    prod_s = statistics.fmean(prod_ms) * 1e-3
    flops = 2.0 * N * K * F
    # The product is fp32-accurate on the tensor cores with three bf16 MMAs per
    # real multiply-add, so its tensor ceiling is the bf16 peak / 3.
    t_hbm, t_tc = pbytes / (hbm * 1e9), flops / (bf16 / 3.0 * 1e12)
    if t_hbm >= t_tc:
        roof = {"bound": "hbm", "achieved": pbytes / prod_s / 1e9, "peak": hbm, "unit": "GB/s",
                "peak_source": f"{peak_kind} MEASURED_PEAKS.json hbm_gbs"}
    else:
        roof = {"bound": "tensor", "achieved": flops / prod_s / 1e12, "peak": bf16 / 3.0,
                "unit": "TFLOP/s (2 N K F; fp32-accurate = 3 bf16 MMAs per multiply-add)",
                "peak_source": f"{peak_kind} MEASURED_PEAKS.json bf16_tflops / 3"}
    roof.update({"kernel": f"product ({'Y W~' if mode == 'weights' else 'H~ W'})",
                 "frac": roof["achieved"] / roof["peak"],
                 "traffic": profile_file_traffic(f"ablation_product_{mode}_{w.name}.txt",
                                                 ["ablation.cu"]),
                 "other_bound_frac": (t_tc if roof["bound"] == "hbm" else t_hbm) / prod_s})
    line = {
        "metric": f"Bi-GCN ablation layer fwd nodes/s ({mode} binarized only)",
        "value": units / (max_ms * 1e-3), "unit": "nodes/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": max_ms / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f32 (3 x bf16 parts) x b1", "data": "synthetic",
        "config": {"workload": w.description + f" -- layer 1, {mode} binarized only",
                   "name": w.name, "N": N, "K": K, "F": F, "nnz": nnz,
                   "l2": "flushed before every step outside the timed events" if flush_needed
                         else "inputs larger than L2 (no flush)",
                   "launch": "bigcn_layer_forward_ablation (pack, product, aggregation)"},
        "components": {"product_us": 1e3 * statistics.fmean(prod_ms),
                       "product_algorithmic_bytes": pbytes, "product_flops": flops,
                       "layer_us": 1e3 * statistics.fmean(layer_ms)},
        "roofline": roof, "cpu_baseline": None, "e2e": None,
        "gpu_launches": (3 if mode == "weights" else 4) * args.steps,
        "clocks": clocks.summary(),
    }
    print(json.dumps(line), flush=True)
    return 0


def run_inductive(args, rank, world, local_rank):
    """Layer 1 of a workload as a binarized inductive GNN layer (Sec. 6.3,
    Table 3): ``--inductive mean`` (Bi-inductiveGCN's aggregator) or
    ``--inductive sage`` (Bi-GraphSAGE: a second, seeded neighbour weight
    matrix). One bigcn_inductive_layer_forward call per step; C1..C4 with L2
    flushed before every step outside the timed events. The roofline is the
    whole layer's algorithmic bytes (X read once, packed rows, the factored
    product written and read once, the CSR, H written) against HBM."""
    import torch

    from paper_2010_07565_gb300 import binding as B
    from paper_2010_07565_gb300 import inputs

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    agg = args.inductive
    w, data = build_workload(args.workload)
    N, K, F = w.N, w.K, w.hidden
    d = {k: torch.from_numpy(np.ascontiguousarray(v)).to(dev)
         for k, v in data.items() if k in ("X", "s", "t", "W1", "rowptr", "colidx")}
    Wn = torch.from_numpy(inputs.weights(K, F, 3200 + w.index)).to(dev) if agg == "sage" else None
    nnz = int(data["colidx"].shape[0])
    ws = torch.empty(B.bigcn_inductive_layer_workspace_bytes(agg, N, K, F), dtype=torch.uint8,
                     device=dev)
    H = torch.empty((N, F), device=dev)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    flush_half = flush[: flush.numel() // 2]

    def step():
        B.bigcn_inductive_layer_forward(agg, d["X"], d["s"], d["t"], d["W1"], d["rowptr"],
                                        d["colidx"], ws, H, W_neigh=Wn)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    times = []
    with ClockSampler(local_rank) as clocks:
        for _ in range(args.steps):
            flush.zero_()
            flush_half.sum()
            e0.record()
            step()
            e1.record()
            e1.synchronize()
            times.append(e0.elapsed_time(e1))
    assert B.device_timeouts() == 0
    total_ms = float(sum(times))
    max_ms, units = aggregate_over_ranks(total_ms, float(N) * args.steps, world)
    if rank != 0:
        return 0
    peaks, peak_kind = load_peaks()
    hbm = float(peaks.get("hbm_gbs", FALLBACK_HBM_GBS))
    words = (K + 63) // 64
    Fz = 2 * ((F + 7) // 8 * 8) if agg == "sage" else (F + 7) // 8 * 8
    zrow = 2.0 * Fz + 4.0 if K <= 32767 else 4.0 * Fz
    layer_bytes = (4.0 * N * K + 2 * 8.0 * N * words + 2.0 * N * zrow + 8.0 * (N + 1) +
                   4.0 * nnz + 4.0 * N * F)
    mean_ms = max_ms / args.steps
    achieved = layer_bytes / (mean_ms * 1e-3) / 1e9
    line = {
        "metric": f"Bi-GCN inductive layer fwd nodes/s ({agg} aggregator)",
        "value": units / (max_ms * 1e-3), "unit": "nodes/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": mean_ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32+b1",
        "data": "synthetic",
        "config": {"workload": w.description + f" -- layer 1, {agg} aggregator", "name": w.name,
                   "N": N, "K": K, "F": F, "nnz": nnz,
                   "l2": "flushed before every step outside the timed events",
                   "launch": "bigcn_inductive_layer_forward (pack rows, pack weights, XNOR "
                             "product, aggregation" + (", plus the weight concatenation copies"
                                                       if agg == "sage" else "") + ")"},
        "roofline": {"kernel": "whole layer", "bound": "hbm", "achieved": achieved, "peak": hbm,
                     "unit": "GB/s", "frac": achieved / hbm,
                     "traffic": profile_file_traffic(f"inductive_layer_{agg}_{w.name}.txt",
                                                     INDUCTIVE_SOURCES[agg]),
                     "traffic_note": "DRAM bytes of one whole call (its 4 kernels)",
                     "peak_source": f"{peak_kind} MEASURED_PEAKS.json hbm_gbs",
                     "algorithmic_bytes": layer_bytes},
        "cpu_baseline": None, "e2e": None, "gpu_launches": 4 * args.steps,
        "clocks": clocks.summary(),
    }
    print(json.dumps(line), flush=True)
    return 0


def run_weighted(args, rank, world, local_rank):
    """Layer 1 of a workload over a weighted adjacency (Sec. 3's general a_ij,
    Eq. 1's operator on A + I): seeded symmetric edge weights, uniform in
    [0.5, 2), on the workload's graph. One bigcn_weighted_layer_forward call
    per step (pack rows, pack weights, the weighted-degree pass, the XNOR
    product, the weighted aggregation), L2 flushed before every step outside
    the timed events. The roofline is the whole layer's algorithmic bytes
    against HBM: X once, the packed rows and the factored product written and
    read once, the row pointers and the weights read by the degree pass and
    the aggregation, the column indices, dinv and s written and read, H."""
    import torch

    from paper_2010_07565_gb300 import binding as B
    from paper_2010_07565_gb300 import inputs

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    w, data = build_workload(args.workload)
    N, K, F = w.N, w.K, w.hidden
    d = {k: torch.from_numpy(np.ascontiguousarray(v)).to(dev)
         for k, v in data.items() if k in ("X", "s", "t", "W1", "rowptr", "colidx")}
    values = torch.from_numpy(inputs.edge_weights(data["rowptr"], data["colidx"],
                                                  4100 + w.index)).to(dev)
    nnz = int(data["colidx"].shape[0])
    ws = torch.empty(B.bigcn_weighted_layer_workspace_bytes(N, K, F), dtype=torch.uint8,
                     device=dev)
    H = torch.empty((N, F), device=dev)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    flush_half = flush[: flush.numel() // 2]

    def step():
        B.bigcn_weighted_layer_forward(d["X"], d["s"], d["t"], d["W1"], d["rowptr"],
                                       d["colidx"], values, ws, H)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    times = []
    with ClockSampler(local_rank) as clocks:
        for _ in range(args.steps):
            flush.zero_()
            flush_half.sum()
            e0.record()
            step()
            e1.record()
            e1.synchronize()
            times.append(e0.elapsed_time(e1))
    assert B.device_timeouts() == 0
    total_ms = float(sum(times))
    max_ms, units = aggregate_over_ranks(total_ms, float(N) * args.steps, world)
    if rank != 0:
        return 0
    peaks, peak_kind = load_peaks()
    hbm = float(peaks.get("hbm_gbs", FALLBACK_HBM_GBS))
    words = (K + 63) // 64
    Fz = (F + 7) // 8 * 8
    zrow = 2.0 * Fz + 4.0 if K <= 32767 else 4.0 * Fz
    layer_bytes = (4.0 * N * K + 2 * 8.0 * N * words + 2.0 * N * zrow + 2 * 8.0 * (N + 1) +
                   4.0 * nnz + 2 * 4.0 * nnz + 4 * 4.0 * N + 4.0 * N * F)
    mean_ms = max_ms / args.steps
    achieved = layer_bytes / (mean_ms * 1e-3) / 1e9
    line = {
        "metric": "Bi-GCN weighted-adjacency layer fwd nodes/s",
        "value": units / (max_ms * 1e-3), "unit": "nodes/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": mean_ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32+b1",
        "data": "synthetic",
        "config": {"workload": w.description + " -- layer 1, edge weights uniform in [0.5, 2), "
                                               "symmetric", "name": w.name,
                   "N": N, "K": K, "F": F, "nnz": nnz,
                   "l2": "flushed before every step outside the timed events",
                   "launch": "bigcn_weighted_layer_forward (pack rows, pack weights, weighted "
                             "degrees, XNOR product, weighted aggregation)"},
        "roofline": {"kernel": "whole layer", "bound": "hbm", "achieved": achieved, "peak": hbm,
                     "unit": "GB/s", "frac": achieved / hbm,
                     "traffic": profile_file_traffic(f"weighted_layer_{w.name}.txt",
                                                     WEIGHTED_SOURCES),
                     "traffic_note": "DRAM bytes of one whole call (its 5 kernels)",
                     "peak_source": f"{peak_kind} MEASURED_PEAKS.json hbm_gbs",
                     "algorithmic_bytes": layer_bytes},
        "cpu_baseline": None, "e2e": None, "gpu_launches": 5 * args.steps,
        "clocks": clocks.summary(),
    }
    print(json.dumps(line), flush=True)
    return 0


def run_bucketed(args, rank, world, local_rank):
    """Layer 1 of a workload with sub-row bucketing (Sec. 4.1): buckets of
    ``--bucket`` B features, each with its own scales. One
    bigcn_layer_forward_bucketed call per step, L2 flushed before every step
    outside the timed events; also the bucketed product alone, against the
    POPC peak (its bit-ops) like the plain product."""
    import torch

    from paper_2010_07565_gb300 import binding as B

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    Bk = args.bucket
    w, data = build_workload(args.workload)
    N, K, F = w.N, w.K, w.hidden
    d = {k: torch.from_numpy(np.ascontiguousarray(v)).to(dev)
         for k, v in data.items() if k in ("X", "s", "t", "W1", "rowptr", "colidx")}
    nnz = int(data["colidx"].shape[0])
    ws = torch.empty(B.bigcn_layer_bucketed_workspace_bytes(N, K, F, Bk), dtype=torch.uint8,
                     device=dev)
    H = torch.empty((N, F), device=dev)
    words, nb = (K + 63) // 64, (K + Bk - 1) // Bk
    a_bits = torch.empty((N, words), dtype=torch.int64, device=dev)
    alpha = torch.empty((N, nb), device=dev)
    b_bits = torch.empty((F, words), dtype=torch.int64, device=dev)
    beta = torch.empty((F, nb), device=dev)
    Z = torch.empty((N, F), device=dev)
    B.bigcn_pack_rows_bucketed(d["X"], d["s"], d["t"], Bk, a_bits, alpha)
    B.bigcn_pack_weights_bucketed(d["W1"], Bk, b_bits, beta)

    def layer():
        B.bigcn_layer_forward_bucketed(Bk, d["X"], d["s"], d["t"], d["W1"], d["rowptr"],
                                       d["colidx"], ws, H)

    def product():
        B.bigcn_xnor_gemm_bucketed(a_bits, alpha, b_bits, beta, K, Bk, Z)

    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    flush_half = flush[: flush.numel() // 2]
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    def timed(fn):
        out = []
        for _ in range(args.steps):
            flush.zero_()
            flush_half.sum()
            e0.record()
            fn()
            e1.record()
            e1.synchronize()
            out.append(e0.elapsed_time(e1))
        return out

    for _ in range(args.warmup):
        layer()
        product()
    torch.cuda.synchronize()
    with ClockSampler(local_rank) as clocks:
        layer_ms = timed(layer)
        prod_ms = timed(product)
    total_ms = float(sum(layer_ms))
    max_ms, units = aggregate_over_ranks(total_ms, float(N) * args.steps, world)
    if rank != 0:
        return 0
    prod_s = statistics.fmean(prod_ms) * 1e-3
    bitops = float(N) * K * F
    peaks, _ = load_peaks()
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    sm_max = float(peaks.get("sm_max_mhz", 2070.0))
    peak = POPC_PER_CLK_PER_SM * 32 * sms * sm_max * 1e6 / 1e12
    achieved = bitops / prod_s / 1e12
    line = {
        "metric": f"Bi-GCN bucketed layer fwd nodes/s (buckets of {Bk} features)",
        "value": units / (max_ms * 1e-3), "unit": "nodes/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": max_ms / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32+b1",
        "data": "synthetic",
        "config": {"workload": w.description + f" -- layer 1, buckets of {Bk}", "name": w.name,
                   "N": N, "K": K, "F": F, "nnz": nnz, "bucket": Bk,
                   "l2": "flushed before every step outside the timed events",
                   "launch": "bigcn_layer_forward_bucketed (pack rows, pack weights, product, "
                             "aggregation)"},
        "components": {"product_us": 1e3 * statistics.fmean(prod_ms),
                       "layer_us": 1e3 * statistics.fmean(layer_ms)},
        "roofline": {"kernel": "bucketed product", "bound": "alu", "achieved": achieved,
                     "peak": peak, "unit": "T bit-ops/s (N K F)", "frac": achieved / peak,
                     "traffic": profile_file_traffic(f"bucketed_product_B{Bk}_{w.name}.txt",
                                                     ["bucket.cu"]),
                     "peak_source": f"measured {POPC_PER_CLK_PER_SM} POPC/clk/SM x 32 bits x "
                                    f"{sms} SMs x {sm_max:.0f} MHz"},
        "cpu_baseline": None, "e2e": None, "gpu_launches": 4 * args.steps,
        "clocks": clocks.summary(),
    }
    print(json.dumps(line), flush=True)
    return 0


def run_forward_only(args):
    """R plain forwards of the workload on cuda:0, nothing timed or printed."""
    import torch

    from paper_2010_07565_gb300.runner import GCN2Forward
    dev = torch.device("cuda", 0)
    w, data = build_workload(args.workload)
    model = GCN2Forward(w.N, w.K, w.hidden, w.out, int(data["colidx"].shape[0]), dev)
    model.load(non_blocking=False, **{k: torch.from_numpy(np.ascontiguousarray(v))
                                      for k, v in data.items()})
    for _ in range(args.forward_only):
        model.launch()
    torch.cuda.synchronize()
    return 0


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["bigcn", "reference"], default="bigcn")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD,
                    help="C1..C4, or a one-layer sweep point such as C5_K4096_F256")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--backward", action="store_true",
                    help="time layer 1's back-propagation (bigcn_layer_backward) instead")
    ap.add_argument("--ablation", choices=["weights", "features"], default=None,
                    help="time layer 1 with only the weights (or only the features) "
                         "binarized (bigcn_layer_forward_ablation) instead")
    ap.add_argument("--inductive", choices=["gcn", "mean", "sage"], default=None,
                    help="time layer 1 as a binarized inductive layer "
                         "(bigcn_inductive_layer_forward) instead")
    ap.add_argument("--weighted", action="store_true",
                    help="time layer 1 over seeded symmetric edge weights "
                         "(bigcn_weighted_layer_forward) instead")
    ap.add_argument("--bucket", type=int, default=0, metavar="B",
                    help="time layer 1 with sub-row bucketing, buckets of B features "
                         "(a multiple of 64; bigcn_layer_forward_bucketed) instead")
    ap.add_argument("--sweep-nodes", type=int, default=0, metavar="N",
                    help="run a sweep point on N nodes (mean degree 16) instead of 2^20: a "
                         "smaller case of the same kernels for profiler captures")
    ap.add_argument("--forward-only", type=int, default=0, metavar="R",
                    help="run R plain forwards (no graph, no timing, no output) and exit: "
                         "a fixed launch sequence for profilers")
    args = ap.parse_args(argv)
    if args.warmup < 3:
        ap.error("--warmup must be at least 3")
    if args.weighted and args.workload.startswith("C5_"):
        ap.error("--weighted runs layer 1 of C1..C4")
    rank, world, local_rank = dist_env()
    if args.impl == "reference":
        return run_reference(args, rank, world)
    if args.forward_only > 0:
        return run_forward_only(args)
    if args.ablation is not None:
        return run_ablation(args, rank, world, local_rank)
    if args.inductive is not None:
        return run_inductive(args, rank, world, local_rank)
    if args.bucket > 0:
        return run_bucketed(args, rank, world, local_rank)
    if args.weighted:
        return run_weighted(args, rank, world, local_rank)
    if args.workload.startswith("C5_"):
        return run_sweep(args, rank, world, local_rank)
    if args.backward:
        return run_backward(args, rank, world, local_rank)
    if world > 1:
        import torch
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local_rank)
        dist.init_process_group(backend=backend)
    try:
        return run_gpu(args, rank, world, local_rank)
    finally:
        if world > 1:
            import torch.distributed as dist
            if dist.is_initialized():
                dist.destroy_process_group()


if __name__ == "__main__":
    sys.exit(main())
