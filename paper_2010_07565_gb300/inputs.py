"""Seeded synthetic workloads for the Bi-GCN layer forward.

This module only draws inputs: node features, graphs (CSR), weights and the
inference-form batch-normalisation statistics of the features. It holds none of
the layer's arithmetic, and it is the one module that both the CUDA path's
callers and the CPU oracle's callers use, so that both see identical inputs.

The workloads stand in for the datasets of the paper's Table 1 / Table 2
(Cora, Citeseer, PubMed, Reddit), whose files are not used: shapes, value
distributions and degree structure are reproduced from seeds.

  C1  2708 nodes, 1433 Bernoulli(0.0127) {0,1} features, preferential
      attachment m=2 (~5.4k undirected edges), hidden 64, out 7
  C2  3327 nodes, 3703 Bernoulli(0.0085) features, preferential attachment
      with m in {1, 2} (~4.7k edges), ~1% isolated nodes, hidden 64, out 6
  C3  19717 nodes, 500 features, 10% nonzero Exponential(1), rows
      L2-normalised, preferential attachment m in {2, 3} (~44.3k edges),
      hidden 64, out 3
  C4  232965 nodes, 602 N(0,1) features, Chung-Lu graph with power-law
      expected degrees truncated at 20000 and mean 492 (~57.3M undirected
      edges, 114.6M CSR entries), hidden 128, out 41
  C5  2**20 nodes, K in {512, 1024, 4096, 8192} N(0,1) features, Erdos-Renyi
      graph with 8 * 2**20 undirected edges (mean CSR degree ~16), one layer
      with F in {64, 256}

Seeds: features 1000 + c, graph 2000 + c, layer-1 weights 3000 + c, layer-2
weights 3100 + c, for config index c (C1 -> 1). Generators are numpy PCG64.
"""
from __future__ import annotations

import dataclasses
import math
import re

import numpy as np

BN_EPS = 1e-5  # batch-normalisation epsilon (the paper does not state one)


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    index: int
    N: int
    K: int
    hidden: int
    out: int
    features: str           # "bernoulli", "exp_l2", "normal"
    feature_p: float = 0.0  # Bernoulli p or nonzero fraction
    graph: str = "ba"       # "ba", "chung_lu", "er"
    ba_m: tuple = (2,)
    ba_p: tuple = (1.0,)
    isolated: int = 0
    undirected_edges: int = 0
    max_degree: int = 0
    layers: int = 2
    description: str = ""


WORKLOADS = {
    "C1": Workload("C1", 1, 2708, 1433, 64, 7, "bernoulli", 0.0127, "ba", (2,), (1.0,),
                   description="2-layer Bi-GCN, Cora-shaped: N=2708, K=1433, hidden 64, out 7"),
    "C2": Workload("C2", 2, 3327, 3703, 64, 6, "bernoulli", 0.0085, "ba", (1, 2), (0.58, 0.42),
                   isolated=33,
                   description="2-layer Bi-GCN, Citeseer-shaped: N=3327, K=3703, hidden 64, out 6"),
    "C3": Workload("C3", 3, 19717, 500, 64, 3, "exp_l2", 0.10, "ba", (2, 3), (0.75, 0.25),
                   description="2-layer Bi-GCN, PubMed-shaped: N=19717, K=500, hidden 64, out 3"),
    "C4": Workload("C4", 4, 232965, 602, 128, 41, "normal", 0.0, "chung_lu",
                   undirected_edges=57_300_000, max_degree=20_000,
                   description="2-layer Bi-GCN, Reddit-shaped: N=232965, K=602, ~114.6M CSR "
                               "entries, hidden 128, out 41"),
}


def sweep_workload(K: int, F: int) -> Workload:
    """C5: one layer on 2**20 nodes, K input and F output features."""
    assert K in (512, 1024, 4096, 8192) and F in (64, 256)
    return Workload(f"C5_K{K}_F{F}", 5, 1 << 20, K, F, F, "normal", 0.0, "er",
                    undirected_edges=8 << 20, layers=1,
                    description=f"1-layer Bi-GCN sweep: N=2^20, K={K}, F={F}, "
                                "Erdos-Renyi mean degree 16")


def get_workload(name: str) -> Workload:
    """C1..C4 by name, or a sweep point named like ``C5_K4096_F256``."""
    if name in WORKLOADS:
        return WORKLOADS[name]
    m = re.fullmatch(r"C5_K(\d+)_F(\d+)", name)
    if m:
        return sweep_workload(int(m.group(1)), int(m.group(2)))
    raise KeyError(name)


# ------------------------------------------------------------- features ----
def features(w: Workload, seed: int | None = None) -> np.ndarray:
    """Node features X (N x K, fp32, row-major) for workload ``w``."""
    rng = np.random.Generator(np.random.PCG64(1000 + w.index if seed is None else seed))
    return draw_features(rng, w.N, w.K, w.features, w.feature_p)


def draw_features(rng, N: int, K: int, kind: str, p: float = 0.0) -> np.ndarray:
    if kind == "bernoulli":
        return (rng.random((N, K), dtype=np.float32) < np.float32(p)).astype(np.float32)
    if kind == "exp_l2":
        nz = rng.random((N, K), dtype=np.float32) < np.float32(p)
        vals = rng.standard_exponential((N, K), dtype=np.float64) * nz
        norms = np.sqrt((vals * vals).sum(axis=1, keepdims=True))
        norms[norms == 0.0] = 1.0
        return (vals / norms).astype(np.float32)
    if kind == "normal":
        return rng.standard_normal((N, K), dtype=np.float32)
    raise ValueError(kind)


def bn_stats(X: np.ndarray, eps: float = BN_EPS):
    """Inference-form batch-normalisation parameters of Sec. 6.2's input BN.

    gamma = 1 and beta = 0 ("zero mean and variance one"); the running
    statistics are the biased per-feature mean and variance of X itself,
    accumulated in float64. Returns (s, t), fp32, with s = 1/sqrt(var + eps)
    and t = -mean * s, so that the normalised feature is x * s + t.
    """
    X64 = X.astype(np.float64, copy=False)
    mean = X64.mean(axis=0)
    var = X64.var(axis=0)
    s = 1.0 / np.sqrt(var + eps)
    return s.astype(np.float32), (-mean * s).astype(np.float32)


def weights(K: int, F: int, seed: int) -> np.ndarray:
    """W (K x F, fp32, row-major), entries N(0, 1/K)."""
    rng = np.random.Generator(np.random.PCG64(seed))
    return (rng.standard_normal((K, F)) / math.sqrt(K)).astype(np.float32)


def layer_weights(w: Workload):
    """(W1, W2) for the workload's layers (W2 is None for a 1-layer sweep)."""
    W1 = weights(w.K, w.hidden, 3000 + w.index)
    W2 = weights(w.hidden, w.out, 3100 + w.index) if w.layers == 2 else None
    return W1, W2


# ---------------------------------------------------------------- graphs ----
def edges_to_csr(u: np.ndarray, v: np.ndarray, N: int):
    """Undirected unique edges (u < v) -> symmetric CSR (rowptr int64, colidx
    int32), both directions stored, columns ascending within a row, no
    self-loops."""
    u = np.asarray(u, np.int64)
    v = np.asarray(v, np.int64)
    key = np.concatenate([u * N + v, v * N + u])
    key.sort()
    rows = key // N
    rowptr = np.zeros(N + 1, np.int64)
    np.cumsum(np.bincount(rows, minlength=N), out=rowptr[1:])
    key -= rows * N
    return rowptr, key.astype(np.int32)


def _sorted_unique(keys: np.ndarray) -> np.ndarray:
    """Distinct values of an int64 array, ascending (sort + adjacent compare)."""
    keys = np.sort(keys)
    if keys.size == 0:
        return keys
    keep = np.empty(keys.size, bool)
    keep[0] = True
    np.not_equal(keys[1:], keys[:-1], out=keep[1:])
    return keys[keep]


def _unique_pairs(a: np.ndarray, b: np.ndarray, N: int) -> np.ndarray:
    lo = np.minimum(a, b).astype(np.int64)
    hi = np.maximum(a, b).astype(np.int64)
    keep = lo != hi
    return _sorted_unique(lo[keep] * N + hi[keep])


def preferential_attachment(N: int, m_choices, m_probs, rng, isolated: int = 0):
    """Barabasi-Albert-style growth: each new node links to m distinct existing
    nodes chosen with probability proportional to degree (m drawn per node).
    ``isolated`` nodes take no part and keep degree 0. Node ids are randomly
    permuted so that hubs are not clustered at low ids."""
    n = N - isolated
    mmax = max(m_choices)
    ms = rng.choice(np.asarray(m_choices), size=n, p=np.asarray(m_probs))
    ends = np.empty(2 * int(ms.sum()) + 2 * mmax * mmax, np.int64)
    ne = 0
    us, vs = [], []
    for i in range(1, n):
        m = min(int(ms[i]), i)
        chosen = set()
        while len(chosen) < m:
            if ne == 0 or i <= mmax:
                c = int(rng.integers(0, i))
            else:
                c = int(ends[rng.integers(0, ne)])
            chosen.add(c)
        for c in chosen:
            us.append(c)
            vs.append(i)
            ends[ne] = c
            ends[ne + 1] = i
            ne += 2
    perm = rng.permutation(N)
    u = perm[np.asarray(us, np.int64)]
    v = perm[np.asarray(vs, np.int64)]
    keys = _unique_pairs(u, v, N)
    return keys // N, keys % N


def _iid_endpoints(p: np.ndarray, M: int, rng) -> np.ndarray:
    """M i.i.d. draws from the categorical distribution p, in random order
    (multinomial counts per category, expanded and shuffled)."""
    counts = rng.multinomial(M, p)
    ends = np.repeat(np.arange(p.shape[0], dtype=np.int64), counts)
    rng.shuffle(ends)
    return ends


def _sample_unique_edges(p: np.ndarray, target_edges: int, rng) -> np.ndarray:
    """Undirected edge keys lo * N + hi (lo < hi): endpoint pairs drawn i.i.d.
    from p, self-loops and repeats dropped, topped up and then subsampled to
    exactly ``target_edges`` distinct edges."""
    N = p.shape[0]
    keys = np.empty(0, np.int64)
    batch = int(target_edges * 1.08) + 64
    while keys.size < target_edges:
        fresh = _unique_pairs(_iid_endpoints(p, batch, rng), _iid_endpoints(p, batch, rng), N)
        keys = fresh if keys.size == 0 else _sorted_unique(np.concatenate([keys, fresh]))
        batch = max(int((target_edges - keys.size) * 1.5), 1024)
    if keys.size > target_edges:
        keep = rng.choice(keys.size, size=target_edges, replace=False)
        keys = keys[np.sort(keep)]
    return keys


def chung_lu(N: int, target_edges: int, mean_degree: float, max_degree: int, rng,
             exponent: float = 2.5):
    """Chung-Lu graph: expected degrees w_i from a power law (tail exponent
    ``exponent``) truncated at ``max_degree`` and scaled to ``mean_degree``;
    endpoints drawn proportional to w; self-loops and duplicates dropped;
    exactly ``target_edges`` unique undirected edges kept."""
    w = rng.pareto(exponent - 1.0, size=N) + 1.0
    for _ in range(50):
        w = np.minimum(w * (mean_degree / w.mean()), max_degree)
    keys = _sample_unique_edges(w / w.sum(), target_edges, rng)
    return keys // N, keys % N


def erdos_renyi(N: int, target_edges: int, rng):
    """G(n, m): ``target_edges`` distinct undirected edges chosen uniformly."""
    keys = _sample_unique_edges(np.full(N, 1.0 / N), target_edges, rng)
    return keys // N, keys % N


def graph(w: Workload, seed: int | None = None):
    """Symmetric CSR (rowptr int64 N+1, colidx int32 nnz) for workload ``w``."""
    rng = np.random.Generator(np.random.PCG64(2000 + w.index if seed is None else seed))
    if w.graph == "ba":
        u, v = preferential_attachment(w.N, w.ba_m, w.ba_p, rng, w.isolated)
    elif w.graph == "chung_lu":
        u, v = chung_lu(w.N, w.undirected_edges, 2.0 * w.undirected_edges / w.N,
                        w.max_degree, rng)
    elif w.graph == "er":
        u, v = erdos_renyi(w.N, w.undirected_edges, rng)
    else:
        raise ValueError(w.graph)
    return edges_to_csr(u, v, w.N)


def edge_weights(rowptr, colidx, seed: int, low: float = 0.5, high: float = 2.0) -> np.ndarray:
    """Symmetric positive edge weights for a CSR (fp32, one per entry, in the
    order of colidx): the entries (i, j) and (j, i) get the same weight,
    uniform between low and high. Each node draws a 32-bit key from the seeded
    PCG64; an entry's weight comes from a 32-bit integer hash of the sum of its
    two nodes' keys (the same sum from either end, so no pairing of the two
    entries is needed)."""
    rowptr = np.asarray(rowptr, np.int64)
    N = rowptr.shape[0] - 1
    key = np.random.Generator(np.random.PCG64(seed)).integers(0, 1 << 32, size=N,
                                                               dtype=np.uint32)
    x = np.repeat(key, np.diff(rowptr))
    x += key[np.asarray(colidx)]                 # wraps modulo 2^32
    m = np.uint32(0x45D9F3B)
    x ^= x >> np.uint32(16)
    x *= m
    x ^= x >> np.uint32(16)
    x *= m
    x ^= x >> np.uint32(16)
    u = (x >> np.uint32(8)).astype(np.float32)
    u *= np.float32(1.0 / (1 << 24))
    u *= np.float32(high - low)
    u += np.float32(low)
    return u


def random_graph(N: int, mean_degree: float, seed: int, hub_degree: int = 0):
    """Small test graph: G(n, m) with about ``mean_degree`` CSR entries per row,
    plus (optionally) node 0 joined to ``hub_degree`` other nodes."""
    rng = np.random.Generator(np.random.PCG64(seed))
    m = int(round(N * mean_degree / 2.0))
    m = min(m, N * (N - 1) // 2)
    if m > 0:
        u, v = erdos_renyi(N, m, rng)
    else:
        u = v = np.empty(0, np.int64)
    if hub_degree > 0:
        others = rng.choice(np.arange(1, N), size=min(hub_degree, N - 1), replace=False)
        keys = _sorted_unique(np.concatenate([u * N + v,
                                              _unique_pairs(np.zeros_like(others), others, N)]))
        u, v = keys // N, keys % N
    return edges_to_csr(u, v, N)


def layer_case(N: int, K: int, F: int, seed: int, mean_degree: float = 4.0,
               features_kind: str = "normal", hub_degree: int = 0, centred: bool = True):
    """A self-contained single-layer case: X, (s, t), W, rowptr, colidx."""
    rng = np.random.Generator(np.random.PCG64(seed))
    X = draw_features(rng, N, K, features_kind, 0.05)
    s, t = bn_stats(X) if centred else (None, None)
    W = weights(K, F, seed + 7)
    rowptr, colidx = random_graph(N, mean_degree, seed + 11, hub_degree)
    return dict(X=X, s=s, t=t, W=W, rowptr=rowptr, colidx=colidx)
