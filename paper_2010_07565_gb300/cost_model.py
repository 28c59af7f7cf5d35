"""Analytic size and operation counts of Sec. 5 (model size, data size,
cycle operations), as the paper uses them to fill Tables 2 and 3.

Counting rules (each pinned by the test suite against the printed tables):

* Model size (Sec. 5.1, Eq. 16): a full-precision layer stores d_in * d_out
  32-bit floats; a binarized layer stores d_in * d_out bits plus d_out 32-bit
  scales. Reported in KiB (1K = 1024 bytes).
* Data size (Sec. 5.2, Eq. 17): N * d 32-bit features versus N * d bits plus N
  32-bit scales. Reported in MiB.
* Cycle operations (Sec. 5.3, Eqs. 18-19): one multiply-add counts one cycle,
  64 binary operations count one cycle. A full-precision layer costs
  N d_in d_out (feature extraction) + |E| d_out (aggregation); a binarized
  layer costs N d_in d_out / 64 + 2 N d_out + |E| d_out. |E| is the paper's
  undirected edge count, self-loops not counted.

* GraphSAGE-style layers (Table 3's GraphSAGE rows) carry two weight
  matrices per layer, W_self and W_neigh (the concatenation [h_i || mean_j h_j]
  times a 2 d_in x d_out matrix): twice the parameters and twice the feature
  extraction (each binarized product with its own 2 N d_out scalings), and one
  aggregation of d_out-wide rows.

Nothing here is on the compute path; the benchmark reports these figures as
the paper's context next to measured numbers.
"""
from __future__ import annotations


def model_size_kib(dims, binary: bool, weights: int = 1) -> float:
    """Sum over layers of the parameter storage, in KiB (Eq. 16's terms);
    ``weights`` weight matrices per layer."""
    total_bits = 0
    for d_in, d_out in zip(dims[:-1], dims[1:]):
        if binary:
            total_bits += d_in * d_out + 32 * d_out
        else:
            total_bits += 32 * d_in * d_out
    return weights * total_bits / 8.0 / 1024.0


def data_size_mib(N: int, d: int, binary: bool) -> float:
    """Storage of the node features, in MiB (Eq. 17's terms)."""
    bits = N * d + 32 * N if binary else 32 * N * d
    return bits / 8.0 / 1024.0 / 1024.0


def cycle_ops(N: int, edges: int, dims, binary: bool, weights: int = 1) -> float:
    """Cycle operations of a GCN / Bi-GCN forward (Eq. 18-19's numerators and
    denominators summed over layers); ``weights`` products per layer."""
    total = 0.0
    for d_in, d_out in zip(dims[:-1], dims[1:]):
        if binary:
            total += weights * (N * d_in * d_out / 64.0 + 2.0 * N * d_out) + edges * d_out
        else:
            total += weights * float(N) * d_in * d_out + edges * d_out
    return total


def pc(d_in: int) -> float:
    """Eq. 16: per-layer model-size compression ratio."""
    return 32.0 * d_in / (d_in + 32.0)


def dc(d: int) -> float:
    """Eq. 17: data-size compression ratio."""
    return 32.0 * d / (d + 32.0)


def s_fe(d_in: int) -> float:
    """Eq. 18: feature-extraction acceleration ratio of one layer."""
    return 64.0 * d_in / (d_in + 128.0)


def s_full(d_in: int, mean_degree: float) -> float:
    """Eq. 19: whole-layer acceleration ratio with |E| = N * deg / 2."""
    return (64.0 * d_in + 32.0 * mean_degree) / (d_in + 128.0 + 32.0 * mean_degree)
