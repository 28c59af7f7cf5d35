"""Shared helpers of the GPU parity tests.

Tolerance for fp32 results: |gpu - oracle| <= ATOL + RTOL * |oracle| with
RTOL = 1e-4 and ATOL = 1e-6 (element by element). Packed bits and integer
dots are compared exactly.

Sums whose terms take both signs (the aggregation of real rows, the backward
products, the mixed real x binary products) are checked with ``check_sum``:
the relative part may be taken against the sum of the terms' magnitudes
(the error scale of any fp32 evaluation order), but only where the plain
|oracle|-relative form asks for more than fp32 resolves -- below
sqrt(n) 2^-24 times that magnitude the terms have cancelled. Every element
that passes only by that exemption is counted in EXEMPTIONS (label ->
[exempt, checked]), and the counts are printed in pytest's terminal summary.
"""
import numpy as np
import torch

RTOL = 1e-4
ATOL = 1e-6


def dev():
    return torch.device("cuda", 0)


def to_dev(a):
    if a is None:
        return None
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint64:
        a = a.view(np.int64)
    return torch.from_numpy(a).to(dev())


def bits_np(t):
    return t.cpu().numpy().view(np.uint64)


def assert_close(gpu, ref, what, rtol=RTOL, atol=ATOL):
    g = np.asarray(gpu.cpu().numpy() if isinstance(gpu, torch.Tensor) else gpu, np.float64)
    o = np.asarray(ref, np.float64)
    assert g.shape == o.shape, (what, g.shape, o.shape)
    err = np.abs(g - o)
    bound = atol + rtol * np.abs(o)
    bad = err > bound
    if bad.any():
        idx = np.unravel_index(np.argmax(err - bound), err.shape)
        raise AssertionError(
            f"{what}: {int(bad.sum())} of {bad.size} elements out of tolerance; worst at "
            f"{idx}: gpu={g[idx]!r} oracle={o[idx]!r} err={err[idx]:.3e} bound={bound[idx]:.3e}")


def assert_bits_equal(gpu_bits, ref_bits, what):
    g = bits_np(gpu_bits) if isinstance(gpu_bits, torch.Tensor) else gpu_bits
    if not np.array_equal(g, ref_bits):
        diff = np.argwhere(g != ref_bits)
        r, w = diff[0]
        raise AssertionError(f"{what}: {len(diff)} words differ; first at row {r} word {w}: "
                             f"gpu={int(g[r, w]):#018x} oracle={int(ref_bits[r, w]):#018x}")


def padded(t, rows, cols, ld, fill=0.0):
    """(view, buffer): a (rows x cols) view of ``t``'s values inside a
    (rows x ld) buffer whose padding columns hold ``fill``."""
    buf = torch.full((rows, ld), fill, dtype=t.dtype, device=t.device)
    buf[:, :cols] = t
    return buf[:, :cols], buf


# label -> [elements that passed only by the cancellation exemption, elements checked]
EXEMPTIONS = {}


def check_sum(gpu, ref, scale, what, nterms):
    """Parity of a sum of ``nterms`` terms of both signs: |g - o| <= ATOL +
    RTOL max(|o|, scale) everywhere (``scale`` = the sum of the terms'
    magnitudes), and the plain form wherever RTOL |o| exceeds the typical
    rounding error of an fp32 sum of nterms terms, sqrt(nterms) 2^-24 scale.
    Elements that need the exemption are counted under ``what``."""
    gpu = np.asarray(gpu.cpu().numpy() if isinstance(gpu, torch.Tensor) else gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    scale = np.asarray(scale, np.float64)
    assert gpu.shape == ref.shape, (what, gpu.shape, ref.shape)
    assert np.isfinite(gpu).all(), f"{what}: non-finite output"
    err = np.abs(gpu - ref)
    bound = ATOL + RTOL * np.maximum(np.abs(ref), scale)
    bad = err > bound
    if bad.any():
        q = np.unravel_index(np.argmax(err - bound), err.shape)
        raise AssertionError(f"{what}: {int(bad.sum())} of {bad.size} out of tolerance; worst "
                             f"at {q}: gpu={gpu[q]!r} oracle={ref[q]!r} scale={scale[q]!r}")
    plain = err > ATOL + RTOL * np.abs(ref)
    resolved = RTOL * np.abs(ref) > np.sqrt(nterms) * 2.0 ** -24 * scale
    stray = plain & resolved
    assert not stray.any(), f"{what}: {int(stray.sum())} |o|-relative misses outside cancellation"
    rec = EXEMPTIONS.setdefault(what, [0, 0])
    rec[0] += int(plain.sum())
    rec[1] += int(plain.size)
