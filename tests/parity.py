"""Comparison helpers for CUDA-vs-oracle parity.

Tolerances: per-token scores within 2e-3 relative / 1e-5 absolute (bf16
inputs, fp32 accumulation on the GPU, double in the oracle); kept index sets
identical except at the top-B boundary, where a swap is allowed only when the
oracle's own scores of the swapped positions lie within that tolerance of the
boundary score; compacted K/V bit-exact given the GPU's indices.
"""

from __future__ import annotations

import numpy as np

RTOL = 2e-3
ATOL = 1e-5


def tol(x):
    return ATOL + RTOL * np.abs(x)


def check_scores(name, gpu, orc, rtol=RTOL, atol=ATOL):
    gpu = np.asarray(gpu, dtype=np.float64)
    orc = np.asarray(orc, dtype=np.float64)
    assert gpu.shape == orc.shape, (name, gpu.shape, orc.shape)
    err = np.abs(gpu - orc)
    bad = err > atol + rtol * np.abs(orc)
    if bad.any():
        i = int(np.argmax(err - (atol + rtol * np.abs(orc))))
        raise AssertionError(f"{name}: {int(bad.sum())} of {bad.size} outside tolerance; worst at "
                             f"{i}: gpu {gpu.flat[i]!r} oracle {orc.flat[i]!r}")
    rel = err / np.maximum(np.abs(orc), 1e-30)
    return float(err.max(initial=0.0)), float(rel[np.abs(orc) > 1e-6].max(initial=0.0))


def check_selection(gpu_idx, orc_idx, orc_S, N, W, budget, keep_window=True):
    """Returns the number of boundary swaps; raises on any other mismatch."""
    gpu_idx = np.asarray(gpu_idx)
    orc_idx = np.asarray(orc_idx)
    kept = min(budget, N)
    assert gpu_idx.shape == (kept,), (gpu_idx.shape, kept)
    assert np.all(np.diff(gpu_idx) > 0), "indices must be strictly ascending"
    assert gpu_idx.min(initial=0) >= 0 and gpu_idx.max(initial=0) < N
    if keep_window and W:
        assert np.array_equal(gpu_idx[kept - W:], np.arange(N - W, N)), "window must be kept"
    g, o = set(gpu_idx.tolist()), set(orc_idx.tolist())
    if g == o:
        return 0
    extra, missing = sorted(g - o), sorted(o - g)
    assert len(extra) == len(missing)
    n_cand = N - (W if keep_window else 0)
    keep = kept - (W if keep_window else 0)
    order = np.lexsort((np.arange(n_cand), -orc_S[:n_cand]))
    thr = orc_S[order[keep - 1]]
    band = tol(thr)
    for i in extra:
        assert orc_S[i] >= thr - band, f"kept {i}: oracle score {orc_S[i]} far below boundary {thr}"
    for j in missing:
        assert orc_S[j] <= thr + band, f"dropped {j}: oracle score {orc_S[j]} far above boundary {thr}"
    return len(extra)


def gather_rows(x, idx):
    """Reference gather for the bit-exactness check (numpy fancy indexing)."""
    return x[np.asarray(idx)]
