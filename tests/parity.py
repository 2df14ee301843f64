"""Comparison helpers for CUDA-vs-oracle parity.

Tolerances: per-token scores within 2e-3 relative / 1e-5 absolute (bf16
inputs, fp32 accumulation on the GPU, double in the oracle); kept index sets
identical except at the top-B boundary, where a swap is allowed only when the
oracle's own scores of the swapped positions lie within that tolerance of the
boundary score; compacted K/V bit-exact given the GPU's indices.
"""

from __future__ import annotations

import json
import os

import numpy as np

RTOL = 2e-3
ATOL = 1e-5

# Every boundary swap seen by the parity tests of this session, per case
# (config and budget): written as JSON at the end of the session to the path
# in the environment variable BACON_SWAP_LOG, when it is set.
SWAP_LOG: dict = {}


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


def check_selection(gpu_idx, orc_idx, orc_S, N, W, budget, keep_window=True, log=None,
                    unit=None):
    """Returns the number of boundary swaps; raises on any other mismatch.

    A swap is a position the GPU keeps and the oracle drops, paired with one
    the oracle keeps and the GPU drops.  With `log` (a list), one record per
    unit with swaps is appended: the positions on each side, their oracle
    scores S, the oracle's boundary score (its budget-th best candidate) and
    the tolerance band around it, and the largest distance from the boundary
    as a fraction of the band (at most 1 for an allowed swap)."""
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
    if log is not None:
        gap = max(abs(float(orc_S[i]) - float(thr)) for i in extra + missing)
        log.append({"unit": list(unit) if unit is not None else None,
                    "gpu_only": [int(i) for i in extra],
                    "oracle_only": [int(j) for j in missing],
                    "oracle_S_gpu_only": [float(orc_S[i]) for i in extra],
                    "oracle_S_oracle_only": [float(orc_S[j]) for j in missing],
                    "boundary_S": float(thr), "band": float(band),
                    "max_gap_over_band": gap / float(band)})
    return len(extra)


def record_swaps(case: str, config: str, budget, units_checked: int, selected_per_unit,
                 records: list, path: str = "whole step"):
    """Adds one case's swap records to the session log."""
    SWAP_LOG[case] = {"config": config, "budget": budget, "path": path,
                      "units_checked": int(units_checked),
                      "selected_per_unit": selected_per_unit,
                      "swaps": int(sum(len(r["gpu_only"]) for r in records)),
                      "units_with_swaps": len(records),
                      "max_gap_over_band": max((r["max_gap_over_band"] for r in records),
                                               default=0.0),
                      "records": records}


def write_swap_log(code_digest: str | None = None):
    """Writes SWAP_LOG to $BACON_SWAP_LOG (no-op when unset or empty)."""
    path = os.environ.get("BACON_SWAP_LOG")
    if not path or not SWAP_LOG:
        return None
    try:
        with open(path) as f:
            old = json.load(f).get("cases", {})
    except (FileNotFoundError, ValueError):
        old = {}
    old.update(SWAP_LOG)
    doc = {"what": "boundary swaps of the CUDA path against the oracle: positions kept by "
                   "one side only, allowed when the oracle's score of each lies within "
                   f"{ATOL} + {RTOL} |S| of the oracle's boundary score",
           "tolerance": {"rtol": RTOL, "atol": ATOL},
           "code_sha256_16": code_digest,
           "cases": dict(sorted(old.items()))}
    os.makedirs(os.path.dirname(os.path.abspath(path)), exist_ok=True)
    with open(path, "w") as f:
        json.dump(doc, f, indent=1)
        f.write("\n")
    return path


def gather_rows(x, idx):
    """Reference gather for the bit-exactness check (numpy fancy indexing)."""
    return x[np.asarray(idx)]
