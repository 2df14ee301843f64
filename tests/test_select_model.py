"""Model of the selection kernels' algorithm, run on the CPU.

The calibration and adaptive-selection kernels choose "the k best" (larger
value first, equal values -> lower position first, as the oracle's stable
sort does) without sorting: a range-adaptive radix select finds the k-th
best key tau and how many of the keys equal to tau are taken, and a walk
over each warp's contiguous segment in index order decides membership.
Once a pass leaves at most 32 keys in the boundary range, one warp sorts
them across its lanes (a bitonic network over (valid, key) pairs) instead
of running more passes.  This file replays those steps in Python, with the
kernels' integer key mapping, bin widths, buffer rule, 32-lane bitonic
network and segment cut, and checks every result against a plain stable
sort on inputs with many ties, narrow and wide key ranges, and k from 1 to
n.  Mistakes in the tie rule, the boundary-bin arithmetic or the network's
direction fail it.
"""

import random
import struct

import numpy as np
import pytest

SEL_BITS = 11
SEL_BINS = 1 << SEL_BITS
SEL_CAP = 2048


def float_key(f):
    """Order-preserving 32-bit key of an fp32 value (the kernels' mapping)."""
    u = struct.unpack("<I", struct.pack("<f", float(np.float32(f))))[0]
    return u ^ 0xFFFFFFFF if u & 0x80000000 else u | 0x80000000


def bitonic_desc32(vals):
    """The warp's network: lane l exchanges with lane l ^ j; the lower lane of
    a pair keeps the maximum in blocks whose bit k is clear."""
    v = list(vals)
    k = 2
    while k <= 32:
        j = k >> 1
        while j > 0:
            o = [v[l ^ j] for l in range(32)]
            v = [max(v[l], o[l]) if ((l & k) == 0) == ((l & j) == 0) else min(v[l], o[l])
                 for l in range(32)]
            j >>= 1
        k <<= 1
    return v


def radix_select(keys, k, warp_sort=True):
    """(tau, need, count_eq) for the k-th best key, as the kernel computes it."""
    lo, hi = min(keys), max(keys)
    span = hi - lo + 1
    shift = 0
    while ((span - 1) >> shift) >= SEL_BINS:
        shift += 1
    width, remaining = span, k
    in_range, buf = -1, None
    while True:
        collect = buf is None and 0 <= in_range <= SEL_CAP
        src = buf if buf is not None else keys
        hist = [0] * SEL_BINS
        new_buf = []
        for key in src:
            if lo <= key < lo + width:
                hist[(key - lo) >> shift] += 1
                if collect:
                    new_buf.append(key)
        if collect:
            buf = new_buf
        # the bin where the count from the top reaches `remaining`
        before = 0
        for b in range(SEL_BINS - 1, -1, -1):
            if before + hist[b] >= remaining:
                break
            before += hist[b]
        lo += b << shift
        remaining -= before
        in_bin = hist[b]
        in_range = in_bin
        width = 1 << shift
        if shift == 0:
            return lo, remaining, in_bin
        if warp_sort and in_bin <= 32:
            src = buf if buf is not None else keys
            few = [key for key in src if lo <= key < lo + width]
            assert len(few) == in_bin
            lanes = [(1 << 32) | key for key in few] + [0] * (32 - len(few))
            v = bitonic_desc32(lanes)
            tau = v[remaining - 1] & 0xFFFFFFFF
            eq = sum(1 for x in v if x >> 32 and (x & 0xFFFFFFFF) == tau)
            gt = sum(1 for x in v if x >> 32 and (x & 0xFFFFFFFF) > tau)
            return tau, remaining - gt, eq
        shift = shift - SEL_BITS if shift > SEL_BITS else 0


def members(keys, sel, nwarps):
    """Membership by the warp-segmented index-ordered walk."""
    tau, need, count_eq = sel
    n = len(keys)
    per = (((n + nwarps - 1) // nwarps) + 31) & ~31
    # equal keys before each segment (skipped by the kernels when every tie is taken)
    out = []
    eq_before = 0
    for w in range(nwarps):
        s0, s1 = min(n, w * per), min(n, w * per + per)
        running = eq_before if need != count_eq else 0
        for i in range(s0, s1):
            eq = keys[i] == tau
            if keys[i] > tau or (eq and (need == count_eq or running < need)):
                out.append(i)
            running += eq
        eq_before += sum(1 for i in range(s0, s1) if keys[i] == tau)
    return out


def reference(values, k):
    order = sorted(range(len(values)), key=lambda i: (-float(np.float32(values[i])), i))
    return sorted(order[:k])


def cases():
    rng = random.Random(7)
    out = []
    for trial in range(60):
        n = rng.choice([1, 2, 31, 32, 33, 100, 640, 992, 2047, 4000])
        kind = trial % 6
        if kind == 0:    # heavy ties: few distinct values
            vals = [rng.choice([0.25, 0.5, 0.125, 1e-6]) for _ in range(n)]
        elif kind == 1:  # plateaus like a max-pooled score
            base = [rng.random() * 1e-3 for _ in range(n)]
            vals = [max(base[max(0, i - 3):i + 4]) for i in range(n)]
        elif kind == 2:  # wide dynamic range
            vals = [10 ** rng.uniform(-12, -1) for _ in range(n)]
        elif kind == 3:  # all equal
            vals = [3.0] * n
        elif kind == 4:  # signed values
            vals = [rng.gauss(0, 1) for _ in range(n)]
        else:            # near-equal keys (a few ulps apart)
            vals = [float(np.nextafter(np.float32(1.0), np.float32(2.0)) * (1 + rng.randint(0, 3) * 1e-7))
                    for _ in range(n)]
        for k in sorted({1, n, max(1, n // 3), max(1, n - 1), rng.randint(1, n)}):
            out.append((vals, k))
    return out


@pytest.mark.parametrize("warp_sort", [True, False])
def test_select_matches_stable_sort(warp_sort):
    for vals, k in cases():
        keys = [float_key(v) for v in vals]
        sel = radix_select(keys, k, warp_sort)
        for nwarps in (8, 32):
            got = members(keys, sel, nwarps)
            assert got == reference(vals, k), (len(vals), k, nwarps)


def test_bitonic_network_sorts_descending():
    rng = random.Random(3)
    for _ in range(500):
        m = rng.randint(1, 32)
        lanes = [(1 << 32) | rng.randint(0, 40) for _ in range(m)] + [0] * (32 - m)
        assert bitonic_desc32(lanes) == sorted(lanes, reverse=True)


def test_wrong_network_direction_is_caught():
    """A network whose lower lane keeps the minimum sorts ascending: the
    selected tau is then wrong and the check above would fail."""
    vals = [0.5, 0.25, 0.75, 0.125, 1.0]
    keys = [float_key(v) for v in vals]
    lanes = [(1 << 32) | key for key in keys] + [0] * 27
    v = bitonic_desc32(lanes)
    assert (v[1] & 0xFFFFFFFF) == float_key(0.75)   # second best
    asc = sorted(lanes)
    assert (asc[1] & 0xFFFFFFFF) != float_key(0.75)


def test_float_key_orders_like_floats():
    xs = [-np.inf, -3.5, -1e-30, -0.0, 0.0, 1e-30, 2.0, np.inf]
    ks = [float_key(x) for x in xs]
    assert ks == sorted(ks)
    assert float_key(-0.0) < float_key(0.0)


# ------------------------------------------------ calibration kernel's runs

def slot_major(T, PER):
    """Storage index of each position in the calibration kernel's
    shared-memory arrays (thread t owns positions t PER .. t PER + PER - 1;
    slot k of thread t is stored at k T + t), and its inverse."""
    at = lambda i: (i % PER) * T + i // PER
    pos = lambda s: (s % T) * PER + s // T
    return at, pos


def members_by_runs(keys, sel, T, PER):
    """Membership as the calibration kernel decides it: every thread walks
    its own run in position order; its tie rank starts from the keys equal
    to tau in the runs of lower threads (an exclusive scan in thread order),
    and the members are written at the scan of the per-thread member counts."""
    tau, need, count_eq = sel
    n = len(keys)
    eq_counts = [sum(1 for i in range(t * PER, min(n, t * PER + PER)) if keys[i] == tau)
                 for t in range(T)]
    eq_before = [0] * T
    for t in range(1, T):
        eq_before[t] = eq_before[t - 1] + eq_counts[t - 1]
    masks = []
    for t in range(T):
        rank = eq_before[t] if need != count_eq else 0
        m = []
        for i in range(t * PER, min(n, t * PER + PER)):
            eq = keys[i] == tau
            if keys[i] > tau or (eq and (need == count_eq or rank < need)):
                m.append(i)
            rank += eq
        masks.append(m)
    out = [None] * sum(len(m) for m in masks)
    pos = 0
    for m in masks:              # exclusive scan of the member counts
        for j, i in enumerate(m):
            out[pos + j] = i
        pos += len(m)
    return out


@pytest.mark.parametrize("T,PER", [(128, 8), (256, 8), (512, 8), (1024, 8), (1024, 16)])
def test_run_membership_matches_stable_sort(T, PER):
    for vals, k in cases():
        if len(vals) > T * PER:
            continue
        keys = [float_key(v) for v in vals]
        # the radix select walks storage indices: the key multiset is the same
        at, pos = slot_major(T, PER)
        stored = [None] * (T * PER)
        for i, key in enumerate(keys):
            stored[at(i)] = key
        walked = [stored[s] for s in range(T * PER) if pos(s) < len(keys)]
        assert sorted(walked) == sorted(keys)
        sel = radix_select(walked, k)
        assert members_by_runs(keys, sel, T, PER) == reference(vals, k), (len(vals), k)


@pytest.mark.parametrize("T,PER", [(128, 8), (256, 8), (512, 8), (1024, 8), (1024, 16), (1024, 24)])
def test_slot_major_layout_is_a_conflict_free_bijection(T, PER):
    at, pos = slot_major(T, PER)
    assert sorted(at(i) for i in range(T * PER)) == list(range(T * PER))
    assert all(pos(at(i)) == i for i in range(T * PER))
    # a warp's threads reading their own position plus one offset d touch
    # 32 consecutive words: 32 distinct banks
    for w in range(0, T, 32):
        for d in (-3, -1, 0, 1, 5, PER - 1, PER + 2):
            words = [at(t * PER + d) for t in range(w, w + 32)
                     if 0 <= t * PER + d < T * PER]
            if len(words) == 32:
                assert len({x % 32 for x in words}) == 32, (w, d)


def test_run_membership_without_the_tie_scan_is_caught():
    """Ranking ties inside each run only (no scan over lower threads) keeps
    too many equal keys: the comparison above would fail."""
    vals = [1.0] * 64
    keys = [float_key(v) for v in vals]
    sel = radix_select(keys, 10)
    tau, need, count_eq = sel
    per_run_only = [i for t in range(8) for j, i in enumerate(range(t * 8, t * 8 + 8))
                    if keys[i] > tau or j < need]
    assert per_run_only != reference(vals, 10)
    assert members_by_runs(keys, sel, 8, 8) == reference(vals, 10)


# ---------------------------------- boundary search of one histogram pass

def boundary_direct(hist, remaining):
    """The bin where the count from the top reaches `remaining`: (bin, keys
    still needed inside it, its count)."""
    before = 0
    for b in range(len(hist) - 1, -1, -1):
        if before + hist[b] >= remaining:
            return b, remaining - before, hist[b]
        before += hist[b]
    raise AssertionError("fewer keys than requested")


def boundary_by_warp(hist, remaining):
    """The single warp's search: lane l owns bins [64 l, 64 l + 64); suffix
    sums over the lanes find the highest lane whose count from the top
    reaches `remaining`; its 64 bins, two per lane, go through the same
    suffix-sum search; the chosen pair's upper bin is taken if it alone
    completes the count, else the lower one."""
    assert len(hist) == 2048
    mine = [sum(hist[64 * l:64 * l + 64]) for l in range(32)]
    incl = [sum(mine[l:]) for l in range(32)]           # shfl_down suffix scan
    hit = [incl[l] >= remaining for l in range(32)]
    lb = max(l for l in range(32) if hit[l])
    above = incl[lb] - mine[lb]
    pairs = [(hist[64 * lb + 2 * l], hist[64 * lb + 2 * l + 1]) for l in range(32)]
    inc2 = [sum(c0 + c1 for c0, c1 in pairs[l:]) for l in range(32)]
    l2 = max(l for l in range(32) if above + inc2[l] >= remaining)
    c0, c1 = pairs[l2]
    before = above + inc2[l2] - (c0 + c1)
    b0 = 64 * lb + 2 * l2
    if before + c1 >= remaining:
        return b0 + 1, remaining - before, c1
    return b0, remaining - before - c1, c0


def test_warp_boundary_search_matches_direct_scan():
    rng = random.Random(11)
    for trial in range(400):
        kind = trial % 4
        if kind == 0:      # sparse: few occupied bins, long runs of zeros
            hist = [0] * 2048
            for _ in range(rng.randint(1, 40)):
                hist[rng.randrange(2048)] += rng.randint(1, 50)
        elif kind == 1:    # dense
            hist = [rng.randint(0, 9) for _ in range(2048)]
        elif kind == 2:    # one heavy bin
            hist = [0] * 2048
            hist[rng.randrange(2048)] = rng.randint(1, 16000)
        else:              # occupied bins only at a lane's edges
            hist = [0] * 2048
            for l in range(32):
                if rng.random() < 0.5:
                    hist[64 * l + rng.choice([0, 1, 62, 63])] = rng.randint(1, 5)
            if not sum(hist):
                hist[0] = 1
        total = sum(hist)
        for remaining in sorted({1, total, max(1, total // 2), rng.randint(1, total)}):
            assert boundary_by_warp(hist, remaining) == boundary_direct(hist, remaining), (
                trial, remaining)


def test_warp_boundary_search_with_the_wrong_pair_order_is_caught():
    """Taking the pair's lower bin first (the wrong end of the suffix order)
    picks a bin below the boundary: the comparison above would fail."""
    hist = [0] * 2048
    hist[100], hist[101] = 3, 4        # one pair, upper bin 101 holds 4
    b, need, cnt = boundary_direct(hist, 2)
    assert (b, need, cnt) == (101, 2, 4)
    assert boundary_by_warp(hist, 2) == (101, 2, 4)
    # lower bin first: 100 would be reported
    assert b != 100
