"""Model of the calibration kernel's per-thread layout, run on the CPU.

The calibration kernel gives each of T threads PER consecutive positions and
keeps a thread's run in registers.  The width-7 max-pool and the coherence
window (Eqs. 5-7) take the values beyond a run from the adjacent lanes' runs
by warp shuffles; lanes 0 and 31 read theirs from global memory, and values
outside the array count as -inf (pooling, over the candidates) or 0
(coherence, over [0, N)).  The coherence window sum slides along the run
with the radius compiled as a constant for r in {3, 5, 7, 9} when the run,
its halo and V fit in registers; any other radius reads its window from
global memory in the same order.  lambda (Eqs. 12-15) is two walks over the
M members: the pooled backbone's moments about its M-th value together
with the members' V sum, then V's squared deviations from its mean.

This file replays those steps in numpy float32, thread by thread and lane
by lane, and checks: the shuffle-halo slide equals the global-memory slide
bit for bit (a wrong halo index, lane test or padding changes a sum), the
pooled backbone equals the oracle's max-pool exactly, the coherence and V
match the oracle within fp32 rounding, and lambda matches the oracle's
two-pass population statistics.  Ragged N, threads wholly past N, and
windows reaching across warps and past both ends are covered.
"""

import numpy as np
import pytest

import oracle

F32 = np.float32


def run_fits(per, r):
    """The kernel's rule for compiling a radius as a constant."""
    return r <= per and 2 * per + 2 * r <= 56


def thread_runs(a, T, PER, fill=0.0):
    """[T][PER] runs of a (fill at and past len(a))."""
    out = np.full(T * PER, fill, dtype=F32)
    out[:len(a)] = a
    return out.reshape(T, PER)


def pool_model(B, n_cand, T, PER):
    """Width-7 max-pool over the candidates, neighbours by shuffles."""
    N = len(B)
    x = thread_runs(B, T, PER)
    pos = np.arange(T * PER).reshape(T, PER)
    x[pos >= n_cand] = -np.inf
    out = np.zeros((T, PER), dtype=F32)
    for t in range(T):
        lane, i0 = t % 32, t * PER
        hl, hr = [], []
        for m in range(3):
            jl, jr = i0 - 3 + m, i0 + PER + m
            if lane == 0:
                hl.append(F32(B[jl]) if 0 <= jl < n_cand else F32(-np.inf))
            else:
                hl.append(x[t - 1][PER - 3 + m])
            if lane == 31:
                hr.append(F32(B[jr]) if jr < n_cand else F32(-np.inf))
            else:
                hr.append(x[t + 1][m])

        def at(j):
            return hl[j + 3] if j < 0 else (hr[j - PER] if j >= PER else x[t][j])

        for k in range(PER):
            if i0 + k < n_cand:
                out[t][k] = max(at(k + d) for d in range(-3, 4))
    return out.reshape(-1)[:N]


def coherence_shuffle_model(E, T, PER, R):
    """The constant-radius slide: halo by shuffles, 0 outside [0, N)."""
    N = len(E)
    x = thread_runs(E, T, PER)
    L = np.zeros((T, PER), dtype=F32)
    inv_full = F32(1) / F32(2 * R + 1)
    for t in range(T):
        lane, i0 = t % 32, t * PER
        e = np.zeros(PER + 2 * R, dtype=F32)
        for m in range(R):
            jl, jh = i0 - R + m, i0 + PER + m
            if lane == 0:
                e[m] = E[jl] if 0 <= jl < N else 0
            else:
                e[m] = x[t - 1][PER - R + m] if jl >= 0 else 0
            if lane == 31:
                e[R + PER + m] = E[jh] if jh < N else 0
            else:
                e[R + PER + m] = x[t + 1][m] if jh < N else 0
        e[R:R + PER] = x[t]
        s = F32(0)
        for j in range(2 * R + 1):
            s = F32(s + e[j])
        for k in range(PER):
            i = i0 + k
            if i < N:
                cnt = min(N - 1, i + R) - max(0, i - R) + 1
                w = inv_full if cnt == 2 * R + 1 else F32(1) / F32(cnt)
                L[t][k] = F32(max(s, F32(0)) * w)
            if k + 1 < PER:
                s = F32(s - e[k])
                s = F32(s + e[k + 2 * R + 1])
    return L.reshape(-1)[:N]


def coherence_global_model(E, T, PER, r):
    """Any radius: the window read from global memory, the same slide."""
    N = len(E)
    L = np.zeros((T, PER), dtype=F32)
    inv_full = F32(1) / F32(2 * r + 1)
    for t in range(T):
        i0 = t * PER
        lo, hi = max(0, i0 - r), min(N - 1, i0 + r)
        s = F32(0)
        for j in range(lo, hi + 1):
            s = F32(s + E[j])
        for k in range(PER):
            i = i0 + k
            if i < N:
                cnt = hi - lo + 1
                w = inv_full if cnt == 2 * r + 1 else F32(1) / F32(cnt)
                L[t][k] = F32(max(s, F32(0)) * w)
                if i - r >= 0:
                    s = F32(s - E[i - r])
                if i + 1 + r <= N - 1:
                    s = F32(s + E[i + 1 + r])
                lo, hi = max(0, i + 1 - r), min(N - 1, i + 1 + r)
    return L.reshape(-1)[:N]


def coherence_model(E, T, PER, r):
    if r in (3, 5, 7, 9) and run_fits(PER, r):
        return coherence_shuffle_model(E, T, PER, r)
    return coherence_global_model(E, T, PER, r)


def lambda_model(Bt, V, members, gamma=1.0, eps=1e-8):
    """Two walks over the members in fp32 (the kernel's per-thread sums are
    combined by a tree; the order only changes rounding)."""
    M = len(members)
    b, v = Bt[members].astype(F32), V[members].astype(F32)
    pb = b.min()  # the M-th best value: every member is at or above it
    db = b - pb
    sx, syy, sz = F32(db.sum(dtype=F32)), F32((db * db).sum(dtype=F32)), F32(v.sum(dtype=F32))
    inv_m = F32(1) / F32(M)
    mb, mv = sx * inv_m, sz * inv_m
    dv = v - mv
    varv = F32((dv * dv).sum(dtype=F32)) * inv_m
    stdb = np.sqrt(max(F32(syy * inv_m - mb * mb), F32(0)))
    stdv = np.sqrt(varv)
    return float(F32(gamma) * stdb / (stdv + F32(eps)))


def residual_like(rng, N):
    """Non-negative residuals: half zeros, a long tail, a few spikes."""
    e = rng.exponential(1e-4, N) * (rng.random(N) < 0.5)
    spikes = rng.choice(N, size=max(1, N // 97), replace=False)
    e[spikes] += rng.exponential(5e-3, len(spikes))
    return e.astype(F32)


def backbone_like(rng, N):
    """Positive scores with plateaus of equal values and ties."""
    b = rng.exponential(1e-4, N)
    b[rng.random(N) < 0.2] = 1e-4
    b[rng.choice(N, size=max(1, N // 50), replace=False)] += rng.exponential(1e-2, max(1, N // 50))
    return b.astype(F32)


SHAPES = [  # (threads, positions per thread, N): ragged N, tail threads past N
    (64, 8, 512), (64, 8, 509), (128, 8, 640), (64, 16, 1000), (96, 16, 1531),
    (64, 24, 1500), (32, 16, 17),
]


@pytest.mark.parametrize("T,PER,N", SHAPES)
@pytest.mark.parametrize("r", [3, 5, 7, 9])
def test_shuffle_halo_slide_equals_global_slide(T, PER, N, r):
    rng = np.random.default_rng(1000 * T + 10 * PER + r)
    E = residual_like(rng, N)
    if not run_fits(PER, r):
        pytest.skip("radius read from global memory at this run length")
    got = coherence_shuffle_model(E, T, PER, r)
    want = coherence_global_model(E, T, PER, r)
    assert np.array_equal(got.view(np.uint32), want.view(np.uint32))


@pytest.mark.parametrize("T,PER,N", SHAPES)
@pytest.mark.parametrize("r", [0, 1, 3, 5, 7, 9, 12])
def test_coherence_matches_oracle(T, PER, N, r):
    rng = np.random.default_rng(7 * T + PER + 31 * r)
    E = residual_like(rng, N)
    got = coherence_model(E, T, PER, r).astype(np.float64)
    want = oracle.coherence(E, r)
    # fp32 sliding sums of values up to ~2e-2: error ~ few ulp of the window sum
    tol = 1e-5 * np.maximum(want, 1e-3) + 1e-9
    assert np.all(np.abs(got - want) <= tol), np.max(np.abs(got - want))
    assert np.all(got >= 0)


@pytest.mark.parametrize("T,PER,N", SHAPES)
@pytest.mark.parametrize("window", [0, 1, 32])
def test_pooling_matches_oracle_exactly(T, PER, N, window):
    rng = np.random.default_rng(3 * T + PER + window)
    B = backbone_like(rng, N)
    n_cand = N - window
    if n_cand <= 0:
        pytest.skip("no candidates")
    got = pool_model(B, n_cand, T, PER)
    want = oracle.maxpool(B[:n_cand], 7)
    assert np.array_equal(got[:n_cand].astype(np.float64), want)
    assert np.all(got[n_cand:] == 0)


@pytest.mark.parametrize("T,PER,N", [(64, 16, 1000), (96, 16, 1531), (128, 8, 640)])
@pytest.mark.parametrize("m,nprev_layers", [(4, 4), (4, 2), (2, 2), (8, 1)])
def test_evidence_matches_oracle(T, PER, N, m, nprev_layers):
    """V = E + L + T with T the fp32 layer-ordered sum times 1/min(m, l)."""
    rng = np.random.default_rng(N + 10 * m + nprev_layers)
    E = residual_like(rng, N)
    prev = [residual_like(rng, N) for _ in range(nprev_layers)]
    r = 5
    v = np.zeros(N, dtype=F32)
    for e in prev:
        v = (v + e).astype(F32)
    v = (v * (F32(1) / F32(len(prev)))).astype(F32)
    v = (v + E).astype(F32)
    v = (v + coherence_model(E, T, PER, r)).astype(F32)
    L = oracle.coherence(E, r)
    Tm = oracle.persistence(prev, N)
    want = oracle.evidence(E, L, Tm)
    tol = 1e-5 * np.maximum(want, 1e-3) + 1e-9
    assert np.all(np.abs(v.astype(np.float64) - want) <= tol)


@pytest.mark.parametrize("N,keep,rho", [(1000, 100, 2), (1531, 300, 2), (640, 32, 3), (4096, 480, 2)])
def test_lambda_two_walks_matches_oracle(N, keep, rho):
    rng = np.random.default_rng(N + keep)
    Bt = backbone_like(rng, N)
    V = (residual_like(rng, N) * 3).astype(F32)
    want, M = oracle.calibration_lambda(Bt, V, keep, rho=rho)
    members = oracle.rank_topk(Bt, M)
    got = lambda_model(Bt, V, members)
    assert abs(got - want) <= 2e-3 * abs(want) + 1e-6, (got, want)


def test_lambda_model_catches_a_sample_std():
    """A plausible mistake (n - 1 in V's variance) moves lambda by more than
    the tolerance on a small member set, so the comparison above can see it."""
    rng = np.random.default_rng(5)
    N, keep = 200, 4
    Bt = backbone_like(rng, N)
    V = (residual_like(rng, N) * 3 + 1e-3).astype(F32)
    want, M = oracle.calibration_lambda(Bt, V, keep, rho=2)
    members = oracle.rank_topk(Bt, M)
    v = V[members].astype(np.float64)
    b = Bt[members].astype(np.float64)
    wrong = b.std() / (v.std(ddof=1) + 1e-8)
    assert abs(wrong - want) > 2e-3 * abs(want)
    assert abs(lambda_model(Bt, V, members) - want) <= 2e-3 * abs(want) + 1e-6


def test_lambda_shift_keeps_precision():
    """Pooled scores near 1 with a spread of ~1e-4: fp32 moments about zero
    lose the variance to cancellation (E[b^2] - E[b]^2 ~ 1e-8 next to an
    ulp of 1.2e-7); about the M-th value they keep it."""
    rng = np.random.default_rng(11)
    N, keep = 2000, 200
    Bt = (1.0 + 1e-4 * rng.random(N)).astype(F32)
    V = (residual_like(rng, N) * 3 + 1e-3).astype(F32)
    want, M = oracle.calibration_lambda(Bt, V, keep, rho=2)
    members = oracle.rank_topk(Bt, M)
    assert abs(lambda_model(Bt, V, members) - want) <= 2e-3 * abs(want)
    b = Bt[members].astype(F32)
    inv_m = F32(1) / F32(M)
    mb = F32(b.sum(dtype=F32)) * inv_m
    unshifted = np.sqrt(max(F32(F32((b * b).sum(dtype=F32)) * inv_m - mb * mb), F32(0)))
    v = V[members].astype(np.float64)
    assert abs(unshifted / (v.std() + 1e-8) - want) > 2e-3 * abs(want)
