"""Pins of the CPU oracle against what the paper and the mathematics fix.

Every expected value here is either a closed form worked by hand from the
definitions (exact fractions, arithmetic shown), a library routine that the
definition reduces to in a special case, an invariant, or a brute-force
recomputation on tiny inputs.  The paper prints no worked numeric example.
"""

import itertools
import math
from fractions import Fraction as F

import numpy as np
import pytest
import torch

import oracle
from oracle import Params


def _close(a, b, tol=1e-13):
    np.testing.assert_allclose(np.asarray(a, dtype=float), np.asarray(b, dtype=float),
                               rtol=0, atol=tol)


# ---------------------------------------------------------------- bf16 input

def test_bf16_widening_matches_torch():
    g = torch.Generator().manual_seed(1)
    x = torch.randn(4096, generator=g) * torch.logspace(-30, 30, 4096)
    x = torch.cat([x, torch.tensor([0.0, -0.0, 1.0, -2.5, 65504.0, 1e-40])])
    xb = x.to(torch.bfloat16)
    bits = xb.view(torch.int16).numpy().view(np.uint16)
    got = oracle.bf16_bits_to_f64(bits)
    want = xb.to(torch.float64).numpy()
    assert np.array_equal(got, want)


# ------------------------------------------------------------ Eqs. 1 and 2

def _line_keys(logits_first_coord, d=4):
    """keys k_i = (a_i, 0, ..., 0) so that q = (sqrt(d), 0, ...) has logit a_i."""
    k = np.zeros((len(logits_first_coord), d))
    k[:, 0] = logits_first_coord
    return k


def test_window_scores_closed_form_single_head():
    # d = 4 (scale 1/2), q = (2, 0, 0, 0): logit of key i = a_i = ln(i + 1),
    # so exp(logit) = 1, 2, 3.  W = 2 window queries at positions 1 and 2.
    d = 4
    k = _line_keys([math.log(1), math.log(2), math.log(3)], d)
    q = np.zeros((1, 2, d))
    q[0, :, 0] = 2.0
    B, Q = oracle.window_scores(q, k)
    # position 1 sees keys 0, 1: (1, 2)/3;  position 2 sees 0..2: (1, 2, 3)/6
    row1 = [F(1, 3), F(2, 3), F(0)]
    row2 = [F(1, 6), F(2, 6), F(3, 6)]
    want_B = [(a + b) / 2 for a, b in zip(row1, row2)]  # = 1/4, 1/2, 1/4
    assert want_B == [F(1, 4), F(1, 2), F(1, 4)]
    _close(B, [float(x) for x in want_B])
    _close(Q, [float(x) for x in row2])


def test_window_scores_closed_form_gqa_group_mean():
    # two query heads on one kv-head: head 1 uses q = (-2, 0, 0, 0), so its
    # weights are 1, 1/2, 1/3 (normalised 6/11, 3/11, 2/11 over three keys,
    # 2/3, 1/3 over two).
    d = 4
    k = _line_keys([math.log(1), math.log(2), math.log(3)], d)
    q = np.zeros((2, 2, d))
    q[0, :, 0] = 2.0
    q[1, :, 0] = -2.0
    B, Q = oracle.window_scores(q, k)
    h0 = [[F(1, 3), F(2, 3), F(0)], [F(1, 6), F(1, 3), F(1, 2)]]
    h1 = [[F(2, 3), F(1, 3), F(0)], [F(6, 11), F(3, 11), F(2, 11)]]
    want_B = [sum(r[i] for r in h0 + h1) / 4 for i in range(3)]
    want_Q = [(h0[1][i] + h1[1][i]) / 2 for i in range(3)]
    _close(B, [float(x) for x in want_B])
    _close(Q, [float(x) for x in want_Q])


def _brute_force_scores(qwin, k):
    """Full N x N causal attention of a prompt whose last W query rows are
    the window queries (other rows random), then the rows of the window."""
    G, W, d = qwin.shape
    N = k.shape[0]
    rng = np.random.default_rng(7)
    B = np.zeros(N)
    Q = np.zeros(N)
    for g in range(G):
        Qfull = rng.standard_normal((N, d))
        Qfull[N - W:] = qwin[g]
        logits = Qfull @ k.T / np.sqrt(d)
        mask = np.tril(np.ones((N, N), dtype=bool))
        logits = np.where(mask, logits, -np.inf)
        A = np.exp(logits - logits.max(axis=1, keepdims=True))
        A = A / A.sum(axis=1, keepdims=True)
        B += A[N - W:].sum(axis=0)
        Q += A[N - 1]
    return B / (G * W), Q / G


@pytest.mark.parametrize("G,W,N,d", [(1, 1, 9, 8), (1, 5, 40, 8), (3, 4, 33, 16), (2, 7, 7, 4)])
def test_window_scores_brute_force(G, W, N, d):
    rng = np.random.default_rng(G * 100 + W)
    qwin = rng.standard_normal((G, W, d)) * 1.5
    k = rng.standard_normal((N, d))
    B, Q = oracle.window_scores(qwin, k)
    Bb, Qb = _brute_force_scores(qwin, k)
    _close(B, Bb, 1e-13)
    _close(Q, Qb, 1e-13)


@pytest.mark.parametrize("G,W,N,d", [(1, 32, 640, 64), (7, 64, 700, 128), (4, 3, 50, 32)])
def test_window_scores_rows_sum_to_one(G, W, N, d):
    rng = np.random.default_rng(N)
    qwin = rng.standard_normal((G, W, d)) * 2
    k = rng.standard_normal((N, d))
    B, Q = oracle.window_scores(qwin, k)
    assert abs(B.sum() - 1) < 1e-12 and abs(Q.sum() - 1) < 1e-12
    assert (B >= 0).all() and (Q >= 0).all()


def test_window_of_one_is_last_query():
    rng = np.random.default_rng(3)
    qwin = rng.standard_normal((3, 1, 16))
    k = rng.standard_normal((30, 16))
    B, Q = oracle.window_scores(qwin, k)
    assert np.array_equal(B, Q)
    assert np.all(oracle.residual(Q, B) == 0)


def test_large_logits_stay_finite():
    # logits beyond the double exponent range (exp(800) overflows): the
    # softmax value is still well defined and must come out finite
    k = _line_keys([0.0, 500.0, 750.0, 800.0], 4)
    q = np.zeros((1, 2, 4))
    q[0, :, 0] = 2.0
    B, Q = oracle.window_scores(q, k)
    # position 3 row: exp(-800), exp(-300), exp(-50), 1 -> ~ (0, 0, e^-50, 1)
    _close(Q, [0, 0, math.exp(-50) / (1 + math.exp(-50)), 1 / (1 + math.exp(-50))], 1e-15)
    assert np.isfinite(B).all()


# ------------------------------------------------------------------ Eq. 4

def test_residual_sign_and_clip():
    Q = [0.5, 0.2, 0.3, 0.0]
    B = [0.3, 0.4, 0.3, 0.0]
    _close(oracle.residual(Q, B), [0.2, 0.0, 0.0, 0.0], 1e-16)


def test_residual_total_variation():
    rng = np.random.default_rng(5)
    qwin = rng.standard_normal((2, 6, 8))
    k = rng.standard_normal((50, 8))
    B, Q = oracle.window_scores(qwin, k)
    E = oracle.residual(Q, B)
    assert abs(E.sum() - 0.5 * np.abs(Q - B).sum()) < 1e-14
    assert (E >= 0).all()


# --------------------------------------------------------------- Eqs. 5-7

def test_coherence_hand_worked_radius_1_and_2():
    E = [1, 0, 0, 0, 0, 0, 0, 2]
    # r = 1: ends average 2 positions, interior 3
    _close(oracle.coherence(E, 1), [F(1, 2), F(1, 3), 0, 0, 0, 0, F(2, 3), F(2, 2)])
    # r = 2: |N_2(i)| = 3, 4, 5, 5, 5, 5, 4, 3
    _close(oracle.coherence(E, 2), [F(1, 3), F(1, 4), F(1, 5), 0, 0, F(2, 5), F(2, 4), F(2, 3)])


def test_coherence_special_cases():
    rng = np.random.default_rng(2)
    E = rng.random(23)
    assert np.array_equal(oracle.coherence(E, 0), E)               # P_0 = I
    _close(oracle.coherence(np.full(17, 0.25), 5), np.full(17, 0.25), 1e-16)
    _close(oracle.coherence(E, 100), np.full(23, E.mean()), 1e-15)
    L = oracle.coherence(E, 5)
    assert L.min() >= E.min() - 1e-16 and L.max() <= E.max() + 1e-16


def test_coherence_is_uniform_filter_in_interior():
    # away from the ends the operator is a plain moving average (library routine)
    rng = np.random.default_rng(4)
    E = rng.random(64)
    r = 5
    L = oracle.coherence(E, r)
    ma = np.convolve(E, np.ones(2 * r + 1) / (2 * r + 1), mode="valid")
    _close(L[r:64 - r], ma, 1e-15)


# --------------------------------------------------------------- Eqs. 8-9

def test_persistence_layer_sets():
    # P_m(l) = {j : max(1, l - m) <= j < l} in 1-based layers; 0-based below
    assert oracle.persistence_layers(0, 4) == []
    assert oracle.persistence_layers(1, 4) == [0]
    assert oracle.persistence_layers(3, 4) == [0, 1, 2]
    assert oracle.persistence_layers(6, 4) == [2, 3, 4, 5]
    assert oracle.persistence_layers(6, 0) == []
    assert oracle.persistence_layers(6, 1) == [5]


def test_persistence_values():
    _close(oracle.persistence([[1, 2], [3, 4]], 2), [2, 3])
    _close(oracle.persistence([], 3), [0, 0, 0])
    e = np.array([0.5, 0.0, 0.25])
    assert np.array_equal(oracle.persistence([e], 3), e)          # m = 1


# ----------------------------------------------------------------- Eq. 10

def test_evidence_switches():
    E, L, T = [1.0, 2.0], [10.0, 20.0], [100.0, 200.0]
    _close(oracle.evidence(E, L, T), [111, 222])
    _close(oracle.evidence(E, L, T, use_L=False), [101, 202])
    _close(oracle.evidence(E, L, T, use_E=False), [110, 220])
    _close(oracle.evidence(E, L, T, use_T=False), [11, 22])
    _close(oracle.evidence(E, L, T, False, False, False), [0, 0])


# --------------------------------------------------------------- pooling

def test_maxpool_hand_worked():
    x = [0, 5, 0, 0, 0, 0, 0, 0, 1, 0]
    _close(oracle.maxpool(x, 3), [5, 5, 5, 0, 0, 0, 0, 1, 1, 1])
    _close(oracle.maxpool(x, 1), x)
    _close(oracle.maxpool(x, 7), [5, 5, 5, 5, 5, 1, 1, 1, 1, 1])


@pytest.mark.parametrize("kernel", [1, 3, 7, 9])
def test_maxpool_is_torch_max_pool1d(kernel):
    rng = np.random.default_rng(kernel)
    x = rng.standard_normal(101)
    want = torch.nn.functional.max_pool1d(torch.tensor(x).view(1, 1, -1), kernel, 1,
                                          kernel // 2).view(-1).numpy()
    assert np.array_equal(oracle.maxpool(x, kernel), want)


# ------------------------------------------------------------------ TopK

def _dominance_subset(x, k):
    """Brute force: the unique k-subset whose members all precede all
    non-members under (value desc, index asc)."""
    n = len(x)
    found = []
    for sub in itertools.combinations(range(n), k):
        s = set(sub)
        if all((x[i] > x[j]) or (x[i] == x[j] and i < j)
               for i in s for j in range(n) if j not in s):
            found.append(sub)
    assert len(found) == 1
    return list(found[0])


@pytest.mark.parametrize("seed", range(6))
def test_topk_brute_force_with_ties(seed):
    rng = np.random.default_rng(seed)
    n = 10
    x = rng.integers(0, 4, n).astype(float)  # many ties
    for k in range(0, n + 1):
        got = oracle.rank_topk(x, k)
        assert sorted(got.tolist()) == _dominance_subset(x, k)
        # rank order: best first
        assert all((x[a] > x[b]) or (x[a] == x[b] and a < b) for a, b in zip(got, got[1:]))


def test_topk_matches_lexsort():
    rng = np.random.default_rng(11)
    x = rng.integers(0, 50, 5000).astype(float)
    order = np.lexsort((np.arange(x.size), -x))
    assert np.array_equal(oracle.rank_topk(x, 777), order[:777])


# -------------------------------------------------------------- Eqs. 12-15

def test_lambda_hand_worked():
    Bt = [4.0, 1.0, 3.0, 2.0]
    V = [0.0, 10.0, 2.0, 6.0]
    # keep 1, rho 2 -> M = 2, set = top-2 of Bt = {0, 2}
    # Std(4, 3) = 1/2, Std(0, 2) = 1 -> lambda = 1/2 (eps = 0)
    lam, M = oracle.calibration_lambda(Bt, V, keep=1, rho=2, gamma=1.0, eps=0.0)
    assert M == 2 and lam == 0.5
    lam, _ = oracle.calibration_lambda(Bt, V, keep=1, rho=2, gamma=3.0, eps=0.0)
    assert lam == 1.5
    # M capped by the candidate count: all four -> Std(Bt) = sqrt(5/4),
    # Std(V) = sqrt(14) (mean 4.5, squares 20.25+30.25+6.25+2.25 = 59/4 ... )
    lam, M = oracle.calibration_lambda(Bt, V, keep=3, rho=2, gamma=1.0, eps=0.0)
    assert M == 4
    sb = math.sqrt(sum((b - 2.5) ** 2 for b in Bt) / 4)
    sv = math.sqrt(sum((v - 4.5) ** 2 for v in V) / 4)
    assert abs(lam - sb / sv) < 1e-15


def test_lambda_postcondition_and_scaling():
    rng = np.random.default_rng(8)
    Bt = rng.random(300)
    V = rng.random(300) * 1e-3
    keep = 40
    lam, M = oracle.calibration_lambda(Bt, V, keep, 2, gamma=0.7, eps=0.0)
    sel = oracle.rank_topk(Bt, M)
    assert M == 80
    assert abs(np.std(lam * V[sel]) - 0.7 * np.std(Bt[sel])) < 1e-14
    lam2, _ = oracle.calibration_lambda(Bt * 5.0, V, keep, 2, gamma=0.7, eps=0.0)
    assert abs(lam2 - 5.0 * lam) < 1e-12 * lam2
    lam0, _ = oracle.calibration_lambda(Bt, V, keep, 2, gamma=0.0)
    assert lam0 == 0.0
    assert oracle.calibration_lambda(Bt, V, 0, 2)[0] == 0.0


def test_lambda_population_std_when_eps_matters():
    # Eq. 15's ratio cancels the Std convention except through eps; the
    # reading taken is the population Std.  Bt = (4, 3), V = (0, 2e-8):
    # Std_pop(Bt) = 1/2, Std_pop(V) = 1e-8 -> lambda = 0.5 / (1e-8 + 1e-8)
    lam, M = oracle.calibration_lambda([4.0, 3.0, 0.0], [0.0, 2e-8, 5.0], keep=1,
                                       rho=2, gamma=1.0, eps=1e-8)
    assert M == 2
    assert abs(lam - 0.5 / 2e-8) < 1e-6 * lam


# ------------------------------------------------------- whole unit, select

def _rand_unit(G=2, W=8, N=120, d=16, seed=0):
    rng = np.random.default_rng(seed)
    return rng.standard_normal((G, W, d)), rng.standard_normal((N, d))


def test_gamma_zero_is_pooled_window_score():
    q, k = _rand_unit()
    p = Params(gamma=0.0)
    out = oracle.score_unit(q, k, [], p, budget=24)
    nc = 120 - 8
    B, _ = oracle.window_scores(q, k)
    assert np.array_equal(out["Bt"][:nc], oracle.maxpool(B[:nc], 7))
    assert np.array_equal(out["S"][:nc], out["Bt"][:nc])
    assert out["lambda"] == 0.0


def test_pool_stops_at_the_window():
    # window keys aligned with the window queries get a large score; the pool
    # over the candidates [0, N - W) must not see them.
    d, N, W = 8, 40, 4
    rng = np.random.default_rng(12)
    q = rng.standard_normal((1, W, d))
    k = 0.1 * rng.standard_normal((N, d))
    k[N - W:] = 3.0 * q[0]
    B, _ = oracle.window_scores(q, k)
    nc = N - W
    assert B[nc:].min() > 10 * B[:nc].max()
    out = oracle.score_unit(q, k, [], Params(gamma=0.0), budget=W + 5)
    for i in range(nc - 3, nc):
        assert out["Bt"][i] == B[max(0, i - 3):nc].max()
    assert np.all(out["S"][nc:] == 0.0)


def test_unit_composes_the_equations():
    q, k = _rand_unit(seed=3)
    rng = np.random.default_rng(9)
    prev = [rng.random(120) * 1e-2 for _ in range(3)]
    p = Params(r=2, m=4, gamma=0.5)
    out = oracle.score_unit(q, k, prev, p, budget=30)
    B, Q = oracle.window_scores(q, k)
    E = oracle.residual(Q, B)
    L = oracle.coherence(E, 2)
    T = oracle.persistence(prev, 120)
    V = oracle.evidence(E, L, T)
    nc = 112
    Bt = oracle.maxpool(B[:nc], 7)
    lam, _ = oracle.calibration_lambda(Bt, V[:nc], 30 - 8, 2, 0.5, 1e-8)
    for name, want in [("B", B), ("Q", Q), ("E", E), ("L", L), ("T", T), ("V", V)]:
        assert np.array_equal(out[name], want), name
    assert out["lambda"] == lam
    assert np.array_equal(out["S"][:nc], Bt + lam * V[:nc])


def test_select_budget_at_least_n_keeps_everything():
    S = np.random.default_rng(0).random(50)
    for budget in (50, 51, 500):
        idx, gap = oracle.select(S, 50, 6, budget, Params())
        assert np.array_equal(idx, np.arange(50)) and gap == math.inf


def test_select_layout_and_window():
    S = np.array([0.1, 0.9, 0.3, 0.9, 0.2, 0.8, 0.0, 0.0, 0.0, 0.0])
    # W = 4: candidates 0..5, keep budget - W = 3 -> 1, 3, 5 (0.9, 0.9, 0.8)
    idx, gap = oracle.select(S, 10, 4, 7, Params())
    assert idx.tolist() == [1, 3, 5, 6, 7, 8, 9]
    assert abs(gap - (0.8 - 0.3)) < 1e-16
    idx, _ = oracle.select(S, 10, 4, 4, Params())
    assert idx.tolist() == [6, 7, 8, 9]
    with pytest.raises(ValueError):
        oracle.select(S, 10, 4, 3, Params())
    # no window reservation: top-3 over all positions
    idx, _ = oracle.select(S, 10, 4, 3, Params(keep_window=False))
    assert idx.tolist() == [1, 3, 5]


def test_gather_bitwise():
    rng = np.random.default_rng(1)
    x = rng.integers(0, 65535, (40, 8)).astype(np.uint16)
    idx = np.array([0, 5, 39, 7], dtype=np.int32)
    assert np.array_equal(oracle.gather(x, idx), x[idx])


# ---------------------------------------------------- planted evidence

def planted_case(d=64, N=256, W=16, evidence=(120, 121, 122), decoys=12, seed=0):
    """Window queries 0..W-2 share a direction u; the last query is
    orthogonal to u.  Decoy keys lie along u (logits 2 to 3 for the shared
    queries), evidence keys along the last query (logit 4 for it only)."""
    rng = np.random.default_rng(seed)
    u = rng.standard_normal(d)
    u /= np.linalg.norm(u)
    qd = rng.standard_normal(d)
    qd -= (qd @ u) * u
    qd /= np.linalg.norm(qd)
    qwin = np.zeros((1, W, d))
    qwin[0, :W - 1] = 3.0 * u + 0.3 * rng.standard_normal((W - 1, d))
    qwin[0, W - 1] = 3.0 * qd
    k = 0.3 * rng.standard_normal((N, d))
    dec = np.linspace(20, N - W - 20, decoys).astype(int)
    for j, p in enumerate(dec):  # logits 2.0 .. 3.0 for the shared queries
        k[p] = ((2.0 + j / (decoys - 1)) * np.sqrt(d) / 3.0) * u
    for p in evidence:
        k[p] = (4.0 * np.sqrt(d) / 3.0) * qd
    return qwin, k, list(evidence), dec


def test_planted_evidence_needs_calibration():
    qwin, k, ev, dec = planted_case()
    N, W, budget = k.shape[0], qwin.shape[1], 16 + 8
    kept = {}
    for gamma in (0.0, 1.0):
        p = Params(gamma=gamma)
        out = oracle.score_unit(qwin, k, [], p, budget)
        idx, _ = oracle.select(out["S"], N, W, budget, p)
        kept[gamma] = set(idx.tolist())
    assert not (set(ev) & kept[0.0]), "window score alone must dilute the evidence"
    assert set(ev) <= kept[1.0], "calibration must recover the evidence"


# ------------------------------------------------------------ host driver

def test_compress_driver_threads_and_subsets():
    from paper_2606_14782_gb300 import workloads
    wl = workloads.CONFIGS["tiny"].with_(layers=6, seq_len=200, visual=(16, 150))
    x = workloads.generate(wl, seed=3)
    qb, kb, vb = (workloads.bf16_bits(t) for t in (x.qwin, x.k, x.v))
    p = Params(m=2)
    full1 = oracle.compress(qb, kb, vb, 64, p, threads=1)
    full4 = oracle.compress(qb, kb, vb, 64, p, threads=4)
    assert full1.keys() == full4.keys()
    for key in full1:
        assert np.array_equal(full1[key]["idx"], full4[key]["idx"])
        assert full1[key]["lambda"] == full4[key]["lambda"]
    sub = oracle.compress(qb, kb, vb, 64, p, threads=2, units=[(0, 5, 1), (0, 0, 3)])
    for key in sub:
        assert np.array_equal(sub[key]["idx"], full1[key]["idx"])
        assert np.array_equal(sub[key]["Kc"], kb[key[0], key[1], key[2]][full1[key]["idx"]])
    # the persistence chain: layer 5 (m = 2) uses the residuals of layers 3, 4
    r, h = 0, 1
    Es = []
    for l in range(6):
        q = oracle.bf16_bits_to_f64(qb[r, l, h:h + 1])
        kk = oracle.bf16_bits_to_f64(kb[r, l, h])
        B, Q = oracle.window_scores(q, kk)
        Es.append(oracle.residual(Q, B))
    q = oracle.bf16_bits_to_f64(qb[r, 5, h:h + 1])
    kk = oracle.bf16_bits_to_f64(kb[r, 5, h])
    want = oracle.score_unit(q, kk, Es[3:5], p, 64)
    got = oracle.compress(qb, kb, vb, 64, p, units=[(0, 5, 1)], keep_scores=True)[(0, 5, 1)]
    assert np.array_equal(got["T"], want["T"]) and got["lambda"] == want["lambda"]


# ------------------------------------------------ PyramidKV layer budgets

def test_pyramid_budgets_hand_worked():
    # K = 10 candidates per layer on average, beta 5: K_min = 2, K_max = 18,
    # three layers -> 18, 10, 2 (+ window 4)
    assert oracle.pyramid_budgets(3, 4, 14, 5).tolist() == [22, 14, 6]
    # a single layer keeps the uniform budget
    assert oracle.pyramid_budgets(1, 8, 64, 20).tolist() == [64]


@pytest.mark.parametrize("layers,window,budget,beta", [(28, 64, 1024, 20), (32, 32, 64, 20),
                                                     (28, 32, 256, 5), (7, 16, 100, 3)])
def test_pyramid_budgets_properties(layers, window, budget, beta):
    b = oracle.pyramid_budgets(layers, window, budget, beta)
    K = budget - window
    assert b[0] - window == 2 * K - K // beta
    assert b[-1] - window == K // beta
    assert all(x >= y for x, y in zip(b, b[1:]))          # pyramid: never grows with depth
    assert all(x >= window for x in b)
    # the schedule spends the uniform budget, never more (floor per layer)
    assert layers * K - (layers - 1) <= int((b - window).sum()) <= layers * K


def test_compress_accepts_layer_budgets():
    from paper_2606_14782_gb300 import workloads
    wl = workloads.CONFIGS["tiny"].with_(layers=3, seq_len=300, visual=(16, 280))
    x = workloads.generate(wl, seed=2)
    qb, kb, vb = (workloads.bf16_bits(t) for t in (x.qwin, x.k, x.v))
    budgets = oracle.pyramid_budgets(3, wl.window, 64, 4)
    res = oracle.compress(qb, kb, vb, budgets, oracle.Params(), threads=2)
    for (r, l, h), o in res.items():
        assert o["idx"].size == budgets[l]
        # each layer matches a uniform run at that layer's budget
    one = oracle.compress(qb, kb, vb, int(budgets[1]), oracle.Params(), threads=2,
                          units=[(0, 1, 2)])
    assert np.array_equal(one[(0, 1, 2)]["idx"], res[(0, 1, 2)]["idx"])


# ---------------------------------------------- AdaKV adaptive head budgets

def test_adaptive_alpha_one_is_per_head_topk():
    rng = np.random.default_rng(21)
    H, N, W, budget = 3, 60, 6, 20
    S = rng.random((H, N))
    S[:, N - W:] = 0.0
    kept = oracle.select_adaptive(S, W, budget, 1.0, Params())
    for h in range(H):
        want, _ = oracle.select(S[h], N, W, budget, Params())
        assert np.array_equal(kept[h], want)


def test_adaptive_single_head_is_topk():
    rng = np.random.default_rng(22)
    S = rng.random((1, 50))
    for alpha in (0.0, 0.2, 0.5):
        kept = oracle.select_adaptive(S, 5, 17, alpha, Params())
        want, _ = oracle.select(S[0], 50, 5, 17, Params())
        assert np.array_equal(kept[0], want)


def test_adaptive_hand_worked():
    # two heads, 6 candidates each + window 2, budget 5 -> K = 3, H K = 6;
    # alpha 1/3 -> g = 1 guaranteed per head, 4 slots jointly.
    S = np.array([[9, 8, 7, 6, 0.5, 0.4, 0, 0],
                  [5, 1, 1, 1, 1, 1, 0, 0]], dtype=float)
    kept = oracle.select_adaptive(S, 2, 5, 1 / 3, Params())
    # guaranteed: head 0 -> 0 (9), head 1 -> 0 (5); jointly the best of the
    # rest: 8, 7, 6 (head 0) then the first 1 of head 1 (ties: lower position)
    assert kept[0].tolist() == [0, 1, 2, 3, 6, 7]
    assert kept[1].tolist() == [0, 1, 6, 7]


@pytest.mark.parametrize("seed", range(4))
def test_adaptive_invariants(seed):
    rng = np.random.default_rng(30 + seed)
    H, N, W, budget, alpha = 4, 80, 8, 24, 0.25
    S = rng.integers(0, 6, (H, N)).astype(float)  # ties everywhere
    kept = oracle.select_adaptive(S, W, budget, alpha, Params())
    K, g = budget - W, int(alpha * (budget - W))
    cand = [k[:-W] for k in kept]
    assert sum(len(c) for c in cand) == H * K
    assert all(len(c) >= g for c in cand)
    for k in kept:
        assert np.all(np.diff(k) > 0) and np.array_equal(k[-W:], np.arange(N - W, N))
    # every jointly chosen candidate dominates every candidate left out
    # (score desc, head asc, position asc), guaranteed ones aside
    guaranteed = set()
    for h in range(H):
        for i in oracle.rank_topk(S[h, :N - W], g):
            guaranteed.add((h, int(i)))
    chosen = {(h, int(i)) for h in range(H) for i in cand[h]} - guaranteed
    left = {(h, i) for h in range(H) for i in range(N - W)} - {(h, int(i)) for h in range(H) for i in cand[h]}
    key = lambda t: (-S[t[0], t[1]], t[0], t[1])
    assert max(key(t) for t in chosen) < min(key(t) for t in left)


# ------------------------------------------ ablation / sensitivity sweep

def _sweep_case(seed=5):
    from paper_2606_14782_gb300 import workloads
    wl = workloads.CONFIGS["tiny"].with_(layers=5, seq_len=260, visual=(16, 220))
    x = workloads.generate(wl, seed=seed)
    return wl, tuple(workloads.bf16_bits(t) for t in (x.qwin, x.k, x.v))


def test_sweep_all_terms_off_is_the_backbone_score():
    # V = 0 when E, L and T are all switched off (Eq. 10), so S = B~ + lambda 0
    # = B~ (Eq. 16): the same selection as gamma = 0 with every term on.
    wl, (qb, kb, vb) = _sweep_case()
    off, g0 = oracle.sweep(qb, kb, vb, 48, [dict(use_E=0, use_L=0, use_T=0), dict(gamma=0.0)],
                           threads=4)
    for key in off:
        assert np.array_equal(off[key]["idx"], g0[key]["idx"]), key


def test_sweep_m_zero_is_no_persistence():
    # P_0(l) is empty for every l (Eq. 8), so T = 0 (Eq. 9) and m = 0 selects
    # what use_T = 0 selects, with the same lambda.
    wl, (qb, kb, vb) = _sweep_case()
    m0, noT = oracle.sweep(qb, kb, vb, 48, [dict(m=0), dict(use_T=0)], threads=4)
    for key in m0:
        assert np.array_equal(m0[key]["idx"], noT[key]["idx"]), key
        assert m0[key]["lambda"] == noT[key]["lambda"]


def test_sweep_radius_covering_the_prompt_makes_L_a_constant():
    # r >= N - 1: every window of Eq. 6 is the whole prompt, L is the constant
    # mean of E, so V is the no-L evidence shifted by a constant: Std over M
    # and hence lambda (Eq. 15) are unchanged and S is shifted uniformly.
    wl, (qb, kb, vb) = _sweep_case()
    big, noL = oracle.sweep(qb, kb, vb, 48, [dict(r=wl.seq_len), dict(use_L=0)], threads=4)
    for key in big:
        assert np.array_equal(big[key]["idx"], noL[key]["idx"]), key
        assert abs(big[key]["lambda"] - noL[key]["lambda"]) <= 1e-9 * abs(noL[key]["lambda"])


def test_sweep_first_layer_ignores_m():
    # layer 0 has no preceding layer: T = 0 whatever m is (Eq. 8).
    wl, (qb, kb, vb) = _sweep_case()
    res = oracle.sweep(qb, kb, vb, 48, [dict(m=m) for m in (0, 1, 4, 8)], threads=4,
                       units=[(0, 0, h) for h in range(wl.kv_heads)])
    for key in res[0]:
        for other in res[1:]:
            assert np.array_equal(res[0][key]["idx"], other[key]["idx"]), key


def test_sweep_variant_grid_is_distinct_and_covers_the_study():
    from paper_2606_14782_gb300 import workloads
    full = dict(use_E=1, use_L=1, use_T=1, m=4, r=5)
    seen = set()
    for v in workloads.SWEEP_VARIANTS:
        k = tuple(sorted({**full, **v}.items()))
        assert k not in seen, v
        seen.add(k)
    comps = {(d["use_E"], d["use_L"], d["use_T"]) for d in map(dict, seen)}
    assert comps == {(1, 1, 1), (0, 0, 0), (1, 0, 1), (1, 1, 0), (0, 1, 1)}
    ms = {d["m"] for d in map(dict, seen) if d["r"] == 5 and d["use_T"]}
    rs = {d["r"] for d in map(dict, seen) if d["m"] == 4 and d["use_L"]}
    assert ms == {2, 4, 6, 8} and rs == {3, 5, 7, 9}
