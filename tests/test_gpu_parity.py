"""CUDA path (through the C ABI) against the CPU oracle on the same seeded
inputs: every configuration of the paper-shaped workloads, edge cases, the
layer-by-layer path and the host-buffer path."""

import os

import numpy as np
import pytest
import torch

import oracle
from paper_2606_14782_gb300 import bacon, build, workloads
from parity import ATOL, RTOL, check_scores, check_selection, record_swaps

pytestmark = pytest.mark.gpu

THREADS = os.cpu_count() or 4


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    bacon.load()


def oracle_params(**kw):
    return oracle.Params(**kw)


def run_gpu(wl, x, budget, **kw):
    p = bacon.default_params(keep_scores=1, max_seq_len=max(wl.seq_len, 64),
                             max_requests=wl.requests)
    for k, v in kw.items():
        setattr(p, k, v)
    ctx = bacon.Context(wl.layers, wl.kv_heads, wl.q_heads, wl.head_dim, wl.window, wl.pool,
                        budget, params=p)
    ko, vo, idx = ctx.compress_all_layers(x.qwin, x.k, x.v, budget)
    ctx.sync()
    R, Ly, H, N = wl.requests, wl.layers, wl.kv_heads, wl.seq_len
    out = {"Kc": ko.cpu(), "Vc": vo.cpu(), "idx": idx.cpu().numpy()}
    for kind in ("B", "Q", "E", "V", "Bpool", "S"):
        out[kind] = ctx.scores(kind).cpu().numpy().reshape(R, Ly, H, N)
    out["lambda"] = ctx.scores("lambda").cpu().numpy().reshape(R, Ly, H)
    ctx.close()
    return out


def compare(wl, x, budget, gpu, orc, report=None, case=None, path="whole step"):
    """Element-wise comparison of every oracle unit; returns the swap count.
    With `case`, every boundary swap goes to the session's swap log."""
    N, W = wl.seq_len, wl.window
    kb = workloads.bf16_bits(x.k)
    vb = workloads.bf16_bits(x.v)
    swaps = 0
    worst = 0.0
    log = []
    n_units = 0
    kw = orc.get("_keep_window", True)
    for key, o in orc.items():
        if not isinstance(key, tuple):
            continue
        r, l, h = key
        where = f"unit ({r},{l},{h})"
        for name, okey in (("B", "B"), ("Q", "Q"), ("E", "E"), ("V", "V"), ("Bpool", "Bt"),
                           ("S", "S")):
            e, _ = check_scores(f"{where} {name}", gpu[name][r, l, h], o[okey])
            worst = max(worst, e)
        lam_g, lam_o = float(gpu["lambda"][r, l, h]), o["lambda"]
        assert abs(lam_g - lam_o) <= RTOL * abs(lam_o) + ATOL, (where, lam_g, lam_o)
        gi = gpu["idx"][r, l, h]
        swaps += check_selection(gi, o["idx"], o["S"], N, W, budget, keep_window=kw, log=log,
                                 unit=key)
        n_units += 1
        # compacted cache: bit-exact against the GPU's own indices
        Kc = gpu["Kc"][r, l, h].view(torch.int16).numpy().view(np.uint16)
        Vc = gpu["Vc"][r, l, h].view(torch.int16).numpy().view(np.uint16)
        assert np.array_equal(Kc, kb[r, l, h][gi]), where
        assert np.array_equal(Vc, vb[r, l, h][gi]), where
    if report is not None:
        report.update(swaps=swaps, worst_abs=worst)
    if case is not None:
        kept = min(budget, N)
        record_swaps(case, wl.name, budget, n_units, kept - (W if kw else 0), log, path)
    return swaps


def oracle_run(wl, x, budget, units=None, adaptive_alpha=None, **kw):
    qb = workloads.bf16_bits(x.qwin)
    kb = workloads.bf16_bits(x.k)
    vb = workloads.bf16_bits(x.v)
    p = oracle_params(pool_kernel=wl.pool, **kw)
    res = oracle.compress(qb, kb, vb, budget, p, threads=THREADS, units=units, keep_scores=True,
                          adaptive_alpha=adaptive_alpha)
    res["_keep_window"] = p.keep_window
    return res


# ------------------------------------------------------------ configs

def test_tiny_full_parity():
    wl = workloads.CONFIGS["tiny"]
    x = workloads.generate(wl, seed=0, device="cuda")
    gpu = run_gpu(wl, x, 64)
    orc = oracle_run(wl, x, 64)
    rep = {}
    compare(wl, x, 64, gpu, orc, rep, case="tiny B=64")
    assert rep["swaps"] <= 2
    # rows of the window softmax sum to one per unit
    np.testing.assert_allclose(gpu["B"].sum(-1), 1.0, atol=1e-4)
    np.testing.assert_allclose(gpu["Q"].sum(-1), 1.0, atol=1e-4)


@pytest.mark.parametrize("budget", [64, 128, 256])
def test_llava_full_parity(budget):
    wl = workloads.CONFIGS["llava"]
    x = workloads.generate(wl, seed=0, device="cuda")
    gpu = run_gpu(wl, x, budget)
    orc = oracle_run(wl, x, budget)
    swaps = compare(wl, x, budget, gpu, orc, case=f"llava B={budget}")
    units = wl.layers * wl.kv_heads
    assert swaps <= max(2, units * (budget - wl.window) // 1000)


FULL_SIZE = [("qwen-img", 128), ("qwen-img", 256), ("qwen-img", 512), ("video", 326),
             ("video", 652), ("gui", 256), ("gui", 1024)]


@pytest.mark.parametrize("name,budget", FULL_SIZE)
def test_full_size_parity(name, budget):
    """Full-size launch (every request, layer and kv-head in one call, as the
    benchmark runs it), compared with the oracle at every unit: scores
    element by element, selections up to logged boundary swaps, gathers bit
    for bit."""
    wl = workloads.CONFIGS[name]
    x = workloads.generate(wl, seed=0, device="cuda")
    gpu = run_gpu(wl, x, budget)
    orc = oracle_run(wl, x, budget)
    assert len([k for k in orc if isinstance(k, tuple)]) == wl.requests * wl.layers * wl.kv_heads
    swaps = compare(wl, x, budget, gpu, orc, case=f"{name} B={budget}")
    units = wl.requests * wl.layers * wl.kv_heads
    assert swaps <= max(2, units * (budget - wl.window) // 1000)
    # whole-launch properties at every unit
    np.testing.assert_allclose(gpu["B"].sum(-1), 1.0, atol=2e-4)
    np.testing.assert_allclose(gpu["Q"].sum(-1), 1.0, atol=2e-4)
    assert (gpu["E"] >= 0).all() and (gpu["V"] >= 0).all() and (gpu["lambda"] >= 0).all()
    idx = gpu["idx"]
    assert (np.diff(idx, axis=-1) > 0).all()
    assert (idx[..., -wl.window:] == np.arange(wl.seq_len - wl.window, wl.seq_len)).all()


# --------------------------------------------------------- edge cases

EDGE = [
    # name, overrides of the tiny workload, budget, oracle/GPU parameter overrides
    ("ragged", dict(seq_len=777, visual=(16, 700)), 100, {}),
    ("ragged_gqa_d128", dict(seq_len=1000, q_heads=6, kv_heads=2, head_dim=128,
                             visual=(16, 900)), 96, {}),
    ("odd_window", dict(seq_len=300, window=5, q_heads=6, kv_heads=2, visual=(16, 280)), 40, {}),
    ("window_one", dict(seq_len=200, window=1, visual=(16, 190)), 30, {}),
    ("no_candidates", dict(seq_len=32, visual=(0, 0), planted=0), 32, {}),
    ("budget_is_window", dict(seq_len=400, visual=(16, 380)), 32, {}),
    ("budget_above_n", dict(seq_len=300, visual=(16, 280)), 500, {}),
    ("gamma_zero", dict(seq_len=640), 64, dict(gamma=0.0)),
    ("no_window_reserve", dict(seq_len=500, visual=(16, 460)), 64, dict(keep_window=False)),
    ("ablate_L", dict(seq_len=640, layers=6), 64, dict(use_L=False)),
    ("ablate_E", dict(seq_len=640, layers=6), 64, dict(use_E=False)),
    ("ablate_T", dict(seq_len=640, layers=6), 64, dict(use_T=False)),
    ("r0_m1", dict(seq_len=640, layers=4), 64, dict(r=0, m=1)),
    ("m0_r9", dict(seq_len=640, layers=4), 64, dict(m=0, r=9)),
    ("m8_deep", dict(seq_len=256, layers=12, visual=(16, 200)), 48, dict(m=8)),
    ("pool1_rho3", dict(seq_len=640), 64, dict(rho=3)),
    ("two_requests", dict(seq_len=513, requests=2, visual=(16, 480)), 80, {}),
    ("long_tail_chunks", dict(seq_len=3000, layers=2, visual=(16, 2900)), 200, {}),
    # more chunks than SMs, units of 9 tiles: each CTA's range of chunks
    # crosses unit boundaries with an odd number of tiles per unit
    ("odd_tiles_many_units", dict(seq_len=1152, layers=24, q_heads=8, kv_heads=8,
                                  visual=(16, 1100)), 100, {}),
    # the largest window block the kernels take: G W = 512 rows at d = 128
    ("rows_512_d128", dict(seq_len=1500, layers=2, q_heads=16, kv_heads=2, head_dim=128,
                           window=64, visual=(16, 1400)), 200, {}),
    # the longest prompt the library takes (24 positions per calibration
    # thread), and a ragged one just below it with the GQA 7:1, W = 64 window
    # blocks of the paper's long shapes
    ("max_prompt", dict(seq_len=24576, layers=2, q_heads=8, kv_heads=2, head_dim=128,
                        window=32, visual=(16, 24000)), 1024, {}),
    ("near_max_gqa7", dict(seq_len=24000, layers=2, q_heads=14, kv_heads=2, head_dim=128,
                           window=64, visual=(16, 23500)), 1024, {}),
]


@pytest.mark.parametrize("name,over,budget,pk", EDGE, ids=[e[0] for e in EDGE])
def test_edge_cases(name, over, budget, pk):
    wl = workloads.CONFIGS["tiny"].with_(**over)
    if name == "pool1_rho3":
        wl = wl.with_(pool=1)
    x = workloads.generate(wl, seed=1, device="cuda")
    gpu_kw = {k: (int(v) if isinstance(v, bool) else v) for k, v in pk.items()}
    gpu = run_gpu(wl, x, budget, **gpu_kw)
    orc = oracle_run(wl, x, budget, **pk)
    compare(wl, x, budget, gpu, orc, case=f"edge {name} B={budget}")
    if name == "gamma_zero":
        nc = wl.seq_len - wl.window
        assert np.array_equal(gpu["S"][..., :nc], gpu["Bpool"][..., :nc])
    if name == "window_one":
        assert np.array_equal(gpu["B"], gpu["Q"]) and not gpu["E"].any()
    if name == "budget_above_n":
        assert (gpu["idx"] == np.arange(wl.seq_len)).all()


# ---------------------------------------------------- planted evidence

def test_planted_evidence_on_gpu():
    from test_oracle_pins import planted_case
    qwin, k, ev, _ = planted_case()
    W, d = qwin.shape[1], qwin.shape[2]
    N = k.shape[0]
    wl = workloads.CONFIGS["tiny"].with_(layers=1, q_heads=1, kv_heads=1, head_dim=d,
                                         seq_len=N, window=W)
    qt = torch.tensor(qwin, dtype=torch.float32).to(torch.bfloat16).reshape(1, 1, 1, W, d)
    kt = torch.tensor(k, dtype=torch.float32).to(torch.bfloat16).reshape(1, 1, 1, N, d)
    x = workloads.Inputs(qt.cuda(), kt.cuda(), kt.clone().cuda(), None)
    budget = W + 8
    kept = {}
    for gamma in (0.0, 1.0):
        gpu = run_gpu(wl, x, budget, gamma=gamma)
        orc = oracle_run(wl, x, budget, gamma=gamma)
        compare(wl, x, budget, gpu, orc)
        kept[gamma] = set(gpu["idx"][0, 0, 0].tolist())
    assert not (set(ev) & kept[0.0])
    assert set(ev) <= kept[1.0]


# --------------------------------------------- other entry points

def test_layer_path_matches_whole_step():
    wl = workloads.CONFIGS["tiny"].with_(layers=7, q_heads=8, kv_heads=2, seq_len=900,
                                         visual=(16, 850))
    x = workloads.generate(wl, seed=2, device="cuda")
    budget = 96
    whole = run_gpu(wl, x, budget)
    p = bacon.default_params(max_seq_len=wl.seq_len, max_requests=1)
    ctx = bacon.Context(wl.layers, wl.kv_heads, wl.q_heads, wl.head_dim, wl.window, wl.pool,
                        budget, params=p)
    st = bacon.State(ctx)
    for l in range(wl.layers):
        S = st.score_layer(l, x.qwin[0, l], x.k[0, l], scores_out=True)
        idx = st.select(budget, wl.seq_len)
        ko, vo = ctx.compact(x.k[0, l], x.v[0, l], idx)
        ctx.sync()
        assert np.array_equal(idx.cpu().numpy(), whole["idx"][0, l]), l
        assert np.array_equal(S.cpu().numpy(), whole["S"][0, l]), l
        assert torch.equal(ko.cpu(), whole["Kc"][0, l]) and torch.equal(vo.cpu(), whole["Vc"][0, l])
    # out-of-order layer and a second state's select before scoring
    with pytest.raises(bacon.BaconError, match="ESTATE"):
        st.score_layer(3, x.qwin[0, 3], x.k[0, 3])
    st2 = bacon.State(ctx)
    with pytest.raises(bacon.BaconError, match="ESTATE"):
        st2.select(budget, wl.seq_len)
    st2.close()
    st.reset()
    st.score_layer(0, x.qwin[0, 0], x.k[0, 0])
    st.close()
    ctx.close()


@pytest.mark.parametrize("name,layers", [("gui", 3), ("qwen-img", 5)])
def test_layer_path_matches_whole_step_at_paper_shapes(name, layers):
    """The layer-by-layer calls (score, select, compact) against the whole
    step, bit for bit, at the paper shapes whose window kernels are compiled
    as specialised plans (jobs per tile, job sizes and window as constants)."""
    wl = workloads.CONFIGS[name].with_(layers=layers, requests=1)
    x = workloads.generate(wl, seed=12, device="cuda")
    budget = max(wl.budgets)
    whole = run_gpu(wl, x, budget)
    p = bacon.default_params(max_seq_len=wl.seq_len, max_requests=1)
    ctx = bacon.Context(wl.layers, wl.kv_heads, wl.q_heads, wl.head_dim, wl.window, wl.pool,
                        budget, params=p)
    st = bacon.State(ctx)
    for l in range(wl.layers):
        S = st.score_layer(l, x.qwin[0, l], x.k[0, l], scores_out=True)
        idx = st.select(budget, wl.seq_len)
        ko, vo = ctx.compact(x.k[0, l], x.v[0, l], idx)
        ctx.sync()
        assert np.array_equal(idx.cpu().numpy(), whole["idx"][0, l]), l
        assert np.array_equal(S.cpu().numpy(), whole["S"][0, l]), l
        assert torch.equal(ko.cpu(), whole["Kc"][0, l]) and torch.equal(vo.cpu(), whole["Vc"][0, l])
    st.close()
    ctx.close()


def test_host_path_matches_device_path_at_gui_shape():
    """bacon_compress_host (page-locked inputs) against the device path, bit
    for bit, at the GUI shape (specialised window plans) with two layers."""
    wl = workloads.CONFIGS["gui"].with_(layers=2, requests=2)
    x = workloads.generate(wl, seed=13, device="cuda")
    budget = max(wl.budgets)
    dev = run_gpu(wl, x, budget)
    p = bacon.default_params(max_seq_len=wl.seq_len, max_requests=2)
    ctx = bacon.Context(wl.layers, wl.kv_heads, wl.q_heads, wl.head_dim, wl.window, wl.pool,
                        budget, params=p)
    qh, kh, vh = (t.cpu().pin_memory() for t in (x.qwin, x.k, x.v))
    ko, vo, idx = ctx.compress_host(qh, kh, vh, budget)
    assert np.array_equal(idx.numpy(), dev["idx"])
    assert torch.equal(ko, dev["Kc"]) and torch.equal(vo, dev["Vc"])
    ctx.close()


@pytest.mark.parametrize("pinned", ["all", "none", "values_pageable"])
def test_host_path_matches_device_path(pinned):
    """Page-locked values are gathered in place, pageable ones uploaded."""
    wl = workloads.CONFIGS["tiny"].with_(requests=2, layers=3, seq_len=700, visual=(16, 650))
    x = workloads.generate(wl, seed=4, device="cuda")
    budget = 80
    dev = run_gpu(wl, x, budget)
    p = bacon.default_params(max_seq_len=wl.seq_len, max_requests=2)
    ctx = bacon.Context(wl.layers, wl.kv_heads, wl.q_heads, wl.head_dim, wl.window, wl.pool,
                        budget, params=p)
    qh, kh, vh = (t.cpu() for t in (x.qwin, x.k, x.v))
    if pinned == "all":
        qh, kh, vh = (t.pin_memory() for t in (qh, kh, vh))
    elif pinned == "values_pageable":
        qh, kh = qh.pin_memory(), kh.pin_memory()
    ko, vo, idx = ctx.compress_host(qh, kh, vh, budget)
    assert np.array_equal(idx.numpy(), dev["idx"])
    assert torch.equal(ko, dev["Kc"]) and torch.equal(vo, dev["Vc"])
    # a second call reuses the staging buffers
    ko2, _, idx2 = ctx.compress_host(qh, kh, vh, budget)
    assert torch.equal(ko2, ko) and torch.equal(idx2, idx)
    # switching between in-place and uploaded values on one context
    other = vh.pin_memory() if not vh.is_pinned() else vh.clone()
    _, vo3, idx3 = ctx.compress_host(qh, kh, other, budget)
    assert torch.equal(vo3, dev["Vc"]) and np.array_equal(idx3.numpy(), dev["idx"])
    ctx.close()


def test_out_of_range_gather_index_is_reported():
    wl = workloads.CONFIGS["tiny"]
    x = workloads.generate(wl, seed=0, device="cuda")
    ctx = bacon.Context(wl.layers, wl.kv_heads, wl.q_heads, wl.head_dim, wl.window, wl.pool, 64)
    idx = torch.zeros((wl.kv_heads, 8), dtype=torch.int32, device="cuda")
    idx[1, 3] = wl.seq_len + 5  # checked and skipped by the kernel
    ctx.compact(x.k[0, 0], x.v[0, 0], idx)
    with pytest.raises(bacon.BaconError, match="gather index"):
        ctx.sync()
    ctx.sync()  # the flag is cleared once reported
    ctx.close()


def test_invalid_calls_on_gpu():
    wl = workloads.CONFIGS["tiny"]
    x = workloads.generate(wl, seed=0, device="cuda")
    ctx = bacon.Context(wl.layers, wl.kv_heads, wl.q_heads, wl.head_dim, wl.window, wl.pool, 64,
                        max_seq_len=640, max_requests=1)
    with pytest.raises(bacon.BaconError, match="EINVAL"):
        ctx.compress_all_layers(x.qwin, x.k, x.v, 16)  # budget below the window
    big = workloads.CONFIGS["tiny"].with_(seq_len=700)
    xb = workloads.generate(big, seed=0, device="cuda")
    with pytest.raises(bacon.BaconError, match="max_seq_len"):
        ctx.compress_all_layers(xb.qwin, xb.k, xb.v, 64)
    with pytest.raises(bacon.BaconError, match="aligned"):
        ctx.compact(x.k[0, 0].flatten()[1:].view(-1)[: 4 * 639 * 64].view(4, 639, 64),
                    x.v[0, 0], torch.zeros((4, 8), dtype=torch.int32, device="cuda"))
    ctx.close()


@pytest.mark.parametrize("over,one_pass", [
    # 4 query heads per kv head x 32 window rows = 128 rows: the two passes
    (dict(q_heads=16, kv_heads=4), False),
    # 32 window rows, 640 tokens: logits resident in tensor memory, one pass
    ({}, True),
])
def test_profile_hooks_count_launches(over, one_pass):
    wl = workloads.CONFIGS["tiny"].with_(**over)
    x = workloads.generate(wl, seed=0, device="cuda")
    ctx = bacon.Context(wl.layers, wl.kv_heads, wl.q_heads, wl.head_dim, wl.window, wl.pool, 64)
    ctx.profile(True)
    for _ in range(3):
        ctx.compress_all_layers(x.qwin, x.k, x.v, 64)
    prof = ctx.profile_read()
    skipped = {"window_stats", "window_combine"} if one_pass else set()
    for name, (ms, n) in prof.items():
        assert n == (0 if name in skipped else 3), (name, n)
        assert (ms == 0) if name in skipped else (ms > 0), (name, ms)
    ctx.close()


# ------------------------------------------------ per-layer budgets (PyramidKV)

def _compare_layer_budgets(wl, x, budgets, ko, vo, ix, orc, log=None):
    N, W = wl.seq_len, wl.window
    kb = workloads.bf16_bits(x.k)
    vb = workloads.bf16_bits(x.v)
    swaps = 0
    for key, o in orc.items():
        if not isinstance(key, tuple):
            continue
        r, l, h = key
        gi = ix[r][l][h].cpu().numpy()
        swaps += check_selection(gi, o["idx"], o["S"], N, W, int(budgets[l]), log=log, unit=key)
        Kc = ko[r][l][h].cpu().view(torch.int16).numpy().view(np.uint16)
        Vc = vo[r][l][h].cpu().view(torch.int16).numpy().view(np.uint16)
        assert np.array_equal(Kc, kb[r, l, h][gi]) and np.array_equal(Vc, vb[r, l, h][gi])
    return swaps


@pytest.mark.parametrize("name,budget,beta", [("tiny", 64, 4), ("llava", 128, 20),
                                              ("qwen-img", 256, 20)])
def test_pyramid_layer_budgets_parity(name, budget, beta):
    wl = workloads.CONFIGS[name].with_(layers=min(8, workloads.CONFIGS[name].layers))
    x = workloads.generate(wl, seed=3, device="cuda")
    budgets = bacon.pyramid_budgets(wl.layers, wl.window, budget, beta)
    assert budgets == oracle.pyramid_budgets(wl.layers, wl.window, budget, beta).tolist()
    p = bacon.default_params(keep_scores=1, max_seq_len=wl.seq_len, max_requests=wl.requests)
    ctx = bacon.Context(wl.layers, wl.kv_heads, wl.q_heads, wl.head_dim, wl.window, wl.pool,
                        budget, params=p)
    ko, vo, ix = ctx.compress_layer_budgets(x.qwin, x.k, x.v, budgets)
    ctx.sync()
    S = ctx.scores("S").cpu().numpy().reshape(wl.requests, wl.layers, wl.kv_heads, wl.seq_len)
    ctx.close()
    units = None if name == "tiny" else [(0, l, h) for l in (0, 3, wl.layers - 1)
                                           for h in (0, wl.kv_heads - 1)]
    orc = oracle_run(wl, x, budgets, units=units)
    for key, o in orc.items():
        if isinstance(key, tuple):
            check_scores(f"S {key}", S[key], o["S"])
    _compare_layer_budgets(wl, x, budgets, ko, vo, ix, orc)
    # the first layer keeps the most tokens, the last the fewest
    assert ix[0][0].shape[1] >= ix[0][-1].shape[1]


PYRAMID_FULL = [("qwen-img", 512, 20), ("video", 652, 20), ("gui", 1024, 20)]


@pytest.mark.parametrize("name,budget,beta", PYRAMID_FULL)
def test_pyramid_layer_budgets_full_size(name, budget, beta):
    """Per-layer budgets on the full-size launch (every request, layer and
    kv-head in one call), every unit against the oracle: S element by
    element, selections up to logged boundary swaps, gathers bit for bit."""
    wl = workloads.CONFIGS[name]
    x = workloads.generate(wl, seed=3, device="cuda")
    budgets = bacon.pyramid_budgets(wl.layers, wl.window, budget, beta)
    assert budgets == oracle.pyramid_budgets(wl.layers, wl.window, budget, beta).tolist()
    p = bacon.default_params(keep_scores=1, max_seq_len=wl.seq_len, max_requests=wl.requests)
    ctx = bacon.Context(wl.layers, wl.kv_heads, wl.q_heads, wl.head_dim, wl.window, wl.pool,
                        budget, params=p)
    ko, vo, ix = ctx.compress_layer_budgets(x.qwin, x.k, x.v, budgets)
    ctx.sync()
    R, Ly, H, N = wl.requests, wl.layers, wl.kv_heads, wl.seq_len
    S = ctx.scores("S").cpu().numpy().reshape(R, Ly, H, N)
    Bp = ctx.scores("Bpool").cpu().numpy().reshape(R, Ly, H, N)
    ctx.close()
    orc = oracle_run(wl, x, budgets)
    units = [k for k in orc if isinstance(k, tuple)]
    assert len(units) == R * Ly * H
    for key in units:
        check_scores(f"S {key}", S[key], orc[key]["S"])
        check_scores(f"Bpool {key}", Bp[key], orc[key]["Bt"])
    log = []
    swaps = _compare_layer_budgets(wl, x, budgets, ko, vo, ix, orc, log=log)
    record_swaps(f"{name} pyramid B={budget} beta={beta}", wl.name, [int(b) for b in budgets],
                 len(units), [int(min(b, N)) - wl.window for b in budgets], log, "layer budgets")
    assert swaps <= max(2, len(units) * (budget - wl.window) // 1000)
    # budgets fall from the first layer to the last and are kept exactly
    for r in range(R):
        for l in range(Ly):
            assert tuple(ix[r][l].shape) == (H, min(budgets[l], N))


def test_uniform_layer_budgets_match_whole_step():
    wl = workloads.CONFIGS["tiny"].with_(layers=4, requests=2, seq_len=700, visual=(16, 650))
    x = workloads.generate(wl, seed=6, device="cuda")
    whole = run_gpu(wl, x, 96)
    p = bacon.default_params(max_seq_len=wl.seq_len, max_requests=2)
    ctx = bacon.Context(wl.layers, wl.kv_heads, wl.q_heads, wl.head_dim, wl.window, wl.pool, 96,
                        params=p)
    ko, vo, ix = ctx.compress_layer_budgets(x.qwin, x.k, x.v, [96] * wl.layers)
    ctx.sync()
    for r in range(2):
        for l in range(wl.layers):
            assert np.array_equal(ix[r][l].cpu().numpy(), whole["idx"][r, l])
            assert torch.equal(ko[r][l].cpu(), whole["Kc"][r, l])
    ctx.close()


# ------------------------------------------------ adaptive head budgets (AdaKV)

def _head_threshold(S_cand, k):
    order = np.lexsort((np.arange(S_cand.size), -S_cand))
    return S_cand[order[k - 1]] if k > 0 else np.inf


def _adaptive_parity(wl, x, budget, alpha, case=None):
    """AdaKV-style head budgets through the C ABI against the oracle at every
    unit of the launch: S per token, per-head counts, each head's kept set
    ascending with its window, K/V bit for bit, and the joint kept set of
    each (request, layer) equal up to swaps whose oracle scores lie within
    the tolerance of one of the thresholds that decide it (a head's
    guaranteed-share boundary or the joint boundary).  Returns the swaps."""
    N, W, H = wl.seq_len, wl.window, wl.kv_heads
    p = bacon.default_params(keep_scores=1, max_seq_len=N, max_requests=wl.requests)
    ctx = bacon.Context(wl.layers, H, wl.q_heads, wl.head_dim, wl.window, wl.pool, budget,
                        params=p)
    ko, vo, ix, counts = ctx.compress_adaptive(x.qwin, x.k, x.v, budget, alpha)
    ctx.sync()
    S = ctx.scores("S").cpu().numpy().reshape(wl.requests, wl.layers, H, N)
    ctx.close()
    ko, vo, ix, counts = ko.cpu(), vo.cpu(), ix.cpu().numpy(), counts.cpu().numpy()
    orc = oracle_run(wl, x, budget, adaptive_alpha=alpha)
    assert len([k for k in orc if isinstance(k, tuple)]) == wl.requests * wl.layers * H
    kb = workloads.bf16_bits(x.k)
    vb = workloads.bf16_bits(x.v)
    K = min(budget, N) - W
    g = int(np.floor(alpha * K))
    swaps = 0
    log = []
    for r in range(wl.requests):
        for l in range(wl.layers):
            cnt = counts[r, l]
            assert cnt.sum() == H * min(budget, N) and (cnt >= g + W).all()
            off = np.concatenate([[0], np.cumsum(cnt)])
            gpu_sets, orc_sets, S_orc = set(), set(), {}
            thresholds = []
            for h in range(H):
                o = orc[(r, l, h)]
                check_scores(f"S {(r, l, h)}", S[r, l, h], o["S"])
                seg = ix[r, l, off[h]:off[h + 1]]
                assert np.all(np.diff(seg) > 0)
                assert np.array_equal(seg[-W:], np.arange(N - W, N))
                Kc = ko[r, l, off[h]:off[h + 1]].view(torch.int16).numpy().view(np.uint16)
                Vc = vo[r, l, off[h]:off[h + 1]].view(torch.int16).numpy().view(np.uint16)
                assert np.array_equal(Kc, kb[r, l, h][seg]) and np.array_equal(Vc, vb[r, l, h][seg])
                gpu_sets |= {(h, int(i)) for i in seg[:-W]}
                orc_sets |= {(h, int(i)) for i in o["idx"][:-W]}
                S_orc.update({(h, i): o["S"][i] for i in range(N - W)})
                thresholds.append(_head_threshold(o["S"][:N - W], g))
            # joint threshold: the lowest oracle score among the oracle's picks
            thresholds.append(min(S_orc[t] for t in orc_sets))
            diff = sorted(gpu_sets ^ orc_sets)
            worst = 0.0
            for t in diff:
                sv = S_orc[t]
                gap = min(abs(sv - th) for th in thresholds)
                assert gap <= 1e-5 + 2e-3 * abs(sv), (r, l, t, sv)
                worst = max(worst, gap / (1e-5 + 2e-3 * abs(sv)))
            extra = sorted(gpu_sets - orc_sets)
            swaps += len(extra)
            if diff:
                missing = sorted(orc_sets - gpu_sets)
                log.append({"unit": [r, l], "gpu_only": [list(t) for t in extra],
                            "oracle_only": [list(t) for t in missing],
                            "oracle_S_gpu_only": [float(S_orc[t]) for t in extra],
                            "oracle_S_oracle_only": [float(S_orc[t]) for t in missing],
                            "thresholds": [float(th) for th in thresholds],
                            "max_gap_over_band": worst})
    if case is not None:
        record_swaps(case, wl.name, budget, wl.requests * wl.layers * H,
                     f"{H * K} per (request, layer), shared by its heads", log,
                     f"adaptive head budgets, alpha {alpha}")
    return swaps


@pytest.mark.parametrize("name,budget,alpha", [("tiny", 64, 0.2), ("tiny", 64, 1.0),
                                               ("llava", 128, 0.2), ("qwen-img", 256, 0.0)])
def test_adaptive_head_budgets_parity(name, budget, alpha):
    base = workloads.CONFIGS[name]
    wl = base.with_(layers=min(3, base.layers))
    x = workloads.generate(wl, seed=8, device="cuda")
    swaps = _adaptive_parity(wl, x, budget, alpha)
    K = min(budget, wl.seq_len) - wl.window
    assert swaps <= max(2, wl.requests * wl.layers * wl.kv_heads * K // 500)


@pytest.mark.parametrize("name,budget,alpha", [("qwen-img", 512, 0.2), ("video", 652, 0.5),
                                               ("gui", 1024, 0.2)])
def test_adaptive_head_budgets_full_size(name, budget, alpha):
    """The full-size launch (every request, layer and kv-head in one call),
    every unit against the oracle, swaps logged."""
    wl = workloads.CONFIGS[name]
    x = workloads.generate(wl, seed=8, device="cuda")
    swaps = _adaptive_parity(wl, x, budget, alpha, case=f"{name} adaptive B={budget} alpha={alpha}")
    K = min(budget, wl.seq_len) - wl.window
    assert swaps <= max(2, wl.requests * wl.layers * wl.kv_heads * K // 500)


def test_adaptive_alpha_one_equals_uniform():
    wl = workloads.CONFIGS["tiny"].with_(layers=3)
    x = workloads.generate(wl, seed=9, device="cuda")
    whole = run_gpu(wl, x, 64)
    ctx = bacon.Context(wl.layers, wl.kv_heads, wl.q_heads, wl.head_dim, wl.window, wl.pool, 64,
                        max_seq_len=wl.seq_len, max_requests=1)
    ko, vo, ix, counts = ctx.compress_adaptive(x.qwin, x.k, x.v, 64, 1.0)
    ctx.sync()
    ctx.close()
    assert (counts.cpu().numpy() == 64).all()
    assert np.array_equal(ix.cpu().numpy().reshape(whole["idx"].shape), whole["idx"])
    assert torch.equal(ko.cpu().reshape(whole["Kc"].shape), whole["Kc"])


# --------------------------------------- normalisers supplied by the prefill

def prefill_lse(wl, x):
    """ln sum_{i <= pos} exp(q . k_i / sqrt(d)) per window row [R, L, Hq, W],
    computed with plain fp32 PyTorch on the GPU (the quantity a fused
    prefill attention kernel keeps for every query row)."""
    R, Ly, Hq, W, d = x.qwin.shape
    H, N, G = wl.kv_heads, wl.seq_len, wl.group
    out = torch.empty((R, Ly, Hq, W), dtype=torch.float32, device=x.qwin.device)
    pos = torch.arange(N, device=x.qwin.device)
    vis = pos[None, :] <= (N - W + torch.arange(W, device=x.qwin.device))[:, None]
    for r in range(R):
        for l in range(Ly):
            q = x.qwin[r, l].float().view(H, G, W, d)
            k = x.k[r, l].float()
            s = torch.einsum("hgwd,hnd->hgwn", q, k) / (d ** 0.5)
            s = s.masked_fill(~vis, float("-inf"))
            out[r, l] = torch.logsumexp(s, dim=-1).reshape(Hq, W)
    return out


def prefill_lse_from_attention(wl, x):
    """The same normalisers as a prefill attention kernel exports them:
    PyTorch's fused memory-efficient attention over the window rows (bf16
    inputs, bottom-right causal mask as an additive bias, keys repeated over
    each kv-head's query group) returns its log-sum-exp beside the output."""
    R, Ly, Hq, W, d = x.qwin.shape
    N, G = wl.seq_len, wl.group
    op = getattr(torch.ops.aten, "_scaled_dot_product_efficient_attention", None)
    if op is None:
        pytest.skip("this PyTorch has no fused memory-efficient attention")
    pos = torch.arange(N, device=x.qwin.device)
    hidden = pos[None, :] > (N - W + torch.arange(W, device=x.qwin.device))[:, None]
    bias = torch.zeros((W, N), dtype=torch.bfloat16, device=x.qwin.device)
    bias.masked_fill_(hidden, float("-inf"))
    bias = bias.expand(1, Hq, W, N).contiguous()
    out = torch.empty((R, Ly, Hq, W), dtype=torch.float32, device=x.qwin.device)
    for r in range(R):
        for l in range(Ly):
            q = x.qwin[r, l].unsqueeze(0)
            k = x.k[r, l].repeat_interleave(G, dim=0).unsqueeze(0)
            v = x.v[r, l].repeat_interleave(G, dim=0).unsqueeze(0)
            try:
                res = op(q, k, v, bias, True, 0.0, False, scale=d ** -0.5)
            except RuntimeError as e:  # no kernel for this device or shape
                pytest.skip(f"fused attention unavailable: {e}")
            out[r, l] = res[1][0, :, :W].float()
    return out


def run_with_lse(wl, x, lse, budget):
    p = bacon.default_params(keep_scores=1, max_seq_len=wl.seq_len, max_requests=wl.requests)
    ctx = bacon.Context(wl.layers, wl.kv_heads, wl.q_heads, wl.head_dim, wl.window, wl.pool,
                        budget, params=p)
    ko, vo, idx = ctx.compress_with_lse(x.qwin, x.k, x.v, lse, budget)
    ctx.sync()
    R, Ly, H, N = wl.requests, wl.layers, wl.kv_heads, wl.seq_len
    out = {"Kc": ko.cpu(), "Vc": vo.cpu(), "idx": idx.cpu().numpy()}
    for kind in ("B", "Q", "E", "V", "Bpool", "S"):
        out[kind] = ctx.scores(kind).cpu().numpy().reshape(R, Ly, H, N)
    out["lambda"] = ctx.scores("lambda").cpu().numpy().reshape(R, Ly, H)
    ctx.close()
    return out


@pytest.mark.parametrize("name,budget", [("tiny", 64), ("qwen-img", 256), ("video", 652),
                                         ("gui", 1024)])
def test_prefill_normalisers_path(name, budget):
    """bacon_compress_with_lse (one pass over K) against the oracle at the
    full shape, every unit: the oracle computes its own normalisers in
    double precision; the GPU path is given fp32 ones."""
    wl = workloads.CONFIGS[name]
    x = workloads.generate(wl, seed=11, device="cuda")
    lse = prefill_lse(wl, x)
    gpu = run_with_lse(wl, x, lse, budget)
    del lse
    orc = oracle_run(wl, x, budget)
    swaps = compare(wl, x, budget, gpu, orc, case=f"{name} B={budget} normalisers from the prefill",
                    path="bacon_compress_with_lse")
    units = wl.requests * wl.layers * wl.kv_heads
    assert swaps <= max(2, units * (budget - wl.window) // 1000)


def test_prefill_normalisers_from_fused_attention():
    """The normalisers as a fused attention kernel exports them (its
    log-sum-exp output) give the oracle's result too: Qwen2-VL image shape,
    every unit of the first six layers."""
    wl = workloads.CONFIGS["qwen-img"].with_(layers=6)
    x = workloads.generate(wl, seed=12, device="cuda")
    lse = prefill_lse_from_attention(wl, x)
    ref = prefill_lse(wl, x)
    # the exported values agree with a plain fp32 computation to well under
    # the score tolerance (an error of e nats scales a row's weights by e^e)
    assert torch.allclose(lse, ref, rtol=0, atol=2e-4), float((lse - ref).abs().max())
    gpu = run_with_lse(wl, x, lse, 256)
    orc = oracle_run(wl, x, 256)
    compare(wl, x, 256, gpu, orc, case="qwen-img (6 layers) B=256 normalisers from fused attention",
            path="bacon_compress_with_lse")
