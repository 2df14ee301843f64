"""Ablation / sensitivity sweep (bacon_sweep) on the GPU: every variant
against the oracle on small shapes, and against the whole-step call under
the same parameters at full size (same kernels, so the indices and lambdas
must be identical)."""

import os

import numpy as np
import pytest

import oracle
from paper_2606_14782_gb300 import bacon, build, workloads
from parity import ATOL, RTOL, check_selection

pytestmark = pytest.mark.gpu

THREADS = os.cpu_count() or 4
EXTRA = [dict(gamma=0.5), dict(gamma=2.0, rho=3), dict(r=0, m=1), dict(rho=0)]


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    bacon.load()


def _ctx(wl, budget, **over):
    p = bacon.default_params(max_seq_len=max(wl.seq_len, 64), max_requests=wl.requests, **over)
    return bacon.Context(wl.layers, wl.kv_heads, wl.q_heads, wl.head_dim, wl.window, wl.pool,
                         budget, params=p)


def _whole_step(wl, x, budget, variant):
    """idx and lambda of bacon_compress_all_layers with the variant's fields."""
    p = bacon.default_params(max_seq_len=max(wl.seq_len, 64), max_requests=wl.requests,
                             keep_scores=1)
    for f, v in variant.items():
        setattr(p, f, v)
    ctx = bacon.Context(wl.layers, wl.kv_heads, wl.q_heads, wl.head_dim, wl.window, wl.pool,
                        budget, params=p)
    _, _, idx = ctx.compress_all_layers(x.qwin, x.k, x.v, budget)
    lam = ctx.scores("lambda")
    ctx.sync()
    out = idx.cpu().numpy(), lam.cpu().numpy().reshape(idx.shape[:3])
    ctx.close()
    return out


@pytest.mark.parametrize("name,over,budget", [
    ("tiny", dict(layers=10, seq_len=640), 64),
    ("tiny", dict(layers=9, seq_len=777, q_heads=6, kv_heads=2, head_dim=128,
                  visual=(16, 700)), 100),
])
def test_sweep_matches_oracle(name, over, budget):
    wl = workloads.CONFIGS[name].with_(**over)
    x = workloads.generate(wl, seed=7, device="cuda")
    variants = list(workloads.SWEEP_VARIANTS) + EXTRA
    ctx = _ctx(wl, budget)
    idx, lam = ctx.sweep(x.qwin, x.k, budget, variants)
    ctx.sync()
    idx, lam = idx.cpu().numpy(), lam.cpu().numpy()
    ctx.close()
    qb, kb, vb = (workloads.bf16_bits(t) for t in (x.qwin, x.k, x.v))
    orc = oracle.sweep(qb, kb, vb, budget, variants, oracle.Params(pool_kernel=wl.pool),
                       threads=THREADS, keep_scores=True)
    N, W = wl.seq_len, wl.window
    # each swap is checked against the tolerance band; their number is only
    # bounded loosely (at most 1% of the kept candidates of a variant)
    max_swaps = max(2, wl.requests * wl.layers * wl.kv_heads * (min(budget, N) - W) // 100)
    for j, (var, res) in enumerate(zip(variants, orc)):
        swaps = 0
        for (r, l, h), o in res.items():
            where = (j, var, r, l, h)
            swaps += check_selection(idx[j, r, l, h], o["idx"], o["S"], N, W, budget)
            g, want = float(lam[j, r, l, h]), o["lambda"]
            assert abs(g - want) <= RTOL * abs(want) + ATOL, (where, g, want)
        assert swaps <= max_swaps, (var, swaps)


@pytest.mark.parametrize("name,budget,picks", [
    ("qwen-img", 256, [0, 2, 6, 10]),
    ("gui", 1024, [0, 1, 5, 9]),
])
def test_sweep_equals_whole_step_at_full_size(name, budget, picks):
    """The launch the benchmark times: every variant of the grid, with a few
    of them recomputed one by one through bacon_compress_all_layers."""
    wl = workloads.CONFIGS[name]
    x = workloads.generate(wl, seed=0, device="cuda")
    variants = list(workloads.SWEEP_VARIANTS)
    ctx = _ctx(wl, budget)
    idx, lam = ctx.sweep(x.qwin, x.k, budget, variants)
    ctx.sync()
    idx, lam = idx.cpu().numpy(), lam.cpu().numpy()
    ctx.close()
    kept = min(budget, wl.seq_len)
    assert idx.shape == (len(variants), wl.requests, wl.layers, wl.kv_heads, kept)
    assert (np.diff(idx, axis=-1) > 0).all()
    assert (idx[..., -wl.window:] == np.arange(wl.seq_len - wl.window, wl.seq_len)).all()
    for j in picks:
        want_idx, want_lam = _whole_step(wl, x, budget, variants[j])
        assert np.array_equal(idx[j], want_idx), variants[j]
        assert np.array_equal(lam[j], want_lam), variants[j]


def test_sweep_sampled_oracle_at_gui_size():
    """A non-default variant (deep persistence, wide coherence) at the GUI
    shape, two units recomputed by the oracle."""
    wl = workloads.CONFIGS["gui"].with_(requests=1, layers=10)
    x = workloads.generate(wl, seed=3, device="cuda")
    budget = 1024
    variants = [dict(m=8, r=9), dict(use_E=0, use_L=1, use_T=1)]
    ctx = _ctx(wl, budget)
    idx, lam = ctx.sweep(x.qwin, x.k, budget, variants)
    ctx.sync()
    idx, lam = idx.cpu().numpy(), lam.cpu().numpy()
    ctx.close()
    qb, kb, vb = (workloads.bf16_bits(t) for t in (x.qwin, x.k, x.v))
    units = [(0, 9, 0), (0, 8, 3)]
    orc = oracle.sweep(qb, kb, vb, budget, variants, oracle.Params(pool_kernel=wl.pool),
                       threads=THREADS, units=units, keep_scores=True)
    for j, res in enumerate(orc):
        for (r, l, h), o in res.items():
            check_selection(idx[j, r, l, h], o["idx"], o["S"], wl.seq_len, wl.window, budget)
            assert abs(lam[j, r, l, h] - o["lambda"]) <= RTOL * abs(o["lambda"]) + ATOL


def test_sweep_rejects_bad_variants():
    wl = workloads.CONFIGS["tiny"]
    x = workloads.generate(wl, seed=0, device="cuda")
    ctx = _ctx(wl, 64)
    bad = [[], [dict()] * (bacon.MAX_VARIANTS + 1), [dict(r=-1)], [dict(m=-2)],
           [dict(rho=-1)], [dict(gamma=float("nan"))], [dict(gamma=-1.0)],
           [dict(gamma=float("inf"))]]
    for vs in bad:
        with pytest.raises(bacon.BaconError) as e:
            ctx.sweep(x.qwin, x.k, 64, vs)
        assert e.value.status == bacon.BACON_EINVAL, vs
    with pytest.raises(bacon.BaconError):
        ctx.sweep(x.qwin, x.k, 16, [dict()])  # budget below the window
    # the context stays usable, and the scores of a sweep are not reported
    idx, _ = ctx.sweep(x.qwin, x.k, 64, [dict()])
    ctx.sync()
    assert idx.shape[0] == 1
    with pytest.raises(bacon.BaconError) as e:
        ctx._last_units, ctx._last_N = 1, wl.seq_len
        ctx.scores("S")
    assert e.value.status == bacon.BACON_ESTATE
    ctx.close()
