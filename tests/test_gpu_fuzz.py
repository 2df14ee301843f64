"""Seeded random shapes through the whole-step call against the CPU oracle.

The window kernels cut every call into (request, layer, kv-head) units, the
units into 128-token tiles and 1024-token chunks, and hand each CTA a
contiguous range of chunks; their pipelines (TMA stages, TMEM buffers, the
epilogue groups' exchange slots) must hold for any mix of window rows, head
dim, ragged lengths, budgets and unit counts.  The shapes below are drawn
once from a fixed seed: window sizes from 1 to 64 (multiples of 16 and
not), query-head groups of 1 to 8, head dim 64 and 128, prompt lengths that
end mid-tile and mid-chunk, budgets from the window alone to more than the
prompt, and calls with more chunks than the GPU has SMs (so that CTA ranges
cross unit boundaries after short or odd-length units).  The same shapes go
through the layer-by-layer path (one layer per call, bit-identical to the
whole step) and the path that takes the prefill's row normalisers (one
window pass; within the parity tolerance of the whole step).
"""

import numpy as np
import pytest
import torch

from paper_2606_14782_gb300 import bacon, build, workloads
from test_gpu_parity import compare, oracle_run, prefill_lse, run_gpu, run_with_lse

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    bacon.load()


def _shapes(n=10, seed=20261202):
    rng = np.random.default_rng(seed)
    out = []
    while len(out) < n:
        many = len(out) >= n - 2  # the last two: more chunks than SMs
        d = int(rng.choice([64, 128]))
        group = int(rng.choice([1, 2, 3, 4, 7, 8]))
        window = int(rng.integers(1, 65))
        if group * window > 512:
            continue
        kv = int(rng.integers(1, 9))
        if many:
            layers, requests = int(rng.integers(16, 25)), 1
            kv = max(kv, 8)
            seq = int(rng.integers(1025, 1700))
        else:
            layers, requests = int(rng.integers(1, 7)), int(rng.integers(1, 3))
            seq = int(rng.integers(max(window, 40), 3000))
        units = requests * layers * kv
        if units * group * window * seq * d > 6e8:
            continue
        budget = int(rng.integers(window, seq + 11))
        span = (min(16, seq // 4), max(min(16, seq // 4) + 1, seq - window - 4))
        planted = 2 if span[1] - span[0] >= 64 else 0
        out.append((f"s{len(out)}_d{d}_g{group}_w{window}_kv{kv}_l{layers}_r{requests}_n{seq}_b{budget}",
                    dict(layers=layers, requests=requests, q_heads=kv * group, kv_heads=kv,
                         head_dim=d, seq_len=seq, window=window, visual=span, planted=planted,
                         plant_run=2),
                    budget))
    return out


SHAPES = _shapes()


@pytest.mark.parametrize("name,over,budget", SHAPES, ids=[s[0] for s in SHAPES])
def test_random_shapes(name, over, budget):
    wl = workloads.CONFIGS["tiny"].with_(**over)
    x = workloads.generate(wl, seed=11, device="cuda")
    gpu = run_gpu(wl, x, budget)
    orc = oracle_run(wl, x, budget)
    compare(wl, x, budget, gpu, orc, case=f"fuzz {name} B={budget}")
    # each window softmax row sums to one, so B and Q do per unit
    np.testing.assert_allclose(gpu["B"].sum(-1), 1.0, atol=2e-4)
    np.testing.assert_allclose(gpu["Q"].sum(-1), 1.0, atol=2e-4)


@pytest.mark.parametrize("name,over,budget", SHAPES, ids=[s[0] for s in SHAPES])
def test_random_shapes_layer_path(name, over, budget):
    wl = workloads.CONFIGS["tiny"].with_(**over)
    x = workloads.generate(wl, seed=11, device="cuda")
    whole = run_gpu(wl, x, budget)
    p = bacon.default_params(max_seq_len=wl.seq_len, max_requests=wl.requests)
    ctx = bacon.Context(wl.layers, wl.kv_heads, wl.q_heads, wl.head_dim, wl.window, wl.pool,
                        budget, params=p)
    st = bacon.State(ctx)
    r = wl.requests - 1
    for l in range(wl.layers):
        S = st.score_layer(l, x.qwin[r, l], x.k[r, l], scores_out=True)
        idx = st.select(budget, wl.seq_len)
        ko, vo = ctx.compact(x.k[r, l], x.v[r, l], idx)
        ctx.sync()
        assert np.array_equal(S.cpu().numpy(), whole["S"][r, l]), l
        assert np.array_equal(idx.cpu().numpy(), whole["idx"][r, l]), l
        assert torch.equal(ko.cpu(), whole["Kc"][r, l]) and torch.equal(vo.cpu(), whole["Vc"][r, l])
    st.close()
    ctx.close()


@pytest.mark.parametrize("name,over,budget", SHAPES, ids=[s[0] for s in SHAPES])
def test_random_shapes_prefill_normalisers(name, over, budget):
    """The one-pass path given the prefill's normalisers, against the oracle."""
    wl = workloads.CONFIGS["tiny"].with_(**over)
    x = workloads.generate(wl, seed=11, device="cuda")
    gpu = run_with_lse(wl, x, prefill_lse(wl, x), budget)
    orc = oracle_run(wl, x, budget)
    compare(wl, x, budget, gpu, orc, case=f"fuzz {name} B={budget} normalisers from the prefill",
            path="bacon_compress_with_lse")
