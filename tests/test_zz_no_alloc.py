"""The allocation-free entry point, bacon_window_scores_noalloc.

It serves callers that cannot call cudaMalloc (for example a serving engine
that has reserved all of HBM for its KV cache): its scratch is a static
device array inside the library.  Its B, Q and E must agree with the oracle
(Eqs. 1, 2 and 4) and with the context path (bacon_compress_all_layers +
bacon_get_scores) within the parity tolerance, on two calls in a row that
reuse the same static scratch.  This file is named so that pytest collects
it last.
"""

import ctypes

import numpy as np
import pytest
import torch

import oracle
from paper_2606_14782_gb300 import bacon, build, workloads
from parity import check_scores

pytestmark = pytest.mark.gpu

SHAPES = [
    # layers = requests = 1; (name, overrides of the tiny workload)
    ("tiny_d64", dict(layers=1)),
    ("qwen_layer", dict(layers=1, q_heads=28, kv_heads=4, head_dim=128, seq_len=4096,
                        window=32, visual=(16, 3616))),
    ("gui_layer", dict(layers=1, q_heads=28, kv_heads=4, head_dim=128, seq_len=16384,
                       window=64, visual=(16, 15888))),
    ("video_layer", dict(layers=1, q_heads=28, kv_heads=4, head_dim=128, seq_len=6528,
                         window=64, visual=(16, 6288))),
    ("ragged", dict(layers=1, q_heads=6, kv_heads=2, head_dim=128, seq_len=1000, window=5,
                    visual=(16, 900))),
]


@pytest.fixture(scope="module")
def lib():
    build.build()
    return bacon.load()


def _noalloc(lib, wl, qwin, k, B, Q, E):
    stream = torch.cuda.current_stream().cuda_stream
    return lib.bacon_window_scores_noalloc(wl.kv_heads, wl.q_heads, wl.head_dim, wl.window,
                                           qwin.data_ptr(), k.data_ptr(), wl.seq_len,
                                           B.data_ptr(), Q.data_ptr(), E.data_ptr(), stream)


@pytest.mark.parametrize("name,over", SHAPES, ids=[s[0] for s in SHAPES])
def test_noalloc_matches_context_path(lib, name, over):
    wl = workloads.CONFIGS["tiny"].with_(**over)
    x = workloads.generate(wl, seed=5, device="cuda")
    qwin, k = x.qwin[0, 0], x.k[0, 0]
    # existing entry point (context-owned scratch)
    ctx = bacon.Context(1, wl.kv_heads, wl.q_heads, wl.head_dim, wl.window, wl.pool,
                        wl.window, max_seq_len=wl.seq_len, max_requests=1)
    ctx.compress_all_layers(x.qwin, x.k, x.v, wl.window)
    ref = {kind: ctx.scores(kind).view(wl.kv_heads, wl.seq_len).cpu() for kind in "BQE"}
    ctx.sync()
    ctx.close()
    # two calls in a row sharing the static scratch
    for call in range(2):
        out = {kind: torch.full((wl.kv_heads, wl.seq_len), float("nan"), device="cuda")
               for kind in "BQE"}
        rc = _noalloc(lib, wl, qwin, k, out["B"], out["Q"], out["E"])
        assert rc == bacon.BACON_OK, (call, rc)
        torch.cuda.synchronize()
        for kind in "BQE":
            check_scores(f"call {call} {kind}", out[kind].cpu().numpy(), ref[kind].numpy())


@pytest.mark.parametrize("name,over", SHAPES, ids=[s[0] for s in SHAPES])
def test_noalloc_matches_oracle(lib, name, over):
    """Every kv-head of the layer against the oracle's Eqs. 1, 2 and 4."""
    wl = workloads.CONFIGS["tiny"].with_(**over)
    x = workloads.generate(wl, seed=7, device="cuda")
    qwin, k = x.qwin[0, 0], x.k[0, 0]
    out = {kind: torch.full((wl.kv_heads, wl.seq_len), float("nan"), device="cuda")
           for kind in "BQE"}
    assert _noalloc(lib, wl, qwin, k, out["B"], out["Q"], out["E"]) == bacon.BACON_OK
    torch.cuda.synchronize()
    qf = oracle.bf16_bits_to_f64(workloads.bf16_bits(qwin))
    kf = oracle.bf16_bits_to_f64(workloads.bf16_bits(k))
    G = wl.q_heads // wl.kv_heads
    for h in range(wl.kv_heads):
        B, Q = oracle.window_scores(qf[h * G:(h + 1) * G], kf[h])
        E = oracle.residual(Q, B)
        for kind, ref in (("B", B), ("Q", Q), ("E", E)):
            check_scores(f"{name} kv-head {h} {kind}", out[kind][h].cpu().numpy(), ref)
        assert np.isfinite(out["B"][h].cpu().numpy()).all()


def test_noalloc_rejects_sizes_beyond_its_static_scratch(lib):
    B = torch.empty(64, device="cuda")
    q = torch.empty(64, dtype=torch.bfloat16, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    call = lib.bacon_window_scores_noalloc
    # seq_len above 16384
    assert call(4, 28, 128, 64, q.data_ptr(), q.data_ptr(), 16385, B.data_ptr(), B.data_ptr(),
                B.data_ptr(), stream) == bacon.BACON_EUNSUPPORTED
    # q_heads * window above 4096
    assert call(8, 64, 128, 128, q.data_ptr(), q.data_ptr(), 4096, B.data_ptr(), B.data_ptr(),
                B.data_ptr(), stream) == bacon.BACON_EUNSUPPORTED
    # malformed arguments
    assert call(4, 6, 128, 64, q.data_ptr(), q.data_ptr(), 4096, B.data_ptr(), B.data_ptr(),
                B.data_ptr(), stream) == bacon.BACON_EINVAL
    assert call(4, 28, 128, 64, q.data_ptr() + 2, q.data_ptr(), 4096, B.data_ptr(),
                B.data_ptr(), B.data_ptr(), stream) == bacon.BACON_EINVAL
    assert call(4, 28, 128, 64, None, q.data_ptr(), 4096, B.data_ptr(), B.data_ptr(),
                B.data_ptr(), stream) == bacon.BACON_EINVAL
