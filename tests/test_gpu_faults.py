"""Failure detection: a pipeline wait that runs out is reported, not hung.

Every wait inside the window kernels is bounded (about a second of clock
cycles).  When one runs out, the CTA raises its abort flag, its other roles
leave their loops, the CTA drains its own copies, frees tensor memory and
returns, and the error word reports BACON_ETIMEOUT at the next bacon_sync.
The fault is injected on the host: with BACON_FAULT=missing_arrival set
when the context is created, the next two-pass window step withholds one
K-tile load of CTA 0 in pass 1, so that CTA's MMA thread waits for data
that never comes.  Nothing faults or traps.  The test runs in a child
process (the variable is read at bacon_init) and checks that the error
comes back, that the context stays usable and that its next call matches
a fresh context bit for bit.
"""

import os
import subprocess
import sys
import textwrap

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = textwrap.dedent("""
    import os, sys, time
    sys.path.insert(0, {root!r})
    import torch
    from paper_2606_14782_gb300 import bacon, build, workloads

    build.build()
    # more than 1024 tokens: the two-pass window kernels run
    wl = workloads.CONFIGS["tiny"].with_(seq_len=2048, visual=(16, 2000))
    budget = wl.budgets[0]
    x = workloads.generate(wl, seed=3, device="cuda")

    def context():
        return bacon.Context(wl.layers, wl.kv_heads, wl.q_heads, wl.head_dim, wl.window,
                             wl.pool, budget, max_seq_len=wl.seq_len, max_requests=1)

    ctx = context()                      # BACON_FAULT is set: one fault pending
    os.environ.pop("BACON_FAULT")
    t0 = time.time()
    ctx.compress_all_layers(x.qwin, x.k, x.v, budget)
    try:
        ctx.sync()
        print("STATUS", 0)
    except bacon.BaconError as e:
        print("STATUS", e.status)
    print("SECONDS", round(time.time() - t0, 2))
    ko, vo, idx = ctx.compress_all_layers(x.qwin, x.k, x.v, budget)
    ctx.sync()
    ref = context()
    rko, rvo, ridx = ref.compress_all_layers(x.qwin, x.k, x.v, budget)
    ref.sync()
    same = (torch.equal(idx, ridx) and torch.equal(ko.view(torch.int16), rko.view(torch.int16))
            and torch.equal(vo.view(torch.int16), rvo.view(torch.int16)))
    print("SAME", int(same))
""")


def test_missing_arrival_times_out_and_the_context_recovers():
    env = dict(os.environ, BACON_FAULT="missing_arrival")
    proc = subprocess.run([sys.executable, "-c", CHILD.format(root=ROOT)], env=env,
                          capture_output=True, text=True, timeout=300)
    assert proc.returncode == 0, proc.stderr[-2000:]
    lines = dict(line.split(" ", 1) for line in proc.stdout.splitlines() if " " in line)
    from paper_2606_14782_gb300 import bacon
    assert int(lines["STATUS"]) == bacon.BACON_ETIMEOUT, proc.stdout
    assert float(lines["SECONDS"]) < 30.0, proc.stdout     # bounded waits, no hang
    assert lines["SAME"].strip() == "1", proc.stdout


NOALLOC_CHILD = textwrap.dedent("""
    import os, sys, time
    sys.path.insert(0, {root!r})
    import torch
    from paper_2606_14782_gb300 import bacon, build, workloads

    build.build()
    lib = bacon.load()
    wl = workloads.CONFIGS["tiny"].with_(layers=1, q_heads=8, kv_heads=2, seq_len=2048,
                                         visual=(16, 2000))
    x = workloads.generate(wl, seed=3, device="cuda")
    qwin, k = x.qwin[0, 0], x.k[0, 0]
    stream = torch.cuda.current_stream().cuda_stream

    def call():
        out = [torch.zeros((wl.kv_heads, wl.seq_len), device="cuda") for _ in range(3)]
        rc = lib.bacon_window_scores_noalloc(wl.kv_heads, wl.q_heads, wl.head_dim, wl.window,
                                             qwin.data_ptr(), k.data_ptr(), wl.seq_len,
                                             *[t.data_ptr() for t in out], stream)
        torch.cuda.synchronize()
        return rc, out

    t0 = time.time()
    rc, out = call()                    # BACON_FAULT is set: this call's pass 1 loses a load
    os.environ.pop("BACON_FAULT")       # (the reference context below must not fault)
    print("RC", rc)
    print("SECONDS", round(time.time() - t0, 2))
    print("ALLNAN", int(all(bool(torch.isnan(t).all()) for t in out)))
    rc2, out2 = call()                  # the next call is clean
    ctx = bacon.Context(1, wl.kv_heads, wl.q_heads, wl.head_dim, wl.window, wl.pool, wl.window,
                        max_seq_len=wl.seq_len, max_requests=1)
    ctx.compress_all_layers(x.qwin, x.k, x.v, wl.window)
    ref = [ctx.scores(kind).view(wl.kv_heads, wl.seq_len) for kind in "BQE"]
    ctx.sync()
    ok = rc2 == 0 and all(torch.allclose(a, b, rtol=2e-3, atol=1e-5) for a, b in zip(out2, ref))
    print("RECOVERED", int(ok))
""")


def test_noalloc_timeout_fills_outputs_with_nan():
    """The allocation-free call returns before its kernels run; a wait that
    runs out inside them turns its B, Q and E into NaN, and the next call
    (same static scratch) is correct again."""
    env = dict(os.environ, BACON_FAULT="missing_arrival")
    proc = subprocess.run([sys.executable, "-c", NOALLOC_CHILD.format(root=ROOT)], env=env,
                          capture_output=True, text=True, timeout=300)
    assert proc.returncode == 0, proc.stderr[-2000:]
    lines = dict(line.split(" ", 1) for line in proc.stdout.splitlines() if " " in line)
    assert int(lines["RC"]) == 0, proc.stdout
    assert float(lines["SECONDS"]) < 30.0, proc.stdout
    assert lines["ALLNAN"].strip() == "1", proc.stdout
    assert lines["RECOVERED"].strip() == "1", proc.stdout
