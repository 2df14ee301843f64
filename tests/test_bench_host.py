"""Host-side logic of bench.py, on the CPU: the traffic record written from an
ncu log and read back (per workload, scaled by the requests of a launch,
voided when the kernel's sources change), and the reference arm's JSON line."""

import json
import os
import subprocess
import sys

import pytest

import bench

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

HEADER = ('"ID","Process ID","Process Name","Host Name","Kernel Name","Context","Stream",'
          '"Block Size","Grid Size","Device","CC","Section Name","Metric Name","Metric Unit",'
          '"Metric Value"\n')


def _row(i, kernel, metric, unit, value):
    return (f'"{i}","1","python3","h","{kernel}","1","7","(576, 1, 1)","(152, 1, 1)","0","10.3",'
            f'"Command line profiler metrics","{metric}","{unit}","{value}"\n')


def _ncu_log(tmp_path):
    k1 = "void unnamed>::window_tc_kernel<128, 1>(TcArgs, unnamed>::Plan)"
    k2 = "void unnamed>::window_tc_kernel<128, 2>(TcArgs, unnamed>::Plan)"
    cal = "void unnamed>::calibrate_select_kernel<1024, 16>(Shape, Calib, CalibArgs)"
    text = ("==PROF== Connected to process 1\n" + HEADER
            + _row(0, k1, "dram__bytes_read.sum", "Mbyte", "480.5")
            + _row(0, k1, "dram__bytes_write.sum", "byte", "500000")
            + _row(0, k1, "gpu__time_duration.sum", "us", "197.0")
            + _row(1, k2, "dram__bytes_read.sum", "Gbyte", "0.48")
            + _row(1, k2, "dram__bytes_write.sum", "Kbyte", "1,625.3")
            + _row(2, cal, "dram__bytes_read.sum", "byte", "14790912")
            + _row(2, cal, "dram__bytes_write.sum", "byte", "0")
            + _row(3, cal, "dram__bytes_read.sum", "byte", "14790000")
            + _row(3, cal, "dram__bytes_write.sum", "byte", "0"))
    p = tmp_path / "log.csv"
    p.write_text(text)
    return str(p)


def test_record_and_read_traffic(tmp_path):
    out = str(tmp_path / "traffic.json")
    found = bench.record_traffic(_ncu_log(tmp_path), "gui", 1, "ncu ...", path=out)
    assert set(found) == {"window_stats", "window_scores", "calibrate_select"}
    rec = json.load(open(out))["gui"]
    assert rec["window_stats"]["dram_bytes_per_request"] == pytest.approx(480.5e6 + 5e5)
    assert rec["window_scores"]["dram_bytes_per_request"] == pytest.approx(0.48e9 + 1625.3e3)
    # two launches of the calibration kernel: their mean
    assert rec["calibrate_select"]["launches"] == 2
    assert rec["calibrate_select"]["dram_bytes_per_request"] == pytest.approx(14790456.0)
    # read back for a 4-request launch of the same workload
    assert bench.kernel_traffic("window_stats", "gui", 4, path=out) == pytest.approx(4 * (480.5e6 + 5e5))
    # another workload, or a kernel without a record: nothing
    assert bench.kernel_traffic("window_stats", "llava", 1, path=out) is None
    assert bench.kernel_traffic("gather", "gui", 1, path=out) is None
    # a record whose sources changed since the capture is void
    rec_all = json.load(open(out))
    rec_all["gui"]["window_stats"]["code_sha256_16"] = "0" * 16
    json.dump(rec_all, open(out, "w"))
    assert bench.kernel_traffic("window_stats", "gui", 4, path=out) is None
    assert bench.kernel_traffic("window_scores", "gui", 4, path=out) is not None


def test_source_digest_ignores_comments():
    # the digest of the committed sources is stable and comment-insensitive by construction
    d = bench.source_digest(["gather.cu", "common.cuh"])
    assert len(d) == 16 and d == bench.source_digest(["gather.cu", "common.cuh"])
    assert d != bench.source_digest(["gather.cu"])


def test_reference_arm_json_line():
    proc = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                           "--config", "tiny", "--steps", "1", "--warmup", "0"],
                          capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert proc.returncode == 0, proc.stderr[-2000:]
    line = json.loads(proc.stdout.strip().splitlines()[-1])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config",
                "cpu_baseline", "e2e"):
        assert key in line, key
    assert line["impl"] == "reference"
    assert line["value"] > 0 and line["higher_is_better"] is True
    assert line["e2e"]["value"] == line["value"]
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["d2h_bytes_per_step"] == 0
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] >= 1
    assert line["config"]["workload"].startswith("tiny")


def test_cpu_baseline_reports_threads_and_one_thread():
    import numpy as np

    import oracle
    from paper_2606_14782_gb300 import workloads
    wl = workloads.CONFIGS["tiny"]
    x = workloads.generate(wl, seed=0, device="cpu")
    host = tuple(workloads.bf16_bits(t) for t in (x.qwin, x.k, x.v))
    # the oracle's own selections stand in for the GPU's: no swaps
    ref = oracle.compress(*host, wl.budgets[0], oracle.Params(pool_kernel=wl.pool))
    idx = np.stack([np.stack([ref[(0, l, h)]["idx"] for h in range(wl.kv_heads)])
                    for l in range(wl.layers)])[None]
    cb = bench.cpu_baseline(wl, wl.budgets[0], host, idx)
    assert cb["kind"] == "oracle" and cb["unit"] == bench.UNIT and cb["value"] > 0
    assert cb["cores"] == min(os.cpu_count() or 1, wl.requests * wl.kv_heads)
    assert cb["single_thread"]["cores"] == 1 and cb["single_thread"]["value"] > 0
    chk = cb["sample_selection_check"]
    assert chk["boundary_swaps"] == 0 and chk["all_within_band"] and chk["units"] == 2 * 4


def test_boundary_swap_count_and_band():
    import numpy as np
    N, W, budget = 12, 2, 6          # 10 candidates, 4 selected
    S = np.array([9, 8, 7, 5, 5.00001, 1, 0, 0, 0, 0, 0, 0], dtype=np.float64)
    orc = np.array([0, 1, 2, 4, 10, 11])
    # position 3 instead of 4: within the band around the boundary score 5
    assert bench.boundary_swaps(np.array([0, 1, 2, 3, 10, 11]), orc, S, N, W, budget) == (1, True)
    # position 5 instead of 4: far below the boundary
    assert bench.boundary_swaps(np.array([0, 1, 2, 5, 10, 11]), orc, S, N, W, budget) == (1, False)
    assert bench.boundary_swaps(orc, orc, S, N, W, budget) == (0, True)


def test_logged_swaps_reads_the_parity_log(tmp_path):
    csrc = os.path.join(ROOT, "paper_2606_14782_gb300", "csrc")
    names = sorted(n for n in os.listdir(csrc) if n.endswith((".cu", ".cuh", ".h")))
    doc = {"code_sha256_16": bench.source_digest(names),
           "cases": {"gui B=1024": {"swaps": 3, "units_checked": 448, "selected_per_unit": 960,
                                    "max_gap_over_band": 0.5},
                     "edge ragged B=100": {"swaps": 0, "units_checked": 8,
                                           "selected_per_unit": 68, "max_gap_over_band": 0}}}
    path = tmp_path / "swaps.json"
    path.write_text(json.dumps(doc))
    got = bench.logged_swaps(str(path))
    assert got["current_code"] is True
    assert got["cases"] == {"gui B=1024": {"swaps": 3, "units": 448, "selected_per_unit": 960,
                                           "max_gap_over_band": 0.5}}
    doc["code_sha256_16"] = "0" * 16
    path.write_text(json.dumps(doc))
    assert bench.logged_swaps(str(path))["current_code"] is False
