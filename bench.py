#!/usr/bin/env python
"""Throughput of the BACON end-of-prefill KV-cache compression step.

One step = the whole path (window scores, calibration, top-B selection,
compaction) for every layer and kv-head of one batch of synthetic prompts,
through the C-ABI call ``bacon_compress_all_layers`` with the inputs already
resident in HBM.  Default workload: the long GUI/screenshot shape (28 layers,
28 query / 4 kv heads, head_dim 128, 16384-token prompts, window 64, pool 7,
budget 1024, 4 requests).  Inputs (1.9 GB of K per step) are far larger than
L2, so no flush is needed between steps.

Prints one JSON line.  ``--impl reference`` times the CPU oracle instead
(bounded sample of the same workload on the host cores).
"""

from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "layer-heads compressed/s"
UNIT = "layer-heads/s"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=("bacon", "reference"), default="bacon")
    ap.add_argument("--config", default="gui")
    ap.add_argument("--budget", type=int, default=None)
    ap.add_argument("--requests", type=int, default=None,
                    help="override the request count (smaller profiling cases)")
    ap.add_argument("--e2e-steps", type=int, default=5)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-extras", action="store_true",
                    help="skip the prefill-normaliser and ablation-sweep measurements")
    ap.add_argument("--record-traffic", metavar="NCU_CSV", default=None,
                    help="store the DRAM bytes of an ncu --csv capture of this --config and "
                         "--requests in profiles/traffic.json, then exit")
    return ap.parse_args()


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return (float(p["hbm_gbs"]), float(p["bf16_tflops"]),
                float(p.get("bf16_tflops_sustained", p["bf16_tflops"])), "measured")
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


def config_dict(wl, budget, n_gpus):
    return {"workload": f"{wl.name}: {wl.layers} layers, {wl.q_heads}/{wl.kv_heads} heads, "
                        f"d {wl.head_dim}, N {wl.seq_len}, W {wl.window}, pool {wl.pool}, "
                        f"budget {budget}, {wl.requests} requests",
            "requests_per_gpu": wl.requests, "seq_len": wl.seq_len, "layers": wl.layers,
            "q_heads": wl.q_heads, "kv_heads": wl.kv_heads, "head_dim": wl.head_dim,
            "window": wl.window, "budget": budget,
            "parallelism": f"replicas x{n_gpus} (independent requests per GPU)",
            "l2": "inputs larger than L2 (K alone %.2f GB per step)" %
                  (wl.requests * wl.layers * wl.kv_heads * wl.seq_len * wl.head_dim * 2 / 1e9)}


# ------------------------------------------------------------- clocks

class ClockSampler:
    FIELDS = ("uuid,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid: str | None):
        self.uuid = uuid
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                if self.uuid and self.uuid not in parts[0]:
                    continue
                rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].replace(".", "", 1).isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "", 1).isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons, "samples": len(rows)}


# --------------------------------------------------------- traffic

def source_digest(names) -> str:
    """sha256[:16] of the named csrc files with comments and blank space
    removed, so that editing a comment does not void a measurement."""
    import re
    h = hashlib.sha256()
    for name in names:
        text = open(os.path.join(ROOT, "paper_2606_14782_gb300", "csrc", name)).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        text = re.sub(r"//[^\n]*", "", text)
        h.update("".join(text.split()).encode())
    return h.hexdigest()[:16]


# ncu kernel name -> (profile stage, the csrc files its code comes from)
KERNEL_SOURCES = [
    ("window_tc_kernel<", ", 1>", "window_stats", ["window_tc.cu", "window_tc.h", "tc.cuh", "common.cuh"]),
    ("window_tc_kernel<", ", 2>", "window_scores", ["window_tc.cu", "window_tc.h", "tc.cuh", "common.cuh"]),
    ("window_onepass_kernel", "", "window_scores",
     ["window_onepass.cu", "window_tc.h", "tc.cuh", "common.cuh"]),
    ("calibrate_select_kernel", "", "calibrate_select", ["calibrate.cu", "select.cuh", "common.cuh"]),
    ("gather_kernel", "", "gather", ["gather.cu", "common.cuh"]),
]


TRAFFIC_PATH = os.path.join(ROOT, "profiles", "traffic.json")


def record_traffic(csv_path: str, workload: str, requests: int, command: str,
                   path: str = TRAFFIC_PATH):
    """Average dram__bytes_read.sum + dram__bytes_write.sum per launch of each
    library kernel in an ncu --csv log, per request, into traffic.json."""
    import csv
    with open(csv_path) as f:
        rows = list(csv.reader(line for line in f if not line.startswith("==")))
    head = rows[0]
    col = {name: i for i, name in enumerate(head)}
    per_launch = {}
    for r in rows[1:]:
        if len(r) != len(head) or r[col["Metric Name"]] not in (
                "dram__bytes_read.sum", "dram__bytes_write.sum"):
            continue
        unit = r[col["Metric Unit"]]
        scale = {"byte": 1, "Kbyte": 1e3, "Mbyte": 1e6, "Gbyte": 1e9}[unit]
        key = (r[col["ID"]], r[col["Kernel Name"]])
        per_launch[key] = per_launch.get(key, 0.0) + float(r[col["Metric Value"]].replace(",", "")) * scale
    try:
        with open(path) as f:
            rec = json.load(f)
    except FileNotFoundError:
        rec = {}
    found = {}
    for (_, name), b in per_launch.items():
        for a, z, stage, srcs in KERNEL_SOURCES:
            if a in name and z in name:
                found.setdefault(stage, (srcs, []))[1].append(b)
                break
    for stage, (srcs, vals) in found.items():
        rec.setdefault(workload, {})[stage] = {
            "sources": srcs, "code_sha256_16": source_digest(srcs),
            "dram_bytes_per_request": sum(vals) / len(vals) / requests,
            "launches": len(vals),
            "measured_on": f"{workload} workload, {requests} request(s): {command}; "
                           "bench.py scales it by the requests of a launch (traffic grows in "
                           "proportion to the (request, layer, kv-head) units processed)"}
    with open(path, "w") as f:
        json.dump(rec, f, indent=1)
        f.write("\n")
    return found


def kernel_traffic(kernel: str, workload: str, requests: int, path: str = TRAFFIC_PATH):
    """DRAM bytes per launch from the committed ncu summary of this kernel on
    this workload (scaled to `requests`: traffic grows with the units), or
    None when there is none or the kernel's sources changed since the
    counters were taken."""
    try:
        with open(path) as f:
            rec = json.load(f)[workload][kernel]
        if source_digest(rec["sources"]) != rec["code_sha256_16"]:
            return None
        return float(rec["dram_bytes_per_request"]) * requests
    except Exception:
        return None


# ---------------------------------------------------- CPU oracle legs

def oracle_sample(wl, budget, units, threads):
    """Time the CPU oracle on `units` of a same-shaped host workload."""
    import oracle
    from paper_2606_14782_gb300 import workloads

    layers_needed = max(l for _, l, _ in units) + 1
    host = workloads.generate(wl.with_(layers=layers_needed), seed=0, device="cpu")
    qb, kb, vb = (workloads.bf16_bits(t) for t in (host.qwin, host.k, host.v))
    p = oracle.Params(pool_kernel=wl.pool)
    t0 = time.perf_counter()
    oracle.compress(qb, kb, vb, budget, p, threads=threads, units=units)
    return time.perf_counter() - t0


def cpu_baseline(wl, budget):
    threads = min(os.cpu_count() or 1, wl.requests * wl.kv_heads)
    layers = min(2, wl.layers)
    units = [(r, l, h) for r in range(wl.requests) for l in range(layers)
             for h in range(wl.kv_heads)]
    secs = oracle_sample(wl, budget, units, threads)
    # the same oracle on one host thread (layer 0 of the first two kv-heads)
    one = units[:min(2, len(units))]
    one_secs = oracle_sample(wl, budget, one, 1)
    return {"value": len(units) / secs, "unit": UNIT, "cores": threads, "kind": "oracle",
            "sample": f"{len(units)} layer-heads (layers 0-{layers - 1} of every request and "
                      f"kv-head) of the same workload, double precision, {threads} threads, "
                      f"{secs:.1f} s wall",
            "single_thread": {"value": len(one) / one_secs, "unit": UNIT, "cores": 1,
                              "sample": f"{len(one)} layer-heads, one thread, "
                                        f"{one_secs:.2f} s wall"}}


def run_reference(args):
    from paper_2606_14782_gb300 import workloads
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    wl = workloads.CONFIGS[args.config]
    if args.requests:
        wl = wl.with_(requests=args.requests)
    budget = args.budget or max(wl.budgets)
    threads = min(os.cpu_count() or 1, wl.requests * wl.kv_heads)
    units = [(r, 0, h) for r in range(wl.requests) for h in range(wl.kv_heads)]
    # one step: layer 0 of every (request, kv-head) of the workload
    import oracle
    host = workloads.generate(wl.with_(layers=1), seed=0, device="cpu")
    qb, kb, vb = (workloads.bf16_bits(t) for t in (host.qwin, host.k, host.v))
    p = oracle.Params(pool_kernel=wl.pool)
    # size the per-step sample so that the whole run stays within a few
    # minutes whatever --steps / --warmup ask for (one untimed probe step)
    t0 = time.perf_counter()
    oracle.compress(qb, kb, vb, budget, p, threads=threads, units=units)
    per_step = time.perf_counter() - t0
    allowed = 150.0 / max(1, args.steps + args.warmup)
    if per_step > allowed:
        keep = max(1, int(len(units) * allowed / per_step))
        units = units[:keep]
    for _ in range(args.warmup):
        oracle.compress(qb, kb, vb, budget, p, threads=threads, units=units)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle.compress(qb, kb, vb, budget, p, threads=threads, units=units)
    secs = time.perf_counter() - t0
    value = len(units) * args.steps / secs
    # n_gpus echoes the launch; the work runs on rank 0's host cores only
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * secs / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "impl": "reference",
            "config": config_dict(wl, budget, 1),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle",
                             "sample": f"each step: {len(units)} layer-heads (layer 0 of "
                                       + ("every (request, kv-head) pair"
                                          if len(units) == wl.requests * wl.kv_heads else
                                          f"the first {len(units)} (request, kv-head) pairs")
                                       + "), double precision"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------ GPU arm

def reduce_step_time(ms: float, world: int, device) -> float:
    """Replicas run independently; the job is as slow as its slowest rank."""
    if world <= 1:
        return ms
    import torch
    import torch.distributed as dist
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(units_per_rank: int, world: int, ms: float) -> float:
    """Whole-job layer-heads per second: every rank's units over the slowest time."""
    return world * units_per_rank / (ms / 1e3)


def main():
    args = parse()
    if args.record_traffic:
        from paper_2606_14782_gb300 import workloads
        wl = workloads.CONFIGS[args.config]
        req = args.requests or wl.requests
        found = record_traffic(args.record_traffic, args.config, req,
                               f"ncu log {os.path.basename(args.record_traffic)}")
        print(json.dumps({k: len(v[1]) for k, v in found.items()}))
        return
    if args.impl == "reference":
        run_reference(args)
        return
    import torch
    import torch.distributed as dist

    from paper_2606_14782_gb300 import bacon, workloads

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)

    def barrier():
        if world > 1:
            dist.barrier()

    wl = workloads.CONFIGS[args.config]
    if args.requests:
        wl = wl.with_(requests=args.requests)
    budget = args.budget or max(wl.budgets)
    x = workloads.generate(wl, seed=rank, device=dev)
    torch.cuda.empty_cache()
    p = bacon.default_params(max_seq_len=wl.seq_len, max_requests=wl.requests)
    ctx = bacon.Context(wl.layers, wl.kv_heads, wl.q_heads, wl.head_dim, wl.window, wl.pool,
                        budget, params=p)
    ko, vo, idx = ctx.compress_all_layers(x.qwin, x.k, x.v, budget)
    stream = torch.cuda.current_stream()
    for _ in range(max(3, args.warmup)):
        ctx.compress_all_layers(x.qwin, x.k, x.v, budget, ko, vo, idx)
    ctx.sync()

    uuid = None
    try:
        uuid = str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:
        pass
    sampler = ClockSampler(uuid)
    sampler.start()
    time.sleep(0.3)
    ctx.profile(True)
    ctx.profile_read()
    barrier()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        ctx.compress_all_layers(x.qwin, x.k, x.v, budget, ko, vo, idx)
    e1.record(stream)
    torch.cuda.synchronize()
    barrier()
    clocks = sampler.stop()
    prof = ctx.profile_read()
    ctx.profile(False)
    ctx.sync()
    ms = reduce_step_time(e0.elapsed_time(e1) / args.steps, world, dev)

    units = wl.requests * wl.layers * wl.kv_heads
    value = job_throughput(units, world, ms)
    hbm, tflops, tflops_sus, peak_src = peaks()

    # per-kernel times measured live (CUDA events around each launch)
    K_bytes = wl.requests * wl.layers * wl.kv_heads * wl.seq_len * wl.head_dim * 2
    Q_bytes = wl.requests * wl.layers * wl.q_heads * wl.window * wl.head_dim * 2
    tok = wl.requests * wl.layers * wl.kv_heads * wl.seq_len
    kept = min(budget, wl.seq_len)
    algo_bytes = {
        "window_stats": K_bytes + Q_bytes,
        "window_scores": K_bytes + Q_bytes + 12 * tok,
        "window_combine": 0,
        "calibrate_select": tok * (4 + 4 * (1 + min(4, wl.layers - 1))) + units * kept * 4,
        "gather": 4 * units * kept * wl.head_dim * 2 + units * kept * 4,
    }
    total = sum(t for t, _ in prof.values())
    kernels = {k: {"ms_per_launch": (t / n if n else None), "share": (t / total if total else None)}
               for k, (t, n) in prof.items() if n}
    dom = max(prof, key=lambda k: prof[k][0])
    dom_ms = prof[dom][0] / max(1, prof[dom][1])
    achieved_gbs = algo_bytes[dom] / (dom_ms / 1e3) / 1e9
    traffic = kernel_traffic(dom, args.config, wl.requests)
    hbm_part = {"achieved": achieved_gbs, "peak": hbm, "unit": "GB/s", "frac": achieved_gbs / hbm,
                "algorithmic_bytes_per_launch": algo_bytes[dom]}
    # one pass of the window contraction: 2 Hq W N d flops per launch
    flops = 2 * wl.requests * wl.layers * wl.q_heads * wl.window * wl.seq_len * wl.head_dim
    if dom.startswith("window") and flops / algo_bytes[dom] > tflops_sus * 1e3 / hbm:
        # a dense contraction above the ridge point: against the sustained
        # bf16 peak (the kernel is timed inside a long step)
        tf = flops / (dom_ms / 1e3) / 1e12
        roofline = {"bound": "tensor", "kernel": dom, "achieved": tf, "peak": tflops_sus,
                    "unit": "TFLOP/s", "frac": tf / tflops_sus,
                    "peak_source": f"{peak_src} (bf16, sustained)", "traffic": traffic,
                    "algorithmic_flops_per_launch": flops, "hbm": hbm_part}
    else:
        roofline = {"bound": "hbm", "kernel": dom, "peak_source": peak_src, "traffic": traffic,
                    **hbm_part}
    step_bytes = wl.bytes_model(budget)

    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
            "ms_per_request": ms / wl.requests,
            "achieved_step_gbs": step_bytes / (ms / 1e3) / 1e9,
            "step_roofline_frac": step_bytes / (ms / 1e3) / 1e9 / hbm,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic (seeded, paper-shaped; no datasets)",
            "config": config_dict(wl, budget, world),
            "gpu_launches": sum(n for _, n in prof.values()), "roofline": roofline, "kernels": kernels,
            "clocks": clocks}

    if not args.no_extras:
        # the same step when the prefill attention supplies the window rows'
        # softmax normalisers (no first pass over K)
        lse = torch.empty((wl.requests, wl.layers, wl.q_heads, wl.window), dtype=torch.float32,
                          device=dev)
        pos = torch.arange(wl.seq_len, device=dev)
        vis = pos[None, :] <= (wl.seq_len - wl.window + torch.arange(wl.window, device=dev))[:, None]
        for r in range(wl.requests):
            for l in range(wl.layers):
                q = x.qwin[r, l].float().view(wl.kv_heads, wl.group, wl.window, wl.head_dim)
                s_ = torch.einsum("hgwd,hnd->hgwn", q, x.k[r, l].float()) / wl.head_dim ** 0.5
                lse[r, l] = torch.logsumexp(s_.masked_fill(~vis, float("-inf")), -1).reshape(
                    wl.q_heads, wl.window)
        del s_
        for _ in range(3):
            ctx.compress_with_lse(x.qwin, x.k, x.v, lse, budget, ko, vo, idx)
        torch.cuda.synchronize()
        g0 = torch.cuda.Event(enable_timing=True)
        g1 = torch.cuda.Event(enable_timing=True)
        g0.record(stream)
        for _ in range(args.steps):
            ctx.compress_with_lse(x.qwin, x.k, x.v, lse, budget, ko, vo, idx)
        g1.record(stream)
        torch.cuda.synchronize()
        line["with_prefill_normalisers"] = {
            "ms_per_step": g0.elapsed_time(g1) / args.steps,
            "what": "bacon_compress_with_lse: the window rows' softmax normalisers come from the "
                    "prefill attention, so the first pass over K is skipped"}
        del lse

        # the paper's ablation / sensitivity grid, every variant selected from
        # one set of window passes (indices only, no gather)
        variants = list(workloads.SWEEP_VARIANTS)
        sidx, slam = ctx.sweep(x.qwin, x.k, budget, variants)
        for _ in range(3):
            ctx.sweep(x.qwin, x.k, budget, variants, sidx, slam)
        torch.cuda.synchronize()
        g0.record(stream)
        for _ in range(args.steps):
            ctx.sweep(x.qwin, x.k, budget, variants, sidx, slam)
        g1.record(stream)
        torch.cuda.synchronize()
        sweep_ms = g0.elapsed_time(g1) / args.steps
        line["ablation_sweep"] = {
            "variants": len(variants), "ms_per_sweep": sweep_ms,
            "ms_per_variant": sweep_ms / len(variants),
            "separate_whole_steps_ms": len(variants) * ms,
            "what": "bacon_sweep over the component ablation and the m / r sensitivity grid: "
                    "one set of window passes, then calibration and selection per variant"}
        del sidx, slam

    # end to end through the host-buffer C call: H2D inputs, compress, D2H outputs
    if not args.no_e2e:
        del x
        torch.cuda.empty_cache()
        hx = workloads.generate(wl, seed=rank, device=dev)
        hq, hk, hv = (t.cpu().pin_memory() for t in (hx.qwin, hx.k, hx.v))
        del hx
        torch.cuda.empty_cache()
        shape_o = (wl.requests, wl.layers, wl.kv_heads, kept, wl.head_dim)
        hko = torch.empty(shape_o, dtype=torch.bfloat16, pin_memory=True)
        hvo = torch.empty(shape_o, dtype=torch.bfloat16, pin_memory=True)
        hidx = torch.empty(shape_o[:-1], dtype=torch.int32, pin_memory=True)
        ctx.compress_host(hq, hk, hv, budget, hko, hvo, hidx)
        barrier()
        torch.cuda.synchronize()
        # the call returns once the outputs are on the host (it overlaps its
        # own copy streams with the compute), so the wall clock is the
        # end-to-end time
        t0 = time.perf_counter()
        for _ in range(args.e2e_steps):
            ctx.compress_host(hq, hk, hv, budget, hko, hvo, hidx)
        torch.cuda.synchronize()
        e2e_ms = reduce_step_time((time.perf_counter() - t0) * 1e3 / args.e2e_steps, world, dev)
        # page-locked values are not uploaded: the gather reads the kept rows
        # in place (the library's host path), so only those rows cross
        v_rows = units * kept * wl.head_dim * hv.element_size()
        h2d = sum(t.numel() * t.element_size() for t in (hq, hk)) + (
            v_rows if hv.is_pinned() else hv.numel() * hv.element_size())
        d2h = sum(t.numel() * t.element_size() for t in (hko, hvo, hidx))
        line["e2e"] = {"value": job_throughput(units, world, e2e_ms), "unit": UNIT,
                       "ms_per_step": e2e_ms, "h2d_bytes_per_step": h2d,
                       "d2h_bytes_per_step": d2h, "steps": args.e2e_steps,
                       "path": "bacon_compress_host (pinned host buffers; queries and keys "
                               "uploaded, kept value rows read in place)"}
    ctx.close()

    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(wl, budget)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
