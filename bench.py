#!/usr/bin/env python3
"""Benchmark of one verification step on GB300: tree attention + argmax/accept
walk + KV compaction through the C ABI, on synthetic inputs of the 7B-class
L=4096 workload (32 heads MHA, D=128, 64-node tree, V=125696, bf16).

Prints ONE JSON line (rank 0).  ``value`` is whole-job verify steps/s with the
inputs resident in HBM, timed with CUDA events over exactly --steps steps
(each step replays a CUDA graph holding the three library calls, the
attention and the argmax/accept call running concurrently on two streams), bracketed by
a barrier and a device synchronize.  Input sets rotate so that their total is
larger than three times the L2 cache.  ``roofline`` reports the attention
kernel's algorithmic bytes per launch over its event-timed duration against
the measured HBM copy bandwidth.  ``e2e`` repeats the step through the public
API from pinned host buffers, copies included.  ``cpu_baseline`` times the fp64
oracle on the host cores.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--impl ours|reference]

Under torchrun (N > 1) every rank runs its own replica of the workload on its
own GPU (sequences are independent: weak scaling, no collective on the data
path); rank 0 prints the line with the max time over ranks.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import torch  # noqa: E402

METRIC = "verify steps/sec and tree-attn achieved HBM GB/s (% of GB300 peak) at 1 GPU"
UNIT = "verify steps/s"
DEFAULT_WORKLOAD = "7b_l4096"
L2_BYTES = 129 * 1000 * 1000
FALLBACK_HBM_GBS = 6800.0
KERNEL_SOURCES = {
    "tree_attn": ["tree_attn_tc.cu", "tc_ptx.cuh", "tmap_host.cuh", "common.cuh", "abi.cu"],
    "accept": ["accept.cu", "common.cuh"],
    "kv_compact": ["kv_compact.cu", "common.cuh"],
}


# ---------------------------------------------------------------------------
# distributed plumbing (also exercised by the CPU gloo tests)
# ---------------------------------------------------------------------------

def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def dist_init(world: int, backend: str):
    import torch.distributed as dist
    if world > 1 and not dist.is_initialized():
        dist.init_process_group(backend=backend)
    return dist if world > 1 else None


def barrier(dist, device=None):
    if dist is not None:
        if device is not None and device.type == "cuda":
            dist.barrier(device_ids=[device.index])
        else:
            dist.barrier()


def max_over_ranks(dist, x: float, device=None) -> float:
    if dist is None:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device if device is not None else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def aggregate(seconds_max: float, steps: int, world: int) -> tuple[float, float]:
    """(whole-job steps/s, ms per step) from the slowest rank's time."""
    ms = 1e3 * seconds_max / steps
    return world * steps / seconds_max, ms


# ---------------------------------------------------------------------------
# workload accounting
# ---------------------------------------------------------------------------

def attn_bytes_per_launch(w, lengths) -> int:
    """Algorithmic bytes of one attention launch: every committed K/V row and
    the T tree K/V rows read once, q read once, out written once."""
    e = w.elem_bytes
    kv = 2 * w.Hkv * w.D * e * sum(L + w.T for L in lengths)
    q = w.B * w.T * w.Hq * w.D * e
    return kv + 2 * q


def attn_flops_per_launch(w, lengths) -> int:
    return 4 * w.Hq * w.T * w.D * sum(L + w.T for L in lengths)


def argmax_bytes_per_launch(w) -> int:
    return w.B * w.T * w.V * w.elem_bytes


def source_hash(kernel: str) -> str:
    h = hashlib.sha256()
    for fn in KERNEL_SOURCES[kernel]:
        with open(os.path.join(ROOT, "paper_2405_00263_gb300", "csrc", fn), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def recorded_traffic(kernel: str, workload: str):
    """DRAM bytes per launch from the committed ncu summary, if it was taken on
    the current kernel source for this workload (else None)."""
    path = os.path.join(ROOT, "profiles", "ncu_traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f).get(kernel, {}).get(workload)
    except (OSError, ValueError):
        return None
    if not rec or rec.get("source_sha256_16") != source_hash(kernel):
        return None
    return rec.get("dram_bytes_per_launch")


def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f), "measured"
    except (OSError, ValueError):
        return {"hbm_gbs": FALLBACK_HBM_GBS}, "fallback"


# ---------------------------------------------------------------------------
# clocks during the timed region
# ---------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ["index", "clocks.sm", "clocks.max.sm", "power.draw", "clocks_event_reasons.active",
              "clocks_event_reasons.hw_slowdown", "clocks_event_reasons.hw_thermal_slowdown",
              "clocks_event_reasons.sw_thermal_slowdown", "clocks_event_reasons.sw_power_cap"]
    REASONS = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]

    def __init__(self, device_index: int):
        self.proc = None
        self.lines = []
        self.t0 = self.t1 = None
        target = str(device_index)
        try:
            uuid = str(torch.cuda.get_device_properties(device_index).uuid)
            target = uuid if uuid.startswith("GPU-") else "GPU-" + uuid
        except Exception:
            pass
        self.cmd = ["nvidia-smi", f"--query-gpu={','.join(self.FIELDS)}", "--format=csv,noheader,nounits",
                    "-lms", "100", "-i", target]

    def start(self):
        try:
            self.proc = subprocess.Popen(self.cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.reader = threading.Thread(target=self._read, daemon=True)
        self.reader.start()
        time.sleep(0.3)

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.time(), line.strip()))

    def mark(self, which: str):
        setattr(self, which, time.time())

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0,
                    "note": "nvidia-smi unavailable"}
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.reader.join(timeout=2)
        rows = []
        for ts, line in self.lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) != len(self.FIELDS):
                continue
            rows.append((ts, parts))
        inside = [r for r in rows if self.t0 is not None and self.t0 <= r[0] <= (self.t1 or 1e30)]
        note = "samples inside the timed region"
        if not inside and rows:
            # region shorter than the sampling period: nearest samples around it
            inside = sorted(rows, key=lambda r: abs(r[0] - (self.t0 or 0)))[:3]
            note = "timed region shorter than the 100 ms sampling period: nearest samples"
        def num(x):
            try:
                return float(x)
            except ValueError:
                return None
        sm = [num(p[1]) for _, p in inside if num(p[1]) is not None]
        smax = [num(p[2]) for _, p in inside if num(p[2]) is not None]
        reasons = set()
        for _, p in inside:
            for name, val in zip(self.REASONS, p[5:9]):
                if val.lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(inside), "note": note,
                "power_w_max": max((num(p[3]) or 0.0) for _, p in inside) if inside else None}


# ---------------------------------------------------------------------------
# the GPU arm
# ---------------------------------------------------------------------------

def make_sets(w, device, n_sets):
    from synth import workloads
    base = workloads.make(w, device=device)
    keys = ("q", "k_new", "v_new", "k_cache", "v_cache", "cache_len", "parent", "cand", "logits")
    sets = [{k: base[k] for k in keys}]
    for _ in range(n_sets - 1):
        sets.append({k: base[k].clone() for k in keys})
    return base, sets


def page_sets(w, sets, page_size, Lcap):
    """Replace every set's dense caches by page pools under a seeded block
    table (synth.paging), giving each sequence pages for L + T slots.  Returns
    the capacity page_size * max_pages."""
    from synth import paging, workloads
    max_pages = -(-Lcap // page_size)
    need = [L + w.T for L in workloads.cache_lengths(w)]
    for i, s in enumerate(sets):
        table, n_pages = paging.page_table(need, page_size, max_pages, seed=w.seed * 131 + i)
        dev = s["k_cache"].device
        s["k_cache"] = paging.to_pages(s["k_cache"].cpu(), table, page_size, n_pages).to(dev)
        s["v_cache"] = paging.to_pages(s["v_cache"].cpu(), table, page_size, n_pages).to(dev)
        s["block_table"] = table.to(dev)
    return max_pages * page_size


def set_bytes(s) -> int:
    return sum(t.numel() * t.element_size() for t in s.values())


def run_gpu_arm(args, world, rank, local, dist):
    import paper_2405_00263_gb300 as pkg
    from synth import workloads

    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    w = workloads.get(args.workload)
    lengths = workloads.cache_lengths(w)
    base, sets = make_sets(w, device, 1)
    per_set = set_bytes(sets[0])
    n_sets = max(2, min(12, math.ceil(3 * L2_BYTES / per_set)))
    del base, sets
    base, sets = make_sets(w, device, n_sets)
    Lcap = base["Lcap"]
    if args.page_size:
        Lcap = page_sets(w, sets, args.page_size, Lcap)
    step = pkg.VerifyStep(w.B, w.T, w.Hq, w.Hkv, w.D, Lcap, w.V, w.torch_dtype, device=device,
                          accept=args.accept, temperature=args.temperature, epsilon=args.epsilon,
                          delta=args.delta, schedule=args.schedule, page_size=args.page_size or None)
    stream = torch.cuda.Stream(device)

    ext_ok = True
    try:
        torch.cuda.Event(enable_timing=True, external=True)
    except TypeError:
        ext_ok = False

    def launch(s, evs=None):
        step.run(s["q"], s["k_new"], s["v_new"], s["k_cache"], s["v_cache"], s["cache_len"], s["parent"],
                 s["cand"], s["logits"], stream=stream, events=evs, block_table=s.get("block_table"))

    # eager warm-up (also initialises per-kernel attributes before capture)
    with torch.cuda.stream(stream):
        for i in range(max(1, args.warmup)):
            launch(sets[i % n_sets])
    stream.synchronize()
    if step.device_status() != 0:
        raise RuntimeError(f"device status {step.device_status()} during warm-up")

    # one CUDA graph per input set and replica; the graphs of the first replica
    # carry two timing events around the attention (an event node costs about
    # a microsecond of the step, so the other calls are timed after the timed
    # region)
    reps = 4
    graphs, graph_events = [], []
    for r in range(reps):
        for s in sets:
            evs = [torch.cuda.Event(enable_timing=True, external=True) for _ in range(2)] \
                if ext_ok and r == 0 else None
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                launch(s, evs)
            graphs.append(g)
            graph_events.append(evs)
    torch.cuda.synchronize(device)
    for i in range(max(3, args.warmup)):
        graphs[i % len(graphs)].replay()
    torch.cuda.synchronize(device)

    sampler = ClockSampler(local) if rank == 0 else None
    if sampler:
        sampler.start()
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    barrier(dist, device)
    torch.cuda.synchronize(device)
    if sampler:
        sampler.mark("t0")
    with torch.cuda.stream(stream):
        start.record(stream)
        for i in range(args.steps):
            graphs[i % len(graphs)].replay()
        end.record(stream)
    end.synchronize()
    torch.cuda.synchronize(device)
    if sampler:
        sampler.mark("t1")
    barrier(dist, device)
    seconds = start.elapsed_time(end) / 1e3
    clocks = sampler.stop() if sampler else None
    seconds_max = max_over_ranks(dist, seconds, device)
    value, ms = aggregate(seconds_max, args.steps, world)
    if step.device_status() != 0:
        raise RuntimeError(f"device status {step.device_status()} in the timed region")

    # per-kernel durations.  The attention: the in-graph events of the last
    # replay of every event-carrying graph inside the timed region.  The accept
    # and commit calls: each launched alone after an L2 flush by a large read
    # (which keeps the GPU busy while the call is queued, so the events bracket
    # the kernel and not the host's launch latency), after the timed region.
    durations = {"tree_attn": []}
    timing_source = {"tree_attn": "events inside the replayed graphs of the timed region",
                     "accept": "launched alone after an L2 flush, events on the launching stream",
                     "kv_commit": "launched alone after an L2 flush, events on the launching stream"}
    timed_graphs = [evs for i, evs in enumerate(graph_events) if evs and i < args.steps]
    for evs in timed_graphs:
        durations["tree_attn"].append(evs[0].elapsed_time(evs[1]) * 1e3)
    if not timed_graphs:
        for i in range(3 * len(sets)):
            evs = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
            with torch.cuda.stream(stream):
                launch(sets[i % n_sets], evs)
            torch.cuda.synchronize(device)
            durations["tree_attn"].append(evs[0].elapsed_time(evs[1]) * 1e3)
        timing_source["tree_attn"] = "eager steps with events after the timed region (no external graph events)"
    us = {k: statistics.mean(v) for k, v in durations.items()}
    flush = torch.zeros(2 * L2_BYTES, dtype=torch.uint8, device=device)
    us["accept"] = accept_kernel_us(pkg, w, sets, stream, device, args.accept, args, flush)
    other = "greedy" if args.accept == "typical" else "typical"
    us_other = accept_kernel_us(pkg, w, sets, stream, device, other, args, flush)
    def commit_call(i):
        c = sets[i % n_sets]
        if args.page_size:
            pkg.clover_kv_commit_paged(c["k_cache"], c["v_cache"], c["block_table"], c["k_new"], c["v_new"],
                                       c["cache_len"], step.path, step.accept_len, step.new_cache_len,
                                       step.src_index, status=step.status_accept, stream=stream)
        else:
            pkg.clover_kv_commit(c["k_cache"], c["v_cache"], c["k_new"], c["v_new"], c["cache_len"], step.path,
                                 step.accept_len, step.new_cache_len, step.src_index, status=step.status_accept,
                                 stream=stream)

    us["kv_commit"] = isolated_us(commit_call, 3 * len(sets), stream, flush)
    del flush
    if step.device_status() != 0:
        raise RuntimeError(f"device status {step.device_status()} in the per-kernel timing")

    peaks, peak_kind = measured_peaks()
    hbm = float(peaks.get("hbm_gbs", FALLBACK_HBM_GBS))
    a_bytes = attn_bytes_per_launch(w, lengths)
    achieved = a_bytes / (us["tree_attn"] * 1e-6) / 1e9
    traffic = recorded_traffic("tree_attn", w.name + (f"_paged{args.page_size}" if args.page_size else ""))
    am_bytes = argmax_bytes_per_launch(w)

    # end to end through the public API from pinned host buffers
    e2e = run_e2e(args, w, step, sets, stream, device, dist, world)

    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16" if w.dtype == "bf16" else "f32", "data": "synthetic",
        "config": {"workload": f"{w.name}: {w.description}", "B": w.B, "T": w.T, "Hq": w.Hq, "Hkv": w.Hkv,
                   "D": w.D, "L": lengths if len(lengths) <= 4 else f"{len(lengths)} lengths, sum {sum(lengths)}",
                   "V": w.V, "Lcap": Lcap, "parallelism": f"replicas x{world} (one per GPU)",
                   "kv_cache": (f"paged, {args.page_size}-slot pages scattered over the pool by a seeded table"
                                if args.page_size else "dense [B, Hkv, Lcap, D]"),
                   "l2": f"{n_sets} rotating input sets of {per_set / 1e6:.1f} MB "
                         f"({n_sets * per_set / 1e6:.0f} MB > 3x the 129 MB L2)",
                   "launch": LAUNCH_DESC[args.schedule],
                   "accept": accept_desc(args)},
        "roofline": {"bound": "hbm", "kernel": "tree_attn", "achieved": achieved, "peak": hbm, "unit": "GB/s",
                     "frac": achieved / hbm, "peak_source": f"{peak_kind} hbm_gbs (MEASURED_PEAKS.json)"
                     if peak_kind == "measured" else "fallback 6.8 TB/s",
                     "traffic": traffic, "bytes_per_launch": a_bytes, "launch_us": us["tree_attn"],
                     "frac_of_8TBs": achieved / 8000.0,
                     "flops_per_launch": attn_flops_per_launch(w, lengths),
                     "timing": timing_source["tree_attn"]},
        "kernels": {"tree_attn_us": us["tree_attn"], "accept_us": us["accept"], "kv_commit_us": us["kv_commit"],
                    "accept_rule": args.accept,
                    "accept_bytes_per_launch": am_bytes,
                    "accept_gbs": am_bytes / (us["accept"] * 1e-6) / 1e9,
                    "accept_frac": am_bytes / (us["accept"] * 1e-6) / 1e9 / hbm,
                    f"accept_{other}": {"us": us_other, "gbs": am_bytes / (us_other * 1e-6) / 1e9,
                                        "frac": am_bytes / (us_other * 1e-6) / 1e9 / hbm,
                                        "timing": timing_source["accept"]}},
        "gpu_launches": (2 if args.schedule == "fused" else 3) * args.steps,
        "timing": timing_source,
        "clocks": clocks,
        "e2e": e2e,
    }
    return line, w, base


LAUNCH_DESC = {
    "commit": "one CUDA graph replay per step: the attention (cache read only) on one stream, argmax/accept "
              "then the commit of the accepted K/V on a second stream",
    "compact": "one CUDA graph replay per step: the attention (appending the tree K/V) on one stream and "
               "argmax/accept on a second, then the compaction of the accepted K/V",
    "fused": "one CUDA graph replay per step, two launches on one stream: the attention (cache read only), then "
             "argmax/accept with the commit of the accepted K/V fused in, launched as a programmatic dependent "
             "of the attention so that it runs beside it",
}


def accept_desc(args) -> str:
    if args.accept == "typical":
        return (f"typical acceptance (temperature {args.temperature}, epsilon {args.epsilon}, "
                f"delta {args.delta})")
    return "greedy"


def isolated_us(call, n, stream, flush) -> float:
    """Mean event-timed duration of call(i), i < n, each launched alone on
    ``stream`` right after a read of ``flush`` (twice the L2: the L2 then holds
    only clean lines of it, so the call pays no write-back of a flush)."""
    times = []
    with torch.cuda.stream(stream):
        for i in range(n + 2):
            torch.amax(flush)
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            call(i)
            b.record(stream)
            b.synchronize()
            if i >= 2:
                times.append(a.elapsed_time(b) * 1e3)
    return statistics.mean(times)


def accept_kernel_us(pkg, w, sets, stream, device, rule, args, flush) -> float:
    """Mean duration of one acceptance call of ``rule`` (own outputs and
    workspace) over the rotating input sets."""
    i32 = dict(dtype=torch.int32, device=device)
    outs = [torch.empty((w.B, w.T), **i32), torch.empty((w.B, w.T), **i32), torch.empty(w.B, **i32),
            torch.empty(w.B, **i32)]
    size = (pkg.clover_verify_accept_typical_workspace_size if rule == "typical"
            else pkg.clover_verify_accept_workspace_size)(w.B, w.T, w.V, w.torch_dtype)
    ws = torch.zeros(size, dtype=torch.uint8, device=device)
    status = torch.zeros(1, **i32)

    def call(i):
        s = sets[i % len(sets)]
        if rule == "typical":
            pkg.clover_verify_accept_typical(s["logits"], s["cand"], s["parent"], args.temperature, args.epsilon,
                                             args.delta, *outs, ws, status=status, stream=stream)
        else:
            pkg.clover_verify_accept(s["logits"], s["cand"], s["parent"], *outs, ws, status=status, stream=stream)

    t = isolated_us(call, 3 * len(sets), stream, flush)
    if int(status.item()) != 0:
        raise RuntimeError(f"device status {int(status.item())} in the {rule} acceptance timing")
    return t


def run_e2e(args, w, step, sets, stream, device, dist, world):
    """Same steps through the public API: inputs copied from pinned host memory,
    the step's results (attention output, path, accepted length, bonus token,
    new length) read back, copies inside the timed region."""
    import paper_2405_00263_gb300 as pkg

    src = sets[0]
    inputs = ("q", "k_new", "v_new", "cache_len", "parent", "cand", "logits")
    host_in = {k: src[k].cpu().pin_memory() for k in inputs}
    dev_in = [{k: s[k] for k in inputs} for s in sets]
    outs = (step.out, step.path, step.accept_len, step.bonus, step.new_cache_len)
    host_out = [torch.empty(o.shape, dtype=o.dtype).pin_memory() for o in outs]
    h2d = sum(t.numel() * t.element_size() for t in host_in.values())
    d2h = sum(t.numel() * t.element_size() for t in host_out)
    n = max(10, min(args.steps, 200))

    def one(i):
        s = sets[i % len(sets)]
        d = dev_in[i % len(sets)]
        for k in inputs:
            d[k].copy_(host_in[k], non_blocking=True)
        step.run(d["q"], d["k_new"], d["v_new"], s["k_cache"], s["v_cache"], d["cache_len"], d["parent"],
                 d["cand"], d["logits"], stream=stream, block_table=s.get("block_table"))
        for h, o in zip(host_out, outs):
            h.copy_(o, non_blocking=True)

    with torch.cuda.stream(stream):
        for i in range(3):
            one(i)
    stream.synchronize()
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    barrier(dist, device)
    torch.cuda.synchronize(device)
    with torch.cuda.stream(stream):
        start.record(stream)
        for i in range(n):
            one(i)
        end.record(stream)
    end.synchronize()
    seconds = max_over_ranks(dist, start.elapsed_time(end) / 1e3, device)
    value, ms = aggregate(seconds, n, world)
    return {"value": value, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "steps": n, "ms_per_step": ms, "api": "paper_2405_00263_gb300.VerifyStep.run (C ABI)"}


# ---------------------------------------------------------------------------
# the oracle on the host cores
# ---------------------------------------------------------------------------

def typical_params(args):
    return (args.temperature, args.epsilon, args.delta) if args.accept == "typical" else None


def oracle_step_seconds(host: dict, threads: int, typical=None) -> float:
    import oracle
    t0 = time.perf_counter()
    oracle.verify_step(host, n_threads=threads, typical=typical)
    return time.perf_counter() - t0


def cpu_baseline(w, host: dict, args, budget_s: float = 8.0) -> dict:
    """Whole oracle verify steps (fp64 attention over every row, argmax over
    every logit row, walk, append, compaction) repeated within a time budget."""
    import oracle
    oracle.build()
    threads = os.cpu_count() or 1
    typ = typical_params(args)
    times = [oracle_step_seconds(host, threads, typ)]
    while sum(times) < budget_s and len(times) < 50:
        times.append(oracle_step_seconds(host, threads, typ))
    per = statistics.median(times)
    return {"value": 1.0 / per, "unit": UNIT, "cores": threads, "kind": "oracle",
            "sample": f"{len(times)} whole verify steps of {w.name} (fp64 oracle, OpenMP over attention rows "
                      f"and logit rows, {accept_desc(args)}), median {per * 1e3:.1f} ms per step"}


def run_reference_arm(args, world, rank):
    from synth import workloads
    if rank != 0:
        return None
    w = workloads.get(args.workload)
    host = workloads.make(w)
    import oracle
    oracle.build()
    threads = os.cpu_count() or 1
    typ = typical_params(args)
    for _ in range(args.warmup):
        oracle_step_seconds(host, threads, typ)
    t = [oracle_step_seconds(host, threads, typ) for _ in range(args.steps)]
    total = sum(t)
    value = args.steps / total
    return {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f64", "data": "synthetic",
            "config": {"workload": f"{w.name}: {w.description}", "parallelism": "host cores (rank 0 only)",
                       "accept": accept_desc(args)},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle",
                             "sample": f"{args.steps} whole verify steps of {w.name} on the host (fp64 oracle)"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "gpu_launches": 0}


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--accept", default="greedy", choices=["greedy", "typical"],
                    help="acceptance rule of the step (typical: tempered softmax with an entropy threshold)")
    ap.add_argument("--page-size", type=int, default=0,
                    help="run on a paged KV cache with pages of this many slots (0: dense cache)")
    ap.add_argument("--schedule", default="commit", choices=["commit", "compact", "fused"],
                    help="call schedule of the step (VerifyStep)")
    ap.add_argument("--temperature", type=float, default=1.0)
    ap.add_argument("--epsilon", type=float, default=0.09)
    ap.add_argument("--delta", type=float, default=0.3)
    args = ap.parse_args(argv)
    if args.warmup < 3:
        args.warmup = 3
    world, rank, local = dist_env()

    if args.impl == "reference":
        line = run_reference_arm(args, world, rank)
        if line is not None:
            print(json.dumps(line), flush=True)
        return 0

    dist = dist_init(world, "nccl" if torch.cuda.is_available() else "gloo")
    line, w, base = run_gpu_arm(args, world, rank, local, dist)
    if rank == 0:
        if world == 1 and not args.no_cpu_baseline:
            host = {k: (v.cpu() if isinstance(v, torch.Tensor) else v) for k, v in base.items()}
            line["cpu_baseline"] = cpu_baseline(w, host, args)
        else:
            line["cpu_baseline"] = None
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
