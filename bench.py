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
STEP_PASSES = 4          # passes over the input sets in one captured graph of steps
FALLBACK_HBM_GBS = 6800.0
FALLBACK_BF16_TFLOPS = 1900.0
FALLBACK_BF16_TFLOPS_SUSTAINED = 1700.0
KERNEL_SOURCES = {
    "tree_attn": ["tree_attn_tc.cu", "tree_attn_tc_pair.cu", "tc_ptx.cuh", "tmap_host.cuh", "common.cuh", "ctx_host.cuh",
                  "abi.cu"],
    "accept": ["accept.cu", "common.cuh", "ctx_host.cuh"],
    "kv_compact": ["kv_compact.cu", "common.cuh", "ctx_host.cuh"],
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
                    "-lms", "20", "-i", target]

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
            note = "timed region shorter than the 20 ms sampling period: nearest samples"
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
                          delta=args.delta, schedule=args.schedule, page_size=args.page_size or None,
                          attn_launch=args.attn_launch)
    stream = torch.cuda.Stream(device)

    def launch(s):
        step.run(s["q"], s["k_new"], s["v_new"], s["k_cache"], s["v_cache"], s["cache_len"], s["parent"],
                 s["cand"], s["logits"], stream=stream, block_table=s.get("block_table"))

    # eager warm-up (also initialises per-kernel attributes before capture)
    with torch.cuda.stream(stream):
        for i in range(max(1, args.warmup)):
            launch(sets[i % n_sets])
    stream.synchronize()
    if step.device_status() != 0:
        raise RuntimeError(f"device status {step.device_status()} during warm-up")

    # CUDA graphs of consecutive steps: the full graph runs STEP_PASSES steps on
    # every input set in turn, each step's calls queued behind the previous
    # step's (as in a decoding loop captured as one graph); single-step graphs
    # time the remainder of K.  The timed graphs carry no timing nodes.
    per_graph = STEP_PASSES * n_sets
    full = torch.cuda.CUDAGraph()
    with torch.cuda.graph(full, stream=stream):
        for _ in range(STEP_PASSES):
            for s in sets:
                launch(s)
    singles = []
    for i in range(args.steps % per_graph):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            launch(sets[i % n_sets])
        singles.append(g)
    torch.cuda.synchronize(device)
    for _ in range(max(1, -(-max(3, args.warmup) // per_graph))):
        full.replay()
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
        for _ in range(args.steps // per_graph):
            full.replay()
        for g in singles:
            g.replay()
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
    del full, singles

    # per-kernel durations, after the timed region.  The attention: its
    # average launch duration over back-to-back launches on the rotating input
    # sets (inputs larger than the L2), one CUDA graph, events around the
    # replays.  The accept and commit calls: each launched alone after an L2
    # flush by a large read (which keeps the GPU busy while the call is queued,
    # so the events bracket the kernel and not the host's launch latency).
    timing_source = {"tree_attn": f"back-to-back attention launches ({step.attn_launch} launch) over the {n_sets} "
                                  "rotating input sets, four passes in one CUDA graph, events around the replays, "
                                  "after the timed region",
                     "accept": "launched alone after an L2 flush (a read of twice the L2), device time: CUDA graphs of (flush, call) pairs less graphs of the flushes alone",
                     "kv_commit": "launched alone after an L2 flush (a read of twice the L2), device time: CUDA graphs of (flush, call) pairs less graphs of the flushes alone"}
    us = {"tree_attn": attn_launch_us(step, sets, stream, device, args, mode=step.attn_launch)}
    us["tree_attn_ordinary"] = (us["tree_attn"] if step.attn_launch == "ordinary"
                                else attn_launch_us(step, sets, stream, device, args, mode="ordinary"))
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
    tc_peak = float(peaks.get("bf16_tflops", FALLBACK_BF16_TFLOPS))
    tc_sustained = float(peaks.get("bf16_tflops_sustained", FALLBACK_BF16_TFLOPS_SUSTAINED))
    a_bytes = attn_bytes_per_launch(w, lengths)
    a_flops = attn_flops_per_launch(w, lengths)
    achieved = a_bytes / (us["tree_attn"] * 1e-6) / 1e9
    tflops = a_flops / (us["tree_attn"] * 1e-6) / 1e12
    # the bound of this shape: HBM when its bytes take longer at the measured
    # copy rate than its flops at the measured bf16 rate, else the tensor pipe
    tensor_bound = a_flops / (tc_peak * 1e12) > a_bytes / (hbm * 1e9)
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
                   "attn_launch": step.attn_launch,
                   "accept": accept_desc(args)},
        "roofline": {"bound": "tensor" if tensor_bound else "hbm", "kernel": "tree_attn",
                     "achieved": tflops if tensor_bound else achieved, "peak": tc_peak if tensor_bound else hbm,
                     "unit": "TFLOP/s" if tensor_bound else "GB/s",
                     "frac": tflops / tc_peak if tensor_bound else achieved / hbm,
                     "peak_source": (f"{peak_kind} " + ("bf16_tflops (burst: the kernel is timed alone)"
                                                        if tensor_bound else "hbm_gbs") + " (MEASURED_PEAKS.json)")
                     if peak_kind == "measured" else ("fallback 1.9 PFLOP/s bf16" if tensor_bound
                                                      else "fallback 6.8 TB/s"),
                     "hbm_gbs": achieved, "frac_hbm": achieved / hbm, "tflops": tflops,
                     "frac_tensor": tflops / tc_peak,
                     # against the sustained bf16 rate (a seconds-long GEMM loop under the power cap)
                     "frac_tensor_sustained": tflops / tc_sustained,
                     "traffic": traffic, "bytes_per_launch": a_bytes, "launch_us": us["tree_attn"],
                     "attn_launch": step.attn_launch,
                     "launch_us_ordinary": us["tree_attn_ordinary"],
                     # an ordinary launch against the same bound's peak, and against HBM
                     "frac_ordinary": (a_flops / (us["tree_attn_ordinary"] * 1e-6) / 1e12 / tc_peak if tensor_bound
                                       else a_bytes / (us["tree_attn_ordinary"] * 1e-6) / 1e9 / hbm),
                     "frac_hbm_ordinary": a_bytes / (us["tree_attn_ordinary"] * 1e-6) / 1e9 / hbm,
                     "frac_of_8TBs": achieved / 8000.0,
                     "flops_per_launch": attn_flops_per_launch(w, lengths),
                     "timing": timing_source["tree_attn"],
                     # the whole step against HBM: the attention's bytes and
                     # the logits read by the argmax (the commit's few rows,
                     # under 0.3 % here, left out) per ms_per_step
                     "step": {"bytes": a_bytes + am_bytes,
                              "gbs": (a_bytes + am_bytes) / (ms * 1e-3) / 1e9,
                              "frac": (a_bytes + am_bytes) / (ms * 1e-3) / 1e9 / hbm}},
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
    "commit": "CUDA graphs of consecutive steps (four passes over the input sets, each step queued behind the last); a step: the "
              "attention (cache read only) on one stream, argmax/accept then the commit of the accepted K/V on a "
              "second stream",
    "compact": "CUDA graphs of consecutive steps (four passes over the input sets, each step queued behind the last); a step: the "
               "attention (appending the tree K/V) on one stream and argmax/accept on a second, then the "
               "compaction of the accepted K/V",
    "fused": "CUDA graphs of consecutive steps (four passes over the input sets, each step queued behind the last); a step: two "
             "launches on one stream, the attention (cache read only), then argmax/accept with the commit of the "
             "accepted K/V fused in, launched as a programmatic dependent of the attention so that it runs "
             "beside it",
}


def accept_desc(args) -> str:
    if args.accept == "typical":
        return (f"typical acceptance (temperature {args.temperature}, epsilon {args.epsilon}, "
                f"delta {args.delta})")
    return "greedy"


def attn_launch_us(step, sets, stream, device, args, mode: str, launches: int = 200, passes: int = 4) -> float:
    """Mean duration of the step's attention call over back-to-back launches
    on the rotating input sets, launched as ``mode`` (VerifyStep.ATTN_LAUNCHES):
    one CUDA graph of ``passes`` launches per set, replayed until about
    ``launches`` launches, CUDA events around the replays."""
    import paper_2405_00263_gb300 as pkg
    kw = pkg.VerifyStep.ATTN_LAUNCHES[mode]

    def attn(s):
        if args.page_size:
            pkg.clover_verify_attn_paged(s["q"], s["k_new"], s["v_new"], s["k_cache"], s["v_cache"],
                                         s["block_table"], s["cache_len"], s["parent"], step.out,
                                         workspace=step.ws_attn, status=step.status, stream=stream, **kw)
        else:
            pkg.clover_verify_attn(s["q"], s["k_new"], s["v_new"], s["k_cache"], s["v_cache"], s["cache_len"],
                                   s["parent"], step.out, workspace=step.ws_attn, status=step.status,
                                   stream=stream, append=args.schedule == "compact", **kw)

    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for _ in range(passes):
            for s in sets:
                attn(s)
    reps = max(3, launches // (passes * len(sets)))
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        for _ in range(3):
            g.replay()
        a.record(stream)
        for _ in range(reps):
            g.replay()
        b.record(stream)
    b.synchronize()
    if step.device_status() != 0:
        raise RuntimeError(f"device status {step.device_status()} in the attention timing")
    return a.elapsed_time(b) * 1e3 / (reps * passes * len(sets))


def isolated_us(call, n, stream, flush, reps: int = 10) -> float:
    """Mean duration of call(i), i < n, each launched alone on ``stream`` right
    after a read of ``flush`` (twice the L2: the L2 then holds only clean lines
    of it, so the call pays no write-back of a flush).  Device time only: one
    CUDA graph holds the n (flush, call) pairs and another the n flushes alone;
    both are replayed ``reps`` times between CUDA events, and the difference is
    the calls' time (with no host launch latency in it)."""
    with torch.cuda.stream(stream):
        for i in range(n):                  # eager first: per-kernel attributes outside the capture
            call(i)
    stream.synchronize()
    g_pairs, g_flush = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_pairs, stream=stream):
        for i in range(n):
            torch.amax(flush)
            call(i)
    with torch.cuda.graph(g_flush, stream=stream):
        for i in range(n):
            torch.amax(flush)

    def timed(g):
        with torch.cuda.stream(stream):
            g.replay()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            for _ in range(reps):
                g.replay()
            b.record(stream)
        b.synchronize()
        return a.elapsed_time(b) * 1e3

    t_pairs, t_flush = timed(g_pairs), timed(g_flush)
    del g_pairs, g_flush
    return (t_pairs - t_flush) / (n * reps)


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


DRAFT_METRIC = "Clover draft head steps/s (one speculative head: embedding, attention decoder, MLP block, " \
               "shared LM head, top-k) and LM-head achieved HBM GB/s at 1 GPU"
DRAFT_UNIT = "head steps/s"


def run_draft_arm(args, world, rank, local, dist):
    """One speculative head step of a 7B-class Clover draft on R rows: the
    weights are synthetic (seeded normal, std 1/sqrt(H)); the LM head alone
    is 1.03 GB of bf16, so every step streams its weights from HBM."""
    import paper_2405_00263_gb300 as pkg

    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    R, H, V, k = args.draft, 4096, 125696, 8
    gen = torch.Generator(device=device).manual_seed(1234 + rank)

    def rnd(*shape, std=1.0):
        return (torch.randn(*shape, generator=gen, device=device, dtype=torch.float32) * std).to(torch.bfloat16)

    w_lm = rnd(V, H, std=H ** -0.5)
    w_v, w_o, w_1 = (rnd(H, H, std=H ** -0.5) for _ in range(3))
    h = rnd(R, H)
    toks = torch.randint(0, V, (R,), generator=gen, device=device, dtype=torch.int32)
    head = pkg.DraftHead(R, H, V, k, device=device)
    stream = torch.cuda.Stream(device)
    with torch.cuda.stream(stream):
        for _ in range(max(3, args.warmup)):
            head.run(h, toks, w_lm, w_v, w_o, w_1, stream=stream)
    stream.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        head.run(h, toks, w_lm, w_v, w_o, w_1, stream=stream)
    with torch.cuda.stream(stream):
        for _ in range(max(3, args.warmup)):
            g.replay()
    torch.cuda.synchronize(device)
    sampler = ClockSampler(local) if rank == 0 else None
    if sampler:
        sampler.start()
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier(dist, device)
    torch.cuda.synchronize(device)
    if sampler:
        sampler.mark("t0")
    with torch.cuda.stream(stream):
        start.record(stream)
        for _ in range(args.steps):
            g.replay()
        end.record(stream)
    end.synchronize()
    if sampler:
        sampler.mark("t1")
    barrier(dist, device)
    clocks = sampler.stop() if sampler else None
    seconds_max = max_over_ranks(dist, start.elapsed_time(end) / 1e3, device)
    value, ms = aggregate(seconds_max, args.steps, world)
    if int(head.status.item()) != 0:
        raise RuntimeError(f"device status {int(head.status.item())} in the draft timing")

    # the LM head alone: events around one launch (its 1 GB read keeps the L2 cold)
    flush = torch.zeros(2 * L2_BYTES, dtype=torch.uint8, device=device)
    lm_us = isolated_us(lambda i: pkg.clover_linear(head.z, w_lm, head.logits, mode="f32", stream=stream),
                        10, stream, flush)
    topk_us = isolated_us(lambda i: pkg.clover_topk(head.logits, k, head.values, head.indices, head.ws,
                                                    stream=stream), 10, stream, flush)
    del flush
    peaks, peak_kind = measured_peaks()
    hbm = float(peaks.get("hbm_gbs", FALLBACK_HBM_GBS))
    lm_bytes = V * H * 2 + R * H * 2 + R * V * 4
    achieved = lm_bytes / (lm_us * 1e-6) / 1e9

    # end to end: h and the tokens from pinned host memory, the top-k back
    h_host = h.cpu().pin_memory()
    t_host = toks.cpu().pin_memory()
    out_host = torch.empty((R, k), dtype=torch.int32).pin_memory()
    h_dev, t_dev = torch.empty_like(h), torch.empty_like(toks)

    def e2e_step():
        h_dev.copy_(h_host, non_blocking=True)
        t_dev.copy_(t_host, non_blocking=True)
        head.run(h_dev, t_dev, w_lm, w_v, w_o, w_1, stream=stream)
        out_host.copy_(head.indices, non_blocking=True)

    n = max(10, min(args.steps, 200))
    with torch.cuda.stream(stream):
        for _ in range(3):
            e2e_step()
    stream.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        e0.record(stream)
        for _ in range(n):
            e2e_step()
        e1.record(stream)
    e1.synchronize()
    e_val, e_ms = aggregate(max_over_ranks(dist, e0.elapsed_time(e1) / 1e3, device), n, world)

    line = {
        "metric": DRAFT_METRIC, "value": value, "unit": DRAFT_UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic (seeded normal weights, std 1/sqrt(H))",
        "config": {"workload": f"Clover head step, 7B shapes: R{R} rows, H{H}, V{V}, top-{k}",
                   "R": R, "H": H, "V": V, "k": k, "parallelism": f"replicas x{world} (one per GPU)",
                   "l2": "the 1.03 GB LM head is read every step (more than 7x the 129 MB L2)",
                   "launch": "one CUDA graph replay per step: embedding, 4 tcgen05 linear layers "
                             "(W_v, W_o + residual, W_1 residual SiLU, LM head), top-k"},
        "roofline": {"bound": "hbm", "kernel": "linear_tc (LM head)", "achieved": achieved, "peak": hbm,
                     "unit": "GB/s", "frac": achieved / hbm,
                     "peak_source": f"{peak_kind} hbm_gbs (MEASURED_PEAKS.json)" if peak_kind == "measured"
                     else "fallback 6.8 TB/s", "traffic": None, "bytes_per_launch": lm_bytes,
                     "launch_us": lm_us, "flops_per_launch": 2 * R * V * H,
                     "timing": "launched alone after an L2 flush by a large read, device time: CUDA graphs of (flush, call) pairs less graphs of the flushes alone"},
        "kernels": {"lm_head_us": lm_us, "topk_us": topk_us,
                    "topk_gbs": R * V * 4 / (topk_us * 1e-6) / 1e9},
        "gpu_launches": 6 * args.steps,
        "clocks": clocks,
        "e2e": {"value": e_val, "unit": DRAFT_UNIT, "h2d_bytes_per_step": R * H * 2 + R * 4,
                "d2h_bytes_per_step": R * k * 4, "steps": n, "ms_per_step": e_ms,
                "api": "paper_2405_00263_gb300.DraftHead.run (C ABI)"},
    }
    return line, (R, H, V, k, w_lm, w_v, w_o, w_1, h, toks)


def draft_cpu_baseline(inputs, budget_s: float = 8.0) -> dict:
    """The oracle's head step for one row of the same weights (host cores),
    its layers on a tenth of their outputs, scaled to whole layers and to R
    rows (every row costs the same)."""
    import oracle
    oracle.build()
    sampler = DraftOracleSampler([t.cpu() if isinstance(t, torch.Tensor) else t for t in inputs])
    times = []
    while not times or (sum(times) < budget_s and len(times) < 20):
        t0 = time.perf_counter()
        times.append(sampler.seconds(0.1))
        if time.perf_counter() - t0 > budget_s:
            break
    per = statistics.median(times)
    return {"value": 1.0 / per, "unit": DRAFT_UNIT, "cores": os.cpu_count() or 1, "kind": "oracle",
            "sample": f"{len(times)} oracle head steps of 1 row, layers on a 0.1 fraction of their outputs, "
                      f"scaled to whole layers and to {inputs[0]} rows; median {per:.2f} s a step"}


def run_e2e(args, w, step, sets, stream, device, dist, world):
    """Same steps through the public API (VerifyStep.run) with host buffers:
    every step's inputs (q, k_new, v_new, cache_len, parent, cand, logits) are
    copied from pinned host memory and its results (attention output, path,
    accepted length, bonus token, new length) read back, copies inside the
    timed region.  One CUDA graph per input set holds step i on set i, and on a
    copy stream the upload of step i+1's inputs into set i+1 (so the upload
    overlaps the step), then the read-back; step 0's upload is a prologue of
    the timed region.  The KV cache is resident device state and not copied."""
    src = sets[0]
    inputs = ("q", "k_new", "v_new", "cache_len", "parent", "cand", "logits")
    # A step's inputs are views of one buffer (each region 256-byte aligned),
    # in pinned host memory and, per input set, on the device: a step's upload
    # is one copy (each copy has a fixed cost on the copy engine, a few us,
    # which seven separate copies paid seven times).
    layout, off = {}, 0
    for k in inputs:
        nbytes = src[k].numel() * src[k].element_size()
        layout[k] = (off, src[k].dtype, tuple(src[k].shape), nbytes)
        off = (off + nbytes + 255) // 256 * 256

    def views(buf):
        return {k: buf[o:o + nb].view(dt).view(shape) for k, (o, dt, shape, nb) in layout.items()}

    host_buf = torch.empty(off, dtype=torch.uint8).pin_memory()
    host_in = views(host_buf)
    for k in inputs:
        host_in[k].copy_(src[k].cpu())
    dev_bufs = [torch.empty(off, dtype=torch.uint8, device=device) for _ in sets]
    dev_in = [views(buf) for buf in dev_bufs]
    # the step's results (out, path, accept_len, bonus, new_cache_len) are one
    # byte range of the step's output buffer: one read-back copy
    host_res = torch.empty(step.results.numel(), dtype=torch.uint8).pin_memory()
    h2d = off
    d2h = step.results.numel()
    n = max(10, min(args.steps, 200))
    n_sets = len(sets)
    copy_stream = torch.cuda.Stream(device)
    fork, join = torch.cuda.Event(), torch.cuda.Event()

    def upload(i, st):
        with torch.cuda.stream(st):
            dev_bufs[i % n_sets].copy_(host_buf, non_blocking=True)

    def one(i):
        s = sets[i % n_sets]
        d = dev_in[i % n_sets]
        fork.record(stream)
        copy_stream.wait_event(fork)
        upload(i + 1, copy_stream)
        step.run(d["q"], d["k_new"], d["v_new"], s["k_cache"], s["v_cache"], d["cache_len"], d["parent"],
                 d["cand"], d["logits"], stream=stream, block_table=s.get("block_table"))
        with torch.cuda.stream(stream):
            host_res.copy_(step.results, non_blocking=True)
        join.record(copy_stream)
        stream.wait_event(join)

    # eager warm-up, then one graph per set (n_sets >= 2, so a step never
    # uploads into the set it reads)
    upload(0, stream)
    for i in range(3):
        one(i)
    stream.synchronize()
    graphs = []
    for i in range(n_sets):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            one(i)
        graphs.append(g)
    with torch.cuda.stream(stream):
        upload(0, stream)
        for i in range(n_sets):
            graphs[i].replay()
    torch.cuda.synchronize(device)
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    barrier(dist, device)
    torch.cuda.synchronize(device)
    with torch.cuda.stream(stream):
        start.record(stream)
        upload(0, stream)
        for i in range(n):
            graphs[i % n_sets].replay()
        end.record(stream)
    end.synchronize()
    if step.device_status() != 0:
        raise RuntimeError(f"device status {step.device_status()} in the end-to-end steps")
    seconds = max_over_ranks(dist, start.elapsed_time(end) / 1e3, device)
    value, ms = aggregate(seconds, n, world)
    return {"value": value, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "steps": n, "ms_per_step": ms,
            "api": "paper_2405_00263_gb300.VerifyStep.run (C ABI), one CUDA graph per input set: step i, the "
                   "upload of step i+1's inputs (one copy of one pinned buffer holding them all) on a copy stream, "
                   "the read-back of step i's results (one copy of VerifyStep.results)"}


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


class OracleSampler:
    """Times the oracle's verify step on a bounded sample of the workload and
    scales it to the whole step: the attention on a fraction f of the query
    rows, the argmax on a fraction of the logit rows (typical acceptance: the
    first fraction of the vocabulary, its cost being linear in V), the walk,
    the append and the compaction in full (they are small).  f = 1 times the
    whole oracle step (oracle.verify_step)."""

    def __init__(self, host: dict, threads: int, typical=None):
        import oracle
        self.oracle = oracle
        self.host, self.threads, self.typ = host, threads, typical
        B, T, Hq, _ = host["q"].shape
        self.n_rows = B * T * Hq
        self.n_logit_rows = B * T
        self.V = host["logits"].shape[-1]
        self.amax = oracle.argmax(host["logits"], n_threads=threads)
        self.sub_logits = {}
        # caches the sampled append and compaction write into (their contents
        # do not matter for the time; the lengths are reset every step)
        self.kc, self.vc = host["k_cache"].clone(), host["v_cache"].clone()

    def step_seconds(self, f: float) -> float:
        if f >= 1.0:
            return oracle_step_seconds(self.host, self.threads, self.typ)
        o, h, th = self.oracle, self.host, self.threads
        # at least one row a thread, so that a sample runs as parallel as the whole
        ra = min(self.n_rows, max(th, round(f * self.n_rows)))
        t0 = time.perf_counter()
        o.tree_attention(h["q"], h["k_new"], h["v_new"], h["k_cache"], h["v_cache"], h["cache_len"], h["parent"],
                         rows=list(range(ra)), n_threads=th)
        t_attn = (time.perf_counter() - t0) * self.n_rows / ra
        if self.typ is None:
            rl = min(self.n_logit_rows, max(th, round(f * self.n_logit_rows)))
            t0 = time.perf_counter()
            o.argmax(h["logits"], rows=list(range(rl)), n_threads=th)
            t_acc = (time.perf_counter() - t0) * self.n_logit_rows / rl
            t0 = time.perf_counter()
            path, alen, _ = o.accept_walk(h["parent"], h["cand"], self.amax)
            t_acc += time.perf_counter() - t0
        else:
            vs = max(1, round(f * self.V))
            if vs not in self.sub_logits:
                self.sub_logits[vs] = h["logits"][..., :vs].contiguous()
            t0 = time.perf_counter()
            r = o.accept_typical(self.sub_logits[vs], h["parent"], h["cand"], *self.typ, n_threads=th)
            t_acc = (time.perf_counter() - t0) * self.V / vs
            path, alen = r["path"], r["accept_len"]
        cl = h["cache_len"].clone().to(torch.int32)
        t0 = time.perf_counter()
        o.append_tree_kv(h["k_new"], h["v_new"], self.kc, self.vc, cl)
        o.kv_compact(self.kc, self.vc, cl, path, alen)
        return t_attn + t_acc + time.perf_counter() - t0


def sample_fraction(t_full: float, n_steps: int, budget_s: float) -> float:
    return min(1.0, budget_s / max(1e-9, n_steps * t_full))


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
    # the same oracle on one core: one step on a sample of the rows sized to
    # about a quarter of the budget (OracleSampler), scaled to the whole step
    one = OracleSampler(host, 1, typ)
    f1 = sample_fraction(per * threads, 1, budget_s / 4)
    t1 = one.step_seconds(f1)
    return {"value": 1.0 / per, "unit": UNIT, "cores": threads, "kind": "oracle",
            "sample": f"{len(times)} whole verify steps of {w.name} (fp64 oracle, OpenMP over attention rows "
                      f"and logit rows, {accept_desc(args)}), median {per * 1e3:.1f} ms per step",
            "single_core": {"value": 1.0 / t1, "unit": UNIT, "cores": 1,
                            "sample": "one verify step" + ("" if f1 >= 1.0 else
                                      f", {f1:.2e} of the attention rows and of the logit rows, scaled to the "
                                      "whole step")}}


def run_reference_arm(args, world, rank, budget_s: float = 120.0):
    """The oracle on the host cores: `--steps` timed steps after `--warmup`,
    each one a bounded sample of the workload (OracleSampler, or one row of a
    draft head step) scaled to the whole step, so that the run stays within
    about `budget_s` seconds whatever the step count."""
    from synth import workloads
    if rank != 0:
        return None
    import oracle
    oracle.build()
    threads = os.cpu_count() or 1
    if args.draft:
        return run_reference_draft(args, world, threads, budget_s)
    w = workloads.get(args.workload)
    host = workloads.make(w)
    typ = typical_params(args)
    sampler = OracleSampler(host, threads, typ)
    t_full = sampler.step_seconds(1.0)
    f = sample_fraction(t_full, args.steps + args.warmup, budget_s)
    for _ in range(args.warmup):
        sampler.step_seconds(f)
    t = [sampler.step_seconds(f) for _ in range(args.steps)]
    total = sum(t)
    value = args.steps / total
    sample = (f"{args.steps} verify steps of {w.name} (fp64 oracle, OpenMP), each timed on "
              + ("the whole step" if f >= 1.0 else f"a {f:.2e} fraction of the attention rows and of the logit "
                 "rows (vocabulary for typical acceptance), scaled to the whole step; walk, append and "
                 "compaction in full"))
    return {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f64", "data": "synthetic",
            "config": {"workload": f"{w.name}: {w.description}", "parallelism": "host cores (rank 0 only)",
                       "accept": accept_desc(args)},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "gpu_launches": 0}


class DraftOracleSampler:
    """Times the oracle's head step on a bounded sample: one row, every layer on
    a fraction f of its output features (the LM head and the top-k on that
    fraction of the vocabulary), each scaled to the whole layer, the total to
    R rows.  Each layer's input is the full one, computed once."""

    def __init__(self, inputs):
        import oracle
        self.o = oracle
        self.R, self.H, self.V, self.k, self.w_lm, self.w_v, self.w_o, self.w_1, h, toks = inputs
        bf = torch.bfloat16
        self.toks = toks[:1]
        self.e = oracle.embed_rows(self.w_lm, self.toks).to(bf)
        self.a = oracle.linear(self.e, self.w_v).to(bf)
        self.h1 = (h[:1].double() + oracle.linear(self.a, self.w_o)).to(bf)
        self.z = oracle.linear(self.h1, self.w_1, res=self.h1, act=1).to(bf)

    def seconds(self, f: float) -> float:
        o, H, V = self.o, self.H, self.V
        th = os.cpu_count() or 1
        # at least a few outputs a thread, so that a sample runs as parallel as the whole
        ns = min(H, max(4 * th, round(f * H)))
        vs = min(V, max(self.k, 4 * th, round(f * V)))
        t0 = time.perf_counter()
        o.embed_rows(self.w_lm, self.toks)
        t = time.perf_counter() - t0
        t0 = time.perf_counter()
        o.linear(self.e, self.w_v[:ns])
        o.linear(self.a, self.w_o[:ns])
        o.linear(self.h1, self.w_1[:ns], res=self.h1[:, :ns].contiguous(), act=1)
        t += (time.perf_counter() - t0) * H / ns
        t0 = time.perf_counter()
        logits = o.linear(self.z, self.w_lm[:vs])
        o.topk(logits, self.k)
        t += (time.perf_counter() - t0) * V / vs
        return t * self.R


def run_reference_draft(args, world, threads, budget_s):
    R, H, V, k = args.draft, 4096, 125696, 8
    g = torch.Generator().manual_seed(1234)
    rnd = lambda *sh, std=1.0: (torch.randn(*sh, generator=g) * std).to(torch.bfloat16)
    w_lm = rnd(V, H, std=H ** -0.5)
    w_v, w_o, w_1 = (rnd(H, H, std=H ** -0.5) for _ in range(3))
    inputs = (R, H, V, k, w_lm, w_v, w_o, w_1, rnd(R, H), torch.randint(0, V, (R,), generator=g, dtype=torch.int32))
    sampler = DraftOracleSampler(inputs)
    t_row = sampler.seconds(0.01) / R                  # one row of a whole step, estimated
    f = sample_fraction(t_row, args.steps + args.warmup, budget_s)
    for _ in range(args.warmup):
        sampler.seconds(f)
    t = [sampler.seconds(f) for _ in range(args.steps)]
    total = sum(t)
    value = args.steps / total
    sample = (f"{args.steps} head steps, each timed on 1 row with every layer (the LM head and top-k included) "
              f"on a {f:.2e} fraction of its outputs, scaled to whole layers and to {R} rows (fp64 oracle, OpenMP)")
    return {"impl": "reference", "metric": DRAFT_METRIC, "value": value, "unit": DRAFT_UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": f"Clover head step, 7B shapes: R{R} rows, H{H}, V{V}, top-{k}",
                       "parallelism": "host cores (rank 0 only)"},
            "cpu_baseline": {"value": value, "unit": DRAFT_UNIT, "cores": threads, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": DRAFT_UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "gpu_launches": 0}


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=40000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--accept", default="greedy", choices=["greedy", "typical"],
                    help="acceptance rule of the step (typical: tempered softmax with an entropy threshold)")
    ap.add_argument("--draft", type=int, default=0,
                    help="time one Clover draft head step on this many rows (7B shapes) instead of verification")
    ap.add_argument("--page-size", type=int, default=0,
                    help="run on a paged KV cache with pages of this many slots (0: dense cache)")
    ap.add_argument("--schedule", default="fused", choices=["commit", "compact", "fused"],
                    help="call schedule of the step (VerifyStep)")
    ap.add_argument("--attn-launch", default="inputs_ready", choices=["ordinary", "pdl", "cache_ready", "inputs_ready"],
                    help="attention launch: ordinary, or a programmatic dependent of the kernel before it, with the "
                         "statement that the caches (cache_ready) or all inputs (inputs_ready) are not being written "
                         "by the kernels that may still run -- true here: consecutive steps serve independent input "
                         "sets, as independent batches do")
    ap.add_argument("--workloads", default="",
                    help="comma-separated workloads: one JSON line each (stdout, and --record FILE if given)")
    ap.add_argument("--record", default="", help="file that --workloads appends its JSON lines to")
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

    if args.page_size and args.schedule == "compact":
        raise SystemExit("a paged cache takes the commit or the fused schedule")
    dist = dist_init(world, "nccl" if torch.cuda.is_available() else "gloo")
    if args.draft:
        line, inputs = run_draft_arm(args, world, rank, local, dist)
        if rank == 0:
            line["cpu_baseline"] = draft_cpu_baseline(inputs) if world == 1 and not args.no_cpu_baseline else None
            print(json.dumps(line), flush=True)
        if dist is not None:
            dist.destroy_process_group()
        return 0
    for name in (args.workloads.split(",") if args.workloads else [args.workload]):
        args.workload = name
        line, w, base = run_gpu_arm(args, world, rank, local, dist)
        if rank == 0:
            if world == 1 and not args.no_cpu_baseline:
                host = {k: (v.cpu() if isinstance(v, torch.Tensor) else v) for k, v in base.items()}
                line["cpu_baseline"] = cpu_baseline(w, host, args)
            else:
                line["cpu_baseline"] = None
            print(json.dumps(line), flush=True)
            if args.record:
                with open(args.record, "a") as f:
                    f.write(json.dumps(line) + "\n")
        del base
        torch.cuda.empty_cache()
    if dist is not None:
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
