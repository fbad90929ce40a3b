"""The roofline arithmetic of bench.py: algorithmic bytes and flops per
launch, pinned to closed forms worked out by hand for the benchmark
workloads (KV rows of every committed and tree key read once, q read once,
out written once; 4 flops per (query row, key, dim) for QK^T and PV)."""

from __future__ import annotations

import bench
from synth import workloads


def test_attention_bytes_7b_l4096():
    w = workloads.get("7b_l4096")
    lengths = workloads.cache_lengths(w)
    # K and V: 2 x 32 heads x 128 dims x 2 bytes per key, 4096 + 64 keys;
    # q and out: 64 x 32 x 128 x 2 bytes each
    kv = 2 * 32 * 128 * 2 * (4096 + 64)
    qo = 2 * 64 * 32 * 128 * 2
    assert bench.attn_bytes_per_launch(w, lengths) == kv + qo == 69_206_016
    assert bench.attn_flops_per_launch(w, lengths) == 4 * 32 * 64 * 128 * (4096 + 64) == 4_362_076_160


def test_attention_bytes_7b_l16384_and_100b_gqa():
    w = workloads.get("7b_l16384")
    assert bench.attn_bytes_per_launch(w, workloads.cache_lengths(w)) == 16384 * 16448 + 1_048_576 == 270_532_608
    w = workloads.get("100b_gqa")
    lengths = workloads.cache_lengths(w)
    # four sequences of 8192 + 64 keys, 8 KV heads; q/out over 64 query heads
    kv = 2 * 8 * 128 * 2 * 4 * (8192 + 64)
    qo = 2 * 4 * 64 * 64 * 128 * 2
    assert bench.attn_bytes_per_launch(w, lengths) == kv + qo == 143_654_912
    assert bench.attn_flops_per_launch(w, lengths) == 4 * 64 * 64 * 128 * 4 * (8192 + 64)


def test_argmax_bytes():
    w = workloads.get("7b_l4096")
    assert bench.argmax_bytes_per_launch(w) == 64 * 125_696 * 2 == 16_089_088


def test_batched_bytes_follow_the_lengths():
    w = workloads.get("7b_batched")
    lengths = workloads.cache_lengths(w)
    assert len(lengths) == w.B == 16
    per_key = 2 * w.Hkv * w.D * 2
    assert bench.attn_bytes_per_launch(w, lengths) == \
        per_key * sum(L + w.T for L in lengths) + 2 * w.B * w.T * w.Hq * w.D * 2


def test_cpu_baseline_reports_all_cores_and_one():
    from types import SimpleNamespace
    w = workloads.get("tiny_f32")
    host = workloads.make(w)
    args = SimpleNamespace(accept="greedy", temperature=1.0, epsilon=0.09, delta=0.3)
    rec = bench.cpu_baseline(w, host, args, budget_s=0.5)
    assert rec["kind"] == "oracle" and rec["value"] > 0 and rec["cores"] >= 1
    assert rec["single_core"]["cores"] == 1 and rec["single_core"]["value"] > 0
