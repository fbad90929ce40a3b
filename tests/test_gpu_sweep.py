"""A seeded sweep over the supported space: random batch sizes, tree sizes and
shapes, head counts and group sizes, head dimensions, cache lengths (ragged or
not, empty included), vocabulary sizes, dtypes, step schedules, attention
launch modes, acceptance rules and cache layouts (dense or paged).  Each case
runs one whole step through VerifyStep and compares it with the oracle:
attention within the dtype's tolerance, argmax, path, accepted length, bonus
token, source indices, new lengths and the committed cache rows bit for bit.

Typical acceptance is drawn with epsilon = 0 (threshold 0: an edge is accepted
iff its candidate has positive probability), so no decision sits near its
threshold; tests/test_gpu_typical.py covers thresholds in general."""

from __future__ import annotations

import random

import pytest
import torch

import oracle
import paper_2405_00263_gb300 as pkg
from synth import paging, workloads
from tests.gpu_util import ATOL, compare_full, to_dev

pytestmark = pytest.mark.gpu

N_CASES = 200


def draw(i: int) -> dict:
    r = random.Random(9000 + i)
    dtype = r.choice(["bf16", "bf16", "bf16", "f32"])
    Hkv = r.choice([1, 2, 4])
    G = r.choice([1, 2, 4, 8])
    T = r.choice([1, 4, 16, 33, 64, 100, 128])
    B = r.choice([1, 2, 3])
    L = r.choice([0, r.randint(1, 300), r.randint(300, 1600)])
    ragged = L > 0 and r.random() < 0.5
    schedule = r.choice(["fused", "fused", "commit", "compact"])
    paged = schedule != "compact" and r.random() < 0.35
    return dict(
        w=workloads.Workload(
            f"sweep{i}", B=B, T=T, Hq=Hkv * G, Hkv=Hkv, D=r.choice([64, 128]), L=L, V=r.choice([1000, 2049, 4099]),
            dtype=dtype, branching=(8, 4, 2, 2, 2, 1), plant_p=r.choice([0.0, 0.5, 1.0]),
            qkv_std=r.choice([1.0, 1.0 / 128 ** 0.5]), seed=500 + i, L_range=(0, L) if ragged else None,
            tree=r.choice(["topk", "random", "chain", "star"])),
        schedule=schedule,
        attn_launch=r.choice(["ordinary", "pdl", "cache_ready", "inputs_ready"]),
        accept=r.choice(["greedy", "greedy", "typical"]),
        page_size=r.choice([16, 32, 64, 128]) if paged else None,
    )


N_LONG = 40


def draw_long(i: int) -> dict:
    """Long caches (up to 8 key ranges a head) and batches up to 6, the
    oracle's work bounded to about 4e9 multiply-adds a case."""
    r = random.Random(77000 + i)
    Hkv = r.choice([1, 2, 4, 8])
    G = r.choice([1, 2, 4, 8])
    T = r.choice([4, 16, 64, 128])
    B = r.choice([1, 2, 4, 6])
    L = r.randint(1600, 9000)
    D = r.choice([64, 128])
    while B * T * Hkv * G * L * D > 4e9 and B > 1:
        B -= 1
    while B * T * Hkv * G * L * D > 4e9 and T > 4:
        T //= 2
    schedule = r.choice(["fused", "fused", "commit", "compact"])
    paged = schedule != "compact" and r.random() < 0.3
    return dict(
        w=workloads.Workload(
            f"long{i}", B=B, T=T, Hq=Hkv * G, Hkv=Hkv, D=D, L=L, V=r.choice([1000, 4099]),
            dtype=r.choice(["bf16", "bf16", "f32"]), branching=(8, 4, 2, 2, 2, 1), plant_p=r.choice([0.0, 0.5, 1.0]),
            qkv_std=r.choice([1.0, 1.0 / 128 ** 0.5]), seed=8000 + i, L_range=(0, L) if r.random() < 0.6 else None,
            tree=r.choice(["topk", "random", "chain", "star"])),
        schedule=schedule,
        attn_launch=r.choice(["ordinary", "pdl", "cache_ready", "inputs_ready"]),
        accept=r.choice(["greedy", "typical"]),
        page_size=r.choice([16, 64, 256]) if paged else None,
    )


def describe(i: int) -> str:
    c = draw(i)
    w = c["w"]
    return (f"{i}-{w.dtype}-B{w.B}-T{w.T}-{w.tree}-h{w.Hq}x{w.Hkv}-D{w.D}-L{w.L}{'r' if w.L_range else ''}-"
            f"{c['schedule']}-{c['attn_launch']}-{c['accept']}" + (f"-p{c['page_size']}" if c["page_size"] else ""))


@pytest.mark.parametrize("i", range(N_CASES), ids=[describe(i) for i in range(N_CASES)])
def test_sweep_step_matches_oracle(i, cuda):
    check_case(draw(i), cuda)


@pytest.mark.parametrize("i", range(N_LONG))
def test_sweep_long_caches_match_oracle(i, cuda):
    check_case(draw_long(i), cuda)


def check_case(c: dict, cuda):
    run, check = prepare_case(c, cuda)
    run(None)
    torch.cuda.synchronize()
    check()


def prepare_case(c: dict, cuda):
    """The case's device inputs and VerifyStep; returns run(stream), which
    issues one step, and check(), which compares the finished step with the
    oracle."""
    w = c["w"]
    host = workloads.make(w)
    B, T, Hq, D = host["q"].shape
    V = host["logits"].shape[-1]
    typical = (1.0, 0.0, 0.3) if c["accept"] == "typical" else None
    kw = dict(schedule=c["schedule"], attn_launch=c["attn_launch"], accept=c["accept"])
    if typical is not None:
        kw.update(temperature=typical[0], epsilon=typical[1], delta=typical[2])
    if c["page_size"] is None:
        t = to_dev(host, cuda)
        step = pkg.VerifyStep(B, T, Hq, w.Hkv, D, t["Lcap"], V, w.torch_dtype, device=cuda, **kw)

        def run(stream):
            step.run(t["q"], t["k_new"], t["v_new"], t["k_cache"], t["v_cache"], t["cache_len"], t["parent"],
                     t["cand"], t["logits"], stream=stream)

        return run, lambda: compare_full(host, step, t)

    # paged: the pools hold the dense cache, padded to whole pages, under a seeded table
    ps = c["page_size"]
    cap = -(-host["Lcap"] // max(256, ps)) * max(256, ps)
    pad = torch.full((B, w.Hkv, cap - host["Lcap"], D), float("nan"), dtype=host["k_cache"].dtype)
    kc = torch.cat([host["k_cache"], pad], 2)
    vc = torch.cat([host["v_cache"], pad], 2)
    table, n_pages = paging.page_table([int(L) + T for L in host["cache_len"]], ps, cap // ps, seed=w.seed)
    kp = paging.to_pages(kc, table, ps, n_pages).to(cuda)
    vp = paging.to_pages(vc, table, ps, n_pages).to(cuda)
    t = to_dev(host, cuda)
    table_dev = table.to(cuda)
    step = pkg.VerifyStep(B, T, Hq, w.Hkv, D, cap, V, w.torch_dtype, device=cuda, page_size=ps, **kw)

    def run(stream):
        step.run(t["q"], t["k_new"], t["v_new"], kp, vp, t["cache_len"], t["parent"], t["cand"], t["logits"],
                 block_table=table_dev, stream=stream)

    def check():
        ref = oracle.verify_step(host, typical=typical)
        assert step.device_status() == 0
        err = (step.out.double().cpu() - ref["out"]).abs().max().item()
        assert err <= ATOL[w.torch_dtype], err
        for name in ("argmax", "path", "accept_len", "bonus"):
            assert torch.equal(getattr(step, name).cpu(), ref[name]), name
        assert torch.equal(step.src_index.cpu(), ref["path"])
        assert torch.equal(step.new_cache_len.cpu(), ref["cache_len"])
        iview = torch.int16 if w.torch_dtype == torch.bfloat16 else torch.int32
        for pool, want in ((kp, ref["k_cache"]), (vp, ref["v_cache"])):
            view = paging.from_pages(pool.cpu(), table, ps, cap)
            for b in range(B):
                n = int(ref["cache_len"][b])
                assert torch.equal(view[b, :, :n].view(iview), want[b, :, :n].view(iview)), b

    return run, check


N_STREAMS = 6


@pytest.mark.parametrize("group", range(4))
def test_independent_steps_on_separate_streams(group, cuda):
    """Six seeded cases (dense and paged caches, every schedule, launch mode
    and acceptance rule that draw() gives), each with its own VerifyStep on its
    own stream, issued interleaved three times over without any dependency
    between the streams, so that their kernels run at the same time: every
    case still matches the oracle, so steps share no device state."""
    cases = [prepare_case(draw(3000 + N_STREAMS * group + k), cuda) for k in range(N_STREAMS)]
    streams = [torch.cuda.Stream() for _ in cases]
    torch.cuda.synchronize()
    for _ in range(3):
        for (run, _), s in zip(cases, streams):
            with torch.cuda.stream(s):
                run(s)
    torch.cuda.synchronize()
    for _, check in cases:
        check()


N_ERRORS = 40


def draw_error(i: int) -> dict:
    """A seeded small case (from draw) with one invalid input: a parent array
    that is not a topologically numbered tree, a cache length past the
    capacity, or (paged) a block-table entry outside the pool."""
    c = draw(1000 + i)
    r = random.Random(61000 + i)
    kinds = ["tree", "capacity"] + (["page"] if c["page_size"] else [])
    c["error"] = r.choice(kinds)
    c["r"] = r
    return c


@pytest.mark.parametrize("i", range(N_ERRORS))
def test_sweep_device_errors_are_reported(i, cuda):
    """The step completes, the status word carries the error's bit
    (CLOVER_ERR_BAD_TREE 4, CLOVER_ERR_CAPACITY 8, CLOVER_ERR_INVALID_ARG 1)
    and never CLOVER_ERR_TIMEOUT: every kernel turns the invalid input into a
    reported error and winds down without a wait running out."""
    c = draw_error(i)
    w, r = c["w"], c["r"]
    host = workloads.make(w)
    B, T, Hq, D = host["q"].shape
    V = host["logits"].shape[-1]
    bit = {"tree": 4, "capacity": 8, "page": 1}[c["error"]]
    b = r.randrange(B)
    if c["error"] == "tree":
        if T == 1 or r.random() < 0.3:
            host["parent"][b, 0] = r.choice([0, 5, -7])
        else:
            j = r.randrange(1, T)
            host["parent"][b, j] = r.choice([j, j + 1 if j + 1 < T else j, -3, T + 4])
    elif c["error"] == "capacity":
        host["cache_len"][b] = host["Lcap"] - T + 1 + r.randrange(40)
    kw = dict(schedule=c["schedule"], attn_launch=c["attn_launch"], accept=c["accept"])
    t = to_dev(host, cuda)
    if c["page_size"] is None:
        step = pkg.VerifyStep(B, T, Hq, w.Hkv, D, t["Lcap"], V, w.torch_dtype, device=cuda, **kw)
        step.run(t["q"], t["k_new"], t["v_new"], t["k_cache"], t["v_cache"], t["cache_len"], t["parent"],
                 t["cand"], t["logits"])
    else:
        ps = c["page_size"]
        cap = -(-host["Lcap"] // max(256, ps)) * max(256, ps)
        lens = [min(int(L), host["Lcap"] - T) for L in host["cache_len"]]
        table, n_pages = paging.page_table([L + T for L in lens], ps, cap // ps, seed=w.seed)
        if c["error"] == "capacity":
            t["cache_len"][b] = cap - T + 1           # past the paged capacity
        if c["error"] == "page":
            # an entry the step always uses: the page of slot 0 (read when L > 0) or of slot L (the commit
            # writes the accepted root there)
            k = 0 if lens[b] > 0 and r.random() < 0.5 else lens[b] // ps
            table[b, k] = r.choice([-2, n_pages, n_pages + 9])
        pool = torch.zeros((n_pages, w.Hkv, ps, D), dtype=w.torch_dtype, device=cuda)
        step = pkg.VerifyStep(B, T, Hq, w.Hkv, D, cap, V, w.torch_dtype, device=cuda, page_size=ps, **kw)
        step.run(t["q"], t["k_new"], t["v_new"], pool, pool.clone(), t["cache_len"], t["parent"], t["cand"],
                 t["logits"], block_table=table.to(cuda))
    torch.cuda.synchronize()
    status = step.device_status()
    assert status & bit, (c["error"], status)
    assert not status & 32, status
