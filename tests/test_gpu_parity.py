"""GPU parity: the CUDA path through the C ABI against the oracle on the same
seeded inputs.  Attention within max-abs 1e-4 (fp32) / 2e-2 (bf16) of the fp64
oracle; argmax, path, accepted length, bonus token, source indices, new cache
lengths and committed cache bytes bit-exact."""

import pytest
import torch

import oracle
import paper_2405_00263_gb300 as pkg
from synth import workloads
from tests.gpu_util import ATOL, compare_full, run_gpu, to_dev

pytestmark = pytest.mark.gpu

SMALL = {
    "tiny": ("tiny_f32", {}),
    "f32_d128_splits_raggedV": ("tiny_f32", dict(D=128, L=1000, Hq=4, Hkv=4, V=5003)),
    "f32_gqa_T64": ("tiny_f32", dict(T=64, Hq=16, Hkv=2, branching=(8, 4, 2, 2, 1), L=200)),
    "bf16_d64_gqa_raggedV": ("7b_l2048", dict(B=2, T=16, Hq=8, Hkv=2, D=64, L=777, V=4099,
                                               branching=(4, 2, 1, 1))),
    "bf16_chain": ("7b_l2048", dict(T=64, Hq=4, Hkv=4, L=300, V=2048, tree="chain")),
    "bf16_star": ("7b_l2048", dict(T=40, Hq=4, Hkv=4, L=129, V=2048, tree="star")),
    "bf16_random_trees": ("7b_l2048", dict(B=3, T=37, Hq=4, Hkv=4, L=513, V=2048, tree="random")),
    "bf16_single_node": ("7b_l2048", dict(B=2, T=1, Hq=4, Hkv=4, L=1500, V=3000, branching=())),
    "bf16_empty_cache": ("7b_l2048", dict(T=16, Hq=4, Hkv=4, L=0, V=2048, branching=(4, 2, 1, 1))),
    "bf16_ragged_batch": ("7b_batched", dict(B=5, Hq=8, Hkv=8, L_range=(0, 700), V=3001)),
    "bf16_sharp_scores": ("7b_l2048", dict(T=64, Hq=4, Hkv=2, L=900, V=2048, qkv_std=1.5)),
    "bf16_gqa8_T64": ("100b_gqa", dict(B=1, Hq=16, Hkv=2, L=640, V=2048)),
    # two 128-row tiles per key range: a cluster of two sharing K/V tiles by multicast, with split merges
    "bf16_gqa4_T64_pairs": ("100b_gqa", dict(B=2, Hq=16, Hkv=4, L=900, V=2048)),
    # trees past 64 nodes: two mask words, two FMA tree tiles, four nodes per lane in the walk
    "bf16_T128_topk": ("7b_l2048", dict(T=128, Hq=4, Hkv=4, L=700, V=3000, branching=(8, 4, 2, 2, 2, 1))),
    "bf16_T128_chain": ("7b_l2048", dict(T=128, Hq=2, Hkv=2, L=300, V=2048, tree="chain", plant_p=1.0)),
    "bf16_T100_random_gqa": ("100b_gqa", dict(B=2, T=100, Hq=16, Hkv=2, L=450, V=4099, tree="random")),
    "bf16_T65_d64": ("7b_l2048", dict(B=2, T=65, Hq=8, Hkv=8, D=64, L=333, V=2048, tree="random")),
    "f32_T100_random": ("tiny_f32", dict(B=2, T=100, Hq=4, Hkv=2, L=260, V=5003, tree="random")),
    "f32_T128_d128": ("tiny_f32", dict(T=128, D=128, Hq=2, Hkv=2, L=500, V=1024, branching=(8, 4, 2, 2, 2, 1))),
}


@pytest.mark.parametrize("case", sorted(SMALL))
def test_small_step_matches_oracle(case, cuda):
    name, over = SMALL[case]
    w = workloads.get(name, **over)
    host = workloads.make(w)
    t = to_dev(host, cuda)
    step = run_gpu(t)
    compare_full(host, step, t)


@pytest.mark.parametrize("case", sorted(c for c in SMALL if not c.startswith("f32")))
def test_small_step_inputs_ready_plan(case, cuda):
    """The inputs-ready launch plan (one CTA takes every key of a head tile, no
    split) on every bf16 shape, in the bench's fused schedule: the whole step
    against the oracle."""
    name, over = SMALL[case]
    host = workloads.make(workloads.get(name, **over))
    t = to_dev(host, cuda)
    step = run_gpu(t, schedule="fused", attn_launch="inputs_ready")
    compare_full(host, step, t)


# Grouped-query shapes whose inputs-ready launch takes one CTA per (sequence,
# KV head, row tile) -- at least 30 row tiles -- with two or more row tiles a
# head: that launch runs two row tiles per CTA (tree_attn_tc_pair.cu).
PAIR = {
    "pair_gqa8_T64": ("100b_gqa", dict(B=2, Hq=32, Hkv=4, L=900, V=2048)),
    # three row tiles a head: the second CTA has one (64 rows) and no second tile
    "pair_odd_tiles_T40": ("100b_gqa", dict(B=2, T=40, Hq=40, Hkv=5, L=700, V=2048, tree="random")),
    # four row tiles a head, the last of 16 rows
    "pair_partial_T100_G4": ("7b_l2048", dict(B=1, T=100, Hq=32, Hkv=8, L=1000, V=2048, tree="random")),
    "pair_empty_cache": ("100b_gqa", dict(B=2, Hq=32, Hkv=4, L=0, V=2048)),
    "pair_whole_tiles_L1024": ("100b_gqa", dict(B=2, Hq=32, Hkv=4, L=1024, V=2048)),
    "pair_ragged_lengths": ("100b_gqa", dict(B=3, Hq=24, Hkv=3, L=1500, L_range=(0, 1500), V=2048)),
    "pair_sharp_scores": ("100b_gqa", dict(B=2, Hq=32, Hkv=4, L=800, V=2048, qkv_std=1.5)),
}


@pytest.mark.parametrize("case", sorted(PAIR))
def test_pair_kernel_step_matches_oracle(case, cuda):
    """The bench's step (fused schedule, inputs-ready attention) on
    grouped-query shapes that take the two-row-tile kernel: every output
    against the oracle."""
    name, over = PAIR[case]
    host = workloads.make(workloads.get(name, **over))
    t = to_dev(host, cuda)
    step = run_gpu(t, schedule="fused", attn_launch="inputs_ready")
    compare_full(host, step, t)


def test_pair_kernel_equals_single_tile_kernel(cuda):
    """100b_gqa at full size: an ordinary launch (one row tile a CTA; its 128
    CTAs fill the GPU, so one key range each) and an inputs-ready launch (two
    row tiles a CTA) compute every row the same way: equal bytes."""
    w = workloads.get("100b_gqa")
    t = workloads.make(w, device=cuda, logits=False)
    ws_n = pkg.clover_verify_attn_workspace_size(w.B, w.T, w.Hq, w.Hkv, w.D, t["Lcap"], torch.bfloat16)
    ws = torch.zeros(max(16, ws_n), dtype=torch.uint8, device=cuda)
    st = torch.zeros(1, dtype=torch.int32, device=cuda)
    outs = []
    for kw in (dict(), dict(pdl=True, inputs_ready=True)):
        out = torch.full_like(t["q"], float("nan"))
        pkg.clover_verify_attn(t["q"], t["k_new"], t["v_new"], t["k_cache"], t["v_cache"], t["cache_len"],
                               t["parent"], out, workspace=ws, status=st, append=False, **kw)
        torch.cuda.synchronize()
        outs.append(out)
    assert int(st.item()) == 0
    assert torch.equal(outs[0].view(torch.int16), outs[1].view(torch.int16))


@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("T,Hq,Hkv,lengths", [(33, 8, 4, [651, 1219]), (33, 8, 4, [0, 1219]),
                                               (64, 8, 4, [512, 1219]), (33, 16, 4, [700, 1219, 40])],
                         ids=["T33_G2_651", "T33_G2_empty", "T64_G2_512", "T33_G4_three"])
def test_full_row_tiles_with_empty_splits(T, Hq, Hkv, lengths, D, cuda):
    """More than 64 query rows a head (full 128-row tiles: two softmax warps
    a lane quadrant) with ragged lengths, so that a short sequence leaves some
    of its non-tree key ranges empty: such a range has no O and reports no
    error, and the whole step matches the oracle.  (A range with no keys once
    raised CLOVER_ERR_TIMEOUT in this layout.)"""
    w = workloads.get("7b_l2048", B=len(lengths), T=T, Hq=Hq, Hkv=Hkv, D=D, L=max(lengths), V=2048,
                      tree="random", seed=620)
    host = workloads.make(w)
    host["cache_len"] = torch.tensor(lengths, dtype=torch.int32)
    t = to_dev(host, cuda)
    for schedule in ("commit", "fused"):
        t = to_dev(host, cuda)
        step = run_gpu(t, schedule=schedule)
        compare_full(host, step, t)


def test_scale_argument(cuda):
    w = workloads.get("tiny_f32", L=300)
    host = workloads.make(w)
    t = to_dev(host, cuda)
    step = run_gpu(t, scale=0.37)
    compare_full(host, step, t, scale=0.37)


def test_repeated_calls_reuse_workspace(cuda):
    """Counters in the workspaces are reset by every call: a second step on
    fresh copies of the inputs gives the same bytes."""
    w = workloads.get("7b_l2048", T=64, Hq=8, Hkv=8, L=1800, V=5000)
    host = workloads.make(w)
    t1 = to_dev(host, cuda)
    step = run_gpu(t1)
    first = [x.clone() for x in (step.out, step.argmax, step.path, step.accept_len, step.bonus)]
    for _ in range(3):
        t2 = to_dev(host, cuda)
        run_gpu(t2, step=step)
        again = (step.out, step.argmax, step.path, step.accept_len, step.bonus)
        for a, b in zip(first, again):
            assert torch.equal(a, b)
    compare_full(host, step, t2)


FULL = ["7b_l2048", "7b_l4096", "7b_l16384", "7b_batched", "100b_gqa", "paper_t4_b4", "paper_t4_b16", "paper_t4_b48",
        "7b_t128"]


@pytest.mark.parametrize("schedule", ["commit", "fused", "fused_inputs_ready"])
@pytest.mark.parametrize("name", FULL)
def test_full_size_workloads(name, schedule, cuda):
    """The workloads at their full sizes: attention on sampled rows (the
    oracle computes them one by one), argmax / walk / indices everywhere, the
    tree slots of the cache everywhere, and the committed prefix untouched.
    "fused_inputs_ready" is the bench's step: the fused schedule with the
    attention launched inputs-ready (one CTA per head tile)."""
    w = workloads.get(name)
    t = workloads.make(w, device=cuda)
    host = {k: (v.cpu() if isinstance(v, torch.Tensor) else v) for k, v in t.items()}
    kc0, vc0 = t["k_cache"].clone(), t["v_cache"].clone()
    if schedule == "fused_inputs_ready":
        step = run_gpu(t, schedule="fused", attn_launch="inputs_ready")
    else:
        step = run_gpu(t, schedule=schedule)
    assert step.device_status() == 0

    B, T, Hq, D = w.B, w.T, w.Hq, w.D
    n_rows = B * T * Hq
    g = torch.Generator().manual_seed(0)
    rows = sorted(set([0, n_rows - 1] + torch.randint(0, n_rows, (46,), generator=g).tolist()))
    ref = oracle.tree_attention(host["q"], host["k_new"], host["v_new"], host["k_cache"], host["v_cache"],
                                host["cache_len"], host["parent"], rows=rows)
    got = step.out.view(-1, D)[rows].double().cpu()
    err = (got - ref).abs().max().item()
    assert err <= ATOL[torch.bfloat16], err

    amax = oracle.argmax(host["logits"])
    assert torch.equal(step.argmax.cpu(), amax)
    path, alen, bonus = oracle.accept_walk(host["parent"], host["cand"], amax)
    assert torch.equal(step.path.cpu(), path)
    assert torch.equal(step.accept_len.cpu(), alen)
    assert torch.equal(step.bonus.cpu(), bonus)
    L = host["cache_len"]
    assert torch.equal(step.new_cache_len.cpu(), L + alen)

    # expected tree slots: the oracle's append + compaction on an empty cache of T slots
    zk = torch.zeros((B, w.Hkv, T, D), dtype=host["k_new"].dtype)
    zv = torch.zeros_like(zk)
    zl = torch.zeros(B, dtype=torch.int32)
    oracle.append_tree_kv(host["k_new"], host["v_new"], zk, zv, zl)
    src = oracle.kv_compact(zk, zv, zl, path, alen)
    exp_src = path if step.schedule in ("commit", "fused") else torch.where(src >= 0, src + L.unsqueeze(1), src)
    assert torch.equal(step.src_index.cpu(), exp_src)
    for b in range(B):
        l0, a = int(L[b]), int(alen[b])
        assert torch.equal(t["k_cache"][b, :, l0:l0 + a].cpu().view(torch.int16), zk[b, :, :a].view(torch.int16))
        assert torch.equal(t["v_cache"][b, :, l0:l0 + a].cpu().view(torch.int16), zv[b, :, :a].view(torch.int16))
        assert torch.equal(t["k_cache"][b, :, :l0].view(torch.int16), kc0[b, :, :l0].view(torch.int16))
        assert torch.equal(t["v_cache"][b, :, :l0].view(torch.int16), vc0[b, :, :l0].view(torch.int16))


# ---------------------------------------------------------------------------
# every split count of the tensor-core path's split merge
# ---------------------------------------------------------------------------

# One KV head, so the launcher's split count is min(8, Lcap / 256 rounded up):
# these cache lengths give 2, 3, 4, 5, 6, 7 and 8 splits.
SPLIT_LENGTHS = [300, 700, 1000, 1200, 1500, 1700, 3000]


@pytest.mark.parametrize("L", SPLIT_LENGTHS)
@pytest.mark.parametrize("Hq,D", [(4, 128), (8, 128), (8, 64)])
def test_split_counts_and_row_groups(L, Hq, D, cuda):
    """T=16 with 4 query heads per KV head is a 64-row tile (two key groups per
    row); 8 heads make a 128-row tile (one key group); D=64 takes the smaller
    shared-memory plan."""
    w = workloads.get("7b_l2048", B=1, T=16, Hq=Hq, Hkv=1, D=D, L=L, V=1000, branching=(4, 2, 1, 1))
    host = workloads.make(w)
    t = to_dev(host, cuda)
    step = run_gpu(t)
    compare_full(host, step, t)


@pytest.mark.parametrize("dtype_name", ["tiny_f32", "7b_l2048"])
def test_one_workspace_serves_smaller_capacities(dtype_name, cuda):
    """A workspace sized for the largest capacity serves calls with smaller
    ones (fewer splits, a smaller partial area): the arrival counters sit at
    the start, where every split count finds them.  Calls alternate between
    capacities; every output equals a call with its own fresh workspace."""
    over = dict(T=16, Hq=4, Hkv=4, D=128, V=1000, branching=(4, 2, 1, 1))
    lens = [2900, 700, 1300, 2900, 300, 1700]
    sets = [to_dev(workloads.make(workloads.get(dtype_name, L=L, seed=90 + i, **over), logits=False), cuda)
            for i, L in enumerate(lens)]
    dt = sets[0]["q"].dtype
    size = lambda s: pkg.clover_verify_attn_workspace_size(1, 16, 4, 4, 128, s["Lcap"], dt)
    sizes = [size(s) for s in sets]
    assert len(set(sizes)) > 2                            # several split counts
    ws = torch.zeros(max(sizes), dtype=torch.uint8, device=cuda)
    st = torch.zeros(1, dtype=torch.int32, device=cuda)
    for rep in range(2):
        for i, s in enumerate(sets):
            out = torch.empty_like(s["q"])
            pkg.clover_verify_attn(s["q"], s["k_new"], s["v_new"], s["k_cache"], s["v_cache"], s["cache_len"],
                                   s["parent"], out, workspace=ws, status=st, append=False)
            own = torch.zeros(max(sizes[i], 16), dtype=torch.uint8, device=cuda)
            ref = torch.empty_like(s["q"])
            pkg.clover_verify_attn(s["q"], s["k_new"], s["v_new"], s["k_cache"], s["v_cache"], s["cache_len"],
                                   s["parent"], ref, workspace=own if sizes[i] else None, status=st, append=False)
            torch.cuda.synchronize()
            assert int(st.item()) == 0
            bits = torch.int16 if dt == torch.bfloat16 else torch.int32
            assert torch.equal(out.view(bits), ref.view(bits)), (rep, i)


# ---------------------------------------------------------------------------
# programmatic dependent launch of the tensor-core attention
# ---------------------------------------------------------------------------

def _attn_chain(sets, ws, st, pdl, cache_ready, graph=False):
    """Attention calls back to back on one stream, call i+1 taking call i's
    output as its q, k_new and v_new (MHA: out has their shape) and its own
    cache; returns the outputs (optionally captured and replayed as one CUDA
    graph)."""
    outs = [torch.full_like(s["q"], float("nan")) for s in sets]

    def run():
        q = kn = vn = None
        for i, s in enumerate(sets):
            q, kn, vn = (s["q"], s["k_new"], s["v_new"]) if i == 0 else (outs[i - 1],) * 3
            pkg.clover_verify_attn(q, kn, vn, s["k_cache"], s["v_cache"], s["cache_len"], s["parent"], outs[i],
                                   workspace=ws, status=st, append=False, pdl=pdl, cache_ready=cache_ready)

    if graph:
        stream = torch.cuda.Stream()
        with torch.cuda.stream(stream):
            run()                       # eager first: per-kernel attributes are set outside the capture
        torch.cuda.synchronize()
        for o in outs:
            o.fill_(float("nan"))
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            run()
        g.replay()
    else:
        run()
    torch.cuda.synchronize()
    return outs


@pytest.mark.parametrize("graph", [False, True])
@pytest.mark.parametrize("cache_ready", [False, True])
def test_pdl_chain_reads_inputs_after_the_previous_kernel(cache_ready, graph, cuda):
    """CLOVER_ATTN_PDL (and CLOVER_ATTN_CACHE_READY, true here: every call has
    its own cache): a call may start while the previous one runs, but its q,
    k_new and v_new are that call's output, so it must read them only after it
    completes.  The outputs equal ordinary launches' bit for bit (same split
    plan, shared workspace), and the first matches the oracle."""
    n = 4
    ws_ = [workloads.get("7b_l2048", T=64, Hq=8, Hkv=8, L=1900 + 97 * i, V=1000, seed=50 + i) for i in range(n)]
    hosts = [workloads.make(w, logits=False) for w in ws_]
    sets = [to_dev(h, cuda) for h in hosts]
    need = max(pkg.clover_verify_attn_workspace_size(1, 64, 8, 8, 128, s["Lcap"], torch.bfloat16) for s in sets)
    assert need > 0                                       # several splits per head: the L2 merge runs
    ws = torch.zeros(need, dtype=torch.uint8, device=cuda)
    st = torch.zeros(1, dtype=torch.int32, device=cuda)
    ref = _attn_chain(sets, ws, st, pdl=False, cache_ready=False)
    got = _attn_chain(sets, ws, st, pdl=True, cache_ready=cache_ready, graph=graph)
    assert int(st.item()) == 0
    for i in range(n):
        assert torch.equal(got[i].view(torch.int16), ref[i].view(torch.int16)), f"call {i}"
    h = hosts[0]
    want = oracle.tree_attention(h["q"], h["k_new"], h["v_new"], h["k_cache"], h["v_cache"], h["cache_len"],
                                 h["parent"])
    assert (ref[0].double().cpu() - want).abs().max().item() <= ATOL[torch.bfloat16]


@pytest.mark.parametrize("graph", [False, True])
def test_pdl_inputs_ready_independent_calls(graph, cuda):
    """CLOVER_ATTN_INPUTS_READY: calls on independent inputs (the statement
    holds) run their key loops while the previous calls finish; their writes
    (the output) still wait for them.  Such calls take every key of a head in
    one CTA, so they are compared with the same calls made one at a time
    (synchronised): six calls, three of them into one output buffer, every
    output equal bit for bit, the shared buffer holding the last call's; and
    every output within the tolerance of the oracle."""
    n = 6
    ws_ = [workloads.get("7b_l2048", T=64, Hq=8, Hkv=8, L=1500 + 211 * i, V=1000, seed=70 + i) for i in range(n)]
    hosts = [workloads.make(w, logits=False) for w in ws_]
    sets = [to_dev(h, cuda) for h in hosts]
    need = max(pkg.clover_verify_attn_workspace_size(1, 64, 8, 8, 128, s["Lcap"], torch.bfloat16) for s in sets)
    assert need > 0
    ws = torch.zeros(need, dtype=torch.uint8, device=cuda)
    st = torch.zeros(1, dtype=torch.int32, device=cuda)

    def run(outs, sync):
        for i, s in enumerate(sets):
            pkg.clover_verify_attn(s["q"], s["k_new"], s["v_new"], s["k_cache"], s["v_cache"], s["cache_len"],
                                   s["parent"], outs[i], workspace=ws, status=st, append=False, pdl=True,
                                   inputs_ready=True)
            if sync:
                torch.cuda.synchronize()

    ref = [torch.empty_like(s["q"]) for s in sets]
    run(ref, True)
    shared = torch.full_like(sets[0]["q"], float("nan"))
    outs = [torch.full_like(s["q"], float("nan")) for s in sets]
    outs[1] = outs[3] = outs[5] = shared
    if graph:
        stream = torch.cuda.Stream()
        with torch.cuda.stream(stream):
            run(outs, False)
        torch.cuda.synchronize()
        for o in outs:
            o.fill_(float("nan"))
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            run(outs, False)
        g.replay()
    else:
        run(outs, False)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    for i in (0, 2, 4):
        assert torch.equal(outs[i].view(torch.int16), ref[i].view(torch.int16)), f"call {i}"
    assert torch.equal(shared.view(torch.int16), ref[5].view(torch.int16))
    for i, h in enumerate(hosts):
        want = oracle.tree_attention(h["q"], h["k_new"], h["v_new"], h["k_cache"], h["v_cache"], h["cache_len"],
                                     h["parent"])
        assert (ref[i].double().cpu() - want).abs().max().item() <= ATOL[torch.bfloat16], i


@pytest.mark.parametrize("mode", ["pdl", "cache_ready", "inputs_ready"])
@pytest.mark.parametrize("schedule", ["commit", "fused"])
def test_step_attention_launch_modes(mode, schedule, cuda):
    """VerifyStep with the attention launched as a programmatic dependent, on
    three independent input sets (the statement holds): steps made one at a
    time match the oracle and, with pdl and cache_ready (the same split plan),
    an ordinary step's outputs bit for bit; three steps queued back to back
    (each its own VerifyStep, so that each keeps its outputs) give the same
    outputs as the steps made one at a time."""
    hosts = [workloads.make(workloads.get("7b_l2048", T=64, Hq=8, Hkv=8, L=1100 + 300 * i, V=3000, seed=40 + i))
             for i in range(3)]
    ref = [run_gpu(to_dev(h, cuda), schedule=schedule) for h in hosts]
    ref_out = [r.out.clone() for r in ref]
    B, T, Hq, D = ref_out[0].shape
    Lcap = max(h["Lcap"] for h in hosts)

    def new_step():
        return pkg.VerifyStep(B, T, Hq, 8, D, Lcap, 3000, torch.bfloat16, device=cuda, schedule=schedule,
                              attn_launch=mode)

    def run(step, t):
        step.run(t["q"], t["k_new"], t["v_new"], t["k_cache"], t["v_cache"], t["cache_len"], t["parent"],
                 t["cand"], t["logits"])

    alone = []
    for i, h in enumerate(hosts):
        t = to_dev(h, cuda)
        step = new_step()
        run(step, t)
        torch.cuda.synchronize()
        if mode != "inputs_ready":
            assert torch.equal(step.out.view(torch.int16), ref_out[i].view(torch.int16)), i
        compare_full(h, step, t)
        alone.append(step.out.clone())
    sets = [to_dev(h, cuda) for h in hosts]
    steps = [new_step() for _ in hosts]
    for step, t in zip(steps, sets):
        run(step, t)
    torch.cuda.synchronize()
    for i, (h, step, t) in enumerate(zip(hosts, steps, sets)):
        assert torch.equal(step.out.view(torch.int16), alone[i].view(torch.int16)), i
        compare_full(h, step, t)


# ---------------------------------------------------------------------------
# the two schedules of a step
# ---------------------------------------------------------------------------

SCHEDULE_CASES = {
    "f32_splits": ("tiny_f32", dict(D=128, L=1000, Hq=4, Hkv=4, V=5003)),
    "bf16_ragged_batch": ("7b_batched", dict(B=5, Hq=8, Hkv=8, L_range=(0, 700), V=3001)),
    "bf16_gqa8": ("100b_gqa", dict(B=2, Hq=16, Hkv=2, L=900, V=2048)),
}


@pytest.mark.parametrize("concurrent", [True, False])
@pytest.mark.parametrize("case", sorted(SCHEDULE_CASES))
def test_commit_and_compact_schedules_agree(case, concurrent, cuda):
    """Attention without the append plus clover_kv_commit, and attention with the
    append plus clover_kv_compact, leave the same bytes in slots [0, L + a)
    and give the same outputs; both match the oracle."""
    name, over = SCHEDULE_CASES[case]
    host = workloads.make(workloads.get(name, **over))
    t1, t2, t3 = to_dev(host, cuda), to_dev(host, cuda), to_dev(host, cuda)
    s1 = run_gpu(t1, schedule="commit", concurrent=concurrent)
    s2 = run_gpu(t2, schedule="compact", concurrent=concurrent)
    s3 = run_gpu(t3, schedule="fused", concurrent=concurrent)
    compare_full(host, s1, t1)
    compare_full(host, s2, t2)
    compare_full(host, s3, t3)
    assert torch.equal(s1.out, s2.out) and torch.equal(s1.out, s3.out)
    assert torch.equal(s1.src_index, s3.src_index) and torch.equal(s1.new_cache_len, s3.new_cache_len)
    L = host["cache_len"].to(cuda)
    assert torch.equal(torch.where(s1.src_index >= 0, s1.src_index + L.unsqueeze(1), s1.src_index), s2.src_index)
    bits = torch.int16 if host["q"].dtype == torch.bfloat16 else torch.int32
    for b in range(host["q"].shape[0]):
        n = int(s1.new_cache_len[b])
        for t in (t2, t3):
            assert torch.equal(t1["k_cache"][b, :, :n].view(bits), t["k_cache"][b, :, :n].view(bits))
            assert torch.equal(t1["v_cache"][b, :, :n].view(bits), t["v_cache"][b, :, :n].view(bits))


@pytest.mark.parametrize("name", ["tiny_f32", "7b_l2048"])
def test_attention_without_append_only_reads_the_cache(name, cuda):
    """CLOVER_ATTN_NO_APPEND: every byte of both caches (the NaN tail included)
    is unchanged, and the output is the appending call's, bit for bit."""
    w = workloads.get(name, **({} if name == "tiny_f32" else dict(T=64, Hq=8, Hkv=8, L=1500, V=1000)))
    host = workloads.make(w, logits=False)
    t = to_dev(host, cuda)
    bits = torch.int16 if host["q"].dtype == torch.bfloat16 else torch.int32
    kc0, vc0 = t["k_cache"].clone(), t["v_cache"].clone()
    B, T, Hq, D = t["q"].shape
    Hkv = t["k_new"].shape[2]
    nbytes = pkg.clover_verify_attn_workspace_size(B, T, Hq, Hkv, D, t["Lcap"], t["q"].dtype)
    ws = torch.zeros(max(nbytes, 16), dtype=torch.uint8, device=cuda) if nbytes else None
    st = torch.zeros(1, dtype=torch.int32, device=cuda)
    out_ro, out_ap = torch.empty_like(t["q"]), torch.empty_like(t["q"])
    pkg.clover_verify_attn(t["q"], t["k_new"], t["v_new"], t["k_cache"], t["v_cache"], t["cache_len"], t["parent"],
                           out_ro, workspace=ws, status=st, append=False)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert torch.equal(t["k_cache"].view(bits), kc0.view(bits)) and torch.equal(t["v_cache"].view(bits), vc0.view(bits))
    pkg.clover_verify_attn(t["q"], t["k_new"], t["v_new"], t["k_cache"], t["v_cache"], t["cache_len"], t["parent"],
                           out_ap, workspace=ws, status=st)
    torch.cuda.synchronize()
    assert torch.equal(out_ro.view(bits), out_ap.view(bits))


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_kv_commit_matches_oracle(dtype, cuda):
    """clover_kv_commit on chosen paths (root only, a chain through every node,
    branches) against the oracle's commit: cache bytes, source nodes, lengths."""
    B, T, Hkv, D = 4, 16, 3, 128
    g = torch.Generator().manual_seed(5)
    Lcap = 320
    kc = torch.randn(B, Hkv, Lcap, D, generator=g).to(dtype)
    vc = torch.randn(B, Hkv, Lcap, D, generator=g).to(dtype)
    kn = torch.randn(B, T, Hkv, D, generator=g).to(dtype)
    vn = torch.randn(B, T, Hkv, D, generator=g).to(dtype)
    L = torch.tensor([0, 17, 150, Lcap - T], dtype=torch.int32)
    paths = [[0], list(range(T)), [0, 2, 9, 15], [0, 1, 5]]
    path = torch.full((B, T), -1, dtype=torch.int32)
    for b, p in enumerate(paths):
        path[b, :len(p)] = torch.tensor(p)
    alen = torch.tensor([len(p) for p in paths], dtype=torch.int32)
    ko, vo, lo = kc.clone(), vc.clone(), L.clone()
    src_ref = oracle.kv_commit(ko, vo, kn, vn, lo, path, alen)
    d = lambda x: x.to(cuda)
    kd, vd = d(kc), d(vc)
    i32 = dict(dtype=torch.int32, device=cuda)
    new_len, src, st = torch.empty(B, **i32), torch.empty((B, T), **i32), torch.zeros(1, **i32)
    pkg.clover_kv_commit(kd, vd, d(kn), d(vn), d(L), d(path), d(alen), new_len, src, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert torch.equal(new_len.cpu(), lo) and torch.equal(src.cpu(), src_ref)
    bits = torch.int16 if dtype == torch.bfloat16 else torch.int32
    assert torch.equal(kd.cpu().view(bits), ko.view(bits)) and torch.equal(vd.cpu().view(bits), vo.view(bits))


# ---------------------------------------------------------------------------
# edge cases
# ---------------------------------------------------------------------------

def _accept_only(logits, cand, parent, cuda):
    B, T, V = logits.shape
    ws = torch.zeros(pkg.clover_verify_accept_workspace_size(B, T, V, logits.dtype), dtype=torch.uint8, device=cuda)
    i32 = dict(dtype=torch.int32, device=cuda)
    out = dict(argmax=torch.empty((B, T), **i32), path=torch.empty((B, T), **i32),
               alen=torch.empty(B, **i32), bonus=torch.empty(B, **i32), status=torch.zeros(1, **i32))
    pkg.clover_verify_accept(logits.to(cuda), cand.to(cuda), parent.to(cuda), out["argmax"], out["path"],
                             out["alen"], out["bonus"], ws, status=out["status"])
    torch.cuda.synchronize()
    return {k: v.cpu() for k, v in out.items()}


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_argmax_ties_signed_zero_infinities(dtype, cuda):
    B, T, V = 2, 8, 125696
    g = torch.Generator().manual_seed(5)
    x = (torch.randn(B, T, V, generator=g) * 4).to(dtype)
    x[0, 0, [70000, 3, 125695]] = 40.0                   # three-way tie
    x[0, 1] = -1.0
    x[0, 1, 9000] = -0.0
    x[0, 1, 8999] = 0.0                                  # -0 == +0
    x[0, 2] = float("-inf")                              # all -inf -> 0
    x[0, 3, V - 1] = 100.0                               # last index
    x[0, 4, 0] = 100.0                                   # first index
    x[0, 5, 77] = float("inf")
    x[0, 6] = 0.0                                        # all equal -> 0
    x[1, :, 1000:2000] = 50.0                            # long runs of ties in every row
    parent = torch.tensor([[-1, 0, 1, 2, 3, 4, 5, 6]] * B, dtype=torch.int32)
    cand = torch.zeros((B, T), dtype=torch.int32)
    r = _accept_only(x, cand, parent, cuda)
    amax = oracle.argmax(x)
    assert torch.equal(r["argmax"], amax)
    assert amax[0, :7].tolist() == [3, 8999, 0, V - 1, 0, 77, 0] and amax[1].tolist() == [1000] * T


def test_argmax_unaligned_rows(cuda):
    """V odd: bf16 rows start off 16-byte boundaries; every split point is exercised."""
    for V in (1, 7, 1001, 40001):
        g = torch.Generator().manual_seed(V)
        x = (torch.randn(3, 5, V, generator=g) * 4).to(torch.bfloat16)
        parent = torch.tensor([[-1, 0, 0, 1, 2]] * 3, dtype=torch.int32)
        cand = torch.randint(0, V, (3, 5), generator=g, dtype=torch.int32)
        r = _accept_only(x, cand, parent, cuda)
        amax = oracle.argmax(x)
        assert torch.equal(r["argmax"], amax), V
        path, alen, bonus = oracle.accept_walk(parent, cand, amax)
        assert torch.equal(r["path"], path) and torch.equal(r["alen"], alen) and torch.equal(r["bonus"], bonus)


def test_walk_duplicates_and_deep_chain(cuda):
    V = 16
    parent = torch.tensor([[-1, 0, 0, 1, 2] + [-1] * 59,
                           [-1] + list(range(63))], dtype=torch.int32)
    parent[0, 5:] = 0                                    # extra root children
    cand = torch.zeros((2, 64), dtype=torch.int32)
    cand[0, :5] = torch.tensor([9, 5, 5, 7, 7])
    cand[0, 5:] = torch.arange(59) % 3 + 10
    logits = torch.zeros((2, 64, V), dtype=torch.float32)
    logits[0, 0, 5] = 1.0                                # root argmax 5: nodes 1 and 2 both match
    logits[0, 1, 1] = 1.0
    logits[0, 2, 7] = 1.0
    logits[1, :, 3] = 1.0                                # chain: every node predicts 3
    cand[1, 1:] = 3
    r = _accept_only(logits, cand, parent, cuda)
    amax = oracle.argmax(logits)
    path, alen, bonus = oracle.accept_walk(parent, cand, amax)
    assert torch.equal(r["path"], path) and torch.equal(r["alen"], alen) and torch.equal(r["bonus"], bonus)
    assert int(alen[0]) == 2 and int(alen[1]) == 64


def test_bad_tree_reports_status(cuda):
    w = workloads.get("7b_l2048", T=8, Hq=4, Hkv=4, L=300, V=1000, branching=(2, 2, 1))
    host = workloads.make(w)
    host["parent"][0, 5] = 6                             # a node whose parent comes after it
    t = to_dev(host, cuda)
    step = run_gpu(t)
    assert step.device_status() & pkg.api.ERR_BAD_TREE


def test_capacity_reports_status(cuda):
    w = workloads.get("7b_l2048", T=8, Hq=4, Hkv=4, L=300, V=1000, branching=(2, 2, 1))
    host = workloads.make(w)
    host["cache_len"][0] = host["Lcap"] - w.T + 1
    t = to_dev(host, cuda)
    step = run_gpu(t)
    assert step.device_status() & pkg.api.ERR_CAPACITY


def test_host_errors_raise(cuda):
    w = workloads.get("tiny_f32")
    t = to_dev(workloads.make(w), cuda)
    out = torch.empty_like(t["q"])
    with pytest.raises(pkg.CloverError):
        pkg.clover_verify_attn(t["q"], t["k_new"], t["v_new"], t["k_cache"], t["v_cache"], t["cache_len"],
                               t["parent"], out, scale=float("inf"))
    new_len = t["cache_len"]
    with pytest.raises(pkg.CloverError):   # new length may not alias the old one
        pkg.clover_kv_compact(t["k_cache"], t["v_cache"], t["cache_len"], torch.zeros_like(t["parent"]),
                              torch.ones_like(t["cache_len"]), new_len)


def test_accept_ex_commit_capacity_and_overlap_flag(cuda):
    """clover_verify_accept_ex with the commit fused in: a sequence whose cache
    has no room for T more slots raises CLOVER_ERR_CAPACITY and is left
    untouched, the others match clover_kv_commit; the overlap flag changes
    nothing in the results (here the preceding kernel is unrelated work)."""
    w = workloads.get("7b_l2048", B=3, T=16, Hq=4, Hkv=2, D=64, L=200, V=3000, branching=(4, 2, 1, 1))
    host = workloads.make(w)
    Lcap = host["Lcap"]
    host["cache_len"][1] = Lcap - w.T + 1                   # one slot short
    for overlap in (False, True):
        t = to_dev(host, cuda)
        i32 = dict(dtype=torch.int32, device=cuda)
        am, path = torch.empty((w.B, w.T), **i32), torch.empty((w.B, w.T), **i32)
        alen, bonus, ncl = torch.empty(w.B, **i32), torch.empty(w.B, **i32), torch.full((w.B,), -7, **i32)
        src = torch.empty((w.B, w.T), **i32)
        st = torch.zeros(1, **i32)
        ws = torch.zeros(pkg.clover_verify_accept_ex_workspace_size(w.B, w.T, w.V, w.torch_dtype, 2),
                         dtype=torch.uint8, device=cuda)
        scratch = torch.zeros(1 << 20, device=cuda)
        scratch.mul_(2.0)                                      # some unrelated kernel before the call
        pkg.clover_verify_accept_ex(t["logits"], t["cand"], t["parent"], am, path, alen, bonus, ws,
                                    commit=(t["k_cache"], t["v_cache"], t["k_new"], t["v_new"], t["cache_len"],
                                            ncl, src), overlap=overlap, status=st)
        torch.cuda.synchronize()
        assert int(st.item()) == 8                             # CLOVER_ERR_CAPACITY
        amax = oracle.argmax(host["logits"])
        rpath, ralen, rbonus = oracle.accept_walk(host["parent"], host["cand"], amax)
        assert torch.equal(path.cpu(), rpath) and torch.equal(alen.cpu(), ralen) and torch.equal(bonus.cpu(), rbonus)
        ok = torch.tensor([0, 2])
        kc_ok, vc_ok = host["k_cache"][ok].contiguous(), host["v_cache"][ok].contiguous()
        rsrc = oracle.kv_commit(kc_ok, vc_ok, host["k_new"][ok].contiguous(), host["v_new"][ok].contiguous(),
                                host["cache_len"][ok].contiguous(), rpath[ok], ralen[ok])
        for n, b in enumerate(ok.tolist()):
            m = int(host["cache_len"][b]) + int(ralen[b])
            assert int(ncl[b]) == m
            assert torch.equal(src[b].cpu(), rsrc[n])
            assert torch.equal(t["k_cache"][b, :, :m].cpu().view(torch.int16), kc_ok[n, :, :m].view(torch.int16))
            assert torch.equal(t["v_cache"][b, :, :m].cpu().view(torch.int16), vc_ok[n, :, :m].view(torch.int16))
        assert int(ncl[1]) == -7                              # not committed
        assert torch.equal(t["k_cache"][1].cpu().view(torch.int16), host["k_cache"][1].view(torch.int16))


@pytest.mark.parametrize("shared_step", [False, True])
@pytest.mark.parametrize("name,over", [("7b_l2048", dict(T=64, Hq=8, Hkv=8, L=1500, V=3000)),
                                       ("100b_gqa", dict(B=2, Hq=32, Hkv=4, L=900, V=2048))],
                         ids=["mha", "gqa_pair"])
def test_graph_of_overlapping_steps(name, over, shared_step, cuda):
    """The bench's arrangement: a CUDA graph of 30 fused steps (inputs-ready
    attention, accept + commit as its programmatic dependent) over three
    independent input sets, consecutive steps overlapping, replayed three
    times.  With one VerifyStep a set (or one shared by all, whose outputs
    then hold the last step's), every set's outputs and committed cache rows
    match the oracle afterwards (a step repeated on the same set rewrites the
    same rows), and no status bit is set."""
    hosts = [workloads.make(workloads.get(name, seed=90 + k, **over)) for k in range(3)]
    sets = [to_dev(h, cuda) for h in hosts]
    B, T, Hq, D = sets[0]["q"].shape
    Hkv = sets[0]["k_new"].shape[2]
    V = sets[0]["logits"].shape[-1]
    Lcap = max(s["Lcap"] for s in sets)
    assert all(s["Lcap"] == Lcap for s in sets)

    def new_step():
        return pkg.VerifyStep(B, T, Hq, Hkv, D, Lcap, V, torch.bfloat16, device=cuda, schedule="fused",
                              attn_launch="inputs_ready")

    steps = [new_step()] * 3 if shared_step else [new_step() for _ in range(3)]
    stream = torch.cuda.Stream()

    def run_all():
        for _ in range(10):
            for step, s in zip(steps, sets):
                step.run(s["q"], s["k_new"], s["v_new"], s["k_cache"], s["v_cache"], s["cache_len"], s["parent"],
                         s["cand"], s["logits"], stream=stream)

    with torch.cuda.stream(stream):
        run_all()                                  # eager warm-up (kernel attributes set before capture)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        run_all()
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    if shared_step:
        compare_full(hosts[2], steps[2], sets[2])
    else:
        for h, step, s in zip(hosts, steps, sets):
            compare_full(h, step, s)
