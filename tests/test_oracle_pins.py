"""Pins for the oracle: every function is checked against something other than
itself -- brute force on tiny inputs, library routines (torch SDPA, numpy argmax),
closed forms, hand-worked examples and invariants -- so that a dropped term, a
wrong index, a wrong sign or a transposed operand fails at least one test.

Pure CPU; marked neither gpu nor slow.
"""

import itertools
import json
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
from synth import trees, workloads

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ---------------------------------------------------------------------------
# helpers (independent formulations used only as pins)
# ---------------------------------------------------------------------------

def reach_matrix(parent):
    """Ancestor-or-self relation as the transitive closure of the parent map:
    R = (I + A)^(T) with boolean products, A[i][p] = 1 iff p = parent[i]."""
    T = len(parent)
    A = np.zeros((T, T), dtype=np.int64)
    for i in range(1, T):
        A[i, parent[i]] = 1
    R = np.eye(T, dtype=np.int64)
    step = np.eye(T, dtype=np.int64) + A
    for _ in range(T):
        R = np.minimum(R @ step, 1)
    return R.astype(bool)


def root_path(parent, i):
    path = []
    n = i
    while n >= 0:
        path.append(n)
        n = parent[n]
    return path[::-1]


def rand_inputs(B, T, Hq, Hkv, D, L, seed, dtype=torch.float32, Lcap=None, std=1.0):
    g = torch.Generator().manual_seed(seed)
    Lmax = max(L) if isinstance(L, (list, tuple)) else L
    Lcap = Lcap or Lmax + T + 3
    def r(*s):
        return (torch.randn(*s, generator=g, dtype=torch.float64) * std).to(dtype)
    inp = dict(q=r(B, T, Hq, D), k_new=r(B, T, Hkv, D), v_new=r(B, T, Hkv, D),
               k_cache=r(B, Hkv, Lcap, D), v_cache=r(B, Hkv, Lcap, D))
    Ls = list(L) if isinstance(L, (list, tuple)) else [L] * B
    inp["cache_len"] = torch.tensor(Ls, dtype=torch.int32)
    return inp


def sdpa_decode(q, K, V, scale):
    """One query row against a key/value list, via torch's SDPA in fp64."""
    return F.scaled_dot_product_attention(
        q.double().view(1, 1, 1, -1), K.double().view(1, 1, K.shape[0], -1),
        V.double().view(1, 1, V.shape[0], -1), scale=scale).view(-1)


def sequence_attention(inp, parent, scale):
    """Tree attention by its definition in terms of the speculated sequences:
    node i is the last token of the sequence root..i appended to the cache, so
    its output is plain decode attention over cache ++ k_new[root path of i]."""
    q, kn, vn, kc, vc, cl = (inp[k] for k in ("q", "k_new", "v_new", "k_cache", "v_cache", "cache_len"))
    B, T, Hq, D = q.shape
    Hkv = kn.shape[2]
    G = Hq // Hkv
    out = torch.empty((B, T, Hq, D), dtype=torch.float64)
    for b in range(B):
        L = int(cl[b])
        par = parent[b]
        for i in range(T):
            nodes = root_path(par, i)
            for h in range(Hq):
                g = h // G
                K = torch.cat([kc[b, g, :L], kn[b, nodes, g]], 0)
                V = torch.cat([vc[b, g, :L], vn[b, nodes, g]], 0)
                out[b, i, h] = sdpa_decode(q[b, i, h], K, V, scale)
    return out


def run_oracle_attn(inp, parent, scale=0.0):
    par = torch.tensor(parent, dtype=torch.int32)
    if par.dim() == 1:
        par = par.unsqueeze(0)
    return oracle.tree_attention(inp["q"], inp["k_new"], inp["v_new"], inp["k_cache"],
                                 inp["v_cache"], inp["cache_len"], par, scale=scale)


# ---------------------------------------------------------------------------
# A0: tree encoding
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("T", [1, 2, 3, 4, 5])
def test_tree_mask_all_small_trees_vs_transitive_closure(T):
    for parent in trees.all_trees(T):
        mask, depth = oracle.tree_mask(parent)
        R = reach_matrix(parent)
        assert np.array_equal(mask.numpy(), R), parent
        assert depth.tolist() == [int(R[i].sum()) - 1 for i in range(T)]


def test_tree_mask_invariants_random_64():
    for seed in range(20):
        parent = trees.random_tree(64, seed)
        mask, depth = oracle.tree_mask(parent)
        m = mask.numpy()
        assert np.array_equal(m, reach_matrix(parent))
        for i in range(64):
            assert m[i, 0] and m[i, i]
            assert not m[i, i + 1:].any()
            if i:
                expect = m[parent[i]].copy()
                expect[i] = True
                assert np.array_equal(m[i], expect)
            assert m[i].sum() == depth[i] + 1


@pytest.mark.parametrize("bad", [[0, 0, 1], [-1, 1], [-1, 0, 2], [-1, 0, -1], [-1, 0, 5], [-1, -1]])
def test_tree_mask_rejects_invalid(bad):
    with pytest.raises(oracle.OracleError) as e:
        oracle.tree_mask(bad)
    assert e.value.code == oracle.BAD_TREE


def test_topk_tree_shapes_match_reading():
    t16 = trees.topk_tree(16, [4, 2, 1, 1])
    assert t16 == json.load(open(os.path.join(GOLDEN, "topk_trees.json")))["T16_b4211"]["parent"]
    for T, br, counts in [(16, [4, 2, 1, 1], [1, 3, 4, 4, 4]), (64, [8, 4, 2, 2, 1], [1, 6, 12, 13, 16, 16]),
                          (32, [8, 4, 2, 1], [1, 4, 8, 11, 8])]:
        _, depth = oracle.tree_mask(trees.topk_tree(T, br))
        assert np.bincount(depth.numpy()).tolist() == counts


# ---------------------------------------------------------------------------
# A1: tree-masked attention
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("T", [1, 2, 3, 4])
@pytest.mark.parametrize("L", [0, 1, 3])
def test_attention_brute_force_all_small_trees(T, L):
    inp = rand_inputs(1, T, 2, 2, 4, L, seed=100 * T + L)
    for parent in trees.all_trees(T):
        got = run_oracle_attn(inp, [parent])
        ref = sequence_attention(inp, [parent], 0.5)
        assert torch.allclose(got, ref, atol=1e-13, rtol=0), parent


def test_attention_sequences_gqa_batched_random_trees():
    B, T, Hq, Hkv, D = 3, 12, 8, 2, 16
    inp = rand_inputs(B, T, Hq, Hkv, D, [5, 0, 9], seed=7)
    parents = [trees.random_tree(T, 11, tag=b) for b in range(B)]
    got = run_oracle_attn(inp, parents)
    ref = sequence_attention(inp, parents, 1 / math.sqrt(D))
    assert torch.allclose(got, ref, atol=1e-13, rtol=0)


def test_attention_chain_equals_causal():
    B, T, H, D, L = 2, 9, 3, 8, 6
    inp = rand_inputs(B, T, H, H, D, L, seed=3)
    got = run_oracle_attn(inp, [trees.chain_tree(T)] * B)
    # causal attention of the whole sequence cache ++ tree, last T positions
    causal = torch.ones(L + T, L + T, dtype=torch.bool).tril()[L:]
    for b in range(B):
        K = torch.cat([inp["k_cache"][b, :, :L], inp["k_new"][b].transpose(0, 1)], 1)
        V = torch.cat([inp["v_cache"][b, :, :L], inp["v_new"][b].transpose(0, 1)], 1)
        Q = inp["q"][b].transpose(0, 1)
        ref = F.scaled_dot_product_attention(Q.double(), K.double(), V.double(), attn_mask=causal,
                                             scale=1 / math.sqrt(D))
        assert torch.allclose(got[b], ref.transpose(0, 1), atol=1e-13, rtol=0)


def test_attention_single_node_is_plain_decode():
    B, H, D, L = 2, 4, 32, 17
    inp = rand_inputs(B, 1, H, H, D, L, seed=4)
    got = run_oracle_attn(inp, [[-1]] * B)
    for b in range(B):
        K = torch.cat([inp["k_cache"][b, :, :L], inp["k_new"][b].transpose(0, 1)], 1)
        V = torch.cat([inp["v_cache"][b, :, :L], inp["v_new"][b].transpose(0, 1)], 1)
        ref = F.scaled_dot_product_attention(inp["q"][b].transpose(0, 1).double(), K.double(), V.double())
        assert torch.allclose(got[b], ref.transpose(0, 1), atol=1e-13, rtol=0)


def test_attention_star_tree():
    T, H, D, L = 6, 2, 8, 4
    inp = rand_inputs(1, T, H, H, D, L, seed=5)
    got = run_oracle_attn(inp, [trees.star_tree(T)])
    for i in range(T):
        nodes = [0] if i == 0 else [0, i]
        for h in range(H):
            K = torch.cat([inp["k_cache"][0, h, :L], inp["k_new"][0, nodes, h]], 0)
            V = torch.cat([inp["v_cache"][0, h, :L], inp["v_new"][0, nodes, h]], 0)
            assert torch.allclose(got[0, i, h], sdpa_decode(inp["q"][0, i, h], K, V, 1 / math.sqrt(D)),
                                  atol=1e-13, rtol=0)


def test_attention_uniform_values_and_empty_cache():
    T, H, D, L = 5, 2, 8, 7
    inp = rand_inputs(1, T, H, H, D, L, seed=6)
    row = torch.arange(D, dtype=torch.float64) * 0.25 - 1
    inp["v_cache"][:] = row
    inp["v_new"][:] = row
    got = run_oracle_attn(inp, [trees.random_tree(T, 1)])
    assert torch.allclose(got, row.expand_as(got), atol=1e-14, rtol=0)
    # L = 0 and T = 1: the only visible key is the node itself
    inp0 = rand_inputs(1, 1, 3, 3, 8, 0, seed=8)
    got0 = run_oracle_attn(inp0, [[-1]])
    assert torch.equal(got0[0, 0], inp0["v_new"][0, 0])


def test_attention_zero_query_is_mean_of_visible_values():
    """q = 0 gives equal weights: out = mean of the values of the visible keys,
    of which there are L + depth(i) + 1 (closed form)."""
    T, H, D, L = 16, 2, 1, 5
    parent = trees.topk_tree(T, [4, 2, 1, 1])
    inp = rand_inputs(1, T, H, H, D, L, seed=9)
    inp["q"][:] = 0
    inp["v_cache"][0, :, :, 0] = torch.arange(inp["v_cache"].shape[2], dtype=torch.float64)
    inp["v_new"][0, :, :, 0] = 1000.0 * torch.arange(1, T + 1, dtype=torch.float64).unsqueeze(1)
    got = run_oracle_attn(inp, [parent])
    for i in range(T):
        nodes = root_path(parent, i)
        expect = (sum(range(L)) + 1000.0 * sum(n + 1 for n in nodes)) / (L + len(nodes))
        assert got[0, i, :, 0].tolist() == pytest.approx([expect] * H, abs=1e-9)


def test_attention_cache_key_permutation_invariance():
    T, H, D, L = 8, 2, 8, 11
    inp = rand_inputs(1, T, H, H, D, L, seed=10)
    parent = [trees.random_tree(T, 3)]
    base = run_oracle_attn(inp, parent)
    perm = torch.randperm(L, generator=torch.Generator().manual_seed(1))
    inp2 = dict(inp)
    for k in ("k_cache", "v_cache"):
        c = inp[k].clone()
        c[:, :, :L] = inp[k][:, :, perm]
        inp2[k] = c
    assert torch.allclose(run_oracle_attn(inp2, parent), base, atol=1e-13, rtol=0)


def test_attention_gqa_equals_mha_with_repeated_kv_heads():
    B, T, Hq, Hkv, D, L = 2, 6, 8, 2, 8, 5
    G = Hq // Hkv
    inp = rand_inputs(B, T, Hq, Hkv, D, L, seed=12)
    parents = [trees.random_tree(T, 5, tag=b) for b in range(B)]
    got = run_oracle_attn(inp, parents)
    mha = dict(inp)
    for k, dim in (("k_new", 2), ("v_new", 2), ("k_cache", 1), ("v_cache", 1)):
        mha[k] = inp[k].repeat_interleave(G, dim=dim).contiguous()
    assert torch.allclose(run_oracle_attn(mha, parents), got, atol=1e-13, rtol=0)


def test_attention_scale_closed_form():
    """One cache key with score s*a and the root with score 0: out =
    (v_c * e^{s a} + v_0) / (e^{s a} + 1)."""
    inp = rand_inputs(1, 1, 1, 1, 1, 1, seed=13)
    a, vc, v0 = 1.5, 2.0, -3.0
    inp["q"][:] = 1.0
    inp["k_cache"][0, 0, 0, 0] = a
    inp["k_new"][:] = 0.0
    inp["v_cache"][0, 0, 0, 0] = vc
    inp["v_new"][:] = v0
    for s in (0.0, 0.3, 2.0):
        got = run_oracle_attn(inp, [[-1]], scale=s)
        ss = 1.0 if s == 0.0 else s   # scale 0 selects 1/sqrt(D) = 1 for D = 1
        w = math.exp(ss * a)
        assert float(got[0, 0, 0, 0]) == pytest.approx((vc * w + v0) / (w + 1), abs=1e-15)


def test_attention_huge_scores_closed_form():
    """Scores far past exp's range (s*a up to 1e4): the softmax is taken
    relative to the row maximum, so the output is the closed form of
    test_attention_scale_closed_form with e^{-s a} underflowing to 0: v_c
    when the cache key dominates, v_0 when its score is hugely negative, and
    the plain mean when both scores are equal and huge."""
    inp = rand_inputs(1, 1, 1, 1, 1, 1, seed=14)
    vc, v0 = 2.0, -3.0
    inp["v_cache"][0, 0, 0, 0] = vc
    inp["v_new"][:] = v0
    for qv, a, kr, want in ((1.0, 800.0, 0.0, vc), (1.0, -5000.0, 0.0, v0), (10.0, 1000.0, 1000.0, (vc + v0) / 2)):
        inp["q"][:] = qv
        inp["k_cache"][0, 0, 0, 0] = a
        inp["k_new"][:] = kr
        got = run_oracle_attn(inp, [[-1]], scale=1.0)
        assert float(got[0, 0, 0, 0]) == want


def test_attention_hand_worked_example():
    ex = json.load(open(os.path.join(GOLDEN, "hand_tree_attention.json")))
    T = len(ex["parent"])
    t32 = lambda x: torch.tensor(x, dtype=torch.float32)
    q = t32(ex["q"]).view(1, T, 1, 1)
    k_new = t32(ex["k_new"]).view(1, T, 1, 1)
    v_new = t32(ex["v_new"]).view(1, T, 1, 1)
    L = len(ex["k_cache"])
    k_cache = t32(ex["k_cache"] + [0.0] * T).view(1, 1, L + T, 1)
    v_cache = t32(ex["v_cache"] + [0.0] * T).view(1, 1, L + T, 1)
    got = oracle.tree_attention(q, k_new, v_new, k_cache, v_cache, torch.tensor([L], dtype=torch.int32),
                                torch.tensor([ex["parent"]], dtype=torch.int32), scale=ex["scale"])
    assert got.view(-1).tolist() == pytest.approx(ex["expected_out"], abs=1e-6)


def test_attention_bf16_widening_matches_f32():
    """bf16 bytes are widened exactly: inputs representable in bf16 give the
    same fp64 result whether stored as bf16 or fp32."""
    inp = rand_inputs(2, 7, 4, 2, 16, [3, 8], seed=14, dtype=torch.float32)
    inp = {k: (v.to(torch.bfloat16).to(torch.float32) if v.is_floating_point() else v) for k, v in inp.items()}
    bf = {k: (v.to(torch.bfloat16) if v.is_floating_point() else v) for k, v in inp.items()}
    parents = [trees.random_tree(7, 2, tag=b) for b in range(2)]
    assert torch.equal(run_oracle_attn(inp, parents), run_oracle_attn(bf, parents))


def test_attention_sharp_scores_stable():
    inp = rand_inputs(1, 8, 2, 2, 16, 20, seed=15, std=6.0)   # scores up to ~hundreds
    parents = [trees.random_tree(8, 9)]
    got = run_oracle_attn(inp, parents)
    assert torch.isfinite(got).all()
    assert torch.allclose(got, sequence_attention(inp, parents, 0.25), atol=1e-12, rtol=0)


def test_attention_rows_subset_matches_full_and_ignores_tail():
    w = workloads.get("tiny_f32")
    t = workloads.make(w)           # cache tail slots hold NaN
    full = oracle.tree_attention(t["q"], t["k_new"], t["v_new"], t["k_cache"], t["v_cache"],
                                 t["cache_len"], t["parent"])
    assert torch.isfinite(full).all()
    rows = [0, 5, 77, w.T * w.Hq - 1]
    sub = oracle.tree_attention(t["q"], t["k_new"], t["v_new"], t["k_cache"], t["v_cache"],
                                t["cache_len"], t["parent"], rows=rows)
    assert torch.equal(sub, full.view(-1, w.D)[rows])
    one = oracle.tree_attention(t["q"], t["k_new"], t["v_new"], t["k_cache"], t["v_cache"],
                                t["cache_len"], t["parent"], n_threads=1)
    assert torch.equal(one, full)


def test_attention_rejects_bad_tree():
    inp = rand_inputs(1, 3, 1, 1, 2, 1, seed=16)
    with pytest.raises(oracle.OracleError) as e:
        run_oracle_attn(inp, [[-1, 0, 2]])
    assert e.value.code == oracle.BAD_TREE


# ---------------------------------------------------------------------------
# A2: argmax
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("V", [1, 7, 1024, 5003])
def test_argmax_vs_numpy_first_index(dtype, V):
    g = torch.Generator().manual_seed(V)
    x = (torch.randn(6, 5, V, generator=g) * 4).to(dtype)
    got = oracle.argmax(x)
    ref = np.argmax(x.to(torch.float64).numpy(), axis=-1)   # numpy returns the first maximum
    assert np.array_equal(got.numpy(), ref)


def test_argmax_planted_ties_signed_zero_and_infinities():
    V = 300
    x = torch.full((8, V), -5.0, dtype=torch.float32)
    x[0, [17, 3, 250]] = 9.0                        # tie -> smallest index 3
    x[1, :] = -1.0
    x[1, 40] = -0.0
    x[1, 20] = 0.0                                   # -0 == +0 -> index 20
    x[2, :] = -1.0
    x[2, 10] = 0.0
    x[2, 5] = -0.0                                   # -> index 5
    x[3, 0] = 1.0                                    # max at index 0
    x[4, V - 1] = 1.0                                # max at the last index
    x[5, :] = float("-inf")
    x[5, 123] = -1e30                                # finite beats -inf
    x[6, 99] = float("inf")
    x[6, 7] = 1e38                                   # +inf wins
    x[7, :] = float("-inf")                          # all -inf -> index 0
    assert oracle.argmax(x).tolist() == [3, 20, 5, 0, V - 1, 123, 99, 0]
    assert oracle.argmax(x.to(torch.bfloat16)).tolist()[:5] == [3, 20, 5, 0, V - 1]


def test_argmax_row_subset():
    x = torch.randn(10, 50, generator=torch.Generator().manual_seed(2)).to(torch.bfloat16)
    full = oracle.argmax(x)
    assert oracle.argmax(x, rows=[9, 0, 4]).tolist() == full[[9, 0, 4]].tolist()


# ---------------------------------------------------------------------------
# A3: acceptance walk
# ---------------------------------------------------------------------------

def brute_force_walk(parent, cand, amax):
    """All root-to-node paths; keep those whose every step matches (child's
    candidate == parent's argmax) and that cannot be extended; the accepted
    path is the lexicographically smallest of them (node-index order)."""
    T = len(parent)
    children = [[c for c in range(T) if parent[c] == n] for n in range(T)]
    good = []
    for i in range(T):
        p = root_path(parent, i)
        if all(cand[p[k]] == amax[p[k - 1]] for k in range(1, len(p))):
            if not any(cand[c] == amax[i] for c in children[i]):
                good.append(p)
    best = min(good)
    return best, len(best), amax[best[-1]]


@pytest.mark.parametrize("T", [1, 2, 3, 4, 5])
def test_walk_exhaustive_small(T):
    """Every tree with T <= 5 nodes, every candidate/argmax assignment over a
    2-token vocabulary (duplicates among siblings included)."""
    n = 0
    for parent in trees.all_trees(T):
        for cand in itertools.product([0, 1], repeat=T):
            for amax in itertools.product([0, 1], repeat=T):
                path, alen, bonus = oracle.accept_walk(torch.tensor([parent]), torch.tensor([cand]),
                                                       torch.tensor([amax]))
                bp, bl, bb = brute_force_walk(parent, cand, amax)
                assert path[0, :bl].tolist() == bp and int(alen[0]) == bl and int(bonus[0]) == bb
                assert (path[0, bl:] == -1).all()
                n += 1
                if n > 4000:
                    return


def test_walk_distinct_siblings_gives_deepest_path_and_bounds():
    for seed in range(30):
        w = workloads.get("tiny_f32", seed=seed, tree="random" if seed % 2 else "topk")
        t = workloads.make(w)
        amax = oracle.argmax(t["logits"])
        path, alen, bonus = oracle.accept_walk(t["parent"], t["cand"], amax)
        parent = t["parent"][0].tolist()
        cand = t["cand"][0].tolist()
        a = amax[0].tolist()
        T = len(parent)
        full = [i for i in range(T)
                if all(cand[p] == a[parent[p]] for p in root_path(parent, i)[1:])]
        deepest = max(len(root_path(parent, i)) for i in full)
        assert int(alen[0]) == deepest
        _, depth = oracle.tree_mask(parent)
        assert 1 <= int(alen[0]) <= int(depth.max()) + 1
        assert int(bonus[0]) == a[path[0, int(alen[0]) - 1]]


def test_walk_plant_all_and_plant_none():
    for seed in range(5):
        w = workloads.get("tiny_f32", seed=seed, plant_p=1.0)
        t = workloads.make(w)
        amax = oracle.argmax(t["logits"])
        path, alen, _ = oracle.accept_walk(t["parent"], t["cand"], amax)
        last = int(path[0, int(alen[0]) - 1])
        assert last not in t["parent"][0].tolist()          # reached a leaf
        _, depth = oracle.tree_mask(t["parent"][0].tolist())
        assert int(alen[0]) == int(depth[last]) + 1
        # with no planting the root row's argmax is a random token: the walk
        # stops at the root unless a child's id happens to equal it
        w0 = workloads.get("tiny_f32", seed=seed, plant_p=0.0)
        t0 = workloads.make(w0)
        a0 = oracle.argmax(t0["logits"])
        _, alen0, _ = oracle.accept_walk(t0["parent"], t0["cand"], a0)
        kids = [c for c in range(w0.T) if t0["parent"][0, c] == 0]
        if all(int(t0["cand"][0, c]) != int(a0[0, 0]) for c in kids):
            assert int(alen0[0]) == 1


def test_walk_duplicate_siblings_smallest_index_wins():
    parent = [-1, 0, 0, 1, 2]
    cand = [9, 5, 5, 7, 7]
    amax = [5, 1, 7, 0, 0]        # node 1 is a dead end, node 2 continues to 4
    path, alen, bonus = oracle.accept_walk(torch.tensor([parent]), torch.tensor([cand]),
                                           torch.tensor([amax]))
    assert path[0].tolist() == [0, 1, -1, -1, -1] and int(alen[0]) == 2 and int(bonus[0]) == 1


# ---------------------------------------------------------------------------
# A4: append + compaction
# ---------------------------------------------------------------------------

def test_append_places_tree_kv_after_cache():
    B, T, Hkv, D = 2, 5, 3, 4
    inp = rand_inputs(B, T, Hkv, Hkv, D, [2, 6], seed=20, dtype=torch.float32)
    kc, vc = inp["k_cache"].clone(), inp["v_cache"].clone()
    oracle.append_tree_kv(inp["k_new"], inp["v_new"], kc, vc, inp["cache_len"])
    for b, L in enumerate(inp["cache_len"].tolist()):
        assert torch.equal(kc[b, :, L:L + T], inp["k_new"][b].permute(1, 0, 2))
        assert torch.equal(vc[b, :, L:L + T], inp["v_new"][b].permute(1, 0, 2))
        assert torch.equal(kc[b, :, :L], inp["k_cache"][b, :, :L])


def test_compact_equals_out_of_place_gather():
    B, T, Hkv, D = 3, 8, 2, 4
    for dtype in (torch.float32, torch.bfloat16):
        g = torch.Generator().manual_seed(21)
        Lcap = 30
        kc = torch.randn(B, Hkv, Lcap, D, generator=g).to(dtype)
        vc = torch.randn(B, Hkv, Lcap, D, generator=g).to(dtype)
        L = torch.tensor([0, 7, 22], dtype=torch.int32)
        paths = [[0, 2, 5, 7], [0], [0, 1, 2, 3, 4, 5, 6, 7]]
        path = torch.full((B, T), -1, dtype=torch.int32)
        for b, p in enumerate(paths):
            path[b, :len(p)] = torch.tensor(p)
        alen = torch.tensor([len(p) for p in paths], dtype=torch.int32)
        k2, v2, L2 = kc.clone(), vc.clone(), L.clone()
        src = oracle.kv_compact(k2, v2, L2, path, alen)
        for b, p in enumerate(paths):
            l0 = int(L[b])
            gather_k = kc[b, :, [l0 + j for j in p]]          # read from the untouched copy
            assert torch.equal(k2[b, :, l0:l0 + len(p)], gather_k)
            assert torch.equal(v2[b, :, l0:l0 + len(p)], vc[b, :, [l0 + j for j in p]])
            assert torch.equal(k2[b, :, :l0], kc[b, :, :l0])
            assert src[b].tolist() == [l0 + j for j in p] + [-1] * (T - len(p))
            assert int(L2[b]) == l0 + len(p)


def test_commit_equals_append_then_compact():
    """The commit from k_new/v_new reaches the end state of append + compaction
    (slots < L + a; the tree slots past L + a are unspecified afterwards)."""
    B, T, Hkv, D = 3, 8, 2, 4
    for dtype in (torch.float32, torch.bfloat16):
        inp = rand_inputs(B, T, Hkv, Hkv, D, [0, 5, 19], seed=22, dtype=dtype)
        paths = [[0, 3, 6], [0], [0, 1, 2, 3, 4, 5, 6, 7]]
        path = torch.full((B, T), -1, dtype=torch.int32)
        for b, q in enumerate(paths):
            path[b, :len(q)] = torch.tensor(q)
        alen = torch.tensor([len(q) for q in paths], dtype=torch.int32)
        k1, v1, L1 = inp["k_cache"].clone(), inp["v_cache"].clone(), inp["cache_len"].clone().to(torch.int32)
        oracle.append_tree_kv(inp["k_new"], inp["v_new"], k1, v1, L1)
        src1 = oracle.kv_compact(k1, v1, L1, path, alen)
        k2, v2, L2 = inp["k_cache"].clone(), inp["v_cache"].clone(), inp["cache_len"].clone().to(torch.int32)
        src2 = oracle.kv_commit(k2, v2, inp["k_new"], inp["v_new"], L2, path, alen)
        assert torch.equal(L1, L2)
        for b, q in enumerate(paths):
            n = int(L2[b])
            assert torch.equal(k1[b, :, :n], k2[b, :, :n]) and torch.equal(v1[b, :, :n], v2[b, :, :n])
            l0 = int(inp["cache_len"][b])
            assert src2[b].tolist() == q + [-1] * (T - len(q))
            assert src1[b].tolist() == [l0 + j for j in q] + [-1] * (T - len(q))
            # slots past the new length are not written by the commit
            assert torch.equal(k2[b, :, n:], inp["k_cache"][b, :, n:])


def test_commit_rejects_bad_paths():
    B, T, Hkv, D = 1, 4, 1, 4
    inp = rand_inputs(B, T, Hkv, Hkv, D, [3], seed=23, dtype=torch.float32)
    for path, alen in (([0, 4, -1, -1], 2), ([0, -1, -1, -1], 0), ([0, 1, 2, 3], 5)):
        k, v, L = inp["k_cache"].clone(), inp["v_cache"].clone(), inp["cache_len"].clone().to(torch.int32)
        with pytest.raises(Exception):
            oracle.kv_commit(k, v, inp["k_new"], inp["v_new"], L, torch.tensor([path], dtype=torch.int32),
                             torch.tensor([alen], dtype=torch.int32))


def test_verify_step_tiny_invariants():
    w = workloads.get("tiny_f32")
    t = workloads.make(w)
    r = oracle.verify_step(t)
    a = int(r["accept_len"][0])
    L = int(t["cache_len"][0])
    assert int(r["cache_len"][0]) == L + a
    assert torch.equal(r["k_cache"][0, :, :L], t["k_cache"][0, :, :L])
    p = r["path"][0, :a].tolist()
    assert torch.equal(r["k_cache"][0, :, L:L + a], t["k_new"][0, p].permute(1, 0, 2))
    assert torch.equal(r["v_cache"][0, :, L:L + a], t["v_new"][0, p].permute(1, 0, 2))


def test_verify_step_typical_at_small_temperature_is_greedy():
    """The whole step under typical acceptance at temperature 1e-3: every
    argmax candidate has probability ~1 (the logits' top gap is far above the
    temperature) and every other candidate ~0, so with epsilon = delta = 0.3
    exactly the argmax children pass and the step equals the greedy step
    (siblings are distinct by construction)."""
    w = workloads.get("tiny_f32")
    t = workloads.make(w)
    top2 = t["logits"].double().topk(2, dim=-1).values
    assert (top2[..., 0] - top2[..., 1]).min() > 0.05
    g = oracle.verify_step(t)
    ty = oracle.verify_step(t, typical=(1e-3, 0.3, 0.3))
    for key in ("out", "argmax", "path", "accept_len", "bonus", "src_index", "cache_len"):
        assert torch.equal(ty[key], g[key]), key
    a = int(g["accept_len"][0])
    L = int(t["cache_len"][0])
    assert torch.equal(ty["k_cache"][0, :, :L + a], g["k_cache"][0, :, :L + a])


# ---------------------------------------------------------------------------
# A6: typical acceptance (the sampling-side acceptance rule)
# ---------------------------------------------------------------------------

def typical_by_library(logits, parent, cand, tau, eps, delta):
    """Independent statement with library routines: scipy's softmax and
    entropy in fp64, the threshold compared in the probability domain, and
    the path chosen among every fully accepted root path by sort order."""
    special = pytest.importorskip("scipy.special")
    stats = pytest.importorskip("scipy.stats")
    x = logits.double().numpy()
    T, V = x.shape
    p = special.softmax(x / tau, axis=-1)
    theta = np.minimum(eps, delta * np.exp(-stats.entropy(p, axis=-1)))
    ok = [True] + [0 <= cand[c] < V and bool(p[parent[c], cand[c]] > theta[parent[c]]) for c in range(1, T)]
    good = [root_path(parent, i) for i in range(T) if all(ok[n] for n in root_path(parent, i))]
    best = sorted(good, key=lambda q: (-len(q), q))[0]
    log_margin = [math.inf] + [
        (math.log(p[parent[c], cand[c]]) - math.log(theta[parent[c]]) if theta[parent[c]] > 0 else math.inf)
        if 0 <= cand[c] < V else -math.inf for c in range(1, T)]
    return best, int(np.argmax(x[best[-1]])), np.argmax(x, axis=-1), log_margin


def run_typical(logits, parent, cand, tau, eps, delta):
    T, V = logits.shape
    r = oracle.accept_typical(logits.reshape(1, T, V), torch.tensor([parent]), torch.tensor([cand]), tau, eps, delta)
    a = int(r["accept_len"][0])
    return r["path"][0, :a].tolist(), int(r["bonus"][0]), r["argmax"][0], r["margin"][0], r["path"][0, a:]


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_typical_brute_force_vs_library(dtype):
    g = torch.Generator().manual_seed(11)
    n = 0
    for T in (1, 2, 4, 6, 9):
        for V in (1, 2, 7, 33):
            for tau, eps, delta in ((1.0, 0.09, 0.3), (0.3, 0.3, 0.55), (2.5, 0.0, 0.3), (0.7, 0.2, 0.0),
                                    (1.0, 0.05, 0.9)):
                for rep in range(3):
                    parent = trees.random_tree(T, seed=100 * T + rep, tag=V)
                    logits = (torch.randn(T, V, generator=g, dtype=torch.float64) * 2.0).to(dtype)
                    cand = torch.randint(-1, V + 1, (T,), generator=g).tolist()
                    path, bonus, amax, margin, tail = run_typical(logits, parent, cand, tau, eps, delta)
                    bp, bb, ba, bm = typical_by_library(logits, parent, cand, tau, eps, delta)
                    assert amax.tolist() == ba.tolist()
                    for c in range(T):
                        if math.isinf(bm[c]):
                            assert float(margin[c]) == bm[c]
                        else:
                            assert float(margin[c]) == pytest.approx(bm[c], rel=1e-9, abs=1e-9)
                    assert min(abs(float(m)) for m in margin) > 1e-9       # no edge on the boundary
                    assert path == bp and bonus == bb and (tail == -1).all()
                    n += 1
    assert n == 2 * 0 + 5 * 4 * 5 * 3


def test_typical_two_token_worked_example():
    """V = 2, logits (ln 4, 0) at temperature 1: p = (0.8, 0.2), entropy
    0.5004024 nats, e^-H = 0.6062866.  Child token 1 has p = 0.2.
    (eps, delta) = (0.09, 0.3): theta = min(0.09, 0.1818860) = 0.09, accepted,
    margin ln(0.2 / 0.09) = 0.7985077.  (0.25, 0.4): theta = 0.2425147,
    rejected, margin ln(0.2 / 0.2425147) = -0.1927447.  Doubling both the
    logits and the temperature changes nothing."""
    for scale in (1.0, 2.0):
        logits = torch.tensor([[math.log(4.0) * scale, 0.0], [0.0, 0.0]], dtype=torch.float64).float()
        path, bonus, amax, margin, _ = run_typical(logits, [-1, 0], [7, 1], scale, 0.09, 0.3)
        assert path == [0, 1] and bonus == 0 and amax.tolist() == [0, 0]
        assert float(margin[1]) == pytest.approx(0.7985077, abs=2e-6)
        path, bonus, _, margin, _ = run_typical(logits, [-1, 0], [7, 1], scale, 0.25, 0.4)
        assert path == [0] and bonus == 0
        assert float(margin[1]) == pytest.approx(-0.1927447, abs=2e-6)
        # token 0 (p = 0.8) passes either threshold
        path, _, _, margin, _ = run_typical(logits, [-1, 0], [7, 0], scale, 0.25, 0.4)
        assert path == [0, 1] and float(margin[1]) == pytest.approx(math.log(0.8 / 0.2425147), abs=2e-6)


def test_typical_uniform_logits_accept_every_edge():
    """Uniform logits: p = 1/V and H = ln V, so theta = min(eps, delta / V);
    with delta < 1 < eps * V every edge passes with margin -ln(delta)."""
    V, delta = 1000, 0.5
    for branching, T in (([3, 2, 2], 10), ([1, 1, 1, 1], 5), ([4], 5)):
        parent = trees.topk_tree(T, branching)
        logits = torch.zeros(T, V, dtype=torch.bfloat16)
        cand = [0] + [(7 * c) % V for c in range(1, T)]
        path, bonus, _, margin, _ = run_typical(logits, parent, cand, 0.8, 0.09, delta)
        _, depth = oracle.tree_mask(parent)
        deepest = [i for i in range(T) if int(depth[i]) == int(depth.max())]
        assert path == min(root_path(parent, i) for i in deepest)
        assert bonus == 0
        assert np.allclose(margin[1:].numpy(), -math.log(delta), atol=1e-12)


def test_typical_zero_epsilon_and_degenerate_candidates():
    """eps = 0: theta = 0 and every finite candidate passes, however unlikely
    (here p ~ e^-2000); a -inf logit (p = 0) and a token outside [0, V) do not."""
    V = 16
    parent = [-1, 0, 0, 1, 2, 4]
    logits = torch.zeros(6, V, dtype=torch.float32)
    logits[:, 3] = 2000.0
    cand = [0, 5, 9, 1, 2, 8]
    path, bonus, _, margin, _ = run_typical(logits, parent, cand, 1.0, 0.0, 0.3)
    assert path == [0, 2, 4, 5] and bonus == 3
    assert all(math.isinf(float(m)) and float(m) > 0 for m in margin)
    logits[4, 8] = -math.inf                   # node 5's token under its parent 4
    path, _, _, margin, _ = run_typical(logits, parent, cand, 1.0, 0.0, 0.3)
    assert path == [0, 1, 3] and float(margin[5]) == -math.inf
    cand[3] = V                                 # out of range: rejected
    path, _, _, margin, _ = run_typical(logits, parent, cand, 1.0, 0.0, 0.3)
    assert path == [0, 2, 4] and float(margin[3]) == -math.inf


def test_typical_small_temperature_is_greedy_on_distinct_siblings():
    """As the temperature goes to 0 the tempered softmax puts all mass on the
    argmax: with logit gaps >= 0.01 and temperature 1e-3 the runner-up has
    p < e^-10, the argmax p > 1 - V e^-10 and H ~ 0, so the accepted edges
    are exactly those whose token is the parent's argmax.  With distinct
    siblings that is a single chain: the greedy walk."""
    g = torch.Generator().manual_seed(5)
    V = 40
    for seed in range(40):
        T = 2 + seed % 20
        parent = trees.random_tree(T, seed=seed, tag=3)
        logits = torch.stack([torch.randperm(V, generator=g).double() * 0.01 for _ in range(T)]).float()
        amax = logits.argmax(-1).tolist()
        cand = [0] * T
        for n in range(T):
            kids = [c for c in range(T) if parent[c] == n]
            toks = torch.randperm(V, generator=g)[:len(kids)].tolist()
            if kids and torch.rand(1, generator=g).item() < 0.7:
                j = int(torch.randint(len(kids), (1,), generator=g))
                if amax[n] in toks:
                    toks[toks.index(amax[n])] = toks[j]
                toks[j] = amax[n]
            for c, tok in zip(kids, toks):
                cand[c] = tok
        path, bonus, _, _, _ = run_typical(logits, parent, cand, 1e-3, 0.09, 0.3)
        gp, ga, gb = oracle.accept_walk(torch.tensor([parent]), torch.tensor([cand]), torch.tensor([amax]))
        assert path == gp[0, :int(ga[0])].tolist() and bonus == int(gb[0])


def test_typical_epsilon_monotone_and_rejects_bad_arguments():
    g = torch.Generator().manual_seed(9)
    T, V = 12, 64
    parent = trees.topk_tree(T, [3, 2, 2])
    logits = (torch.randn(T, V, generator=g) * 1.5).to(torch.bfloat16)
    top = logits.float().topk(3, -1).indices
    cand = [0] * T
    for n in range(T):                       # children take the parent's top tokens in sibling order
        for k, c in enumerate(c for c in range(T) if parent[c] == n):
            cand[c] = int(top[n, k])
    # delta = 10 keeps delta e^-H above eps, so theta = eps
    for delta in (10.0, 0.3):
        lens = [len(run_typical(logits, parent, cand, 1.0, eps, delta)[0])
                for eps in (0.0, 0.02, 0.05, 0.1, 0.2, 0.5)]
        assert lens == sorted(lens, reverse=True)
        assert delta != 10.0 or lens[0] == 4 > lens[-1]
    lg = logits.reshape(1, T, V)
    par, cd = torch.tensor([parent]), torch.tensor([cand])
    for tau, eps, delta in ((0.0, 0.1, 0.3), (-1.0, 0.1, 0.3), (math.nan, 0.1, 0.3), (math.inf, 0.1, 0.3),
                            (1.0, -0.1, 0.3), (1.0, math.nan, 0.3), (1.0, 0.1, -1.0), (1.0, 0.1, math.inf)):
        with pytest.raises(oracle.OracleError) as e:
            oracle.accept_typical(lg, par, cd, tau, eps, delta)
        assert e.value.code == oracle.BAD_ARG
    bad = torch.tensor([parent])
    bad[0, 3] = 5
    with pytest.raises(oracle.OracleError) as e:
        oracle.accept_typical(lg, bad, cd, 1.0, 0.1, 0.3)
    assert e.value.code == oracle.BAD_TREE


# ---------------------------------------------------------------------------
# A8: draft side (the Clover head's linear layers, embedding, top-k)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_linear_vs_library_matmul_and_silu(dtype):
    special = pytest.importorskip("scipy.special")
    g = torch.Generator().manual_seed(21)
    for R, N, K in ((1, 1, 1), (3, 7, 5), (8, 33, 64), (17, 9, 130)):
        x = torch.randn(R, K, generator=g).to(dtype)
        w = torch.randn(N, K, generator=g).to(dtype)
        res = torch.randn(R, N, generator=g).to(dtype)
        ref = (x.double().numpy() @ w.double().numpy().T)
        assert np.allclose(oracle.linear(x, w).numpy(), ref, rtol=1e-12, atol=1e-12)
        got = oracle.linear(x, w, res=res, act=1).numpy()
        assert np.allclose(got, res.double().numpy() + ref * special.expit(ref), rtol=1e-12, atol=1e-12)


def test_linear_identity_and_zero_weight():
    x = torch.randn(5, 16).bfloat16()
    res = torch.randn(5, 16).bfloat16()
    eye = torch.eye(16).bfloat16()
    assert torch.equal(oracle.linear(x, eye), x.double())
    assert torch.equal(oracle.linear(x, torch.zeros(16, 16).bfloat16(), res=res, act=1), res.double())
    with pytest.raises(oracle.OracleError):
        oracle.linear(x, eye, act=1)                  # the residual block needs its residual


def test_embed_rows_unit_norm_and_direction():
    g = torch.Generator().manual_seed(4)
    w = torch.randn(50, 24, generator=g).bfloat16()
    w[7] = 0
    toks = [3, 7, 49, 3, 0]
    e = oracle.embed_rows(w, toks)
    for r, t in enumerate(toks):
        row = w[t].double()
        if t == 7:
            assert (e[r] == 0).all()
            continue
        assert abs(e[r].norm().item() - 1.0) < 1e-12
        assert torch.allclose(e[r] * row.norm(), row, rtol=1e-12, atol=1e-12)
    # scaling a row does not change its embedding
    w2 = w.clone()
    w2[3] = (w[3].float() * 4).bfloat16()
    assert torch.allclose(oracle.embed_rows(w2, [3]), e[:1], rtol=1e-12, atol=1e-12)
    with pytest.raises(oracle.OracleError):
        oracle.embed_rows(w, [50])


def test_topk_vs_stable_sort_with_ties():
    g = torch.Generator().manual_seed(8)
    for R, V, k in ((1, 1, 1), (4, 10, 3), (3, 200, 8), (2, 64, 64)):
        x = torch.randint(-5, 6, (R, V), generator=g).double()     # many ties
        vals, idx = oracle.topk(x, k)
        for r in range(R):
            order = np.lexsort((np.arange(V), -x[r].numpy()))[:k]
            assert idx[r].tolist() == order.tolist()
            assert vals[r].tolist() == x[r, order].tolist()
    with pytest.raises(oracle.OracleError):
        oracle.topk(torch.zeros(1, 4), 5)


def test_head_step_special_cases():
    """W_v = 0: the decoder adds nothing; W_1 = 0 as well: the MLP block is the
    identity (silu(0) = 0), so the logits are the LM head of bf16(h).  The
    embedding ignores the scale of the LM-head rows."""
    g = torch.Generator().manual_seed(12)
    R, H, V, k = 3, 32, 300, 4
    bf = torch.bfloat16
    h = torch.randn(R, H, generator=g).to(bf)
    toks = torch.tensor([5, 77, 299], dtype=torch.int32)
    w_lm = torch.randn(V, H, generator=g).to(bf)
    z0 = torch.zeros(H, H, dtype=bf)
    w_o = torch.randn(H, H, generator=g).to(bf)
    out = oracle.clover_head_step(h, toks, w_lm, z0, w_o, z0, k)
    assert torch.equal(out["h"], h.double())
    assert torch.equal(out["z"], h.double())
    assert torch.equal(out["logits"], oracle.linear(h, w_lm))
    ref_v, ref_i = oracle.topk(out["logits"], k)
    assert torch.equal(out["top_indices"], ref_i)
    w_v = torch.randn(H, H, generator=g).to(bf)
    full = oracle.clover_head_step(h, toks, w_lm, w_v, w_o, z0, k)
    e = oracle.embed_rows(w_lm, toks)
    assert torch.allclose(full["attn"], oracle.linear(oracle.linear(e.to(bf), w_v).to(bf), w_o))
    assert torch.allclose(full["h"], h.double() + full["attn"])


def test_head_step_exact_hand_example():
    """A head step worked by hand (H = 2, V = 3, token 0).  The LM-head row
    (3, 4) has norm 5, so e = (0.6, 0.8); W_v = I gives v = e; W_o = [[1, 1],
    [0, 2]] gives (1.4, 1.6); with h = (0.5, -1), h' = (1.9, 0.6); W_1 =
    [[1, 0], [0, 0]] gives W_1 h' = (1.9, 0) and silu(1.9) = 1.9 / (1 +
    e^-1.9) = 1.652793898710304, silu(0) = 0, so z = (3.552793898710304, 0.6);
    the LM head rows (3, 4), (1, 0), (0, 2) give 3 z0 + 4 z1, z0 and 2 z1."""
    bf = torch.bfloat16
    w_lm = torch.tensor([[3.0, 4.0], [1.0, 0.0], [0.0, 2.0]]).to(bf)
    w_v = torch.eye(2).to(bf)
    w_o = torch.tensor([[1.0, 1.0], [0.0, 2.0]]).to(bf)
    w_1 = torch.tensor([[1.0, 0.0], [0.0, 0.0]]).to(bf)
    h = torch.tensor([[0.5, -1.0]]).to(bf)
    out = oracle.clover_head_step_exact(h, torch.tensor([0], dtype=torch.int32), w_lm, w_v, w_o, w_1, 2)
    close = lambda a, b: torch.allclose(a, torch.tensor([b], dtype=torch.float64), rtol=1e-14, atol=1e-14)
    assert close(out["e"], [0.6, 0.8])
    assert close(out["v"], [0.6, 0.8])
    assert close(out["attn"], [1.4, 1.6])
    assert close(out["h"], [1.9, 0.6])
    assert close(out["z"], [3.552793898710304, 0.6])
    assert close(out["logits"], [13.058381696130912, 3.552793898710304, 1.2])
    assert out["top_indices"].tolist() == [[0, 1]]


def test_head_step_exact_special_cases():
    """W_v = W_1 = 0: the step reduces to the LM head of h (the oracle's C
    linear layer, an independent fp64 sum)."""
    g = torch.Generator().manual_seed(21)
    R, H, V = 3, 48, 200
    bf = torch.bfloat16
    h = torch.randn(R, H, generator=g).to(bf)
    w_lm = torch.randn(V, H, generator=g).to(bf)
    z0 = torch.zeros(H, H, dtype=bf)
    w_o = torch.randn(H, H, generator=g).to(bf)
    out = oracle.clover_head_step_exact(h, torch.tensor([1, 2, 3], dtype=torch.int32), w_lm, z0, w_o, z0, 5)
    assert torch.equal(out["z"], h.double())
    assert torch.allclose(out["logits"], oracle.linear(h, w_lm), rtol=1e-13, atol=1e-13)


def test_head_step_bf16_reading_within_derived_bound():
    """The oracle's bf16-input reading of the head step stays within the
    worst-case rounding bound of tests/draft_bound.py of the exact step, the
    bound is small against the logits, and plausible mistakes (the residual
    dropped, W_o's sign flipped) break it."""
    from tests.draft_bound import head_step_bound
    g = torch.Generator().manual_seed(22)
    R, H, V, k = 4, 128, 600, 4
    bf = torch.bfloat16
    rnd = lambda *s, std=1.0: (torch.randn(*s, generator=g, dtype=torch.float64) * std).to(bf)
    h = rnd(R, H)
    w_lm = rnd(V, H, std=H ** -0.5)
    w_v, w_o, w_1 = (rnd(H, H, std=H ** -0.5) for _ in range(3))
    toks = torch.randint(0, V, (R,), generator=g, dtype=torch.int32)
    ex = oracle.clover_head_step_exact(h, toks, w_lm, w_v, w_o, w_1, k)
    rd = oracle.clover_head_step(h, toks, w_lm, w_v, w_o, w_1, k)
    E = head_step_bound(h, w_lm, w_v, w_o, w_1, ex)
    assert ((rd["logits"] - ex["logits"]).abs() <= E).all()
    assert E.max() < 0.25 * ex["logits"].abs().max()
    no_res = oracle.clover_head_step_exact(torch.zeros_like(h), toks, w_lm, w_v, w_o, w_1, k)
    assert ((no_res["logits"] - ex["logits"]).abs() > E).any()
    flip = oracle.clover_head_step_exact(h, toks, w_lm, w_v, (-w_o.double()).to(bf), w_1, k)
    assert ((flip["logits"] - ex["logits"]).abs() > E).any()
