"""GPU parity of typical acceptance (clover_verify_accept_typical) with the oracle.

Every decision p(cand) > theta is an fp32 comparison on the GPU and an fp64 one
in the oracle.  The kernel's ln p - ln theta is within about 1e-4 of the exact
value (fp32 sums over up to 125,696 terms, base-2 exponent and logarithm
instructions), so both sides decide an edge alike whenever its exact margin is
larger than MARGIN.  Each case therefore first moves every candidate whose
oracle margin is below MARGIN to its parent's argmax token: the argmax has
p >= e^-H >= theta / delta, so that edge then passes by ln(1 / delta) or more.
The argmax, the path, its length and the bonus token must then be identical.
"""

from __future__ import annotations

import math
import random

import pytest
import torch

import oracle
import paper_2405_00263_gb300 as pkg
from synth import trees, workloads

pytestmark = pytest.mark.gpu

MARGIN = 5e-3          # nats


def peaked_logits(B, T, V, dtype, seed):
    """Normal logits with a per-row scale in {0.5, 1, 2, 4} plus, in half of
    the rows, a few boosted tokens (peaked rows with low entropy)."""
    g = torch.Generator().manual_seed(seed)
    x = torch.randn(B * T, V, generator=g, dtype=torch.float64)
    scales = torch.tensor([0.5, 1.0, 2.0, 4.0], dtype=torch.float64)
    x *= scales[torch.randint(4, (B * T, 1), generator=g)]
    for r in range(B * T):
        if torch.rand(1, generator=g).item() < 0.5:
            k = min(V, 1 + int(torch.randint(4, (1,), generator=g)))
            idx = torch.randperm(V, generator=g)[:k]
            x[r, idx] += torch.rand(k, generator=g, dtype=torch.float64) * 14.0
    return x.reshape(B, T, V).to(dtype)


def tree_and_cand(B, T, V, logits, kind, seed):
    """Parents (top-k style, random or chain trees) and candidates: each child takes
    a uniform token, or with probability 1/2 one of its parent's top-4 tokens."""
    g = torch.Generator().manual_seed(seed + 1)
    par = []
    for b in range(B):
        if kind == "random":
            par.append(trees.random_tree(T, seed=seed, tag=b))
        elif kind == "chain":
            par.append(trees.chain_tree(T))
        else:
            par.append(trees.topk_tree(T, [8, 4, 2, 2, 1]))
    top = logits.float().topk(min(4, V), -1).indices
    cand = torch.randint(V, (B, T), generator=g, dtype=torch.int32)
    for b in range(B):
        for c in range(1, T):
            if torch.rand(1, generator=g).item() < 0.5:
                cand[b, c] = top[b, par[b][c], int(torch.randint(top.shape[-1], (1,), generator=g))]
    return torch.tensor(par, dtype=torch.int32), cand


def clear_margins(logits, parent, cand, tau, eps, delta):
    r = oracle.accept_typical(logits, parent, cand, tau, eps, delta)
    near = r["margin"].abs() < MARGIN
    if near.any():
        cand = cand.clone()
        for b, c in near.nonzero().tolist():
            cand[b, c] = r["argmax"][b, parent[b, c]]
        r = oracle.accept_typical(logits, parent, cand, tau, eps, delta)
    assert not (r["margin"].abs() < MARGIN).any()
    return cand, r


def run_typical(logits, parent, cand, tau, eps, delta, ws=None, status=None):
    dev = torch.device("cuda")
    B, T, V = logits.shape
    lg, par, cd = logits.to(dev), parent.to(dev), cand.to(dev)
    am = torch.empty((B, T), dtype=torch.int32, device=dev)
    path = torch.empty((B, T), dtype=torch.int32, device=dev)
    alen = torch.empty(B, dtype=torch.int32, device=dev)
    bonus = torch.empty(B, dtype=torch.int32, device=dev)
    if ws is None:
        ws = torch.zeros(pkg.clover_verify_accept_typical_workspace_size(B, T, V, logits.dtype), dtype=torch.uint8,
                         device=dev)
    if status is None:
        status = torch.zeros(1, dtype=torch.int32, device=dev)
    pkg.clover_verify_accept_typical(lg, cd, par, tau, eps, delta, am, path, alen, bonus, ws, status)
    torch.cuda.synchronize()
    return {"argmax": am.cpu(), "path": path.cpu(), "accept_len": alen.cpu(), "bonus": bonus.cpu(),
            "status": int(status.item())}


def assert_same(got, ref):
    assert got["status"] == 0
    assert torch.equal(got["argmax"], ref["argmax"])
    assert torch.equal(got["accept_len"], ref["accept_len"])
    assert torch.equal(got["path"], ref["path"])
    assert torch.equal(got["bonus"], ref["bonus"])


CASES = [
    # B, T, V, dtype, tree, (tau, eps, delta)
    (2, 16, 1000, torch.bfloat16, "topk", (1.0, 0.09, 0.3)),
    (3, 64, 32000, torch.bfloat16, "topk", (0.7, 0.09, 0.3)),
    (1, 1, 17, torch.float32, "topk", (1.0, 0.09, 0.3)),
    (2, 7, 50257, torch.bfloat16, "random", (1.3, 0.2, 0.5)),      # odd V: unaligned rows, scalar heads/tails
    (2, 33, 16385, torch.bfloat16, "random", (2.0, 0.05, 0.2)),    # one element past a chunk
    (4, 9, 125696, torch.float32, "random", (0.5, 0.09, 0.3)),
    (1, 64, 1, torch.float32, "topk", (1.0, 0.09, 0.3)),           # V = 1: p = 1, H = 0
    (2, 24, 4099, torch.float32, "random", (1.0, 0.0, 0.3)),       # eps = 0: theta = 0
    (2, 24, 4099, torch.bfloat16, "random", (1.0, 0.3, 0.0)),      # delta = 0: theta = 0
    (2, 128, 20000, torch.bfloat16, "random", (1.0, 0.09, 0.3)),   # two mask words, two threads a row
    (1, 100, 9000, torch.float32, "topk", (0.8, 0.2, 0.5)),
    # root paths longer than the walk CTA's short walks (8 steps): the masks by pointer jumping
    (2, 40, 3000, torch.bfloat16, "chain", (1.0, 0.09, 0.3)),
    (1, 100, 3000, torch.bfloat16, "chain", (1.0, 0.0, 0.3)),    # theta = 0: the whole chain is accepted
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: f"B{c[0]}_T{c[1]}_V{c[2]}_{str(c[3])[6:]}_{c[5][0]}")
def test_typical_matches_oracle(case):
    B, T, V, dtype, kind, (tau, eps, delta) = case
    seed = B * 1000 + T * 10 + V % 97
    logits = peaked_logits(B, T, V, dtype, seed)
    parent, cand = tree_and_cand(B, T, V, logits, kind, seed)
    cand, ref = clear_margins(logits, parent, cand, tau, eps, delta)
    got = run_typical(logits, parent, cand, tau, eps, delta)
    assert_same(got, ref)
    if V > 1 and T > 1:
        # the cases decide edges both ways
        m = ref["margin"][:, 1:]
        assert (m > 0).any() and ((m < 0).any() or eps == 0.0 or delta == 0.0)


def test_typical_neg_inf_logits_and_out_of_range_candidates():
    B, T, V = 2, 20, 20000                  # fp32 chunks of 8192: row 3's first chunk is all -inf
    logits = peaked_logits(B, T, V, torch.float32, 77)
    parent, cand = tree_and_cand(B, T, V, logits, "random", 77)
    for b in range(B):
        for c in range(1, T, 3):
            logits[b, parent[b, c], cand[b, c]] = -math.inf      # p = 0: rejected even at theta = 0
        cand[b, 2] = V + 5
        cand[b, 4] = -3
        logits[b, 3, :V // 2] = -math.inf
    for tau, eps, delta in ((1.0, 0.0, 0.3), (0.8, 0.09, 0.3)):
        cd, ref = clear_margins(logits, parent, cand, tau, eps, delta)
        assert_same(run_typical(logits, parent, cd, tau, eps, delta), ref)


@pytest.mark.parametrize("name", ["paper_t4_b16", "7b_l4096", "100b_gqa", "7b_t128"])
def test_typical_full_size_workloads(name):
    w = workloads.get(name)
    t = workloads.make(w)
    logits, parent = t["logits"], t["parent"]
    for tau, eps, delta in ((1.0, 0.09, 0.3), (0.7, 0.3, 0.55)):
        cand, ref = clear_margins(logits, parent, t["cand"], tau, eps, delta)
        assert_same(run_typical(logits, parent, cand, tau, eps, delta), ref)


def test_typical_workspace_shared_with_greedy_and_reused():
    """Keys and counters reset themselves: greedy and typical calls alternate
    on one workspace and repeat with identical results."""
    dev = torch.device("cuda")
    B, T, V = 3, 32, 20000
    logits = peaked_logits(B, T, V, torch.bfloat16, 5)
    parent, cand = tree_and_cand(B, T, V, logits, "random", 5)
    cand, ref = clear_margins(logits, parent, cand, 1.0, 0.09, 0.3)
    ws = torch.zeros(pkg.clover_verify_accept_typical_workspace_size(B, T, V, torch.bfloat16), dtype=torch.uint8,
                     device=dev)
    amax = oracle.argmax(logits)
    gpath, glen, gbonus = oracle.accept_walk(parent, cand, amax)
    lg, par, cd = logits.to(dev), parent.to(dev), cand.to(dev)
    for _ in range(3):
        assert_same(run_typical(logits, parent, cand, 1.0, 0.09, 0.3, ws=ws), ref)
        am = torch.empty((B, T), dtype=torch.int32, device=dev)
        path = torch.empty((B, T), dtype=torch.int32, device=dev)
        alen = torch.empty(B, dtype=torch.int32, device=dev)
        bonus = torch.empty(B, dtype=torch.int32, device=dev)
        pkg.clover_verify_accept(lg, cd, par, am, path, alen, bonus, ws)
        torch.cuda.synchronize()
        assert torch.equal(path.cpu(), gpath) and torch.equal(alen.cpu(), glen) and torch.equal(bonus.cpu(), gbonus)


def test_typical_bad_tree_sets_status():
    B, T, V = 2, 8, 512
    logits = peaked_logits(B, T, V, torch.float32, 3)
    parent, cand = tree_and_cand(B, T, V, logits, "random", 3)
    parent[1, 5] = 6
    got = run_typical(logits, parent, cand, 1.0, 0.09, 0.3)
    assert got["status"] & 4                   # CLOVER_ERR_BAD_TREE
    assert int(got["accept_len"][1]) == 1 and int(got["path"][1, 0]) == 0


@pytest.mark.parametrize("schedule", ["commit", "compact", "fused"])
@pytest.mark.parametrize("name,over,params", [
    ("tiny_f32", {}, (1.0, 0.09, 0.3)),
    ("7b_l2048", dict(B=2, T=64, Hq=8, Hkv=2, L=700, V=5003), (0.8, 0.09, 0.3)),
    ("paper_t4_b4", dict(Hq=8, Hkv=8, L_range=(100, 900), V=32000), (1.0, 0.3, 0.55)),
])
def test_typical_verify_step_matches_oracle(name, over, params, schedule):
    """The whole step (attention, typical acceptance, commit or compaction)
    through VerifyStep against the oracle's step with the same rule."""
    from tests.gpu_util import compare_full, run_gpu, to_dev
    host = workloads.make(workloads.get(name, **over))
    host["cand"], _ = clear_margins(host["logits"], host["parent"], host["cand"], *params)
    t = to_dev(host, torch.device("cuda"))
    tau, eps, delta = params
    step = run_gpu(t, schedule=schedule, accept="typical", temperature=tau, epsilon=eps, delta=delta)
    compare_full(host, step, t)


def draw_typical(i: int):
    r = random.Random(53000 + i)
    B = r.choice([1, 2, 3, 5])
    T = r.choice([1, 2, 9, 16, 33, 64, 65, 100, 128])
    V = r.choice([1, 2, 100, 1000, 4099, 16384, 16385, 50257, 125696])
    dtype = r.choice([torch.bfloat16, torch.bfloat16, torch.float32])
    kind = r.choice(["topk", "random", "chain"])
    tau = r.choice([0.3, 0.7, 1.0, 1.5, 3.0])
    eps = r.choice([0.0, 0.01, 0.09, 0.3, 0.9])
    delta = r.choice([0.0, 0.1, 0.3, 0.6, 1.0])
    return B, T, V, dtype, kind, (tau, eps, delta)


N_SWEEP = 60


@pytest.mark.parametrize("i", range(N_SWEEP))
def test_typical_sweep(i):
    """Seeded random shapes, trees and (temperature, epsilon, delta), with
    candidates moved off the threshold's neighbourhood as above."""
    B, T, V, dtype, kind, (tau, eps, delta) = draw_typical(i)
    seed = 53000 + i
    logits = peaked_logits(B, T, V, dtype, seed)
    parent, cand = tree_and_cand(B, T, V, logits, kind, seed)
    cand, ref = clear_margins(logits, parent, cand, tau, eps, delta)
    assert_same(run_typical(logits, parent, cand, tau, eps, delta), ref)
