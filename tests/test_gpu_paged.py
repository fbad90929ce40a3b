"""GPU parity of the paged KV cache (clover_verify_attn_paged, clover_kv_commit_paged).

The cache layout changes nothing in what is computed.  With the same logical
capacity (hence the same split plan) the paged attention reads the same keys in
the same tiles as the dense one, so its output must equal the dense call's bit
for bit; the dense call is itself pinned to the oracle (test_gpu_parity.py), and
a few rows are checked against the oracle here as well.  The paged commit must
leave, in the dense view of the pool, the bytes the dense commit leaves.  Pages
that no table names hold NaN, and table entries past each sequence's slots are
-1, so a read of either shows up.
"""

from __future__ import annotations


import pytest
import torch

import oracle
import paper_2405_00263_gb300 as pkg
from synth import paging, workloads
from tests.gpu_util import ATOL

pytestmark = pytest.mark.gpu


def paged_case(host, page_size, seed):
    """Dense caches padded to a capacity that is a multiple of 256 slots and of
    the page size, and their pools under a seeded table that gives each
    sequence L + T slots."""
    B, Hkv, Lcap, D = host["k_cache"].shape
    T = host["k_new"].shape[1]
    unit = max(256, page_size)
    cap = -(-Lcap // unit) * unit
    pad = torch.full((B, Hkv, cap - Lcap, D), float("nan"), dtype=host["k_cache"].dtype)
    kc = torch.cat([host["k_cache"], pad], 2)
    vc = torch.cat([host["v_cache"], pad], 2)
    need = [int(L) + T for L in host["cache_len"]]
    table, n_pages = paging.page_table(need, page_size, cap // page_size, seed)
    return {"k_dense": kc, "v_dense": vc, "cap": cap, "table": table, "n_pages": n_pages,
            "k_pool": paging.to_pages(kc, table, page_size, n_pages),
            "v_pool": paging.to_pages(vc, table, page_size, n_pages)}


def run_both(host, pc, page_size, dev):
    """(dense output, paged output, dense status, paged status)."""
    q, kn, vn = (host[k].to(dev) for k in ("q", "k_new", "v_new"))
    cl, par = host["cache_len"].to(dev), host["parent"].to(dev)
    B, T, Hq, D = q.shape
    Hkv = kn.shape[2]
    dt = q.dtype
    st_d = torch.zeros(1, dtype=torch.int32, device=dev)
    st_p = torch.zeros(1, dtype=torch.int32, device=dev)
    out_d = torch.empty_like(q)
    out_p = torch.empty_like(q)
    n_ws = pkg.clover_verify_attn_workspace_size(B, T, Hq, Hkv, D, pc["cap"], dt)
    ws = torch.zeros(max(16, n_ws), dtype=torch.uint8, device=dev) if n_ws else None
    pkg.clover_verify_attn(q, kn, vn, pc["k_dense"].to(dev), pc["v_dense"].to(dev), cl, par, out_d, workspace=ws,
                           status=st_d, append=False)
    max_pages = pc["table"].shape[1]
    assert pkg.clover_verify_attn_paged_workspace_size(B, T, Hq, Hkv, D, page_size, max_pages, dt) == n_ws
    pkg.clover_verify_attn_paged(q, kn, vn, pc["k_pool"].to(dev), pc["v_pool"].to(dev), pc["table"].to(dev), cl,
                                 par, out_p, workspace=ws, status=st_p)
    torch.cuda.synchronize()
    return out_d.cpu(), out_p.cpu(), int(st_d.item()), int(st_p.item())


def check_rows_against_oracle(host, out, n=24):
    B, T, Hq, D = host["q"].shape
    g = torch.Generator().manual_seed(1)
    rows = sorted(set([0, B * T * Hq - 1] + torch.randint(0, B * T * Hq, (n,), generator=g).tolist()))
    ref = oracle.tree_attention(host["q"], host["k_new"], host["v_new"], host["k_cache"], host["v_cache"],
                                host["cache_len"], host["parent"], rows=rows)
    err = (out.view(-1, D)[rows].double() - ref).abs().max().item()
    assert err <= ATOL[host["q"].dtype], err


CASES = [
    # workload, overrides, page sizes
    ("7b_l2048", dict(B=3, T=16, Hq=8, Hkv=4, L=1200, L_range=(1, 1200), V=2048, branching=(4, 2, 1, 1)),
     (16, 64, 128, 256)),
    ("7b_l2048", dict(B=2, T=100, Hq=4, Hkv=2, D=64, L=700, L_range=(300, 700), V=2048, tree="random"), (32, 512)),
    ("tiny_f32", dict(B=2, D=128, Hq=4, Hkv=2, L=900, L_range=(0, 900), V=1024), (16, 128)),
]


@pytest.mark.parametrize("name,over,sizes", CASES, ids=["bf16_gqa", "bf16_T100_d64", "f32"])
def test_paged_attention_equals_dense(name, over, sizes):
    host = workloads.make(workloads.get(name, **over))
    dev = torch.device("cuda")
    for i, ps in enumerate(sizes):
        pc = paged_case(host, ps, seed=10 + i)
        out_d, out_p, st_d, st_p = run_both(host, pc, ps, dev)
        assert st_d == 0 and st_p == 0
        assert torch.equal(out_p.view(torch.int16 if out_p.dtype == torch.bfloat16 else torch.int32),
                           out_d.view(torch.int16 if out_d.dtype == torch.bfloat16 else torch.int32)), ps
        if i == 0:
            check_rows_against_oracle(host, out_p)


@pytest.mark.parametrize("name", ["7b_l4096", "paper_t4_b16"])
def test_paged_attention_full_size(name):
    host = workloads.make(workloads.get(name))
    pc = paged_case(host, 64, seed=3)
    out_d, out_p, st_d, st_p = run_both(host, pc, 64, torch.device("cuda"))
    assert st_d == 0 and st_p == 0
    assert torch.equal(out_p.view(torch.int16), out_d.view(torch.int16))
    check_rows_against_oracle(host, out_p)


@pytest.mark.parametrize("ps", [16, 128])
def test_paged_commit_equals_dense_commit(ps):
    w = workloads.get("7b_l2048", B=3, T=32, Hq=4, Hkv=4, L=500, L_range=(0, 500), V=3000, branching=(4, 2, 2, 1))
    host = workloads.make(w)
    pc = paged_case(host, ps, seed=7)
    dev = torch.device("cuda")
    amax = oracle.argmax(host["logits"])
    path, alen, _ = oracle.accept_walk(host["parent"], host["cand"], amax)
    i32 = dict(dtype=torch.int32, device=dev)
    kn, vn = host["k_new"].to(dev), host["v_new"].to(dev)
    cl, p_, a_ = host["cache_len"].to(dev), path.to(dev), alen.to(dev)
    kd, vd = pc["k_dense"].to(dev), pc["v_dense"].to(dev)
    ncl_d, src_d = torch.empty(w.B, **i32), torch.empty((w.B, w.T), **i32)
    pkg.clover_kv_commit(kd, vd, kn, vn, cl, p_, a_, ncl_d, src_d)
    kp, vp = pc["k_pool"].to(dev), pc["v_pool"].to(dev)
    ncl_p, src_p = torch.empty(w.B, **i32), torch.empty((w.B, w.T), **i32)
    st = torch.zeros(1, **i32)
    pkg.clover_kv_commit_paged(kp, vp, pc["table"].to(dev), kn, vn, cl, p_, a_, ncl_p, src_p, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert torch.equal(ncl_p, ncl_d) and torch.equal(src_p, src_d)
    kview = paging.from_pages(kp.cpu(), pc["table"], ps, pc["cap"])
    vview = paging.from_pages(vp.cpu(), pc["table"], ps, pc["cap"])
    for b in range(w.B):
        m = int(ncl_d[b])
        assert torch.equal(kview[b, :, :m].view(torch.int16), kd[b, :, :m].cpu().view(torch.int16))
        assert torch.equal(vview[b, :, :m].view(torch.int16), vd[b, :, :m].cpu().view(torch.int16))
    owned = set(int(x) for x in pc["table"].flatten() if x >= 0)
    spare = [p for p in range(pc["n_pages"]) if p not in owned]
    assert torch.isnan(kp[spare].float()).all() and torch.isnan(vp[spare].float()).all()


def test_paged_invalid_page_ids_report_status():
    """A table entry outside [0, n_pages) for a slot that is read (attention) or
    written (commit) raises CLOVER_ERR_INVALID_ARG; the access goes to page 0."""
    w = workloads.get("7b_l2048", B=2, T=8, Hq=2, Hkv=2, L=300, V=1000, branching=(2, 2, 1))
    host = workloads.make(w)
    dev = torch.device("cuda")
    pc = paged_case(host, 64, seed=5)
    pc["table"][1, 2] = pc["n_pages"] + 7                  # slot 128 of sequence 1 (L = 300)
    _, _, _, st_p = run_both(host, pc, 64, dev)
    assert st_p & 1
    pc = paged_case(host, 64, seed=5)
    pc["table"][0, 4] = -5                                # slot 300 = L + 0 of sequence 0: a commit target
    i32 = dict(dtype=torch.int32, device=dev)
    st = torch.zeros(1, **i32)
    path = torch.zeros((w.B, w.T), **i32)
    alen = torch.ones(w.B, **i32)
    pkg.clover_kv_commit_paged(pc["k_pool"].to(dev), pc["v_pool"].to(dev), pc["table"].to(dev),
                               host["k_new"].to(dev), host["v_new"].to(dev), host["cache_len"].to(dev), path, alen,
                               torch.empty(w.B, **i32), status=st)
    torch.cuda.synchronize()
    assert int(st.item()) & 1


def fused_pair(host, pc, ps, dev, **step_kw):
    """The fused step on the dense padded caches and on the pools: (dense
    step, paged step, dense K/V caches, K/V pools) after one run each."""
    B, T, Hq, D = host["q"].shape
    Hkv = host["k_new"].shape[2]
    V = host["logits"].shape[-1]
    dt = host["q"].dtype
    t = {k: host[k].to(dev) for k in ("q", "k_new", "v_new", "cache_len", "parent", "cand", "logits")}
    args = (t["q"], t["k_new"], t["v_new"])
    tail = (t["cache_len"], t["parent"], t["cand"], t["logits"])
    dense = pkg.VerifyStep(B, T, Hq, Hkv, D, pc["cap"], V, dt, device=dev, schedule="fused", **step_kw)
    paged = pkg.VerifyStep(B, T, Hq, Hkv, D, pc["cap"], V, dt, device=dev, schedule="fused", page_size=ps,
                           **step_kw)
    kd, vd = pc["k_dense"].to(dev), pc["v_dense"].to(dev)
    kp, vp = pc["k_pool"].to(dev), pc["v_pool"].to(dev)
    dense.run(*args, kd, vd, *tail)
    paged.run(*args, kp, vp, *tail, block_table=pc["table"].to(dev))
    torch.cuda.synchronize()
    return dense, paged, (kd.cpu(), vd.cpu()), (kp.cpu(), vp.cpu())


def check_pair(pc, ps, dense, paged, dense_kv, pools):
    """The paged step equals the dense one bit for bit: outputs, indices and
    the committed prefix in the dense view of the pools; unowned pages keep
    their NaN."""
    assert dense.device_status() == 0 and paged.device_status() == 0
    iview = torch.int16 if dense.out.dtype == torch.bfloat16 else torch.int32
    assert torch.equal(paged.out.view(iview), dense.out.view(iview))
    for name in ("argmax", "path", "accept_len", "bonus", "src_index", "new_cache_len"):
        assert torch.equal(getattr(paged, name), getattr(dense, name)), name
    for pool, kd in zip(pools, dense_kv):
        view = paging.from_pages(pool, pc["table"], ps, pc["cap"])
        for b in range(kd.shape[0]):
            m = int(dense.new_cache_len[b])
            assert torch.equal(view[b, :, :m].view(iview), kd[b, :, :m].view(iview))
        owned = set(int(x) for x in pc["table"].flatten() if x >= 0)
        spare = [p for p in range(pc["n_pages"]) if p not in owned]
        assert torch.isnan(pool[spare].float()).all()


@pytest.mark.parametrize("launch", ["ordinary", "pdl", "cache_ready", "inputs_ready"])
@pytest.mark.parametrize("accept", ["greedy", "typical"])
def test_paged_fused_step_equals_dense(launch, accept):
    """The fused schedule on a paged cache (clover_verify_attn_paged_ex, then
    clover_verify_accept_paged_ex with the commit into the pools) in every
    attention launch mode: bit-equal to the dense fused step, whose accept
    outputs are checked against the oracle here too."""
    w = workloads.get("7b_l2048", B=3, T=32, Hq=8, Hkv=4, L=900, L_range=(1, 900), V=3001, branching=(4, 2, 2, 1))
    host = workloads.make(w)
    dev = torch.device("cuda")
    ps = 16 if launch in ("ordinary", "inputs_ready") else 64
    pc = paged_case(host, ps, seed=21)
    dense, paged, dense_kv, pools = fused_pair(host, pc, ps, dev, accept=accept, attn_launch=launch)
    check_pair(pc, ps, dense, paged, dense_kv, pools)
    ref = oracle.verify_step(host, typical=paged.typical if accept == "typical" else None)
    for name in ("argmax", "path", "accept_len", "bonus"):
        assert torch.equal(getattr(paged, name).cpu(), ref[name]), name
    assert torch.equal(paged.new_cache_len.cpu(), ref["cache_len"])
    err = (paged.out.double().cpu() - ref["out"]).abs().max().item()
    assert err <= ATOL[torch.bfloat16], err


def test_paged_fused_step_grouped_query_rows():
    """A grouped-query shape with four 128-row tiles a head, inputs-ready: the
    dense step runs two row tiles per CTA (tree_attn_tc_pair.cu), the paged
    one a row tile per CTA with one key range (tree_attn_tc.cu); the two
    kernels compute every row the same way, so the steps agree bit for bit."""
    w = workloads.get("100b_gqa", B=2, Hq=32, Hkv=4, L=900, L_range=(300, 900), V=2048)
    host = workloads.make(w)
    pc = paged_case(host, 16, seed=8)
    dense, paged, dense_kv, pools = fused_pair(host, pc, 16, torch.device("cuda"), attn_launch="inputs_ready")
    check_pair(pc, 16, dense, paged, dense_kv, pools)
    check_rows_against_oracle(host, paged.out.cpu())


@pytest.mark.parametrize("name,ps", [("7b_l4096", 16), ("paper_t4_b16", 64)])
def test_paged_fused_step_full_size(name, ps):
    """The bench's paged step at full size (inputs-ready attention, fused
    accept + commit): bit-equal to the dense step, attention rows sampled
    against the oracle."""
    host = workloads.make(workloads.get(name))
    pc = paged_case(host, ps, seed=4)
    dense, paged, dense_kv, pools = fused_pair(host, pc, ps, torch.device("cuda"), attn_launch="inputs_ready")
    check_pair(pc, ps, dense, paged, dense_kv, pools)
    check_rows_against_oracle(host, paged.out.cpu())


def test_paged_fused_invalid_page_id_reports_status():
    """A bad table entry for a slot the fused commit writes raises
    CLOVER_ERR_INVALID_ARG in the accept call's status; the row is skipped."""
    w = workloads.get("7b_l2048", B=2, T=8, Hq=2, Hkv=2, L=256, V=1000, branching=(2, 2, 1))
    host = workloads.make(w)
    pc = paged_case(host, 64, seed=5)
    pc["table"][0, 4] = -5                                # slot 256 = L + 0 of sequence 0 (no slot < L on it)
    dev = torch.device("cuda")
    _, paged, _, _ = fused_pair(host, pc, 64, dev)
    assert int(paged.status.item()) == 0
    assert int(paged.status_accept.item()) & 1
