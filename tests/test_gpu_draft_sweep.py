"""A seeded sweep of the draft side's entry points against the oracle: random
linear-layer shapes (rows from 0 to 600, so one or several launches of up to
256 rows; output features from 1 to 5000, tail tiles included; K from 64 to
4096 in steps of 64) in every epilogue, with and without the K-split
workspace, and random top-k shapes (V from 1 to 150,000, k from 1 to 32) with
planted ties, signed zeros and infinities.  Tolerances as in
tests/test_gpu_draft.py: the linear layer within a small multiple of the
absolute sum of its products (plus one bf16 rounding for the bf16 epilogues),
the top-k bit for bit."""

from __future__ import annotations

import random

import pytest
import torch

import oracle
import paper_2405_00263_gb300 as pkg
from tests.test_gpu_draft import BF, DEV, linear_tol, rand

pytestmark = pytest.mark.gpu

N_LINEAR = 60
N_TOPK = 40


def draw_linear(i: int):
    r = random.Random(31000 + i)
    R = r.choice([0, 1, 2, 15, 16, 17, 31, 32, 33, 100, 255, 256, 257, 600])
    N = r.choice([1, 7, 64, 127, 128, 129, 255, 384, 1000, 4097, 5000])
    K = 64 * r.choice([1, 2, 3, 5, 16, 33, 64])
    mode = r.choice(["f32", "bf16", "res_silu", "res"])
    return R, N, K, mode


@pytest.mark.parametrize("i", range(N_LINEAR), ids=[f"{i}-R{draw_linear(i)[0]}-N{draw_linear(i)[1]}-K{draw_linear(i)[2]}-"
                                                     f"{draw_linear(i)[3]}" for i in range(N_LINEAR)])
def test_linear_sweep(i):
    R, N, K, mode = draw_linear(i)
    g = torch.Generator().manual_seed(31000 + i)
    x = rand((R, K), g)
    w = rand((N, K), g, std=K ** -0.5)
    res = rand((R, N), g) if mode in ("res_silu", "res") else None
    if R == 0:                                               # no rows: nothing to compute, nothing reported
        out = torch.empty((0, N), dtype=torch.float32 if mode == "f32" else BF, device=DEV)
        st = torch.zeros(1, dtype=torch.int32, device=DEV)
        pkg.clover_linear(x.to(DEV), w.to(DEV), out, res=None if res is None else res.to(DEV), mode=mode, status=st)
        torch.cuda.synchronize()
        assert int(st.item()) == 0
        return
    if mode == "res":
        ref = oracle.linear(x, w) + res.double()
    else:
        ref = oracle.linear(x, w, res=res, act=1 if mode == "res_silu" else 0)
    tol = linear_tol(x, w, ref, mode != "f32")
    n_ws = pkg.clover_linear_workspace_size(R, N, K)
    for ws in (None, torch.zeros(max(16, n_ws), dtype=torch.uint8, device=DEV)):
        out = torch.full((R, N), float("nan"), dtype=torch.float32 if mode == "f32" else BF, device=DEV)
        st = torch.zeros(1, dtype=torch.int32, device=DEV)
        pkg.clover_linear(x.to(DEV), w.to(DEV), out, res=None if res is None else res.to(DEV), mode=mode,
                          workspace=ws, status=st)
        torch.cuda.synchronize()
        assert int(st.item()) == 0
        err = (out.cpu().double() - ref).abs()
        assert (err <= tol).all(), (err - tol).max().item()


def draw_topk(i: int):
    r = random.Random(47000 + i)
    V = r.choice([1, 2, 31, 32, 33, 1000, 4097, 16384, 16385, 50000, 125696, 150000])
    k = min(V, r.choice([1, 2, 5, 8, 10, 16, 31, 32]))
    R = r.choice([1, 2, 3, 16, 40])
    return R, V, k


@pytest.mark.parametrize("i", range(N_TOPK), ids=[f"{i}-R{draw_topk(i)[0]}-V{draw_topk(i)[1]}-k{draw_topk(i)[2]}"
                                                  for i in range(N_TOPK)])
def test_topk_sweep(i):
    R, V, k = draw_topk(i)
    g = torch.Generator().manual_seed(47000 + i)
    x = torch.randn(R, V, generator=g)
    r = random.Random(i)
    for row in range(R):
        if V > 1 and r.random() < 0.7:                       # ties at the top
            idx = torch.randperm(V, generator=g)[: min(V, r.randint(2, 40))]
            x[row, idx] = x[row].max() + r.choice([0.0, 1.0])
        if V > 10:
            x[row, r.randrange(V)] = -0.0
            x[row, r.randrange(V)] = 0.0
            x[row, r.randrange(V)] = -float("inf")
        if V > 10 and r.random() < 0.2:
            x[row, r.randrange(V)] = float("inf")
    vals, ind = oracle.topk(x, k)
    ws = torch.zeros(max(16, pkg.clover_topk_workspace_size(R, V, k)), dtype=torch.uint8, device=DEV)
    v = torch.empty((R, k), dtype=torch.float32, device=DEV)
    ix = torch.empty((R, k), dtype=torch.int32, device=DEV)
    pkg.clover_topk(x.to(DEV), k, v, ix, ws)
    torch.cuda.synchronize()
    assert torch.equal(ix.cpu(), ind)
    assert torch.equal(v.cpu().double(), vals)
