"""Seeded synthetic verification-step inputs.

The paper measures on internal Baichuan models and datasets (Section 4.1) that
are not available; these tensors stand in for them with the shapes of a 7B-class
and a 100B-class model and the value distributions listed per workload below.

Layouts (row-major, matching the C ABI):
  q        [B, T, Hq,  D]      k_new, v_new [B, T, Hkv, D]
  k_cache  [B, Hkv, Lcap, D]   v_cache      [B, Hkv, Lcap, D]
  cache_len[B] int32           parent, cand [B, T] int32
  logits   [B, T, V]

Cache slots at and past ``cache_len[b]`` hold NaN, so that any read of an
uncommitted slot shows up in the results.

Candidate ids: the root holds a random token; the children of every node get
distinct uniform ids.  With probability ``plant_p`` per node that has children,
one child chosen uniformly is made to match: the parent's logit row gets the
value ``PLANT`` at that child's id.  ``PLANT`` exceeds every Box-Muller draw
(|z| < 8.6 for 53-bit uniforms, times ``logit_std``), so it is then the row's
unique maximum.  No argmax is computed here.
"""

from __future__ import annotations

import math
from dataclasses import dataclass, field, replace

import torch

from . import rng, trees

PLANT = 64.0

_TAG = {"q": 1, "k_new": 2, "v_new": 3, "k_cache": 4, "v_cache": 5, "logits": 6,
        "cand": 7, "plant": 8, "plant_pick": 9, "len": 10, "root": 11}


@dataclass(frozen=True)
class Workload:
    name: str
    B: int
    T: int
    Hq: int
    Hkv: int
    D: int
    L: int                      # cache length (all sequences) when L_range is None
    V: int
    dtype: str                  # "f32" or "bf16"
    branching: tuple = ()
    plant_p: float = 0.5
    qkv_std: float = 1.0
    logit_std: float = 4.0
    seed: int = 0
    L_range: tuple | None = None  # (lo, hi) inclusive: per-sequence lengths ~ U[lo, hi]
    tree: str = "topk"          # "topk", "chain", "star", "random"
    description: str = ""

    @property
    def torch_dtype(self):
        return torch.float32 if self.dtype == "f32" else torch.bfloat16

    @property
    def elem_bytes(self) -> int:
        return 4 if self.dtype == "f32" else 2


WORKLOADS = {
    "tiny_f32": Workload(
        "tiny_f32", B=1, T=16, Hq=8, Hkv=8, D=64, L=128, V=1024, dtype="f32",
        branching=(4, 2, 1, 1), plant_p=0.6, qkv_std=1.0, logit_std=4.0, seed=0,
        description="B1, 8 heads MHA, D64, L128, 16-node tree [4,2,1,1], V1024, fp32"),
    "7b_l2048": Workload(
        "7b_l2048", B=1, T=64, Hq=32, Hkv=32, D=128, L=2048, V=125696, dtype="bf16",
        branching=(8, 4, 2, 2, 1), plant_p=0.5, qkv_std=1 / math.sqrt(128), seed=1,
        description="7B-class: B1, 32 heads MHA, D128, L2048, 64-node tree depth 5, V125696, bf16"),
    "7b_l4096": Workload(
        "7b_l4096", B=1, T=64, Hq=32, Hkv=32, D=128, L=4096, V=125696, dtype="bf16",
        branching=(8, 4, 2, 2, 1), plant_p=0.5, qkv_std=1 / math.sqrt(128), seed=2,
        description="7B-class: B1, 32 heads MHA, D128, L4096, 64-node tree depth 5, V125696, bf16"),
    "7b_l16384": Workload(
        "7b_l16384", B=1, T=64, Hq=32, Hkv=32, D=128, L=16384, V=125696, dtype="bf16",
        branching=(8, 4, 2, 2, 1), plant_p=0.5, qkv_std=1 / math.sqrt(128), seed=2,
        description="7B-class: B1, 32 heads MHA, D128, L16384, 64-node tree depth 5, V125696, bf16"),
    "7b_batched": Workload(
        "7b_batched", B=16, T=32, Hq=32, Hkv=32, D=128, L=8192, V=125696, dtype="bf16",
        branching=(8, 4, 2, 1), plant_p=0.5, qkv_std=1 / math.sqrt(128), seed=3,
        L_range=(512, 8192),
        description="7B-class batched: B16, L_b ~ U[512,8192], 32 heads MHA, D128, "
                    "32-node tree depth 4, V125696, bf16"),
    # the paper's own serving regime (tree size 4, batch 4-48, 7B MHA shapes, L around 2k)
    "paper_t4_b4": Workload(
        "paper_t4_b4", B=4, T=4, Hq=32, Hkv=32, D=128, L=2560, V=125696, dtype="bf16",
        branching=(2, 1), plant_p=0.5, qkv_std=1 / math.sqrt(128), seed=5, L_range=(1536, 2560),
        description="paper regime: B4, L_b ~ U[1536,2560], 32 heads MHA, D128, 4-node tree, V125696, bf16"),
    "paper_t4_b16": Workload(
        "paper_t4_b16", B=16, T=4, Hq=32, Hkv=32, D=128, L=2560, V=125696, dtype="bf16",
        branching=(2, 1), plant_p=0.5, qkv_std=1 / math.sqrt(128), seed=6, L_range=(1536, 2560),
        description="paper regime: B16, L_b ~ U[1536,2560], 32 heads MHA, D128, 4-node tree, V125696, bf16"),
    "paper_t4_b48": Workload(
        "paper_t4_b48", B=48, T=4, Hq=32, Hkv=32, D=128, L=2560, V=125696, dtype="bf16",
        branching=(2, 1), plant_p=0.5, qkv_std=1 / math.sqrt(128), seed=7, L_range=(1536, 2560),
        description="paper regime: B48, L_b ~ U[1536,2560], 32 heads MHA, D128, 4-node tree, V125696, bf16"),
    # a larger tree (the tree-size sweep of the paper's appendix), 7B MHA shapes
    "7b_t128": Workload(
        "7b_t128", B=1, T=128, Hq=32, Hkv=32, D=128, L=4096, V=125696, dtype="bf16",
        branching=(8, 4, 2, 2, 2, 1), plant_p=0.5, qkv_std=1 / math.sqrt(128), seed=8,
        description="7B-class, larger tree: B1, 32 heads MHA, D128, L4096, 128-node tree depth 6, V125696, bf16"),
    "100b_gqa": Workload(
        "100b_gqa", B=4, T=64, Hq=64, Hkv=8, D=128, L=8192, V=125696, dtype="bf16",
        branching=(8, 4, 2, 2, 1), plant_p=0.5, qkv_std=1 / math.sqrt(128), seed=4,
        description="100B-class GQA: B4, 64 q heads / 8 KV heads, D128, L8192, "
                    "64-node tree depth 5, V125696, bf16"),
}


def get(name: str, **overrides) -> Workload:
    w = WORKLOADS[name]
    return replace(w, **overrides) if overrides else w


def cache_lengths(w: Workload) -> list[int]:
    if w.L_range is None:
        return [w.L] * w.B
    lo, hi = w.L_range
    key = rng.derive_key(w.seed, _TAG["len"])
    return [lo + int(v) for v in rng.below(key, w.B, hi - lo + 1).tolist()]


def lcap(w: Workload) -> int:
    need = max(cache_lengths(w)) + w.T
    return ((need + 63) // 64) * 64


def parents(w: Workload) -> list[list[int]]:
    """Parent array of every sequence (all sequences share the shape unless random)."""
    out = []
    for b in range(w.B):
        if w.tree == "topk":
            out.append(trees.topk_tree(w.T, list(w.branching)))
        elif w.tree == "chain":
            out.append(trees.chain_tree(w.T))
        elif w.tree == "star":
            out.append(trees.star_tree(w.T))
        elif w.tree == "random":
            out.append(trees.random_tree(w.T, w.seed, tag=b))
        else:
            raise ValueError(w.tree)
    return out


def _normal_tensor(w: Workload, tag: str, shape, std: float, device) -> torch.Tensor:
    n = math.prod(shape)
    x = rng.normal(rng.derive_key(w.seed, _TAG[tag]), n, device=device)
    if std != 1.0:
        x = x * std
    return rng.round_to(x, w.torch_dtype).reshape(shape)


def candidates(w: Workload, par: list[list[int]]):
    """cand [B,T] (distinct ids among siblings) and the planted (b, node, id) list."""
    key_c = rng.derive_key(w.seed, _TAG["cand"])
    key_r = rng.derive_key(w.seed, _TAG["root"])
    key_p = rng.derive_key(w.seed, _TAG["plant"])
    key_k = rng.derive_key(w.seed, _TAG["plant_pick"])
    cand = [[0] * w.T for _ in range(w.B)]
    plants = []
    for b in range(w.B):
        p = par[b]
        cand[b][0] = int(rng.splitmix64_scalar(key_r, b) % w.V)
        children = [[] for _ in range(w.T)]
        for i in range(1, w.T):
            children[p[i]].append(i)
        for node in range(w.T):
            used = set()
            for c in children[node]:
                attempt = 0
                while True:
                    z = rng.splitmix64_scalar(key_c, (b * w.T + c) * 64 + attempt)
                    tok = int(((z >> 11) * 2.0 ** -53) * w.V)
                    attempt += 1
                    if tok not in used:
                        break
                used.add(tok)
                cand[b][c] = tok
            if children[node]:
                u = (rng.splitmix64_scalar(key_p, b * w.T + node) >> 11) * 2.0 ** -53
                if u < w.plant_p:
                    u2 = (rng.splitmix64_scalar(key_k, b * w.T + node) >> 11) * 2.0 ** -53
                    pick = children[node][min(len(children[node]) - 1, int(u2 * len(children[node])))]
                    plants.append((b, node, cand[b][pick]))
    return cand, plants


def make(w: Workload, device="cpu", logits: bool = True) -> dict:
    """All inputs of one verification step for workload ``w`` on ``device``."""
    L = cache_lengths(w)
    cap = lcap(w)
    par = parents(w)
    cand, plants = candidates(w, par)
    t = {}
    t["q"] = _normal_tensor(w, "q", (w.B, w.T, w.Hq, w.D), w.qkv_std, device)
    t["k_new"] = _normal_tensor(w, "k_new", (w.B, w.T, w.Hkv, w.D), w.qkv_std, device)
    t["v_new"] = _normal_tensor(w, "v_new", (w.B, w.T, w.Hkv, w.D), w.qkv_std, device)
    for name in ("k_cache", "v_cache"):
        c = _normal_tensor(w, name, (w.B, w.Hkv, cap, w.D), w.qkv_std, device)
        for b in range(w.B):
            c[b, :, L[b]:, :] = float("nan")
        t[name] = c
    t["cache_len"] = torch.tensor(L, dtype=torch.int32, device=device)
    t["parent"] = torch.tensor(par, dtype=torch.int32, device=device)
    t["cand"] = torch.tensor(cand, dtype=torch.int32, device=device)
    if logits:
        lg = _normal_tensor(w, "logits", (w.B, w.T, w.V), w.logit_std, device)
        for b, node, tok in plants:
            lg[b, node, tok] = PLANT
        t["logits"] = lg
    t["Lcap"] = cap
    t["plants"] = plants
    return t
