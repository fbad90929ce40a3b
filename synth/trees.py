"""Seeded token-tree shapes (parent arrays).

A token tree with T nodes is given by ``parent[0..T-1]``: node 0 is the root
(``parent[0] == -1``) and every other node has ``0 <= parent[i] < i``, i.e. the
nodes are numbered in a topological order.  The paper merges the speculated
sequences by prefix into such a tree (Section 2.2, Tree Attention); it does not
give the shapes it used, so the shapes here follow a top-k style rule:

``topk_tree(T, branching)``: every rank tuple (r_1..r_k) with r_d < branching[d]
is a candidate continuation whose score is prod 1/(r_d + 1).  The T-1 best
tuples, ordered by (score descending, length ascending, tuple lexicographic),
become nodes 1..T-1 in that order, and the parent of a tuple is its prefix.
The prefix of a tuple has the same or a larger score and is shorter, so the
result is ancestor-closed and topologically numbered.
"""

from __future__ import annotations

import itertools
from fractions import Fraction

from . import rng


def topk_tree(T: int, branching: list[int]) -> list[int]:
    """Parent array of the T-node top-k style tree described in the module doc."""
    if T < 1:
        raise ValueError("T must be >= 1")
    cands = []
    for depth in range(1, len(branching) + 1):
        for ranks in itertools.product(*[range(b) for b in branching[:depth]]):
            score = Fraction(1)
            for r in ranks:
                score /= (r + 1)
            cands.append((-score, depth, ranks))
    cands.sort()
    if T - 1 > len(cands):
        raise ValueError(f"branching {branching} yields only {len(cands) + 1} nodes")
    chosen = [c[2] for c in cands[: T - 1]]
    index = {(): 0}
    parent = [-1]
    for k, ranks in enumerate(chosen, start=1):
        prefix = ranks[:-1]
        if prefix not in index:
            raise AssertionError("top-k rule produced a node before its parent")
        parent.append(index[prefix])
        index[ranks] = k
    return parent


def node_depths_of_topk(T: int, branching: list[int]) -> list[int]:
    """Depth of every node of ``topk_tree(T, branching)`` (tuple length; root 0)."""
    cands = []
    for depth in range(1, len(branching) + 1):
        for ranks in itertools.product(*[range(b) for b in branching[:depth]]):
            score = Fraction(1)
            for r in ranks:
                score /= (r + 1)
            cands.append((-score, depth, ranks))
    cands.sort()
    return [0] + [c[1] for c in cands[: T - 1]]


def chain_tree(T: int) -> list[int]:
    """A single speculated sequence: parent[i] = i - 1."""
    return [-1] + list(range(T - 1))


def star_tree(T: int) -> list[int]:
    """Every node is a child of the root."""
    return [-1] + [0] * (T - 1)


def random_tree(T: int, seed: int, tag: int = 0) -> list[int]:
    """Uniform random topologically numbered tree: parent[i] = floor(u_i * i)."""
    key = rng.derive_key(seed, 0x7EE0 + tag)
    parent = [-1]
    for i in range(1, T):
        u = (rng.splitmix64_scalar(key, i) >> 11) * 2.0 ** -53
        parent.append(min(i - 1, int(u * i)))
    return parent


def all_trees(T: int):
    """Every topologically numbered parent array with T nodes ((T-1)! of them)."""
    for choice in itertools.product(*[range(i) for i in range(1, T)]):
        yield [-1] + list(choice)
