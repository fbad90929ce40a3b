"""Seeded paged layouts of a dense KV cache (input construction only).

A paged cache stores each sequence's slots in fixed-size pages of a shared pool
``[n_pages, Hkv, page_size, D]``; ``block_table[b][k]`` is the pool page that
holds slots ``[k * page_size, (k + 1) * page_size)`` of sequence b.  Here every
sequence gets the pages for ``need[b]`` slots, drawn from a seeded random
permutation of the pool (so neighbouring slots of one sequence are scattered
over the pool), and the table entries past them are -1.  The pool also has
``n_spare`` pages that no table names, filled with NaN, so that a read of a
page nobody owns shows up in the results.
"""

from __future__ import annotations

import math

import torch

from . import rng

_TAG_PERM = 21


def page_table(need, page_size: int, max_pages: int, seed: int, n_spare: int = 3):
    """(block_table [B, max_pages] int32, n_pages): sequence b owns the pages of
    its first ceil(need[b] / page_size) table entries."""
    owned = [math.ceil(n / page_size) for n in need]
    if max(owned, default=0) > max_pages:
        raise ValueError("max_pages too small for the requested slots")
    n_pages = sum(owned) + n_spare
    key = rng.derive_key(seed, _TAG_PERM)
    order = sorted(range(n_pages), key=lambda i: rng.splitmix64_scalar(key, i))
    table = torch.full((len(need), max_pages), -1, dtype=torch.int32)
    k = 0
    for b, n in enumerate(owned):
        for j in range(n):
            table[b, j] = order[k]
            k += 1
    return table, n_pages


def to_pages(cache: torch.Tensor, table: torch.Tensor, page_size: int, n_pages: int) -> torch.Tensor:
    """The pool holding dense cache [B, Hkv, Lcap, D] under `table` (pages no
    entry names are NaN; table entries of -1 are skipped)."""
    B, Hkv, Lcap, D = cache.shape
    pool = torch.full((n_pages, Hkv, page_size, D), float("nan"), dtype=cache.dtype)
    for b in range(B):
        for j in range(table.shape[1]):
            p = int(table[b, j])
            if p < 0:
                continue
            lo = j * page_size
            hi = min(Lcap, lo + page_size)
            if lo >= Lcap:
                continue
            pool[p, :, : hi - lo] = cache[b, :, lo:hi]
    return pool


def from_pages(pool: torch.Tensor, table: torch.Tensor, page_size: int, Lcap: int) -> torch.Tensor:
    """The dense view [B, Hkv, Lcap, D] of a pool (slots without a page are NaN)."""
    n_pages, Hkv, _, D = pool.shape
    B = table.shape[0]
    out = torch.full((B, Hkv, Lcap, D), float("nan"), dtype=pool.dtype)
    for b in range(B):
        for j in range(table.shape[1]):
            p = int(table[b, j])
            lo = j * page_size
            if p < 0 or lo >= Lcap:
                continue
            hi = min(Lcap, lo + page_size)
            out[b, :, lo:hi] = pool[p, :, : hi - lo]
    return out
