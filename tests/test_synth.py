"""The seeded input generator: SplitMix64 against its published test vector,
the torch (vectorised) form against the scalar form, value distributions and
the workload recipes."""

import math

import torch

from synth import rng, trees, workloads


def test_splitmix64_published_vector():
    # first outputs of SplitMix64 seeded with 1234567 (Vigna's splitmix64.c)
    assert [rng.splitmix64_scalar(1234567, n) for n in range(5)] == [
        6457827717110365317, 3203168211198807973, 9817491932198370423,
        4593380528125082431, 16408922859458223821]
    assert rng.splitmix64_scalar(0, 0) == 0xE220A8397B1DCDAF


def test_vectorised_matches_scalar():
    for key in (0, 1234567, rng.derive_key(3, 4), (1 << 64) - 1):
        got = rng.uint64(key, 257, offset=1 << 40)
        ref = [rng.splitmix64_scalar(key, (1 << 40) + n) for n in range(257)]
        assert [v & rng.MASK64 for v in got.tolist()] == ref


def test_normal_and_uniform_moments():
    x = rng.normal(rng.derive_key(0, 1), 1 << 20)
    assert abs(float(x.mean())) < 5e-3 and abs(float(x.std()) - 1) < 5e-3
    assert float(x.abs().max()) < 8.6
    u = rng.uniform(rng.derive_key(0, 2), 1 << 16)
    assert 0 < float(u.min()) and float(u.max()) < 1


def test_round_to_bf16_is_round_to_nearest_even_via_f32():
    x = torch.tensor([1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -(1.0 + 2 ** -8)], dtype=torch.float64)
    y = rng.round_to(x, torch.bfloat16).to(torch.float64).tolist()
    assert y == [1.0, 1.0 + 2 ** -6, -1.0]


def test_workload_shapes_and_recipe():
    w = workloads.get("tiny_f32")
    t = workloads.make(w)
    assert t["q"].shape == (1, 16, 8, 64) and t["k_cache"].shape == (1, 8, 192, 64)
    assert t["parent"][0].tolist() == trees.topk_tree(16, [4, 2, 1, 1])
    assert torch.isnan(t["k_cache"][0, :, 128:]).all() and torch.isfinite(t["k_cache"][0, :, :128]).all()
    # siblings carry distinct candidate ids
    par = t["parent"][0].tolist()
    for n in range(16):
        kids = [int(t["cand"][0, c]) for c in range(16) if par[c] == n]
        assert len(kids) == len(set(kids))
    # every plant is the unique maximum of its row and names a child of that row's node
    for b, node, tok in t["plants"]:
        row = t["logits"][b, node]
        assert float(row[tok]) == workloads.PLANT and int((row == row.max()).sum()) == 1
        assert any(int(t["cand"][b, c]) == tok and par[c] == node for c in range(16))
    # same seed, same bytes
    t2 = workloads.make(w)
    assert torch.equal(t2["logits"], t["logits"]) and torch.equal(t2["q"], t["q"])


def test_batched_lengths_and_capacity():
    w = workloads.get("7b_batched")
    L = workloads.cache_lengths(w)
    assert len(L) == 16 and all(512 <= x <= 8192 for x in L)
    cap = workloads.lcap(w)
    assert cap % 64 == 0 and cap >= max(L) + w.T


def test_bf16_scaled_distribution():
    w = workloads.get("7b_l2048", L=64, V=4096)
    t = workloads.make(w)
    q = t["q"].float()
    assert abs(float(q.std()) - 1 / math.sqrt(128)) < 2e-3
    assert t["q"].dtype == torch.bfloat16 and t["logits"].dtype == torch.bfloat16


def test_paging_round_trip_and_scatter():
    """A dense cache put into pages by a seeded table and read back is unchanged
    where a page exists; the table scatters neighbouring slots; spare pages are
    NaN and entries past each sequence's need are -1."""
    from synth import paging
    need = [100, 0, 257, 64]
    table, n_pages = paging.page_table(need, 64, 6, seed=3)
    assert n_pages == 2 + 0 + 5 + 1 + 3
    owned = sorted(int(x) for x in table.flatten() if x >= 0)
    assert owned == sorted(set(owned)) and len(owned) == n_pages - 3       # each page owned once
    assert (table[1] == -1).all() and int(table[0, 2]) == -1
    cache = torch.randn(4, 2, 384, 8)
    pool = paging.to_pages(cache, table, 64, n_pages)
    spare = sorted(set(range(n_pages)) - set(owned))
    assert torch.isnan(pool[spare]).all()
    back = paging.from_pages(pool, table, 64, 384)
    for b, n in enumerate(need):
        m = -(-n // 64) * 64
        assert torch.equal(back[b, :, :m], cache[b, :, :m])
        assert torch.isnan(back[b, :, m:]).all()
    assert table[2, :5].tolist() != sorted(table[2, :5].tolist()) or table[2, :5].tolist() != list(range(5))
