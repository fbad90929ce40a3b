"""Planted mistakes in the oracle, on the CPU.

Each mutant is clover_oracle.c with one plausible slip -- a dropped term, a
wrong sign, index or bound, a transposed operand, a flipped comparison --
compiled beside the real oracle and swapped in for it.  The pins of its area
(tests/test_oracle_pins.py, which check the oracle against brute force,
closed forms, library routines and the paper's worked examples) must reject
it: a mutant that every pin accepts is a hole in the pins.  The unmutated
copy, built and loaded the same way, passes every pin (the control).

Every mutant keeps each access in bounds and each loop finite, so a mutant can
only compute a wrong answer, never crash the test process."""

from __future__ import annotations

import itertools
import os
import subprocess
from concurrent.futures import ThreadPoolExecutor

import pytest

import oracle
from tests import test_oracle_pins as pins

_SRC = os.path.join(os.path.dirname(oracle.__file__), "clover_oracle.c")
_DIR = os.path.join(os.path.dirname(oracle.__file__), "_build", "mutants")

ATTN = ("test_attention", "test_verify_step")
MASK = ("test_tree_mask",)
ARGMAX = ("test_argmax", "test_verify_step")
WALK = ("test_walk", "test_verify_step")
KV = ("test_append", "test_compact", "test_commit", "test_verify_step")
TYPICAL = ("test_typical",)
DRAFT = ("test_linear", "test_embed", "test_topk_vs", "test_head_step")

# name, the source text replaced (it occurs exactly once), its replacement, the pin areas that must catch it
MUTANTS = [
    # tree-masked attention (Section 3.2, the tree attention mask)
    ("attn_scale_dropped_on_cache_keys",
     "        score[n_keys] = P->scale * s;\n        v_base[n_keys] = P->v_cache;",
     "        score[n_keys] = s;\n        v_base[n_keys] = P->v_cache;", ATTN),
    ("attn_default_scale_one_over_d", "1.0 / sqrt((double)D)", "1.0 / (double)D", ATTN),
    ("attn_tree_keys_from_descendants", "if (!on_root_path(parent, i, m)) continue;",
     "if (!on_root_path(parent, m, i)) continue;", ATTN),
    ("attn_first_cache_key_skipped", "for (int j = 0; j < L; ++j) {", "for (int j = 1; j < L; ++j) {", ATTN),
    ("attn_kv_heads_interleaved", "const int g = h / G;", "const int g = h % P->Hkv;", ATTN),
    ("attn_no_max_subtraction", "score[n] = exp(score[n] - mx);", "score[n] = exp(score[n]);", ATTN),
    ("attn_values_from_key_cache", "v_base[n_keys] = P->v_cache;", "v_base[n_keys] = P->k_cache;", ATTN),
    ("attn_softmax_not_normalised", "out[d] /= z;", "out[d] += 0.0;", ATTN),
    ("attn_row_order_node_major",
     "const int h = (int)(r % Hq);\n        const int i = (int)((r / Hq) % T);",
     "const int h = (int)((r / T) % Hq);\n        const int i = (int)(r % T);", ATTN),
    ("attn_tree_keys_head_major",
     "const int64_t off = (((int64_t)b * P->T + m) * P->Hkv + g) * D;",
     "const int64_t off = (((int64_t)b * P->Hkv + g) * P->T + m) * D;", ATTN),
    ("bf16_widened_half_ulp_high", "(uint32_t)h << 16;", "((uint32_t)h << 16) | 0x8000u;", ATTN),
    # the tree mask
    ("mask_excludes_self", "for (int n = i; n >= 0; n = parent[n])",
     "for (int n = parent[i]; n >= 0; n = parent[n])", MASK + ATTN),
    ("mask_depth_counts_nodes", "depth[i] = d;", "depth[i] = d + 1;", MASK),
    ("mask_accepts_second_root", "if (parent[i] < 0 || parent[i] >= i) return 0;",
     "if (parent[i] < -1 || parent[i] >= i) return 0;", MASK),
    # argmax (the target model's greedy token at every node)
    ("argmax_last_index_of_ties",
     "            double x = load_elem(logits, r * V + v, dtype);\n            if (x > best) {",
     "            double x = load_elem(logits, r * V + v, dtype);\n            if (x >= best) {", ARGMAX),
    # the greedy acceptance walk
    ("walk_child_checked_against_own_argmax", "cd[c] == am[cur]", "cd[c] == am[c]", WALK),
    ("walk_takes_last_matching_child", "next = c;\n                    break;", "next = c;", WALK),
    ("walk_bonus_from_parent", "bonus[b] = am[cur];", "bonus[b] = am[pb[len > 1 ? len - 2 : 0]];", WALK),
    ("walk_length_excludes_root", "accept_len[b] = len;", "accept_len[b] = len - 1;", WALK),
    # cache append, compaction and commit
    ("append_at_slot_zero", "cache_len[b] + m;", "m;", KV),
    ("compact_src_index_is_destination", "src_index[(int64_t)b * T + j] = src_slot;",
     "src_index[(int64_t)b * T + j] = dst_slot;", KV),
    ("compact_k_copied_backwards",
     "memmove((char *)k_cache + (base + dst_slot) * row, (char *)k_cache + (base + src_slot) * row, row);",
     "memmove((char *)k_cache + (base + src_slot) * row, (char *)k_cache + (base + dst_slot) * row, row);", KV),
    ("commit_takes_node_j", "const int node = path[(int64_t)b * T + j];", "const int node = j;", KV),
    ("commit_src_index_offset", "src_index[(int64_t)b * T + j] = node;",
     "src_index[(int64_t)b * T + j] = L + node;", KV),
    # typical acceptance
    ("typical_entropy_sign", "if (p > 0.0) h -= p * log_p;", "if (p > 0.0) h += p * log_p;", TYPICAL),
    ("typical_threshold_max_not_min", "row_log_theta[r] = log_eps < log_dh", "row_log_theta[r] = log_eps > log_dh",
     TYPICAL),
    ("typical_edge_rule_inclusive", "acc[c] = log_p > row_log_theta[r];", "acc[c] = log_p >= row_log_theta[r];",
     TYPICAL),
    ("typical_reach_ignores_ancestors", "reach[c] = reach[par[c]] && acc[c];", "reach[c] = acc[c];", TYPICAL),
    ("typical_ties_largest_path", "better = this_path[k] < best_path[k];", "better = this_path[k] > best_path[k];",
     TYPICAL),
    ("typical_edge_without_temperature", "/ temperature - row_max[r] - row_lse[r]", "- row_max[r] - row_lse[r]",
     TYPICAL),
    ("typical_argmax_last_index_of_ties",
     "const double x = load_elem(logits, r * V + v, dtype);\n            if (x > best) {",
     "const double x = load_elem(logits, r * V + v, dtype);\n            if (x >= best) {", TYPICAL),
    ("typical_bonus_from_root", "bonus[b] = row_amax[(int64_t)b * T + best_path[best_len - 1]];",
     "bonus[b] = row_amax[(int64_t)b * T + best_path[0]];", TYPICAL),
    # the draft side's dense pieces (Section 3)
    ("linear_silu_sign", "s / (1.0 + exp(-s))", "s / (1.0 + exp(s))", DRAFT),
    ("linear_weight_transposed", "load_elem(w, n * K + k, dtype)", "load_elem(w, k * N + n, dtype)", DRAFT),
    ("linear_residual_dropped", "s = load_elem(res, r * N + n, dtype) + s / (1.0 + exp(-s));",
     "s = s / (1.0 + exp(-s));", DRAFT),
    ("embed_not_normalised", "dtype) * inv;", "dtype);", DRAFT),
    ("embed_norm_squared", "1.0 / sqrt(s)", "1.0 / s", DRAFT),
    ("topk_ties_by_largest_index", "row[v] > row[best]", "row[v] >= row[best]", DRAFT),
    ("topk_taken_not_excluded", "if (taken) continue;", "if (0 && taken) continue;", DRAFT),
]


def mutate(src: str, old: str, new: str) -> str:
    assert src.count(old) == 1, f"the mutation site must occur exactly once: {old!r}"
    return src.replace(old, new)


def _compile(name: str, text: str) -> str:
    c_path = os.path.join(_DIR, name + ".c")
    so_path = os.path.join(_DIR, name + ".so")
    with open(c_path, "w") as f:
        f.write(text)
    subprocess.run(["gcc", "-O2", "-fopenmp", "-std=c11", "-w", "-shared", "-fPIC", c_path, "-o", so_path, "-lm"],
                   check=True)
    return so_path


@pytest.fixture(scope="module")
def libs():
    """Every mutant and the unmutated control, compiled in parallel."""
    os.makedirs(_DIR, exist_ok=True)
    with open(_SRC) as f:
        src = f.read()
    texts = {"control": src}
    for name, old, new, _ in MUTANTS:
        texts[name] = mutate(src, old, new)
    with ThreadPoolExecutor(max_workers=min(16, os.cpu_count() or 1)) as ex:
        paths = dict(zip(texts, ex.map(lambda kv: _compile(*kv), texts.items())))
    return {name: oracle._open(path) for name, path in paths.items()}


def expand(fn):
    """The keyword sets of a pin's parametrize marks (their cartesian product)."""
    sets = []
    for mark in getattr(fn, "pytestmark", []):
        if mark.name != "parametrize":
            continue
        names, values = mark.args[0], mark.args[1]
        names = [n.strip() for n in names.split(",")] if isinstance(names, str) else list(names)
        sets.append([dict(zip(names, v if len(names) > 1 else (v,))) for v in values])
    return [dict(kv for d in combo for kv in d.items()) for combo in itertools.product(*sets)]


def pin_cases(areas):
    for name, fn in list(vars(pins).items()):
        if name.startswith(areas) and callable(fn):
            for kw in expand(fn):
                yield name, fn, kw


def failing_pins(lib, areas, monkeypatch) -> list[str]:
    failed = []
    with monkeypatch.context() as m:
        m.setattr(oracle, "_lib", lib)
        for name, fn, kw in pin_cases(areas):
            try:
                fn(**kw)
            except pytest.skip.Exception:
                continue
            except (Exception, pytest.fail.Exception):
                failed.append(f"{name}{kw or ''}")
    return failed


def test_mutation_sites_are_unique():
    with open(_SRC) as f:
        src = f.read()
    names = [m[0] for m in MUTANTS]
    assert len(set(names)) == len(names)
    for name, old, new, _ in MUTANTS:
        assert old != new and src.count(old) == 1, name


def test_unmutated_copy_passes_every_pin(libs, monkeypatch):
    areas = tuple(sorted({a for *_, ar in MUTANTS for a in ar}))
    assert sum(1 for _ in pin_cases(areas)) > 60
    assert failing_pins(libs["control"], areas, monkeypatch) == []


@pytest.mark.parametrize("name,areas", [(m[0], m[3]) for m in MUTANTS], ids=[m[0] for m in MUTANTS])
def test_pins_reject_planted_mistake(name, areas, libs, monkeypatch):
    assert failing_pins(libs[name], areas, monkeypatch), f"no pin of {areas} rejects the mutant {name}"


# ---------------------------------------------------------------------------
# The oracle's Python compositions (oracle/__init__.py): one slip in a
# function's source, the function rebuilt from it beside the real one and
# swapped in for it.
# ---------------------------------------------------------------------------

HEAD = ("test_head_step",)

# name, the oracle function, the source text replaced (once in that function), its replacement, the pin areas
PY_MUTANTS = [
    ("verify_step_without_append", "verify_step",
     '    append_tree_kv(inp["k_new"], inp["v_new"], k_cache, v_cache, cache_len)\n', "", ("test_verify_step",)),
    ("verify_step_typical_outputs_swapped", "verify_step",
     '        amax, path, alen, bonus = r["argmax"], r["path"], r["accept_len"], r["bonus"]\n',
     '        amax, path, alen, bonus = r["argmax"], r["path"], r["accept_len"], r["argmax"][:, 0]\n', ("test_verify_step",)),
    ("head_step_residual_dropped", "clover_head_step", "    h1 = h.double() + d\n", "    h1 = d\n", HEAD),
    ("head_step_decoder_weights_swapped", "clover_head_step",
     "    a = linear(e.to(bf), w_v)\n    d = linear(a.to(bf), w_o)\n",
     "    a = linear(e.to(bf), w_o)\n    d = linear(a.to(bf), w_v)\n", HEAD),
    ("head_step_mlp_residual_from_input", "clover_head_step", "res=h1.to(bf), act=1)", "res=h.to(bf), act=1)", HEAD),
    ("head_step_lm_head_before_mlp", "clover_head_step", "    logits = linear(z.to(bf), w_lm)\n",
     "    logits = linear(h1.to(bf), w_lm)\n", HEAD),
    # the fp64 statement of the head step (the reference of the rounding bound)
    ("exact_step_silu_sign", "clover_head_step_exact", "u / (1.0 + torch.exp(-u))", "u / (1.0 + torch.exp(u))", HEAD),
    ("exact_step_weight_transposed", "clover_head_step_exact", "    a = e @ W_v.T\n", "    a = e @ W_v\n", HEAD),
    ("exact_step_mlp_residual_dropped", "clover_head_step_exact", "    z = h1 + u / (1.0 + torch.exp(-u))\n",
     "    z = u / (1.0 + torch.exp(-u))\n", HEAD),
]


def rebuild(fn_name: str, old: str = "", new: str = ""):
    """The oracle function `fn_name` defined again from its source, with `old`
    replaced by `new` when given, over a copy of the oracle module's globals
    (so that it calls the real library functions)."""
    import inspect
    src = inspect.getsource(getattr(oracle, fn_name))
    if old:
        assert src.count(old) == 1, f"the mutation site must occur exactly once in {fn_name}: {old!r}"
        src = src.replace(old, new)
    ns = dict(vars(oracle))
    exec(compile(src, oracle.__file__, "exec"), ns)
    return ns[fn_name]


def failing_pins_py(fn_name, fn, areas, monkeypatch) -> list[str]:
    failed = []
    with monkeypatch.context() as m:
        m.setattr(oracle, fn_name, fn)
        for name, pin, kw in pin_cases(areas):
            try:
                pin(**kw)
            except pytest.skip.Exception:
                continue
            except (Exception, pytest.fail.Exception):
                failed.append(f"{name}{kw or ''}")
    return failed


def test_unmutated_python_compositions_pass_their_pins(monkeypatch):
    """The control: each function rebuilt from its unchanged source passes
    every pin of its areas."""
    for fn_name in sorted({m[1] for m in PY_MUTANTS}):
        areas = tuple(sorted({a for _, f, _, _, ar in PY_MUTANTS if f == fn_name for a in ar}))
        assert sum(1 for _ in pin_cases(areas)) > 0
        assert failing_pins_py(fn_name, rebuild(fn_name), areas, monkeypatch) == []


@pytest.mark.parametrize("name,fn_name,old,new,areas", PY_MUTANTS, ids=[m[0] for m in PY_MUTANTS])
def test_pins_reject_planted_composition_mistake(name, fn_name, old, new, areas, monkeypatch):
    fn = rebuild(fn_name, old, new)
    assert failing_pins_py(fn_name, fn, areas, monkeypatch), f"no pin of {areas} rejects the mutant {name}"
