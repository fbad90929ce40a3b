"""The oracle: a plain fp64 CPU statement of the verification step.

TEST INFRASTRUCTURE ONLY -- imported by the tests, by ``__graft_entry__.smoke``
and by the benchmark's CPU-baseline leg, never by the library.  It shares no
code with the CUDA path.  ``clover_oracle.c`` holds the arithmetic; this module
compiles it with gcc (on first use, or from ``build()``) and marshals arguments.

Functions take and return torch CPU tensors (bf16 inputs are passed as their
bytes and widened exactly inside the C code).
"""

from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "clover_oracle.c")
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB = os.path.join(_OUT_DIR, "liboracle.so")

OK = 0
BAD_ARG = 1
BAD_TREE = 4
NO_MEMORY = 64

F32 = 0
BF16 = 1

_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile clover_oracle.c into _build/liboracle.so (gcc -O2 -fopenmp)."""
    os.makedirs(_OUT_DIR, exist_ok=True)
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.run(["gcc", "-O2", "-fopenmp", "-std=c11", "-Wall", "-shared", "-fPIC",
                        _SRC, "-o", tmp, "-lm"], check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _open(path: str):
    """Load a compiled copy of clover_oracle.c and declare its signatures."""
    lib = ctypes.CDLL(path)
    P, I, I64, D = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_double
    lib.oracle_tree_mask.argtypes = [P, I, P, P]
    lib.oracle_tree_attention.argtypes = [P, P, P, P, P, P, P, I, I, I, I, I, I, I, D,
                                          P, I64, P, I]
    lib.oracle_argmax.argtypes = [P, I64, I64, I, P, I64, P, I]
    lib.oracle_accept_walk.argtypes = [P, P, P, I, I, P, P, P]
    lib.oracle_append_tree_kv.argtypes = [P, P, P, P, P, I, I, I, I, I, I]
    lib.oracle_kv_compact.argtypes = [P, P, P, P, P, I, I, I, I, I, I, P]
    lib.oracle_kv_commit.argtypes = [P, P, P, P, P, P, P, I, I, I, I, I, I, P]
    lib.oracle_accept_typical.argtypes = [P, P, P, I, I, I64, I, D, D, D, P, P, P, P, P, I]
    lib.oracle_linear.argtypes = [P, P, P, I, I, I, I, I, P, I]
    lib.oracle_embed_rows.argtypes = [P, P, I, I, I, I, P]
    lib.oracle_topk.argtypes = [P, I, I, I, P, P]
    for f in (lib.oracle_tree_mask, lib.oracle_tree_attention, lib.oracle_argmax,
              lib.oracle_accept_walk, lib.oracle_append_tree_kv, lib.oracle_kv_compact,
              lib.oracle_kv_commit):
        f.restype = ctypes.c_int
    return lib


def _load():
    global _lib
    with _lock:
        if _lib is None:
            _lib = _open(build())
    return _lib


class OracleError(RuntimeError):
    def __init__(self, code: int):
        super().__init__(f"oracle returned status {code}")
        self.code = code


def _check(code: int):
    if code != OK:
        raise OracleError(code)


def _cpu(t: torch.Tensor) -> torch.Tensor:
    if t.device.type != "cpu":
        raise ValueError("the oracle takes CPU tensors")
    return t.contiguous()


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return F32
    if t.dtype == torch.bfloat16:
        return BF16
    raise ValueError(f"unsupported dtype {t.dtype}")


def _p(t):
    return ctypes.c_void_p(t.data_ptr()) if t is not None else None


def default_threads() -> int:
    return os.cpu_count() or 1


def tree_mask(parent) -> tuple[torch.Tensor, torch.Tensor]:
    """(mask [T,T] bool, depth [T] int32) of one parent array."""
    par = _cpu(torch.as_tensor(parent, dtype=torch.int32))
    T = par.numel()
    mask = torch.zeros((T, T), dtype=torch.uint8)
    depth = torch.zeros(T, dtype=torch.int32)
    _check(_load().oracle_tree_mask(_p(par), T, _p(mask), _p(depth)))
    return mask.bool(), depth


def tree_attention(q, k_new, v_new, k_cache, v_cache, cache_len, parent, scale: float = 0.0,
                   rows=None, n_threads: int | None = None) -> torch.Tensor:
    """fp64 attention rows; ``rows`` = flattened (b*T+i)*Hq+h ids, or None for all.

    Returns [B,T,Hq,D] float64 when rows is None, else [len(rows), D].
    """
    q, k_new, v_new = _cpu(q), _cpu(k_new), _cpu(v_new)
    k_cache, v_cache = _cpu(k_cache), _cpu(v_cache)
    cl = _cpu(cache_len.to(torch.int32))
    par = _cpu(parent.to(torch.int32))
    B, T, Hq, D = q.shape
    Hkv, Lcap = k_cache.shape[1], k_cache.shape[2]
    dt = _dtype_code(q)
    if rows is None:
        out = torch.empty((B, T, Hq, D), dtype=torch.float64)
        rows_t, n = None, B * T * Hq
    else:
        rows_t = _cpu(torch.as_tensor(rows, dtype=torch.int64))
        n = rows_t.numel()
        out = torch.empty((n, D), dtype=torch.float64)
    _check(_load().oracle_tree_attention(
        _p(q), _p(k_new), _p(v_new), _p(k_cache), _p(v_cache), _p(cl), _p(par),
        B, T, Hq, Hkv, D, Lcap, dt, float(scale), _p(rows_t), n, _p(out),
        n_threads or default_threads()))
    return out


def argmax(logits, rows=None, n_threads: int | None = None) -> torch.Tensor:
    """First-index argmax over the last dim; returns int32 of logits.shape[:-1] or [len(rows)]."""
    lg = _cpu(logits)
    V = lg.shape[-1]
    n_total = lg.numel() // V
    if rows is None:
        out = torch.empty(lg.shape[:-1], dtype=torch.int32)
        rows_t, n = None, n_total
    else:
        rows_t = _cpu(torch.as_tensor(rows, dtype=torch.int64))
        n = rows_t.numel()
        out = torch.empty(n, dtype=torch.int32)
    _check(_load().oracle_argmax(_p(lg), n_total, V, _dtype_code(lg), _p(rows_t), n, _p(out),
                                 n_threads or default_threads()))
    return out


def accept_walk(parent, cand, amax):
    """(path [B,T], accept_len [B], bonus [B]) int32."""
    par = _cpu(parent.to(torch.int32))
    cd = _cpu(cand.to(torch.int32))
    am = _cpu(amax.to(torch.int32))
    B, T = par.shape
    path = torch.empty((B, T), dtype=torch.int32)
    alen = torch.empty(B, dtype=torch.int32)
    bonus = torch.empty(B, dtype=torch.int32)
    _check(_load().oracle_accept_walk(_p(par), _p(cd), _p(am), B, T, _p(path), _p(alen),
                                      _p(bonus)))
    return path, alen, bonus


def accept_typical(logits, parent, cand, temperature: float, epsilon: float, delta: float,
                   n_threads: int | None = None) -> dict:
    """Typical acceptance of every sequence.  logits [B, T, V] (or [B*T, V]),
    parent/cand [B, T].  Returns argmax [B,T], path [B,T], accept_len [B],
    bonus [B] (int32) and margin [B,T] (fp64, ln p - ln theta per edge)."""
    par = _cpu(parent.to(torch.int32))
    cd = _cpu(cand.to(torch.int32))
    B, T = par.shape
    lg = _cpu(logits)
    V = lg.shape[-1]
    assert lg.numel() == B * T * V
    amax = torch.empty((B, T), dtype=torch.int32)
    path = torch.empty((B, T), dtype=torch.int32)
    alen = torch.empty(B, dtype=torch.int32)
    bonus = torch.empty(B, dtype=torch.int32)
    margin = torch.empty((B, T), dtype=torch.float64)
    _check(_load().oracle_accept_typical(_p(lg), _p(par), _p(cd), B, T, V, _dtype_code(lg), float(temperature),
                                         float(epsilon), float(delta), _p(amax), _p(path), _p(alen), _p(bonus),
                                         _p(margin), n_threads or default_threads()))
    return {"argmax": amax, "path": path, "accept_len": alen, "bonus": bonus, "margin": margin}


def append_tree_kv(k_new, v_new, k_cache, v_cache, cache_len):
    """In place on k_cache/v_cache (contiguous CPU tensors)."""
    assert k_cache.is_contiguous() and v_cache.is_contiguous()
    kn, vn = _cpu(k_new), _cpu(v_new)
    cl = _cpu(cache_len.to(torch.int32))
    B, Hkv, Lcap, D = k_cache.shape
    T = kn.shape[1]
    _check(_load().oracle_append_tree_kv(_p(kn), _p(vn), _p(k_cache), _p(v_cache), _p(cl), B, T,
                                         Hkv, D, Lcap, k_cache.element_size()))


def kv_compact(k_cache, v_cache, cache_len, path, accept_len):
    """In place on k_cache/v_cache/cache_len (int32); returns src_index [B,T]."""
    assert k_cache.is_contiguous() and v_cache.is_contiguous() and cache_len.dtype == torch.int32
    B, Hkv, Lcap, D = k_cache.shape
    pa = _cpu(path.to(torch.int32))
    al = _cpu(accept_len.to(torch.int32))
    T = pa.shape[1]
    src = torch.empty((B, T), dtype=torch.int32)
    _check(_load().oracle_kv_compact(_p(k_cache), _p(v_cache), _p(cache_len), _p(pa), _p(al), B, T,
                                     Hkv, D, Lcap, k_cache.element_size(), _p(src)))
    return src


def kv_commit(k_cache, v_cache, k_new, v_new, cache_len, path, accept_len):
    """In place on k_cache/v_cache/cache_len (int32): slot L+j <- node path[j]
    of k_new/v_new; returns src_index [B,T] (the nodes, -1 past a)."""
    assert k_cache.is_contiguous() and v_cache.is_contiguous() and cache_len.dtype == torch.int32
    B, Hkv, Lcap, D = k_cache.shape
    kn, vn = _cpu(k_new), _cpu(v_new)
    pa = _cpu(path.to(torch.int32))
    al = _cpu(accept_len.to(torch.int32))
    T = pa.shape[1]
    src = torch.empty((B, T), dtype=torch.int32)
    _check(_load().oracle_kv_commit(_p(k_cache), _p(v_cache), _p(kn), _p(vn), _p(cache_len), _p(pa), _p(al), B, T,
                                    Hkv, D, Lcap, k_cache.element_size(), _p(src)))
    return src


def verify_step(inp: dict, scale: float = 0.0, n_threads: int | None = None, typical=None) -> dict:
    """The whole step on copies of the inputs: attention, append, argmax, walk
    (greedy, or typical acceptance with ``typical`` = (temperature, epsilon,
    delta)), compact."""
    k_cache = inp["k_cache"].clone()
    v_cache = inp["v_cache"].clone()
    cache_len = inp["cache_len"].clone().to(torch.int32)
    out = tree_attention(inp["q"], inp["k_new"], inp["v_new"], k_cache, v_cache, cache_len,
                         inp["parent"], scale=scale, n_threads=n_threads)
    append_tree_kv(inp["k_new"], inp["v_new"], k_cache, v_cache, cache_len)
    if typical is None:
        amax = argmax(inp["logits"], n_threads=n_threads)
        path, alen, bonus = accept_walk(inp["parent"], inp["cand"], amax)
    else:
        r = accept_typical(inp["logits"], inp["parent"], inp["cand"], *typical, n_threads=n_threads)
        amax, path, alen, bonus = r["argmax"], r["path"], r["accept_len"], r["bonus"]
    src = kv_compact(k_cache, v_cache, cache_len, path, alen)
    return {"out": out, "argmax": amax, "path": path, "accept_len": alen, "bonus": bonus,
            "src_index": src, "k_cache": k_cache, "v_cache": v_cache, "cache_len": cache_len}


def linear(x, w, res=None, act=0, n_threads: int | None = None) -> torch.Tensor:
    """fp64 y [R,N] = x [R,K] . w [N,K]^T (act 0), or res + silu(x . w^T) (act 1);
    x, w, res share one dtype."""
    xc, wc = _cpu(x), _cpu(w)
    R, K = xc.shape
    N = wc.shape[0]
    assert wc.shape[1] == K and wc.dtype == xc.dtype
    rc = _cpu(res) if res is not None else None
    if rc is not None:
        assert rc.shape == (R, N) and rc.dtype == xc.dtype
    y = torch.empty((R, N), dtype=torch.float64)
    _check(_load().oracle_linear(_p(xc), _p(wc), _p(rc), R, N, K, _dtype_code(xc), act, _p(y),
                                 n_threads or default_threads()))
    return y


def embed_rows(w, tokens) -> torch.Tensor:
    """fp64 e [R,H]: row tokens[r] of w [V,H] divided by its L2 norm."""
    wc = _cpu(w)
    V, H = wc.shape
    t = _cpu(torch.as_tensor(tokens, dtype=torch.int32))
    e = torch.empty((t.numel(), H), dtype=torch.float64)
    _check(_load().oracle_embed_rows(_p(wc), _p(t), t.numel(), V, H, _dtype_code(wc), _p(e)))
    return e


def topk(x, k: int):
    """(values fp64 [R,k], indices int32 [R,k]) of each row of x (widened to fp64):
    decreasing value, equal values by increasing index."""
    xc = _cpu(x.to(torch.float64))
    R, V = xc.shape
    vals = torch.empty((R, k), dtype=torch.float64)
    idx = torch.empty((R, k), dtype=torch.int32)
    _check(_load().oracle_topk(_p(xc), R, V, k, _p(vals), _p(idx)))
    return vals, idx


def clover_head_step(h, tokens, w_lm, w_v, w_o, w_1, k: int):
    """One speculative head (Section 3.2 Eq. 1-2, the MLP block, the shared LM
    head), from bf16 inputs h [R,H] (the previous hidden state) and tokens [R]
    (the previous token).  The cross attention has a single key and value (the
    previous token's embedding), so its softmax weight is 1 and its output is
    W_o . W_v . e whatever the query; W_Q and W_K do not enter.  Every layer's
    input is a bf16 tensor (rounded to nearest even), as the layers take them:
      e  = embed_rows(w_lm, tokens)
      h' = h + W_o (W_v e)
      z  = h' + silu(W_1 h')
      logits = W_lm z, and their top-k.
    Returns a dict of the fp64 intermediates, the logits and the top-k."""
    bf = torch.bfloat16
    e = embed_rows(w_lm, tokens)
    a = linear(e.to(bf), w_v)
    d = linear(a.to(bf), w_o)
    h1 = h.double() + d
    z = linear(h1.to(bf), w_1, res=h1.to(bf), act=1)
    logits = linear(z.to(bf), w_lm)
    vals, idx = topk(logits, k)
    return {"e": e, "v": a, "attn": d, "h": h1, "z": z, "logits": logits, "top_values": vals, "top_indices": idx}


def clover_head_step_exact(h, tokens, w_lm, w_v, w_o, w_1, k: int):
    """The same head step (Section 3.2 Eq. 1-2, the MLP block, the shared LM
    head) in fp64 throughout: the bf16 inputs h and weights are widened once
    and no intermediate is rounded, so this is the step's plain definition on
    those inputs.  Each layer is one fp64 matrix product (a library routine),
    silu(x) = x / (1 + e^-x).  Same keys as clover_head_step."""
    W_v, W_o, W_1, W_lm = (_cpu(w).double() for w in (w_v, w_o, w_1, w_lm))
    e = embed_rows(w_lm, tokens)
    a = e @ W_v.T
    d = a @ W_o.T
    h1 = _cpu(h).double() + d
    u = h1 @ W_1.T
    z = h1 + u / (1.0 + torch.exp(-u))
    logits = z @ W_lm.T
    vals, idx = topk(logits, k)
    return {"e": e, "v": a, "attn": d, "h": h1, "z": z, "logits": logits, "top_values": vals, "top_indices": idx}
