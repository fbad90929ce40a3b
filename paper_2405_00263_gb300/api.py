"""Python binding of the C ABI, with the same names.

Each function only checks and marshals its torch arguments (device, dtype,
shape, contiguity) and calls the library; every step of the computation runs
in the CUDA kernels.  Tensors must live on the current CUDA device; the stream
defaults to torch's current stream.
"""

from __future__ import annotations

import ctypes
import math

import torch

from . import _lib

OK = 0
ERR_INVALID_ARG = 1
ERR_UNSUPPORTED = 2
ERR_BAD_TREE = 4
ERR_CAPACITY = 8
ERR_CUDA = 16
ERR_TIMEOUT = 32
ERR_SCRATCH_LIMIT = 64
ERR_CHECK = 128

F32 = 0
BF16 = 1


class CloverError(RuntimeError):
    def __init__(self, code: int, where: str):
        lib = _lib.load()
        super().__init__(f"{where}: {lib.clover_status_string(code).decode()} (status {code})")
        self.code = code


def dtype_code(dt: torch.dtype) -> int:
    if dt == torch.float32:
        return F32
    if dt == torch.bfloat16:
        return BF16
    raise TypeError(f"unsupported dtype {dt}: float32 or bfloat16")


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _dev(*tensors):
    dev = None
    for t in tensors:
        if t is None:
            continue
        if not t.is_cuda:
            raise ValueError("all tensors must be CUDA tensors")
        if not t.is_contiguous():
            raise ValueError("all tensors must be contiguous")
        if dev is None:
            dev = t.device
        elif t.device != dev:
            raise ValueError("all tensors must be on one device")
    return dev


def _check(t, shape, dtype, name):
    if tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name}: expected shape {tuple(shape)}, got {tuple(t.shape)}")
    if t.dtype != dtype:
        raise ValueError(f"{name}: expected {dtype}, got {t.dtype}")


def clover_abi_version() -> int:
    return _lib.load().clover_abi_version()


def clover_build_flags() -> int:
    """Build options of the loaded library (bit 1: device index checks)."""
    return _lib.load().clover_build_flags()


def clover_verify_attn_workspace_size(B, T, Hq, Hkv, D, Lcap, dtype) -> int:
    code = dtype if isinstance(dtype, int) else dtype_code(dtype)
    return int(_lib.load().clover_verify_attn_workspace_size(B, T, Hq, Hkv, D, Lcap, code))


def clover_verify_accept_workspace_size(B, T, V, dtype) -> int:
    code = dtype if isinstance(dtype, int) else dtype_code(dtype)
    return int(_lib.load().clover_verify_accept_workspace_size(B, T, V, code))


def clover_verify_accept_typical_workspace_size(B, T, V, dtype) -> int:
    code = dtype if isinstance(dtype, int) else dtype_code(dtype)
    return int(_lib.load().clover_verify_accept_typical_workspace_size(B, T, V, code))


def clover_verify_attn(q, k_new, v_new, k_cache, v_cache, cache_len, parent, out, scale=0.0,
                       workspace=None, status=None, stream=None, append=True, pdl=False, cache_ready=False,
                       inputs_ready=False):
    """Tree-masked attention; with ``append`` (clover_verify_attn) it also
    writes k_new/v_new at cache slots [L, L+T), without it
    (clover_verify_attn_ex with CLOVER_ATTN_NO_APPEND) the caches are only read.
    ``pdl``: CLOVER_ATTN_PDL (launched as a programmatic dependent of the
    kernel queued before it); ``cache_ready`` (with ``pdl``):
    CLOVER_ATTN_CACHE_READY, the caller's statement that the caches and
    cache_len are not being written by the kernels that may still run;
    ``inputs_ready`` (with ``pdl``): CLOVER_ATTN_INPUTS_READY, the same
    statement of every input."""
    B, T, Hq, D = q.shape
    Hkv, Lcap = k_cache.shape[1], k_cache.shape[2]
    dt = q.dtype
    _check(k_new, (B, T, Hkv, D), dt, "k_new")
    _check(v_new, (B, T, Hkv, D), dt, "v_new")
    _check(k_cache, (B, Hkv, Lcap, D), dt, "k_cache")
    _check(v_cache, (B, Hkv, Lcap, D), dt, "v_cache")
    _check(cache_len, (B,), torch.int32, "cache_len")
    _check(parent, (B, T), torch.int32, "parent")
    _check(out, (B, T, Hq, D), dt, "out")
    if status is not None:
        _check(status, (1,), torch.int32, "status")
    _dev(q, k_new, v_new, k_cache, v_cache, cache_len, parent, out, workspace, status)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    args = (_ptr(q), _ptr(k_new), _ptr(v_new), _ptr(k_cache), _ptr(v_cache), _ptr(cache_len), _ptr(parent),
            _ptr(out), B, T, Hq, Hkv, D, Lcap, dtype_code(dt), float(scale), _ptr(workspace), ws_bytes,
            _ptr(status), _stream(stream))
    flags = (0 if append else _lib.ATTN_NO_APPEND) | (_lib.ATTN_PDL if pdl else 0) | \
        (_lib.ATTN_CACHE_READY if cache_ready else 0) | (_lib.ATTN_INPUTS_READY if inputs_ready else 0)
    if flags == 0:
        code = _lib.load().clover_verify_attn(*args)
    else:
        code = _lib.load().clover_verify_attn_ex(*args, flags)
    if code != OK:
        raise CloverError(code, "clover_verify_attn" if flags == 0 else "clover_verify_attn_ex")


def clover_verify_attn_noalloc(q, k_new, v_new, k_cache, v_cache, cache_len, parent, out, scale=0.0,
                               status=None, stream=None):
    """clover_verify_attn for callers that cannot allocate device memory: the
    scratch is a static 8 MiB device buffer inside the library, shared by every
    call on a device (calls that overlap on the GPU race)."""
    B, T, Hq, D = q.shape
    Hkv, Lcap = k_cache.shape[1], k_cache.shape[2]
    dt = q.dtype
    _check(k_new, (B, T, Hkv, D), dt, "k_new")
    _check(v_new, (B, T, Hkv, D), dt, "v_new")
    _check(k_cache, (B, Hkv, Lcap, D), dt, "k_cache")
    _check(v_cache, (B, Hkv, Lcap, D), dt, "v_cache")
    _check(cache_len, (B,), torch.int32, "cache_len")
    _check(parent, (B, T), torch.int32, "parent")
    _check(out, (B, T, Hq, D), dt, "out")
    if status is not None:
        _check(status, (1,), torch.int32, "status")
    _dev(q, k_new, v_new, k_cache, v_cache, cache_len, parent, out, status)
    code = _lib.load().clover_verify_attn_noalloc(
        _ptr(q), _ptr(k_new), _ptr(v_new), _ptr(k_cache), _ptr(v_cache), _ptr(cache_len), _ptr(parent),
        _ptr(out), B, T, Hq, Hkv, D, Lcap, dtype_code(dt), float(scale), _ptr(status), _stream(stream))
    if code != OK:
        raise CloverError(code, "clover_verify_attn_noalloc")


def clover_verify_accept(logits, cand, parent, argmax_out, path_out, accept_len, bonus_token,
                         workspace, status=None, stream=None):
    """Per-node argmax and the greedy acceptance walk."""
    B, T, V = logits.shape
    _check(cand, (B, T), torch.int32, "cand")
    _check(parent, (B, T), torch.int32, "parent")
    _check(argmax_out, (B, T), torch.int32, "argmax_out")
    _check(path_out, (B, T), torch.int32, "path_out")
    _check(accept_len, (B,), torch.int32, "accept_len")
    _check(bonus_token, (B,), torch.int32, "bonus_token")
    if status is not None:
        _check(status, (1,), torch.int32, "status")
    _dev(logits, cand, parent, argmax_out, path_out, accept_len, bonus_token, workspace, status)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    code = _lib.load().clover_verify_accept(
        _ptr(logits), _ptr(cand), _ptr(parent), B, T, V, dtype_code(logits.dtype), _ptr(argmax_out),
        _ptr(path_out), _ptr(accept_len), _ptr(bonus_token), _ptr(workspace), ws_bytes, _ptr(status),
        _stream(stream))
    if code != OK:
        raise CloverError(code, "clover_verify_accept")


def clover_verify_accept_typical(logits, cand, parent, temperature, epsilon, delta, argmax_out, path_out,
                                 accept_len, bonus_token, workspace, status=None, stream=None):
    """Per-node argmax and the typical (tempered-softmax, entropy-threshold)
    acceptance of the longest accepted path."""
    B, T, V = logits.shape
    _check(cand, (B, T), torch.int32, "cand")
    _check(parent, (B, T), torch.int32, "parent")
    _check(argmax_out, (B, T), torch.int32, "argmax_out")
    _check(path_out, (B, T), torch.int32, "path_out")
    _check(accept_len, (B,), torch.int32, "accept_len")
    _check(bonus_token, (B,), torch.int32, "bonus_token")
    if status is not None:
        _check(status, (1,), torch.int32, "status")
    _dev(logits, cand, parent, argmax_out, path_out, accept_len, bonus_token, workspace, status)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    code = _lib.load().clover_verify_accept_typical(
        _ptr(logits), _ptr(cand), _ptr(parent), B, T, V, dtype_code(logits.dtype), float(temperature),
        float(epsilon), float(delta), _ptr(argmax_out), _ptr(path_out), _ptr(accept_len), _ptr(bonus_token),
        _ptr(workspace), ws_bytes, _ptr(status), _stream(stream))
    if code != OK:
        raise CloverError(code, "clover_verify_accept_typical")


def clover_kv_compact(k_cache, v_cache, cache_len, path, accept_len, new_cache_len, src_index_out=None,
                      status=None, stream=None):
    """Moves the accepted nodes' K/V to slots [L, L+a); new_cache_len = L + a."""
    B, Hkv, Lcap, D = k_cache.shape
    T = path.shape[1]
    _check(v_cache, (B, Hkv, Lcap, D), k_cache.dtype, "v_cache")
    _check(cache_len, (B,), torch.int32, "cache_len")
    _check(path, (B, T), torch.int32, "path")
    _check(accept_len, (B,), torch.int32, "accept_len")
    _check(new_cache_len, (B,), torch.int32, "new_cache_len")
    if src_index_out is not None:
        _check(src_index_out, (B, T), torch.int32, "src_index_out")
    if status is not None:
        _check(status, (1,), torch.int32, "status")
    _dev(k_cache, v_cache, cache_len, path, accept_len, new_cache_len, src_index_out, status)
    code = _lib.load().clover_kv_compact(
        _ptr(k_cache), _ptr(v_cache), _ptr(cache_len), _ptr(path), _ptr(accept_len), _ptr(new_cache_len),
        _ptr(src_index_out), B, T, Hkv, D, Lcap, dtype_code(k_cache.dtype), _ptr(status), _stream(stream))
    if code != OK:
        raise CloverError(code, "clover_kv_compact")


def clover_verify_attn_paged_workspace_size(B, T, Hq, Hkv, D, page_size, max_pages, dtype) -> int:
    code = dtype if isinstance(dtype, int) else dtype_code(dtype)
    return int(_lib.load().clover_verify_attn_paged_workspace_size(B, T, Hq, Hkv, D, page_size, max_pages, code))


def clover_verify_attn_paged(q, k_new, v_new, k_pages, v_pages, block_table, cache_len, parent, out, scale=0.0,
                             workspace=None, status=None, stream=None, pdl=False, cache_ready=False,
                             inputs_ready=False):
    """Tree-masked attention over a paged cache: pools [n_pages, Hkv, page_size, D],
    block_table [B, max_pages] (the pools are only read).  ``pdl``,
    ``cache_ready`` and ``inputs_ready`` as for clover_verify_attn (through
    clover_verify_attn_paged_ex; the statements also cover the block table)."""
    B, T, Hq, D = q.shape
    n_pages, Hkv, page_size = k_pages.shape[0], k_pages.shape[1], k_pages.shape[2]
    max_pages = block_table.shape[1]
    dt = q.dtype
    _check(k_new, (B, T, Hkv, D), dt, "k_new")
    _check(v_new, (B, T, Hkv, D), dt, "v_new")
    _check(k_pages, (n_pages, Hkv, page_size, D), dt, "k_pages")
    _check(v_pages, (n_pages, Hkv, page_size, D), dt, "v_pages")
    _check(block_table, (B, max_pages), torch.int32, "block_table")
    _check(cache_len, (B,), torch.int32, "cache_len")
    _check(parent, (B, T), torch.int32, "parent")
    _check(out, (B, T, Hq, D), dt, "out")
    if status is not None:
        _check(status, (1,), torch.int32, "status")
    _dev(q, k_new, v_new, k_pages, v_pages, block_table, cache_len, parent, out, workspace, status)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    args = (_ptr(q), _ptr(k_new), _ptr(v_new), _ptr(k_pages), _ptr(v_pages), _ptr(block_table), n_pages, page_size,
            max_pages, _ptr(cache_len), _ptr(parent), _ptr(out), B, T, Hq, Hkv, D, dtype_code(dt), float(scale),
            _ptr(workspace), ws_bytes, _ptr(status), _stream(stream))
    flags = (_lib.ATTN_PDL if pdl else 0) | (_lib.ATTN_CACHE_READY if cache_ready else 0) | \
        (_lib.ATTN_INPUTS_READY if inputs_ready else 0)
    if flags == 0:
        code = _lib.load().clover_verify_attn_paged(*args)
    else:
        code = _lib.load().clover_verify_attn_paged_ex(*args, flags)
    if code != OK:
        raise CloverError(code, "clover_verify_attn_paged" if flags == 0 else "clover_verify_attn_paged_ex")


def clover_kv_commit_paged(k_pages, v_pages, block_table, k_new, v_new, cache_len, path, accept_len, new_cache_len,
                           src_index_out=None, status=None, stream=None):
    """clover_kv_commit into a paged cache (slot L+j of sequence b: page
    block_table[b][(L+j) // page_size], row (L+j) % page_size)."""
    n_pages, Hkv, page_size, D = k_pages.shape
    B, max_pages = block_table.shape
    T = path.shape[1]
    dt = k_pages.dtype
    _check(v_pages, (n_pages, Hkv, page_size, D), dt, "v_pages")
    _check(k_new, (B, T, Hkv, D), dt, "k_new")
    _check(v_new, (B, T, Hkv, D), dt, "v_new")
    _check(block_table, (B, max_pages), torch.int32, "block_table")
    _check(cache_len, (B,), torch.int32, "cache_len")
    _check(path, (B, T), torch.int32, "path")
    _check(accept_len, (B,), torch.int32, "accept_len")
    _check(new_cache_len, (B,), torch.int32, "new_cache_len")
    if src_index_out is not None:
        _check(src_index_out, (B, T), torch.int32, "src_index_out")
    if status is not None:
        _check(status, (1,), torch.int32, "status")
    _dev(k_pages, v_pages, block_table, k_new, v_new, cache_len, path, accept_len, new_cache_len, src_index_out,
         status)
    code = _lib.load().clover_kv_commit_paged(
        _ptr(k_pages), _ptr(v_pages), _ptr(block_table), n_pages, page_size, max_pages, _ptr(k_new), _ptr(v_new),
        _ptr(cache_len), _ptr(path), _ptr(accept_len), _ptr(new_cache_len), _ptr(src_index_out), B, T, Hkv, D,
        dtype_code(dt), _ptr(status), _stream(stream))
    if code != OK:
        raise CloverError(code, "clover_kv_commit_paged")


def clover_kv_commit(k_cache, v_cache, k_new, v_new, cache_len, path, accept_len, new_cache_len,
                     src_index_out=None, status=None, stream=None):
    """Writes the accepted nodes' K/V from k_new/v_new to slots [L, L+a);
    new_cache_len = L + a."""
    B, Hkv, Lcap, D = k_cache.shape
    T = path.shape[1]
    _check(v_cache, (B, Hkv, Lcap, D), k_cache.dtype, "v_cache")
    _check(k_new, (B, T, Hkv, D), k_cache.dtype, "k_new")
    _check(v_new, (B, T, Hkv, D), k_cache.dtype, "v_new")
    _check(cache_len, (B,), torch.int32, "cache_len")
    _check(path, (B, T), torch.int32, "path")
    _check(accept_len, (B,), torch.int32, "accept_len")
    _check(new_cache_len, (B,), torch.int32, "new_cache_len")
    if src_index_out is not None:
        _check(src_index_out, (B, T), torch.int32, "src_index_out")
    if status is not None:
        _check(status, (1,), torch.int32, "status")
    _dev(k_cache, v_cache, k_new, v_new, cache_len, path, accept_len, new_cache_len, src_index_out, status)
    code = _lib.load().clover_kv_commit(
        _ptr(k_cache), _ptr(v_cache), _ptr(k_new), _ptr(v_new), _ptr(cache_len), _ptr(path), _ptr(accept_len),
        _ptr(new_cache_len), _ptr(src_index_out), B, T, Hkv, D, Lcap, dtype_code(k_cache.dtype), _ptr(status),
        _stream(stream))
    if code != OK:
        raise CloverError(code, "clover_kv_commit")


def clover_verify_accept_ex_workspace_size(B, T, V, dtype, flags=0) -> int:
    code = dtype if isinstance(dtype, int) else dtype_code(dtype)
    return int(_lib.load().clover_verify_accept_ex_workspace_size(B, T, V, code, flags))


def clover_verify_accept_ex(logits, cand, parent, argmax_out, path_out, accept_len, bonus_token, workspace,
                            typical=None, commit=None, overlap=False, status=None, stream=None):
    """One launch: the greedy rule, or the typical rule with ``typical`` =
    (temperature, epsilon, delta); with ``commit`` = (k_cache, v_cache, k_new,
    v_new, cache_len, new_cache_len, src_index_out or None) also the commit of
    the accepted K/V; with ``overlap`` as a programmatic dependent of the
    kernel queued before it (see CLOVER_ACCEPT_OVERLAP)."""
    B, T, V = logits.shape
    _check(cand, (B, T), torch.int32, "cand")
    _check(parent, (B, T), torch.int32, "parent")
    _check(argmax_out, (B, T), torch.int32, "argmax_out")
    _check(path_out, (B, T), torch.int32, "path_out")
    _check(accept_len, (B,), torch.int32, "accept_len")
    _check(bonus_token, (B,), torch.int32, "bonus_token")
    if status is not None:
        _check(status, (1,), torch.int32, "status")
    flags = 0
    tau = eps = delta = 0.0
    if typical is not None:
        flags |= _lib.ACCEPT_TYPICAL
        tau, eps, delta = (float(x) for x in typical)
    kc = vc = kn = vn = cl = ncl = src = None
    Hkv = D = Lcap = 0
    if commit is not None:
        flags |= _lib.ACCEPT_COMMIT
        kc, vc, kn, vn, cl, ncl, src = commit
        _, Hkv, Lcap, D = kc.shape
        _check(kc, (B, Hkv, Lcap, D), logits.dtype, "k_cache")
        _check(vc, (B, Hkv, Lcap, D), logits.dtype, "v_cache")
        _check(kn, (B, T, Hkv, D), logits.dtype, "k_new")
        _check(vn, (B, T, Hkv, D), logits.dtype, "v_new")
        _check(cl, (B,), torch.int32, "cache_len")
        _check(ncl, (B,), torch.int32, "new_cache_len")
        if src is not None:
            _check(src, (B, T), torch.int32, "src_index_out")
    if overlap:
        flags |= _lib.ACCEPT_OVERLAP
    _dev(logits, cand, parent, argmax_out, path_out, accept_len, bonus_token, workspace, status, kc, vc, kn, vn,
         cl, ncl, src)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    code = _lib.load().clover_verify_accept_ex(
        _ptr(logits), _ptr(cand), _ptr(parent), B, T, V, dtype_code(logits.dtype), tau, eps, delta, _ptr(kc),
        _ptr(vc), _ptr(kn), _ptr(vn), _ptr(cl), Hkv, D, Lcap, _ptr(argmax_out), _ptr(path_out), _ptr(accept_len),
        _ptr(bonus_token), _ptr(ncl), _ptr(src), _ptr(workspace), ws_bytes, flags, _ptr(status), _stream(stream))
    if code != OK:
        raise CloverError(code, "clover_verify_accept_ex")


def clover_verify_accept_paged_ex(logits, cand, parent, argmax_out, path_out, accept_len, bonus_token, workspace,
                                  commit, block_table, typical=None, overlap=False, status=None, stream=None):
    """clover_verify_accept_ex with the commit into a paged cache: ``commit`` =
    (k_pages, v_pages, k_new, v_new, cache_len, new_cache_len, src_index_out
    or None) with pools [n_pages, Hkv, page_size, D] and ``block_table``
    [B, max_pages]; slot L+j of sequence b is row (L+j) % page_size of page
    block_table[b][(L+j) // page_size]."""
    B, T, V = logits.shape
    _check(cand, (B, T), torch.int32, "cand")
    _check(parent, (B, T), torch.int32, "parent")
    _check(argmax_out, (B, T), torch.int32, "argmax_out")
    _check(path_out, (B, T), torch.int32, "path_out")
    _check(accept_len, (B,), torch.int32, "accept_len")
    _check(bonus_token, (B,), torch.int32, "bonus_token")
    if status is not None:
        _check(status, (1,), torch.int32, "status")
    flags = _lib.ACCEPT_COMMIT
    tau = eps = delta = 0.0
    if typical is not None:
        flags |= _lib.ACCEPT_TYPICAL
        tau, eps, delta = (float(x) for x in typical)
    if overlap:
        flags |= _lib.ACCEPT_OVERLAP
    kp, vp, kn, vn, cl, ncl, src = commit
    n_pages, Hkv, page_size, D = kp.shape
    max_pages = block_table.shape[1]
    dt = logits.dtype
    _check(kp, (n_pages, Hkv, page_size, D), dt, "k_pages")
    _check(vp, (n_pages, Hkv, page_size, D), dt, "v_pages")
    _check(block_table, (B, max_pages), torch.int32, "block_table")
    _check(kn, (B, T, Hkv, D), dt, "k_new")
    _check(vn, (B, T, Hkv, D), dt, "v_new")
    _check(cl, (B,), torch.int32, "cache_len")
    _check(ncl, (B,), torch.int32, "new_cache_len")
    if src is not None:
        _check(src, (B, T), torch.int32, "src_index_out")
    _dev(logits, cand, parent, argmax_out, path_out, accept_len, bonus_token, workspace, status, kp, vp, block_table,
         kn, vn, cl, ncl, src)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    code = _lib.load().clover_verify_accept_paged_ex(
        _ptr(logits), _ptr(cand), _ptr(parent), B, T, V, dtype_code(dt), tau, eps, delta, _ptr(kp), _ptr(vp),
        _ptr(block_table), n_pages, page_size, max_pages, _ptr(kn), _ptr(vn), _ptr(cl), Hkv, D, _ptr(argmax_out),
        _ptr(path_out), _ptr(accept_len), _ptr(bonus_token), _ptr(ncl), _ptr(src), _ptr(workspace), ws_bytes, flags,
        _ptr(status), _stream(stream))
    if code != OK:
        raise CloverError(code, "clover_verify_accept_paged_ex")


_LINEAR_MODES = {"f32": 0, "bf16": 1, "res_silu": 2, "res": 3}


def clover_linear_workspace_size(R, N, K) -> int:
    return int(_lib.load().clover_linear_workspace_size(R, N, K))


def clover_linear(x, w, out, res=None, mode="bf16", workspace=None, status=None, stream=None, pdl=False):
    """out = x . w^T (fp32 accumulation) with the epilogue `mode`: "f32" (fp32
    out), "bf16", "res_silu" (res + silu(.)), "res" (res + .); x [R,K], w [N,K],
    res/out [R,N].  With a workspace of clover_linear_workspace_size bytes a
    layer with few weight tiles splits K over more CTAs.  pdl=True launches it
    as a programmatic dependent of the kernel before it in the stream
    (clover_linear_ex with CLOVER_LINEAR_PDL: that kernel must not write w)."""
    code = _LINEAR_MODES[mode]
    R, K = x.shape
    N = w.shape[0]
    _check(x, (R, K), torch.bfloat16, "x")
    _check(w, (N, K), torch.bfloat16, "w")
    _check(out, (R, N), torch.float32 if code == 0 else torch.bfloat16, "out")
    if code >= 2:
        _check(res, (R, N), torch.bfloat16, "res")
    if status is not None:
        _check(status, (1,), torch.int32, "status")
    _dev(x, w, out, res if code >= 2 else None, workspace, status)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    rc = _lib.load().clover_linear_ex(_ptr(x), _ptr(w), _ptr(res if code >= 2 else None), _ptr(out), R, N, K, code,
                                      _lib.LINEAR_PDL if pdl else 0, _ptr(workspace), ws_bytes, _ptr(status),
                                      _stream(stream))
    if rc != OK:
        raise CloverError(rc, "clover_linear")


def clover_embed_rows(w, tokens, out, status=None, stream=None):
    """out[r] = w[tokens[r]] / ||w[tokens[r]]||_2 (bf16), w [V,H], tokens [R]."""
    V, H = w.shape
    R = tokens.shape[0]
    _check(w, (V, H), torch.bfloat16, "w")
    _check(tokens, (R,), torch.int32, "tokens")
    _check(out, (R, H), torch.bfloat16, "out")
    if status is not None:
        _check(status, (1,), torch.int32, "status")
    _dev(w, tokens, out, status)
    rc = _lib.load().clover_embed_rows(_ptr(w), _ptr(tokens), _ptr(out), R, V, H, _ptr(status), _stream(stream))
    if rc != OK:
        raise CloverError(rc, "clover_embed_rows")


def clover_topk_workspace_size(R, V, k) -> int:
    return int(_lib.load().clover_topk_workspace_size(R, V, k))


def clover_topk(x, k, values, indices, workspace, status=None, stream=None):
    """Top-k of each row of fp32 x [R,V]: values [R,k] fp32, indices [R,k] int32."""
    R, V = x.shape
    _check(x, (R, V), torch.float32, "x")
    _check(values, (R, k), torch.float32, "values")
    _check(indices, (R, k), torch.int32, "indices")
    if status is not None:
        _check(status, (1,), torch.int32, "status")
    _dev(x, values, indices, workspace, status)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    rc = _lib.load().clover_topk(_ptr(x), R, V, k, _ptr(values), _ptr(indices), _ptr(workspace), ws_bytes,
                                 _ptr(status), _stream(stream))
    if rc != OK:
        raise CloverError(rc, "clover_topk")


class DraftHead:
    """One speculative head step of a Clover draft (Section 3), on R rows:
    the previous token's embedding e (its row of the LM-head weight,
    normalised), the attention decoder's h' = h + W_o W_v e (one key and value
    per row, so the softmax weight is 1 and the query projections do not
    enter), the MLP block z = h' + silu(W_1 h'), the shared LM head's fp32
    logits and their top-k.  Weights are bf16 [out, in]; every layer's input
    is bf16.  Owns the activations, the logits and the top-k workspace."""

    def __init__(self, R, H, V, k, device="cuda"):
        dev = torch.device(device)
        bf = dict(dtype=torch.bfloat16, device=dev)
        self.e = torch.empty((R, H), **bf)
        self.v = torch.empty((R, H), **bf)
        self.h = torch.empty((R, H), **bf)
        self.z = torch.empty((R, H), **bf)
        self.logits = torch.empty((R, V), dtype=torch.float32, device=dev)
        self.values = torch.empty((R, k), dtype=torch.float32, device=dev)
        self.indices = torch.empty((R, k), dtype=torch.int32, device=dev)
        self.ws = torch.zeros(max(16, clover_topk_workspace_size(R, V, k)), dtype=torch.uint8, device=dev)
        # the three H x H layers (run one after another) share one split workspace
        self.ws_lin = torch.zeros(max(16, clover_linear_workspace_size(R, H, H)), dtype=torch.uint8, device=dev)
        self.status = torch.zeros(1, dtype=torch.int32, device=dev)
        self.k = k

    def run(self, h, tokens, w_lm, w_v, w_o, w_1, stream=None):
        st = dict(status=self.status, stream=stream)
        # each layer a programmatic dependent of the kernel before it: its
        # set-up and first weight tiles overlap that kernel's end
        clover_embed_rows(w_lm, tokens, self.e, **st)
        clover_linear(self.e, w_v, self.v, mode="bf16", workspace=self.ws_lin, pdl=True, **st)
        clover_linear(self.v, w_o, self.h, res=h, mode="res", workspace=self.ws_lin, pdl=True, **st)
        clover_linear(self.h, w_1, self.z, res=self.h, mode="res_silu", workspace=self.ws_lin, pdl=True, **st)
        clover_linear(self.z, w_lm, self.logits, mode="f32", pdl=True, **st)
        clover_topk(self.logits, self.k, self.values, self.indices, self.ws, **st)


class VerifyStep:
    """Device buffers for repeated verification steps of one shape.

    Owns the two zero-initialised workspaces and the output tensors.  ``run``
    issues the three library calls of one step.  Schedules:

    ``"commit"`` (default): the attention (caches only read) on ``stream`` and,
    at the same time on a side stream, the argmax/acceptance walk followed by
    clover_kv_commit, which writes the accepted K/V from k_new/v_new to slots
    [L, L+a) -- outside what the attention reads -- so no call waits for the
    attention but the end of the step.
    ``"compact"``: the attention appends the tree K/V while the accept call
    runs on the side stream; clover_kv_compact follows on ``stream`` once both
    are done.
    ``"fused"``: two launches on ``stream``: the attention (caches only read),
    then clover_verify_accept_ex with the commit fused in, launched as a
    programmatic dependent of the attention so that it runs beside it on the
    SM space the attention leaves (and completes after it).
    With ``concurrent=False`` the calls run in order on ``stream``.
    ``src_index`` holds tree nodes (commit) or cache slots (compact).
    The outputs are views of one device buffer; ``results`` is the byte range
    holding ``out``, ``path``, ``accept_len``, ``bonus`` and ``new_cache_len``,
    for a read-back in one copy.
    ``accept``: ``"greedy"`` (clover_verify_accept) or ``"typical"``
    (clover_verify_accept_typical with ``temperature``, ``epsilon``, ``delta``).
    ``attn_launch``: how the attention is launched (clover_verify_attn_ex
    flags): ``"ordinary"``; ``"pdl"`` (CLOVER_ATTN_PDL); ``"cache_ready"``
    (with CLOVER_ATTN_CACHE_READY) or ``"inputs_ready"`` (with
    CLOVER_ATTN_INPUTS_READY): the caller's statement that the kernels
    queued before a step do not write its inputs, as when consecutive steps
    serve independent batches.
    ``page_size``: a paged cache (the commit or the fused schedule): ``run``
    then takes the page pools as k_cache/v_cache and the ``block_table``, and
    calls clover_verify_attn_paged(_ex) with clover_kv_commit_paged (commit)
    or clover_verify_accept_paged_ex (fused); ``Lcap`` is the capacity
    page_size * max_pages.
    """

    ATTN_LAUNCHES = {"ordinary": {}, "pdl": dict(pdl=True), "cache_ready": dict(pdl=True, cache_ready=True),
                     "inputs_ready": dict(pdl=True, inputs_ready=True)}

    def __init__(self, B, T, Hq, Hkv, D, Lcap, V, dtype, device="cuda", concurrent=True, schedule="commit",
                 accept="greedy", temperature=1.0, epsilon=0.09, delta=0.3, page_size=None, attn_launch="ordinary"):
        if schedule not in ("commit", "compact", "fused"):
            raise ValueError(f"unknown schedule {schedule!r}")
        if attn_launch not in self.ATTN_LAUNCHES:
            raise ValueError(f"unknown attention launch {attn_launch!r}")
        self.attn_launch = attn_launch
        self._attn_kw = self.ATTN_LAUNCHES[attn_launch]
        if page_size is not None and (schedule == "compact" or Lcap % page_size):
            raise ValueError("a paged cache takes the commit or the fused schedule and a capacity of whole pages")
        self.page_size = page_size
        if accept not in ("greedy", "typical"):
            raise ValueError(f"unknown acceptance rule {accept!r}")
        self.shape = dict(B=B, T=T, Hq=Hq, Hkv=Hkv, D=D, Lcap=Lcap, V=V)
        self.dtype = dtype
        self.schedule = schedule
        self.accept = accept
        self.typical = (float(temperature), float(epsilon), float(delta))
        dev = torch.device(device)
        ws_a = clover_verify_attn_workspace_size(B, T, Hq, Hkv, D, Lcap, dtype)
        ws_b = (clover_verify_accept_typical_workspace_size if accept == "typical"
                else clover_verify_accept_workspace_size)(B, T, V, dtype)
        self.ws_attn = torch.zeros(max(ws_a, 16), dtype=torch.uint8, device=dev) if ws_a else None
        self.ws_accept = torch.zeros(max(ws_b, 16), dtype=torch.uint8, device=dev)
        # The outputs are views of one device buffer (each region 256-byte
        # aligned): out, path, accept_len, bonus, new_cache_len, then argmax
        # and src_index.  `results` is the byte range of the first five, the
        # step's results, so that a caller reads them back with one copy.
        fields = [("out", (B, T, Hq, D), dtype), ("path", (B, T), torch.int32), ("accept_len", (B,), torch.int32),
                  ("bonus", (B,), torch.int32), ("new_cache_len", (B,), torch.int32),
                  ("argmax", (B, T), torch.int32), ("src_index", (B, T), torch.int32)]
        offs, off = [], 0
        for _, shape, dt in fields:
            n = math.prod(shape) * torch.empty((), dtype=dt).element_size()
            offs.append((off, n))
            off = (off + n + 255) // 256 * 256
        self._outputs = torch.empty(off, dtype=torch.uint8, device=dev)
        for (name, shape, dt), (o, n) in zip(fields, offs):
            setattr(self, name, self._outputs[o:o + n].view(dt).view(shape))
        self.results = self._outputs[:offs[4][0] + offs[4][1]]
        i32 = dict(dtype=torch.int32, device=dev)
        self.status = torch.zeros((1,), **i32)
        # the side stream's calls get their own status word so that concurrent
        # calls never update one word at the same time from two streams
        self.status_accept = torch.zeros((1,), **i32)
        # the side stream (argmax/accept, commit) at the highest priority: its
        # CTAs are placed ahead of the attention's when both wait for SM space
        lo, hi = torch.cuda.Stream.priority_range() if hasattr(torch.cuda.Stream, "priority_range") else (0, -1)
        self.side = torch.cuda.Stream(device=dev, priority=min(lo, hi)) if concurrent else None
        self._fork = torch.cuda.Event() if concurrent else None
        self._join = torch.cuda.Event() if concurrent else None

    def device_status(self) -> int:
        return int(self.status.item()) | int(self.status_accept.item())

    def clear_status(self):
        self.status.zero_()
        self.status_accept.zero_()

    def run(self, q, k_new, v_new, k_cache, v_cache, cache_len, parent, cand, logits, scale=0.0,
            stream=None, events=None, block_table=None):
        """One step.  ``events`` (optional, up to six CUDA events) brackets the
        attention (0-1), the commit or compaction (2-3) and the accept call
        (4-5), each on the stream it runs on; a shorter list brackets only the
        calls it has events for."""
        stream = stream if stream is not None else torch.cuda.current_stream()
        commit = self.schedule == "commit"
        side = self.side if self.side is not None else stream
        n_ev = len(events) if events else 0

        def ev(i, st):
            if i < n_ev:
                events[i].record(st)

        if self.schedule == "fused":
            ev(0, stream)
            if self.page_size is not None:
                clover_verify_attn_paged(q, k_new, v_new, k_cache, v_cache, block_table, cache_len, parent,
                                         self.out, scale=scale, workspace=self.ws_attn, status=self.status,
                                         stream=stream, **self._attn_kw)
            else:
                clover_verify_attn(q, k_new, v_new, k_cache, v_cache, cache_len, parent, self.out, scale=scale,
                                   workspace=self.ws_attn, status=self.status, stream=stream, append=False,
                                   **self._attn_kw)
            timed_end = n_ev > 1 and self.side is not None
            if timed_end:
                # the attention's end, recorded on the side stream: nothing is
                # queued on `stream` between the attention and the accept call
                self._fork.record(stream)
                self.side.wait_event(self._fork)
                events[1].record(self.side)
                self._join.record(self.side)
            elif n_ev > 1:
                events[1].record(stream)
            typical = self.typical if self.accept == "typical" else None
            commit_args = (k_cache, v_cache, k_new, v_new, cache_len, self.new_cache_len, self.src_index)
            if self.page_size is not None:
                clover_verify_accept_paged_ex(logits, cand, parent, self.argmax, self.path, self.accept_len,
                                              self.bonus, self.ws_accept, commit_args, block_table, typical=typical,
                                              overlap=self.side is not None, status=self.status_accept,
                                              stream=stream)
            else:
                clover_verify_accept_ex(logits, cand, parent, self.argmax, self.path, self.accept_len, self.bonus,
                                        self.ws_accept, typical=typical, commit=commit_args,
                                        overlap=self.side is not None, status=self.status_accept, stream=stream)
            if timed_end:
                stream.wait_event(self._join)
            return

        if self.side is not None:
            self._fork.record(stream)
            self.side.wait_event(self._fork)
        ev(0, stream)
        if self.page_size is not None:
            clover_verify_attn_paged(q, k_new, v_new, k_cache, v_cache, block_table, cache_len, parent, self.out,
                                     scale=scale, workspace=self.ws_attn, status=self.status, stream=stream,
                                     **self._attn_kw)
        else:
            clover_verify_attn(q, k_new, v_new, k_cache, v_cache, cache_len, parent, self.out, scale=scale,
                               workspace=self.ws_attn, status=self.status, stream=stream, append=not commit,
                               **self._attn_kw)
        ev(1, stream)
        ev(4, side)
        if self.accept == "typical":
            clover_verify_accept_typical(logits, cand, parent, *self.typical, self.argmax, self.path,
                                         self.accept_len, self.bonus, self.ws_accept, status=self.status_accept,
                                         stream=side)
        else:
            clover_verify_accept(logits, cand, parent, self.argmax, self.path, self.accept_len, self.bonus,
                                 self.ws_accept, status=self.status_accept, stream=side)
        ev(5, side)
        if commit:
            ev(2, side)
            if self.page_size is not None:
                clover_kv_commit_paged(k_cache, v_cache, block_table, k_new, v_new, cache_len, self.path,
                                       self.accept_len, self.new_cache_len, self.src_index, status=self.status_accept,
                                       stream=side)
            else:
                clover_kv_commit(k_cache, v_cache, k_new, v_new, cache_len, self.path, self.accept_len,
                                 self.new_cache_len, self.src_index, status=self.status_accept, stream=side)
            ev(3, side)
            if self.side is not None:
                self._join.record(self.side)
                stream.wait_event(self._join)
        else:
            if self.side is not None:
                self._join.record(self.side)
                stream.wait_event(self._join)
            ev(2, stream)
            clover_kv_compact(k_cache, v_cache, cache_len, self.path, self.accept_len, self.new_cache_len,
                              self.src_index, status=self.status, stream=stream)
            ev(3, stream)
