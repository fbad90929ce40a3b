"""ctypes loader of libclover_verify.so and the raw C signatures.

The library is built in-tree (``paper_2405_00263_gb300/_build``) by
``paper_2405_00263_gb300.build.build()``.  There is no fallback: if the shared
library is missing, loading raises.
"""

from __future__ import annotations

import ctypes
import os
import threading

from . import build as _build

_lock = threading.Lock()
_lib = None

# Every symbol include/clover_verify.h declares.
EXPORTS = (
    "clover_abi_version",
    "clover_build_flags",
    "clover_status_string",
    "clover_verify_attn_workspace_size",
    "clover_verify_attn",
    "clover_verify_attn_ex",
    "clover_verify_accept_workspace_size",
    "clover_verify_accept",
    "clover_verify_accept_typical_workspace_size",
    "clover_verify_accept_typical",
    "clover_verify_accept_ex_workspace_size",
    "clover_verify_accept_ex",
    "clover_kv_compact",
    "clover_kv_commit",
    "clover_verify_attn_noalloc",
    "clover_verify_attn_paged_workspace_size",
    "clover_verify_attn_paged",
    "clover_verify_attn_paged_ex",
    "clover_verify_accept_paged_ex",
    "clover_kv_commit_paged",
    "clover_linear_workspace_size",
    "clover_linear",
    "clover_linear_ex",
    "clover_embed_rows",
    "clover_topk_workspace_size",
    "clover_topk",
)

# Flags of clover_verify_attn_ex (CLOVER_ATTN_* in include/clover_verify.h).
ATTN_NO_APPEND = 1
ATTN_PDL = 2
ATTN_CACHE_READY = 4
ATTN_INPUTS_READY = 8

# Flags of clover_verify_accept_ex (CLOVER_ACCEPT_* in include/clover_verify.h).
ACCEPT_TYPICAL = 1
ACCEPT_COMMIT = 2
ACCEPT_OVERLAP = 4

# Epilogues of clover_linear (CLOVER_LINEAR_* in include/clover_verify.h).
LINEAR_F32 = 0
LINEAR_BF16 = 1
LINEAR_RES_SILU = 2
LINEAR_RES = 3
# Launch flag of clover_linear_ex (CLOVER_LINEAR_PDL).
LINEAR_PDL = 1

# Bytes of the static scratch buffer behind clover_verify_attn_noalloc
# (CLOVER_NOALLOC_SCRATCH_BYTES in include/clover_verify.h).
NOALLOC_SCRATCH_BYTES = 8 << 20


# Bit of clover_build_flags(): the library was built with -DCLOVER_CHECKED.
BUILD_CHECKED = 1

# Set to 1 to load the checked build (``build(checked=True)``) instead.
CHECKED_ENV = "CLOVER_VERIFY_CHECKED"


def library_path() -> str:
    return _build.CHECKED_LIB if os.environ.get(CHECKED_ENV) == "1" else _build.LIB


def load(build_if_missing: bool = False):
    """The loaded CDLL with argtypes set.  Raises if the library was not built."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        path = library_path()
        if not os.path.exists(path):
            if not build_if_missing:
                raise RuntimeError(
                    f"libclover_verify.so is not built ({path}); run "
                    "`python -c 'import __graft_entry__ as g; g.build()'` first")
            _build.build(checked=path == _build.CHECKED_LIB)
        lib = ctypes.CDLL(path)
        P, I, Z, F = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t, ctypes.c_float
        lib.clover_abi_version.argtypes = []
        lib.clover_abi_version.restype = I
        lib.clover_build_flags.argtypes = []
        lib.clover_build_flags.restype = I
        lib.clover_status_string.argtypes = [I]
        lib.clover_status_string.restype = ctypes.c_char_p
        lib.clover_verify_attn_workspace_size.argtypes = [I, I, I, I, I, I, I]
        lib.clover_verify_attn_workspace_size.restype = Z
        lib.clover_verify_attn.argtypes = [P, P, P, P, P, P, P, P, I, I, I, I, I, I, I, F, P, Z, P, P]
        lib.clover_verify_attn.restype = I
        lib.clover_verify_attn_ex.argtypes = [P, P, P, P, P, P, P, P, I, I, I, I, I, I, I, F, P, Z, P, P,
                                              ctypes.c_uint32]
        lib.clover_verify_attn_ex.restype = I
        lib.clover_verify_accept_workspace_size.argtypes = [I, I, I, I]
        lib.clover_verify_accept_workspace_size.restype = Z
        lib.clover_verify_accept.argtypes = [P, P, P, I, I, I, I, P, P, P, P, P, Z, P, P]
        lib.clover_verify_accept.restype = I
        lib.clover_verify_accept_typical_workspace_size.argtypes = [I, I, I, I]
        lib.clover_verify_accept_typical_workspace_size.restype = Z
        lib.clover_verify_accept_typical.argtypes = [P, P, P, I, I, I, I, ctypes.c_double, ctypes.c_double,
                                                     ctypes.c_double, P, P, P, P, P, Z, P, P]
        lib.clover_verify_accept_typical.restype = I
        lib.clover_verify_accept_ex_workspace_size.argtypes = [I, I, I, I, ctypes.c_uint32]
        lib.clover_verify_accept_ex_workspace_size.restype = Z
        Dd = ctypes.c_double
        lib.clover_verify_accept_ex.argtypes = [P, P, P, I, I, I, I, Dd, Dd, Dd, P, P, P, P, P, I, I, I,
                                                P, P, P, P, P, P, P, Z, ctypes.c_uint32, P, P]
        lib.clover_verify_accept_ex.restype = I
        lib.clover_kv_compact.argtypes = [P, P, P, P, P, P, P, I, I, I, I, I, I, P, P]
        lib.clover_kv_compact.restype = I
        lib.clover_kv_commit.argtypes = [P, P, P, P, P, P, P, P, P, I, I, I, I, I, I, P, P]
        lib.clover_kv_commit.restype = I
        lib.clover_verify_attn_noalloc.argtypes = [P, P, P, P, P, P, P, P, I, I, I, I, I, I, I, F, P, P]
        lib.clover_verify_attn_noalloc.restype = I
        lib.clover_verify_attn_paged_workspace_size.argtypes = [I, I, I, I, I, I, I, I]
        lib.clover_verify_attn_paged_workspace_size.restype = Z
        lib.clover_verify_attn_paged.argtypes = [P, P, P, P, P, P, I, I, I, P, P, P, I, I, I, I, I, I, F, P, Z,
                                                 P, P]
        lib.clover_verify_attn_paged.restype = I
        lib.clover_verify_attn_paged_ex.argtypes = lib.clover_verify_attn_paged.argtypes + [ctypes.c_uint32]
        lib.clover_verify_attn_paged_ex.restype = I
        lib.clover_verify_accept_paged_ex.argtypes = [P, P, P, I, I, I, I, Dd, Dd, Dd, P, P, P, I, I, I, P, P, P, I,
                                                      I, P, P, P, P, P, P, P, Z, ctypes.c_uint32, P, P]
        lib.clover_verify_accept_paged_ex.restype = I
        lib.clover_kv_commit_paged.argtypes = [P, P, P, I, I, I, P, P, P, P, P, P, P, I, I, I, I, I, P, P]
        lib.clover_kv_commit_paged.restype = I
        lib.clover_linear_workspace_size.argtypes = [I, I, I]
        lib.clover_linear_workspace_size.restype = Z
        lib.clover_linear.argtypes = [P, P, P, P, I, I, I, I, P, Z, P, P]
        lib.clover_linear.restype = I
        lib.clover_linear_ex.argtypes = [P, P, P, P, I, I, I, I, ctypes.c_uint, P, Z, P, P]
        lib.clover_linear_ex.restype = I
        lib.clover_embed_rows.argtypes = [P, P, P, I, I, I, P, P]
        lib.clover_embed_rows.restype = I
        lib.clover_topk_workspace_size.argtypes = [I, I, I]
        lib.clover_topk_workspace_size.restype = Z
        lib.clover_topk.argtypes = [P, I, I, I, P, P, P, Z, P, P]
        lib.clover_topk.restype = I
        _lib = lib
        return lib
