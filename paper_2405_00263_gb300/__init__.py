"""GB300 (sm_103a) verification step of Clover-style tree speculative decoding.

The compute lives in libclover_verify.so (CUDA kernels behind a C ABI, see
include/clover_verify.h); this package builds it in-tree and binds it with the
same names.  There is no CPU fallback.
"""

from .api import (  # noqa: F401
    BF16, F32, OK, CloverError, DraftHead, VerifyStep, clover_abi_version, clover_build_flags, clover_embed_rows,
    clover_linear,
    clover_linear_workspace_size,
    clover_topk, clover_topk_workspace_size, clover_kv_commit, clover_kv_commit_paged,
    clover_kv_compact, clover_verify_attn_paged, clover_verify_attn_paged_workspace_size,
    clover_verify_accept, clover_verify_accept_ex, clover_verify_accept_ex_workspace_size,
    clover_verify_accept_typical, clover_verify_accept_typical_workspace_size,
    clover_verify_accept_workspace_size, clover_verify_attn, clover_verify_attn_noalloc,
    clover_verify_attn_workspace_size, dtype_code)
