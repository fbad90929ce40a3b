// Shared device helpers and launch-argument structs of the verification kernels.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "clover_verify.h"
#include "ctx_host.cuh"

namespace clover {

constexpr int kMaxTreeNodes = 128;  // ancestor masks of two 64-bit words per node
constexpr int kMaskWords = 2;

// Everything clover_verify_attn's kernels need, already validated on the host.
struct AttnArgs {
    const void *q, *k_new, *v_new;
    void *k_cache, *v_cache;
    const int32_t *cache_len, *parent;
    void *out;
    int B, T, Hq, Hkv, D, Lcap, G;
    int dtype;             // clover_dtype
    float scale_log2;      // softmax scale * log2(e): scores are kept in base 2
    int rows;              // T * G query rows per KV head
    int row_tile;          // rows per CTA
    int row_tiles;         // ceil(rows / row_tile)
    int n_split;           // cache key ranges per (sequence, KV head, row tile)
    int slot_rows;         // rows of one partial-result slot (<= row_tile)
    int append;            // write k_new/v_new to cache slots [L, L+T) (0: the caches are only read)
    // paged cache (block_table != nullptr): k_cache/v_cache are page pools
    // [n_pages, Hkv, page_size, D]; slot s of sequence b is row s % page_size
    // of page block_table[b * max_pages + s / page_size]; Lcap = page_size * max_pages
    const int32_t *block_table;
    int page_size, page_shift, max_pages, n_pages;
    // split partials (n_split > 1).  FMA kernel: part_o [B, Hkv, row_tiles,
    // n_split, slot_rows, D] and part_ml [..., slot_rows, 2] (max, sum);
    // tensor-core kernel: part_o [B, Hkv, row_tiles, n_split, slot_rows, D + 4]
    // (O, then max and sum), part_ml unused
    float *part_o;
    float *part_ml;
    unsigned *counters;    // [B, Hkv, row_tiles] arrival counters, zero between calls
    int32_t *status;
    int pdl;               // launched as a programmatic dependent of the preceding kernel
    int cache_early;       // caches, lengths and block table may be read before that kernel completes
    int inputs_early;      // every input may be read before that kernel completes (only writes wait)
    size_t ws_bytes;       // workspace bytes (index checks of CLOVER_CHECKED builds)
};

// One acceptance call (clover_verify_accept, _typical or _ex), validated on
// the host.
struct AcceptCall {
    const void *logits;
    const int32_t *cand, *parent;
    int B, T, V, dtype;
    int32_t *argmax_out, *path_out, *accept_len, *bonus;
    void *workspace;
    int32_t *status;
    bool typical;                   // typical rule with the three values below
    float y_scale, log2_eps, log2_delta;
    bool commit;                    // also commit the accepted K/V (from k_new/v_new)
    void *k_cache, *v_cache;
    const void *k_new, *v_new;
    const int32_t *cache_len;
    int32_t *new_cache_len, *src_index;
    int Hkv, D, Lcap;
    // paged cache (block_table != nullptr): k_cache/v_cache are page pools
    // [n_pages, Hkv, page_size, D]; slot s of sequence b is row s % page_size
    // of page block_table[b * max_pages + s / page_size]
    const int32_t *block_table;
    int page_size, max_pages, n_pages;
    bool after_prior;               // launch as a programmatic dependent of the preceding kernel
};

// Programmatic dependent launch: lets the next kernel in the stream, if it
// was launched as a programmatic dependent, start as soon as every CTA of this
// grid has issued this (the dependent then waits for this grid's completion
// itself where it has to).  Without such a dependent it has no effect.
__device__ __forceinline__ void allow_dependent_launch() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Waits until the grids this one was launched as a programmatic dependent of
// have completed and their memory operations are visible; returns at once in a
// grid launched the ordinary way.
__device__ __forceinline__ void wait_prerequisite_grids() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
}

__device__ __forceinline__ void report(int32_t *status, int bits) {
    if (status) atomicOr(status, bits);
}

// Index checks of a CLOVER_CHECKED build: CLOVER_IN(status, i, n) is true
// when 0 <= i < n; otherwise it raises CLOVER_ERR_CHECK in the status word
// (never traps) and is false, and the call site skips the access it guards.
// Ordinary builds compile it to true.
#ifdef CLOVER_CHECKED
__device__ __forceinline__ bool check_in(int32_t *status, long long i, long long n) {
    if (i >= 0 && i < n) return true;
    report(status, CLOVER_ERR_CHECK);
    return false;
}
#define CLOVER_IN(status, i, n) ::clover::check_in((status), (long long)(i), (long long)(n))
#else
#define CLOVER_IN(status, i, n) true
#endif

// Page of cache slot `slot` (< cache_len) of sequence b in a paged cache; an
// id outside [0, n_pages) is reported and replaced by page 0, so that every
// access stays inside the pool (the result is then unspecified).
__device__ __forceinline__ int cache_page(const AttnArgs &a, int b, int slot) {
    const int p = __ldg(a.block_table + (size_t)b * a.max_pages + (slot >> a.page_shift));
    if (p < 0 || p >= a.n_pages) {
        report(a.status, CLOVER_ERR_INVALID_ARG);
        return 0;
    }
    return p;
}

__device__ __forceinline__ float bf16_bits_to_float(uint16_t h) {
    return __uint_as_float(static_cast<uint32_t>(h) << 16);
}

// Eight consecutive elements (16 bytes of bf16 or two 16-byte loads of fp32) -> fp32.
template <typename T>
struct Vec8;

template <>
struct Vec8<float> {
    static __device__ __forceinline__ void load(const float *p, float (&v)[8]) {
        const float4 a = *reinterpret_cast<const float4 *>(p);
        const float4 b = *reinterpret_cast<const float4 *>(p + 4);
        v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
        v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
    }
};

template <>
struct Vec8<__nv_bfloat16> {
    static __device__ __forceinline__ void load(const __nv_bfloat16 *p, float (&v)[8]) {
        const uint4 a = *reinterpret_cast<const uint4 *>(p);
        const uint32_t w[4] = {a.x, a.y, a.z, a.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            v[2 * k] = __uint_as_float(w[k] << 16);
            v[2 * k + 1] = __uint_as_float(w[k] & 0xFFFF0000u);
        }
    }
};

__device__ __forceinline__ float to_float(float x) { return x; }
__device__ __forceinline__ float to_float(__nv_bfloat16 x) { return __bfloat162float(x); }

template <typename T>
__device__ __forceinline__ T from_float(float x);
template <>
__device__ __forceinline__ float from_float<float>(float x) { return x; }
template <>
__device__ __forceinline__ __nv_bfloat16 from_float<__nv_bfloat16>(float x) { return __float2bfloat16_rn(x); }

// Ancestor-or-self bitmasks by pointer jumping in one warp's registers: lane l
// owns nodes l + 32 k (k < NS, T <= 32 NS) with parents parent[k]; node n is
// bit n & 63 of word n >> 6.  After round r a node's mask covers its 2^r
// nearest ancestors, so log2(32 NS) rounds cover every depth.  The parents must
// form a valid tree.
template <int NS>
__device__ __forceinline__ void tree_masks_jump(const int (&parent)[NS], int T, uint64_t (&m)[NS][kMaskWords]) {
    const int lane = threadIdx.x & 31;
    int up[NS];
#pragma unroll
    for (int k = 0; k < NS; ++k) {
        const int i = lane + 32 * k;
#pragma unroll
        for (int w = 0; w < kMaskWords; ++w) m[k][w] = (i < T && (i >> 6) == w) ? (1ull << (i & 63)) : 0ull;
        up[k] = (i < T && i > 0) ? parent[k] : -1;
    }
    constexpr int kRounds = NS <= 2 ? 6 : 7;
#pragma unroll 1
    for (int round = 0; round < kRounds; ++round) {
        uint64_t nm[NS][kMaskWords];
        int nu[NS];
#pragma unroll
        for (int k = 0; k < NS; ++k) {
            const int u = up[k] < 0 ? 0 : up[k];
            // mask and pointer of node u: lane u & 31, slot u >> 5
            uint64_t mu[kMaskWords] = {0ull, 0ull};
            int uu = -1;
#pragma unroll
            for (int sl = 0; sl < NS; ++sl) {
                const int us = __shfl_sync(0xffffffffu, up[sl], u & 31);
#pragma unroll
                for (int w = 0; w < kMaskWords; ++w) {
                    const uint64_t ms = __shfl_sync(0xffffffffu, m[sl][w], u & 31);
                    if ((u >> 5) == sl) mu[w] = ms;
                }
                if ((u >> 5) == sl) uu = us;
            }
#pragma unroll
            for (int w = 0; w < kMaskWords; ++w) nm[k][w] = up[k] < 0 ? m[k][w] : (m[k][w] | mu[w]);
            nu[k] = up[k] < 0 ? -1 : uu;
        }
#pragma unroll
        for (int k = 0; k < NS; ++k) {
#pragma unroll
            for (int w = 0; w < kMaskWords; ++w) m[k][w] = nm[k][w];
            up[k] = nu[k];
        }
    }
}

// The parent array of a tree, read by one warp: lane l holds node l + 32k in
// p[k] (-1 past T).  Split from the mask computation so that a kernel can
// issue these loads at its start, ahead of its bulk traffic.
__device__ __forceinline__ void tree_parents_load(const int32_t *parent, int T, int (&p)[4]) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const int i = lane + 32 * k;
        p[k] = (i < T && (k < 2 || T > 64)) ? __ldg(parent + i) : -1;
    }
}

// Ancestor-or-self bitmask of every tree node into anc[node * kMaskWords + w],
// computed by one warp from the parents loaded by tree_parents_load.  Invalid
// parent arrays set *bad (masks are then only self bits and must not be trusted).
template <int NS>
__device__ __forceinline__ void tree_masks_from(const int (&pl)[4], int T, uint64_t *anc, bool *bad) {
    const int lane = threadIdx.x & 31;
    int p[NS];
    bool invalid = false;
#pragma unroll
    for (int k = 0; k < NS; ++k) {
        const int i = lane + 32 * k;
        p[k] = -1;
        if (i < T) {
            p[k] = pl[k];
            if (i == 0 ? (p[k] != -1) : (p[k] < 0 || p[k] >= i)) invalid = true;
        }
    }
    const bool any_bad = __any_sync(0xffffffffu, invalid);
    uint64_t m[NS][kMaskWords];
    if (any_bad) {
#pragma unroll
        for (int k = 0; k < NS; ++k) {
            const int i = lane + 32 * k;
#pragma unroll
            for (int w = 0; w < kMaskWords; ++w) m[k][w] = (i < T && (i >> 6) == w) ? (1ull << (i & 63)) : 0ull;
        }
    } else {
        tree_masks_jump<NS>(p, T, m);
    }
#pragma unroll
    for (int k = 0; k < NS; ++k) {
        const int i = lane + 32 * k;
        if (i < T) {
#pragma unroll
            for (int w = 0; w < kMaskWords; ++w) anc[i * kMaskWords + w] = m[k][w];
        }
    }
    if (lane == 0) *bad = any_bad;
}

__device__ __forceinline__ void tree_masks_build(const int (&p)[4], int T, uint64_t *anc, bool *bad) {
    if (T <= 64) tree_masks_from<2>(p, T, anc, bad);
    else tree_masks_from<4>(p, T, anc, bad);
}

__device__ __forceinline__ void tree_masks_warp(const int32_t *parent, int T, uint64_t *anc, bool *bad) {
    int p[4];
    tree_parents_load(parent, T, p);
    tree_masks_build(p, T, anc, bad);
}

// Ancestor-or-self bitmasks by walking each node's root path, in one warp:
// lane l holds the parents of nodes l + 32 k in p[k] (tree_parents_load's
// layout) and copies them to `par` in shared memory; then node i's mask
// collects i and every node on the way up to the root (depth(i) + 1 steps,
// as parent[i] < i).  Node n is bit n & 63 of word n >> 6 of anc[i].  An
// invalid parent array (parent[0] != -1, or parent[i] outside [0, i)) sets
// *bad and leaves only the self bits.  Small code, for kernels that run it
// once per launch; its time grows with the tree's depth.
static __device__ __noinline__ void tree_masks_walk(const int (&p)[4], int T, int *par, uint64_t *anc, bool *bad) {
    const int lane = threadIdx.x & 31;
    bool invalid = false;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const int i = lane + 32 * k;
        if (i < T) {
            par[i] = p[k];
            if (i == 0 ? (p[k] != -1) : (p[k] < 0 || p[k] >= i)) invalid = true;
        }
    }
    const bool any_bad = __any_sync(0xffffffffu, invalid);
    __syncwarp();
#pragma unroll 1
    for (int i = lane; i < T; i += 32) {
        uint64_t m[kMaskWords] = {0ull, 0ull};
        int j = i;
        do {
            m[j >> 6] |= 1ull << (j & 63);
            j = any_bad ? -1 : par[j];
        } while (j >= 0);
        anc[i * kMaskWords] = m[0];
        anc[i * kMaskWords + 1] = m[1];
    }
    if (lane == 0) *bad = any_bad;
}

// Raises a kernel's dynamic shared memory limit once per CUDA context.
// Launchers call it before every launch; only the first call in a context
// reaches the driver, so launches captured into a CUDA graph after a first
// eager launch issue no attribute call.  `done` holds, per device ordinal, the
// context in which the attribute was last set: a reset device (or another
// context on it) starts without the attribute and gets it again.
template <typename Kernel>
cudaError_t ensure_smem_attr(Kernel kernel, size_t bytes, unsigned long long (&done)[64]) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const unsigned long long ctx = current_context_id();
    if (ctx != 0 && dev >= 0 && dev < 64 && done[dev] == ctx) return cudaSuccess;
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    if (e == cudaSuccess && dev >= 0 && dev < 64) done[dev] = ctx;
    return e;
}

}  // namespace clover
