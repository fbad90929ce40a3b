// extern "C" entry points of libclover_verify.so: host-side validation, launch
// planning and dispatch to the kernels.  Declarations and the full contract of
// each call are in include/clover_verify.h.
#include <math.h>

#include <mutex>

#include <nvtx3/nvToolsExt.h>

#include "common.cuh"

namespace clover {
int fma_row_tile();
int tc_row_tile();
int tc_max_splits();
cudaError_t launch_tree_attn_fma(const AttnArgs &a, cudaStream_t stream);
cudaError_t launch_tree_attn_tc(const AttnArgs &a, cudaStream_t stream);
bool tc_pair_eligible(const AttnArgs &a);
cudaError_t launch_tree_attn_tc_pair(const AttnArgs &a, cudaStream_t stream);
void accept_plan(int B, int T, int V, int dtype, bool typical, int resident, int *n_chunks, int *chunk);
size_t accept_workspace_bytes(int B, int T, int V, int dtype);
size_t accept_typical_workspace_bytes(int B, int T, int V, int dtype);
cudaError_t launch_linear_tc(const void *x, const void *w, const void *res, void *out, int R, int N, int K, int mode,
                             void *workspace, size_t ws_bytes, int32_t *status, bool pdl, cudaStream_t stream);
size_t linear_workspace_bytes(int R, int N, int K);
size_t topk_workspace_bytes(int R, int V, int k);
int topk_max_k();
cudaError_t launch_topk(const float *x, int R, int V, int k, float *values, int32_t *indices, void *workspace,
                        int32_t *status, cudaStream_t stream);
cudaError_t launch_embed_rows(const void *w, const int32_t *tokens, void *e, int R, int V, int H, int32_t *status,
                              cudaStream_t stream);
cudaError_t launch_accept_call(const AcceptCall &c, cudaStream_t stream);
cudaError_t launch_kv_compact(void *k_cache, void *v_cache, const void *k_new, const void *v_new,
                              const int32_t *cache_len, const int32_t *path, const int32_t *accept_len,
                              int32_t *new_cache_len, int32_t *src_index, int B, int T, int Hkv, int D, int Lcap,
                              int dtype, int32_t *status, cudaStream_t stream, const int32_t *block_table = nullptr,
                              int page_size = 0, int max_pages = 0, int n_pages = 0);

namespace {

constexpr int kAbiVersion = 1;
constexpr int kSms = 152;                  // SMs of a GB300 (planning constant; any GPU runs the plan)
constexpr int kTargetAttnCtas = 2 * kSms;  // FMA path: two resident CTAs per SM
constexpr int kMinKeysPerSplit = 256;
constexpr int kMaxSplits = 64;

// CTAs an inputs-ready attention launch aims for: about a fifth of the SMs
// (see run_attn).
constexpr long kChainCtas = kSms / 5;

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Workspace layout: [arrival counters][split partials (O rows; FMA: then
// max and sum)], each part rounded up to 256 bytes.
struct AttnPlan {
    bool tc;                 // tensor-core (tcgen05) kernel, else the FMA kernel
    int row_tile, row_tiles, n_split, slot_rows;
    size_t o_bytes, ml_bytes, counter_bytes, total;
};

clover_status check_attn_sizes(int B, int T, int Hq, int Hkv, int D, int Lcap, int dtype) {
    if (B < 0 || T < 1 || Hq < 1 || Hkv < 1 || Lcap < 1) return CLOVER_ERR_INVALID_ARG;
    if (dtype != CLOVER_F32 && dtype != CLOVER_BF16) return CLOVER_ERR_INVALID_ARG;
    if (T > kMaxTreeNodes || (D != 64 && D != 128) || Hq % Hkv != 0) return CLOVER_ERR_UNSUPPORTED;
    if (Lcap < T) return CLOVER_ERR_INVALID_ARG;
    if (B > 65535 || Hkv > 65535) return CLOVER_ERR_UNSUPPORTED;
    if ((unsigned long long)B * T * Hq >= (1ull << 32)) return CLOVER_ERR_UNSUPPORTED;   // output rows: 32-bit ids
    return CLOVER_OK;
}

// Kernel choice, split count and workspace layout for one shape.  bf16 runs on
// the tensor cores for any number of query rows: even a 4-row tile is bound by
// HBM there, as the MMA cost of a 128-key tile (about 0.8 us) stays below its
// HBM time.  One CTA per SM: the cache keys of a (sequence, head, row tile)
// split over as many CTAs as fill the SMs in one wave (at most tc_max_splits,
// at least kMinKeysPerSplit keys each), partials merged through the workspace
// (rows of D + 4 floats).  fp32 runs on the FMA kernel with two CTAs per SM
// and merges splits through the workspace too.
AttnPlan plan_attn(int B, int T, int Hq, int Hkv, int D, int Lcap, int dtype) {
    AttnPlan p;
    const int G = Hq / Hkv;
    const int rows = T * G;
    const long Bp = B > 0 ? B : 1;
    const int by_len = (Lcap + kMinKeysPerSplit - 1) / kMinKeysPerSplit;
    int n;
    p.tc = (dtype == CLOVER_BF16);
    if (p.tc) {
        p.row_tile = tc_row_tile();
        p.row_tiles = (rows + p.row_tile - 1) / p.row_tile;
        p.slot_rows = rows < p.row_tile ? rows : p.row_tile;
        const long base = Bp * Hkv * p.row_tiles;
        n = (int)(kSms / base);
        if (n > tc_max_splits()) n = tc_max_splits();
        if (n > by_len) n = by_len;
        if (n < 1) n = 1;
        p.n_split = n;
        const size_t heads = (size_t)Bp * Hkv * p.row_tiles;
        if (n == 1) {
            p.o_bytes = p.ml_bytes = p.counter_bytes = p.total = 0;
        } else {
            p.o_bytes = round_up(sizeof(float) * heads * n * p.slot_rows * (D + 4), 256);
            p.ml_bytes = 0;
            p.counter_bytes = round_up(sizeof(unsigned) * heads, 256);
            p.total = p.o_bytes + p.counter_bytes;
        }
        return p;
    } else {
        p.row_tile = fma_row_tile();
        p.row_tiles = (rows + p.row_tile - 1) / p.row_tile;
        p.slot_rows = p.row_tile;
        const long base = Bp * Hkv * p.row_tiles;
        n = (int)((kTargetAttnCtas + base - 1) / base);
    }
    if (n > by_len) n = by_len;
    if (n > kMaxSplits) n = kMaxSplits;
    if (n < 1) n = 1;
    p.n_split = n;
    const size_t heads = (size_t)Bp * Hkv * p.row_tiles;
    if (n == 1) {
        p.o_bytes = p.ml_bytes = p.counter_bytes = p.total = 0;
    } else {
        p.o_bytes = round_up(sizeof(float) * heads * n * p.slot_rows * D, 256);
        p.ml_bytes = round_up(sizeof(float) * heads * n * p.slot_rows * 2, 256);
        p.counter_bytes = round_up(sizeof(unsigned) * heads, 256);
        p.total = p.o_bytes + p.ml_bytes + p.counter_bytes;
    }
    return p;
}

clover_status from_cuda(cudaError_t e) { return e == cudaSuccess ? CLOVER_OK : CLOVER_ERR_CUDA; }

// An NVTX range (named after the entry point) around each call, so that a
// profiler's timeline shows the library's host-side calls; without a tool
// attached it costs a few nanoseconds.
struct NvtxRange {
    explicit NvtxRange(const char *name) { nvtxRangePushA(name); }
    ~NvtxRange() { nvtxRangePop(); }
    NvtxRange(const NvtxRange &) = delete;
    NvtxRange &operator=(const NvtxRange &) = delete;
};

}  // namespace
}  // namespace clover

using namespace clover;

namespace {

// Checks shared by clover_kv_compact and clover_kv_commit (k_new == v_new ==
// nullptr for the compaction).
clover_status check_commit(void *k_cache, void *v_cache, const void *k_new, const void *v_new,
                           const int32_t *cache_len, const int32_t *path, const int32_t *accept_len,
                           int32_t *new_cache_len, int B, int T, int Hkv, int D, int Lcap, clover_dtype dtype,
                           bool from_new) {
    if (B < 0 || T < 1 || Hkv < 1 || Lcap < 1) return CLOVER_ERR_INVALID_ARG;
    if (dtype != CLOVER_F32 && dtype != CLOVER_BF16) return CLOVER_ERR_INVALID_ARG;
    if (T > kMaxTreeNodes || (D != 64 && D != 128)) return CLOVER_ERR_UNSUPPORTED;
    if (Lcap < T) return CLOVER_ERR_INVALID_ARG;
    if (B > 65535 || Hkv > 65535) return CLOVER_ERR_UNSUPPORTED;
    if (B == 0) return CLOVER_OK;
    if (!k_cache || !v_cache || !cache_len || !path || !accept_len || !new_cache_len) return CLOVER_ERR_INVALID_ARG;
    if (!aligned16(k_cache) || !aligned16(v_cache)) return CLOVER_ERR_INVALID_ARG;
    if (from_new && (!k_new || !v_new || !aligned16(k_new) || !aligned16(v_new))) return CLOVER_ERR_INVALID_ARG;
    const uintptr_t a0 = reinterpret_cast<uintptr_t>(cache_len), a1 = a0 + sizeof(int32_t) * (size_t)B;
    const uintptr_t b0 = reinterpret_cast<uintptr_t>(new_cache_len), b1 = b0 + sizeof(int32_t) * (size_t)B;
    if (a0 < b1 && b0 < a1) return CLOVER_ERR_INVALID_ARG;      // lengths are read by every CTA: no aliasing
    return CLOVER_OK;
}

// Host checks shared by the acceptance entry points; fills c (nothing is
// launched when the result is not CLOVER_OK).
clover_status check_accept(AcceptCall &c, const void *logits, const int32_t *cand, const int32_t *parent, int B,
                           int T, int V, clover_dtype dtype, int32_t *argmax_out, int32_t *path_out,
                           int32_t *accept_len, int32_t *bonus_token, void *workspace, size_t ws_bytes,
                           int32_t *status, bool typical, double temperature, double epsilon, double delta) {
    if (B < 0 || T < 1 || V < 1) return CLOVER_ERR_INVALID_ARG;
    if (dtype != CLOVER_F32 && dtype != CLOVER_BF16) return CLOVER_ERR_INVALID_ARG;
    c = AcceptCall{};
    if (typical) {
        if (!(temperature > 0.0) || !isfinite(temperature) || !(epsilon >= 0.0) || !isfinite(epsilon) ||
            !(delta >= 0.0) || !isfinite(delta))
            return CLOVER_ERR_INVALID_ARG;
        // exponents are kept in base 2: y = x log2(e) / temperature, in fp32
        c.y_scale = (float)(1.4426950408889634 / temperature);
        if (!isfinite(c.y_scale) || !(c.y_scale >= 1.17549435e-38f)) return CLOVER_ERR_UNSUPPORTED;
        c.log2_eps = epsilon > 0.0 ? (float)log2(epsilon) : -INFINITY;
        c.log2_delta = delta > 0.0 ? (float)log2(delta) : -INFINITY;
    }
    if (T > kMaxTreeNodes) return CLOVER_ERR_UNSUPPORTED;
    if ((long)B * T > 0x7FFFFFFFL) return CLOVER_ERR_UNSUPPORTED;
    if (B > 0) {
        if (!logits || !cand || !parent || !argmax_out || !path_out || !accept_len || !bonus_token)
            return CLOVER_ERR_INVALID_ARG;
        const size_t need = typical ? accept_typical_workspace_bytes(B, T, V, dtype)
                                    : accept_workspace_bytes(B, T, V, dtype);
        if (ws_bytes < need || !workspace || !(typical ? aligned16(workspace)
                                                       : (reinterpret_cast<uintptr_t>(workspace) & 7u) == 0))
            return CLOVER_ERR_INVALID_ARG;
        if (reinterpret_cast<uintptr_t>(logits) % (dtype == CLOVER_F32 ? 4 : 2)) return CLOVER_ERR_INVALID_ARG;
    }
    c.logits = logits;
    c.cand = cand;
    c.parent = parent;
    c.B = B;
    c.T = T;
    c.V = V;
    c.dtype = dtype;
    c.argmax_out = argmax_out;
    c.path_out = path_out;
    c.accept_len = accept_len;
    c.bonus = bonus_token;
    c.workspace = workspace;
    c.status = status;
    c.typical = typical;
    return CLOVER_OK;
}

// Logical capacity of a paged cache (page_size * max_pages slots), or -1 when
// the page size is not a power of two in [16, 1024] or the product overflows.
long paged_capacity(int page_size, int max_pages) {
    if (page_size < 16 || page_size > 1024 || (page_size & (page_size - 1)) || max_pages < 1) return -1;
    const long c = (long)page_size * max_pages;
    return c > 0x3FFFFFFFL ? -1 : c;
}

// The attention call after the size checks (B > 0): pointer checks, the
// launch plan and the kernel.  block_table != nullptr: paged cache.
clover_status run_attn(const void *q, const void *k_new, const void *v_new, void *k_cache, void *v_cache,
                       const int32_t *cache_len, const int32_t *parent, void *out, int B, int T, int Hq, int Hkv,
                       int D, int Lcap, clover_dtype dtype, float scale, void *workspace, size_t ws_bytes,
                       int32_t *status, void *stream, bool append, const int32_t *block_table, int page_size,
                       int max_pages, int n_pages, uint32_t launch_flags = 0u) {
    if (!q || !k_new || !v_new || !k_cache || !v_cache || !cache_len || !parent || !out)
        return CLOVER_ERR_INVALID_ARG;
    if (!aligned16(q) || !aligned16(k_new) || !aligned16(v_new) || !aligned16(k_cache) || !aligned16(v_cache) ||
        !aligned16(out))
        return CLOVER_ERR_INVALID_ARG;
    if (!(scale == scale) || isinf(scale)) return CLOVER_ERR_INVALID_ARG;
    const AttnPlan p = plan_attn(B, T, Hq, Hkv, D, Lcap, dtype);
    if (ws_bytes < p.total || (p.total > 0 && (!workspace || !aligned16(workspace)))) return CLOVER_ERR_INVALID_ARG;

    AttnArgs a{};
    a.q = q;
    a.k_new = k_new;
    a.v_new = v_new;
    a.k_cache = k_cache;
    a.v_cache = v_cache;
    a.cache_len = cache_len;
    a.parent = parent;
    a.out = out;
    a.B = B;
    a.T = T;
    a.Hq = Hq;
    a.Hkv = Hkv;
    a.D = D;
    a.Lcap = Lcap;
    a.G = Hq / Hkv;
    a.dtype = dtype;
    const float sc = scale > 0.f ? scale : 1.f / sqrtf((float)D);
    a.scale_log2 = sc * 1.4426950408889634f;
    a.append = append ? 1 : 0;
    a.block_table = block_table;
    if (block_table) {
        a.page_size = page_size;
        while ((1 << a.page_shift) < page_size) ++a.page_shift;
        a.max_pages = max_pages;
        a.n_pages = n_pages;
    }
    a.rows = T * a.G;
    a.row_tile = p.row_tile;
    a.row_tiles = p.row_tiles;
    a.n_split = p.n_split;
    a.slot_rows = p.slot_rows;
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    // counters first: their place does not depend on the split count, so a
    // workspace sized for a capacity serves every smaller one
    a.counters = p.total ? reinterpret_cast<unsigned *>(ws) : nullptr;
    a.part_o = p.total ? reinterpret_cast<float *>(ws + p.counter_bytes) : nullptr;
    a.part_ml = p.total && p.ml_bytes ? reinterpret_cast<float *>(ws + p.counter_bytes + p.o_bytes) : nullptr;
    a.status = status;
    a.ws_bytes = workspace ? ws_bytes : 0;
    // the launch options apply to the tensor-core kernel; the FMA kernel is
    // launched the ordinary way (stream order) whatever they say
    a.pdl = (launch_flags & CLOVER_ATTN_PDL) ? 1 : 0;
    a.cache_early = (a.pdl && (launch_flags & CLOVER_ATTN_CACHE_READY)) ? 1 : 0;
    a.inputs_early = (a.pdl && (launch_flags & CLOVER_ATTN_INPUTS_READY)) ? 1 : 0;
    // A launch that runs its whole key loop beside the kernels before it is
    // one of a chain that shares the GPU: it takes about kChainCtas CTAs (a
    // fifth of the SMs), so that about five launches run at once, each CTA
    // over as long a key range as that allows: one CTA per (sequence, head,
    // row tile) when there are that many, which spends no setup and no merge
    // on split ranges (and does not use the workspace).
    if (p.tc && a.inputs_early) {
        const long base = (long)B * Hkv * p.row_tiles;
        const long want = (kChainCtas + base - 1) / base;
        a.n_split = (int)(want < p.n_split ? want : p.n_split);
        if (a.n_split == 1) {
            a.counters = nullptr;
            a.part_o = nullptr;
            a.part_ml = nullptr;
        }
    }
    const cudaStream_t st = static_cast<cudaStream_t>(stream);
    // Such a launch with one CTA per head and at least two row tiles a head
    // (grouped-query shapes) runs two row tiles per CTA: each K/V tile an SM
    // loads then serves 256 query rows.
    if (p.tc && a.inputs_early && tc_pair_eligible(a)) return from_cuda(launch_tree_attn_tc_pair(a, st));
    return from_cuda(p.tc ? launch_tree_attn_tc(a, st) : launch_tree_attn_fma(a, st));
}

}  // namespace

extern "C" {

int clover_abi_version(void) { return kAbiVersion; }

int clover_build_flags(void) {
#ifdef CLOVER_CHECKED
    return CLOVER_BUILD_CHECKED;
#else
    return 0;
#endif
}

const char *clover_status_string(int status) {
    switch (status) {
        case CLOVER_OK: return "ok";
        case CLOVER_ERR_INVALID_ARG: return "invalid argument";
        case CLOVER_ERR_UNSUPPORTED: return "unsupported size or type";
        case CLOVER_ERR_BAD_TREE: return "parent array is not a topologically numbered tree";
        case CLOVER_ERR_CAPACITY: return "cache length out of range or cache too small";
        case CLOVER_ERR_CUDA: return "CUDA error";
        case CLOVER_ERR_TIMEOUT: return "device wait timed out";
        case CLOVER_ERR_SCRATCH_LIMIT: return "scratch need exceeds the static buffer of clover_verify_attn_noalloc";
        case CLOVER_ERR_CHECK: return "a device index check failed (CLOVER_CHECKED build)";
        default: return "several errors (bitwise OR of codes)";
    }
}

size_t clover_verify_attn_workspace_size(int B, int T, int Hq, int Hkv, int D, int Lcap, clover_dtype dtype) {
    if (check_attn_sizes(B, T, Hq, Hkv, D, Lcap, dtype) != CLOVER_OK) return 0;
    return plan_attn(B, T, Hq, Hkv, D, Lcap, dtype).total;
}

clover_status clover_verify_attn(const void *q, const void *k_new, const void *v_new, void *k_cache,
                                 void *v_cache, const int32_t *cache_len, const int32_t *parent, void *out,
                                 int B, int T, int Hq, int Hkv, int D, int Lcap, clover_dtype dtype,
                                 float scale, void *workspace, size_t ws_bytes, int32_t *status,
                                 void *stream) {
    const NvtxRange nvtx_range("clover_verify_attn");
    return clover_verify_attn_ex(q, k_new, v_new, k_cache, v_cache, cache_len, parent, out, B, T, Hq, Hkv, D,
                                 Lcap, dtype, scale, workspace, ws_bytes, status, stream, 0u);
}

clover_status clover_verify_attn_ex(const void *q, const void *k_new, const void *v_new, void *k_cache,
                                    void *v_cache, const int32_t *cache_len, const int32_t *parent, void *out,
                                    int B, int T, int Hq, int Hkv, int D, int Lcap, clover_dtype dtype,
                                    float scale, void *workspace, size_t ws_bytes, int32_t *status,
                                    void *stream, uint32_t flags) {
    const NvtxRange nvtx_range("clover_verify_attn_ex");
    if (flags & ~(CLOVER_ATTN_NO_APPEND | CLOVER_ATTN_PDL | CLOVER_ATTN_CACHE_READY | CLOVER_ATTN_INPUTS_READY))
        return CLOVER_ERR_INVALID_ARG;
    const clover_status s = check_attn_sizes(B, T, Hq, Hkv, D, Lcap, dtype);
    if (s != CLOVER_OK) return s;
    if (B == 0) return CLOVER_OK;
    return run_attn(q, k_new, v_new, k_cache, v_cache, cache_len, parent, out, B, T, Hq, Hkv, D, Lcap, dtype, scale,
                    workspace, ws_bytes, status, stream, (flags & CLOVER_ATTN_NO_APPEND) == 0, nullptr, 0, 0, 0,
                    flags);
}

size_t clover_verify_attn_paged_workspace_size(int B, int T, int Hq, int Hkv, int D, int page_size, int max_pages,
                                               clover_dtype dtype) {
    const long lcap = paged_capacity(page_size, max_pages);
    if (lcap < 0) return 0;
    return clover_verify_attn_workspace_size(B, T, Hq, Hkv, D, (int)lcap, dtype);
}

static clover_status attn_paged(const void *q, const void *k_new, const void *v_new, const void *k_pages,
                                const void *v_pages, const int32_t *block_table, int n_pages, int page_size,
                                int max_pages, const int32_t *cache_len, const int32_t *parent, void *out, int B,
                                int T, int Hq, int Hkv, int D, clover_dtype dtype, float scale, void *workspace,
                                size_t ws_bytes, int32_t *status, void *stream, uint32_t flags) {
    constexpr uint32_t known = CLOVER_ATTN_NO_APPEND | CLOVER_ATTN_PDL | CLOVER_ATTN_CACHE_READY |
                               CLOVER_ATTN_INPUTS_READY;
    if (flags & ~known) return CLOVER_ERR_INVALID_ARG;
    const long lcap = paged_capacity(page_size, max_pages);
    if (lcap < 0 || n_pages < 1) return CLOVER_ERR_INVALID_ARG;
    const clover_status s = check_attn_sizes(B, T, Hq, Hkv, D, (int)lcap, dtype);
    if (s != CLOVER_OK) return s;
    if ((long)n_pages * Hkv * page_size > 0x7FFFFFFFL) return CLOVER_ERR_UNSUPPORTED;
    if (B == 0) return CLOVER_OK;
    if (!block_table) return CLOVER_ERR_INVALID_ARG;
    return run_attn(q, k_new, v_new, const_cast<void *>(k_pages), const_cast<void *>(v_pages), cache_len, parent, out,
                    B, T, Hq, Hkv, D, (int)lcap, dtype, scale, workspace, ws_bytes, status, stream, false, block_table,
                    page_size, max_pages, n_pages, flags & ~CLOVER_ATTN_NO_APPEND);
}

clover_status clover_verify_attn_paged(const void *q, const void *k_new, const void *v_new, const void *k_pages,
                                       const void *v_pages, const int32_t *block_table, int n_pages, int page_size,
                                       int max_pages, const int32_t *cache_len, const int32_t *parent, void *out,
                                       int B, int T, int Hq, int Hkv, int D, clover_dtype dtype, float scale,
                                       void *workspace, size_t ws_bytes, int32_t *status, void *stream) {
    const NvtxRange nvtx_range("clover_verify_attn_paged");
    return attn_paged(q, k_new, v_new, k_pages, v_pages, block_table, n_pages, page_size, max_pages, cache_len, parent,
                      out, B, T, Hq, Hkv, D, dtype, scale, workspace, ws_bytes, status, stream, 0u);
}

clover_status clover_verify_attn_paged_ex(const void *q, const void *k_new, const void *v_new, const void *k_pages,
                                          const void *v_pages, const int32_t *block_table, int n_pages,
                                          int page_size, int max_pages, const int32_t *cache_len,
                                          const int32_t *parent, void *out, int B, int T, int Hq, int Hkv, int D,
                                          clover_dtype dtype, float scale, void *workspace, size_t ws_bytes,
                                          int32_t *status, void *stream, uint32_t flags) {
    const NvtxRange nvtx_range("clover_verify_attn_paged_ex");
    return attn_paged(q, k_new, v_new, k_pages, v_pages, block_table, n_pages, page_size, max_pages, cache_len, parent,
                      out, B, T, Hq, Hkv, D, dtype, scale, workspace, ws_bytes, status, stream, flags);
}

size_t clover_verify_accept_workspace_size(int B, int T, int V, clover_dtype dtype) {
    if (B < 0 || T < 1 || T > kMaxTreeNodes || V < 1) return 0;
    if (dtype != CLOVER_F32 && dtype != CLOVER_BF16) return 0;
    return accept_workspace_bytes(B > 0 ? B : 1, T, V, dtype);
}

clover_status clover_verify_accept(const void *logits, const int32_t *cand, const int32_t *parent, int B, int T,
                                   int V, clover_dtype dtype, int32_t *argmax_out, int32_t *path_out,
                                   int32_t *accept_len, int32_t *bonus_token, void *workspace, size_t ws_bytes,
                                   int32_t *status, void *stream) {
    const NvtxRange nvtx_range("clover_verify_accept");
    AcceptCall c;
    const clover_status s = check_accept(c, logits, cand, parent, B, T, V, dtype, argmax_out, path_out, accept_len,
                                         bonus_token, workspace, ws_bytes, status, false, 0.0, 0.0, 0.0);
    if (s != CLOVER_OK || B == 0) return s;
    return from_cuda(launch_accept_call(c, static_cast<cudaStream_t>(stream)));
}

size_t clover_verify_accept_typical_workspace_size(int B, int T, int V, clover_dtype dtype) {
    if (B < 0 || T < 1 || T > kMaxTreeNodes || V < 1) return 0;
    if (dtype != CLOVER_F32 && dtype != CLOVER_BF16) return 0;
    return accept_typical_workspace_bytes(B > 0 ? B : 1, T, V, dtype);
}

clover_status clover_verify_accept_typical(const void *logits, const int32_t *cand, const int32_t *parent, int B,
                                           int T, int V, clover_dtype dtype, double temperature, double epsilon,
                                           double delta, int32_t *argmax_out, int32_t *path_out,
                                           int32_t *accept_len, int32_t *bonus_token, void *workspace,
                                           size_t ws_bytes, int32_t *status, void *stream) {
    const NvtxRange nvtx_range("clover_verify_accept_typical");
    AcceptCall c;
    const clover_status s = check_accept(c, logits, cand, parent, B, T, V, dtype, argmax_out, path_out, accept_len,
                                         bonus_token, workspace, ws_bytes, status, true, temperature, epsilon,
                                         delta);
    if (s != CLOVER_OK || B == 0) return s;
    return from_cuda(launch_accept_call(c, static_cast<cudaStream_t>(stream)));
}

size_t clover_verify_accept_ex_workspace_size(int B, int T, int V, clover_dtype dtype, uint32_t flags) {
    return (flags & CLOVER_ACCEPT_TYPICAL) ? clover_verify_accept_typical_workspace_size(B, T, V, dtype)
                                           : clover_verify_accept_workspace_size(B, T, V, dtype);
}

clover_status clover_verify_accept_ex(const void *logits, const int32_t *cand, const int32_t *parent, int B, int T,
                                      int V, clover_dtype dtype, double temperature, double epsilon, double delta,
                                      void *k_cache, void *v_cache, const void *k_new, const void *v_new,
                                      const int32_t *cache_len, int Hkv, int D, int Lcap, int32_t *argmax_out,
                                      int32_t *path_out, int32_t *accept_len, int32_t *bonus_token,
                                      int32_t *new_cache_len, int32_t *src_index_out, void *workspace,
                                      size_t ws_bytes, uint32_t flags, int32_t *status, void *stream) {
    const NvtxRange nvtx_range("clover_verify_accept_ex");
    constexpr uint32_t known = CLOVER_ACCEPT_TYPICAL | CLOVER_ACCEPT_COMMIT | CLOVER_ACCEPT_OVERLAP;
    if (flags & ~known) return CLOVER_ERR_INVALID_ARG;
    AcceptCall c;
    clover_status s = check_accept(c, logits, cand, parent, B, T, V, dtype, argmax_out, path_out, accept_len,
                                   bonus_token, workspace, ws_bytes, status, (flags & CLOVER_ACCEPT_TYPICAL) != 0,
                                   temperature, epsilon, delta);
    if (s != CLOVER_OK) return s;
    if (flags & CLOVER_ACCEPT_COMMIT) {
        // the path and accepted length are this call's own outputs: any
        // non-NULL pointers pass the commit checks on them
        s = check_commit(k_cache, v_cache, k_new, v_new, cache_len, path_out, accept_len, new_cache_len, B, T, Hkv,
                         D, Lcap, dtype, true);
        if (s != CLOVER_OK) return s;
        c.commit = true;
        c.k_cache = k_cache;
        c.v_cache = v_cache;
        c.k_new = k_new;
        c.v_new = v_new;
        c.cache_len = cache_len;
        c.new_cache_len = new_cache_len;
        c.src_index = src_index_out;
        c.Hkv = Hkv;
        c.D = D;
        c.Lcap = Lcap;
    }
    c.after_prior = (flags & CLOVER_ACCEPT_OVERLAP) != 0;
    if (B == 0) return CLOVER_OK;
    return from_cuda(launch_accept_call(c, static_cast<cudaStream_t>(stream)));
}

clover_status clover_verify_accept_paged_ex(const void *logits, const int32_t *cand, const int32_t *parent, int B,
                                            int T, int V, clover_dtype dtype, double temperature, double epsilon,
                                            double delta, void *k_pages, void *v_pages, const int32_t *block_table,
                                            int n_pages, int page_size, int max_pages, const void *k_new,
                                            const void *v_new, const int32_t *cache_len, int Hkv, int D,
                                            int32_t *argmax_out, int32_t *path_out, int32_t *accept_len,
                                            int32_t *bonus_token, int32_t *new_cache_len, int32_t *src_index_out,
                                            void *workspace, size_t ws_bytes, uint32_t flags, int32_t *status,
                                            void *stream) {
    const NvtxRange nvtx_range("clover_verify_accept_paged_ex");
    constexpr uint32_t known = CLOVER_ACCEPT_TYPICAL | CLOVER_ACCEPT_COMMIT | CLOVER_ACCEPT_OVERLAP;
    if (flags & ~known) return CLOVER_ERR_INVALID_ARG;
    const long lcap = paged_capacity(page_size, max_pages);
    if (lcap < 0 || n_pages < 1) return CLOVER_ERR_INVALID_ARG;
    AcceptCall c;
    clover_status s = check_accept(c, logits, cand, parent, B, T, V, dtype, argmax_out, path_out, accept_len,
                                   bonus_token, workspace, ws_bytes, status, (flags & CLOVER_ACCEPT_TYPICAL) != 0,
                                   temperature, epsilon, delta);
    if (s != CLOVER_OK) return s;
    s = check_commit(k_pages, v_pages, k_new, v_new, cache_len, path_out, accept_len, new_cache_len, B, T, Hkv, D,
                     (int)lcap, dtype, true);
    if (s != CLOVER_OK) return s;
    if ((long)n_pages * Hkv * page_size > 0x7FFFFFFFL) return CLOVER_ERR_UNSUPPORTED;
    if (B > 0 && !block_table) return CLOVER_ERR_INVALID_ARG;
    c.commit = true;
    c.k_cache = k_pages;
    c.v_cache = v_pages;
    c.k_new = k_new;
    c.v_new = v_new;
    c.cache_len = cache_len;
    c.new_cache_len = new_cache_len;
    c.src_index = src_index_out;
    c.Hkv = Hkv;
    c.D = D;
    c.Lcap = (int)lcap;
    c.block_table = block_table;
    c.page_size = page_size;
    c.max_pages = max_pages;
    c.n_pages = n_pages;
    c.after_prior = (flags & CLOVER_ACCEPT_OVERLAP) != 0;
    if (B == 0) return CLOVER_OK;
    return from_cuda(launch_accept_call(c, static_cast<cudaStream_t>(stream)));
}

clover_status clover_kv_commit(void *k_cache, void *v_cache, const void *k_new, const void *v_new,
                               const int32_t *cache_len, const int32_t *path, const int32_t *accept_len,
                               int32_t *new_cache_len, int32_t *src_index_out, int B, int T, int Hkv, int D,
                               int Lcap, clover_dtype dtype, int32_t *status, void *stream) {
    const NvtxRange nvtx_range("clover_kv_commit");
    const clover_status s = check_commit(k_cache, v_cache, k_new, v_new, cache_len, path, accept_len, new_cache_len,
                                         B, T, Hkv, D, Lcap, dtype, true);
    if (s != CLOVER_OK || B == 0) return s;
    return from_cuda(launch_kv_compact(k_cache, v_cache, k_new, v_new, cache_len, path, accept_len, new_cache_len,
                                       src_index_out, B, T, Hkv, D, Lcap, dtype, status,
                                       static_cast<cudaStream_t>(stream)));
}

size_t clover_linear_workspace_size(int R, int N, int K) {
    if (R < 0 || N < 1 || K < 64 || K % 64 != 0) return 0;
    return linear_workspace_bytes(R > 0 ? R : 1, N, K);
}

clover_status clover_linear(const void *x, const void *w, const void *res, void *out, int R, int N, int K, int mode,
                            void *workspace, size_t ws_bytes, int32_t *status, void *stream) {
    return clover_linear_ex(x, w, res, out, R, N, K, mode, 0u, workspace, ws_bytes, status, stream);
}

clover_status clover_linear_ex(const void *x, const void *w, const void *res, void *out, int R, int N, int K, int mode,
                               unsigned flags, void *workspace, size_t ws_bytes, int32_t *status, void *stream) {
    const NvtxRange nvtx_range("clover_linear");
    if (flags & ~CLOVER_LINEAR_PDL) return CLOVER_ERR_INVALID_ARG;
    if (R < 0 || N < 1 || K < 64 || K % 64 != 0) return CLOVER_ERR_INVALID_ARG;
    if (mode < CLOVER_LINEAR_F32 || mode > CLOVER_LINEAR_RES) return CLOVER_ERR_INVALID_ARG;
    const bool with_res = mode == CLOVER_LINEAR_RES_SILU || mode == CLOVER_LINEAR_RES;
    if ((long)R * N > 0x7FFFFFFFL * 4L) return CLOVER_ERR_UNSUPPORTED;
    if (R == 0) return CLOVER_OK;
    if (!x || !w || !out || (with_res && !res)) return CLOVER_ERR_INVALID_ARG;
    if (!aligned16(x) || !aligned16(w) || !aligned16(out) || (with_res && !aligned16(res)))
        return CLOVER_ERR_INVALID_ARG;
    if (workspace && !aligned16(workspace)) return CLOVER_ERR_INVALID_ARG;
    return from_cuda(launch_linear_tc(x, w, with_res ? res : nullptr, out, R, N, K, mode, workspace, ws_bytes, status,
                                      (flags & CLOVER_LINEAR_PDL) != 0, static_cast<cudaStream_t>(stream)));
}

clover_status clover_embed_rows(const void *w, const int32_t *tokens, void *e, int R, int V, int H, int32_t *status,
                                void *stream) {
    const NvtxRange nvtx_range("clover_embed_rows");
    if (R < 0 || V < 1 || H < 1) return CLOVER_ERR_INVALID_ARG;
    if (R == 0) return CLOVER_OK;
    if (!w || !tokens || !e) return CLOVER_ERR_INVALID_ARG;
    return from_cuda(launch_embed_rows(w, tokens, e, R, V, H, status, static_cast<cudaStream_t>(stream)));
}

size_t clover_topk_workspace_size(int R, int V, int k) {
    if (R < 0 || V < 1 || k < 1 || k > topk_max_k() || k > V) return 0;
    return topk_workspace_bytes(R > 0 ? R : 1, V, k);
}

clover_status clover_topk(const float *x, int R, int V, int k, float *values, int32_t *indices, void *workspace,
                          size_t ws_bytes, int32_t *status, void *stream) {
    const NvtxRange nvtx_range("clover_topk");
    if (R < 0 || V < 1 || k < 1 || k > V) return CLOVER_ERR_INVALID_ARG;
    if (k > topk_max_k()) return CLOVER_ERR_UNSUPPORTED;
    // the final merge holds two candidates a thread: chunks x k <= 512
    if ((long)((V + 8191) / 8192) * k > 512) return CLOVER_ERR_UNSUPPORTED;
    if (R == 0) return CLOVER_OK;
    if (!x || !values || !indices) return CLOVER_ERR_INVALID_ARG;
    if (ws_bytes < topk_workspace_bytes(R, V, k) || !workspace || (reinterpret_cast<uintptr_t>(workspace) & 7u))
        return CLOVER_ERR_INVALID_ARG;
    return from_cuda(launch_topk(x, R, V, k, values, indices, workspace, status, static_cast<cudaStream_t>(stream)));
}

clover_status clover_kv_commit_paged(void *k_pages, void *v_pages, const int32_t *block_table, int n_pages,
                                     int page_size, int max_pages, const void *k_new, const void *v_new,
                                     const int32_t *cache_len, const int32_t *path, const int32_t *accept_len,
                                     int32_t *new_cache_len, int32_t *src_index_out, int B, int T, int Hkv, int D,
                                     clover_dtype dtype, int32_t *status, void *stream) {
    const NvtxRange nvtx_range("clover_kv_commit_paged");
    const long lcap = paged_capacity(page_size, max_pages);
    if (lcap < 0 || n_pages < 1) return CLOVER_ERR_INVALID_ARG;
    const clover_status s = check_commit(k_pages, v_pages, k_new, v_new, cache_len, path, accept_len, new_cache_len,
                                         B, T, Hkv, D, (int)lcap, dtype, true);
    if (s != CLOVER_OK || B == 0) return s;
    if ((long)n_pages * Hkv * page_size > 0x7FFFFFFFL) return CLOVER_ERR_UNSUPPORTED;
    if (!block_table) return CLOVER_ERR_INVALID_ARG;
    return from_cuda(launch_kv_compact(k_pages, v_pages, k_new, v_new, cache_len, path, accept_len, new_cache_len,
                                       src_index_out, B, T, Hkv, D, (int)lcap, dtype, status,
                                       static_cast<cudaStream_t>(stream), block_table, page_size, max_pages, n_pages));
}

clover_status clover_kv_compact(void *k_cache, void *v_cache, const int32_t *cache_len, const int32_t *path,
                                const int32_t *accept_len, int32_t *new_cache_len, int32_t *src_index_out, int B,
                                int T, int Hkv, int D, int Lcap, clover_dtype dtype, int32_t *status,
                                void *stream) {
    const NvtxRange nvtx_range("clover_kv_compact");
    const clover_status s = check_commit(k_cache, v_cache, nullptr, nullptr, cache_len, path, accept_len,
                                         new_cache_len, B, T, Hkv, D, Lcap, dtype, false);
    if (s != CLOVER_OK || B == 0) return s;
    return from_cuda(launch_kv_compact(k_cache, v_cache, nullptr, nullptr, cache_len, path, accept_len,
                                       new_cache_len, src_index_out, B, T, Hkv, D, Lcap, dtype, status,
                                       static_cast<cudaStream_t>(stream)));
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Allocation-free attention: the split-KV scratch of clover_verify_attn lives in
// a static device array instead of a caller-provided workspace.
// ---------------------------------------------------------------------------

namespace clover {
namespace {

static_assert(CLOVER_NOALLOC_SCRATCH_BYTES % 256 == 0, "scratch size must keep 256-byte alignment");

// Resident on every device that loads this library, until the process exits.
static __device__ __align__(256) unsigned char g_attn_scratch[CLOVER_NOALLOC_SCRATCH_BYTES];

// Device address of g_attn_scratch, looked up with cudaGetSymbolAddress once
// per CUDA context (the context current on the calling thread) and cached
// under that context's id.  A device ordinal alone would not do: after
// cudaDeviceReset, or under a non-primary context of the same device, the
// module (and with it the array) is loaded anew, possibly at another address.
constexpr int kAddrSlots = 64;
struct ScratchAddr {
    unsigned long long ctx;   // current_context_id() of the lookup (0: slot unused)
    void *addr;
};
std::mutex g_attn_scratch_mu;
ScratchAddr g_attn_scratch_addr[kAddrSlots];
int g_attn_scratch_next = 0;   // slot to fill (round robin once every slot is used)

cudaError_t attn_scratch_address(void **addr) {
    const unsigned long long ctx = current_context_id();
    std::lock_guard<std::mutex> lock(g_attn_scratch_mu);
    if (ctx != 0)
        for (const ScratchAddr &s : g_attn_scratch_addr)
            if (s.ctx == ctx) {
                *addr = s.addr;
                return cudaSuccess;
            }
    void *p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_attn_scratch);
    if (e != cudaSuccess) return e;
    if (ctx != 0) {
        g_attn_scratch_addr[g_attn_scratch_next] = ScratchAddr{ctx, p};
        g_attn_scratch_next = (g_attn_scratch_next + 1) % kAddrSlots;
    }
    *addr = p;
    return cudaSuccess;
}

}  // namespace
}  // namespace clover

extern "C" clover_status clover_verify_attn_noalloc(const void *q, const void *k_new, const void *v_new,
                                                    void *k_cache, void *v_cache, const int32_t *cache_len,
                                                    const int32_t *parent, void *out, int B, int T, int Hq,
                                                    int Hkv, int D, int Lcap, clover_dtype dtype, float scale,
                                                    int32_t *status, void *stream) {
    const NvtxRange nvtx_range("clover_verify_attn_noalloc");
    using namespace clover;
    const clover_status s = check_attn_sizes(B, T, Hq, Hkv, D, Lcap, dtype);
    if (s != CLOVER_OK) return s;
    if (B == 0) return CLOVER_OK;
    // the argument checks of clover_verify_attn, repeated so that nothing (not
    // even the counter memset) is issued for a call it would reject
    if (!q || !k_new || !v_new || !k_cache || !v_cache || !cache_len || !parent || !out)
        return CLOVER_ERR_INVALID_ARG;
    if (!aligned16(q) || !aligned16(k_new) || !aligned16(v_new) || !aligned16(k_cache) || !aligned16(v_cache) ||
        !aligned16(out))
        return CLOVER_ERR_INVALID_ARG;
    if (!(scale == scale) || isinf(scale)) return CLOVER_ERR_INVALID_ARG;
    const AttnPlan p = plan_attn(B, T, Hq, Hkv, D, Lcap, dtype);
    if (p.total > CLOVER_NOALLOC_SCRATCH_BYTES) return CLOVER_ERR_SCRATCH_LIMIT;

    void *scratch = nullptr;
    if (attn_scratch_address(&scratch) != cudaSuccess) return CLOVER_ERR_CUDA;
    const cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (p.counter_bytes > 0 &&
        cudaMemsetAsync(scratch, 0, p.counter_bytes, st) !=
            cudaSuccess)
        return CLOVER_ERR_CUDA;
    return clover_verify_attn(q, k_new, v_new, k_cache, v_cache, cache_len, parent, out, B, T, Hq, Hkv, D, Lcap,
                              dtype, scale, scratch, CLOVER_NOALLOC_SCRATCH_BYTES, status, stream);
}
