// Per-node argmax over the vocabulary and the greedy acceptance walk, in one
// launch.
//
// The verification phase keeps the base model's own output (Section 1, and
// Section 2.1): the greedy token at tree node i is the first index of the
// maximum of its logit row.  A speculated child is accepted when its candidate
// token equals its parent's greedy token; the accepted path is walked from the
// root and its length is the paper's tokens/step (Section 4.1).
//
// Grid: one CTA per (logit row, vocabulary chunk of one to four 32 KB rounds).
// Each CTA reduces its chunk with 16-byte loads (eight in flight per thread a
// round) to a packed 64-bit key
// (order-preserving value bits in the high word, bit-inverted index in the low
// word) so that one unsigned max gives "largest value, then smallest index",
// and folds it into the row's key with a 64-bit atomic max.  A per-sequence
// arrival counter finds the CTA that finishes a sequence's last chunk; it
// decodes the argmax of every node and runs the walk in one warp, and resets
// the keys and the counter.
//
// Typical acceptance (the tree sampling rule the paper evaluates with, Section
// 4 setup, after Medusa) is a compile-time mode of the same kernel.  Each chunk
// CTA keeps its loads in registers and, besides the packed maximum, sums over
// its chunk s = sum 2^t and u = sum 2^t t with t = (x - m) log2(e) / tau, the
// base-2 exponent relative to a maximum m (each thread's own, then merged
// across the CTA), and gathers the logits of the candidates that fall in its
// chunk.  The last CTA merges the chunk sums of every row into the tempered
// softmax's normaliser and entropy (H = ln 2 (log2 S - U / S) over the merged
// sums), decides every edge p(cand) > min(eps, delta e^-H) in the log2
// domain, and walks the longest accepted path (ties: the smallest-index child
// at every step).
#include <algorithm>

#include "common.cuh"

namespace clover {
namespace {

constexpr int kThreads = 256;

// Order-preserving map of a float to 32 unsigned bits; -0 is first turned into +0.
__device__ __forceinline__ uint32_t order_bits(float x) {
    uint32_t u = __float_as_uint(x);
    if (u == 0x80000000u) u = 0u;
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__device__ __forceinline__ uint64_t make_key(float x, uint32_t index) {
    return (static_cast<uint64_t>(order_bits(x)) << 32) | static_cast<uint64_t>(0xFFFFFFFFu - index);
}

__device__ __forceinline__ uint64_t umax64(uint64_t a, uint64_t b) { return a > b ? a : b; }

template <typename T>
__device__ __forceinline__ void scan_scalar(const T *row, int64_t lo, int64_t hi, uint64_t &best) {
    for (int64_t v = lo + threadIdx.x; v < hi; v += kThreads) best = umax64(best, make_key(to_float(row[v]), (uint32_t)v));
}

constexpr int kUnits = 8;   // 16-byte loads each thread issues at once

// Largest value of a 16-byte unit (8 bf16 or 4 fp32), as fp32.
__device__ __forceinline__ float unit_max(const uint4 &w, __nv_bfloat16) {
    const __nv_bfloat162 *h = reinterpret_cast<const __nv_bfloat162 *>(&w);
    const __nv_bfloat162 m = __hmax2(__hmax2(h[0], h[1]), __hmax2(h[2], h[3]));
    return fmaxf(__low2float(m), __high2float(m));
}
__device__ __forceinline__ float unit_max(const uint4 &w, float) {
    return fmaxf(fmaxf(__uint_as_float(w.x), __uint_as_float(w.y)), fmaxf(__uint_as_float(w.z), __uint_as_float(w.w)));
}

// Position of the first element of a unit equal to v (which the unit holds).
__device__ __forceinline__ int unit_first(const uint4 &w, float v, __nv_bfloat16) {
    const uint32_t x[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        const float f = __uint_as_float((e & 1) ? (x[e >> 1] & 0xFFFF0000u) : (x[e >> 1] << 16));
        if (f == v) return e;
    }
    return 7;
}
__device__ __forceinline__ int unit_first(const uint4 &w, float v, float) {
    const uint32_t x[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int e = 0; e < 4; ++e)
        if (__uint_as_float(x[e]) == v) return e;
    return 3;
}

// Vector body: 16-byte units [0, n_units) of the row from element `first`,
// n_units <= kThreads * kUnits (one round).  A thread issues its
// kUnits independent loads (units tid + k*kThreads) into w, takes the maximum
// over them, and only then looks for its first position.
template <typename T>
__device__ __forceinline__ void scan_vector(const T *row, int64_t first, int64_t n_units, uint64_t &best,
                                            uint4 (&w)[kUnits]) {
    constexpr int E = 16 / sizeof(T);
    const uint4 *p = reinterpret_cast<const uint4 *>(row + first);
#pragma unroll
    for (int k = 0; k < kUnits; ++k) {
        const int64_t u = threadIdx.x + (int64_t)k * kThreads;
        w[k] = (u < n_units) ? __ldcs(p + u) : make_uint4(0, 0, 0, 0);
    }
    float um[kUnits];
    float m = -INFINITY;
#pragma unroll
    for (int k = 0; k < kUnits; ++k) {
        const int64_t u = threadIdx.x + (int64_t)k * kThreads;
        um[k] = (u < n_units) ? unit_max(w[k], T()) : -INFINITY;
        m = fmaxf(m, um[k]);
    }
    // units are visited in increasing element order, so the first unit
    // reaching m holds the thread's first maximum
    int kf = -1;
#pragma unroll
    for (int k = kUnits - 1; k >= 0; --k)
        if (um[k] == m && threadIdx.x + (int64_t)k * kThreads < n_units) kf = k;
    if (kf >= 0) {
        uint4 wf = w[0];
#pragma unroll
        for (int k = 1; k < kUnits; ++k)
            if (k == kf) wf = w[k];
        const int64_t u = threadIdx.x + (int64_t)kf * kThreads;
        const int e = unit_first(wf, m, T());
        best = umax64(best, make_key(m, (uint32_t)(first + u * E + e)));
    }
}

__device__ __forceinline__ float ex2_approx(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
__device__ __forceinline__ float lg2_approx(float x) {
    float y;
    asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// Softmax sums of a chunk relative to its scaled maximum my: s += 2^t and
// u += 2^t t with t = x * ys - my.  t is clamped at -256 (2^t is then 0 in
// fp32), which also turns the -inf logits (p = 0) into zero terms.
struct ExpSums {
    float s = 0.f, u = 0.f;
    float2 s2 = make_float2(0.f, 0.f), u2 = make_float2(0.f, 0.f);   // two lanes of sums, folded in at the end
    __device__ __forceinline__ void add(float x, float ys, float my) {
        const float t = fmaxf(fmaf(x, ys, -my), -256.f);
        const float e = ex2_approx(t);
        s += e;
        u = fmaf(e, t, u);
    }
    // two terms at once: the exponent arguments and both sums as packed f32x2
    // operations (each lane rounded as the scalar form would be)
    __device__ __forceinline__ void add2(float x0, float x1, float2 ys2, float2 nmy2) {
        float2 t = __ffma2_rn(make_float2(x0, x1), ys2, nmy2);
        t.x = fmaxf(t.x, -256.f);
        t.y = fmaxf(t.y, -256.f);
        const float2 e = make_float2(ex2_approx(t.x), ex2_approx(t.y));
        s2 = __fadd2_rn(s2, e);
        u2 = __ffma2_rn(e, t, u2);
    }
    __device__ __forceinline__ float sum_s() const { return s + (s2.x + s2.y); }
    __device__ __forceinline__ float sum_u() const { return u + (u2.x + u2.y); }
};

__device__ __forceinline__ void unit_sums(const uint4 &w, __nv_bfloat16, float ys, float my, ExpSums &acc) {
    const uint32_t x[4] = {w.x, w.y, w.z, w.w};
    const float2 ys2 = make_float2(ys, ys), nmy2 = make_float2(-my, -my);
#pragma unroll
    for (int k = 0; k < 4; ++k)
        acc.add2(__uint_as_float(x[k] << 16), __uint_as_float(x[k] & 0xFFFF0000u), ys2, nmy2);
}
__device__ __forceinline__ void unit_sums(const uint4 &w, float, float ys, float my, ExpSums &acc) {
    acc.add(__uint_as_float(w.x), ys, my);
    acc.add(__uint_as_float(w.y), ys, my);
    acc.add(__uint_as_float(w.z), ys, my);
    acc.add(__uint_as_float(w.w), ys, my);
}

// (m, s, u) of two disjoint parts -> the sums of their union, relative to the
// larger maximum.  Parts with s = 0 (all -inf) contribute nothing.
__device__ __forceinline__ float3 merge_sums(float3 a, float3 b) {
    if (b.y == 0.f) return a;
    if (a.y == 0.f) return b;
    const float M = fmaxf(a.x, b.x);
    const float da = a.x - M, db = b.x - M;
    const float wa = ex2_approx(da), wb = ex2_approx(db);
    return make_float3(M, wa * a.y + wb * b.y, wa * fmaf(a.y, da, a.z) + wb * fmaf(b.y, db, b.z));
}

__device__ __forceinline__ uint64_t block_max(uint64_t v, uint64_t *s_red) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v = umax64(v, __shfl_xor_sync(0xffffffffu, v, off));
    const int warp = threadIdx.x >> 5;
    if ((threadIdx.x & 31) == 0) s_red[warp] = v;
    __syncthreads();
    if (warp == 0) {
        v = (threadIdx.x < kThreads / 32) ? s_red[threadIdx.x] : 0ull;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) v = umax64(v, __shfl_xor_sync(0xffffffffu, v, off));
    }
    return v;   // valid in thread 0
}

struct AcceptArgs {
    const void *logits;
    const int32_t *cand, *parent;
    int B, T, V, n_chunks, chunk;
    int32_t *argmax_out, *path_out, *accept_len, *bonus;
    unsigned long long *row_key;   // [B*T] running packed maximum of each logit row
    unsigned *seq_count;           // [B] chunks of the sequence finished
    // typical acceptance only
    float4 *chunk_sums;            // [B*T, n_chunks] (scaled maximum, s, u) of every chunk
    float *cand_x;                 // [B*T] logit of each node's candidate under its parent
    float y_scale;                 // log2(e) / temperature
    float log2_eps, log2_delta;    // log2 of the threshold parameters (-inf for 0)
    // commit of the accepted K/V by the sequence's last CTA (commit != 0)
    uint4 *k_cache, *v_cache;      // [B, Hkv, Lcap, D] as 16-byte units
    const uint4 *k_new, *v_new;    // [B, T, Hkv, D]
    const int32_t *cache_len;
    int32_t *new_cache_len, *src_index;
    int Hkv, Lcap, row_units;      // row_units = D * element size / 16
    const int32_t *block_table;    // paged cache: [B, max_pages] page ids, else nullptr
    int page_size, page_shift, max_pages, n_pages;
    int commit;
    int wait_prior;                // the last CTAs end with a wait for the preceding grid
    int32_t *status;
};

constexpr int kNodesPerLane = kMaxTreeNodes / 32;

// Sequence b's tree in warp 0's registers: lane l holds nodes l + 32 k.
struct TreeRegs {
    int p[kNodesPerLane], c[kNodesPerLane];
    bool invalid;
};

__device__ __forceinline__ TreeRegs load_tree(const AcceptArgs &a, int b) {
    const int lane = threadIdx.x & 31;
    const int32_t *par = a.parent + (size_t)b * a.T;
    const int32_t *cd = a.cand + (size_t)b * a.T;
    TreeRegs t;
    t.invalid = false;
#pragma unroll
    for (int k = 0; k < kNodesPerLane; ++k) {
        const int i = lane + 32 * k;
        t.p[k] = -2;
        t.c[k] = 0;
        if (i < a.T) {
            t.p[k] = __ldg(par + i);
            t.c[k] = __ldg(cd + i);
            if (i == 0 ? (t.p[k] != -1) : (t.p[k] < 0 || t.p[k] >= i)) t.invalid = true;
        }
    }
    return t;
}

// First set bit of a warp's per-node predicate (node lane + 32 k for pred[k]);
// -1 if none.
__device__ __forceinline__ int first_node(const bool (&pred)[kNodesPerLane]) {
#pragma unroll
    for (int k = 0; k < kNodesPerLane; ++k) {
        const unsigned bits = __ballot_sync(0xffffffffu, pred[k]);
        if (bits) return 32 * k + __ffs(bits) - 1;
    }
    return -1;
}

// The walk of finish_sequence, by warp 0; the path also goes to s_path/s_len.
template <bool TYPICAL>
__device__ void walk_sequence(const AcceptArgs &a, int b, const TreeRegs &tr, const int (&am)[kNodesPerLane],
                              const float (&xc)[kNodesPerLane], const uint64_t (&anc)[kNodesPerLane][kMaskWords],
                              const float4 *s_row, int *s_path, int *s_len) {
    const int lane = threadIdx.x & 31;
    const int Tn = a.T;
    int32_t *path = a.path_out + (size_t)b * Tn;
    for (int i = lane; i < Tn; i += 32) path[i] = -1;
    __syncwarp();
    int cur = 0, len = 1;
    if (lane == 0) path[0] = s_path[0] = 0;
    auto argmax_of = [&](int node) {
        int v = 0;
#pragma unroll
        for (int k = 0; k < kNodesPerLane; ++k) {
            const int x = __shfl_sync(0xffffffffu, am[k], node & 31);
            if ((node >> 5) == k) v = x;
        }
        return v;
    };
    if (__any_sync(0xffffffffu, tr.invalid)) {
        if (lane == 0) report(a.status, CLOVER_ERR_BAD_TREE);
    } else if (!TYPICAL) {
        // at most T - 1 steps: every step moves to a larger node index
        for (int step = 1; step < Tn; ++step) {
            const int want = argmax_of(cur);
            bool hit[kNodesPerLane];
#pragma unroll
            for (int k = 0; k < kNodesPerLane; ++k) hit[k] = tr.p[k] == cur && tr.c[k] == want;
            const int next = first_node(hit);
            if (next < 0) break;
            cur = next;
            if (lane == 0) path[len] = s_path[len] = cur;
            ++len;
        }
    } else {
        uint64_t acc[kMaskWords];                 // accepted edges (node bits), the root included
#pragma unroll
        for (int k = 0; k < kNodesPerLane; ++k) {
            const int i = lane + 32 * k;
            bool ok = false;
            if (i >= 1 && i < Tn) {
                const float4 r = s_row[tr.p[k]];
                ok = fmaf(xc[k], a.y_scale, -r.x) - r.y > r.z;   // log2 p > log2 theta
            }
            const uint64_t bits = __ballot_sync(0xffffffffu, ok);
            if ((k & 1) == 0) acc[k >> 1] = bits;
            else acc[k >> 1] |= bits << 32;
        }
        acc[0] |= 1ull;
        int depth[kNodesPerLane];
        unsigned dmax = 0;
#pragma unroll
        for (int k = 0; k < kNodesPerLane; ++k) {
            bool reach = lane + 32 * k < Tn;
            int pc = -1;
#pragma unroll
            for (int w = 0; w < kMaskWords; ++w) {
                reach = reach && (anc[k][w] & ~acc[w]) == 0ull;
                pc += __popcll(anc[k][w]);
            }
            depth[k] = reach ? pc : -1;
            dmax = max(dmax, (unsigned)max(depth[k], 0));
        }
        dmax = __reduce_max_sync(0xffffffffu, dmax);
        // G: the nodes on the root paths of the deepest accepted nodes
        uint64_t g[kMaskWords] = {0ull, 0ull};
#pragma unroll
        for (int k = 0; k < kNodesPerLane; ++k)
            if (depth[k] == (int)dmax) {
#pragma unroll
                for (int w = 0; w < kMaskWords; ++w) g[w] |= anc[k][w];
            }
#pragma unroll
        for (int w = 0; w < kMaskWords; ++w)
            g[w] = (static_cast<uint64_t>(__reduce_or_sync(0xffffffffu, (unsigned)(g[w] >> 32))) << 32) |
                   __reduce_or_sync(0xffffffffu, (unsigned)g[w]);
        for (unsigned step = 0; step < dmax; ++step) {
            bool hit[kNodesPerLane];
#pragma unroll
            for (int k = 0; k < kNodesPerLane; ++k) {
                const int i = lane + 32 * k;
                hit[k] = tr.p[k] == cur && ((g[i >> 6] >> (i & 63)) & 1ull);
            }
            const int next = first_node(hit);
            if (next < 0) break;
            cur = next;
            if (lane == 0) path[len] = s_path[len] = cur;
            ++len;
        }
    }
    const int bonus = argmax_of(cur);
    if (lane == 0) {
        a.accept_len[b] = len;
        a.bonus[b] = bonus;
        a.seq_count[b] = 0u;                                       // ready for the next call
        *s_len = len;
    }
}

// Commit of sequence b's accepted path (len nodes in s_path) by the whole CTA:
// slot L + j of every KV head receives node s_path[j]'s K/V from k_new/v_new,
// into a dense cache or, through the block table, a paged one (a page id
// outside [0, n_pages) raises CLOVER_ERR_INVALID_ARG and its row is skipped).
__device__ void commit_sequence(const AcceptArgs &a, int b, const int *s_path, int len) {
    __shared__ int s_page[kMaxTreeNodes];     // paged: the page of slot L + j
    const int Tn = a.T;
    const int L = __ldg(a.cache_len + b);
    if (L < 0 || L + Tn > a.Lcap) {
        if (threadIdx.x == 0) report(a.status, CLOVER_ERR_CAPACITY);
        return;
    }
    if (a.src_index && threadIdx.x < Tn) a.src_index[(size_t)b * Tn + threadIdx.x] = threadIdx.x < len ? s_path[threadIdx.x] : -1;
    if (threadIdx.x == 0) a.new_cache_len[b] = L + len;
    if (a.block_table) {
        if ((int)threadIdx.x < len) {
            const int pg = __ldg(a.block_table + (size_t)b * a.max_pages + ((L + (int)threadIdx.x) >> a.page_shift));
            const bool bad = pg < 0 || pg >= a.n_pages;
            if (bad) report(a.status, CLOVER_ERR_INVALID_ARG);
            s_page[threadIdx.x] = bad ? -1 : pg;
        }
        __syncthreads();
    }
    // The accepted rows (len nodes x Hkv heads x row_units 16-byte units, K
    // and V) in batches: every thread loads its kBatch units of K and V, then
    // stores them, so a batch costs one load round trip.
    const int per_node = a.Hkv * a.row_units;
    const int total = len * per_node;
    constexpr int kBatch = 4;
    for (int e0 = threadIdx.x; e0 < total; e0 += kBatch * kThreads) {
        uint4 kb[kBatch], vb[kBatch];
#pragma unroll
        for (int t = 0; t < kBatch; ++t) {
            const int e = e0 + t * kThreads;
            if (e < total) {
                const int j = e / per_node;
                if (!CLOVER_IN(a.status, s_path[j], Tn)) continue;
                const size_t src = ((size_t)b * Tn + s_path[j]) * per_node + (e - j * per_node);
                kb[t] = __ldg(a.k_new + src);
                vb[t] = __ldg(a.v_new + src);
            }
        }
#pragma unroll
        for (int t = 0; t < kBatch; ++t) {
            const int e = e0 + t * kThreads;
            if (e < total) {
                const int j = e / per_node;
                const int r = e - j * per_node;
                const int g = r / a.row_units;
                const int u = r - g * a.row_units;
                if (!CLOVER_IN(a.status, s_path[j], Tn) || !CLOVER_IN(a.status, L + j, a.Lcap)) continue;
                size_t dst = (((size_t)b * a.Hkv + g) * a.Lcap + L + j) * a.row_units + u;
                if (a.block_table) {
                    if (s_page[j] < 0) continue;
                    dst = (((size_t)s_page[j] * a.Hkv + g) * a.page_size + ((L + j) & (a.page_size - 1))) * a.row_units + u;
                }
                a.k_cache[dst] = kb[t];
                a.v_cache[dst] = vb[t];
            }
        }
    }
}

// The CTA that finished sequence b's last chunk: argmax of every node from the
// merged row keys, then the walk, by warp 0 (the walk reads the current
// node's argmax from registers by warp shuffles, so a step costs no memory
// round trip).  The row keys and the counter are reset for the next call.
//
// Greedy: from the root, the smallest-index child whose candidate equals the
// current node's argmax, until there is none.
// Typical: first every thread of the CTA merges its share of one row's chunk
// sums (4 or 2 threads a row) into the row's (max, log2 S, log2 theta), while
// warp 0 also reads each child's candidate logit (gathered by the chunk CTAs).
// Then warp 0 builds the ancestor masks in registers, decides every edge,
// marks the nodes whose whole root path is accepted, takes the greatest depth
// among them and the union G of the root paths of the accepted nodes at that
// depth, and walks from the root through G, the smallest-index child at every
// step.  With a commit, the whole CTA then writes the accepted K/V.
template <typename T, bool TYPICAL>
__device__ void finish_sequence(const AcceptArgs &a, int b, const TreeRegs &tr) {
    __shared__ float4 s_row[kMaxTreeNodes];
    __shared__ int s_path[kMaxTreeNodes];
    __shared__ int s_par[kMaxTreeNodes];      // typical: the parent array, for the root-path walks
    __shared__ int s_len;
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int Tn = a.T;
    // Typical: tpr threads a row (neighbours in one warp) merge its chunk
    // records.  Each thread's first two records are loaded before warp 0's
    // key loads, so that the two round trips overlap.
    constexpr int kPre = 2;
    const int tpr = Tn <= 64 ? 4 : 2;
    const int row = threadIdx.x / tpr;
    const int q = threadIdx.x % tpr;
    const float4 *cs = a.chunk_sums + ((size_t)b * Tn + row) * a.n_chunks;
    float4 pre[kPre];
    if (TYPICAL) {
#pragma unroll
        for (int p = 0; p < kPre; ++p) {
            const int k = q + p * tpr;
            pre[p] = (row < Tn && k < a.n_chunks) ? __ldcg(cs + k) : make_float4(-INFINITY, 0.f, 0.f, 0.f);
        }
    }
    int am[kNodesPerLane];
    float xc[kNodesPerLane];
    uint64_t anc[kNodesPerLane][kMaskWords];
#pragma unroll
    for (int k = 0; k < kNodesPerLane; ++k) {
        am[k] = 0;
        xc[k] = -INFINITY;
    }
    if (warp == 0) {
        // the row keys and candidate logits are requested first; the typical
        // rule's ancestor masks are built while they are on their way
        unsigned long long key[kNodesPerLane];
#pragma unroll
        for (int k = 0; k < kNodesPerLane; ++k) {
            const int i = lane + 32 * k;
            key[k] = i < Tn ? __ldcg(a.row_key + (size_t)b * Tn + i) : 0ull;
            if (TYPICAL && i > 0 && i < Tn && tr.c[k] >= 0 && tr.c[k] < a.V)
                xc[k] = __ldcg(a.cand_x + (size_t)b * Tn + i);
        }
        if (TYPICAL) {
            // Each lane walks its nodes' root paths through the parent array
            // in shared memory, at most kShortDepth steps a node: the trees
            // of speculative decoding are shallow.  A deeper tree (or an
            // invalid one, which is reported and not walked) takes pointer
            // jumping instead: two nodes a lane and 6 rounds for trees of up
            // to 64 nodes, four nodes and 7 rounds above that.
            constexpr int kShortDepth = 8;
            bool done = !__any_sync(0xffffffffu, tr.invalid);
            if (done) {
#pragma unroll
                for (int k = 0; k < kNodesPerLane; ++k)
                    if (lane + 32 * k < Tn) s_par[lane + 32 * k] = tr.p[k];
                __syncwarp();
#pragma unroll
                for (int k = 0; k < kNodesPerLane; ++k) {
                    uint64_t m0 = 0ull, m1 = 0ull;
                    int j = lane + 32 * k < Tn ? lane + 32 * k : -1;
                    for (int d = 0; d < kShortDepth && j >= 0; ++d) {
                        if (j < 64) m0 |= 1ull << j;
                        else m1 |= 1ull << (j - 64);
                        j = s_par[j];
                    }
                    done = done && j < 0;
                    anc[k][0] = m0;
                    anc[k][1] = m1;
                }
                done = __all_sync(0xffffffffu, done);
            }
            if (!done) {
                if (Tn <= 64) {
                    tree_masks_jump<2>(*reinterpret_cast<const int(*)[2]>(&tr.p[0]), Tn,
                                       *reinterpret_cast<uint64_t(*)[2][kMaskWords]>(&anc[0]));
#pragma unroll
                    for (int k = 2; k < kNodesPerLane; ++k)
#pragma unroll
                        for (int w = 0; w < kMaskWords; ++w) anc[k][w] = 0ull;
                } else {
                    tree_masks_jump<kNodesPerLane>(tr.p, Tn, anc);
                }
            }
        }
#pragma unroll
        for (int k = 0; k < kNodesPerLane; ++k) {
            const int i = lane + 32 * k;
            if (i < Tn) {
                am[k] = (int)(0xFFFFFFFFu - (uint32_t)(key[k] & 0xFFFFFFFFull));
                a.argmax_out[(size_t)b * Tn + i] = am[k];
                a.row_key[(size_t)b * Tn + i] = 0ull;                      // ready for the next call
            }
        }
    }
    if (TYPICAL) {
        // the records of a row in the order k = q, q + tpr, ...
        float3 st = make_float3(-INFINITY, 0.f, 0.f);
#pragma unroll
        for (int p = 0; p < kPre; ++p) st = merge_sums(st, make_float3(pre[p].x, pre[p].y, pre[p].z));
        if (row < Tn) {
            for (int k = q + kPre * tpr; k < a.n_chunks; k += tpr) {
                const float4 v = __ldcg(cs + k);
                st = merge_sums(st, make_float3(v.x, v.y, v.z));
            }
        }
        for (int off = 1; off < tpr; off <<= 1) {
            const float3 o = make_float3(__shfl_xor_sync(0xffffffffu, st.x, off), __shfl_xor_sync(0xffffffffu, st.y, off),
                                         __shfl_xor_sync(0xffffffffu, st.z, off));
            st = merge_sums(st, o);
        }
        if (q == 0 && row < Tn) {
            // S >= 1 (the maximum's own term); entropy in bits H2 = log2 S - U / S
            const float log2s = lg2_approx(st.y);
            const float h2 = log2s - st.z / st.y;
            s_row[row] = make_float4(st.x, log2s, fminf(a.log2_eps, a.log2_delta - h2), 0.f);
        }
        __syncthreads();
    }
    if (warp == 0) walk_sequence<TYPICAL>(a, b, tr, am, xc, anc, s_row, s_path, &s_len);
    if (a.commit || a.wait_prior) {
        __syncthreads();
        if (a.commit) commit_sequence(a, b, s_path, s_len);
        // this grid completes only after the grid it may have overlapped
        if (a.wait_prior) wait_prerequisite_grids();
    }
}

template <typename T, bool TYPICAL>
__device__ __forceinline__ void accept_body(const AcceptArgs &a) {
    __shared__ uint64_t s_red[kThreads / 32];
    __shared__ float4 s_sum[kThreads / 32];
    __shared__ int s_seq_last;
    // a commit queued behind this call as a programmatic dependent may place
    // its CTAs now; it waits for this grid's completion before its first access
    allow_dependent_launch();
    const int warp = threadIdx.x >> 5;
    const int row = blockIdx.x;            // b * T + i
    const int chunk_id = blockIdx.y;
    const int b = row / a.T;
    const int node = row - b * a.T;
    const T *rowp = static_cast<const T *>(a.logits) + (size_t)row * a.V;

    // the tree, for the walk if this CTA turns out to finish the sequence
    // (and the candidate gather below); its loads overlap the scan
    TreeRegs tr;
    if (warp == 0) tr = load_tree(a, b);

    const int64_t lo = (int64_t)chunk_id * a.chunk;
    const int64_t hi = min((int64_t)a.V, lo + a.chunk);
    constexpr int E = 16 / sizeof(T);
    uint64_t best = 0ull;
    uint4 w[kUnits];
    int64_t head = 0, n_units = 0;
    if (lo < hi) {
        // scalar head up to a 16-byte boundary, vector body, scalar tail
        const uintptr_t addr = reinterpret_cast<uintptr_t>(rowp + lo);
        head = (int64_t)(((16 - (addr & 15)) & 15) / sizeof(T));
        if ((addr % sizeof(T)) != 0) head = hi - lo;       // cannot happen for valid tensors
        head = min(head, hi - lo);
        n_units = (hi - lo - head) / E;
        scan_scalar<T>(rowp, lo, lo + head, best);
        // rounds of the vector body (the typical rule's plan has one, whose
        // units stay in w for its sums)
        constexpr int kRound = kThreads * kUnits;
        const int nu = (int)n_units;           // at most four rounds
        for (int u0 = 0; u0 < nu; u0 += kRound)
            scan_vector<T>(rowp, lo + head + (int64_t)u0 * E, min(nu - u0, kRound), best, w);
        scan_scalar<T>(rowp, lo + head + n_units * E, hi, best);
    }

    if (TYPICAL) {
        // the thread's softmax sums relative to its own scaled maximum, from
        // the registers of the scan (head and tail elements are read again),
        // merged across the CTA with the chunk's key
        const int64_t t0 = lo + head + n_units * E;
        float mt = -INFINITY;
#pragma unroll
        for (int k = 0; k < kUnits; ++k)
            if (threadIdx.x + (int64_t)k * kThreads < n_units) mt = fmaxf(mt, unit_max(w[k], T()));
        for (int64_t v = lo + threadIdx.x; v < lo + head; v += kThreads) mt = fmaxf(mt, to_float(rowp[v]));
        for (int64_t v = t0 + threadIdx.x; v < hi; v += kThreads) mt = fmaxf(mt, to_float(rowp[v]));
        const float my = mt * a.y_scale;
        ExpSums acc;
#pragma unroll
        for (int k = 0; k < kUnits; ++k)
            if (threadIdx.x + (int64_t)k * kThreads < n_units) unit_sums(w[k], T(), a.y_scale, my, acc);
        for (int64_t v = lo + threadIdx.x; v < lo + head; v += kThreads) acc.add(to_float(rowp[v]), a.y_scale, my);
        for (int64_t v = t0 + threadIdx.x; v < hi; v += kThreads) acc.add(to_float(rowp[v]), a.y_scale, my);
        float3 st = make_float3(my, acc.sum_s(), acc.sum_u());
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
            const float3 o = make_float3(__shfl_xor_sync(0xffffffffu, st.x, off), __shfl_xor_sync(0xffffffffu, st.y, off),
                                         __shfl_xor_sync(0xffffffffu, st.z, off));
            st = merge_sums(st, o);
        }
        if ((threadIdx.x & 31) == 0) s_sum[warp] = make_float4(st.x, st.y, st.z, 0.f);
        // candidates of this node's children that fall in this chunk: their
        // logits for the walk
        if (warp == 0) {
#pragma unroll
            for (int k = 0; k < kNodesPerLane; ++k) {
                const int i = threadIdx.x + 32 * k;
                if (i >= 1 && i < a.T && tr.p[k] == node && tr.c[k] >= lo && tr.c[k] < hi) {
                    a.cand_x[(size_t)b * a.T + i] = to_float(rowp[tr.c[k]]);
                    __threadfence();
                }
            }
        }
    }
    best = block_max(best, s_red);            // its barrier also publishes s_sum
    if (TYPICAL && threadIdx.x == 0) {
        float3 st = make_float3(s_sum[0].x, s_sum[0].y, s_sum[0].z);
#pragma unroll
        for (int k = 1; k < kThreads / 32; ++k) st = merge_sums(st, make_float3(s_sum[k].x, s_sum[k].y, s_sum[k].z));
        __stcg(a.chunk_sums + (size_t)row * a.n_chunks + chunk_id, make_float4(st.x, st.y, st.z, 0.f));
    }

    // fold this chunk into the row's key and count it for its sequence; the
    // CTA that counts the sequence's last chunk runs the walk
    if (threadIdx.x == 0) {
        atomicMax(a.row_key + row, static_cast<unsigned long long>(best));
        __threadfence();                      // release: the key, sums and candidate logits
        const bool last = atomicAdd(a.seq_count + b, 1u) == (unsigned)(a.T * a.n_chunks) - 1u;
        if (last) __threadfence();            // acquire: every other CTA's; the barrier below
        s_seq_last = last;                    // passes it on, and they are read through L2
    }
    __syncthreads();
    if (!s_seq_last) return;
    finish_sequence<T, TYPICAL>(a, b, tr);
}

// The greedy kernel is held to 56 registers, so that two of its CTAs fit on an
// SM beside an attention CTA (160 registers x 224 threads) when the two calls
// run at the same time; the typical kernel needs more.
template <typename T>
__global__ void __maxnreg__(56) accept_kernel(const AcceptArgs a) {
    accept_body<T, false>(a);
}

// The typical kernel is held to 64 registers: four of its 256-thread CTAs an SM
// (65,536 registers), so that the 512 CTAs of a 7B-vocabulary step (64 rows x
// 8 chunks) are all resident at once on 152 SMs; at 71 registers three fit,
// and the grid took two waves.
template <typename T>
__global__ void __maxnreg__(64) accept_typical_kernel(const AcceptArgs a) {
    accept_body<T, true>(a);
}

}  // namespace

// Vocabulary chunk per CTA: rounds of kUnits 16-byte loads per thread (32 KB
// of bf16 or fp32 logits a round).  The typical rule keeps its one round in
// registers for the sums.  The greedy rule takes as many rounds (up to four)
// as bring the grid within `resident` CTAs, what the GPU holds at once, so
// that a call with many rows (a 128-node tree, a batch of sequences) runs in
// one wave instead of two or more; a grid that fits already keeps one round.
void accept_plan(int B, int T, int V, int dtype, bool typical, int resident, int *n_chunks, int *chunk) {
    constexpr int kMaxRounds = 4;
    const int elems = 16 / (dtype == CLOVER_F32 ? 4 : 2);
    const int round = kThreads * kUnits * elems;
    const long long one_round = (long long)B * T * ((V + round - 1) / round);
    const long long cap = resident > 0 ? resident : one_round;
    const int rounds = typical ? 1 : (int)std::min<long long>(kMaxRounds, std::max<long long>(1, (one_round + cap - 1) / cap));
    *chunk = round * rounds;
    *n_chunks = (V + *chunk - 1) / *chunk;
}

// CTAs of the greedy accept kernel the current device holds at once: four a
// multiprocessor (256 threads at 56 registers).
static int greedy_resident_ctas() {
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return 0;
    return 4 * sms;
}

// Keys and counters, then (typical acceptance) the 16-byte aligned chunk sums
// and the candidates' logits.
static size_t accept_sums_offset(int B, int T) {
    const size_t base = sizeof(unsigned long long) * (size_t)B * T + sizeof(unsigned) * (size_t)B;
    return (base + 15) & ~(size_t)15;
}

size_t accept_workspace_bytes(int B, int T, int V, int dtype) {
    (void)V;
    (void)dtype;
    return sizeof(unsigned long long) * (size_t)B * T + sizeof(unsigned) * (size_t)B;
}

size_t accept_typical_workspace_bytes(int B, int T, int V, int dtype) {
    int n_chunks, chunk;
    accept_plan(B, T, V, dtype, true, 0, &n_chunks, &chunk);
    return accept_sums_offset(B, T) + sizeof(float4) * (size_t)B * T * n_chunks + sizeof(float) * (size_t)B * T;
}

// A launch with after_prior is a programmatic dependent of the preceding
// kernel in the stream (which may let it start early).
template <typename T, bool TYPICAL>
static cudaError_t launch_kernel(const AcceptArgs &a, bool after_prior, cudaStream_t stream) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(a.B * a.T, a.n_chunks);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = after_prior ? 1 : 0;
    if (TYPICAL) return cudaLaunchKernelEx(&cfg, accept_typical_kernel<T>, a);
    return cudaLaunchKernelEx(&cfg, accept_kernel<T>, a);
}

cudaError_t launch_accept_call(const AcceptCall &c, cudaStream_t stream) {
    AcceptArgs a{};
    a.logits = c.logits;
    a.cand = c.cand;
    a.parent = c.parent;
    a.B = c.B;
    a.T = c.T;
    a.V = c.V;
    accept_plan(c.B, c.T, c.V, c.dtype, c.typical, c.typical ? 0 : greedy_resident_ctas(), &a.n_chunks, &a.chunk);
    a.argmax_out = c.argmax_out;
    a.path_out = c.path_out;
    a.accept_len = c.accept_len;
    a.bonus = c.bonus;
    a.row_key = static_cast<unsigned long long *>(c.workspace);
    a.seq_count = reinterpret_cast<unsigned *>(a.row_key + (size_t)c.B * c.T);
    if (c.typical) {
        a.chunk_sums = reinterpret_cast<float4 *>(static_cast<uint8_t *>(c.workspace) + accept_sums_offset(c.B, c.T));
        a.cand_x = reinterpret_cast<float *>(a.chunk_sums + (size_t)c.B * c.T * a.n_chunks);
        a.y_scale = c.y_scale;
        a.log2_eps = c.log2_eps;
        a.log2_delta = c.log2_delta;
    }
    if (c.commit) {
        a.commit = 1;
        a.k_cache = static_cast<uint4 *>(c.k_cache);
        a.v_cache = static_cast<uint4 *>(c.v_cache);
        a.k_new = static_cast<const uint4 *>(c.k_new);
        a.v_new = static_cast<const uint4 *>(c.v_new);
        a.cache_len = c.cache_len;
        a.new_cache_len = c.new_cache_len;
        a.src_index = c.src_index;
        a.Hkv = c.Hkv;
        a.Lcap = c.Lcap;
        a.row_units = c.D * (c.dtype == CLOVER_F32 ? 4 : 2) / 16;
        if (c.block_table) {
            a.block_table = c.block_table;
            a.page_size = c.page_size;
            while ((1 << a.page_shift) < c.page_size) ++a.page_shift;
            a.max_pages = c.max_pages;
            a.n_pages = c.n_pages;
        }
    }
    a.wait_prior = c.after_prior ? 1 : 0;
    a.status = c.status;
    if (c.dtype == CLOVER_F32)
        return c.typical ? launch_kernel<float, true>(a, c.after_prior, stream)
                         : launch_kernel<float, false>(a, c.after_prior, stream);
    return c.typical ? launch_kernel<__nv_bfloat16, true>(a, c.after_prior, stream)
                     : launch_kernel<__nv_bfloat16, false>(a, c.after_prior, stream);
}

}  // namespace clover
