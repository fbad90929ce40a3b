// Draft side of a Clover head step (Section 3): the top-k of the shared LM
// head's logits, and the regressive connection's embedding of the previous
// token (Section 3.4: its row of the LM-head weight, normalised).
//
// Top-k: one CTA per (row, 8192-element chunk).  Every value becomes a packed
// 64-bit key (order-preserving value bits high, bit-inverted index low), so an
// unsigned max picks "largest value, then smallest index".  A CTA takes its
// chunk's k best keys in k rounds of a block-wide max, each thread proposing
// its best key not yet taken; it writes them to the workspace, and the CTA that
// finishes a row's last chunk (an arrival counter) selects the row's k best
// among the chunks' the same way and resets the counter.  In the chunk phase a
// thread keeps its 32 values as 32-bit order bits and its best one between
// rounds: only the thread whose key won a round looks through its values again.
#include "common.cuh"

namespace clover {
namespace {

constexpr int kTkThreads = 256;
constexpr int kTkPer = 32;                               // values per thread per chunk
constexpr int kTkChunk = kTkThreads * kTkPer;            // 8192
constexpr int kTkMaxK = 32;

__device__ __forceinline__ uint32_t tk_order_bits(float x) {
    uint32_t u = __float_as_uint(x);
    if (u == 0x80000000u) u = 0u;                        // -0 == +0
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__device__ __forceinline__ uint64_t tk_key(float x, uint32_t index) {
    return (static_cast<uint64_t>(tk_order_bits(x)) << 32) | static_cast<uint64_t>(0xFFFFFFFFu - index);
}

__device__ __forceinline__ float tk_value(uint64_t key) {
    const uint32_t ob = static_cast<uint32_t>(key >> 32);
    return __uint_as_float((ob & 0x80000000u) ? (ob & 0x7FFFFFFFu) : ~ob);
}

__device__ __forceinline__ uint64_t tk_umax(uint64_t a, uint64_t b) { return a > b ? a : b; }

// Block-wide max of one key per thread; every thread gets the result.
__device__ __forceinline__ uint64_t tk_block_max(uint64_t v, uint64_t *s_red) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v = tk_umax(v, __shfl_xor_sync(0xffffffffu, v, off));
    const int warp = threadIdx.x >> 5;
    __syncthreads();                                     // s_red is free (previous round read it)
    if ((threadIdx.x & 31) == 0) s_red[warp] = v;
    __syncthreads();
    uint64_t m = 0ull;
#pragma unroll
    for (int w = 0; w < kTkThreads / 32; ++w) m = tk_umax(m, s_red[w]);
    return m;
}

// The k best of NK keys per thread (keys[i] == 0: none), into out[0..k).
template <int NK>
__device__ __forceinline__ void tk_select(uint64_t (&keys)[NK], int k, uint64_t *out, uint64_t *s_red) {
    for (int j = 0; j < k; ++j) {
        uint64_t best = 0ull;
        int bi = -1;
#pragma unroll
        for (int i = 0; i < NK; ++i)
            if (keys[i] > best) {
                best = keys[i];
                bi = i;
            }
        const uint64_t m = tk_block_max(best, s_red);
        // keys are distinct (their indices are), so one thread owns the winner
        if (bi >= 0 && best == m) {
#pragma unroll
            for (int i = 0; i < NK; ++i)
                if (i == bi) keys[i] = 0ull;
        }
        if (threadIdx.x == 0) out[j] = m;
    }
}

struct TopkArgs {
    const float *x;
    int R, V, k, n_chunks;
    float *values;
    int32_t *indices;
    unsigned long long *cand;                            // [R, n_chunks, k]
    unsigned *count;                                     // [R]
    int32_t *status;
};

__global__ void __launch_bounds__(kTkThreads) topk_kernel(const TopkArgs a) {
    __shared__ uint64_t s_red[kTkThreads / 32];
    __shared__ uint64_t s_out[kTkMaxK];
    __shared__ int s_last;
    const int r = blockIdx.x;
    const int c = blockIdx.y;
    const float *row = a.x + (size_t)r * a.V;
    const int lo = c * kTkChunk;
    // value j of this thread is element lo + threadIdx.x + j * kTkThreads; its
    // order bits, 0 for none (below every value's, so never proposed)
    uint32_t ob[kTkPer];
#pragma unroll
    for (int j = 0; j < kTkPer; ++j) {
        const int v = lo + threadIdx.x + j * kTkThreads;
        ob[j] = v < a.V ? tk_order_bits(__ldcs(row + v)) : 0u;
    }
    // the thread's best value not yet taken: the largest order bits, the
    // smallest j (so the smallest index) among equal ones
    uint32_t bv = 0u;
    int bj = -1;
    auto rescan = [&]() {
        bv = 0u;
        bj = -1;
#pragma unroll
        for (int j = 0; j < kTkPer; ++j)
            if (ob[j] > bv) {
                bv = ob[j];
                bj = j;
            }
    };
    rescan();
    for (int i = 0; i < a.k; ++i) {
        const uint64_t key = bj >= 0 ? (static_cast<uint64_t>(bv) << 32) |
                                           static_cast<uint64_t>(0xFFFFFFFFu - (uint32_t)(lo + threadIdx.x + bj * kTkThreads))
                                     : 0ull;
        const uint64_t m = tk_block_max(key, s_red);
        // keys are distinct (their indices are), so one thread owns the winner
        if (bj >= 0 && key == m) {
#pragma unroll
            for (int j = 0; j < kTkPer; ++j)
                if (j == bj) ob[j] = 0u;
            rescan();
        }
        if (threadIdx.x == 0) s_out[i] = m;
    }
    if (threadIdx.x == 0) {
        unsigned long long *dst = a.cand + ((size_t)r * a.n_chunks + c) * a.k;
        for (int j = 0; j < a.k; ++j) dst[j] = s_out[j];
        __threadfence();
        const bool last = atomicAdd(a.count + r, 1u) == (unsigned)a.n_chunks - 1u;
        if (last) {
            a.count[r] = 0u;                             // ready for the next call
            __threadfence();
        }
        s_last = last;
    }
    __syncthreads();
    if (!s_last) return;
    // the row's k best among the chunks' k best (at most 16 x 32 keys, two per thread)
    uint64_t ck[2];
    const int n = a.n_chunks * a.k;
#pragma unroll
    for (int j = 0; j < 2; ++j) {
        const int i = threadIdx.x + j * kTkThreads;
        ck[j] = i < n ? __ldcg(a.cand + (size_t)r * a.n_chunks * a.k + i) : 0ull;
    }
    tk_select<2>(ck, a.k, s_out, s_red);
    __syncthreads();
    if (threadIdx.x < a.k) {
        const uint64_t key = s_out[threadIdx.x];
        a.values[(size_t)r * a.k + threadIdx.x] = tk_value(key);
        a.indices[(size_t)r * a.k + threadIdx.x] = (int32_t)(0xFFFFFFFFu - (uint32_t)(key & 0xFFFFFFFFull));
    }
}

// 16-byte chunks of a row that each thread of the embedding keeps in registers
// (rows of up to 8 * 256 * 4 = 8192 bf16 take the one-read path).
constexpr int kEmbedChunks = 4;

__device__ __forceinline__ float bf16_lo(uint32_t u) { return __uint_as_float(u << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t u) { return __uint_as_float(u & 0xFFFF0000u); }

// Sum of squares over a CTA of 256 threads (8 warps).
__device__ __forceinline__ float block_sum(float s, float *s_sum) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
    if ((threadIdx.x & 31) == 0) s_sum[threadIdx.x >> 5] = s;
    __syncthreads();
    float tot = 0.f;
#pragma unroll
    for (int i = 0; i < 8; ++i) tot += s_sum[i];
    return tot;
}

// e[r] = w[t] / ||w[t]||_2, one CTA per row.  Rows of whole 16-byte chunks
// (H a multiple of 8, 16-byte aligned w and e) are read once, all of a
// thread's chunks at the same time, and scaled from registers; others take a
// plain element loop.
__global__ void __launch_bounds__(256) embed_rows_kernel(const __nv_bfloat16 *w, const int32_t *tokens,
                                                         __nv_bfloat16 *e, int V, int H, int32_t *status) {
    // a linear layer queued behind this call as a programmatic dependent may
    // start its set-up now; it waits for this grid before it reads e
    allow_dependent_launch();
    __shared__ float s_sum[8];
    const int r = blockIdx.x;
    const int t = __ldg(tokens + r);
    __nv_bfloat16 *dst = e + (size_t)r * H;
    if (t < 0 || t >= V) {
        if (threadIdx.x == 0) report(status, CLOVER_ERR_INVALID_ARG);
        for (int h = threadIdx.x; h < H; h += blockDim.x) dst[h] = __float2bfloat16_rn(0.f);
        return;
    }
    const __nv_bfloat16 *src = w + (size_t)t * H;
    const int n_chunks = H / 8;
    const bool vec = (H % 8) == 0 && n_chunks <= kEmbedChunks * 256 &&
                     ((reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst)) & 15) == 0;
    if (vec) {
        uint4 c[kEmbedChunks];
#pragma unroll
        for (int k = 0; k < kEmbedChunks; ++k) {
            const int i = threadIdx.x + 256 * k;
            c[k] = i < n_chunks ? __ldg(reinterpret_cast<const uint4 *>(src) + i) : make_uint4(0, 0, 0, 0);
        }
        float s = 0.f;
#pragma unroll
        for (int k = 0; k < kEmbedChunks; ++k) {
            const uint32_t u[4] = {c[k].x, c[k].y, c[k].z, c[k].w};
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                s = fmaf(bf16_lo(u[q]), bf16_lo(u[q]), s);
                s = fmaf(bf16_hi(u[q]), bf16_hi(u[q]), s);
            }
        }
        const float tot = block_sum(s, s_sum);
        const float inv = tot > 0.f ? 1.f / sqrtf(tot) : 0.f;
#pragma unroll
        for (int k = 0; k < kEmbedChunks; ++k) {
            const int i = threadIdx.x + 256 * k;
            if (i >= n_chunks) break;
            const uint32_t u[4] = {c[k].x, c[k].y, c[k].z, c[k].w};
            uint32_t o[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const __nv_bfloat162 v = __floats2bfloat162_rn(bf16_lo(u[q]) * inv, bf16_hi(u[q]) * inv);
                o[q] = *reinterpret_cast<const uint32_t *>(&v);
            }
            reinterpret_cast<uint4 *>(dst)[i] = make_uint4(o[0], o[1], o[2], o[3]);
        }
        return;
    }
    float s = 0.f;
    for (int h = threadIdx.x; h < H; h += blockDim.x) {
        const float v = __bfloat162float(src[h]);
        s = fmaf(v, v, s);
    }
    const float tot = block_sum(s, s_sum);
    const float inv = tot > 0.f ? 1.f / sqrtf(tot) : 0.f;
    for (int h = threadIdx.x; h < H; h += blockDim.x) dst[h] = __float2bfloat16_rn(__bfloat162float(src[h]) * inv);
}

}  // namespace

int topk_max_k() { return kTkMaxK; }

size_t topk_workspace_bytes(int R, int V, int k) {
    const int n_chunks = (V + kTkChunk - 1) / kTkChunk;
    return sizeof(unsigned long long) * (size_t)R * n_chunks * k + sizeof(unsigned) * (size_t)R;
}

int topk_max_chunks() { return 2 * kTkThreads / kTkMaxK; }

cudaError_t launch_topk(const float *x, int R, int V, int k, float *values, int32_t *indices, void *workspace,
                        int32_t *status, cudaStream_t stream) {
    TopkArgs a;
    a.x = x;
    a.R = R;
    a.V = V;
    a.k = k;
    a.n_chunks = (V + kTkChunk - 1) / kTkChunk;
    a.values = values;
    a.indices = indices;
    a.cand = static_cast<unsigned long long *>(workspace);
    a.count = reinterpret_cast<unsigned *>(a.cand + (size_t)R * a.n_chunks * k);
    a.status = status;
    topk_kernel<<<dim3(R, a.n_chunks), kTkThreads, 0, stream>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_embed_rows(const void *w, const int32_t *tokens, void *e, int R, int V, int H, int32_t *status,
                              cudaStream_t stream) {
    embed_rows_kernel<<<R, 256, 0, stream>>>(static_cast<const __nv_bfloat16 *>(w), tokens,
                                             static_cast<__nv_bfloat16 *>(e), V, H, status);
    return cudaGetLastError();
}

}  // namespace clover
