// Tree-masked split-KV attention on CUDA cores (fp32 FMA), any dtype, any GQA
// group size.  This is the general path: it serves fp32 inputs (where the
// 1e-4 tolerance rules out reduced-precision tensor-core products) and shapes
// whose rows per KV head are too few for a dense tensor-core tile.
//
// The operation is the tree attention of the verification phase (Sections 2.1
// and 2.2 of the Clover paper): each tree node attends to every committed
// cache key and to the tree nodes on its own root path.
//
// Work decomposition: one CTA per (row tile of 32 query rows, cache-key split,
// KV head, sequence).  The T*G query rows of a KV head (node i, query head
// g*G + hh for row i*G + hh) share every K/V tile that CTA streams.  The split
// that owns the last cache range also processes the T tree keys under the
// ancestor mask and appends k_new/v_new to cache slots [L, L+T).  Partial
// (max, sum, unnormalised output) triples are merged by the CTA that arrives
// last at a per-head counter, which also resets the counter.
#include "common.cuh"

namespace clover {
namespace {

constexpr int kRT = 32;    // query rows per CTA
constexpr int kKT = 64;    // keys per tile
constexpr int kThreads = 256;

template <int D>
struct FmaSmem {
    static constexpr int DQ = D + 4;          // padded fp32 row of the Q and K tiles
    static constexpr int PS = kKT + 4;        // padded row of the P tile
    static constexpr int q_off = 0;
    static constexpr int k_off = q_off + kRT * DQ;
    static constexpr int v_off = k_off + kKT * DQ;
    static constexpr int p_off = v_off + kKT * D;
    static constexpr int floats = p_off + kRT * PS;
    static constexpr size_t bytes = sizeof(float) * floats;
};

// Raw 16-byte units of one K or V tile held by a thread between the global load
// and the shared-memory store.
template <typename T, int D>
struct TileRegs {
    static constexpr int kPerChunk = 16 / sizeof(T);                 // elements per 16 bytes
    static constexpr int kChunks = kKT * D / kPerChunk / kThreads;   // per thread, per tensor
    uint4 k[kChunks];
    uint4 v[kChunks];
};

template <typename T, int D>
__device__ __forceinline__ void chunk_coords(int j, int &key, int &col) {
    constexpr int per_row = D / TileRegs<T, D>::kPerChunk;
    const int c = threadIdx.x + kThreads * j;
    key = c / per_row;
    col = (c % per_row) * TileRegs<T, D>::kPerChunk;
}

// Global -> registers for one tile.  Cache tile: keys [base, base+kKT) of head g,
// valid below `end`.  Tree tile (tree == true): nodes [base, base+kKT) below T.
template <typename T, int D>
__device__ __forceinline__ void load_tile(const AttnArgs &a, int b, int g, bool tree, int base,
                                          int end, TileRegs<T, D> &r) {
    const T *kc = static_cast<const T *>(a.k_cache);
    const T *vc = static_cast<const T *>(a.v_cache);
    const T *kn = static_cast<const T *>(a.k_new);
    const T *vn = static_cast<const T *>(a.v_new);
#pragma unroll
    for (int j = 0; j < TileRegs<T, D>::kChunks; ++j) {
        int key, col;
        chunk_coords<T, D>(j, key, col);
        r.k[j] = make_uint4(0, 0, 0, 0);
        r.v[j] = make_uint4(0, 0, 0, 0);
        if (!tree) {
            const int slot = base + key;
            if (slot < end) {
                // dense: plane (b, g) of the cache; paged: row slot % page of
                // plane (page, g) of the pool
                const size_t row = a.block_table
                                       ? ((size_t)cache_page(a, b, slot) * a.Hkv + g) * a.page_size +
                                             (slot & (a.page_size - 1))
                                       : (size_t)(b * a.Hkv + g) * a.Lcap + slot;
                const size_t off = row * D + col;
                r.k[j] = __ldg(reinterpret_cast<const uint4 *>(kc + off));
                r.v[j] = __ldg(reinterpret_cast<const uint4 *>(vc + off));
            }
        } else if (base + key < a.T) {
            const size_t off = ((size_t)(b * a.T + base + key) * a.Hkv + g) * D + col;
            r.k[j] = __ldg(reinterpret_cast<const uint4 *>(kn + off));
            r.v[j] = __ldg(reinterpret_cast<const uint4 *>(vn + off));
        }
    }
}

template <typename T>
__device__ __forceinline__ void unpack(const uint4 &u, float *dst);

template <>
__device__ __forceinline__ void unpack<float>(const uint4 &u, float *dst) {
    *reinterpret_cast<float4 *>(dst) =
        make_float4(__uint_as_float(u.x), __uint_as_float(u.y), __uint_as_float(u.z), __uint_as_float(u.w));
}

template <>
__device__ __forceinline__ void unpack<__nv_bfloat16>(const uint4 &u, float *dst) {
    *reinterpret_cast<float4 *>(dst) = make_float4(__uint_as_float(u.x << 16), __uint_as_float(u.x & 0xFFFF0000u),
                                                   __uint_as_float(u.y << 16), __uint_as_float(u.y & 0xFFFF0000u));
    *reinterpret_cast<float4 *>(dst + 4) = make_float4(__uint_as_float(u.z << 16), __uint_as_float(u.z & 0xFFFF0000u),
                                                       __uint_as_float(u.w << 16), __uint_as_float(u.w & 0xFFFF0000u));
}

template <typename T, int D>
__global__ void __launch_bounds__(kThreads, 2) tree_attn_fma_kernel(const AttnArgs a) {
    allow_dependent_launch();
    using S = FmaSmem<D>;
    extern __shared__ float4 smem4[];
    float *smem = reinterpret_cast<float *>(smem4);
    float *sQ = smem + S::q_off;
    float *sK = smem + S::k_off;
    float *sV = smem + S::v_off;
    float *sP = smem + S::p_off;
    __shared__ uint64_t s_anc[kMaxTreeNodes * kMaskWords];
    __shared__ bool s_bad;
    __shared__ int s_is_last;

    const int tid = threadIdx.x;
    const int split = blockIdx.x % a.n_split;
    const int rt = blockIdx.x / a.n_split;
    const int g = blockIdx.y;
    const int b = blockIdx.z;
    const bool tree_cta = (split == a.n_split - 1);

    // committed length; an out-of-range one is reported and clamped so that
    // every access stays inside the cache (the result is then unspecified)
    int L = __ldg(a.cache_len + b);
    const bool cap_bad = (L < 0 || L + a.T > a.Lcap);
    if (cap_bad) {
        if (tid == 0 && split == 0 && rt == 0 && g == 0) report(a.status, CLOVER_ERR_CAPACITY);
        L = L < 0 ? 0 : a.Lcap - a.T;
    }

    if (tree_cta && tid < 32) {
        tree_masks_warp(a.parent + (size_t)b * a.T, a.T, s_anc, &s_bad);
    }

    // this split's cache keys [kbeg, kend)
    const int chunk = (((L + a.n_split - 1) / a.n_split) + kKT - 1) / kKT * kKT;
    const int kbeg = min(L, split * chunk);
    const int kend = min(L, kbeg + chunk);
    const int n_cache_tiles = (kend - kbeg + kKT - 1) / kKT;
    // the tree CTA ends with the tree keys, in tiles of kKT nodes
    const int n_tiles = n_cache_tiles + (tree_cta ? (a.T + kKT - 1) / kKT : 0);
    // first key (cache tile) or first node (tree tile) of tile t
    auto tile_base = [&](int t) { return t < n_cache_tiles ? kbeg + t * kKT : (t - n_cache_tiles) * kKT; };

    // Q tile, pre-multiplied by scale*log2(e)
    {
        const T *q = static_cast<const T *>(a.q);
        constexpr int per_row = D / 8;
        for (int c = tid; c < kRT * per_row; c += kThreads) {
            const int r = c / per_row;
            const int col = (c % per_row) * 8;
            const int R = rt * kRT + r;
            float v[8] = {0, 0, 0, 0, 0, 0, 0, 0};
            if (R < a.rows) {
                const int i = R / a.G;
                const int h = g * a.G + (R % a.G);
                Vec8<T>::load(q + ((size_t)(b * a.T + i) * a.Hq + h) * D + col, v);
            }
#pragma unroll
            for (int e = 0; e < 8; ++e) sQ[r * S::DQ + col + e] = v[e] * a.scale_log2;
        }
    }

    // thread roles: rows r0 = 2*(tid/16), r1 = r0 + 1; score keys kg + 16*j;
    // output columns dg*4.. (+64 for D = 128)
    const int r0 = 2 * (tid >> 4);
    const int kg = tid & 15;
    constexpr int NC = D / 64;   // float4 column groups per row per thread
    float o[2][NC][4];
#pragma unroll
    for (int r = 0; r < 2; ++r)
#pragma unroll
        for (int c = 0; c < NC; ++c)
#pragma unroll
            for (int e = 0; e < 4; ++e) o[r][c][e] = 0.f;
    float m_run[2] = {-INFINITY, -INFINITY};
    float l_run[2] = {0.f, 0.f};

    // tree node of each of this thread's rows (padding rows use the root)
    int node[2];
#pragma unroll
    for (int r = 0; r < 2; ++r) {
        const int R = rt * kRT + r0 + r;
        node[r] = R < a.rows ? R / a.G : 0;
    }

    TileRegs<T, D> regs;
    if (n_tiles > 0) load_tile<T, D>(a, b, g, n_cache_tiles == 0, tile_base(0), kend, regs);

    for (int t = 0; t < n_tiles; ++t) {
        const bool tree_tile = (t >= n_cache_tiles);
        const int base = tile_base(t);
        // registers -> shared memory (and, for the tree tile, the cache append)
#pragma unroll
        for (int j = 0; j < TileRegs<T, D>::kChunks; ++j) {
            int key, col;
            chunk_coords<T, D>(j, key, col);
            constexpr int per = TileRegs<T, D>::kPerChunk;
            unpack<T>(regs.k[j], sK + key * S::DQ + col);
            unpack<T>(regs.v[j], sV + key * D + col);
            if (tree_tile && a.append && rt == 0 && !cap_bad && base + key < a.T) {
                const size_t off = ((size_t)(b * a.Hkv + g) * a.Lcap + L + base + key) * D + col;
                *reinterpret_cast<uint4 *>(static_cast<T *>(a.k_cache) + off) = regs.k[j];
                *reinterpret_cast<uint4 *>(static_cast<T *>(a.v_cache) + off) = regs.v[j];
            }
            (void)per;
        }
        __syncthreads();
        if (t + 1 < n_tiles) load_tile<T, D>(a, b, g, t + 1 >= n_cache_tiles, tile_base(t + 1), kend, regs);

        // scores s[r][j] for rows r0+r and keys kg + 16 j
        float s[2][4];
#pragma unroll
        for (int r = 0; r < 2; ++r)
#pragma unroll
            for (int j = 0; j < 4; ++j) s[r][j] = 0.f;
#pragma unroll 8
        for (int d = 0; d < D; d += 4) {
            const float4 qa = *reinterpret_cast<const float4 *>(sQ + r0 * S::DQ + d);
            const float4 qb = *reinterpret_cast<const float4 *>(sQ + (r0 + 1) * S::DQ + d);
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const float4 k = *reinterpret_cast<const float4 *>(sK + (kg + 16 * j) * S::DQ + d);
                s[0][j] = fmaf(qa.x, k.x, fmaf(qa.y, k.y, fmaf(qa.z, k.z, fmaf(qa.w, k.w, s[0][j]))));
                s[1][j] = fmaf(qb.x, k.x, fmaf(qb.y, k.y, fmaf(qb.z, k.z, fmaf(qb.w, k.w, s[1][j]))));
            }
        }
        // mask: cache keys past kend, tree keys outside the root path
#pragma unroll
        for (int r = 0; r < 2; ++r)
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int kk = kg + 16 * j;
                bool ok;
                if (tree_tile) {
                    const int n = base + kk;
                    ok = (n < a.T) && ((s_anc[node[r] * kMaskWords + (n >> 6)] >> (n & 63)) & 1ull);
                }
                else ok = (base + kk < kend);
                if (!ok) s[r][j] = -INFINITY;
            }
        // online softmax over the 16 lanes that share a row
        float alpha[2];
#pragma unroll
        for (int r = 0; r < 2; ++r) {
            float mx = fmaxf(fmaxf(s[r][0], s[r][1]), fmaxf(s[r][2], s[r][3]));
#pragma unroll
            for (int off = 8; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
            const float m_new = fmaxf(m_run[r], mx);
            const float ref = (m_new == -INFINITY) ? 0.f : m_new;
            alpha[r] = exp2f(m_run[r] - ref);
            float sum = 0.f;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                s[r][j] = exp2f(s[r][j] - ref);
                sum += s[r][j];
            }
#pragma unroll
            for (int off = 8; off > 0; off >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
            l_run[r] = l_run[r] * alpha[r] + sum;
            m_run[r] = m_new;
#pragma unroll
            for (int j = 0; j < 4; ++j) sP[(r0 + r) * S::PS + kg + 16 * j] = s[r][j];
        }
        __syncthreads();

        // o = o * alpha + P V
#pragma unroll
        for (int r = 0; r < 2; ++r)
#pragma unroll
            for (int c = 0; c < NC; ++c)
#pragma unroll
                for (int e = 0; e < 4; ++e) o[r][c][e] *= alpha[r];
#pragma unroll 4
        for (int k = 0; k < kKT; k += 4) {
            const float4 pa = *reinterpret_cast<const float4 *>(sP + r0 * S::PS + k);
            const float4 pb = *reinterpret_cast<const float4 *>(sP + (r0 + 1) * S::PS + k);
            const float pav[4] = {pa.x, pa.y, pa.z, pa.w};
            const float pbv[4] = {pb.x, pb.y, pb.z, pb.w};
#pragma unroll
            for (int kk = 0; kk < 4; ++kk) {
#pragma unroll
                for (int c = 0; c < NC; ++c) {
                    const float4 v = *reinterpret_cast<const float4 *>(sV + (k + kk) * D + c * 64 + kg * 4);
                    o[0][c][0] = fmaf(pav[kk], v.x, o[0][c][0]);
                    o[0][c][1] = fmaf(pav[kk], v.y, o[0][c][1]);
                    o[0][c][2] = fmaf(pav[kk], v.z, o[0][c][2]);
                    o[0][c][3] = fmaf(pav[kk], v.w, o[0][c][3]);
                    o[1][c][0] = fmaf(pbv[kk], v.x, o[1][c][0]);
                    o[1][c][1] = fmaf(pbv[kk], v.y, o[1][c][1]);
                    o[1][c][2] = fmaf(pbv[kk], v.z, o[1][c][2]);
                    o[1][c][3] = fmaf(pbv[kk], v.w, o[1][c][3]);
                }
            }
        }
        __syncthreads();
    }

    if (tree_cta && tid == 0 && rt == 0 && s_bad) report(a.status, CLOVER_ERR_BAD_TREE);

    T *out = static_cast<T *>(a.out);
    if (a.n_split == 1) {
#pragma unroll
        for (int r = 0; r < 2; ++r) {
            const int R = rt * kRT + r0 + r;
            if (R >= a.rows) continue;
            const int i = R / a.G;
            const int h = g * a.G + (R % a.G);
            if (!CLOVER_IN(a.status, ((size_t)b * a.T + i) * a.Hq + h, (size_t)a.B * a.T * a.Hq)) continue;
            const float inv = 1.f / l_run[r];
            T *dst = out + ((size_t)(b * a.T + i) * a.Hq + h) * D;
#pragma unroll
            for (int c = 0; c < NC; ++c)
#pragma unroll
                for (int e = 0; e < 4; ++e) dst[c * 64 + kg * 4 + e] = from_float<T>(o[r][c][e] * inv);
        }
        return;
    }

    // publish this split's partial result
    const size_t head_tile = (size_t)(b * a.Hkv + g) * a.row_tiles + rt;
    float *po = a.part_o + (head_tile * a.n_split + split) * kRT * D;
    float *pml = a.part_ml + (head_tile * a.n_split + split) * kRT * 2;
    // the workspace starts with the counters: slots must end inside it
    if (CLOVER_IN(a.status, (const char *)(pml + kRT * 2) - (const char *)a.counters - 1, a.ws_bytes) &&
        CLOVER_IN(a.status, head_tile, (size_t)a.B * a.Hkv * a.row_tiles)) {
#pragma unroll
        for (int r = 0; r < 2; ++r) {
#pragma unroll
            for (int c = 0; c < NC; ++c)
                *reinterpret_cast<float4 *>(po + (r0 + r) * D + c * 64 + kg * 4) =
                    make_float4(o[r][c][0], o[r][c][1], o[r][c][2], o[r][c][3]);
            if (kg == 0) {
                pml[(r0 + r) * 2] = m_run[r];
                pml[(r0 + r) * 2 + 1] = l_run[r];
            }
        }
    }
    __threadfence();
    __syncthreads();
    if (tid == 0) {
        const unsigned prev = atomicAdd(a.counters + head_tile, 1u);
        s_is_last = (prev == (unsigned)a.n_split - 1u);
    }
    __syncthreads();
    if (!s_is_last) return;
    __threadfence();

    // last CTA of this (sequence, head, row tile): merge the n_split partials
    const float *po_all = a.part_o + head_tile * a.n_split * kRT * D;
    const float *pml_all = a.part_ml + head_tile * a.n_split * kRT * 2;
    constexpr int kColsPerThread = D / 8;       // 8 threads per row
    const int r = tid / 8;
    const int c0 = (tid % 8) * kColsPerThread;
    const int R = rt * kRT + r;
    if (R < a.rows) {
        float M = -INFINITY;
        for (int sp = 0; sp < a.n_split; ++sp) M = fmaxf(M, __ldcg(pml_all + (sp * kRT + r) * 2));
        float acc[kColsPerThread];
#pragma unroll
        for (int e = 0; e < kColsPerThread; ++e) acc[e] = 0.f;
        float lsum = 0.f;
        for (int sp = 0; sp < a.n_split; ++sp) {
            const float ms = __ldcg(pml_all + (sp * kRT + r) * 2);
            const float ls = __ldcg(pml_all + (sp * kRT + r) * 2 + 1);
            const float w = (ms == -INFINITY) ? 0.f : exp2f(ms - M);
            lsum += w * ls;
            const float *src = po_all + ((size_t)sp * kRT + r) * D + c0;
#pragma unroll
            for (int e = 0; e < kColsPerThread; e += 4) {
                const float4 x = __ldcg(reinterpret_cast<const float4 *>(src + e));
                acc[e] = fmaf(w, x.x, acc[e]);
                acc[e + 1] = fmaf(w, x.y, acc[e + 1]);
                acc[e + 2] = fmaf(w, x.z, acc[e + 2]);
                acc[e + 3] = fmaf(w, x.w, acc[e + 3]);
            }
        }
        const float inv = 1.f / lsum;
        const int i = R / a.G;
        const int h = g * a.G + (R % a.G);
        T *dst = out + ((size_t)(b * a.T + i) * a.Hq + h) * D + c0;
        if (CLOVER_IN(a.status, ((size_t)b * a.T + i) * a.Hq + h, (size_t)a.B * a.T * a.Hq)) {
#pragma unroll
            for (int e = 0; e < kColsPerThread; ++e) dst[e] = from_float<T>(acc[e] * inv);
        }
    }
    if (tid == 0) a.counters[head_tile] = 0u;   // ready for the next call
}

template <typename T, int D>
cudaError_t launch(const AttnArgs &a, cudaStream_t stream) {
    static unsigned long long done[64];
    auto kernel = tree_attn_fma_kernel<T, D>;
    cudaError_t e = ensure_smem_attr(kernel, FmaSmem<D>::bytes, done);
    if (e != cudaSuccess) return e;
    dim3 grid(a.n_split * a.row_tiles, a.Hkv, a.B);
    kernel<<<grid, kThreads, FmaSmem<D>::bytes, stream>>>(a);
    return cudaGetLastError();
}

}  // namespace

int fma_row_tile() { return kRT; }

cudaError_t launch_tree_attn_fma(const AttnArgs &a, cudaStream_t stream) {
    if (a.dtype == CLOVER_F32) return a.D == 64 ? launch<float, 64>(a, stream) : launch<float, 128>(a, stream);
    return a.D == 64 ? launch<__nv_bfloat16, 64>(a, stream) : launch<__nv_bfloat16, 128>(a, stream);
}

}  // namespace clover
