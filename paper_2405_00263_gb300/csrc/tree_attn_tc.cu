// Tree-masked split-KV attention on the 5th-generation tensor cores (tcgen05,
// sm_103a) for bf16 inputs.
//
// The operation is the tree attention of the verification phase (Sections 2.1
// and 2.2 of the Clover paper): every tree node attends to all committed cache
// keys and to the tree nodes on its own root path (the tree topology as mask).
//
// One CTA per (row tile of up to 128 query rows, cache-key split, sequence x
// KV head).  The T*G query rows of a KV head (row i*G + hh = node i, query head
// g*G + hh) share every K/V tile, so per 128-key tile:
//   S  = Q K^T        tcgen05.mma M=128 N=128, D/16 instructions of K=16
//                     (Q in TMEM, K K-major in smem; S in TMEM)
//   P  = 2^(S*c - m)  online softmax in registers; bf16 P written back to TMEM
//                     over the S tile it came from
//   O += P V          tcgen05.mma M=128 N=D, 8 instructions of K=16 over the
//                     tile's 128 keys (P in TMEM, V MN-major in smem)
// Q and O stay in TMEM for the whole key range, so the tensor core reads only
// K and V from shared memory (which the TMA writes fill at the same time).
// Each row keeps a reference max m; P is taken relative to it, and m (with O
// and the row sum) is only moved when a tile's max exceeds it by more than
// 2^8, so O is rarely rescaled.  A tile of at most 64 real rows repeats its Q
// rows in TMEM lanes 64-127, and the rows' keys split into two halves, each a
// separate online softmax merged after the loop, so all four softmax warps work.
// Warp roles (224 threads): warp w in 0-3 writes the Q rows of TMEM lanes
// 32w.. and runs the softmax, rescales and the epilogue of those lanes (the
// lanes warp w may access); warp 4 issues the TMA loads of the K tiles (its
// own ring); warp 6 those of the V tiles; warp 5 allocates TMEM and issues the
// MMAs from one thread.  A full 128-row tile (KS = 1) adds warps 7-10 (352
// threads): a second softmax warp per lane quadrant, the two taking 64 keys
// of a tile each and sharing one reference max through shared memory.  The
// cache tiles are read with an L2 evict-first policy: they are read once, and
// must not push out of L2 what is reused.
// The split that owns the last cache range also takes the tile of T tree keys
// (read from k_new/v_new) under the ancestor bitmask, as its first tile; its
// producers also append the tree keys and values to the cache when asked, by
// TMA stores of that tile.
//
// Split merge: every CTA of a (sequence, head, row tile) group but the last
// (the one with the tree tile, which ends last) combines its two key halves,
// copies its partial result (unnormalised O rows with their max m and sum l)
// from shared memory to its workspace slot by one bulk copy and counts itself
// in at the group's arrival counter; then it exits, so its SM is free.  The
// last CTA waits (bounded) for the others' arrival, bulk-loads their rows and
// merges every source of a row (its own key halves and the other splits' rows)
// straight into the output.
//
// Programmatic dependent launch (AttnArgs::pdl): the grid may start while the
// kernel before it in the stream still runs.  Barrier setup and the TMEM
// allocation come first.  Every read of an input comes after
// griddepcontrol.wait, except when the caller states that they are not being
// written by the kernels that may still run: with cache_early the cache
// length, the block table and the cache tiles of the free ring stages are read
// before it; with inputs_early every input is, and only the writes (the
// append, the workspace, the output) wait.
//
// Every mbarrier wait is bounded; on a timeout the CTA reports
// CLOVER_ERR_TIMEOUT, winds down, waits (bounded) for its copies in flight and
// frees its TMEM.
#include "common.cuh"
#include "tc_ptx.cuh"
#include "tmap_host.cuh"

namespace clover {
namespace {

using namespace tc;

constexpr int BM = 128;                 // query rows per CTA (MMA M)
constexpr int BN = 128;                 // keys per tile (the N of the S MMA)
constexpr int kMinPage = 16;             // smallest page of a paged cache (rows)
constexpr int kMaxBoxes = BN / kMinPage; // TMA boxes of one paged cache tile
static_assert(kMaxBoxes * 2 <= 32, "a paged tile's boxes and column blocks go one to a producer lane");
constexpr int kPageSmem = 512;           // page ids of a split staged in shared memory
constexpr int kKProducerWarp = 4;
constexpr int kMmaWarp = 5;
constexpr int kVProducerWarp = 6;
constexpr int kSoft2Warp = 7;           // KS = 1: warps 7-10 are a second softmax group
// Threads of a CTA: 7 warps; with KS = 1 (full 128-row tiles) 4 more, so that
// two softmax warps share each TMEM lane quadrant, 64 keys of a tile each.
template <int KS>
constexpr int threads_of() { return KS == 1 ? 352 : 224; }
constexpr int kMaxSplits = 8;           // key ranges per (sequence, head, row tile)
constexpr int kMaxSrc = kMaxSplits + 2;  // partial rows merged into one output row (own halves + others)
constexpr float kRescale = 8.0f;        // move the reference max only past 2^8 growth
constexpr uint64_t kWaitNs = 500ull * 1000 * 1000;   // 0.5 s per wait

// Shared-memory plan: the K and V rings (Q lives in TMEM).  KS = key groups
// per tile row: with KS = 2 (a tile of at most 64 real query rows) the Q rows
// of TMEM lanes 64-127 repeat those of lanes 0-63, so every real row's scores
// sit in two lane quadrants and the four softmax warps each take half of a
// tile's keys.
template <int D, int KS>
struct TcSmem {
    static constexpr int NSK = (D == 128) ? 3 : 4;   // K ring stages
    static constexpr int NSV = (D == 128) ? 3 : 4;   // V ring stages
    static constexpr int DH = D / 64;                // 128-byte column blocks per row
    static constexpr int kv_bytes = BN * D * 2;      // one K or V tile: [DH][BN][128 B]
    static constexpr int k_off = 0;
    static constexpr int v_off = k_off + NSK * kv_bytes;
    static constexpr int bar_off = v_off + NSV * kv_bytes;
    static constexpr int n_bars = 2 * NSK + 2 * NSV + 14;
    static constexpr int misc_off = bar_off + 8 * n_bars;          // tmem addr, abort, bad
    static constexpr int anc_off = misc_off + 16;                  // ancestor masks [128][2]
    static constexpr int pages_off = anc_off + kMaxTreeNodes * kMaskWords * 8;   // paged: page ids of the split
    static constexpr int wts_off = pages_off + kPageSmem * 4;      // merge weights [BM][kMaxSrc]
    static constexpr int par_off = wts_off + BM * kMaxSrc * 4;     // the tree's parent array [128]
    static constexpr int orow_off = par_off + kMaxTreeNodes * 4;   // output row of each tile row [BM]
    static constexpr int x_off = orow_off + BM * 4;              // KS = 1: pair exchange [2][2][BM] + flags [2][2][4]
    static constexpr int total = x_off + 2 * 2 * BM * 4 + 2 * 2 * 4 * 4;
    static constexpr size_t alloc = total + 1024;                  // base rounded up to 1024 bytes
    // TMEM columns: S/P 2 x BN, O D, Q D / 2 (two bf16 per column), rounded up
    // to a power of two.  All 512 columns of an SM go to one CTA only when
    // the shared memory already keeps a second CTA off the SM (a second CTA
    // would wait in tcgen05.alloc).
    static constexpr uint32_t tmem_cols = (2 * BN + D + D / 2 <= 256) ? 256 : 512;
    static_assert(tmem_cols < 512 || 2 * alloc > 228 * 1024, "512 TMEM columns need one CTA per SM");
    // After the key loop the rings hold the partial results: this CTA's at the
    // start of the K ring, one fp32 row of D + 4 floats per query row (O, then
    // m and l; with KS = 2 rows 64-127 first carry the second key half's
    // rows), and, in the merging CTA, the other splits' rows after it, in the
    // same row format (the workspace's format too).
    static constexpr int po_stride = D + 4;
    static constexpr int own_bytes = BM * po_stride * 4;
    static constexpr int recv_bytes = (NSK + NSV) * kv_bytes - own_bytes;
    static_assert(own_bytes % 16 == 0 && (po_stride * 4) % 16 == 0, "bulk copies move 16-byte units");
    static_assert(own_bytes <= NSK * kv_bytes, "partial result must fit in the K ring");
    static_assert(recv_bytes >= (kMaxSplits - 1) * po_stride * 4, "a merge pass must hold one row of each split");
    static_assert(KS == 1 || BM == 128, "the second key half's rows sit 64 rows below the first's");
    static_assert(alloc <= 227 * 1024, "shared memory budget");
};

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t *>(&v);
}

__device__ __forceinline__ float rcp_approx(float x) {
    float y;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// One pass of the merge of partial softmax results into output rows (Section
// 2.2's attention over the whole key range, from per-range partial results):
//   O = sum_s 2^(m_s - M) O_s / sum_s 2^(m_s - M) l_s,  M = max_s m_s,
// over the sources s of a row, with the weights w[row][s] = 2^(m_s - M) /
// sum_s 2^(m_s - M) l_s already in shared memory.  Source s < KS of row rr is
// this CTA's row rr + 64 s of `own` (its key halves); source KS + k is the
// k-th other split's, row rr - p0 of slot k of `recv`.  Rows [p0, p1).  A warp
// takes 8 rows at a time and lane l their columns [4 l, 4 l + 4) (D = 128;
// D = 64 uses lanes 0-15): each shared-memory load of the warp reads one row's
// contiguous 512 bytes, free of bank conflicts, and 8 are in flight per
// source.  Output row rr goes to out + orow[rr] * D; with `out` == nullptr the
// result (weights not normalised) goes back to `own` row rr instead.
template <int D, int KS>
__device__ __forceinline__ void merge_pass(float *own, const float *recv, const float *wts, const unsigned *orow,
                                           int n_src, int rpp, int p0, int p1, __nv_bfloat16 *out) {
    constexpr int PS = D + 4;
    constexpr int RG = 8;                     // rows per warp step
    const int lane = threadIdx.x & 31;
    const int c = lane * 4;
    if (c >= D) return;
    const int n_warps = blockDim.x >> 5;
    for (int r0 = p0 + (int)(threadIdx.x >> 5) * RG; r0 < p1; r0 += n_warps * RG) {
        const int nr = min(RG, p1 - r0);
        float4 acc[RG];
#pragma unroll
        for (int k = 0; k < RG; ++k) acc[k] = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 1
        for (int sidx = 0; sidx < n_src; ++sidx) {
            const float *base = sidx < KS ? own + (r0 + 64 * sidx) * PS : recv + ((sidx - KS) * rpp + r0 - p0) * PS;
#pragma unroll
            for (int k = 0; k < RG; ++k) {
                if (k < nr) {
                    const float w = wts[(r0 + k) * kMaxSrc + sidx];
                    const float4 x = *reinterpret_cast<const float4 *>(base + k * PS + c);
                    acc[k].x = fmaf(w, x.x, acc[k].x);
                    acc[k].y = fmaf(w, x.y, acc[k].y);
                    acc[k].z = fmaf(w, x.z, acc[k].z);
                    acc[k].w = fmaf(w, x.w, acc[k].w);
                }
            }
        }
#pragma unroll
        for (int k = 0; k < RG; ++k) {
            if (k >= nr) continue;
            const int rr = r0 + k;
            if (out == nullptr) {
                *reinterpret_cast<float4 *>(own + rr * PS + c) = acc[k];
            } else {
                uint2 w2;
                w2.x = pack_bf16x2(acc[k].x, acc[k].y);
                w2.y = pack_bf16x2(acc[k].z, acc[k].w);
#ifdef CLOVER_CHECKED
                if (orow[rr] == ~0u) continue;   // its index check failed (reported)
#endif
                *reinterpret_cast<uint2 *>(out + (size_t)orow[rr] * D + c) = w2;
            }
        }
    }
}

// Merge weights of the sources of rows [p0, p1) (one thread a row), from the
// (m, l) stored after each source row's O: source s < KS is `own` row
// rr + 64 s, source KS + k row rr - p0 of slot k of `recv` (both in shared
// memory).  w[rr][s] = 2^(m_s - M) with M the largest m, divided by
// sum_s 2^(m_s - M) l_s when `normalise`; otherwise the combined row's M and
// sum go to w[rr][kMaxSrc - 2] and w[rr][kMaxSrc - 1].
template <int D, int KS>
__device__ __forceinline__ void row_weights(const float *own, const float *recv, int rpp, int p0, int p1, int n_src,
                                            float *wts, bool normalise) {
    constexpr int PS = D + 4;
    const int rr = p0 + (int)threadIdx.x;
    if (rr >= p1) return;
    float2 v[kMaxSrc];
#pragma unroll
    for (int sidx = 0; sidx < kMaxSrc; ++sidx) {
        const float *row = sidx < KS ? own + (rr + 64 * sidx) * PS : recv + ((sidx - KS) * rpp + rr - p0) * PS;
        v[sidx] = sidx < n_src ? *reinterpret_cast<const float2 *>(row + D) : make_float2(-INFINITY, 0.f);
    }
    float M = v[0].x;
#pragma unroll
    for (int sidx = 1; sidx < kMaxSrc; ++sidx) M = fmaxf(M, v[sidx].x);
    float w[kMaxSrc];
    float lsum = 0.f;
#pragma unroll
    for (int sidx = 0; sidx < kMaxSrc; ++sidx) {
        w[sidx] = (v[sidx].x == -INFINITY) ? 0.f : ex2_approx(v[sidx].x - M);
        lsum = fmaf(w[sidx], v[sidx].y, lsum);
    }
    const float inv = normalise ? (lsum > 0.f ? rcp_approx(lsum) : 0.f) : 1.f;
#pragma unroll
    for (int sidx = 0; sidx < kMaxSrc; ++sidx)
        if (sidx < n_src) wts[rr * kMaxSrc + sidx] = w[sidx] * inv;
    if (!normalise) {
        wts[rr * kMaxSrc + kMaxSrc - 2] = M;
        wts[rr * kMaxSrc + kMaxSrc - 1] = lsum;
    }
}

// At most 160 registers a thread (35,840 for the CTA): two 56-register CTAs
// of the accept kernel (28,672) still fit beside it on an SM, so that the
// argmax running beside the attention is not held back to one CTA an SM.
template <int D, int KS, bool PAGED>
__global__ void __maxnreg__(160)
    tree_attn_tc_kernel(const __grid_constant__ CUtensorMap tm_kc, const __grid_constant__ CUtensorMap tm_vc,
                        const __grid_constant__ CUtensorMap tm_kn, const __grid_constant__ CUtensorMap tm_vn,
                        const __grid_constant__ CUtensorMap tm_ks,
                        const __grid_constant__ CUtensorMap tm_vs, const AttnArgs a) {
    using S = TcSmem<D, KS>;
    constexpr int NSK = S::NSK;
    constexpr int NSV = S::NSV;
    // a kernel queued behind this one as a programmatic dependent may start
    // on the SM space this grid leaves free
    allow_dependent_launch();
    extern __shared__ uint8_t smem_raw[];
    // base rounded up to 1024 bytes by pointer arithmetic on the shared array,
    // so that every access below stays a shared-memory access
    uint8_t *sm = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    uint8_t *sK = sm + S::k_off;
    uint8_t *sV = sm + S::v_off;
    uint64_t *bars = reinterpret_cast<uint64_t *>(sm + S::bar_off);
    uint64_t *k_full = bars;
    uint64_t *k_empty = k_full + NSK;
    uint64_t *v_full = k_empty + NSK;
    uint64_t *v_empty = v_full + NSV;
    uint64_t *s_full = v_empty + NSV;         // [2] S of a tile is in TMEM
    uint64_t *p_full = s_full + 2;            // [2] P of a tile is in TMEM
    uint64_t *o_full = p_full + 2;            // [2] the tile's P.V product is done
    uint64_t *mma_done = o_full + 2;
    uint64_t *q_full = mma_done + 1;          // the four lane quadrants hold their Q rows in TMEM
    uint64_t *g_full = q_full + 1;            // the merging CTA: a pass of the other splits' partials is here
    uint64_t *anc_full = g_full + 1;          // the tree CTA: the ancestor masks are in shared memory
    uint64_t *x_bar = anc_full + 1;           // [4] KS = 1: the two softmax warps of a lane quadrant exchanged a value
    uint32_t *s_tmem = reinterpret_cast<uint32_t *>(sm + S::misc_off);
    volatile int *s_abort = reinterpret_cast<volatile int *>(sm + S::misc_off + 4);
    bool *s_bad = reinterpret_cast<bool *>(sm + S::misc_off + 8);
    uint64_t *s_anc = reinterpret_cast<uint64_t *>(sm + S::anc_off);
    int *s_pages = reinterpret_cast<int *>(sm + S::pages_off);
    float *s_wts = reinterpret_cast<float *>(sm + S::wts_off);
    float *s_xv = reinterpret_cast<float *>(sm + S::x_off);               // [parity][group][row]
    volatile int *s_xf = reinterpret_cast<volatile int *>(sm + S::x_off + 2 * 2 * BM * 4);   // [parity][group][quad]
    int *s_par = reinterpret_cast<int *>(sm + S::par_off);
    unsigned *s_orow = reinterpret_cast<unsigned *>(sm + S::orow_off);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    // grid (row tiles, split, sequence x KV head) with a group's tree split
    // (the merging one, which has the most work) at y = 0: CTAs are placed in
    // block order, so when SMs free up one by one it starts first in its group
    const int rt = blockIdx.x;
    const int split = a.n_split - 1 - (int)blockIdx.y;
    const int bg = blockIdx.z;
    const int b = bg / a.Hkv;
    const int g = bg % a.Hkv;
    const int n_split = a.n_split;
    const bool tree_cta = (split == n_split - 1);
    const int rows_here = min(BM, a.rows - rt * BM);
    const int q_act = (rows_here + 31) >> 5;        // 32-row quadrants holding real rows
    constexpr int NG = (KS == 1) ? 2 : 1;            // softmax warps per TMEM lane quadrant
    const int n_soft_warps = 2 * q_act;              // softmax warps of this tile (KS * NG per quadrant)

    // ------------------------------------------ setup that reads no input
    // Each producer initialises the barriers of its ring (the K producer also
    // every other one); warp 5 allocates TMEM.
    if (warp == kVProducerWarp && lane == 0) {
        for (int i = 0; i < NSV; ++i) {
            mbar_init(&v_full[i], 1);
            mbar_init(&v_empty[i], 1);
        }
        fence_barrier_init();
        prefetch_tensormap(&tm_vc);
        prefetch_tensormap(&tm_vn);
    }
    if (warp == kKProducerWarp && lane == 0) {
        for (int i = 0; i < NSK; ++i) {
            mbar_init(&k_full[i], 1);
            mbar_init(&k_empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&s_full[i], 1);
            mbar_init(&p_full[i], n_soft_warps);
            mbar_init(&o_full[i], 1);
        }
        mbar_init(mma_done, 1);
        mbar_init(q_full, 4);
        mbar_init(g_full, 1);
        mbar_init(anc_full, 1);
        for (int i = 0; i < 4; ++i) mbar_init(&x_bar[i], 2);
        *s_abort = 0;
        *s_bad = false;
        fence_barrier_init();
        prefetch_tensormap(&tm_kc);
        prefetch_tensormap(&tm_kn);
    }
    if (warp == kMmaWarp) {
        tmem_alloc(s_tmem, S::tmem_cols);
        tmem_relinquish();
    }

    // Q rows of this warp's TMEM lane quadrant (row (node, head in group) =
    // lane-quadrant row; with KS = 2 lanes 64-127 take rows 0-63 again); rows
    // past the tile's real rows are zero.  The tree CTA's warp 3 reads the
    // parent array.
    constexpr int QW = D / 2;                 // 32-bit TMEM columns of a Q row (two bf16 each)
    const int rq = ((KS == 2) ? (warp & 1) : (warp & 3)) * 32 + lane;
    const bool q_real = warp < 4 && rq < rows_here &&
                        CLOVER_IN(a.status, ((size_t)b * a.T + (rt * BM + rq) / a.G) * a.Hq + g * a.G +
                                                (rt * BM + rq) % a.G, (size_t)a.B * a.T * a.Hq);
    const uint4 *q_src = reinterpret_cast<const uint4 *>(
        static_cast<const __nv_bfloat16 *>(a.q) +
        ((size_t)(b * a.T + (q_real ? (rt * BM + rq) / a.G : 0)) * a.Hq + g * a.G +
         (q_real ? (rt * BM + rq) % a.G : 0)) * D);
    uint32_t qrow[QW];
    int parents[4];
    // Plain loads (L1-cached, so that a row's 16-byte pieces share their
    // lines; coherent, since in a programmatic launch the preceding kernel may
    // have written these inputs while this grid already ran).
    auto load_q_and_parents = [&]() {
        if (warp < 4) {
#pragma unroll
            for (int k = 0; k < QW / 4; ++k) {
                const uint4 v = q_real ? q_src[k] : make_uint4(0, 0, 0, 0);
                qrow[4 * k] = v.x;
                qrow[4 * k + 1] = v.y;
                qrow[4 * k + 2] = v.z;
                qrow[4 * k + 3] = v.w;
            }
        }
        if (warp == 3 && tree_cta) {
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const int i = lane + 32 * k;
                parents[k] = (i < a.T && (k < 2 || a.T > 64)) ? a.parent[(size_t)b * a.T + i] : -1;
            }
        }
    };

    // ------------------------------------ cache length and this CTA's keys
    // Launch modes: an ordinary launch (or pdl alone) reads every input after
    // the prerequisite grids complete; with cache_early the cache length, the
    // block table and the cache tiles of the free ring stages are read before
    // that; with inputs_early every input is, and only the writes wait.
    const bool in_early = a.inputs_early != 0;
    const bool c_early = in_early || a.cache_early != 0;
    if (!c_early) wait_prerequisite_grids();
    int L = a.cache_len[b];
    // the Q and parent loads go out while the length is read, ahead of the
    // ring's bulk traffic (issued once the length is known), so that they do
    // not queue behind it
    if (!c_early || in_early) load_q_and_parents();
    const bool cap_bad = (L < 0 || L + a.T > a.Lcap);
    if (cap_bad) {
        if (threadIdx.x == 0 && split == 0 && rt == 0 && g == 0) report(a.status, CLOVER_ERR_CAPACITY);
        L = L < 0 ? 0 : a.Lcap - a.T;
    }
    const int chunk = (((L + n_split - 1) / n_split) + BN - 1) / BN * BN;
    const int kbeg = min(L, split * chunk);
    const int kend = min(L, kbeg + chunk);
    const int n_cache_tiles = (CLOVER_IN(a.status, kbeg, a.Lcap + 1) && CLOVER_IN(a.status, kend, a.Lcap + 1))
                                  ? (kend - kbeg + BN - 1) / BN : 0;
    const int n_tiles = n_cache_tiles + (tree_cta ? 1 : 0);
    // The tree CTA takes its tree tile first, in every launch mode (so that
    // the result does not depend on the mode): the one CTA with an extra tile
    // then does not end on a load whose latency nothing hides.  With
    // cache_early the free ring stages after stage 0 fill with cache tiles
    // before k_new/v_new may be read.
    const bool split_wait = c_early && !in_early;
    const int tree_j = tree_cta ? 0 : -1;
    const int tree_shift = tree_cta ? 1 : 0;   // tile j is cache tile j - tree_shift
    // this CTA appends the tree K/V to cache slots [L, L+T)
    const bool appender = a.append && tree_cta && rt == 0 && !cap_bad;

    // Paged cache: a cache tile is read as boxes of `box` rows, each inside one
    // page (box = min(page size, BN); tiles start at multiples of BN).  The
    // page ids of tile j, looked up before the producer waits for the stage.
    // PAGED is a template flag: the dense kernel carries none of this code
    constexpr bool paged = PAGED;
    const int box = paged ? min(a.page_size, BN) : BN;
    const int first_page = kbeg >> a.page_shift;     // the split's first page (paged)
    // A paged cache tile is read by the whole producer warp at once: lane l
    // takes box l / DH (rows [box (l / DH), +box) of the tile) in 64-column
    // block l % DH, with its own page id (at most 8 boxes x 2 blocks).  The
    // page id of a lane's box of tile j, looked up before the producer waits
    // for the stage; staged: the split's first kPageSmem page ids are in
    // s_pages (after the setup barrier); later ones, and all of them before
    // it, come from the table.
    const int n_box_issues = paged ? (BN / box) * S::DH : 0;
    auto lane_page = [&](int j, bool staged) -> int {
        if (!paged || j == tree_j || lane >= n_box_issues) return 0;
        const int slot = kbeg + (j - tree_shift) * BN + (lane / S::DH) * box;
        const int pi = (slot >> a.page_shift) - first_page;
        return slot >= kend ? 0 : (staged && pi < kPageSmem) ? s_pages[pi] : cache_page(a, b, slot);
    };
    // tile j of K (is_v == false) or V into ring stage `dst`: a cache tile (an
    // evict-first read) or the tree tile.  Dense: run by the producer's lane 0;
    // paged: by all its lanes together (lane 0 alone for the tree tile).
    const uint64_t pol = l2_policy_evict_first();
    auto issue_tile = [&](int j, bool is_v, uint8_t *dst, uint64_t *bar, int pg) {
        const CUtensorMap *cache_map = is_v ? &tm_vc : &tm_kc;
        const CUtensorMap *new_map = is_v ? &tm_vn : &tm_kn;
        if (j != tree_j && paged) {
            if (lane == 0) mbar_arrive_expect_tx(bar, S::kv_bytes);
            __syncwarp();
            if (lane < n_box_issues) {
                const int r = (lane / S::DH) * box;
                const int dh = lane % S::DH;
                const int row = (kbeg + (j - tree_shift) * BN + r) & (a.page_size - 1);
                tma_load_3d_hint(dst + dh * BN * 128 + r * 128, cache_map, bar, dh * 64, row, pg * a.Hkv + g, pol);
            }
        } else if (lane == 0) {
            mbar_arrive_expect_tx(bar, S::kv_bytes);
            if (j != tree_j) {
#pragma unroll
                for (int dh = 0; dh < S::DH; ++dh)
                    tma_load_3d_hint(dst + dh * BN * 128, cache_map, bar, dh * 64, kbeg + (j - tree_shift) * BN, bg,
                                     pol);
            } else {
#pragma unroll
                for (int dh = 0; dh < S::DH; ++dh) tma_load_3d(dst + dh * BN * 128, new_map, bar, dh * 64, g, b * a.T);
            }
        }
    };
    // The first ring stages start empty: their tiles are issued without a
    // wait, in phase 0 (before the prerequisite grids complete, with
    // cache_early alone: the cache tiles among them) or phase 1 (the rest).
    auto issue_first = [&](bool is_v, int &issued, int phase) {
        constexpr int NSmax = NSK > NSV ? NSK : NSV;
        const int ns = is_v ? NSV : NSK;
        uint8_t *ring = is_v ? sV : sK;
        uint64_t *full = is_v ? v_full : k_full;
        const int upto = min(ns, n_tiles);
        int pg[NSmax];
        for (int j = 0; j < upto; ++j)
            if ((phase == 0) == (split_wait && j != tree_j)) pg[j] = lane_page(j, false);
        for (int j = 0; j < upto; ++j)
            if ((phase == 0) == (split_wait && j != tree_j)) issue_tile(j, is_v, ring + j * S::kv_bytes, &full[j], pg[j]);
        if (phase == 1) issued = upto;
    };

    // The tree tile (the tree CTA's last tile) holds the T new keys or values in
    // its first T rows once it has landed; TMA stores those rows straight from
    // the ring to cache slots [L, L+T), then waits until the store has read
    // them (the rings hold the partial result after the loop).
    auto append_tile = [&](bool is_v) {
        const int jt = tree_j;
        const int ns = is_v ? NSV : NSK;
        const int s = jt % ns;
        const uint32_t ph = (jt / ns) & 1;
        uint64_t *full = is_v ? &v_full[s] : &k_full[s];
        const uint8_t *src = (is_v ? sV : sK) + s * S::kv_bytes;
        if (*s_abort || !mbar_wait(full, ph, kWaitNs)) {
            *s_abort = 1;
            return;
        }
        fence_proxy_async_smem();
#pragma unroll
        for (int dh = 0; dh < S::DH; ++dh) tma_store_3d(is_v ? &tm_vs : &tm_ks, src + dh * BN * 128, dh * 64, L, bg);
        bulk_commit_group();
        bulk_wait_group_read0();
    };

    // The first ring stages, in two phases: with cache_early only, phase 0
    // issues the cache tiles among them before the prerequisite grids
    // complete (after an L2 prefetch of the Q rows); phase 1 stages the
    // split's page ids (paged), waits for those grids and loads Q (with
    // cache_early), and issues the rest of the first stages.
    const bool producer = (warp == kVProducerWarp || warp == kKProducerWarp) && (paged || lane == 0);
    const bool prod_v = warp == kVProducerWarp;
    int k_issued = 0, v_issued = 0;
#pragma unroll 1
    for (int phase = split_wait ? 0 : 1; phase < 2; ++phase) {
        if (phase == 0 && q_real)
            for (int c = 0; c < D * 2; c += 128) prefetch_l2(reinterpret_cast<const uint8_t *>(q_src) + c);
        if (phase == 1 && paged && warp == kMmaWarp && kend > kbeg) {
            const int n_pg = min(kPageSmem, ((kend - 1) >> a.page_shift) - first_page + 1);
            for (int i = lane; i < n_pg; i += 32) s_pages[i] = cache_page(a, b, (first_page + i) << a.page_shift);
        }
        if (phase == 1 && split_wait) {
            wait_prerequisite_grids();
            load_q_and_parents();
        }
        if (producer) issue_first(prod_v, prod_v ? v_issued : k_issued, phase);
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *s_tmem;
    const uint32_t tS = tmem;                 // S tiles (and their P): columns [0, 2*BN)
    const uint32_t tO = tmem + 2 * BN;        // O: columns [2*BN, 2*BN + D)
    const uint32_t tQ = tmem + 2 * BN + D;    // Q (the A operand of S): D / 2 columns after O
    if (warp < 4) {
        const uint32_t lanes = static_cast<uint32_t>(warp * 32) << 16;
#pragma unroll
        for (int c = 0; c < QW; c += 32)
            tmem_st32(tQ + lanes + c, *reinterpret_cast<const float(*)[32]>(qrow + c));
        tmem_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(q_full);
    }
    // The tree CTA's ancestor masks, built by warp 3 while the first tiles
    // are still on their way (they are needed by the tree tile's step only).
    if (warp == 3 && tree_cta) {
        tree_masks_walk(parents, a.T, s_par, s_anc, s_bad);
        __syncwarp();
        if (lane == 0) mbar_arrive(anc_full);
    }

    // ----------------------------------------------------- TMA producer warps
    // (lane 0; with a paged cache the whole warp, its waits and exits uniform)
    if (producer) {
        const bool is_v = warp == kVProducerWarp;
        const int ns = is_v ? NSV : NSK;
        uint8_t *ring = is_v ? sV : sK;
        uint64_t *full = is_v ? v_full : k_full;
        uint64_t *empty = is_v ? v_empty : k_empty;
        int &issued = is_v ? v_issued : k_issued;
        // the append reads the tree tile's stage: before the stage takes its
        // next tile, or after the loop (a write: after the prerequisite grids)
        bool appended = false;
        auto append = [&]() {
            if (in_early) wait_prerequisite_grids();
            append_tile(is_v);
            appended = true;
        };
        for (int j = issued; j < n_tiles; ++j) {
            const int s = j % ns;
            if (appender && !appended && j == tree_j + ns) append();
            const int pg = lane_page(j, true);
            bool ok = mbar_wait(&empty[s], ((j / ns) - 1) & 1, kWaitNs);
            if (paged) ok = __all_sync(0xffffffffu, ok);
            if (!ok) {
                *s_abort = 1;
                break;
            }
            if (paged ? __any_sync(0xffffffffu, *s_abort != 0) : *s_abort != 0) break;
            issue_tile(j, is_v, ring + s * S::kv_bytes, &full[s], pg);
            issued = j + 1;
        }
        if (appender && !appended && issued == n_tiles) append();
    }

    // --------------------------------------------------------- MMA issuer warp
    // Per tile j: S_j (needs K_j) is issued one tile ahead, then P_j.V_j (needs
    // P_j and V_j).  MMAs from this thread execute in issue order, so S_{j+2}
    // overwriting the TMEM of P_j comes after the P.V product reading it.
    if (warp == kMmaWarp && lane == 0) {
        const uint32_t idS = idesc_bf16(BM, BN, false, false);
        const uint32_t idO = idesc_bf16(BM, D, false, true);
        bool ok = mbar_wait(q_full, 0, kWaitNs);
        tc_fence_after();
        auto issue_s = [&](int j) -> bool {
            const int s = j % NSK;
            const int sb = j & 1;
            if (!mbar_wait(&k_full[s], (j / NSK) & 1, kWaitNs)) return false;
            tc_fence_after();
            const uint32_t k_base = smem_u32(sK + s * S::kv_bytes);
#pragma unroll
            for (int k = 0; k < D / 16; ++k) {
                const uint64_t bd = sdesc_sw128(k_base + (k >> 2) * (BN * 128) + (k & 3) * 32, 16, 1024);
                mma_bf16_tmem_a(tS + sb * BN, tQ + k * 8, bd, idS, k > 0 ? 1u : 0u);
            }
            mma_commit(&s_full[sb]);
            mma_commit(&k_empty[s]);
            return true;
        };
        int s_issued = 0;
        for (int j = 0; ok && j < n_tiles; ++j) {
            if (*s_abort) {
                ok = false;
                break;
            }
            // S of tiles j and j + 1 are issued before the P.V product of tile j
            while (ok && s_issued < min(j + 2, n_tiles)) ok = issue_s(s_issued++);
            if (!ok) break;
            const int s = j % NSV;
            const int sb = j & 1;
            if (!mbar_wait(&p_full[sb], (j >> 1) & 1, kWaitNs) || !mbar_wait(&v_full[s], (j / NSV) & 1, kWaitNs)) {
                ok = false;
                break;
            }
            tc_fence_after();
            const uint32_t v_base = smem_u32(sV + s * S::kv_bytes);
#pragma unroll
            for (int k = 0; k < BN / 16; ++k) {
                const uint64_t bd = sdesc_sw128(v_base + k * 16 * 128, BN * 128, 1024);
                mma_bf16_tmem_a(tO, tS + sb * BN + k * 8, bd, idO, (j > 0 || k > 0) ? 1u : 0u);
            }
            mma_commit(&o_full[sb]);
            mma_commit(&v_empty[s]);
        }
        if (!ok) *s_abort = 1;
        mma_commit(mma_done);
    }

    // ------------------------------------------------------------ softmax warps
    // A softmax warp reads S in the TMEM lanes of its quadrant (warp % 4, the
    // lanes it may access), one 64-key block of every tile, writes that
    // block's P back over S, keeps the reference max m_ref and the sum l, and
    // rescales its share of the O rows in TMEM when m_ref has to move.
    //   KS = 2 (a tile of at most 64 real rows): warps 0-3; lanes 32w.. are
    //   rows 32 (w & 1).. and the warp takes key block w >> 1; the two key
    //   halves of a row are two separate online softmaxes (own m, l and O
    //   rows), merged after the loop.
    //   KS = 1: warps 0-3 (group 0) and 7-10 (group 1); lanes 32 (w % 4).. are
    //   rows 32 (w % 4).. and group g takes key block g.  The two warps of a
    //   quadrant exchange their block maxima through shared memory (an
    //   mbarrier of two arrivals a tile, its wait bounded), so that both use
    //   one reference max and the P of a row is one softmax; each rescales
    //   half of the O columns, and their sums add up after the loop.
    const int sgroup = warp < 4 ? 0 : (NG == 2 && warp >= kSoft2Warp && warp < kSoft2Warp + 4) ? 1 : -1;
    const int quad = warp & 3;
    const int rquad = (KS == 2) ? (quad & 1) : quad;
    const int half = (KS == 2) ? (quad >> 1) : 0;
    const bool softmax_warp = sgroup >= 0 && rquad < q_act;
    const int r = rquad * 32 + lane;          // tile row
    const int blk = (KS == 2) ? half : sgroup;   // this thread's 64-key block of a tile
    const int soft_rank = (((KS == 2) ? half : sgroup) * q_act + rquad) * 32 + lane;
    const uint32_t lane_base = static_cast<uint32_t>(quad * 32) << 16;
    constexpr int OC = D / 32 / NG;           // 32-column chunks of O a softmax warp rescales and stores
    const int oc0 = (sgroup > 0 ? sgroup : 0) * OC;
    float m_ref = -INFINITY, l_run = 0.f;
    bool o_ready = false;
    int xn = 0;                               // exchanges made with the other warp of the quadrant
    // KS = 1: swap v (and a stop flag) with the quadrant's other warp; on a
    // timeout the partner's value reads as -inf and the flag as set
    auto exchange = [&](float v, bool &stop) -> float {
        const int par = xn & 1;
        s_xv[(par * 2 + sgroup) * BM + r] = v;
        if (lane == 0) s_xf[(par * 2 + sgroup) * 4 + quad] = stop ? 1 : 0;
        __syncwarp();
        if (lane == 0) mbar_arrive(&x_bar[quad]);
        const bool got = __all_sync(0xffffffffu, mbar_wait(&x_bar[quad], par, kWaitNs));
        ++xn;
        stop = stop || !got || s_xf[(par * 2 + 1 - sgroup) * 4 + quad] != 0;
        return got ? s_xv[(par * 2 + 1 - sgroup) * BM + r] : -INFINITY;
    };
    if (softmax_warp) {
        const int R = rt * BM + r;
        const int node = (r < rows_here) ? R / a.G : 0;
        const float sc = a.scale_log2;
        for (int j = 0; j < n_tiles; ++j) {
            const int sb = j & 1;
            const uint32_t ph = (j >> 1) & 1;
            const bool tree_tile = j == tree_j;
            bool stop = !__all_sync(0xffffffffu, mbar_wait(&s_full[sb], ph, kWaitNs)) ||
                        __any_sync(0xffffffffu, *s_abort != 0);
            if (!stop && tree_tile) stop = !__all_sync(0xffffffffu, mbar_wait(anc_full, 0, kWaitNs));
            const int key0 = kbeg + (j - tree_shift) * BN;
            const int n_valid = tree_tile ? a.T : min(BN, kend - key0);
            // Keys of the thread's 64-key block that its row sees: a prefix of
            // the cache keys, or the row's ancestors among the (at most 128)
            // tree keys, word blk of its mask.  Every tile runs the same
            // instructions, so the one tree tile brings no code into the
            // instruction cache (a miss then waits on a saturated memory system).
            float sv[64];
            float mxb = -INFINITY;
            if (!stop) {
                tc_fence_after();
                const uint32_t col = tS + lane_base + sb * BN + blk * 64;
                tmem_ld32(col, *reinterpret_cast<float(*)[32]>(sv));
                tmem_ld32(col + 32, *reinterpret_cast<float(*)[32]>(sv + 32));
                tmem_wait_ld();
                const int nv = n_valid - 64 * blk;
                const uint64_t prefix = nv >= 64 ? ~0ull : (nv <= 0 ? 0ull : ((1ull << nv) - 1ull));
                const uint64_t vis = tree_tile ? s_anc[node * kMaskWords + blk] : prefix;
                // a full block (every cache block but a tile's last) needs no
                // mask: warp-uniform there, so the branch costs nothing
                if (vis != ~0ull) {
#pragma unroll
                    for (int c = 0; c < 64; ++c) sv[c] = ((vis >> c) & 1ull) ? sv[c] : -INFINITY;
                }
                float mx4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
                for (int c = 0; c < 64; c += 8) {
                    mx4[0] = fmax3(mx4[0], sv[c], sv[c + 1]);
                    mx4[1] = fmax3(mx4[1], sv[c + 2], sv[c + 3]);
                    mx4[2] = fmax3(mx4[2], sv[c + 4], sv[c + 5]);
                    mx4[3] = fmax3(mx4[3], sv[c + 6], sv[c + 7]);
                }
                mxb = fmaxf(fmaxf(mx4[0], mx4[1]), fmaxf(mx4[2], mx4[3]));
            }
            // the row's max over the tile (KS = 1: over both warps' blocks;
            // group 0's first, so both warps compute the same value)
            if (NG == 2) {
                const float other = exchange(mxb, stop);
                mxb = sgroup == 0 ? fmaxf(mxb, other) : fmaxf(other, mxb);
            }
            if (stop) {
                *s_abort = 1;
                break;
            }
            const float mx = mxb * sc;            // sc > 0

            // move the reference max when this tile exceeds it by more than 2^8
            const bool move = (mx > m_ref + kRescale);
            if (j == 0) {
                m_ref = mx;
            } else if (__any_sync(0xffffffffu, move)) {
                // O must hold every earlier tile before it is rescaled
                const bool got_o =
                    __all_sync(0xffffffffu, mbar_wait(&o_full[(j - 1) & 1], ((j - 1) >> 1) & 1, kWaitNs));
                if (!got_o) {
                    *s_abort = 1;
                    break;
                }
                tc_fence_after();
                const float f = move ? ex2_approx(m_ref - mx) : 1.f;
                l_run *= f;
                if (move) m_ref = mx;
#pragma unroll 1
                for (int cc = oc0; cc < oc0 + OC; ++cc) {
                    float x[32];
                    tmem_ld32(tO + lane_base + cc * 32, x);
                    tmem_wait_ld();
#pragma unroll
                    for (int c = 0; c < 32; c += 2) {
                        const float2 y = __fmul2_rn(make_float2(x[c], x[c + 1]), make_float2(f, f));
                        x[c] = y.x;
                        x[c + 1] = y.y;
                    }
                    tmem_st32(tO + lane_base + cc * 32, x);
                }
            }
            const float ref = (m_ref == -INFINITY) ? 0.f : m_ref;
            // P of the block (two keys per column) goes to packed columns
            // [32 blk, 32 blk + 32) of the tile's TMEM, over S values already
            // read: this thread's own (block 0) or, for block 1, those of
            // block 0, which its reader had loaded before the exchange
            // (KS = 1) or which sit in other lanes (KS = 2).  The exponent
            // arguments and the running sums go two at a time (packed f32x2
            // FMA and add: the same roundings as one at a time).
            const float2 sc2 = make_float2(sc, sc);
            const float2 nref2 = make_float2(-ref, -ref);
            float2 sum01 = make_float2(0.f, 0.f), sum23 = make_float2(0.f, 0.f);
            {
                float pk[32];
#pragma unroll
                for (int c = 0; c < 64; c += 4) {
                    const float2 t01 = __ffma2_rn(make_float2(sv[c], sv[c + 1]), sc2, nref2);
                    const float2 t23 = __ffma2_rn(make_float2(sv[c + 2], sv[c + 3]), sc2, nref2);
                    const float2 p01 = make_float2(ex2_approx(t01.x), ex2_approx(t01.y));
                    const float2 p23 = make_float2(ex2_approx(t23.x), ex2_approx(t23.y));
                    sum01 = __fadd2_rn(sum01, p01);
                    sum23 = __fadd2_rn(sum23, p23);
                    pk[c >> 1] = __uint_as_float(pack_bf16x2(p01.x, p01.y));
                    pk[(c >> 1) + 1] = __uint_as_float(pack_bf16x2(p23.x, p23.y));
                }
                tmem_st32(tS + lane_base + sb * BN + blk * 32, pk);
            }
            l_run += (sum01.x + sum01.y) + (sum23.x + sum23.y);
            if (KS == 2) {
                // the other half's keys of this row read as zero
                float z[32];
#pragma unroll
                for (int c = 0; c < 32; ++c) z[c] = 0.f;
                tmem_st32(tS + lane_base + sb * BN + (1 - half) * 32, z);
            }
            // value rows of keys past the valid ones may hold anything (even NaN): zero them
            if (n_valid < BN) {
                const int s = j % NSV;
                const bool got_v = __all_sync(0xffffffffu, mbar_wait(&v_full[s], (j / NSV) & 1, kWaitNs));
                if (!got_v) {
                    *s_abort = 1;
                    break;
                }
                uint4 *vrows = reinterpret_cast<uint4 *>(sV + s * S::kv_bytes);
                const int n_zero = (BN - n_valid) * S::DH * 8;
                for (int e = soft_rank; e < n_zero; e += n_soft_warps * 32) {
                    const int row = n_valid + e / (S::DH * 8);
                    const int rest = e % (S::DH * 8);
                    vrows[(rest >> 3) * (BN * 8) + row * 8 + (rest & 7)] = make_uint4(0, 0, 0, 0);
                }
                fence_proxy_async_smem();
            }
            tmem_wait_st();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&p_full[sb]);
        }
        // the last P.V product completes O
        if (n_tiles > 0 && !__any_sync(0xffffffffu, *s_abort != 0)) {
            const int jl = n_tiles - 1;
            o_ready = __all_sync(0xffffffffu, mbar_wait(&o_full[jl & 1], (jl >> 1) & 1, kWaitNs));
            if (!o_ready) *s_abort = 1;
            tc_fence_after();
        }
    }

    // ------------------------------------------------------------- epilogue
    tc_fence_before();
    __syncthreads();                          // every role is out of its key loop
    if (*s_abort && lane == 0) {
        // wind down: wait (bounded) for the loads still in flight before the
        // rings are reused below
        if (warp == kKProducerWarp)
            for (int j = max(0, k_issued - NSK); j < k_issued; ++j) mbar_wait(&k_full[j % NSK], (j / NSK) & 1, kWaitNs);
        if (warp == kVProducerWarp)
            for (int j = max(0, v_issued - NSV); j < v_issued; ++j) mbar_wait(&v_full[j % NSV], (j / NSV) & 1, kWaitNs);
    }
    __syncthreads();
    tc_fence_after();
    // (1) every softmax warp moves the O rows, m and l of its TMEM lanes to
    // part_o row 32 quad + lane: KS = 1, tile row r (each warp of the quadrant
    // its half of the columns, group 0 m and the sum of both warps' l); KS =
    // 2, the first key half of tile row r in rows 0-63 and the second half in
    // rows 64-127.  The TMEM loads are warp-collective: every lane runs them,
    // rows past the tile's real rows only skip the stores.
    float *part_o = reinterpret_cast<float *>(sK);            // [BM][D + 4] fp32
    if (softmax_warp) {
        const bool real = r < rows_here;
        float *dst = part_o + (quad * 32 + lane) * S::po_stride;
        float l_tot = l_run;
        if (NG == 2) {
            // a split with no keys (a short sequence's empty range) has no O
            // and is not a failure: its rows carry m = -inf and l = 0
            bool stop = n_tiles > 0 && !o_ready;
            const float other = exchange(l_run, stop);
            l_tot = sgroup == 0 ? l_run + other : other + l_run;
            if (stop) *s_abort = 1;
        }
        constexpr int NP = (OC % 2 == 0) ? 2 : 1;             // chunks per TMEM round trip
#pragma unroll 1
        for (int cc = oc0; cc < oc0 + OC; cc += NP) {
            float x[NP][32];
            if (o_ready) {
#pragma unroll
                for (int p = 0; p < NP; ++p) tmem_ld32(tO + lane_base + (cc + p) * 32, x[p]);
                tmem_wait_ld();
            } else {
#pragma unroll
                for (int p = 0; p < NP; ++p)
#pragma unroll
                    for (int c = 0; c < 32; ++c) x[p][c] = 0.f;
            }
            if (real) {
#pragma unroll
                for (int p = 0; p < NP; ++p)
#pragma unroll
                    for (int c = 0; c < 32; c += 4)
                        *reinterpret_cast<float4 *>(dst + (cc + p) * 32 + c) =
                            make_float4(x[p][c], x[p][c + 1], x[p][c + 2], x[p][c + 3]);
            }
        }
        if (real && sgroup == 0)
            *reinterpret_cast<float4 *>(dst + D) =
                make_float4(o_ready ? m_ref : -INFINITY, o_ready ? l_tot : 0.f, 0.f, 0.f);
    }
    // every TMEM access and MMA is finished before TMEM is released
    tc_fence_before();
    __syncthreads();
    if (warp == kMmaWarp) {
        if (lane == 0) mbar_wait(mma_done, 0, kWaitNs);
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem, S::tmem_cols);
    }
    if (tree_cta && rt == 0 && threadIdx.x == 0 && *s_bad) report(a.status, CLOVER_ERR_BAD_TREE);
    // every global write below comes after the prerequisite grids complete
    if (in_early) wait_prerequisite_grids();
    // the appended tree K/V is in global memory before the CTA exits
    if (appender && (warp == kKProducerWarp || warp == kVProducerWarp) && lane == 0) bulk_wait_group0();

    // (2) The split merge.  Every split but the last (the tree split, which
    // has the most work and ends last) combines its two key halves, copies its
    // rows to its workspace slot and counts itself in at the group's counter
    // (release); then it is done.  The last split waits (bounded) until the
    // others are in (acquire), loads their rows and merges every source of a
    // row (its own halves and the other splits' rows) into the output.  With
    // one split there are no others.
    const int grp = bg * a.row_tiles + rt;
    float *slots = n_split > 1 ? a.part_o + (size_t)grp * n_split * a.slot_rows * S::po_stride : nullptr;
    constexpr uint32_t row_bytes = S::po_stride * 4;
    const int others = tree_cta ? n_split - 1 : 0;
    const int n_src = KS + others;
    __nv_bfloat16 *out = static_cast<__nv_bfloat16 *>(a.out);
    if (n_split > 1 && !tree_cta) {
        if (KS == 2) {
            row_weights<D, KS>(part_o, nullptr, 0, 0, rows_here, KS, s_wts, false);
            __syncthreads();
            merge_pass<D, KS>(part_o, nullptr, s_wts, nullptr, KS, 0, 0, rows_here, nullptr);
            if (threadIdx.x < rows_here)
                *reinterpret_cast<float2 *>(part_o + threadIdx.x * S::po_stride + D) =
                    make_float2(s_wts[threadIdx.x * kMaxSrc + kMaxSrc - 2], s_wts[threadIdx.x * kMaxSrc + kMaxSrc - 1]);
        }
        fence_proxy_async_smem();             // the bulk copy reads these rows
        __syncthreads();
        if (threadIdx.x == 0 &&
            CLOVER_IN(a.status, (((size_t)grp * n_split + split) * a.slot_rows + rows_here) * row_bytes - 1,
                      a.ws_bytes) &&
            CLOVER_IN(a.status, grp, (size_t)a.B * a.Hkv * a.row_tiles)) {
            bulk_store_s2g(slots + (size_t)split * a.slot_rows * S::po_stride, part_o, rows_here * row_bytes);
            bulk_commit_group();
            bulk_wait_group0();
            fence_proxy_async_global();
            red_add_release_gpu(a.counters + grp, 1u);
        }
    } else {
        if (others > 0 && threadIdx.x == 0 &&
            !(CLOVER_IN(a.status, grp, (size_t)a.B * a.Hkv * a.row_tiles) &&
              CLOVER_IN(a.status, (((size_t)grp * n_split + others - 1) * a.slot_rows + rows_here) * row_bytes - 1,
                        a.ws_bytes)))
            *s_abort = 1;
        if (others > 0 && threadIdx.x == 0 && !*s_abort) {
            bool in = ld_acquire_gpu(a.counters + grp) >= (unsigned)others;
            if (!in) {
                const uint64_t t0 = globaltimer_ns();
                while (!(in = ld_acquire_gpu(a.counters + grp) >= (unsigned)others) && globaltimer_ns() - t0 < kWaitNs)
                    __nanosleep(64);
            }
            if (in) {
                a.counters[grp] = 0u;                 // ready for the next call
                fence_proxy_async_global();
            } else {
                *s_abort = 1;
            }
        }
        __syncthreads();
        // output row (node i, query head h) of tile row rr: (b T + i) Hq + h
        if ((int)threadIdx.x < rows_here) {
            const int R = rt * BM + (int)threadIdx.x;
            const int i = R / a.G;
            const size_t orow = ((size_t)b * a.T + i) * a.Hq + g * a.G + (R - i * a.G);
            s_orow[threadIdx.x] = CLOVER_IN(a.status, orow, (size_t)a.B * a.T * a.Hq) ? (unsigned)orow : ~0u;
        }
        if (!*s_abort) {
            float *recv = reinterpret_cast<float *>(sK + S::own_bytes);
            const int rpp = others > 0 ? min(rows_here, S::recv_bytes / (others * (int)row_bytes)) : rows_here;
            int pass = 0;
            for (int p0 = 0; p0 < rows_here; p0 += rpp, ++pass) {
                const int p1 = min(rows_here, p0 + rpp);
                if (others > 0 && threadIdx.x == 0) {
                    const uint32_t bytes = (uint32_t)(p1 - p0) * row_bytes;
                    mbar_arrive_expect_tx(g_full, bytes * others);
                    for (int k = 0; k < others; ++k)
                        bulk_load_g2s(recv + (size_t)k * rpp * S::po_stride,
                                      slots + ((size_t)k * a.slot_rows + p0) * S::po_stride, bytes, g_full);
                }
                const bool got = others == 0 || mbar_wait(g_full, pass & 1, kWaitNs);
                if (got) row_weights<D, KS>(part_o, recv, rpp, p0, p1, n_src, s_wts, true);
                else *s_abort = 1;
                __syncthreads();   // the weights are in shared memory
                if (!*s_abort) merge_pass<D, KS>(part_o, recv, s_wts, s_orow, n_src, rpp, p0, p1, out);
                // the received rows are read before the next pass overwrites them
                __syncthreads();
                if (*s_abort) break;
            }
        }
    }
    if (*s_abort && threadIdx.x == 0) report(a.status, CLOVER_ERR_TIMEOUT);
}

template <int D, int KS, bool PAGED>
cudaError_t launch(AttnArgs a, cudaStream_t stream) {
    static unsigned long long done[64];
    auto kernel = tree_attn_tc_kernel<D, KS, PAGED>;
    cudaError_t err = ensure_smem_attr(kernel, TcSmem<D, KS>::alloc, done);
    if (err != cudaSuccess) return err;
    if (a.n_split < 1 || a.n_split > kMaxSplits) return cudaErrorInvalidValue;
    if (a.n_split > 1 && (!a.part_o || !a.counters)) return cudaErrorInvalidValue;

    CUtensorMap kc, vc, kn, vn, ks, vs;
    const uint64_t e = 2;
    bool ok = make_tmap_bf16_3d(&kn, a.k_new, D, a.Hkv, (uint64_t)a.B * a.T, D * e, (uint64_t)a.Hkv * D * e, 64, 1, BN) &&
              make_tmap_bf16_3d(&vn, a.v_new, D, a.Hkv, (uint64_t)a.B * a.T, D * e, (uint64_t)a.Hkv * D * e, 64, 1, BN);
    if (PAGED) {
        // page pools [n_pages * Hkv planes][page_size rows][D]; a paged call
        // never appends, so the append maps are not used
        const uint32_t box = (uint32_t)(a.page_size < BN ? a.page_size : BN);
        const uint64_t plane = (uint64_t)a.page_size * D * e;
        ok = ok &&
             make_tmap_bf16_3d(&kc, a.k_cache, D, a.page_size, (uint64_t)a.n_pages * a.Hkv, D * e, plane, 64, box, 1) &&
             make_tmap_bf16_3d(&vc, a.v_cache, D, a.page_size, (uint64_t)a.n_pages * a.Hkv, D * e, plane, 64, box, 1);
        ks = kc;
        vs = vc;
    } else {
        const uint64_t plane = (uint64_t)a.Lcap * D * e;
        ok = ok &&
             make_tmap_bf16_3d(&kc, a.k_cache, D, a.Lcap, (uint64_t)a.B * a.Hkv, D * e, plane, 64, BN, 1) &&
             make_tmap_bf16_3d(&vc, a.v_cache, D, a.Lcap, (uint64_t)a.B * a.Hkv, D * e, plane, 64, BN, 1) &&
             // the append: T rows of one (sequence, head) plane of the cache
             make_tmap_bf16_3d(&ks, a.k_cache, D, a.Lcap, (uint64_t)a.B * a.Hkv, D * e, plane, 64, a.T, 1) &&
             make_tmap_bf16_3d(&vs, a.v_cache, D, a.Lcap, (uint64_t)a.B * a.Hkv, D * e, plane, 64, a.T, 1);
    }
    if (!ok) return cudaErrorInvalidValue;

    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(a.row_tiles, a.n_split, a.B * a.Hkv);
    cfg.blockDim = dim3(threads_of<KS>(), 1, 1);
    cfg.dynamicSmemBytes = TcSmem<D, KS>::alloc;
    cfg.stream = stream;
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr.val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = &attr;
    cfg.numAttrs = a.pdl ? 1 : 0;
    err = cudaLaunchKernelEx(&cfg, kernel, kc, vc, kn, vn, ks, vs, a);
    if (err != cudaSuccess) return err;
    return cudaGetLastError();
}

}  // namespace

int tc_row_tile() { return BM; }
int tc_max_splits() { return kMaxSplits; }

cudaError_t launch_tree_attn_tc(const AttnArgs &a, cudaStream_t stream) {
    // a tile of at most 64 real rows: two key groups per row (KS = 2)
    if (a.block_table) {
        if (a.rows <= 64) return a.D == 64 ? launch<64, 2, true>(a, stream) : launch<128, 2, true>(a, stream);
        return a.D == 64 ? launch<64, 1, true>(a, stream) : launch<128, 1, true>(a, stream);
    }
    if (a.rows <= 64) return a.D == 64 ? launch<64, 2, false>(a, stream) : launch<128, 2, false>(a, stream);
    return a.D == 64 ? launch<64, 1, false>(a, stream) : launch<128, 1, false>(a, stream);
}

}  // namespace clover
