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
// own ring); warp 6 those of the V tiles (a deeper ring: a V tile is held
// until its P.V product, a K tile only until its S); warp 5 allocates TMEM and
// issues the MMAs from one thread.  The tree CTA's producers also append the
// tree keys and values to the cache when asked, by TMA stores of the tree
// tile they loaded.
// The split that owns the last cache range also takes the tile of T tree keys
// (read from k_new/v_new) under the ancestor bitmask.  The n_split CTAs of a
// (sequence, head, row tile) form one thread-block cluster: each sends every
// other CTA its rows of the partial result (O, m, l) by shared-to-shared bulk
// copy, and merges its own rows, so no partial result touches global memory.
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
constexpr int kPageSmem = 512;           // page ids of a split staged in shared memory
constexpr int kKProducerWarp = 4;
constexpr int kMmaWarp = 5;
constexpr int kVProducerWarp = 6;
constexpr int kThreads = 224;
constexpr int kMaxCluster = 8;          // portable cluster size: splits per head
constexpr float kRescale = 8.0f;        // move the reference max only past 2^8 growth
constexpr uint64_t kWaitNs = 500ull * 1000 * 1000;   // 0.5 s per wait

// Shared-memory plan: the K and V rings only (Q lives in TMEM).  KS = key
// groups per tile row: with KS = 2 (a tile of at most 64 real query rows) the
// Q rows of TMEM lanes 64-127 repeat those of lanes 0-63, so every real row's
// scores sit in two lane quadrants and the four softmax warps each take half
// of a tile's keys.
template <int D, int KS>
struct TcSmem {
    static constexpr int NSK = (D == 128) ? 3 : 4;   // K ring stages
    static constexpr int NSV = (D == 128) ? 3 : 4;   // V ring stages
    static constexpr int DH = D / 64;                // 128-byte column blocks per row
    static constexpr int kv_bytes = BN * D * 2;      // one K or V tile: [DH][BN][128 B]
    static constexpr int k_off = 0;
    static constexpr int v_off = k_off + NSK * kv_bytes;
    static constexpr int bar_off = v_off + NSV * kv_bytes;
    static constexpr int n_bars = 2 * NSK + 2 * NSV + 11;
    static constexpr int misc_off = bar_off + 8 * n_bars;          // tmem addr, abort, bad flags
    static constexpr int anc_off = misc_off + 16;                  // ancestor masks [128][2]
    static constexpr int pages_off = anc_off + kMaxTreeNodes * kMaskWords * 8;   // paged: page ids of the split
    static constexpr int total = pages_off + kPageSmem * 4;
    static constexpr size_t alloc = total + 1024;                  // base rounded up to 1024 bytes
    // TMEM columns: S/P 2 x BN, O D, Q D / 2 (two bf16 per column), rounded up
    // to a power of two.  All 512 columns of an SM go to one CTA only when
    // the shared memory already keeps a second CTA off the SM (a CTA waiting
    // in tcgen05.alloc would stall its cluster).
    static constexpr uint32_t tmem_cols = (2 * BN + D + D / 2 <= 256) ? 256 : 512;
    static_assert(tmem_cols < 512 || 2 * alloc > 228 * 1024, "512 TMEM columns need one CTA per SM");
    // After the key loop the K ring holds this CTA's partial result, one fp32
    // row of D + 4 floats per query row (O, then m and l in the padding; with
    // KS = 2 rows 64-127 first carry the second key half's rows), and the V
    // ring receives the other splits' partials of the rows this CTA merges:
    // [n_split][rows per split][D + 4].
    static constexpr int po_stride = D + 4;
    static constexpr int rows_max = (KS == 2) ? 64 : BM;         // real rows of a tile
    static_assert(BM * po_stride * 4 <= NSK * kv_bytes, "partial result must fit in the K ring");
    static_assert((rows_max + kMaxCluster - 1) * po_stride * 4 <= NSV * kv_bytes,
                  "received partials must fit in the V ring");
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

// Merge of the NS split partials of rows [r0, r1) of a tile (Section 2.2's
// attention over the whole key range, from per-range partial softmax results):
//   O = sum_k 2^(m_k - M) O_k / sum_k 2^(m_k - M) l_k,  M = max_k m_k.
// Row rr of split k is `own` (this CTA's) or row (k * per + rr - r0) of `recv`;
// each row holds O (D floats), then m and l.  A thread takes one (row, 4
// columns) item at a time.  NS is a template argument so the whole item is
// one short chain of independent loads and arithmetic (with few warps per
// SM, the latency of a long chain is not hidden).
template <int D, int NS>
__device__ __forceinline__ void merge_rows(const float *own, const float *recv, int po_stride, int split, int per,
                                           int r0, int r1, int row0, const AttnArgs &a, int b, int g,
                                           __nv_bfloat16 *out) {
    const int n_items = (r1 - r0) * (D / 4);
    const float inv_g = 1.f / (float)a.G;
    for (int e = threadIdx.x; e < n_items; e += blockDim.x) {
        const int rr = r0 + e / (D / 4);
        const int c4 = (e % (D / 4)) * 4;
        float2 ml[NS];
        float4 x[NS];
#pragma unroll
        for (int k = 0; k < NS; ++k) {
            const float *row = (k == split) ? own + rr * po_stride : recv + (k * per + rr - r0) * po_stride;
            ml[k] = *reinterpret_cast<const float2 *>(row + D);
            x[k] = *reinterpret_cast<const float4 *>(row + c4);
        }
        float M = ml[0].x;
#pragma unroll
        for (int k = 1; k < NS; ++k) M = fmaxf(M, ml[k].x);
        float w[NS];
        float lsum = 0.f;
#pragma unroll
        for (int k = 0; k < NS; ++k) {
            w[k] = (ml[k].x == -INFINITY) ? 0.f : ex2_approx(ml[k].x - M);
            lsum = fmaf(w[k], ml[k].y, lsum);
        }
        const float inv = rcp_approx(lsum);
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int k = 0; k < NS; ++k) {
            const float wk = w[k] * inv;
            acc.x = fmaf(wk, x[k].x, acc.x);
            acc.y = fmaf(wk, x[k].y, acc.y);
            acc.z = fmaf(wk, x[k].z, acc.z);
            acc.w = fmaf(wk, x[k].w, acc.w);
        }
        // row R = node * G + head-in-group; (R + 1/2) / G is never within
        // float rounding of an integer, so the truncation is exact
        const int R = row0 + rr;
        const int i = __float2int_rz(((float)R + 0.5f) * inv_g);
        const int h = g * a.G + (R - i * a.G);
        uint2 w2;
        w2.x = pack_bf16x2(acc.x, acc.y);
        w2.y = pack_bf16x2(acc.z, acc.w);
        *reinterpret_cast<uint2 *>(out + ((size_t)(b * a.T + i) * a.Hq + h) * D + c4) = w2;
    }
}

template <int D, int KS, bool PAGED>
__global__ void __launch_bounds__(kThreads, 1)
    tree_attn_tc_kernel(const __grid_constant__ CUtensorMap tm_kc, const __grid_constant__ CUtensorMap tm_vc,
                        const __grid_constant__ CUtensorMap tm_kn, const __grid_constant__ CUtensorMap tm_vn,
                        const __grid_constant__ CUtensorMap tm_ks,
                        const __grid_constant__ CUtensorMap tm_vs, const AttnArgs a) {
    using S = TcSmem<D, KS>;
    constexpr int NSK = S::NSK;
    constexpr int NSV = S::NSV;
    // an accept call queued behind this one as a programmatic dependent may
    // take the SM space this grid leaves free
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
    uint64_t *m_free = q_full + 1;            // every CTA of the cluster is out of its key loop
    uint64_t *m_done = m_free + 1;            // every CTA has received this CTA's partial rows
    uint64_t *m_data = m_done + 1;            // the other splits' partials of this CTA's rows are here
    uint32_t *s_tmem = reinterpret_cast<uint32_t *>(sm + S::misc_off);
    volatile int *s_abort = reinterpret_cast<volatile int *>(sm + S::misc_off + 4);
    bool *s_bad = reinterpret_cast<bool *>(sm + S::misc_off + 8);
    uint64_t *s_anc = reinterpret_cast<uint64_t *>(sm + S::anc_off);
    int *s_pages = reinterpret_cast<int *>(sm + S::pages_off);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int rt = blockIdx.x;
    const int split = blockIdx.y;
    const int bg = blockIdx.z;
    const int b = bg / a.Hkv;
    const int g = bg % a.Hkv;
    const int n_split = a.n_split;
    const bool tree_cta = (split == n_split - 1);
    const int rows_here = min(BM, a.rows - rt * BM);
    const int q_act = (rows_here + 31) >> 5;        // 32-row quadrants holding real rows
    const int n_soft_warps = KS * q_act;             // softmax warps of this tile

    // The loads that do not depend on the cache length go out first, ahead of
    // the ring's bulk traffic (issued once the length is known), so that they
    // do not queue behind it.  Q rows of this warp's TMEM lane quadrant (row
    // (node, head in group) = lane-quadrant row; with KS = 2 lanes 64-127 take
    // rows 0-63 again) are written to TMEM once its address is known; rows past
    // the tile's real rows are zero.  The tree CTA's warp 3 loads the parents.
    constexpr int QW = D / 2;                 // 32-bit TMEM columns of a Q row (two bf16 each)
    uint32_t qrow[QW];
    if (warp < 4) {
        const int rq = ((KS == 2) ? (warp & 1) : warp) * 32 + lane;
        const int R = rt * BM + rq;
        const bool real = rq < rows_here;
        const uint4 *src = reinterpret_cast<const uint4 *>(static_cast<const __nv_bfloat16 *>(a.q) +
                                                           ((size_t)(b * a.T + (real ? R / a.G : 0)) * a.Hq +
                                                            g * a.G + (real ? R % a.G : 0)) * D);
#pragma unroll
        for (int k = 0; k < QW / 4; ++k) {
            const uint4 v = real ? __ldg(src + k) : make_uint4(0, 0, 0, 0);
            qrow[4 * k] = v.x;
            qrow[4 * k + 1] = v.y;
            qrow[4 * k + 2] = v.z;
            qrow[4 * k + 3] = v.w;
        }
    }
    int parents[4];
    if (warp == 3 && tree_cta) tree_parents_load(a.parent + (size_t)b * a.T, a.T, parents);

    int L = __ldg(a.cache_len + b);
    const bool cap_bad = (L < 0 || L + a.T > a.Lcap);
    if (cap_bad) {
        if (threadIdx.x == 0 && split == 0 && rt == 0 && g == 0) report(a.status, CLOVER_ERR_CAPACITY);
        L = L < 0 ? 0 : a.Lcap - a.T;
    }
    const int chunk = (((L + n_split - 1) / n_split) + BN - 1) / BN * BN;
    const int kbeg = min(L, split * chunk);
    const int kend = min(L, kbeg + chunk);
    const int n_cache_tiles = (kend - kbeg + BN - 1) / BN;
    const int n_tiles = n_cache_tiles + (tree_cta ? 1 : 0);
    // the tree CTA takes its tree tile first (tile 0), so the one CTA with an
    // extra tile does not finish on a load whose latency nothing hides
    const int first_cache = tree_cta ? 1 : 0;
    // this CTA appends the tree K/V to cache slots [L, L+T)
    const bool appender = a.append && tree_cta && rt == 0 && !cap_bad;

    // Paged cache: a cache tile is read as boxes of `box` rows, each inside one
    // page (box = min(page size, BN); tiles start at multiples of BN).  The
    // page ids of tile j, looked up before the producer waits for the stage.
    // PAGED is a template flag: the dense kernel carries none of this code
    constexpr bool paged = PAGED;
    const int box = paged ? min(a.page_size, BN) : BN;
    const int first_page = kbeg >> a.page_shift;     // the split's first page (paged)
    // staged: the split's first kPageSmem page ids are in s_pages (after the
    // setup barrier); later ones, and all of them before it, come from the table
    auto tile_pages = [&](int j, int (&pg)[kMaxBoxes], bool staged) {
        if (!paged || j < first_cache) return;
        const int key0 = kbeg + (j - first_cache) * BN;
        for (int r = 0, x = 0; r < BN; r += box, ++x) {
            const int slot = key0 + r;
            const int pi = (slot >> a.page_shift) - first_page;
            pg[x] = slot >= kend ? 0 : (staged && pi < kPageSmem) ? s_pages[pi] : cache_page(a, b, slot);
        }
    };
    // tile j of K (is_v == false) or V into ring stage `dst`
    auto issue_tile = [&](int j, bool is_v, uint8_t *dst, uint64_t *bar, const int (&pg)[kMaxBoxes]) {
        mbar_arrive_expect_tx(bar, S::kv_bytes);
        const CUtensorMap *cache_map = is_v ? &tm_vc : &tm_kc;
        const CUtensorMap *new_map = is_v ? &tm_vn : &tm_kn;
        if (j >= first_cache && paged) {
            const int key0 = kbeg + (j - first_cache) * BN;
            for (int r = 0, x = 0; r < BN; r += box, ++x) {
                const int row = (key0 + r) & (a.page_size - 1);
#pragma unroll
                for (int dh = 0; dh < S::DH; ++dh)
                    tma_load_3d(dst + dh * BN * 128 + r * 128, cache_map, bar, dh * 64, row, pg[x] * a.Hkv + g);
            }
        } else if (j >= first_cache) {
#pragma unroll
            for (int dh = 0; dh < S::DH; ++dh) tma_load_3d(dst + dh * BN * 128, cache_map, bar, dh * 64, kbeg + (j - first_cache) * BN, bg);
        } else {
#pragma unroll
            for (int dh = 0; dh < S::DH; ++dh) tma_load_3d(dst + dh * BN * 128, new_map, bar, dh * 64, g, b * a.T);
        }
    };

    // The tree tile (tile 0 of the tree CTA, ring stage 0) holds the T new
    // keys or values in its first T rows once it has landed; TMA stores those
    // rows straight from the ring to cache slots [L, L+T), then waits until the
    // store has read them.  The producer does this before stage 0 takes its
    // next tile (or after its loop when there is none).
    auto append_tile = [&](bool is_v) {
        uint64_t *full = is_v ? &v_full[0] : &k_full[0];
        const uint8_t *src = is_v ? sV : sK;
        if (*s_abort || !mbar_wait(full, 0, kWaitNs)) {
            *s_abort = 1;
            return;
        }
        fence_proxy_async_smem();
#pragma unroll
        for (int dh = 0; dh < S::DH; ++dh) tma_store_3d(is_v ? &tm_vs : &tm_ks, src + dh * BN * 128, dh * 64, L, bg);
        bulk_commit_group();
        bulk_wait_group_read0();
    };

    // ---------------------------------------------------------------- setup
    // Each producer initialises the barriers of its ring (the K producer also
    // every other one) and issues its first ring loads at once (the stages
    // start empty), the K producer also the Q load, so that they overlap the
    // TMEM allocation.
    int k_issued = 0, v_issued = 0;
    if (warp == kVProducerWarp && lane == 0) {
        for (int i = 0; i < NSV; ++i) {
            mbar_init(&v_full[i], 1);
            mbar_init(&v_empty[i], 1);
        }
        fence_barrier_init();
        prefetch_tensormap(&tm_vc);
        prefetch_tensormap(&tm_vn);
        int pg[NSV][kMaxBoxes];
        for (int j = 0; j < min(NSV, n_tiles); ++j) tile_pages(j, pg[j], false);
        for (; v_issued < min(NSV, n_tiles); ++v_issued)
            issue_tile(v_issued, true, sV + v_issued * S::kv_bytes, &v_full[v_issued], pg[v_issued]);
    }
    if (warp == kKProducerWarp) {
        if (lane == 0) {
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
            mbar_init(m_free, n_split);
            mbar_init(m_done, n_split);
            mbar_init(m_data, 1);
            if (n_split > 1) {
                // every other split sends this CTA its rows [r0, r1) of the tile
                const int per = (rows_here + n_split - 1) / n_split;
                const int mine = max(0, min(rows_here, (split + 1) * per) - split * per);
                mbar_arrive_expect_tx(m_data, (uint32_t)((n_split - 1) * mine * S::po_stride * 4));
            }
            *s_abort = 0;
            *s_bad = false;
            fence_barrier_init();
            prefetch_tensormap(&tm_kc);
            prefetch_tensormap(&tm_kn);
            int pg[NSK][kMaxBoxes];
            for (int j = 0; j < min(NSK, n_tiles); ++j) tile_pages(j, pg[j], false);
            for (; k_issued < min(NSK, n_tiles); ++k_issued)
                issue_tile(k_issued, false, sK + k_issued * S::kv_bytes, &k_full[k_issued], pg[k_issued]);
        }
    }
    if (warp == kMmaWarp) {
        tmem_alloc(s_tmem, S::tmem_cols);
        tmem_relinquish();
        // paged: the split's page ids, for the producers' loops
        if (paged && kend > kbeg) {
            const int n_pg = min(kPageSmem, ((kend - 1) >> a.page_shift) - first_page + 1);
            for (int i = lane; i < n_pg; i += 32) s_pages[i] = cache_page(a, b, (first_page + i) << a.page_shift);
        }
    }
    // the tree CTA's ancestor masks (warp 3 is otherwise idle here)
    if (warp == 3 && tree_cta) tree_masks_build(parents, a.T, s_anc, s_bad);
    // The cluster barrier is split: its wait (before the first remote arrive,
    // in the merge) lets the key loop start without waiting for the other
    // CTAs' setup.  The arrive is relaxed: fence_barrier_init has already
    // published this CTA's barriers to the cluster, and a releasing arrive
    // would hold each producer until its ring loads have landed.
    tc_fence_before();
    __syncwarp();
    if (n_split > 1) cluster_arrive_relaxed();
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

    // ----------------------------------------------------- TMA producer warps
    if (warp == kVProducerWarp) {
        if (lane == 0) {
            bool appended = false;
            for (int j = v_issued; j < n_tiles; ++j) {
                const int s = j % NSV;
                if (appender && j == NSV) {
                    append_tile(true);
                    appended = true;
                }
                int pg[kMaxBoxes];
                tile_pages(j, pg, true);
                if (!mbar_wait(&v_empty[s], ((j / NSV) - 1) & 1, kWaitNs)) {
                    *s_abort = 1;
                    break;
                }
                if (*s_abort) break;
                issue_tile(j, true, sV + s * S::kv_bytes, &v_full[s], pg);
                v_issued = j + 1;
            }
            if (appender && !appended && v_issued == n_tiles) append_tile(true);
        }
    }
    if (warp == kKProducerWarp) {
        if (lane == 0) {
            bool appended = false;
            for (int j = k_issued; j < n_tiles; ++j) {
                const int s = j % NSK;
                if (appender && j == NSK) {
                    append_tile(false);
                    appended = true;
                }
                int pg[kMaxBoxes];
                tile_pages(j, pg, true);
                if (!mbar_wait(&k_empty[s], ((j / NSK) - 1) & 1, kWaitNs)) {
                    *s_abort = 1;
                    break;
                }
                if (*s_abort) break;
                issue_tile(j, false, sK + s * S::kv_bytes, &k_full[s], pg);
                k_issued = j + 1;
            }
            if (appender && !appended && k_issued == n_tiles) append_tile(false);
        }
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
        if (ok && n_tiles > 0) ok = issue_s(0);
        for (int j = 0; ok && j < n_tiles; ++j) {
            if (*s_abort) {
                ok = false;
                break;
            }
            if (j + 1 < n_tiles && !(ok = issue_s(j + 1))) break;
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
    // Warp w owns TMEM lanes 32w.. (the lanes it may access); it reads S there,
    // writes P back over it, keeps the reference max m_ref and sum l, and
    // rescales its O rows in TMEM when m_ref has to move.  KS = 1: lanes 32w..
    // are tile rows 32w.. and the warp takes every key of a tile.  KS = 2:
    // lanes 32w.. are rows 32(w & 1).. and the warp takes keys
    // [32 (w >> 1), +32) of every tile; the two key halves of a row are two
    // separate online softmaxes (own m, l and O rows), merged after the loop.
    constexpr int NK = BN / KS;               // keys of a tile per thread
    const int quad = warp & 3;
    const int rquad = (KS == 2) ? (quad & 1) : quad;
    const int half = (KS == 2) ? (quad >> 1) : 0;
    const bool softmax_warp = warp < 4 && rquad < q_act;
    const int r = rquad * 32 + lane;          // tile row
    const int soft_rank = ((KS == 2) ? half * q_act + rquad : quad) * 32 + lane;
    const uint32_t lane_base = static_cast<uint32_t>(quad * 32) << 16;
    float m_ref = -INFINITY, l_run = 0.f;
    bool o_ready = false;
    if (softmax_warp) {
        const int R = rt * BM + r;
        const int node = (r < rows_here) ? R / a.G : 0;
        const float sc = a.scale_log2;
        for (int j = 0; j < n_tiles; ++j) {
            const int sb = j & 1;
            const uint32_t ph = (j >> 1) & 1;
            const bool got = __all_sync(0xffffffffu, mbar_wait(&s_full[sb], ph, kWaitNs));
            if (!got || __any_sync(0xffffffffu, *s_abort != 0)) {
                *s_abort = 1;
                break;
            }
            tc_fence_after();
            const bool tree_tile = tree_cta && j == 0;
            const int key0 = kbeg + (j - first_cache) * BN;
            const int n_valid = tree_tile ? a.T : min(BN, kend - key0);
            // Keys of a 64-key block of the tile that this row sees: a prefix
            // of the cache keys, or the row's ancestors among the (at most
            // 128) tree keys, word blk of its mask.  Every tile runs the same
            // instructions, so the one tree tile, late in the loop, brings no
            // code into the instruction cache (a miss then waits on a
            // saturated memory system).
            auto block_vis = [&](int blk) -> uint64_t {
                const int nv = n_valid - 64 * blk;
                const uint64_t prefix = nv >= 64 ? ~0ull : (nv <= 0 ? 0ull : ((1ull << nv) - 1ull));
                return tree_tile ? s_anc[node * kMaskWords + blk] : prefix;
            };
            // this thread's NB blocks of 64 keys start at block blk0 (KS = 2:
            // the key half; KS = 1: both halves, S re-read from TMEM per pass)
            constexpr int NB = NK / 64;
            const int blk0 = half * NB;
            float sv[64];
            auto load_block = [&](int blk) {
                const uint32_t col = tS + lane_base + sb * BN + blk * 64;
                tmem_ld32(col, *reinterpret_cast<float(*)[32]>(sv));
                tmem_ld32(col + 32, *reinterpret_cast<float(*)[32]>(sv + 32));
                tmem_wait_ld();
                const uint64_t vis = block_vis(blk);
#pragma unroll
                for (int c = 0; c < 64; ++c) sv[c] = ((vis >> c) & 1ull) ? sv[c] : -INFINITY;
            };
            float mx4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll 1
            for (int bi = 0; bi < NB; ++bi) {
                load_block(blk0 + bi);
#pragma unroll
                for (int c = 0; c < 64; ++c) mx4[c & 3] = fmaxf(mx4[c & 3], sv[c]);
            }
            const float mx = fmaxf(fmaxf(mx4[0], mx4[1]), fmaxf(mx4[2], mx4[3])) * sc;   // sc > 0

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
                for (int cc = 0; cc < D / 32; ++cc) {
                    float x[32];
                    tmem_ld32(tO + lane_base + cc * 32, x);
                    tmem_wait_ld();
#pragma unroll
                    for (int c = 0; c < 32; ++c) x[c] *= f;
                    tmem_st32(tO + lane_base + cc * 32, x);
                }
            }
            const float ref = (m_ref == -INFINITY) ? 0.f : m_ref;
            // P of block blk (two keys per column) goes to packed columns
            // [32 blk, 32 blk + 32) of the tile's TMEM: over S values this
            // thread has already read (blocks in increasing order)
            float sum4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 1
            for (int bi = 0; bi < NB; ++bi) {
                if (NB > 1) load_block(blk0 + bi);
                float pk[32];
#pragma unroll
                for (int c = 0; c < 64; c += 2) {
                    const float p0 = ex2_approx(fmaf(sv[c], sc, -ref));
                    const float p1 = ex2_approx(fmaf(sv[c + 1], sc, -ref));
                    sum4[c & 3] += p0;
                    sum4[(c + 1) & 3] += p1;
                    pk[c >> 1] = __uint_as_float(pack_bf16x2(p0, p1));
                }
                tmem_st32(tS + lane_base + sb * BN + (blk0 + bi) * 32, pk);
            }
            l_run += (sum4[0] + sum4[1]) + (sum4[2] + sum4[3]);
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
    if (n_split > 1) {
        // this CTA's rings are free: the other splits may send their partials
        cluster_wait_acquire();               // every CTA's barriers exist
        if (warp == 1 && lane < n_split) mbar_arrive_remote(mapa_shared(smem_u32(m_free), lane));
    }
    __nv_bfloat16 *out = static_cast<__nv_bfloat16 *>(a.out);
    const bool row_ok = softmax_warp && r < rows_here;
    float *part_o = reinterpret_cast<float *>(sK);            // [BM][D + 4] fp32, this CTA's partial
    float *recv = reinterpret_cast<float *>(sV);              // [n_split][per][D + 4]
    // 64 O columns of this warp's lanes.  The TMEM loads are warp-collective:
    // every lane runs them, rows past the tile's real rows only skip the stores
    auto load_o = [&](int cc, float (&x0)[32], float (&x1)[32]) {
        if (o_ready) {
            tmem_ld32(tO + lane_base + cc * 32, x0);
            tmem_ld32(tO + lane_base + cc * 32 + 32, x1);
            tmem_wait_ld();
        } else {
#pragma unroll
            for (int c = 0; c < 32; ++c) x0[c] = x1[c] = 0.f;
        }
    };
    // KS = 2: the second key half's rows (O, m, l) go to rows 64.. of part_o,
    // where the warps of the first half merge them into their own.  Those
    // warps load their first 64 O columns meanwhile.
    float x0[32], x1[32];
    if (KS == 2) {
        if (softmax_warp && half == 1) {
            float *dst = part_o + (64 + r) * S::po_stride;
#pragma unroll 1
            for (int cc = 0; cc < D / 32; cc += 2) {
                load_o(cc, x0, x1);
                if (row_ok) {
#pragma unroll
                    for (int c = 0; c < 32; c += 4) {
                        *reinterpret_cast<float4 *>(dst + cc * 32 + c) =
                            make_float4(x0[c], x0[c + 1], x0[c + 2], x0[c + 3]);
                        *reinterpret_cast<float4 *>(dst + cc * 32 + 32 + c) =
                            make_float4(x1[c], x1[c + 1], x1[c + 2], x1[c + 3]);
                    }
                }
            }
            if (row_ok)
                *reinterpret_cast<float2 *>(dst + D) =
                    make_float2(o_ready ? m_ref : -INFINITY, o_ready ? l_run : 0.f);
        }
        if (softmax_warp && half == 0) load_o(0, x0, x1);
        __syncthreads();
    }
    if (softmax_warp && half == 0) {
        // this row's (m, l) and the weights of its key halves
        float m_row = o_ready ? m_ref : -INFINITY;
        float l_row = o_ready ? l_run : 0.f;
        float wa = 1.f, wb = 0.f;
        const float *ob = part_o + (64 + r) * S::po_stride;
        if (KS == 2 && row_ok) {
            const float2 mlb = *reinterpret_cast<const float2 *>(ob + D);
            const float M = fmaxf(m_row, mlb.x);
            wa = (m_row == -INFINITY) ? 0.f : ex2_approx(m_row - M);
            wb = (mlb.x == -INFINITY) ? 0.f : ex2_approx(mlb.x - M);
            m_row = M;
            l_row = wa * l_row + wb * mlb.y;
        }
        // 64 columns of the row: the output (one split) or the partial row.
        // The other half's 64 values are read in one batch before any store.
        auto emit = [&](int cc, float (&y0)[32], float (&y1)[32]) {
            if (KS == 2) {
                float4 yb[16];
#pragma unroll
                for (int c = 0; c < 16; ++c) yb[c] = *reinterpret_cast<const float4 *>(ob + cc * 32 + 4 * c);
#pragma unroll
                for (int c = 0; c < 8; ++c) {
                    y0[4 * c] = fmaf(wb, yb[c].x, wa * y0[4 * c]);
                    y0[4 * c + 1] = fmaf(wb, yb[c].y, wa * y0[4 * c + 1]);
                    y0[4 * c + 2] = fmaf(wb, yb[c].z, wa * y0[4 * c + 2]);
                    y0[4 * c + 3] = fmaf(wb, yb[c].w, wa * y0[4 * c + 3]);
                    y1[4 * c] = fmaf(wb, yb[8 + c].x, wa * y1[4 * c]);
                    y1[4 * c + 1] = fmaf(wb, yb[8 + c].y, wa * y1[4 * c + 1]);
                    y1[4 * c + 2] = fmaf(wb, yb[8 + c].z, wa * y1[4 * c + 2]);
                    y1[4 * c + 3] = fmaf(wb, yb[8 + c].w, wa * y1[4 * c + 3]);
                }
            }
            if (n_split == 1) {
                // the output row (node, head); only this path needs it
                const int R = rt * BM + r;
                const int i = R / a.G;
                const int h = g * a.G + (R % a.G);
                const float inv = l_row > 0.f ? rcp_approx(l_row) : 1.f;
                __nv_bfloat16 *dst = out + ((size_t)(b * a.T + i) * a.Hq + h) * D + cc * 32;
#pragma unroll
                for (int c = 0; c < 64; c += 8) {
                    const float *x = c < 32 ? y0 + c : y1 + (c - 32);
                    uint4 w;
                    w.x = pack_bf16x2(x[0] * inv, x[1] * inv);
                    w.y = pack_bf16x2(x[2] * inv, x[3] * inv);
                    w.z = pack_bf16x2(x[4] * inv, x[5] * inv);
                    w.w = pack_bf16x2(x[6] * inv, x[7] * inv);
                    *reinterpret_cast<uint4 *>(dst + c) = w;
                }
            } else {
                float *po = part_o + r * S::po_stride + cc * 32;
#pragma unroll
                for (int c = 0; c < 32; c += 4) {
                    *reinterpret_cast<float4 *>(po + c) = make_float4(y0[c], y0[c + 1], y0[c + 2], y0[c + 3]);
                    *reinterpret_cast<float4 *>(po + 32 + c) = make_float4(y1[c], y1[c + 1], y1[c + 2], y1[c + 3]);
                }
            }
        };
        // two TMEM loads in flight per wait (the first pair is loaded already with KS = 2)
#pragma unroll 1
        for (int cc = 0; cc < D / 32; cc += 2) {
            if (KS == 1 || cc > 0) load_o(cc, x0, x1);
            if (row_ok) emit(cc, x0, x1);
        }
        if (row_ok && n_split > 1)
            *reinterpret_cast<float2 *>(part_o + r * S::po_stride + D) = make_float2(m_row, l_row);
        if (n_split > 1) fence_proxy_async_smem();   // the bulk copies below read these rows
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
    if (n_split > 1) {
        // ------------------------------------------ split merge in the cluster
        // CTA `split` merges rows [r0, r1) of the tile.  Once every CTA is out
        // of its key loop (m_free), lane k of warp 0 sends CTA k (k != split)
        // that CTA's rows of this CTA's partial with one bulk copy into its V
        // ring (completing on its m_data); then every CTA merges its own rows
        // from shared memory.
        const int per = (rows_here + n_split - 1) / n_split;
        const int r0 = split * per;
        const int r1 = min(rows_here, r0 + per);
        constexpr uint32_t row_bytes = S::po_stride * 4;
        bool ok = true;
        if (warp == 0) {
            if (lane < n_split) {
                ok = mbar_wait_cluster(m_free, 0, kWaitNs);
                const int k0 = lane * per;
                const int k1 = min(rows_here, k0 + per);
                if (ok && lane != split && k1 > k0)
                    bulk_copy_to_cluster(mapa_shared(smem_u32(recv) + split * per * row_bytes, lane),
                                         part_o + k0 * S::po_stride, (k1 - k0) * row_bytes,
                                         mapa_shared(smem_u32(m_data), lane));
            }
            ok = __all_sync(0xffffffffu, ok);
            if (lane == 0 && ok) ok = mbar_wait_cluster(m_data, 0, kWaitNs);
        }
        // one thread waited; every thread acquires the received rows itself
        const bool got = __syncthreads_and(ok) && mbar_test_cluster(m_data, 0);
        // every partial row this CTA needs is here: its senders may exit
        if (warp == 1 && lane < n_split) mbar_arrive_remote(mapa_shared(smem_u32(m_done), lane));
        if (got) {
            switch (n_split) {
#define CLOVER_MERGE_CASE(NS) \
    case NS: merge_rows<D, NS>(part_o, recv, S::po_stride, split, per, r0, r1, rt * BM, a, b, g, out); break;
                CLOVER_MERGE_CASE(2)
                CLOVER_MERGE_CASE(3)
                CLOVER_MERGE_CASE(4)
                CLOVER_MERGE_CASE(5)
                CLOVER_MERGE_CASE(6)
                CLOVER_MERGE_CASE(7)
                CLOVER_MERGE_CASE(8)
#undef CLOVER_MERGE_CASE
                default: break;
            }
        } else {
            *s_abort = 1;
        }
        // the copies reading this CTA's partial are complete before its
        // shared memory goes away
        ok = true;
        if (threadIdx.x == 0) ok = mbar_wait_cluster(m_done, 0, kWaitNs);
        if (!__syncthreads_and(ok)) *s_abort = 1;
    }
    // the appended tree K/V is in global memory before the CTA exits
    if (appender && (warp == kKProducerWarp || warp == kVProducerWarp) && lane == 0) bulk_wait_group0();
    if (*s_abort && threadIdx.x == 0) report(a.status, CLOVER_ERR_TIMEOUT);
}

struct TcLaunchCache {
    int sms = 0;
    int max_clusters[kMaxCluster + 1] = {0};   // co-resident clusters per cluster size (0: not queried)
};

template <int D, int KS, bool PAGED>
int max_active_clusters(int n, TcLaunchCache &cache) {
    if (cache.max_clusters[n] == 0) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(1, n, n);
        cfg.blockDim = dim3(kThreads, 1, 1);
        cfg.dynamicSmemBytes = TcSmem<D, KS>::alloc;
        cudaLaunchAttribute attr;
        attr.id = cudaLaunchAttributeClusterDimension;
        attr.val.clusterDim.x = 1;
        attr.val.clusterDim.y = n;
        attr.val.clusterDim.z = 1;
        cfg.attrs = &attr;
        cfg.numAttrs = 1;
        int num = 0;
        if (cudaOccupancyMaxActiveClusters(&num, tree_attn_tc_kernel<D, KS, PAGED>, &cfg) != cudaSuccess) {
            cudaGetLastError();
            num = -1;
        }
        cache.max_clusters[n] = num > 0 ? num : -1;
    }
    return cache.max_clusters[n];
}

template <int D, int KS, bool PAGED>
cudaError_t launch(AttnArgs a, cudaStream_t stream) {
    static unsigned long long done[64];
    static TcLaunchCache caches[64];
    auto kernel = tree_attn_tc_kernel<D, KS, PAGED>;
    cudaError_t err = ensure_smem_attr(kernel, TcSmem<D, KS>::alloc, done);
    if (err != cudaSuccess) return err;
    int dev = 0;
    if ((err = cudaGetDevice(&dev)) != cudaSuccess) return err;
    TcLaunchCache &cache = caches[dev < 64 ? dev : 63];
    if (cache.sms == 0 && (err = cudaDeviceGetAttribute(&cache.sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
        return err;

    // splits per head: as many as fill the SMs in one wave of clusters
    const long base = (long)a.B * a.Hkv * a.row_tiles;
    const int by_len = (a.Lcap + 255) / 256;
    int n = 1;
    for (int c = kMaxCluster; c >= 2; --c) {
        if (c > by_len || base * c > cache.sms) continue;
        if (max_active_clusters<D, KS, PAGED>(c, cache) >= base) {
            n = c;
            break;
        }
    }
    a.n_split = n;

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
    cfg.gridDim = dim3(a.row_tiles, n, a.B * a.Hkv);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = TcSmem<D, KS>::alloc;
    cfg.stream = stream;
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeClusterDimension;
    attr.val.clusterDim.x = 1;
    attr.val.clusterDim.y = n;
    attr.val.clusterDim.z = 1;
    cfg.attrs = &attr;
    cfg.numAttrs = n > 1 ? 1 : 0;
    err = cudaLaunchKernelEx(&cfg, kernel, kc, vc, kn, vn, ks, vs, a);
    if (err != cudaSuccess) return err;
    return cudaGetLastError();
}

}  // namespace

int tc_row_tile() { return BM; }

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
