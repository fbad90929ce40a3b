// Linear layer of the draft heads on the tensor cores: y[R, N] = x[R, K] . w[N, K]^T
// (bf16 inputs, fp32 accumulation), with the epilogue the Clover head needs
// (Section 3: the attention decoder's projections, the residual SiLU block of
// the MLP and the shared LM head).
//
// The draft rows are few (R <= 256 per launch) and the weights large (the LM
// head is V x H = 125696 x 4096), so the layer is a weight stream: each weight
// byte is read once, and the R rows of x stay in L2.  The weight is the MMA's A
// operand (M = 128 weight rows), x the B operand (N = R rounded up to 16), so
// D[m][r] = y[r][row0 + m] accumulates in TMEM.
//
// One persistent CTA per SM takes a contiguous range of 128-row weight tiles
// and walks it two tiles at a time (one x chunk serves both, halving x's reads
// from L2).  Warp 0 issues the TMA loads of a 3-stage ring (per stage: 64 K
// columns of the two weight tiles and of x), warp 1 issues the MMAs (two
// accumulators), warps 2-5 read the accumulators and write y.  Every wait is
// bounded; a wait that gives up sets CLOVER_ERR_TIMEOUT and the CTA winds down.
//
// Programmatic dependent launch: every CTA lets a dependent grid launch as soon
// as it starts, and waits for the grid it depends on (griddepcontrol.wait)
// only before its first touch of x, res, out or the workspace: the weight
// tiles of the first stages are requested before that wait (the weight is
// never written by the kernel before it), so a layer's set-up and first
// weight loads overlap the end of the layer before it.  Launched without the
// attribute the wait returns at once.
#include "common.cuh"
#include "tc_ptx.cuh"
#include "tmap_host.cuh"

namespace clover {
namespace {

using namespace tc;

constexpr int LM = 128;                    // weight rows per tile (the MMA's M)
constexpr int LK = 64;                     // K columns per stage (one 128-byte swizzle row)
constexpr int kMaxRows = 256;              // x rows per launch (the MMA's N)
constexpr int kStages = 3;
constexpr int kThreadsL = 192;             // producer, MMA, 4 epilogue warps
constexpr int kProducer = 0;
constexpr int kMma = 1;
constexpr uint64_t kWaitL = 500000000ull;  // 0.5 s
constexpr int kMaxSplit = 8;               // K ranges per tile pair at most

struct LinSmem {
    static constexpr int w_bytes = LM * LK * 2;                      // one weight tile's stage: 16 KB
    static constexpr int x_bytes = kMaxRows * LK * 2;                // x's stage: up to 32 KB
    static constexpr int stage_bytes = 2 * w_bytes + x_bytes;        // 64 KB
    static constexpr int bar_off = kStages * stage_bytes;
    static constexpr int n_bars = 2 * kStages + 3;                   // full, empty; acc full, acc empty, mma done
    static constexpr int misc_off = bar_off + 8 * n_bars;            // tmem address, abort flag
    static constexpr int total = misc_off + 16;
    static constexpr size_t alloc = total + 1024;
    static_assert(alloc <= 227 * 1024, "shared memory budget");
};

struct LinArgs {
    const __nv_bfloat16 *res;              // [R, N] (modes with a residual)
    void *out;                             // [R, N]: fp32 (mode 0) or bf16
    int R, Rp, N, K, mode;
    int n_tiles;                           // ceil(N / LM)
    // split K (n_split > 1): CTA = (tile pair, K range); fp32 partials in
    // part [n_split, R, N], one arrival counter per tile pair
    int n_split;
    float *part;
    unsigned *counters;
    int32_t *status;
};

// The epilogue of one output element from its fp32 sum.
__device__ __forceinline__ void store_out(const LinArgs &a, size_t o, float y);

__device__ __forceinline__ float silu(float v) { return v / (1.f + ex2_approx(-v * 1.4426950408889634f)); }

__device__ __forceinline__ void store_out(const LinArgs &a, size_t o, float y) {
    if (a.mode == CLOVER_LINEAR_F32) {
        static_cast<float *>(a.out)[o] = y;
        return;
    }
    if (a.mode == CLOVER_LINEAR_RES_SILU) y = __bfloat162float(a.res[o]) + silu(y);
    else if (a.mode == CLOVER_LINEAR_RES) y = __bfloat162float(a.res[o]) + y;
    static_cast<__nv_bfloat16 *>(a.out)[o] = __float2bfloat16_rn(y);
}

__global__ void __launch_bounds__(kThreadsL, 1)
    linear_tc_kernel(const __grid_constant__ CUtensorMap tm_w, const __grid_constant__ CUtensorMap tm_x,
                     const LinArgs a) {
    using S = LinSmem;
    allow_dependent_launch();
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    uint64_t *full = reinterpret_cast<uint64_t *>(sm + S::bar_off);
    uint64_t *empty = full + kStages;
    uint64_t *acc_full = empty + kStages;
    uint64_t *acc_empty = acc_full + 1;
    uint64_t *mma_done = acc_empty + 1;
    uint32_t *s_tmem = reinterpret_cast<uint32_t *>(sm + S::misc_off);
    volatile int *s_abort = reinterpret_cast<volatile int *>(sm + S::misc_off + 4);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    // this CTA's tiles [t0, t1), walked in pairs, and its K chunks [c_lo, c_hi)
    const int n_chunks = a.K / LK;
    const bool split = a.n_split > 1;
    const int pair = blockIdx.x / a.n_split;
    const int ks = blockIdx.x % a.n_split;
    const int t0 = split ? 2 * pair : (int)((long)blockIdx.x * a.n_tiles / gridDim.x);
    const int t1 = split ? min(a.n_tiles, 2 * pair + 2) : (int)((long)(blockIdx.x + 1) * a.n_tiles / gridDim.x);
    const int c_lo = split ? ks * n_chunks / a.n_split : 0;
    const int c_hi = split ? (ks + 1) * n_chunks / a.n_split : n_chunks;
    // accumulator of tile h at TMEM columns [h * RS, h * RS + Rp); the
    // epilogue reads 32 columns at a time, so RS and the allocation are whole
    // multiples of 32 covering both
    const int RS = (a.Rp + 31) / 32 * 32;
    const uint32_t tmem_cols = (2 * RS <= 32) ? 32 : (2 * RS <= 64) ? 64 : (2 * RS <= 128) ? 128
                                                 : (2 * RS <= 256) ? 256 : 512;

    if (threadIdx.x == 0) {
        for (int i = 0; i < kStages; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        mbar_init(acc_full, 1);
        mbar_init(acc_empty, 4);
        mbar_init(mma_done, 1);
        *s_abort = 0;
        fence_barrier_init();
    }
    if (warp == kMma) {
        tmem_alloc(s_tmem, tmem_cols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *s_tmem;

    int issued = 0;                        // stages issued by the producer (for the wind-down)
    if (warp == kProducer && lane == 0) {
        prefetch_tensormap(&tm_w);
        prefetch_tensormap(&tm_x);
        // the x chunks of the first stages wait for the prerequisite grid
        // (which writes x); their weight tiles are requested before it
        int pend_c[kStages];
        int n_pend = 0;
        bool waited = false;
        auto release_x = [&]() {
            wait_prerequisite_grids();
            for (int i = 0; i < n_pend; ++i)
                tma_load_3d(sm + i * S::stage_bytes + 2 * S::w_bytes, &tm_x, &full[i], pend_c[i] * LK, 0, 0);
            waited = true;
        };
        int it = 0;
        for (int t = t0; t < t1 && !*s_abort; t += 2) {
            const bool two = t + 1 < t1;
            const uint32_t bytes = (uint32_t)((two ? 2 : 1) * S::w_bytes + a.Rp * LK * 2);
            for (int c = c_lo; c < c_hi; ++c, ++it) {
                const int s = it % kStages;
                if (it >= kStages && !waited) release_x();
                if (!mbar_wait(&empty[s], ((it / kStages) - 1) & 1, kWaitL)) {
                    *s_abort = 1;
                    break;
                }
                uint8_t *st = sm + s * S::stage_bytes;
                mbar_arrive_expect_tx(&full[s], bytes);
                tma_load_3d(st, &tm_w, &full[s], c * LK, t * LM, 0);
                if (two) tma_load_3d(st + S::w_bytes, &tm_w, &full[s], c * LK, (t + 1) * LM, 0);
                if (waited) tma_load_3d(st + 2 * S::w_bytes, &tm_x, &full[s], c * LK, 0, 0);
                else pend_c[n_pend++] = c;            // stage s == n_pend here (it < kStages)
                issued = it + 1;
            }
        }
        if (!waited) release_x();
    }

    if (warp == kMma && lane == 0) {
        const uint32_t idesc = idesc_bf16(LM, a.Rp, false, false);
        int it = 0, item = 0;
        for (int t = t0; t < t1 && !*s_abort; t += 2, ++item) {
            const bool two = t + 1 < t1;
            // the epilogue has read the accumulators of the previous item
            if (!mbar_wait(acc_empty, (item - 1) & 1, kWaitL)) {
                *s_abort = 1;
                break;
            }
            tc_fence_after();
            bool ok = true;
            for (int c = c_lo; c < c_hi; ++c, ++it) {
                const int s = it % kStages;
                if (!mbar_wait(&full[s], (it / kStages) & 1, kWaitL)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t st = smem_u32(sm + s * S::stage_bytes);
#pragma unroll
                for (int k = 0; k < LK / 16; ++k) {
                    const uint64_t bd = sdesc_sw128(st + 2 * S::w_bytes + k * 32, 16, 1024);
                    mma_bf16(tmem, sdesc_sw128(st + k * 32, 16, 1024), bd, idesc, (c - c_lo) + k != 0);
                    if (two) mma_bf16(tmem + RS, sdesc_sw128(st + S::w_bytes + k * 32, 16, 1024), bd, idesc,
                                      (c - c_lo) + k != 0);
                }
                mma_commit(&empty[s]);         // the stage is free once these MMAs have read it
            }
            if (!ok) {
                *s_abort = 1;
                break;
            }
            mma_commit(acc_full);
        }
        // every MMA of this thread (and the stage releases they carry) has
        // completed before the accumulators' TMEM is released
        mma_commit(mma_done);
        if (!mbar_wait(mma_done, 0, kWaitL)) *s_abort = 1;
    }

    if (warp >= 2) {
        // res, out, the partials and the counters after the prerequisite grid
        wait_prerequisite_grids();
        // warp w reads TMEM lanes 32 (w % 4) .. +31: weight rows m of the tile
        const int quad = warp & 3;
        const int m = quad * 32 + lane;
        const uint32_t lane_base = static_cast<uint32_t>(quad * 32) << 16;
        int item = 0;
        for (int t = t0; t < t1; t += 2, ++item) {
            const bool two = t + 1 < t1;
            const bool got = __all_sync(0xffffffffu, mbar_wait(acc_full, item & 1, kWaitL));
            if (!got || *s_abort) {
                *s_abort = 1;
                break;
            }
            tc_fence_after();
            for (int half = 0; half < (two ? 2 : 1); ++half) {
                const int n = (t + half) * LM + m;
                for (int c0 = 0; c0 < a.Rp; c0 += 32) {
                    float v[32];
                    tmem_ld32(tmem + lane_base + half * RS + c0, v);
                    tmem_wait_ld();
                    if (n < a.N) {
#pragma unroll
                        for (int c = 0; c < 32; ++c) {
                            const int r = c0 + c;
                            if (r >= a.R) break;
                            const size_t o = (size_t)r * a.N + n;
                            if (split) a.part[(size_t)ks * a.R * a.N + o] = v[c];    // this K range's partial
                            else store_out(a, o, v[c]);
                        }
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(acc_empty);
            if (split) {
                // this warp's rows (quadrant `quad` of both tiles) are its own:
                // the last K range to finish them, by a per-(pair, quadrant)
                // arrival counter, sums the partials in split order (the
                // result does not depend on the arrival order)
                __threadfence();
                __syncwarp();
                unsigned last = 0;
                if (lane == 0) {
                    unsigned *cnt = a.counters + pair * 4 + quad;
                    last = atomicAdd(cnt, 1u) == (unsigned)a.n_split - 1u;
                    if (last) {
                        *cnt = 0u;                                          // ready for the next call
                        __threadfence();
                    }
                }
                if (__shfl_sync(0xffffffffu, last, 0)) {
                    __threadfence();
                    // 8 rows a round: all their partials are loaded at once,
                    // then summed in split order
                    constexpr int RB = 8;
                    const size_t plane = (size_t)a.R * a.N;
                    for (int half = 0; half < (two ? 2 : 1); ++half) {
                        const int n = (t + half) * LM + m;
                        if (n >= a.N) continue;
                        for (int r0 = 0; r0 < a.R; r0 += RB) {
                            float p[kMaxSplit][RB];
#pragma unroll
                            for (int q = 0; q < kMaxSplit; ++q)
#pragma unroll
                                for (int j = 0; j < RB; ++j)
                                    p[q][j] = (q < a.n_split && r0 + j < a.R)
                                                  ? __ldcg(a.part + q * plane + (size_t)(r0 + j) * a.N + n) : 0.f;
#pragma unroll
                            for (int j = 0; j < RB; ++j) {
                                if (r0 + j >= a.R) break;
                                float y = 0.f;
#pragma unroll
                                for (int q = 0; q < kMaxSplit; ++q) y += p[q][j];
                                store_out(a, (size_t)(r0 + j) * a.N + n, y);
                            }
                        }
                    }
                }
            }
        }
    }

    // ------------------------------------------------------------ wind-down
    tc_fence_before();
    __syncthreads();
    if (*s_abort && threadIdx.x == 0) {
        report(a.status, CLOVER_ERR_TIMEOUT);
    }
    if (*s_abort && warp == kProducer && lane == 0) {
        // the loads still in flight land before the CTA's shared memory goes away
        for (int j = max(0, issued - kStages); j < issued; ++j) mbar_wait(&full[j % kStages], (j / kStages) & 1, kWaitL);
    }
    __syncthreads();
    tc_fence_after();
    if (warp == kMma) {
        __syncwarp();
        tmem_dealloc(tmem, tmem_cols);
    }
}

}  // namespace

int linear_max_rows() { return kMaxRows; }

constexpr int kSmsPlan = 152;              // SMs of a GB300 (planning constant; any GPU runs the plan)

// K ranges per tile pair: a layer with fewer weight tiles than SMs splits K so
// that about one CTA per SM streams it (at least 4 stages of K per range).
// The ranges' sum costs one L2 round trip per 8 rows at the end; measured at
// H = 4096 it pays off up to 32 rows (a head step at R = 4: 287 -> 252 us,
// R = 16: 303 -> 288 us) and not at 48 (355 -> 410 us).
constexpr int kSplitMaxRows = 32;

int linear_split(int R, int N, int K) {
    const int n_tiles = (N + LM - 1) / LM;
    if (n_tiles >= kSmsPlan || R > kSplitMaxRows) return 1;
    const int n_pairs = (n_tiles + 1) / 2;
    int s = kSmsPlan / n_pairs;
    s = min(s, (K / LK) / 4);
    s = min(s, kMaxSplit);
    return s < 1 ? 1 : s;
}

// Partials of one launch (at most kMaxRows rows) and the per-(pair, quadrant)
// counters, 16-byte aligned.
size_t linear_workspace_bytes(int R, int N, int K) {
    const int s = linear_split(R, N, K);
    if (s <= 1) return 0;
    const int rows = min(R, kMaxRows);
    const int n_pairs = ((N + LM - 1) / LM + 1) / 2;
    const size_t part = ((size_t)s * rows * N * 4 + 15) / 16 * 16;
    return part + sizeof(unsigned) * 4 * (size_t)n_pairs;
}

// One launch per slice of at most kMaxRows rows of x.  With a workspace of
// linear_workspace_bytes(R, N, K) bytes (zero-filled before first use) the
// plan's K split is used; without one, none.
cudaError_t launch_linear_tc(const void *x, const void *w, const void *res, void *out, int R, int N, int K, int mode,
                             void *workspace, size_t ws_bytes, int32_t *status, bool pdl, cudaStream_t stream) {
    static unsigned long long done[64];
    static int sms[64];
    cudaError_t err = ensure_smem_attr(linear_tc_kernel, LinSmem::alloc, done);
    if (err != cudaSuccess) return err;
    int dev = 0;
    if ((err = cudaGetDevice(&dev)) != cudaSuccess) return err;
    int &n_sm = sms[dev < 64 ? dev : 63];
    if (n_sm == 0 && (err = cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
        return err;
    const int n_tiles = (N + LM - 1) / LM;
    const int n_pairs = (n_tiles + 1) / 2;
    const size_t need = linear_workspace_bytes(R, N, K);
    const int n_split = (need > 0 && workspace && ws_bytes >= need) ? linear_split(R, N, K) : 1;
    const size_t out_elem = mode == CLOVER_LINEAR_F32 ? 4 : 2;
    CUtensorMap tw;
    if (!make_tmap_bf16_3d(&tw, w, K, N, 1, (uint64_t)K * 2, (uint64_t)N * K * 2, LK, LM, 1)) return cudaErrorInvalidValue;
    for (int r0 = 0; r0 < R; r0 += kMaxRows) {
        const int Rs = min(kMaxRows, R - r0);
        const int Rp = (Rs + 15) / 16 * 16;
        CUtensorMap tx;
        const void *xs = static_cast<const __nv_bfloat16 *>(x) + (size_t)r0 * K;
        if (!make_tmap_bf16_3d(&tx, xs, K, Rs, 1, (uint64_t)K * 2, (uint64_t)Rs * K * 2, LK, Rp, 1))
            return cudaErrorInvalidValue;
        LinArgs a;
        a.res = res ? static_cast<const __nv_bfloat16 *>(res) + (size_t)r0 * N : nullptr;
        a.out = static_cast<uint8_t *>(out) + (size_t)r0 * N * out_elem;
        a.R = Rs;
        a.Rp = Rp;
        a.N = N;
        a.K = K;
        a.mode = mode;
        a.n_tiles = n_tiles;
        a.n_split = n_split;
        a.part = n_split > 1 ? static_cast<float *>(workspace) : nullptr;
        a.counters = n_split > 1 ? reinterpret_cast<unsigned *>(static_cast<uint8_t *>(workspace) + need -
                                                                sizeof(unsigned) * 4 * (size_t)n_pairs)
                                 : nullptr;
        a.status = status;
        const int grid = n_split > 1 ? n_pairs * n_split : min(n_sm, n_tiles);
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(grid, 1, 1);
        cfg.blockDim = dim3(kThreadsL, 1, 1);
        cfg.dynamicSmemBytes = LinSmem::alloc;
        cfg.stream = stream;
        cudaLaunchAttribute attr;
        attr.id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr.val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = &attr;
        cfg.numAttrs = pdl ? 1 : 0;
        if ((err = cudaLaunchKernelEx(&cfg, linear_tc_kernel, tw, tx, a)) != cudaSuccess) return err;
        if ((err = cudaGetLastError()) != cudaSuccess) return err;
    }
    return cudaSuccess;
}

}  // namespace clover
