// Per-node argmax over the vocabulary and the greedy acceptance walk, in one
// launch.
//
// The verification phase keeps the base model's own output (Section 1, and
// Section 2.1): the greedy token at tree node i is the first index of the
// maximum of its logit row.  A speculated child is accepted when its candidate
// token equals its parent's greedy token; the accepted path is walked from the
// root and its length is the paper's tokens/step (Section 4.1).
//
// Grid: one CTA per (logit row, vocabulary chunk).  Each CTA reduces its chunk
// with 16-byte loads to a packed 64-bit key (order-preserving value bits in the
// high word, bit-inverted index in the low word) so that one unsigned max
// gives "largest value, then smallest index", and folds it into the row's key
// with a 64-bit atomic max.  Per-row and per-sequence arrival counters find
// the CTA that finishes a sequence's last chunk; it decodes the argmax of
// every node and runs the walk in one warp, and resets the keys and counters.
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

// Vector body: 16-byte units [0, n_units) of the row from element `first`.
// Each round a thread issues kUnits independent loads (units tid + k*kThreads),
// takes the maximum over them, and only then looks for its first position.
template <typename T>
__device__ __forceinline__ void scan_vector(const T *row, int64_t first, int64_t n_units, uint64_t &best) {
    constexpr int E = 16 / sizeof(T);
    const uint4 *p = reinterpret_cast<const uint4 *>(row + first);
    for (int64_t base = 0; base < n_units; base += (int64_t)kThreads * kUnits) {
        uint4 w[kUnits];
#pragma unroll
        for (int k = 0; k < kUnits; ++k) {
            const int64_t u = base + threadIdx.x + (int64_t)k * kThreads;
            w[k] = (u < n_units) ? __ldcs(p + u) : make_uint4(0, 0, 0, 0);
        }
        float um[kUnits];
        float m = -INFINITY;
#pragma unroll
        for (int k = 0; k < kUnits; ++k) {
            const int64_t u = base + threadIdx.x + (int64_t)k * kThreads;
            um[k] = (u < n_units) ? unit_max(w[k], T()) : -INFINITY;
            m = fmaxf(m, um[k]);
        }
        // units are visited in increasing element order, so the first unit
        // reaching m holds this round's first maximum of the thread
        int kf = -1;
#pragma unroll
        for (int k = kUnits - 1; k >= 0; --k)
            if (um[k] == m && base + threadIdx.x + (int64_t)k * kThreads < n_units) kf = k;
        if (kf >= 0) {
            uint4 wf = w[0];
#pragma unroll
            for (int k = 1; k < kUnits; ++k)
                if (k == kf) wf = w[k];
            const int64_t u = base + threadIdx.x + (int64_t)kf * kThreads;
            const int e = unit_first(wf, m, T());
            best = umax64(best, make_key(m, (uint32_t)(first + u * E + e)));
        }
    }
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
    unsigned *row_count;           // [B*T] chunks of the row finished
    unsigned *seq_count;           // [B] rows of the sequence finished
    int32_t *status;
};

// Argmax of every node of sequence b from the merged row keys, then the greedy
// walk, by one warp: lane l owns nodes l and l + 32.  The walk reads the argmax
// of the current node from registers (warp shuffles), so each step costs no
// memory round trip.  The row keys and the counter are reset for the next call.
__device__ void accept_walk_warp(const AcceptArgs &a, int b) {
    const int lane = threadIdx.x & 31;
    const int T = a.T;
    const int32_t *par = a.parent + (size_t)b * T;
    const int32_t *cd = a.cand + (size_t)b * T;
    int p[2], c[2], am[2];
    bool invalid = false;
#pragma unroll
    for (int k = 0; k < 2; ++k) {
        const int i = lane + 32 * k;
        p[k] = -2;
        c[k] = 0;
        am[k] = 0;
        if (i < T) {
            const unsigned long long key = __ldcg(a.row_key + (size_t)b * T + i);
            am[k] = (int)(0xFFFFFFFFu - (uint32_t)(key & 0xFFFFFFFFull));
            a.argmax_out[(size_t)b * T + i] = am[k];
            a.row_key[(size_t)b * T + i] = 0ull;                      // ready for the next call
            p[k] = __ldg(par + i);
            c[k] = __ldg(cd + i);
            if (i == 0 ? (p[k] != -1) : (p[k] < 0 || p[k] >= i)) invalid = true;
        }
    }
    int32_t *path = a.path_out + (size_t)b * T;
    for (int i = lane; i < T; i += 32) path[i] = -1;
    __syncwarp();
    int cur = 0, len = 1;
    if (lane == 0) path[0] = 0;
    auto argmax_of = [&](int node) {
        const int lo = __shfl_sync(0xffffffffu, am[0], node & 31);
        const int hi = __shfl_sync(0xffffffffu, am[1], node & 31);
        return (node >> 5) ? hi : lo;
    };
    if (__any_sync(0xffffffffu, invalid)) {
        if (lane == 0) report(a.status, CLOVER_ERR_BAD_TREE);
    } else {
        // at most T - 1 steps: every step moves to a larger node index
        for (int step = 1; step < T; ++step) {
            const int want = argmax_of(cur);
            const unsigned lo = __ballot_sync(0xffffffffu, p[0] == cur && c[0] == want);
            const unsigned hi = __ballot_sync(0xffffffffu, p[1] == cur && c[1] == want);
            const uint64_t hits = (static_cast<uint64_t>(hi) << 32) | lo;
            if (hits == 0ull) break;
            cur = __ffsll(static_cast<long long>(hits)) - 1;
            if (lane == 0) path[len] = cur;
            ++len;
        }
    }
    const int bonus = argmax_of(cur);
    if (lane == 0) {
        a.accept_len[b] = len;
        a.bonus[b] = bonus;
        a.seq_count[b] = 0u;                                       // ready for the next call
    }
}

template <typename T>
__global__ void __launch_bounds__(kThreads) accept_kernel(const AcceptArgs a) {
    __shared__ uint64_t s_red[kThreads / 32];
    __shared__ int s_seq_last;
    const int row = blockIdx.x;               // b * T + i
    const int chunk_id = blockIdx.y;
    const int b = row / a.T;
    const T *rowp = static_cast<const T *>(a.logits) + (size_t)row * a.V;

    const int64_t lo = (int64_t)chunk_id * a.chunk;
    const int64_t hi = min((int64_t)a.V, lo + a.chunk);
    uint64_t best = 0ull;
    if (lo < hi) {
        // scalar head up to a 16-byte boundary, vector body, scalar tail
        constexpr int E = 16 / sizeof(T);
        const uintptr_t addr = reinterpret_cast<uintptr_t>(rowp + lo);
        int64_t head = (int64_t)(((16 - (addr & 15)) & 15) / sizeof(T));
        if ((addr % sizeof(T)) != 0) head = hi - lo;       // cannot happen for valid tensors
        head = min(head, hi - lo);
        const int64_t n_units = (hi - lo - head) / E;
        scan_scalar<T>(rowp, lo, lo + head, best);
        scan_vector<T>(rowp, lo + head, n_units, best);
        scan_scalar<T>(rowp, lo + head + n_units * E, hi, best);
    }
    best = block_max(best, s_red);

    // fold this chunk into the row's key and count it; the CTA finishing a
    // row's last chunk counts the row for its sequence, and the one finishing
    // the sequence's last row runs the walk (two levels keep each counter to a
    // few arrivals)
    if (threadIdx.x == 0) {
        atomicMax(a.row_key + row, static_cast<unsigned long long>(best));
        __threadfence();
        bool last = false;
        if (atomicAdd(a.row_count + row, 1u) == (unsigned)a.n_chunks - 1u) {
            a.row_count[row] = 0u;                              // ready for the next call
            __threadfence();
            last = (atomicAdd(a.seq_count + b, 1u) == (unsigned)a.T - 1u);
        }
        s_seq_last = last;
    }
    __syncthreads();
    if (!s_seq_last) return;
    if (threadIdx.x < 32) {
        __threadfence();
        accept_walk_warp(a, b);
    }
}

}  // namespace

// Vocabulary chunk per CTA: one round of kUnits 16-byte loads per thread
// (32 KB of bf16 or fp32 logits).
void accept_plan(int B, int T, int V, int dtype, int *n_chunks, int *chunk) {
    (void)B;
    (void)T;
    const int elems = 16 / (dtype == CLOVER_F32 ? 4 : 2);
    const int c = kThreads * kUnits * elems;
    *chunk = c;
    *n_chunks = (V + c - 1) / c;
}

size_t accept_workspace_bytes(int B, int T, int V, int dtype) {
    (void)V;
    (void)dtype;
    return sizeof(unsigned long long) * (size_t)B * T + sizeof(unsigned) * ((size_t)B * T + B);
}

cudaError_t launch_accept(const void *logits, const int32_t *cand, const int32_t *parent, int B, int T,
                          int V, int dtype, int32_t *argmax_out, int32_t *path_out, int32_t *accept_len,
                          int32_t *bonus, void *workspace, int32_t *status, cudaStream_t stream) {
    AcceptArgs a;
    a.logits = logits;
    a.cand = cand;
    a.parent = parent;
    a.B = B;
    a.T = T;
    a.V = V;
    accept_plan(B, T, V, dtype, &a.n_chunks, &a.chunk);
    a.argmax_out = argmax_out;
    a.path_out = path_out;
    a.accept_len = accept_len;
    a.bonus = bonus;
    a.row_key = static_cast<unsigned long long *>(workspace);
    a.row_count = reinterpret_cast<unsigned *>(a.row_key + (size_t)B * T);
    a.seq_count = a.row_count + (size_t)B * T;
    a.status = status;
    dim3 grid(B * T, a.n_chunks);
    if (dtype == CLOVER_F32) accept_kernel<float><<<grid, kThreads, 0, stream>>>(a);
    else accept_kernel<__nv_bfloat16><<<grid, kThreads, 0, stream>>>(a);
    return cudaGetLastError();
}

}  // namespace clover
