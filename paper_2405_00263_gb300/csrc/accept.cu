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
// with a 64-bit atomic max.  The CTA that finishes the last chunk of a
// sequence (per-sequence arrival counter) decodes the argmax of every node and
// runs the walk in one warp; it also resets the keys and the counter.
#include "common.cuh"

namespace clover {
namespace {

constexpr int kThreads = 256;
constexpr int kTargetCtas = 2 * 152 * 2;   // about four resident CTAs per SM on a 152-SM GPU

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

// Vector body: 16-byte units [u_lo, u_hi) of the row starting at element `first`.
template <typename T>
__device__ __forceinline__ void scan_vector(const T *row, int64_t first, int64_t n_units, uint64_t &best) {
    constexpr int E = 16 / sizeof(T);
    const uint4 *p = reinterpret_cast<const uint4 *>(row + first);
    int64_t u = threadIdx.x;
    // four independent 16-byte loads in flight per thread
    for (; u + 3 * kThreads < n_units; u += 4 * kThreads) {
        uint4 w[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) w[k] = __ldcs(p + u + k * kThreads);
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            float f[E];
            if constexpr (E == 8) {
                const uint32_t x[4] = {w[k].x, w[k].y, w[k].z, w[k].w};
#pragma unroll
                for (int h = 0; h < 4; ++h) {
                    f[2 * h] = __uint_as_float(x[h] << 16);
                    f[2 * h + 1] = __uint_as_float(x[h] & 0xFFFF0000u);
                }
            } else {
                f[0] = __uint_as_float(w[k].x); f[1] = __uint_as_float(w[k].y);
                f[2] = __uint_as_float(w[k].z); f[3] = __uint_as_float(w[k].w);
            }
            const int64_t base = first + (u + k * kThreads) * E;
#pragma unroll
            for (int e = 0; e < E; ++e) best = umax64(best, make_key(f[e], (uint32_t)(base + e)));
        }
    }
    for (; u < n_units; u += kThreads) {
        const uint4 w = __ldcs(p + u);
        float f[E];
        if constexpr (E == 8) {
            const uint32_t x[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
            for (int h = 0; h < 4; ++h) {
                f[2 * h] = __uint_as_float(x[h] << 16);
                f[2 * h + 1] = __uint_as_float(x[h] & 0xFFFF0000u);
            }
        } else {
            f[0] = __uint_as_float(w.x); f[1] = __uint_as_float(w.y);
            f[2] = __uint_as_float(w.z); f[3] = __uint_as_float(w.w);
        }
        const int64_t base = first + u * E;
#pragma unroll
        for (int e = 0; e < E; ++e) best = umax64(best, make_key(f[e], (uint32_t)(base + e)));
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
    unsigned *seq_count;           // [B] chunks of the sequence's rows finished
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

    // fold this chunk into the row's key, then count the chunk as done for the
    // sequence; the CTA finishing the sequence's last chunk runs the walk
    if (threadIdx.x == 0) {
        atomicMax(a.row_key + row, static_cast<unsigned long long>(best));
        __threadfence();
        const unsigned prev = atomicAdd(a.seq_count + b, 1u);
        s_seq_last = (prev == (unsigned)(a.T * a.n_chunks) - 1u);
    }
    __syncthreads();
    if (!s_seq_last) return;
    if (threadIdx.x < 32) {
        __threadfence();
        accept_walk_warp(a, b);
    }
}

}  // namespace

void accept_plan(int B, int T, int V, int dtype, int *n_chunks, int *chunk) {
    const int rows = B * T;
    int n = (kTargetCtas + rows - 1) / rows;
    const int elems = 16 / (dtype == CLOVER_F32 ? 4 : 2);
    const int max_by_size = (V + 4096 - 1) / 4096;          // at least 4096 elements per chunk
    if (n > max_by_size) n = max_by_size;
    if (n < 1) n = 1;
    int c = (V + n - 1) / n;
    c = (c + elems - 1) / elems * elems;
    n = (V + c - 1) / c;
    *n_chunks = n;
    *chunk = c;
}

size_t accept_workspace_bytes(int B, int T, int V, int dtype) {
    (void)V;
    (void)dtype;
    return sizeof(unsigned long long) * (size_t)B * T + sizeof(unsigned) * (size_t)B;
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
    a.seq_count = reinterpret_cast<unsigned *>(a.row_key + (size_t)B * T);
    a.status = status;
    dim3 grid(B * T, a.n_chunks);
    if (dtype == CLOVER_F32) accept_kernel<float><<<grid, kThreads, 0, stream>>>(a);
    else accept_kernel<__nv_bfloat16><<<grid, kThreads, 0, stream>>>(a);
    return cudaGetLastError();
}

}  // namespace clover
