// Commit of the accepted path to the KV cache: for sequence b with committed
// length L and accepted nodes path[0..a-1], slot L + j receives the K/V of
// node path[j].  The paper leaves this engine step implicit.  Two sources:
//   compaction  the rows at slots L + path[j] (where the attention kernel
//               appended the tree's K/V) move to slots L + j; the result is
//               that of copying in increasing j, which equals a gather
//               because path[j] >= j;
//   commit      the rows come straight from k_new/v_new [B, T, Hkv, D] (no
//               append before it), into a dense cache or a paged one (slot
//               L + j is row (L + j) % page of page block_table[b][(L + j) / page]).
//
// One CTA per (KV head, sequence) stages the a accepted rows of K and V in
// shared memory and only then writes them, so a row that is both a source and
// a destination is read before it is overwritten.  The CTA of head 0 also
// writes the source indices and the new length.
#include "common.cuh"

namespace clover {
namespace {

constexpr int kThreads = 128;

__global__ void __launch_bounds__(kThreads) kv_compact_kernel(
    uint8_t *k_cache, uint8_t *v_cache, const uint8_t *k_new, const uint8_t *v_new, const int32_t *cache_len,
    const int32_t *path,
    const int32_t *accept_len, int32_t *new_cache_len, int32_t *src_index, int T, int Hkv,
    int row_bytes, int Lcap, const int32_t *block_table, int page_size, int page_shift, int max_pages,
    int n_pages, int32_t *status) {
    extern __shared__ uint4 stage[];          // [2][T][row_bytes / 16]
    __shared__ int s_src[kThreads];
    __shared__ int s_dst_page[kThreads];      // paged cache: page of slot L + j (-1: invalid id, skipped)
    __shared__ int s_ok;
    const int g = blockIdx.x;
    const int b = blockIdx.y;
    // launched as a programmatic dependent of the kernel before it in the
    // stream: every global access comes after that grid has completed
    wait_prerequisite_grids();
    // the length, the accepted count and the whole path row are loaded at
    // once, one path entry per thread (T <= kThreads)
    static_assert(kMaxTreeNodes <= kThreads, "one path entry per thread");
    const int L = __ldg(cache_len + b);
    const int a = __ldg(accept_len + b);
    const int jt = threadIdx.x;
    const int p = jt < T ? __ldg(path + (size_t)b * T + jt) : -1;
    const bool len_ok = (a >= 1 && a <= T);
    const bool cap_ok = (L >= 0 && L + T <= Lcap);
    const bool bad = jt < a && (p < 0 || p >= T);
    s_src[jt] = bad ? jt : p;
    bool bad_page = false;
    if (block_table && jt < a && a <= T && L >= 0 && L + T <= Lcap) {
        const int pg = __ldg(block_table + (size_t)b * max_pages + ((L + jt) >> page_shift));
        bad_page = pg < 0 || pg >= n_pages;
        s_dst_page[jt] = bad_page ? -1 : pg;
    }
    const bool bad_path = __syncthreads_or(bad || bad_page);
    if (threadIdx.x == 0) {
        s_ok = len_ok && cap_ok;
        if (g == 0 && !cap_ok) report(status, CLOVER_ERR_CAPACITY);
        if (g == 0 && (!len_ok || bad_path)) report(status, CLOVER_ERR_INVALID_ARG);
    }
    if (g == 0 && len_ok && cap_ok) {
        if (src_index && jt < T) {
            const int base = k_new ? 0 : L;         // a tree node (commit) or a cache slot
            src_index[(size_t)b * T + jt] = (jt < a) ? base + s_src[jt] : -1;
        }
        if (threadIdx.x == 0) new_cache_len[b] = L + a;
    }
    __syncthreads();
    if (!s_ok) return;

    const int units = row_bytes / 16;
    const size_t head_base = ((size_t)b * Hkv + g) * Lcap;
    const uint4 *ks = reinterpret_cast<const uint4 *>(k_new ? k_new : k_cache);
    const uint4 *vs = reinterpret_cast<const uint4 *>(v_new ? v_new : v_cache);
    for (int e = threadIdx.x; e < a * units; e += kThreads) {
        const int j = e / units;
        const int u = e % units;
        if (!CLOVER_IN(status, k_new ? s_src[j] : L + s_src[j], k_new ? T : Lcap)) continue;
        const size_t src = (k_new ? ((size_t)b * T + s_src[j]) * Hkv + g : head_base + L + s_src[j]) * units + u;
        stage[e] = ks[src];
        stage[T * units + e] = vs[src];
    }
    __syncthreads();
    uint4 *kd = reinterpret_cast<uint4 *>(k_cache);
    uint4 *vd = reinterpret_cast<uint4 *>(v_cache);
    for (int e = threadIdx.x; e < a * units; e += kThreads) {
        const int j = e / units;
        const int u = e % units;
        if (!CLOVER_IN(status, L + j, Lcap)) continue;
        size_t dst = (head_base + L + j) * units + u;
        if (block_table) {
            if (s_dst_page[j] < 0) continue;
            dst = (((size_t)s_dst_page[j] * Hkv + g) * page_size + ((L + j) & (page_size - 1))) * units + u;
        }
        kd[dst] = stage[e];
        vd[dst] = stage[T * units + e];
    }
}

}  // namespace

cudaError_t launch_kv_compact(void *k_cache, void *v_cache, const void *k_new, const void *v_new,
                              const int32_t *cache_len, const int32_t *path, const int32_t *accept_len,
                              int32_t *new_cache_len, int32_t *src_index, int B, int T, int Hkv, int D, int Lcap,
                              int dtype, int32_t *status, cudaStream_t stream, const int32_t *block_table,
                              int page_size, int max_pages, int n_pages) {
    int page_shift = 0;
    while (block_table && (1 << page_shift) < page_size) ++page_shift;
    const int row_bytes = D * (dtype == CLOVER_F32 ? 4 : 2);
    const size_t smem = (size_t)2 * T * row_bytes;
    static unsigned long long done[64];
    cudaError_t e = ensure_smem_attr(kv_compact_kernel, (size_t)2 * kMaxTreeNodes * 128 * 4, done);
    if (e != cudaSuccess) return e;
    // A programmatic dependent of the preceding kernel in the stream: its CTAs
    // may be placed while that kernel runs (an accept call lets them in at its
    // start) and wait in the kernel for its completion, so the copy starts
    // without a launch gap.
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(Hkv, B);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, kv_compact_kernel, static_cast<uint8_t *>(k_cache), static_cast<uint8_t *>(v_cache),
                           static_cast<const uint8_t *>(k_new), static_cast<const uint8_t *>(v_new), cache_len, path,
                           accept_len, new_cache_len, src_index, T, Hkv, row_bytes, Lcap, block_table, page_size,
                           page_shift, max_pages, n_pages, status);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace clover
