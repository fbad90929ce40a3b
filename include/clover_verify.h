/*
 * clover_verify.h -- C ABI of the GB300 (sm_103a) verification step of
 * Clover-style tree speculative decoding (arXiv 2405.00263).
 *
 * One verification step (Section 2.1, "verification phase"): the base model
 * scores all T speculated tokens, arranged as a token tree, in one pass.  The
 * library provides the data-parallel hot path of that pass:
 *
 *   clover_verify_attn    tree-masked attention of the T tree queries against
 *                         the committed KV cache plus the T new keys
 *                         (Section 2.2, Tree Attention);
 *   clover_verify_accept  per-node argmax of the logits and the greedy walk
 *                         that selects the accepted path (Section 2.1; the
 *                         tokens/step metric of Section 4.1);
 *   clover_verify_accept_typical
 *                         the same with the sampling-side (typical) acceptance
 *                         rule of the paper's tree sampling algorithm (Section 4);
 *   clover_verify_accept_ex
 *                         either rule, optionally fused with the commit of the
 *                         accepted K/V and launched to overlap the attention;
 *   clover_kv_compact     moves the accepted nodes' K/V to the front of the
 *                         tree slots (an engine step the paper leaves implicit);
 *   clover_verify_attn_paged, clover_kv_commit_paged
 *                         the attention and the commit on a paged KV cache;
 *   clover_linear(_ex), clover_embed_rows, clover_topk
 *                         the draft side: the dense layers of a Clover head,
 *                         the LM-head row embedding and the top-k of its
 *                         logits (Section 3).
 *
 * A second schedule of the same step: clover_verify_attn_ex with
 * CLOVER_ATTN_NO_APPEND leaves the caches untouched, and clover_kv_commit then
 * writes the accepted nodes' K/V straight from k_new/v_new.  The commit needs
 * only the accept result, so it can run while the attention still runs (its
 * writes, slots >= cache_len, are outside what the attention reads); the
 * final cache equals that of the append + compact schedule.
 *
 * Conventions shared by every entry point
 *   - All tensor pointers are DEVICE pointers owned by the caller; the library
 *     never allocates, frees or retains them.  Tensors are dense row-major.
 *   - Calls are asynchronous on `stream` (a cudaStream_t passed as void*;
 *     NULL = the legacy default stream).  The return value reports errors
 *     found on the host before anything is launched (and launch failures);
 *     nothing is launched when it is not CLOVER_OK.  Stream order holds for
 *     every call.  clover_kv_commit, clover_kv_commit_paged and
 *     clover_kv_compact launch as programmatic dependents of the kernel before
 *     them in the stream: their CTAs may be placed early, but they wait for
 *     that kernel's completion before their first memory access.
 *   - Errors found on the device (an invalid parent array, a cache that is too
 *     small, an invalid path) are OR-ed into `*status` (a device int32 the
 *     caller zeroes; may be NULL).  Kernels never trap and never wait without
 *     a bound; outputs are unspecified when a status bit is set.
 *   - Token tree: parent[b][0] == -1 (node 0 is the root) and
 *     0 <= parent[b][i] < i for i >= 1, so nodes are topologically numbered.
 *     Node i attends to node j iff j is i or an ancestor of i (the tree's
 *     topology as the attention mask, Section 2.2).
 *   - Limits: 1 <= T <= 128, D in {64, 128}, Hq a multiple of Hkv (query head h
 *     reads KV head h / (Hq/Hkv)), cache_len[b] + T <= Lcap.
 */
#ifndef CLOVER_VERIFY_H
#define CLOVER_VERIFY_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define CLOVER_API __attribute__((visibility("default")))
#else
#define CLOVER_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    CLOVER_OK = 0,
    CLOVER_ERR_INVALID_ARG = 1,  /* bad size, NULL or misaligned pointer, short workspace */
    CLOVER_ERR_UNSUPPORTED = 2,  /* outside the limits above (T > 128, D not 64/128, ...) */
    CLOVER_ERR_BAD_TREE = 4,     /* device: parent array is not a topologically numbered tree */
    CLOVER_ERR_CAPACITY = 8,     /* device: cache_len[b] < 0 or cache_len[b] + T > Lcap */
    CLOVER_ERR_CUDA = 16,        /* a CUDA launch or query failed */
    CLOVER_ERR_TIMEOUT = 32,     /* device: a bounded wait gave up (see below) */
    CLOVER_ERR_SCRATCH_LIMIT = 64, /* clover_verify_attn_noalloc: scratch need exceeds its static buffer */
    CLOVER_ERR_CHECK = 128       /* device, CLOVER_CHECKED builds only: an index check failed (see below) */
} clover_status;

/*
 * CLOVER_ERR_CHECK: a library built with -DCLOVER_CHECKED checks, on the
 * device, the indices its kernels compute before the global accesses they
 * guard: query rows and key ranges of the attention against B*T and the
 * sequence's key count, output rows against B*T, split-KV workspace slots and
 * arrival counters against ws_bytes, committed and compacted cache slots
 * against Lcap, and the source nodes of a commit against T.  A failed check
 * sets this bit and skips the access; it never traps.  Ordinary builds
 * compile the checks out and never set it; clover_build_flags() tells the two
 * apart.
 */

/*
 * CLOVER_ERR_TIMEOUT is raised by the kernels that wait on barriers: the bf16
 * tensor-core attention (clover_verify_attn, _ex, _paged, _noalloc with bf16)
 * and clover_linear.  Each of their waits gives up after about 0.5 s; the
 * kernel then winds down (waits, again bounded, for its copies in flight and
 * frees its tensor memory) and sets this bit.  The outputs of that call are
 * unspecified; the context stays usable.  The other kernels never wait.
 */

typedef enum {
    CLOVER_F32 = 0,   /* float32 storage, fp32 arithmetic (no TF32) */
    CLOVER_BF16 = 1   /* bfloat16 storage, fp32 accumulation, bf16 output (round to nearest even) */
} clover_dtype;

/* Version of this ABI (incremented on any incompatible change). */
CLOVER_API int clover_abi_version(void);

/* Build options of the loaded library: CLOVER_BUILD_CHECKED when it was
 * compiled with -DCLOVER_CHECKED (device index checks, CLOVER_ERR_CHECK). */
#define CLOVER_BUILD_CHECKED 1
CLOVER_API int clover_build_flags(void);

/* Short English name of a status code (static storage). */
CLOVER_API const char *clover_status_string(int status);

/*
 * Bytes of device workspace clover_verify_attn needs for these sizes
 * (split-KV partial results and per-head arrival counters).  0 when none is
 * needed (one key range per head: no split) and when the sizes are outside
 * the limits.
 */
CLOVER_API size_t clover_verify_attn_workspace_size(int B, int T, int Hq, int Hkv, int D, int Lcap,
                                         clover_dtype dtype);

/*
 * Tree-masked attention of one verification step (Section 2.1 verification
 * phase; Section 2.2 Tree Attention with the tree topology as the mask).
 *
 * For every sequence b, node i and query head h (g = h / (Hq/Hkv)):
 *   out[b,i,h,:] = softmax_j(scale * q[b,i,h,:] . key_j) . value_j
 * over the keys j = cache slots 0..cache_len[b]-1 of KV head g, and the tree
 * nodes m that are i or an ancestor of i (key k_new[b,m,g,:], value v_new[b,m,g,:]).
 *
 *   q        [B,T,Hq,D]      dtype   query rows of the tree nodes (positions already applied)
 *   k_new    [B,T,Hkv,D]     dtype   keys of the tree nodes
 *   v_new    [B,T,Hkv,D]     dtype   values of the tree nodes
 *   k_cache  [B,Hkv,Lcap,D]  dtype   in/out: slots [0, cache_len[b]) are read;
 *   v_cache  [B,Hkv,Lcap,D]  dtype   slots [cache_len[b], cache_len[b]+T) receive
 *                                    k_new/v_new of nodes 0..T-1 (the append)
 *   cache_len[B]             int32   committed length of each sequence (read only)
 *   parent   [B,T]           int32   the token tree (see conventions)
 *   out      [B,T,Hq,D]      dtype   attention output
 *   scale                    float   softmax scale; <= 0 selects 1/sqrt(D)
 *   workspace, ws_bytes              device scratch of at least
 *                                    clover_verify_attn_workspace_size(...) bytes,
 *                                    16-byte aligned.  It must be zero-filled before
 *                                    its first use; every call leaves it ready for the
 *                                    next one.  One workspace serves calls with the
 *                                    same B, T, Hq, Hkv, D and dtype and any Lcap up to
 *                                    the one it was sized for; for other sizes zero it
 *                                    again.  After a call that raised
 *                                    CLOVER_ERR_TIMEOUT, zero it again.  Calls sharing
 *                                    a workspace must not overlap on the device, apart
 *                                    from the overlap of CLOVER_ATTN_PDL launches
 *                                    (clover_verify_attn_ex), which is safe.
 *   status                           device int32 error bits (may be NULL)
 * q, k_new, v_new, caches and out must be 16-byte aligned.
 */
CLOVER_API clover_status clover_verify_attn(const void *q, const void *k_new, const void *v_new,
                                 void *k_cache, void *v_cache, const int32_t *cache_len,
                                 const int32_t *parent, void *out,
                                 int B, int T, int Hq, int Hkv, int D, int Lcap,
                                 clover_dtype dtype, float scale,
                                 void *workspace, size_t ws_bytes,
                                 int32_t *status, void *stream);

/* Flags of clover_verify_attn_ex. */
#define CLOVER_ATTN_NO_APPEND 1u    /* the call only reads k_cache/v_cache (no append) */
#define CLOVER_ATTN_PDL 2u          /* launch as a programmatic dependent of the kernel queued before it */
#define CLOVER_ATTN_CACHE_READY 4u  /* with CLOVER_ATTN_PDL: the cache may be read before that kernel ends */
#define CLOVER_ATTN_INPUTS_READY 8u /* with CLOVER_ATTN_PDL: every input may be read before that kernel ends */

/*
 * clover_verify_attn with flags: 0 is clover_verify_attn itself.
 *   CLOVER_ATTN_NO_APPEND skips the append, so slots >= cache_len[b] are
 *     neither read for the result nor written.
 *   CLOVER_ATTN_PDL launches the bf16 (tensor-core) kernel as a programmatic
 *     dependent of the kernel queued just before it on `stream`: its CTAs may
 *     be placed once every CTA of that kernel has started (this library's
 *     attention kernels allow it at their start), and they set up their
 *     barriers and tensor memory while it runs.  Every read of an input still
 *     waits for that kernel's completion (griddepcontrol.wait), so the results
 *     and stream order are those of an ordinary launch.
 *   CLOVER_ATTN_CACHE_READY (with CLOVER_ATTN_PDL) states that cache_len, the
 *     cache slots [0, cache_len[b]) and (paged) the block table are not
 *     written by the kernel queued before this call, nor by any kernel that
 *     may still run beside it (with programmatic launches, every kernel of the
 *     chain of programmatic dependents that ends in it).  The kernel then
 *     reads those before the preceding kernel completes: it loads the lengths
 *     and streams its first cache tiles while that kernel finishes.  q, k_new,
 *     v_new and parent are still read only after it completes, and every write
 *     (out, the append, the workspace) comes after that too.  Example: the
 *     attention launched right behind the projection that produced q, k_new
 *     and v_new.
 *   CLOVER_ATTN_INPUTS_READY (with CLOVER_ATTN_PDL) states the same of every
 *     input: q, k_new, v_new, parent, cache_len, the cache slots
 *     [0, cache_len[b]) and the block table.  The kernel then reads all of
 *     them, and runs its whole key loop, while the preceding kernel finishes;
 *     only its writes (out, the append, the workspace) wait for that kernel's
 *     completion.  Example: the attention of one micro-batch launched right
 *     behind the attention of another micro-batch, whose inputs were produced
 *     earlier.  Neither statement is checked: a kernel that does write one of
 *     these inputs while this call reads it gives unspecified results.  Such a
 *     launch is planned for a chain of them, several sharing the GPU at once:
 *     it takes about a fifth of the SMs' worth of CTAs, each over as long a
 *     key range as that allows; with at least that many (sequence, KV head,
 *     128-row tile) groups, one CTA takes every key of a group, with no split
 *     of the keys and no use of the workspace.  Fewer, longer CTAs then spend
 *     less of the GPU on setup and on merging splits, and the chain keeps the
 *     memory busy; a single such call on its own takes longer than an
 *     ordinary one.  With two or more 128-row tiles per (sequence, KV head)
 *     (grouped-query shapes, T * Hq / Hkv > 128), D = 128, a dense cache and
 *     no append, one CTA takes two row tiles, so each K/V tile it loads
 *     serves both.  Its results may differ from an ordinary launch's in the
 *     last bits (the key ranges are summed in another order); they do not
 *     depend on what runs beside it.
 * The fp32 (CUDA-core) kernel is launched the ordinary way whatever the launch
 * flags say.  Other flag bits: CLOVER_ERR_INVALID_ARG.
 */
CLOVER_API clover_status clover_verify_attn_ex(const void *q, const void *k_new, const void *v_new,
                                    void *k_cache, void *v_cache, const int32_t *cache_len,
                                    const int32_t *parent, void *out,
                                    int B, int T, int Hq, int Hkv, int D, int Lcap,
                                    clover_dtype dtype, float scale,
                                    void *workspace, size_t ws_bytes,
                                    int32_t *status, void *stream, uint32_t flags);

/*
 * Paged KV cache (an engine's block-table layout; the paper leaves the cache
 * layout implicit).  The pools k_pages, v_pages are [n_pages, Hkv, page_size, D]
 * (dtype, 16-byte aligned); block_table [B, max_pages] int32 maps cache slot s
 * of sequence b to row s % page_size of page block_table[b][s / page_size].
 * page_size is a power of two in [16, 1024]; the cache capacity is
 * Lcap = page_size * max_pages slots.  Entries for slots < cache_len[b] (and,
 * for the commit, < cache_len[b] + accept_len[b]) must be page ids in
 * [0, n_pages); another id found on the device raises CLOVER_ERR_INVALID_ARG
 * (device bit) and the access goes to page 0 (results unspecified).  Entries
 * past those are not read.
 */

/* Bytes of device workspace clover_verify_attn_paged needs (0 outside the limits). */
CLOVER_API size_t clover_verify_attn_paged_workspace_size(int B, int T, int Hq, int Hkv, int D, int page_size,
                                                          int max_pages, clover_dtype dtype);

/*
 * Tree-masked attention over a paged cache: clover_verify_attn_ex with
 * CLOVER_ATTN_NO_APPEND on the cache the block table describes (the pools are
 * only read; commit the accepted K/V with clover_kv_commit_paged).  Same
 * arguments, limits and results, with Lcap = page_size * max_pages; bf16 runs
 * on the tensor-core kernel (a 128-key tile is read as 128 / page_size boxes
 * when pages are smaller), fp32 on the FMA kernel.
 */
CLOVER_API clover_status clover_verify_attn_paged(const void *q, const void *k_new, const void *v_new,
                                   const void *k_pages, const void *v_pages, const int32_t *block_table,
                                   int n_pages, int page_size, int max_pages,
                                   const int32_t *cache_len, const int32_t *parent, void *out,
                                   int B, int T, int Hq, int Hkv, int D, clover_dtype dtype, float scale,
                                   void *workspace, size_t ws_bytes, int32_t *status, void *stream);

/*
 * clover_verify_attn_paged with the launch flags of clover_verify_attn_ex:
 * CLOVER_ATTN_PDL, CLOVER_ATTN_CACHE_READY, CLOVER_ATTN_INPUTS_READY (the
 * statements cover the pools, the block table and the lengths), and
 * CLOVER_ATTN_NO_APPEND, accepted and implied (a paged call never appends).
 * Other flag bits: CLOVER_ERR_INVALID_ARG.
 */
CLOVER_API clover_status clover_verify_attn_paged_ex(const void *q, const void *k_new, const void *v_new,
                                   const void *k_pages, const void *v_pages, const int32_t *block_table,
                                   int n_pages, int page_size, int max_pages,
                                   const int32_t *cache_len, const int32_t *parent, void *out,
                                   int B, int T, int Hq, int Hkv, int D, clover_dtype dtype, float scale,
                                   void *workspace, size_t ws_bytes, int32_t *status, void *stream,
                                   uint32_t flags);

/*
 * clover_kv_commit into a paged cache: for every sequence b with L = cache_len[b]
 * and a = accept_len[b], slot L+j (its page from block_table) of every KV head
 * receives k_new/v_new of node path[j]; src_index_out[b][j] = path[j] (-1 past
 * a; may be NULL); new_cache_len[b] = L + a.  Errors as for clover_kv_commit,
 * with Lcap = page_size * max_pages.
 */
CLOVER_API clover_status clover_kv_commit_paged(void *k_pages, void *v_pages, const int32_t *block_table,
                                   int n_pages, int page_size, int max_pages,
                                   const void *k_new, const void *v_new, const int32_t *cache_len,
                                   const int32_t *path, const int32_t *accept_len, int32_t *new_cache_len,
                                   int32_t *src_index_out, int B, int T, int Hkv, int D, clover_dtype dtype,
                                   int32_t *status, void *stream);

/*
 * Draft side: the dense pieces of one Clover head step (Section 3).  All
 * tensors are device pointers, row-major, bf16 unless stated; no workspace
 * unless stated.
 */

/* Epilogues of clover_linear (y = x . w^T accumulated in fp32). */
#define CLOVER_LINEAR_F32 0       /* out fp32 = y (the LM head's logits) */
#define CLOVER_LINEAR_BF16 1      /* out bf16 = y */
#define CLOVER_LINEAR_RES_SILU 2  /* out bf16 = res + silu(y): the residual SiLU block of a head's MLP */
#define CLOVER_LINEAR_RES 3       /* out bf16 = res + y: a residual add (the attention decoder's Eq. 2) */

/*
 * Linear layer on the tensor cores: x [R,K], w [N,K] (output features by input
 * features), res [R,N] (modes 2-3; else may be NULL), out [R,N] (fp32 for
 * CLOVER_LINEAR_F32, else bf16).  Rounding: one fp32 accumulation, then one
 * rounding to bf16 (after the residual and SiLU) for the bf16 modes.
 * K a multiple of 64 (64 <= K); R >= 0, N >= 1; x, w, res, out 16-byte
 * aligned; out must not overlap x, w or res.  A bounded device wait that gives
 * up raises CLOVER_ERR_TIMEOUT (device bit).
 * workspace, ws_bytes: with at least clover_linear_workspace_size(R, N, K)
 * bytes (16-byte aligned, zero-filled before first use, left ready for the
 * next call; calls sharing it must not overlap on the device), a layer of at
 * most 32 rows with fewer 128-row weight tiles than a GB300 has SMs splits K
 * over more CTAs and sums the parts in a fixed order; with NULL (or a smaller
 * one), or more rows, it does not (the size is then 0).
 * The result is the same function either way (the fp32 summation order differs).
 */
CLOVER_API size_t clover_linear_workspace_size(int R, int N, int K);
CLOVER_API clover_status clover_linear(const void *x, const void *w, const void *res, void *out,
                                   int R, int N, int K, int mode, void *workspace, size_t ws_bytes,
                                   int32_t *status, void *stream);

/*
 * clover_linear with launch flags (clover_linear is this call with flags 0).
 * CLOVER_LINEAR_PDL: the layer is launched as a programmatic dependent of the
 * kernel before it in the stream.  Its set-up and the weight tiles of its
 * first pipeline stages are requested before that kernel completes; x, res,
 * out, the workspace and the status word are touched only after it does.  The
 * caller states that the kernel before it does not write w (the layers of a
 * head step: each reads the activations the one before writes, never a
 * weight).  Any other flag bit -> CLOVER_ERR_INVALID_ARG.
 */
#define CLOVER_LINEAR_PDL 1u
CLOVER_API clover_status clover_linear_ex(const void *x, const void *w, const void *res, void *out,
                                      int R, int N, int K, int mode, unsigned flags, void *workspace,
                                      size_t ws_bytes, int32_t *status, void *stream);

/*
 * The regressive connection's embedding (Section 3.4): e[r] = w[t[r]] / ||w[t[r]]||_2
 * (the token's row of the LM-head weight, normalised), w [V,H], tokens [R]
 * int32, e [R,H] bf16.  A token outside [0, V) -> CLOVER_ERR_INVALID_ARG
 * (device bit; that row of e is zero).  A zero row gives a zero embedding.
 */
CLOVER_API clover_status clover_embed_rows(const void *w, const int32_t *tokens, void *e,
                                   int R, int V, int H, int32_t *status, void *stream);

/* Bytes of device workspace clover_topk needs (0 outside the limits). */
CLOVER_API size_t clover_topk_workspace_size(int R, int V, int k);

/*
 * Top-k of each row of fp32 x [R,V] (the LM head's logits): values [R,k] fp32
 * and indices [R,k] int32, in decreasing value, equal values by increasing
 * index (-0 == +0).  1 <= k <= 32, k <= V.  The workspace (zero-filled before
 * first use) is left ready for the next call; calls sharing it must not
 * overlap on the device.  NaN in x: unspecified.
 */
CLOVER_API clover_status clover_topk(const float *x, int R, int V, int k, float *values, int32_t *indices,
                                   void *workspace, size_t ws_bytes, int32_t *status, void *stream);

/* Bytes of device workspace clover_verify_accept needs (0 outside the limits). */
CLOVER_API size_t clover_verify_accept_workspace_size(int B, int T, int V, clover_dtype dtype);

/*
 * Per-node greedy token and acceptance walk (Section 2.1: the base model
 * rejects wrong speculations; Section 1: outputs stay those of the base model;
 * Section 4.1: tokens/step is the accepted length).
 *
 *   logits   [B,T,V]  dtype  base-model logits at every tree node (any alignment)
 *   cand     [B,T]    int32  candidate token of every node; cand[b][0] (the root,
 *                            already emitted by the base model) is not checked
 *   parent   [B,T]    int32  the token tree
 *   argmax_out [B,T]  int32  smallest index v with logits[b,i,v] equal to the row
 *                            maximum (-0 == +0)
 *   path_out [B,T]    int32  accepted nodes from the root: path[0] = 0 and
 *                            path[k+1] = the smallest-index child c of path[k]
 *                            with cand[c] == argmax[path[k]]; padded with -1
 *   accept_len [B]    int32  number of accepted nodes (1 .. depth+1)
 *   bonus_token [B]   int32  argmax at the last accepted node (the next root)
 *   workspace, ws_bytes      >= clover_verify_accept_workspace_size(...) bytes,
 *                            8-byte aligned, zero-filled before first use; left
 *                            ready for the next call.  Calls sharing it must not
 *                            overlap on the device.
 */
CLOVER_API clover_status clover_verify_accept(const void *logits, const int32_t *cand, const int32_t *parent,
                                   int B, int T, int V, clover_dtype dtype,
                                   int32_t *argmax_out, int32_t *path_out,
                                   int32_t *accept_len, int32_t *bonus_token,
                                   void *workspace, size_t ws_bytes,
                                   int32_t *status, void *stream);

/* Bytes of device workspace clover_verify_accept_typical needs (0 outside the limits). */
CLOVER_API size_t clover_verify_accept_typical_workspace_size(int B, int T, int V, clover_dtype dtype);

/*
 * Typical acceptance: the sampling-side acceptance rule of the tree sampling
 * algorithm the paper evaluates with (Section 4, experiment setup; the rule
 * is Medusa's), beside the greedy rule of clover_verify_accept.  For node i
 * with logit row x_i:
 *     p_i = softmax(x_i / temperature),  H_i = -sum_v p_i(v) ln p_i(v),
 *     theta_i = min(epsilon, delta * exp(-H_i)).
 * The edge into child c (parent i) is accepted iff p_i(cand[c]) > theta_i; a
 * candidate outside [0, V) is rejected.  The accepted path ends at the deepest
 * node whose every edge from the root is accepted; among equally deep ones it
 * is the one that takes the smallest-index child at every step (the
 * lexicographically smallest node sequence).  No random numbers are drawn.
 *
 *   logits, cand, parent     as for clover_verify_accept; logits must be finite
 *                            or -inf (p = 0), with a finite maximum in every row
 *                            (+inf or NaN: outputs unspecified)
 *   temperature              > 0 and finite, with log2(e)/temperature a normal
 *                            fp32 number (else CLOVER_ERR_UNSUPPORTED)
 *   epsilon, delta           >= 0 and finite (0 makes theta 0: every candidate
 *                            of positive probability passes)
 *   argmax_out, path_out, accept_len, bonus_token
 *                            as for clover_verify_accept (the bonus token is the
 *                            argmax at the last accepted node)
 *   workspace, ws_bytes      >= clover_verify_accept_typical_workspace_size(...)
 *                            bytes, 16-byte aligned, zero-filled before first
 *                            use; left ready for the next call.  Calls sharing
 *                            it must not overlap on the device.
 * Precision: the softmax sums, the entropy and the comparison are fp32
 * (base-2 exponent and logarithm instructions); an edge whose ln p - ln theta
 * is within about 1e-4 of zero may be decided either way.
 */
CLOVER_API clover_status clover_verify_accept_typical(const void *logits, const int32_t *cand,
                                   const int32_t *parent, int B, int T, int V, clover_dtype dtype,
                                   double temperature, double epsilon, double delta,
                                   int32_t *argmax_out, int32_t *path_out,
                                   int32_t *accept_len, int32_t *bonus_token,
                                   void *workspace, size_t ws_bytes,
                                   int32_t *status, void *stream);

/* Flags of clover_verify_accept_ex. */
#define CLOVER_ACCEPT_TYPICAL 1u   /* typical rule (temperature, epsilon, delta) instead of greedy */
#define CLOVER_ACCEPT_COMMIT 2u    /* also commit the accepted K/V, as clover_kv_commit would */
#define CLOVER_ACCEPT_OVERLAP 4u   /* may start while the kernel queued before it still runs */

/* Bytes of device workspace clover_verify_accept_ex needs with these flags. */
CLOVER_API size_t clover_verify_accept_ex_workspace_size(int B, int T, int V, clover_dtype dtype, uint32_t flags);

/*
 * The acceptance step with options, in one launch:
 *   - the greedy rule (clover_verify_accept) or, with CLOVER_ACCEPT_TYPICAL,
 *     the typical rule (clover_verify_accept_typical; temperature, epsilon
 *     and delta are read only then);
 *   - with CLOVER_ACCEPT_COMMIT, the commit of the accepted path from the
 *     tree's K/V, with the effect of clover_kv_commit on the path and length
 *     this call produces: for every sequence b with L = cache_len[b] and a =
 *     accept_len[b], slot L+j of every KV head receives k_new/v_new of node
 *     path[j] (j < a), src_index_out[b][j] = path[j] (-1 past a; may be NULL),
 *     new_cache_len[b] = L + a.  k_cache, v_cache [B,Hkv,Lcap,D], k_new, v_new
 *     [B,T,Hkv,D] (16-byte aligned), cache_len, new_cache_len [B] (not
 *     overlapping), D in {64, 128}, Lcap >= T.  cache_len[b] < 0 or
 *     cache_len[b] + T > Lcap -> CLOVER_ERR_CAPACITY (device bit; that sequence
 *     is not committed).  Without the flag these arguments are not read.
 *   - with CLOVER_ACCEPT_OVERLAP, the launch is a programmatic dependent of
 *     the kernel queued just before it on `stream`: it may start once that
 *     kernel's CTAs have all started (this library's attention kernels allow
 *     that at their start) and run beside it.  The caller guarantees that the
 *     two touch disjoint memory apart from reads of the same inputs and the
 *     status word, as clover_verify_attn_ex with CLOVER_ATTN_NO_APPEND does
 *     with a commit into slots >= cache_len.  This call still completes only
 *     after that kernel has, so stream order is kept for everything queued
 *     later.  Where the overlap is unavailable the launch simply runs after it.
 * Other flag bits: CLOVER_ERR_INVALID_ARG.  Workspace: as for the chosen rule
 * (clover_verify_accept_ex_workspace_size).
 */
CLOVER_API clover_status clover_verify_accept_ex(const void *logits, const int32_t *cand, const int32_t *parent,
                                   int B, int T, int V, clover_dtype dtype,
                                   double temperature, double epsilon, double delta,
                                   void *k_cache, void *v_cache, const void *k_new, const void *v_new,
                                   const int32_t *cache_len, int Hkv, int D, int Lcap,
                                   int32_t *argmax_out, int32_t *path_out,
                                   int32_t *accept_len, int32_t *bonus_token,
                                   int32_t *new_cache_len, int32_t *src_index_out,
                                   void *workspace, size_t ws_bytes, uint32_t flags,
                                   int32_t *status, void *stream);

/*
 * clover_verify_accept_ex with the commit (CLOVER_ACCEPT_COMMIT, implied and
 * accepted) into a paged cache: slot L+j of every KV head lives in row
 * (L+j) % page_size of page block_table[b][(L+j) / page_size] of the pools
 * k_pages, v_pages [n_pages, Hkv, page_size, D]; Lcap = page_size * max_pages;
 * page ids as for clover_verify_attn_paged (an id outside [0, n_pages) found
 * on the device raises CLOVER_ERR_INVALID_ARG and that row is not written).
 * Every other argument, flag and result as for clover_verify_accept_ex.
 */
CLOVER_API clover_status clover_verify_accept_paged_ex(const void *logits, const int32_t *cand, const int32_t *parent,
                                   int B, int T, int V, clover_dtype dtype,
                                   double temperature, double epsilon, double delta,
                                   void *k_pages, void *v_pages, const int32_t *block_table,
                                   int n_pages, int page_size, int max_pages,
                                   const void *k_new, const void *v_new, const int32_t *cache_len, int Hkv, int D,
                                   int32_t *argmax_out, int32_t *path_out,
                                   int32_t *accept_len, int32_t *bonus_token,
                                   int32_t *new_cache_len, int32_t *src_index_out,
                                   void *workspace, size_t ws_bytes, uint32_t flags,
                                   int32_t *status, void *stream);

/*
 * Commit the accepted path to the cache (no counterpart in the paper, which
 * leaves the engine's cache handling implicit).  For every sequence b with
 * L = cache_len[b] and a = accept_len[b]:
 *   cache[b,g,L+j,:] <- cache[b,g,L+path[b][j],:]  for j < a, every KV head g,
 * for K and V, with the result of copying in increasing j (all reads happen
 * before any write); slots < L are not touched.
 *   k_cache, v_cache [B,Hkv,Lcap,D] dtype  in place, 16-byte aligned
 *   cache_len [B]        int32   length before the step (read only)
 *   path, accept_len             as produced by clover_verify_accept
 *   new_cache_len [B]    int32   out: L + a.  Must not overlap cache_len.
 *   src_index_out [B,T]  int32   out: L + path[b][j] for j < a, else -1 (may be NULL)
 */
CLOVER_API clover_status clover_kv_compact(void *k_cache, void *v_cache, const int32_t *cache_len,
                                const int32_t *path, const int32_t *accept_len,
                                int32_t *new_cache_len, int32_t *src_index_out,
                                int B, int T, int Hkv, int D, int Lcap, clover_dtype dtype,
                                int32_t *status, void *stream);

/*
 * Commit of the accepted path straight from the tree's K/V (the engine step of
 * clover_kv_compact without the append before it).  For every sequence b with
 * L = cache_len[b] and a = accept_len[b]:
 *   cache[b,g,L+j,:] <- new[b,path[b][j],g,:]  for j < a, every KV head g, K and V;
 * slots < L are not touched.
 *   k_cache, v_cache [B,Hkv,Lcap,D] dtype  out, 16-byte aligned
 *   k_new, v_new     [B,T,Hkv,D]    dtype  in, 16-byte aligned
 *   cache_len [B]        int32   length before the step (read only)
 *   path, accept_len             as produced by clover_verify_accept
 *   new_cache_len [B]    int32   out: L + a.  Must not overlap cache_len.
 *   src_index_out [B,T]  int32   out: path[b][j] (a tree node) for j < a, else -1 (may be NULL)
 * Errors: cache_len[b] + T > Lcap -> CLOVER_ERR_CAPACITY; a path entry outside
 * [0, T) or an accept_len outside [1, T] -> CLOVER_ERR_INVALID_ARG (device bits).
 */
CLOVER_API clover_status clover_kv_commit(void *k_cache, void *v_cache, const void *k_new, const void *v_new,
                               const int32_t *cache_len, const int32_t *path, const int32_t *accept_len,
                               int32_t *new_cache_len, int32_t *src_index_out,
                               int B, int T, int Hkv, int D, int Lcap, clover_dtype dtype,
                               int32_t *status, void *stream);

/*
 * Bytes of the static device scratch buffer behind clover_verify_attn_noalloc.
 */
#define CLOVER_NOALLOC_SCRATCH_BYTES ((size_t)8 << 20)

/*
 * clover_verify_attn without a caller-provided workspace.  The paper has no
 * counterpart; this entry point exists for deployment.
 *
 * Who needs it: callers that cannot allocate device memory themselves.  Two
 * examples are a plugin inside a serving process whose memory manager has
 * already reserved the free HBM for its own pool, and latency-critical code
 * that must not make a call that may synchronise the device (cudaMalloc can).
 * Such callers cannot supply the workspace clover_verify_attn asks for.
 *
 * Behaviour: the same computation, arguments and results as clover_verify_attn
 * (inputs and outputs are still caller-owned device memory).  The split-KV
 * scratch lives in one file-scope static device array of
 * CLOVER_NOALLOC_SCRATCH_BYTES (8 MiB).  Every GPU that loads the library holds
 * that array until the process exits.  This call allocates nothing: it calls no
 * cudaMalloc, cudaFree or allocating library routine.
 *   - The first call in a CUDA context (normally once per device; again after
 *     cudaDeviceReset or under another context of the device) looks up the
 *     array's device address with that context current (cudaGetSymbolAddress)
 *     and caches it under the context's id.  Make this first call before any
 *     stream capture that contains later calls.
 *   - Each call clears the part of the array that must start at zero (the
 *     arrival counters) with an asynchronous memset on `stream`, then launches.
 *     The rest of the array keeps the previous call's contents, which are
 *     overwritten before they are read.
 *   - All calls on a device share the one array: calls whose executions
 *     overlap on the GPU (on any streams) race and give wrong results.
 *     Serialise them.
 *   - Sizes whose scratch need (clover_verify_attn_workspace_size) exceeds the
 *     buffer are rejected with CLOVER_ERR_SCRATCH_LIMIT before anything is
 *     launched; other errors are those of clover_verify_attn.
 */
CLOVER_API clover_status clover_verify_attn_noalloc(const void *q, const void *k_new, const void *v_new,
                                                    void *k_cache, void *v_cache, const int32_t *cache_len,
                                                    const int32_t *parent, void *out,
                                                    int B, int T, int Hq, int Hkv, int D, int Lcap,
                                                    clover_dtype dtype, float scale,
                                                    int32_t *status, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* CLOVER_VERIFY_H */
