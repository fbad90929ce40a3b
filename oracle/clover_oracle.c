/*
 * clover_oracle.c -- plain, slow fp64 CPU statement of the tree-speculative
 * verification step (Clover, arXiv 2405.00263).
 *
 * TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check and the CPU
 * baseline of the benchmark use this file.  It shares no code, header,
 * table or constant with the CUDA library; it reads the same input bytes and
 * widens them exactly (bf16 -> fp32 by a 16-bit shift, fp32 -> fp64).
 *
 * What it computes, step by step:
 *   tree      Section 2.2 (Tree Attention) and the caption of the tree-attention
 *             figure: the speculations form a token tree whose topology is a
 *             2-D matrix used as the attention mask.  Node i sees node j iff j
 *             lies on the path from the root to i (ancestor or self).
 *   attention Section 2.1 (verification phase) and Section 2.2: the target model
 *             scores all speculated tokens in one pass; each tree node attends
 *             to every committed cache key and to the tree nodes the mask allows.
 *             softmax(scale * q.k) . v in fp64, scale = 1/sqrt(D) unless given.
 *   argmax    Section 1 (outputs consistent with the base model) and Section 2.1:
 *             the base model's greedy token at every node; smallest index among
 *             equal maxima, -0 == +0.
 *   walk      Section 4.1 (tokens/step metric) and Section 2.1: from the root,
 *             repeatedly accept the smallest-index child whose candidate token
 *             equals the current node's argmax; the accepted length is the
 *             number of nodes on the path, the bonus token the argmax at its end.
 *   typical   Section 4 (experiment setup): the tree sampling algorithm taken
 *             over from Medusa; the edge into a child is accepted when its
 *             token's probability under the tempered softmax of the parent's
 *             logits exceeds min(epsilon, delta * exp(-entropy)); the longest
 *             accepted path wins (ties: lexicographically smallest).
 *   draft     Section 3 (the Clover heads): a linear layer with an optional
 *             residual SiLU (the heads' MLP block), the LM-head row embedding
 *             of the regressive connection (Section 3.4), and the top-k of the
 *             shared LM head's logits.
 *   append /  (engine step; the paper is silent) the T tree keys/values occupy
 *   compact   cache slots [L, L+T); the accepted nodes' K/V are then moved, in
 *             path order, to slots [L, L+a) and the length becomes L + a.
 *
 * Every pinned function is checked by the CPU tests against brute force,
 * library routines, closed forms and invariants; none is "parity unpinned".
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_OK 0
#define ORACLE_BAD_TREE 4
#define ORACLE_BAD_ARG 1
#define ORACLE_NO_MEMORY 64

#define ORACLE_F32 0
#define ORACLE_BF16 1

/* Exact widening of one stored element to double. */
static double load_elem(const void *base, int64_t index, int dtype)
{
    if (dtype == ORACLE_F32) {
        return (double)((const float *)base)[index];
    }
    uint16_t h = ((const uint16_t *)base)[index];
    uint32_t bits = (uint32_t)h << 16;
    float f;
    memcpy(&f, &bits, sizeof f);
    return (double)f;
}

/* parent[0] must be -1 and 0 <= parent[i] < i for i >= 1. */
static int tree_is_valid(const int32_t *parent, int T)
{
    if (T < 1 || parent[0] != -1) return 0;
    for (int i = 1; i < T; ++i)
        if (parent[i] < 0 || parent[i] >= i) return 0;
    return 1;
}

/* Is node j on the path from the root to node i?  Follows parent pointers. */
static int on_root_path(const int32_t *parent, int i, int j)
{
    for (int n = i; n >= 0; n = parent[n])
        if (n == j) return 1;
    return 0;
}

/*
 * The tree as the paper's 2-D mask matrix: mask[i*T + j] = 1 iff node j is an
 * ancestor of node i or i itself; depth[i] = number of edges from the root.
 */
int oracle_tree_mask(const int32_t *parent, int T, uint8_t *mask, int32_t *depth)
{
    if (!tree_is_valid(parent, T)) return ORACLE_BAD_TREE;
    for (int i = 0; i < T; ++i) {
        for (int j = 0; j < T; ++j) mask[(int64_t)i * T + j] = (uint8_t)on_root_path(parent, i, j);
        int d = 0;
        for (int n = i; parent[n] >= 0; n = parent[n]) ++d;
        depth[i] = d;
    }
    return ORACLE_OK;
}

typedef struct {
    const void *q, *k_new, *v_new, *k_cache, *v_cache;
    const int32_t *cache_len, *parent;
    int B, T, Hq, Hkv, D, Lcap, dtype;
    double scale;
} attn_problem;

/*
 * One output row: node i of sequence b, query head h.  KV head g = h / (Hq/Hkv).
 * Keys: cache slots 0..L-1 of head g, then tree nodes m on the root path of i.
 */
static int attention_row(const attn_problem *P, int b, int i, int h, double *out)
{
    const int G = P->Hq / P->Hkv;
    const int g = h / G;
    const int L = P->cache_len[b];
    const int D = P->D;
    const int32_t *parent = P->parent + (int64_t)b * P->T;

    double *q_row = (double *)malloc(sizeof(double) * (size_t)D);
    double *score = (double *)malloc(sizeof(double) * (size_t)(L + P->T));
    const void **v_base = (const void **)malloc(sizeof(void *) * (size_t)(L + P->T));
    int64_t *v_off = (int64_t *)malloc(sizeof(int64_t) * (size_t)(L + P->T));
    if (!q_row || !score || !v_base || !v_off) {
        free(q_row);
        free(score);
        free(v_base);
        free(v_off);
        return ORACLE_NO_MEMORY;
    }
    const int64_t q_off = (((int64_t)b * P->T + i) * P->Hq + h) * D;
    for (int d = 0; d < D; ++d) q_row[d] = load_elem(P->q, q_off + d, P->dtype);

    /* The keys this row may see: every committed cache slot, then the tree
     * nodes on its root path.  Each key's value row is remembered beside it. */
    int n_keys = 0;
    for (int j = 0; j < L; ++j) {
        const int64_t off = (((int64_t)b * P->Hkv + g) * P->Lcap + j) * D;
        double s = 0.0;
        for (int d = 0; d < D; ++d) s += q_row[d] * load_elem(P->k_cache, off + d, P->dtype);
        score[n_keys] = P->scale * s;
        v_base[n_keys] = P->v_cache;
        v_off[n_keys] = off;
        ++n_keys;
    }
    for (int m = 0; m < P->T; ++m) {
        if (!on_root_path(parent, i, m)) continue;
        const int64_t off = (((int64_t)b * P->T + m) * P->Hkv + g) * D;
        double s = 0.0;
        for (int d = 0; d < D; ++d) s += q_row[d] * load_elem(P->k_new, off + d, P->dtype);
        score[n_keys] = P->scale * s;
        v_base[n_keys] = P->v_new;
        v_off[n_keys] = off;
        ++n_keys;
    }

    /* softmax over the visible keys, then the weighted sum of their values */
    double mx = -INFINITY;
    for (int n = 0; n < n_keys; ++n)
        if (score[n] > mx) mx = score[n];
    double z = 0.0;
    for (int n = 0; n < n_keys; ++n) {
        score[n] = exp(score[n] - mx);
        z += score[n];
    }
    for (int d = 0; d < D; ++d) out[d] = 0.0;
    for (int n = 0; n < n_keys; ++n)
        for (int d = 0; d < D; ++d) out[d] += score[n] * load_elem(v_base[n], v_off[n] + d, P->dtype);
    for (int d = 0; d < D; ++d) out[d] /= z;

    free(q_row);
    free(score);
    free(v_base);
    free(v_off);
    return ORACLE_OK;
}

/*
 * Tree-masked attention output, in fp64.
 * rows: flattened row ids r = (b*T + i)*Hq + h to compute (NULL = all B*T*Hq,
 * in order); out: [n_rows, D].  scale <= 0 selects 1/sqrt(D).
 */
int oracle_tree_attention(const void *q, const void *k_new, const void *v_new,
                          const void *k_cache, const void *v_cache,
                          const int32_t *cache_len, const int32_t *parent,
                          int B, int T, int Hq, int Hkv, int D, int Lcap, int dtype,
                          double scale, const int64_t *rows, int64_t n_rows,
                          double *out, int n_threads)
{
    if (B < 1 || T < 1 || Hq < 1 || Hkv < 1 || D < 1 || Hq % Hkv != 0) return ORACLE_BAD_ARG;
    for (int b = 0; b < B; ++b) {
        if (!tree_is_valid(parent + (int64_t)b * T, T)) return ORACLE_BAD_TREE;
        if (cache_len[b] < 0 || cache_len[b] > Lcap) return ORACLE_BAD_ARG;
    }
    attn_problem P = {q, k_new, v_new, k_cache, v_cache, cache_len, parent,
                      B, T, Hq, Hkv, D, Lcap, dtype, scale > 0 ? scale : 1.0 / sqrt((double)D)};
    const int64_t total = rows ? n_rows : (int64_t)B * T * Hq;
    int status = ORACLE_OK;
#pragma omp parallel for schedule(dynamic, 4) num_threads(n_threads > 0 ? n_threads : 1)
    for (int64_t n = 0; n < total; ++n) {
        const int64_t r = rows ? rows[n] : n;
        const int h = (int)(r % Hq);
        const int i = (int)((r / Hq) % T);
        const int b = (int)(r / ((int64_t)Hq * T));
        int s = attention_row(&P, b, i, h, out + n * D);
        if (s != ORACLE_OK) {
#pragma omp atomic write
            status = s;
        }
    }
    return status;
}

/*
 * Argmax of each selected logit row: the smallest index whose value equals the
 * row maximum (values compared after exact widening, so -0 == +0).
 * rows: row ids in [0, n_rows_total) (NULL = all); out: [n_sel].
 */
int oracle_argmax(const void *logits, int64_t n_rows_total, int64_t V, int dtype,
                  const int64_t *rows, int64_t n_sel, int32_t *out, int n_threads)
{
    if (V < 1) return ORACLE_BAD_ARG;
    const int64_t total = rows ? n_sel : n_rows_total;
#pragma omp parallel for schedule(static) num_threads(n_threads > 0 ? n_threads : 1)
    for (int64_t n = 0; n < total; ++n) {
        const int64_t r = rows ? rows[n] : n;
        double best = load_elem(logits, r * V, dtype);
        int64_t best_v = 0;
        for (int64_t v = 1; v < V; ++v) {
            double x = load_elem(logits, r * V + v, dtype);
            if (x > best) {
                best = x;
                best_v = v;
            }
        }
        out[n] = (int32_t)best_v;
    }
    return ORACLE_OK;
}

/*
 * Greedy acceptance walk per sequence.  path [B,T] receives node indices from
 * the root, padded with -1; accept_len [B] the path length; bonus [B] the
 * argmax at the last accepted node.  cand[b][0] (the root token) is not checked.
 */
int oracle_accept_walk(const int32_t *parent, const int32_t *cand, const int32_t *amax,
                       int B, int T, int32_t *path, int32_t *accept_len, int32_t *bonus)
{
    for (int b = 0; b < B; ++b)
        if (!tree_is_valid(parent + (int64_t)b * T, T)) return ORACLE_BAD_TREE;
    for (int b = 0; b < B; ++b) {
        const int32_t *par = parent + (int64_t)b * T;
        const int32_t *cd = cand + (int64_t)b * T;
        const int32_t *am = amax + (int64_t)b * T;
        int32_t *pb = path + (int64_t)b * T;
        for (int j = 0; j < T; ++j) pb[j] = -1;
        int cur = 0, len = 1;
        pb[0] = 0;
        for (;;) {
            int next = -1;
            for (int c = cur + 1; c < T; ++c) {
                if (par[c] == cur && cd[c] == am[cur]) {
                    next = c;
                    break;
                }
            }
            if (next < 0) break;
            pb[len++] = next;
            cur = next;
        }
        accept_len[b] = len;
        bonus[b] = am[cur];
    }
    return ORACLE_OK;
}

/* The T tree keys/values of sequence b go to cache slots [L_b, L_b + T). */
int oracle_append_tree_kv(const void *k_new, const void *v_new, void *k_cache, void *v_cache,
                          const int32_t *cache_len, int B, int T, int Hkv, int D, int Lcap,
                          int elem_bytes)
{
    for (int b = 0; b < B; ++b)
        if (cache_len[b] < 0 || cache_len[b] + T > Lcap) return ORACLE_BAD_ARG;
    const size_t row = (size_t)D * elem_bytes;
    for (int b = 0; b < B; ++b)
        for (int g = 0; g < Hkv; ++g)
            for (int m = 0; m < T; ++m) {
                const int64_t src = ((int64_t)b * T + m) * Hkv + g;
                const int64_t dst = ((int64_t)b * Hkv + g) * Lcap + cache_len[b] + m;
                memcpy((char *)k_cache + dst * row, (const char *)k_new + src * row, row);
                memcpy((char *)v_cache + dst * row, (const char *)v_new + src * row, row);
            }
    return ORACLE_OK;
}

/*
 * Compaction, sequential semantics: for j = 0..a-1 copy slot L+path[j] to slot
 * L+j (K and V, every KV head); src_index[b][j] = L + path[j] (-1 past a);
 * cache_len[b] += a.
 */
int oracle_kv_compact(void *k_cache, void *v_cache, int32_t *cache_len, const int32_t *path,
                      const int32_t *accept_len, int B, int T, int Hkv, int D, int Lcap,
                      int elem_bytes, int32_t *src_index)
{
    const size_t row = (size_t)D * elem_bytes;
    for (int b = 0; b < B; ++b) {
        const int L = cache_len[b];
        const int a = accept_len[b];
        if (a < 1 || a > T || L < 0 || L + T > Lcap) return ORACLE_BAD_ARG;
        for (int j = 0; j < a; ++j)
            if (path[(int64_t)b * T + j] < 0 || path[(int64_t)b * T + j] >= T) return ORACLE_BAD_ARG;
    }
    for (int b = 0; b < B; ++b) {
        const int L = cache_len[b];
        const int a = accept_len[b];
        for (int j = 0; j < T; ++j) src_index[(int64_t)b * T + j] = -1;
        for (int j = 0; j < a; ++j) {
            const int src_slot = L + path[(int64_t)b * T + j];
            const int dst_slot = L + j;
            src_index[(int64_t)b * T + j] = src_slot;
            for (int g = 0; g < Hkv; ++g) {
                const int64_t base = ((int64_t)b * Hkv + g) * Lcap;
                memmove((char *)k_cache + (base + dst_slot) * row, (char *)k_cache + (base + src_slot) * row, row);
                memmove((char *)v_cache + (base + dst_slot) * row, (char *)v_cache + (base + src_slot) * row, row);
            }
        }
        cache_len[b] = L + a;
    }
    return ORACLE_OK;
}

/*
 * Commit from the tree's K/V (the same end state as append + compaction):
 * for j = 0..a-1, slot L+j of every KV head receives k_new/v_new of node
 * path[j]; src_index[b][j] = path[j] (-1 past a); cache_len[b] += a.
 */
int oracle_kv_commit(void *k_cache, void *v_cache, const void *k_new, const void *v_new, int32_t *cache_len,
                     const int32_t *path, const int32_t *accept_len, int B, int T, int Hkv, int D, int Lcap,
                     int elem_bytes, int32_t *src_index)
{
    const size_t row = (size_t)D * elem_bytes;
    for (int b = 0; b < B; ++b) {
        const int L = cache_len[b];
        const int a = accept_len[b];
        if (a < 1 || a > T || L < 0 || L + T > Lcap) return ORACLE_BAD_ARG;
        for (int j = 0; j < a; ++j)
            if (path[(int64_t)b * T + j] < 0 || path[(int64_t)b * T + j] >= T) return ORACLE_BAD_ARG;
    }
    for (int b = 0; b < B; ++b) {
        const int L = cache_len[b];
        const int a = accept_len[b];
        for (int j = 0; j < T; ++j) src_index[(int64_t)b * T + j] = -1;
        for (int j = 0; j < a; ++j) {
            const int node = path[(int64_t)b * T + j];
            src_index[(int64_t)b * T + j] = node;
            for (int g = 0; g < Hkv; ++g) {
                const int64_t src = ((int64_t)b * T + node) * Hkv + g;
                const int64_t dst = ((int64_t)b * Hkv + g) * Lcap + L + j;
                memcpy((char *)k_cache + dst * row, (const char *)k_new + src * row, row);
                memcpy((char *)v_cache + dst * row, (const char *)v_new + src * row, row);
            }
        }
        cache_len[b] = L + a;
    }
    return ORACLE_OK;
}

/*
 * Typical acceptance: the sampling-side acceptance rule of the tree sampling
 * algorithm the paper evaluates with (Section 4, experiment setup; the rule is
 * Medusa's).  All in fp64 on exactly widened logits x of each node i:
 *   p_i    = softmax(x_i / temperature)
 *   H_i    = -sum_v p_i(v) ln p_i(v)            (terms with p = 0 add nothing)
 *   theta_i = min(epsilon, delta * exp(-H_i))
 * The edge into child c (parent i) is accepted iff p_i(cand[c]) > theta_i,
 * decided as ln p > ln theta (ln 0 = -inf, so theta = 0 accepts every token of
 * positive probability); a candidate outside [0, V) is rejected.  A node is
 * accepted when every edge on its path from the root is; the root always is.
 * The chosen path ends at the deepest accepted node; among equally deep ones
 * it is the lexicographically smallest sequence of node indices.  accept_len
 * is its node count, bonus the argmax of the last node's logits.
 * argmax_out [B,T] (first index of the maximum), path [B,T] (-1 padded),
 * margin [B,T]: ln p - ln theta of the edge into each node (root: +inf;
 * p = 0 or an invalid candidate: -inf).
 */
int oracle_accept_typical(const void *logits, const int32_t *parent, const int32_t *cand, int B, int T,
                          int64_t V, int dtype, double temperature, double epsilon, double delta,
                          int32_t *argmax_out, int32_t *path, int32_t *accept_len, int32_t *bonus,
                          double *margin, int n_threads)
{
    if (V < 1 || T < 1 || !(temperature > 0.0) || !isfinite(temperature) || !(epsilon >= 0.0) ||
        !isfinite(epsilon) || !(delta >= 0.0) || !isfinite(delta))
        return ORACLE_BAD_ARG;
    for (int b = 0; b < B; ++b)
        if (!tree_is_valid(parent + (int64_t)b * T, T)) return ORACLE_BAD_TREE;
    const int64_t rows = (int64_t)B * T;
    double *row_max = malloc(sizeof(double) * (size_t)rows);     /* max of x / temperature */
    double *row_lse = malloc(sizeof(double) * (size_t)rows);     /* ln sum exp(z - max) */
    double *row_log_theta = malloc(sizeof(double) * (size_t)rows);
    int32_t *row_amax = malloc(sizeof(int32_t) * (size_t)rows);
    if (!row_max || !row_lse || !row_log_theta || !row_amax) {
        free(row_max);
        free(row_lse);
        free(row_log_theta);
        free(row_amax);
        return ORACLE_NO_MEMORY;
    }
#pragma omp parallel for schedule(static) num_threads(n_threads > 0 ? n_threads : 1)
    for (int64_t r = 0; r < rows; ++r) {
        double best = load_elem(logits, r * V, dtype);
        int64_t best_v = 0;
        double m = -INFINITY;
        for (int64_t v = 0; v < V; ++v) {
            const double x = load_elem(logits, r * V + v, dtype);
            if (x > best) {
                best = x;
                best_v = v;
            }
            const double z = x / temperature;
            if (z > m) m = z;
        }
        double s = 0.0;
        for (int64_t v = 0; v < V; ++v) s += exp(load_elem(logits, r * V + v, dtype) / temperature - m);
        const double lse = log(s);
        double h = 0.0;
        for (int64_t v = 0; v < V; ++v) {
            const double log_p = load_elem(logits, r * V + v, dtype) / temperature - m - lse;
            const double p = exp(log_p);
            if (p > 0.0) h -= p * log_p;
        }
        row_amax[r] = (int32_t)best_v;
        row_max[r] = m;
        row_lse[r] = lse;
        const double log_eps = log(epsilon);           /* -inf for 0 */
        const double log_dh = log(delta) - h;          /* ln(delta e^-H) */
        row_log_theta[r] = log_eps < log_dh ? log_eps : log_dh;
    }
    int32_t *acc = malloc(sizeof(int32_t) * (size_t)T);
    int32_t *reach = malloc(sizeof(int32_t) * (size_t)T);
    int32_t *depth = malloc(sizeof(int32_t) * (size_t)T);
    int32_t *best_path = malloc(sizeof(int32_t) * (size_t)T);
    int32_t *this_path = malloc(sizeof(int32_t) * (size_t)T);
    int status = ORACLE_OK;
    if (!acc || !reach || !depth || !best_path || !this_path) status = ORACLE_NO_MEMORY;
    for (int b = 0; b < B && status == ORACLE_OK; ++b) {
        const int32_t *par = parent + (int64_t)b * T;
        const int32_t *cd = cand + (int64_t)b * T;
        double *mg = margin + (int64_t)b * T;
        for (int c = 0; c < T; ++c) argmax_out[(int64_t)b * T + c] = row_amax[(int64_t)b * T + c];
        /* each edge on its own */
        acc[0] = 1;
        mg[0] = INFINITY;
        for (int c = 1; c < T; ++c) {
            const int64_t r = (int64_t)b * T + par[c];
            if (cd[c] < 0 || (int64_t)cd[c] >= V) {
                acc[c] = 0;
                mg[c] = -INFINITY;
                continue;
            }
            const double log_p = load_elem(logits, r * V + cd[c], dtype) / temperature - row_max[r] - row_lse[r];
            acc[c] = log_p > row_log_theta[r];
            mg[c] = log_p == -INFINITY ? -INFINITY : log_p - row_log_theta[r];
        }
        /* accepted nodes and their depths (parents come before children) */
        reach[0] = 1;
        depth[0] = 0;
        for (int c = 1; c < T; ++c) {
            reach[c] = reach[par[c]] && acc[c];
            depth[c] = depth[par[c]] + 1;
        }
        /* deepest accepted node; ties by the lexicographically smallest path */
        int best_len = 0;
        for (int c = 0; c < T; ++c) {
            if (!reach[c]) continue;
            const int len = depth[c] + 1;
            for (int n = c, k = len - 1; n >= 0; n = par[n], --k) this_path[k] = n;
            int better = len > best_len;
            if (len == best_len) {
                for (int k = 0; k < len; ++k) {
                    if (this_path[k] != best_path[k]) {
                        better = this_path[k] < best_path[k];
                        break;
                    }
                }
            }
            if (better) {
                best_len = len;
                memcpy(best_path, this_path, sizeof(int32_t) * (size_t)len);
            }
        }
        int32_t *pb = path + (int64_t)b * T;
        for (int k = 0; k < T; ++k) pb[k] = k < best_len ? best_path[k] : -1;
        accept_len[b] = best_len;
        bonus[b] = row_amax[(int64_t)b * T + best_path[best_len - 1]];
    }
    free(acc);
    free(reach);
    free(depth);
    free(best_path);
    free(this_path);
    free(row_max);
    free(row_lse);
    free(row_log_theta);
    free(row_amax);
    return status;
}

/*
 * Draft side (Section 3: the Clover heads), the dense pieces of one head step.
 *
 * Linear layer, fp64 on exactly widened inputs:
 *   y[r][n] = sum_k x[r][k] * w[n][k]                       (act 0)
 *   y[r][n] = res[r][n] + silu(sum_k x[r][k] * w[n][k])      (act 1: the
 *            residual SiLU block of the speculative heads' MLP)
 * with silu(v) = v / (1 + exp(-v)).  x [R,K], w [N,K] (output features by
 * input features), res [R,N] (act 1 only), y [R,N].
 */
int oracle_linear(const void *x, const void *w, const void *res, int R, int N, int K, int dtype, int act,
                  double *y, int n_threads)
{
    if (R < 0 || N < 1 || K < 1 || (act != 0 && act != 1) || (act == 1 && !res)) return ORACLE_BAD_ARG;
#pragma omp parallel for schedule(static) num_threads(n_threads > 0 ? n_threads : 1)
    for (int64_t rn = 0; rn < (int64_t)R * N; ++rn) {
        const int64_t r = rn / N, n = rn % N;
        double s = 0.0;
        for (int k = 0; k < K; ++k) s += load_elem(x, r * K + k, dtype) * load_elem(w, n * K + k, dtype);
        if (act == 1) s = load_elem(res, r * N + n, dtype) + s / (1.0 + exp(-s));
        y[rn] = s;
    }
    return ORACLE_OK;
}

/*
 * The regressive connection's embedding (Section 3.4): the token's row of the
 * LM-head weight after normalisation, e = w[t] / ||w[t]||_2.  w [V,H], tokens
 * [R] in [0, V), e [R,H].
 */
int oracle_embed_rows(const void *w, const int32_t *tokens, int R, int V, int H, int dtype, double *e)
{
    for (int r = 0; r < R; ++r)
        if (tokens[r] < 0 || tokens[r] >= V) return ORACLE_BAD_ARG;
    for (int r = 0; r < R; ++r) {
        double s = 0.0;
        for (int h = 0; h < H; ++h) {
            const double v = load_elem(w, (int64_t)tokens[r] * H + h, dtype);
            s += v * v;
        }
        const double inv = s > 0.0 ? 1.0 / sqrt(s) : 0.0;
        for (int h = 0; h < H; ++h) e[(int64_t)r * H + h] = load_elem(w, (int64_t)tokens[r] * H + h, dtype) * inv;
    }
    return ORACLE_OK;
}

/*
 * Top-k of each row of fp64 values x [R,V]: the k largest, in decreasing
 * order, equal values by increasing index.  values, indices [R,k].
 */
int oracle_topk(const double *x, int R, int V, int k, double *values, int32_t *indices)
{
    if (k < 1 || k > V) return ORACLE_BAD_ARG;
    for (int r = 0; r < R; ++r) {
        const double *row = x + (int64_t)r * V;
        for (int j = 0; j < k; ++j) {
            /* the best element not yet taken: larger value, then smaller index */
            int best = -1;
            for (int v = 0; v < V; ++v) {
                int taken = 0;
                for (int q = 0; q < j; ++q)
                    if (indices[(int64_t)r * k + q] == v) taken = 1;
                if (taken) continue;
                if (best < 0 || row[v] > row[best]) best = v;
            }
            indices[(int64_t)r * k + j] = best;
            values[(int64_t)r * k + j] = row[best];
        }
    }
    return ORACLE_OK;
}
