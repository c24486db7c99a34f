/*
 * parason_oracle.c -- fp64 CPU oracle for fork-tree decode attention.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may call, link or
 * load this file: only the tests, the smoke check and the benchmark's CPU
 * baseline use it.  It shares no code, header, table or helper with the CUDA
 * library; both read the same raw input buffers and nothing else.
 *
 * What it computes.  The paper runs every Subtask and Trial branch of a
 * <Parallel> region as an independent worker (Sec. 3.4) and concatenates the
 * branch outputs into the context that follows (Fig. 1 caption, Sec. 3.1
 * "Trial Parallelism").  One decode step therefore needs, for every live
 * branch b, plain softmax attention of b's query over b's whole context: the
 * KV of every fork-tree node on the path root -> b, in root-first order.
 * The oracle evaluates exactly that definition, branch by branch, with no
 * sharing between branches, no tiling and no split of the KV range:
 *
 *   KV_b   = concat over nodes n on root->b of tokens t = 0 .. len(n)-1,
 *            token t of node n at physical page page_ids[node_page_ptr[n] + t/P],
 *            slot t % P   (P = page_size)
 *   s_t    = scale * sum_d q[b,h,d] * k_t[kvh,d]          kvh = h / (H_q/H_kv)
 *   m      = max_t s_t,   l = sum_t exp(s_t - m)
 *   o      = sum_t exp(s_t - m) * v_t[kvh] / l,   lse = m + ln l
 *
 * All arithmetic is fp64.  Inputs are widened exactly: bf16 and fp32 are
 * exact in fp64, an e4m3 byte is decoded from the OCP FP8 definition and
 * multiplied by its per-kv-head fp32 scale.  A branch whose whole path holds
 * no token gets o = 0 and lse = -inf (an empty softmax).
 *
 * The standalone LSE merge follows the same definition: two normalised
 * attention results over disjoint key sets A and B combine into the result
 * over A u B with weights exp(lse_A) and exp(lse_B).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

enum { ORACLE_BF16 = 0, ORACLE_FP32 = 1, ORACLE_FP8_E4M3_KV = 2 };
enum { ORACLE_OK = 0, ORACLE_EINVAL = 1, ORACLE_ENOMEM = 2 };

/* bf16 is the upper half of an IEEE binary32. */
double parason_oracle_bf16_to_double(uint16_t bits)
{
    uint32_t u = (uint32_t)bits << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* OCP FP8 E4M3: 1 sign bit, 4 exponent bits (bias 7), 3 mantissa bits,
 * no infinities, S.1111.111 is NaN, exponent field 0 is subnormal. */
double parason_oracle_e4m3_to_double(uint8_t bits)
{
    int sign = bits >> 7;
    int expo = (bits >> 3) & 0xF;
    int mant = bits & 0x7;
    double mag;
    if (expo == 0xF && mant == 0x7)
        return NAN;
    if (expo == 0)
        mag = ldexp((double)mant / 8.0, 1 - 7);
    else
        mag = ldexp(1.0 + (double)mant / 8.0, expo - 7);
    return sign ? -mag : mag;
}

static double load_elem(const void *base, int64_t idx, int dtype_code, double scale)
{
    switch (dtype_code) {
    case ORACLE_BF16:
        return parason_oracle_bf16_to_double(((const uint16_t *)base)[idx]);
    case ORACLE_FP32:
        return (double)((const float *)base)[idx];
    default: /* e4m3 byte times its fp32 scale */
        return parason_oracle_e4m3_to_double(((const uint8_t *)base)[idx]) * scale;
    }
}

/* Root-first list of the nodes on the path root -> node.  Returns its length,
 * or -1 if the parent chain is malformed. */
static int path_to_root(int32_t node, const int32_t *parent, int32_t num_nodes,
                        int32_t *path)
{
    int n = 0;
    int32_t cur = node;
    while (cur >= 0) {
        if (cur >= num_nodes || n >= num_nodes)
            return -1;
        path[n++] = cur;
        cur = parent[cur];
    }
    for (int i = 0; i < n / 2; ++i) {
        int32_t t = path[i];
        path[i] = path[n - 1 - i];
        path[n - 1 - i] = t;
    }
    return n;
}

/*
 * Decode-step attention for the selected branches.
 *
 * q       [num_leaves, H_q, d]          bf16 (fp32 in FP32 mode)
 * k_pages [num_pages, H_kv, page_size, d] bf16 / fp32 / e4m3 bytes
 * v_pages same layout as k_pages
 * k_scale, v_scale [H_kv] fp32, FP8 mode only
 * sel     branch indices to evaluate (NULL: all, in order)
 * out     [num_sel, H_q, d] fp64;  lse [num_sel, H_q] fp64 (natural log)
 */
int parason_oracle_decode(int32_t num_q_heads, int32_t num_kv_heads, int32_t head_dim,
                          int32_t page_size, int32_t mode, double sm_scale,
                          int32_t num_nodes, const int32_t *parent,
                          const int32_t *node_len, const int32_t *node_page_ptr,
                          const int32_t *page_ids, int32_t num_leaves,
                          const int32_t *leaf_node, const void *q,
                          const void *k_pages, const void *v_pages,
                          const float *k_scale, const float *v_scale,
                          int32_t num_sel, const int32_t *sel, double *out,
                          double *lse, int32_t num_threads)
{
    if (num_q_heads <= 0 || num_kv_heads <= 0 || num_q_heads % num_kv_heads != 0 ||
        head_dim <= 0 || page_size <= 0 || num_nodes < 0 || num_leaves < 0)
        return ORACLE_EINVAL;
    if (mode != ORACLE_BF16 && mode != ORACLE_FP32 && mode != ORACLE_FP8_E4M3_KV)
        return ORACLE_EINVAL;
    if (mode == ORACLE_FP8_E4M3_KV && (!k_scale || !v_scale))
        return ORACLE_EINVAL;
    if (!sel)
        num_sel = num_leaves;

    const int group = num_q_heads / num_kv_heads;
    const double scale = sm_scale > 0.0 ? sm_scale : 1.0 / sqrt((double)head_dim);
    const int q_code = (mode == ORACLE_FP32) ? ORACLE_FP32 : ORACLE_BF16;
    const int kv_code = mode;
    int status = ORACLE_OK;

#ifdef _OPENMP
    if (num_threads > 0)
        omp_set_num_threads(num_threads);
#else
    (void)num_threads;
#endif

#pragma omp parallel
    {
        int32_t *path = (int32_t *)malloc(sizeof(int32_t) * (size_t)(num_nodes > 0 ? num_nodes : 1));
        double *qv = (double *)malloc(sizeof(double) * (size_t)head_dim);
        double *acc = (double *)malloc(sizeof(double) * (size_t)head_dim);
        double *scores = NULL;
        int64_t scores_cap = 0;
        if (!path || !qv || !acc) {
#pragma omp atomic write
            status = ORACLE_ENOMEM;
        }

#pragma omp for schedule(dynamic, 1)
        for (int64_t task = 0; task < (int64_t)num_sel * num_q_heads; ++task) {
            if (status != ORACLE_OK)
                continue;
            const int32_t si = (int32_t)(task / num_q_heads);
            const int32_t h = (int32_t)(task % num_q_heads);
            const int32_t b = sel ? sel[si] : si;
            const int32_t kvh = h / group;
            double *o = out + ((int64_t)si * num_q_heads + h) * head_dim;
            double *lse_out = lse ? lse + (int64_t)si * num_q_heads + h : NULL;

            if (b < 0 || b >= num_leaves) {
#pragma omp atomic write
                status = ORACLE_EINVAL;
                continue;
            }
            const int plen = path_to_root(leaf_node[b], parent, num_nodes, path);
            if (plen < 0) {
#pragma omp atomic write
                status = ORACLE_EINVAL;
                continue;
            }
            int64_t total = 0;
            for (int i = 0; i < plen; ++i)
                total += node_len[path[i]];

            const double ks = (mode == ORACLE_FP8_E4M3_KV) ? (double)k_scale[kvh] : 1.0;
            const double vs = (mode == ORACLE_FP8_E4M3_KV) ? (double)v_scale[kvh] : 1.0;
            for (int dd = 0; dd < head_dim; ++dd)
                qv[dd] = load_elem(q, ((int64_t)b * num_q_heads + h) * head_dim + dd, q_code, 1.0);

            if (total == 0) {
                for (int dd = 0; dd < head_dim; ++dd)
                    o[dd] = 0.0;
                if (lse_out)
                    *lse_out = -INFINITY;
                continue;
            }
            if (total > scores_cap) {
                free(scores);
                scores = (double *)malloc(sizeof(double) * (size_t)total);
                scores_cap = scores ? total : 0;
                if (!scores) {
#pragma omp atomic write
                    status = ORACLE_ENOMEM;
                    continue;
                }
            }

            /* pass 1: scores s_t over the concatenated path, root first */
            int64_t pos = 0;
            double m = -INFINITY;
            for (int i = 0; i < plen; ++i) {
                const int32_t n = path[i];
                for (int32_t t = 0; t < node_len[n]; ++t) {
                    const int64_t page = page_ids[node_page_ptr[n] + t / page_size];
                    const int64_t row = ((page * num_kv_heads + kvh) * page_size + t % page_size) * head_dim;
                    double dot = 0.0;
                    for (int dd = 0; dd < head_dim; ++dd)
                        dot += qv[dd] * load_elem(k_pages, row + dd, kv_code, ks);
                    const double s = scale * dot;
                    scores[pos++] = s;
                    if (s > m)
                        m = s;
                }
            }

            /* pass 2: l = sum exp(s - m), o = sum exp(s - m) v / l */
            double l = 0.0;
            for (int dd = 0; dd < head_dim; ++dd)
                acc[dd] = 0.0;
            pos = 0;
            for (int i = 0; i < plen; ++i) {
                const int32_t n = path[i];
                for (int32_t t = 0; t < node_len[n]; ++t) {
                    const int64_t page = page_ids[node_page_ptr[n] + t / page_size];
                    const int64_t row = ((page * num_kv_heads + kvh) * page_size + t % page_size) * head_dim;
                    const double p = exp(scores[pos++] - m);
                    l += p;
                    for (int dd = 0; dd < head_dim; ++dd)
                        acc[dd] += p * load_elem(v_pages, row + dd, kv_code, vs);
                }
            }
            for (int dd = 0; dd < head_dim; ++dd)
                o[dd] = acc[dd] / l;
            if (lse_out)
                *lse_out = m + log(l);
        }
        free(scores);
        free(acc);
        free(qv);
        free(path);
    }
    return status;
}

/*
 * Tree-masked prefill (the join of a parallel block: the threads' text
 * becomes context of the main trajectory, Fig. 1, Sec. 3.1; each new token
 * attends causally).  Every token of every chunk node is a query:
 * queries are numbered chunk by chunk (query k = token t of chunk c, with k =
 * qbase_c + t), and query k attends to every token of every ancestor of
 * chunk_node[c] (root first) and to tokens 0 .. t of chunk_node[c] itself.
 *
 * q [num_queries, H_q, d]; sel query indices to evaluate (NULL: all);
 * out [num_sel, H_q, d] fp64; lse [num_sel, H_q] fp64 (natural log).
 */
int parason_oracle_prefill(int32_t num_q_heads, int32_t num_kv_heads, int32_t head_dim,
                           int32_t page_size, int32_t mode, double sm_scale,
                           int32_t num_nodes, const int32_t *parent,
                           const int32_t *node_len, const int32_t *node_page_ptr,
                           const int32_t *page_ids, int32_t num_chunks,
                           const int32_t *chunk_node, const void *q,
                           const void *k_pages, const void *v_pages,
                           const float *k_scale, const float *v_scale,
                           int32_t num_sel, const int32_t *sel, double *out,
                           double *lse, int32_t num_threads)
{
    if (num_q_heads <= 0 || num_kv_heads <= 0 || num_q_heads % num_kv_heads != 0 ||
        head_dim <= 0 || page_size <= 0 || num_nodes < 0 || num_chunks < 0)
        return ORACLE_EINVAL;
    if (mode != ORACLE_BF16 && mode != ORACLE_FP32 && mode != ORACLE_FP8_E4M3_KV)
        return ORACLE_EINVAL;
    if (mode == ORACLE_FP8_E4M3_KV && (!k_scale || !v_scale))
        return ORACLE_EINVAL;
    int64_t num_queries = 0;
    for (int32_t c = 0; c < num_chunks; ++c) {
        if (chunk_node[c] < 0 || chunk_node[c] >= num_nodes)
            return ORACLE_EINVAL;
        num_queries += node_len[chunk_node[c]];
    }
    if (!sel)
        num_sel = (int32_t)num_queries;

    const int group = num_q_heads / num_kv_heads;
    const double scale = sm_scale > 0.0 ? sm_scale : 1.0 / sqrt((double)head_dim);
    const int q_code = (mode == ORACLE_FP32) ? ORACLE_FP32 : ORACLE_BF16;
    const int kv_code = mode;
    int status = ORACLE_OK;

#ifdef _OPENMP
    if (num_threads > 0)
        omp_set_num_threads(num_threads);
#else
    (void)num_threads;
#endif

#pragma omp parallel
    {
        int32_t *path = (int32_t *)malloc(sizeof(int32_t) * (size_t)(num_nodes > 0 ? num_nodes : 1));
        double *qv = (double *)malloc(sizeof(double) * (size_t)head_dim);
        double *acc = (double *)malloc(sizeof(double) * (size_t)head_dim);
        double *scores = NULL;
        int64_t scores_cap = 0;
        if (!path || !qv || !acc) {
#pragma omp atomic write
            status = ORACLE_ENOMEM;
        }

#pragma omp for schedule(dynamic, 1)
        for (int64_t task = 0; task < (int64_t)num_sel * num_q_heads; ++task) {
            if (status != ORACLE_OK)
                continue;
            const int32_t si = (int32_t)(task / num_q_heads);
            const int32_t h = (int32_t)(task % num_q_heads);
            const int64_t k = sel ? sel[si] : si;
            const int32_t kvh = h / group;
            double *o = out + ((int64_t)si * num_q_heads + h) * head_dim;
            double *lse_out = lse ? lse + (int64_t)si * num_q_heads + h : NULL;
            if (k < 0 || k >= num_queries) {
#pragma omp atomic write
                status = ORACLE_EINVAL;
                continue;
            }
            /* the query's chunk and token */
            int32_t c = 0;
            int64_t base = 0;
            while (base + node_len[chunk_node[c]] <= k) {
                base += node_len[chunk_node[c]];
                ++c;
            }
            const int32_t own = chunk_node[c];
            const int32_t t_q = (int32_t)(k - base);
            const int plen = path_to_root(own, parent, num_nodes, path);
            if (plen < 0) {
#pragma omp atomic write
                status = ORACLE_EINVAL;
                continue;
            }
            /* visible tokens: all of every ancestor, tokens 0 .. t_q of own */
            int64_t total = 0;
            for (int i = 0; i < plen; ++i)
                total += (path[i] == own) ? t_q + 1 : node_len[path[i]];

            const double ks = (mode == ORACLE_FP8_E4M3_KV) ? (double)k_scale[kvh] : 1.0;
            const double vs = (mode == ORACLE_FP8_E4M3_KV) ? (double)v_scale[kvh] : 1.0;
            for (int dd = 0; dd < head_dim; ++dd)
                qv[dd] = load_elem(q, (k * num_q_heads + h) * head_dim + dd, q_code, 1.0);
            if (total > scores_cap) {
                free(scores);
                scores = (double *)malloc(sizeof(double) * (size_t)total);
                scores_cap = scores ? total : 0;
                if (!scores) {
#pragma omp atomic write
                    status = ORACLE_ENOMEM;
                    continue;
                }
            }

            /* pass 1: scores over the visible tokens, root first */
            int64_t pos = 0;
            double m = -INFINITY;
            for (int i = 0; i < plen; ++i) {
                const int32_t n = path[i];
                const int32_t vis = (n == own) ? t_q + 1 : node_len[n];
                for (int32_t t = 0; t < vis; ++t) {
                    const int64_t page = page_ids[node_page_ptr[n] + t / page_size];
                    const int64_t row = ((page * num_kv_heads + kvh) * page_size + t % page_size) * head_dim;
                    double dot = 0.0;
                    for (int dd = 0; dd < head_dim; ++dd)
                        dot += qv[dd] * load_elem(k_pages, row + dd, kv_code, ks);
                    const double s = scale * dot;
                    scores[pos++] = s;
                    if (s > m)
                        m = s;
                }
            }

            /* pass 2: l = sum exp(s - m), o = sum exp(s - m) v / l */
            double l = 0.0;
            for (int dd = 0; dd < head_dim; ++dd)
                acc[dd] = 0.0;
            pos = 0;
            for (int i = 0; i < plen; ++i) {
                const int32_t n = path[i];
                const int32_t vis = (n == own) ? t_q + 1 : node_len[n];
                for (int32_t t = 0; t < vis; ++t) {
                    const int64_t page = page_ids[node_page_ptr[n] + t / page_size];
                    const int64_t row = ((page * num_kv_heads + kvh) * page_size + t % page_size) * head_dim;
                    const double p = exp(scores[pos++] - m);
                    l += p;
                    for (int dd = 0; dd < head_dim; ++dd)
                        acc[dd] += p * load_elem(v_pages, row + dd, kv_code, vs);
                }
            }
            for (int dd = 0; dd < head_dim; ++dd)
                o[dd] = acc[dd] / l;
            if (lse_out)
                *lse_out = m + log(l);
        }
        free(scores);
        free(acc);
        free(qv);
        free(path);
    }
    return status;
}

/*
 * Merge of two attention results over disjoint key sets A and B, each given
 * as its normalised output o and its log-sum-exp lse (natural log):
 *   w_A = exp(lse_A), w_B = exp(lse_B)
 *   o   = (w_A o_A + w_B o_B) / (w_A + w_B),   lse = ln(w_A + w_B)
 * evaluated relative to M = max(lse_A, lse_B) so that the exponentials stay
 * finite.  Both sets empty (lse = -inf on both sides) gives o = 0, lse = -inf.
 * o_* are [rows, head_dim], lse_* are [rows].
 */
void parason_oracle_lse_merge(const double *o_a, const double *lse_a,
                              const double *o_b, const double *lse_b,
                              double *o_out, double *lse_out, int64_t rows,
                              int32_t head_dim)
{
    for (int64_t r = 0; r < rows; ++r) {
        const double la = lse_a[r], lb = lse_b[r];
        double *o = o_out + r * head_dim;
        if (la == -INFINITY && lb == -INFINITY) {
            for (int dd = 0; dd < head_dim; ++dd)
                o[dd] = 0.0;
            lse_out[r] = -INFINITY;
            continue;
        }
        const double mx = la > lb ? la : lb;
        const double wa = exp(la - mx), wb = exp(lb - mx);
        for (int dd = 0; dd < head_dim; ++dd)
            o[dd] = (wa * o_a[r * head_dim + dd] + wb * o_b[r * head_dim + dd]) / (wa + wb);
        lse_out[r] = mx + log(wa + wb);
    }
}

/* Number of OpenMP threads a parallel region of the oracle uses. */
int parason_oracle_num_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
