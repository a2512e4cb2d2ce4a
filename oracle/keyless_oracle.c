/*
 * keyless_oracle.c -- plain fp64 CPU oracle for the decode step of Keyless Attention
 * over a paged Value-Only Cache.
 *
 * TEST INFRASTRUCTURE. Only the test suite, the package smoke check and the benchmark's
 * CPU-baseline leg load this library. The CUDA library never calls it, and the two share
 * no source, header, table or helper.
 *
 * What it computes ("Keyless Attention: Value-Space Routing and Value-Only Caching for
 * Efficient Transformers"):
 *   - the routing projection q_r = q W^R of a query row (Eq. 2 and the keyless score of
 *     Eq. 4, Section 2.2; W^R maps query space to value space and is d_k x d_k, Section 2.2);
 *   - the decode step over the Value-Only Cache (Section 3): with the cached rows v_1..v_{n+1},
 *     which include the row of the current token,
 *         O_{n+1} = sum_i alpha_{n+1,i} v_i,
 *         alpha_{n+1,i} = exp(lambda <q_{n+1}, v_i> / sqrt(d_k)) / sum_i' exp(... v_i' ...),
 *     where q_{n+1} is the routed query; the same cached row forms the score and the output;
 *   - the head mapping of Section 3 ("Multi-Head", "Multi-Query", "Grouped Query" paragraphs):
 *     heads that share a value group read the same cached value rows;
 *   - for the comparison only: standard decode softmax(q K^T / sqrt(d_k)) V (Eq. 1) over a
 *     paged K cache and a paged V cache;
 *   - prefill of a chunk of new tokens (Eq. 3 under a causal mask) and the chunk append;
 *   - decode over a latent value-only cache (Section 3, latent value-only cache paragraph);
 *   - the FP8 (E4M3, one fp32 scale per cached row) value cache: encoding, append, decode.
 *
 * Readings taken where the paper is silent:
 *   - lambda / sqrt(d_k) is the caller's `scale`; lambda = 1 gives 1/sqrt(d_k);
 *   - query head h reads value head h / (Hq / Hkv) (contiguous groups);
 *   - W^R holds either Hkv matrices (indexed by value head) or Hq matrices (by query head);
 *   - q_r = q W^R with q a row vector and W^R stored row-major, W^R[k][j] at k*D + j;
 *   - the softmax is evaluated as exp(s_i - max s) / sum exp(s_j - max s): the same number as
 *     the paper's ratio (the factor exp(max s) cancels), without overflow;
 *   - a sequence of length 0 gives a zero output;
 *   - in prefill, query i of a chunk of n new tokens of a sequence of length L (after the
 *     append) sits at position L - n + i and attends tokens 0..L - n + i.
 * Paging follows PagedAttention, which the paper cites for KV-cache management: token t of
 * sequence b is row t % P of physical page block_table[b][t / P]; the cache is laid out as
 * [num_pages][Hkv][P][D].
 *
 * Inputs in bf16 are passed as their 16-bit patterns and widened to double exactly.
 * Every function returns 0, or -1 when a page id, a position or a length is out of range.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* A bf16 value is the upper half of an IEEE binary32 value; widening is exact. */
static double bf16_to_f64(uint16_t bits)
{
    uint32_t u = ((uint32_t)bits) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* Routing projection of one query row: q_r[j] = sum_k q[k] W[k][j] (Section 2.2). */
static void route_row(int D, const uint16_t *q, const uint16_t *W, double *qr)
{
    for (int j = 0; j < D; ++j)
        qr[j] = 0.0;
    for (int k = 0; k < D; ++k) {
        double qk = bf16_to_f64(q[k]);
        for (int j = 0; j < D; ++j)
            qr[j] += qk * bf16_to_f64(W[(size_t)k * D + j]);
    }
}

/* Widen an unrouted query row (the standard-attention comparison). */
static void widen_row(int D, const uint16_t *q, double *out)
{
    for (int j = 0; j < D; ++j)
        out[j] = bf16_to_f64(q[j]);
}

/* Row t of head g of one sequence, or NULL when the page id is outside the pool. */
static const uint16_t *cache_row(const uint16_t *cache, const int32_t *bt_row, int t, int g,
                                 int Hkv, int P, int D, int num_pages)
{
    int page = bt_row[t / P];
    if (page < 0 || page >= num_pages)
        return NULL;
    return cache + (((size_t)page * Hkv + g) * P + (size_t)(t % P)) * D;
}

/*
 * Softmax attention of one query row over tokens [t0, t1) of one sequence and head g.
 * Scores come from `score_cache` (the value cache itself for Keyless Attention, the key
 * cache for the comparison); the output rows come from `value_cache`.
 *   s_t = scale * <qv, score row t>,  m = max_t s_t,  l = sum_t exp(s_t - m),
 *   o = sum_t exp(s_t - m) * value row t / l.
 * An empty range gives m = -inf, l = 0, o = 0. `s` is scratch of at least t1 - t0 doubles.
 */
static int attend(int D, int Hkv, int P, int num_pages, double scale, const double *qv,
                  const uint16_t *score_cache, const uint16_t *value_cache,
                  const int32_t *bt_row, int g, int t0, int t1, double *s,
                  double *o, double *m_out, double *l_out)
{
    for (int j = 0; j < D; ++j)
        o[j] = 0.0;
    *m_out = -INFINITY;
    *l_out = 0.0;
    if (t1 <= t0)
        return 0;

    double m = -INFINITY;
    for (int t = t0; t < t1; ++t) {
        const uint16_t *row = cache_row(score_cache, bt_row, t, g, Hkv, P, D, num_pages);
        if (!row)
            return -1;
        double dot = 0.0;
        for (int j = 0; j < D; ++j)
            dot += qv[j] * bf16_to_f64(row[j]);
        s[t - t0] = scale * dot;
        if (s[t - t0] > m)
            m = s[t - t0];
    }
    double l = 0.0;
    for (int t = t0; t < t1; ++t) {
        double e = exp(s[t - t0] - m);
        s[t - t0] = e;
        l += e;
    }
    for (int t = t0; t < t1; ++t) {
        const uint16_t *row = cache_row(value_cache, bt_row, t, g, Hkv, P, D, num_pages);
        if (!row)
            return -1;
        double w = s[t - t0] / l;
        for (int j = 0; j < D; ++j)
            o[j] += w * bf16_to_f64(row[j]);
    }
    *m_out = m;
    *l_out = l;
    return 0;
}

static int check_dims(int B, int Hq, int Hkv, int D)
{
    if (B < 0 || Hq <= 0 || Hkv <= 0 || D <= 0 || Hq % Hkv != 0)
        return -1;
    return 0;
}

/* q_r[b][h][:] = q[b][h][:] W^R[w(h)] for every head; w(h) = h / G, or h when per query head. */
int ko_route(int B, int Hq, int Hkv, int D, int wr_per_query_head,
             const uint16_t *q, const uint16_t *w_r, double *q_r)
{
    if (check_dims(B, Hq, Hkv, D))
        return -1;
    int G = Hq / Hkv;
    for (int b = 0; b < B; ++b)
        for (int h = 0; h < Hq; ++h) {
            int w = wr_per_query_head ? h : h / G;
            route_row(D, q + ((size_t)b * Hq + h) * D, w_r + (size_t)w * D * D,
                      q_r + ((size_t)b * Hq + h) * D);
        }
    return 0;
}

/*
 * Shared driver of the decode variants. `routed` selects Keyless Attention (scores from the
 * value cache with the routed query) or the standard comparison (scores from `k_cache` with
 * the query as given). With sel == NULL every (b, h) is computed and `out` is [B][Hq][D];
 * otherwise sel holds n_sel pairs (b, h) and `out` is [n_sel][D].
 */
static int decode_impl(int routed, int B, int Hq, int Hkv, int D, int P, int num_pages,
                       int max_pages, int wr_per_query_head, double scale,
                       const uint16_t *q, const uint16_t *w_r, const uint16_t *k_cache,
                       const uint16_t *v_cache, const int32_t *block_table,
                       const int32_t *seq_lens, int n_sel, const int32_t *sel, double *out)
{
    if (check_dims(B, Hq, Hkv, D) || P <= 0 || max_pages < 0)
        return -1;
    int G = Hq / Hkv;
    long n_items = sel ? n_sel : (long)B * Hq;
    int err = 0;

#pragma omp parallel for schedule(dynamic, 1) reduction(| : err)
    for (long it = 0; it < n_items; ++it) {
        int b = sel ? sel[2 * it] : (int)(it / Hq);
        int h = sel ? sel[2 * it + 1] : (int)(it % Hq);
        double *o = out + (size_t)it * D;
        if (b < 0 || b >= B || h < 0 || h >= Hq) {
            err |= 1;
            continue;
        }
        int L = seq_lens[b];
        if (L < 0 || L > max_pages * P) {
            err |= 1;
            continue;
        }
        int g = h / G;
        double *qv = (double *)malloc(sizeof(double) * (size_t)D);
        double *s = (double *)malloc(sizeof(double) * (size_t)(L > 0 ? L : 1));
        const uint16_t *qrow = q + ((size_t)b * Hq + h) * D;
        if (routed) {
            int w = wr_per_query_head ? h : g;
            route_row(D, qrow, w_r + (size_t)w * D * D, qv);
        } else {
            widen_row(D, qrow, qv);
        }
        double m, l;
        const uint16_t *score_cache = routed ? v_cache : k_cache;
        if (attend(D, Hkv, P, num_pages, scale, qv, score_cache, v_cache,
                   block_table + (size_t)b * max_pages, g, 0, L, s, o, &m, &l))
            err |= 1;
        free(s);
        free(qv);
    }
    return err ? -1 : 0;
}

/* Keyless decode (Section 3) for all heads or for the selected (b, h) pairs. */
int ko_decode(int B, int Hq, int Hkv, int D, int P, int num_pages, int max_pages,
              int wr_per_query_head, double scale, const uint16_t *q, const uint16_t *w_r,
              const uint16_t *v_cache, const int32_t *block_table, const int32_t *seq_lens,
              int n_sel, const int32_t *sel, double *out)
{
    return decode_impl(1, B, Hq, Hkv, D, P, num_pages, max_pages, wr_per_query_head, scale,
                       q, w_r, NULL, v_cache, block_table, seq_lens, n_sel, sel, out);
}

/* Standard decode softmax(q K^T * scale) V over paged K and V caches (Eq. 1), comparison only. */
int ko_standard_decode(int B, int Hq, int Hkv, int D, int P, int num_pages, int max_pages,
                       double scale, const uint16_t *q, const uint16_t *k_cache,
                       const uint16_t *v_cache, const int32_t *block_table,
                       const int32_t *seq_lens, int n_sel, const int32_t *sel, double *out)
{
    return decode_impl(0, B, Hq, Hkv, D, P, num_pages, max_pages, 0, scale, q, NULL, k_cache,
                       v_cache, block_table, seq_lens, n_sel, sel, out);
}

/* The attention weights alpha_{n+1,i} of one (b, h) (Section 3), written to alpha[0..L_b). */
int ko_attention_weights(int B, int Hq, int Hkv, int D, int P, int num_pages, int max_pages,
                         int wr_per_query_head, double scale, const uint16_t *q,
                         const uint16_t *w_r, const uint16_t *v_cache,
                         const int32_t *block_table, const int32_t *seq_lens, int b, int h,
                         double *alpha)
{
    if (check_dims(B, Hq, Hkv, D) || b < 0 || b >= B || h < 0 || h >= Hq)
        return -1;
    int G = Hq / Hkv, g = h / G, L = seq_lens[b];
    if (L < 0 || L > max_pages * P)
        return -1;
    double *qr = (double *)malloc(sizeof(double) * (size_t)D);
    int w = wr_per_query_head ? h : g;
    route_row(D, q + ((size_t)b * Hq + h) * D, w_r + (size_t)w * D * D, qr);
    const int32_t *bt_row = block_table + (size_t)b * max_pages;
    int err = 0;
    double m = -INFINITY;
    for (int t = 0; t < L && !err; ++t) {
        const uint16_t *row = cache_row(v_cache, bt_row, t, g, Hkv, P, D, num_pages);
        if (!row) {
            err = 1;
            break;
        }
        double dot = 0.0;
        for (int j = 0; j < D; ++j)
            dot += qr[j] * bf16_to_f64(row[j]);
        alpha[t] = scale * dot;
        if (alpha[t] > m)
            m = alpha[t];
    }
    if (!err) {
        double z = 0.0;
        for (int t = 0; t < L; ++t) {
            alpha[t] = exp(alpha[t] - m);
            z += alpha[t];
        }
        for (int t = 0; t < L; ++t)
            alpha[t] /= z;
    }
    free(qr);
    return err ? -1 : 0;
}

/*
 * Split-sequence partial states: split s of sequence b covers tokens
 * [s * chunk, min((s + 1) * chunk, L_b)). For every (b, h, s):
 *   part_o[b][h][s][:] = normalized output of the split, part_ml[b][h][s] = {m, l}
 * with m the largest score of the split and l = sum exp(s_t - m); an empty split gives
 * {-inf, 0} and a zero output. These are the states that `ko_combine` merges.
 */
int ko_decode_partial(int B, int Hq, int Hkv, int D, int P, int num_pages, int max_pages,
                      int wr_per_query_head, double scale, const uint16_t *q,
                      const uint16_t *w_r, const uint16_t *v_cache,
                      const int32_t *block_table, const int32_t *seq_lens, int chunk, int S,
                      double *part_o, double *part_ml)
{
    if (check_dims(B, Hq, Hkv, D) || chunk <= 0 || S <= 0)
        return -1;
    int G = Hq / Hkv;
    int err = 0;
#pragma omp parallel for schedule(dynamic, 1) reduction(| : err)
    for (long it = 0; it < (long)B * Hq; ++it) {
        int b = (int)(it / Hq), h = (int)(it % Hq), g = h / G;
        int L = seq_lens[b];
        if (L < 0 || L > max_pages * P || (long)S * chunk < L) {
            err |= 1;
            continue;
        }
        double *qr = (double *)malloc(sizeof(double) * (size_t)D);
        double *s = (double *)malloc(sizeof(double) * (size_t)chunk);
        int w = wr_per_query_head ? h : g;
        route_row(D, q + ((size_t)b * Hq + h) * D, w_r + (size_t)w * D * D, qr);
        for (int sp = 0; sp < S; ++sp) {
            int t0 = sp * chunk, t1 = (sp + 1) * chunk;
            if (t1 > L)
                t1 = L;
            size_t slot = ((size_t)it * S + sp);
            if (attend(D, Hkv, P, num_pages, scale, qr, v_cache, v_cache,
                       block_table + (size_t)b * max_pages, g, t0, t1, s,
                       part_o + slot * D, &part_ml[2 * slot], &part_ml[2 * slot + 1]))
                err |= 1;
        }
        free(s);
        free(qr);
    }
    return err ? -1 : 0;
}

/*
 * Merge of split states into one softmax over the union of the splits:
 *   M = max over non-empty splits of m_s,  w_s = l_s exp(m_s - M),
 *   out = sum_s w_s o_s / sum_s w_s.
 * This equals one softmax over all tokens because each split's normalized output times its
 * l_s exp(m_s - M) is its share of the unnormalized sum sum_t exp(s_t - M) v_t. All splits
 * empty gives a zero output.
 */
int ko_combine(int B, int Hq, int D, int S, const double *part_o, const double *part_ml,
               double *out)
{
    if (B < 0 || Hq <= 0 || D <= 0 || S <= 0)
        return -1;
    for (long it = 0; it < (long)B * Hq; ++it) {
        const double *ml = part_ml + (size_t)it * S * 2;
        const double *po = part_o + (size_t)it * S * D;
        double *o = out + (size_t)it * D;
        double M = -INFINITY;
        for (int s = 0; s < S; ++s)
            if (ml[2 * s + 1] > 0.0 && ml[2 * s] > M)
                M = ml[2 * s];
        for (int j = 0; j < D; ++j)
            o[j] = 0.0;
        if (M == -INFINITY)
            continue;
        double z = 0.0;
        for (int s = 0; s < S; ++s) {
            if (!(ml[2 * s + 1] > 0.0))
                continue;
            double w = ml[2 * s + 1] * exp(ml[2 * s] - M);
            z += w;
            for (int j = 0; j < D; ++j)
                o[j] += w * po[(size_t)s * D + j];
        }
        for (int j = 0; j < D; ++j)
            o[j] /= z;
    }
    return 0;
}

/*
 * Append of the current token's value rows to the Value-Only Cache (Section 3: the cache
 * holds the rows of the previous steps and the row obtained at the current step):
 *   cache[block_table[b][pos_b / P]][g][pos_b % P][:] = v_new[b][g][:]  for every g.
 * Bit copies; a position or page id out of range leaves the cache untouched and returns -1.
 */
int ko_append(int B, int Hkv, int D, int P, int num_pages, int max_pages,
              const uint16_t *v_new, const int32_t *block_table, const int32_t *positions,
              uint16_t *v_cache)
{
    int err = 0;
    for (int b = 0; b < B; ++b) {
        int pos = positions[b];
        if (pos < 0 || pos >= max_pages * P) {
            err = 1;
            continue;
        }
        int page = block_table[(size_t)b * max_pages + pos / P];
        if (page < 0 || page >= num_pages) {
            err = 1;
            continue;
        }
        for (int g = 0; g < Hkv; ++g)
            memcpy(v_cache + (((size_t)page * Hkv + g) * P + (size_t)(pos % P)) * D,
                   v_new + ((size_t)b * Hkv + g) * D, sizeof(uint16_t) * (size_t)D);
    }
    return err ? -1 : 0;
}

/*
 * Keyless prefill over the Value-Only Cache: the full attention of Eq. 3 for the rows of a
 * chunk of new tokens, under the causal mask of an autoregressive model (Section 5 builds it
 * on the fly; a token attends itself and the tokens before it).
 * Sequence b holds L_b = seq_lens[b] cached rows. Its last n_b = cu_q[b + 1] - cu_q[b] rows are
 * the chunk, already appended; query row r = cu_q[b] + i (0 <= i < n_b) sits at position
 * p = L_b - n_b + i and, for query head h,
 *     q_r = q[r][h] W^R[w(h)],  s_t = scale * <q_r, v_t>  (t = 0..p),  out = sum_t alpha_t v_t.
 * q and out are [T][Hq][D] with T = cu_q[B]; with sel != NULL only the n_sel pairs (r, h) are
 * computed and out is [n_sel][D].
 */
int ko_prefill(int B, int Hq, int Hkv, int D, int P, int num_pages, int max_pages,
               int wr_per_query_head, double scale, const uint16_t *q, const uint16_t *w_r,
               const uint16_t *v_cache, const int32_t *block_table, const int32_t *seq_lens,
               const int32_t *cu_q, int n_sel, const int32_t *sel, double *out)
{
    if (check_dims(B, Hq, Hkv, D) || P <= 0 || max_pages < 0 || cu_q[0] != 0)
        return -1;
    for (int b = 0; b < B; ++b) {
        int n = cu_q[b + 1] - cu_q[b];
        if (n < 0 || n > seq_lens[b] || seq_lens[b] > max_pages * P)
            return -1;
    }
    int G = Hq / Hkv, T = cu_q[B];
    long n_items = sel ? n_sel : (long)T * Hq;
    int err = 0;

#pragma omp parallel for schedule(dynamic, 1) reduction(| : err)
    for (long it = 0; it < n_items; ++it) {
        int r = sel ? sel[2 * it] : (int)(it / Hq);
        int h = sel ? sel[2 * it + 1] : (int)(it % Hq);
        double *o = out + (size_t)it * D;
        if (r < 0 || r >= T || h < 0 || h >= Hq) {
            err |= 1;
            continue;
        }
        int b = 0;
        while (cu_q[b + 1] <= r)
            ++b;
        int n = cu_q[b + 1] - cu_q[b];
        int p = seq_lens[b] - n + (r - cu_q[b]);
        int g = h / G, w = wr_per_query_head ? h : g;
        double *qr = (double *)malloc(sizeof(double) * (size_t)D);
        double *s = (double *)malloc(sizeof(double) * (size_t)(p + 1));
        route_row(D, q + ((size_t)r * Hq + h) * D, w_r + (size_t)w * D * D, qr);
        double m, l;
        if (attend(D, Hkv, P, num_pages, scale, qr, v_cache, v_cache,
                   block_table + (size_t)b * max_pages, g, 0, p + 1, s, o, &m, &l))
            err |= 1;
        free(s);
        free(qr);
    }
    return err ? -1 : 0;
}

/*
 * Append of a chunk: the n_b = cu_q[b + 1] - cu_q[b] value rows of sequence b go to positions
 * L_b - n_b .. L_b - 1 (L_b = seq_lens[b], the length after the append):
 *   cache[block_table[b][p / P]][g][p % P][:] = v_new[cu_q[b] + i][g][:],  p = L_b - n_b + i.
 * v_new is [T][Hkv][D]. Rows whose position or page id is out of range are skipped; -1 then.
 */
int ko_append_chunk(int B, int Hkv, int D, int P, int num_pages, int max_pages,
                    const uint16_t *v_new, const int32_t *block_table, const int32_t *seq_lens,
                    const int32_t *cu_q, uint16_t *v_cache)
{
    int err = 0;
    for (int b = 0; b < B; ++b) {
        int n = cu_q[b + 1] - cu_q[b];
        for (int i = 0; i < n; ++i) {
            int pos = seq_lens[b] - n + i;
            if (pos < 0 || pos >= max_pages * P) {
                err = 1;
                continue;
            }
            int page = block_table[(size_t)b * max_pages + pos / P];
            if (page < 0 || page >= num_pages) {
                err = 1;
                continue;
            }
            for (int g = 0; g < Hkv; ++g)
                memcpy(v_cache + (((size_t)page * Hkv + g) * P + (size_t)(pos % P)) * D,
                       v_new + ((size_t)(cu_q[b] + i) * Hkv + g) * D,
                       sizeof(uint16_t) * (size_t)D);
        }
    }
    return err ? -1 : 0;
}

/*
 * Multi-head attention over a latent value-only cache (Section 3, "Multihead with Latent
 * Value-only Cache"): the cache holds V* = X W^V_pre (width r) and head h expands it with
 * W^V_{h,post} (r x d_k). For query head h of latent group g = h / (Hq / Hl):
 *   q_r = q W^R[w(h)]                                (Section 2.2)
 *   q*[k] = sum_j q_r[j] W_post[h][k][j]              (absorbed query Q* = Q (W_post)^T)
 *   s_t = scale * <q*, v*_t>,  alpha = softmax(s),  o*[k] = sum_t alpha_t v*_t[k]
 *   out[j] = sum_k o*[k] W_post[h][k][j]              (output V* W_post)
 * with scale = 1 / sqrt(r) in the paper (the caller's `scale`). W_post is [Hq][r][D] row-major
 * (row k = latent dimension); the latent cache is [num_pages][Hl][P][r]; out is [B][Hq][D], or
 * [n_sel][D] for the selected (b, h) pairs.
 */
int ko_latent_decode(int B, int Hq, int Hl, int D, int r, int P, int num_pages, int max_pages,
                     int wr_per_query_head, double scale, const uint16_t *q, const uint16_t *w_r,
                     const uint16_t *w_post, const uint16_t *v_lat, const int32_t *block_table,
                     const int32_t *seq_lens, int n_sel, const int32_t *sel, double *out)
{
    if (check_dims(B, Hq, Hl, D) || r <= 0 || P <= 0 || max_pages < 0)
        return -1;
    int G = Hq / Hl;
    long n_items = sel ? n_sel : (long)B * Hq;
    int err = 0;

#pragma omp parallel for schedule(dynamic, 1) reduction(| : err)
    for (long it = 0; it < n_items; ++it) {
        int b = sel ? sel[2 * it] : (int)(it / Hq);
        int h = sel ? sel[2 * it + 1] : (int)(it % Hq);
        double *o = out + (size_t)it * D;
        if (b < 0 || b >= B || h < 0 || h >= Hq) {
            err |= 1;
            continue;
        }
        int L = seq_lens[b];
        if (L < 0 || L > max_pages * P) {
            err |= 1;
            continue;
        }
        int g = h / G, w = wr_per_query_head ? h : g;
        const uint16_t *Wp = w_post + (size_t)h * r * D;
        double *qr = (double *)malloc(sizeof(double) * (size_t)D);
        double *qs = (double *)malloc(sizeof(double) * (size_t)r);
        double *os = (double *)malloc(sizeof(double) * (size_t)r);
        double *s = (double *)malloc(sizeof(double) * (size_t)(L > 0 ? L : 1));
        route_row(D, q + ((size_t)b * Hq + h) * D, w_r + (size_t)w * D * D, qr);
        for (int k = 0; k < r; ++k) {
            double acc = 0.0;
            for (int j = 0; j < D; ++j)
                acc += qr[j] * bf16_to_f64(Wp[(size_t)k * D + j]);
            qs[k] = acc;
        }
        double m, l;
        if (attend(r, Hl, P, num_pages, scale, qs, v_lat, v_lat,
                   block_table + (size_t)b * max_pages, g, 0, L, s, os, &m, &l))
            err |= 1;
        for (int j = 0; j < D; ++j) {
            double acc = 0.0;
            for (int k = 0; k < r; ++k)
                acc += os[k] * bf16_to_f64(Wp[(size_t)k * D + j]);
            o[j] = acc;
        }
        free(s);
        free(os);
        free(qs);
        free(qr);
    }
    return err ? -1 : 0;
}

/*
 * FP8 value cache. Section 3 states that the value-only cache is orthogonal to other
 * KV-cache reduction methods, so it composes with a quantized cache; the paper fixes no format,
 * and this one is the reading taken. Values are stored as OCP FP8 E4M3 codes (1 sign bit, 4 exponent bits
 * with bias 7, 3 mantissa bits; exponent field 0 encodes subnormals m/8 * 2^-6; the all-ones
 * exponent with all-ones mantissa is NaN; no infinities; largest finite value 448) with one
 * fp32 scale per cached row: v = scale * value(code).
 */
static double e4m3_value(uint8_t c)
{
    int sign = c >> 7, e = (c >> 3) & 15, m = c & 7;
    double v;
    if (e == 15 && m == 7)
        return NAN;
    if (e == 0)
        v = (double)m / 8.0 * ldexp(1.0, -6);
    else
        v = (1.0 + (double)m / 8.0) * ldexp(1.0, e - 7);
    return sign ? -v : v;
}

/* Nearest E4M3 code of x, ties to the code with an even mantissa, magnitudes above 448 clamped
 * to 448 (saturating conversion). The grid values are exact in double, so the comparisons are
 * exact. */
uint8_t ko_e4m3_from_f32(float x)
{
    uint8_t sign = (x < 0.0f || (x == 0.0f && signbit(x))) ? 0x80 : 0;
    double a = fabs((double)x);
    if (a >= 448.0)
        return sign | 0x7E;
    int lo = 0;                       /* largest code with value <= a (codes 0..126 ascend) */
    for (int c = 1; c <= 126; ++c)
        if (e4m3_value((uint8_t)c) <= a)
            lo = c;
    if (lo == 126)
        return sign | 126;
    double vl = e4m3_value((uint8_t)lo), vh = e4m3_value((uint8_t)(lo + 1));
    int pick;
    if (a - vl < vh - a)
        pick = lo;
    else if (a - vl > vh - a)
        pick = lo + 1;
    else
        pick = (lo & 1) ? lo + 1 : lo;    /* tie: even mantissa */
    return sign | (uint8_t)pick;
}

double ko_e4m3_value(uint8_t c) { return e4m3_value(c); }

/* Quantize one row of D bf16 values: scale = max |v| / 448 (fp32), code_j = e4m3(v_j / scale)
 * with the division in fp32; an all-zero row gets scale 0 and zero codes. */
static void quantize_row(int D, const uint16_t *v, uint8_t *codes, float *scale)
{
    float amax = 0.0f;
    for (int j = 0; j < D; ++j) {
        uint32_t u = ((uint32_t)v[j]) << 16;
        float f;
        memcpy(&f, &u, sizeof f);
        if (fabsf(f) > amax)
            amax = fabsf(f);
    }
    float s = amax / 448.0f;
    *scale = s;
    for (int j = 0; j < D; ++j) {
        uint32_t u = ((uint32_t)v[j]) << 16;
        float f;
        memcpy(&f, &u, sizeof f);
        codes[j] = s > 0.0f ? ko_e4m3_from_f32(f / s) : 0;
    }
}

int ko_quantize_rows(int n, int D, const uint16_t *v, uint8_t *codes, float *scales)
{
    for (int i = 0; i < n; ++i)
        quantize_row(D, v + (size_t)i * D, codes + (size_t)i * D, scales + i);
    return 0;
}

/* Append to the FP8 cache: row pos_b of sequence b, every value head, quantized as above.
 * Codes are [num_pages][Hkv][P][D], scales [num_pages][Hkv][P]. */
int ko_append_fp8(int B, int Hkv, int D, int P, int num_pages, int max_pages,
                  const uint16_t *v_new, const int32_t *block_table, const int32_t *positions,
                  uint8_t *codes, float *scales)
{
    int err = 0;
    for (int b = 0; b < B; ++b) {
        int pos = positions[b];
        if (pos < 0 || pos >= max_pages * P) {
            err = 1;
            continue;
        }
        int page = block_table[(size_t)b * max_pages + pos / P];
        if (page < 0 || page >= num_pages) {
            err = 1;
            continue;
        }
        for (int g = 0; g < Hkv; ++g) {
            size_t row = ((size_t)page * Hkv + g) * P + (size_t)(pos % P);
            quantize_row(D, v_new + ((size_t)b * Hkv + g) * D, codes + row * D, scales + row);
        }
    }
    return err ? -1 : 0;
}

/*
 * Keyless decode (Section 3) over the FP8 cache: every cached value is scale * value(code),
 * widened exactly to double; otherwise as ko_decode (routing, GQA mapping, softmax, output).
 */
int ko_decode_fp8(int B, int Hq, int Hkv, int D, int P, int num_pages, int max_pages,
                  int wr_per_query_head, double scale, const uint16_t *q, const uint16_t *w_r,
                  const uint8_t *codes, const float *scales, const int32_t *block_table,
                  const int32_t *seq_lens, int n_sel, const int32_t *sel, double *out)
{
    if (check_dims(B, Hq, Hkv, D) || P <= 0 || max_pages < 0)
        return -1;
    int G = Hq / Hkv;
    long n_items = sel ? n_sel : (long)B * Hq;
    int err = 0;

#pragma omp parallel for schedule(dynamic, 1) reduction(| : err)
    for (long it = 0; it < n_items; ++it) {
        int b = sel ? sel[2 * it] : (int)(it / Hq);
        int h = sel ? sel[2 * it + 1] : (int)(it % Hq);
        double *o = out + (size_t)it * D;
        for (int j = 0; j < D; ++j)
            o[j] = 0.0;
        if (b < 0 || b >= B || h < 0 || h >= Hq) {
            err |= 1;
            continue;
        }
        int L = seq_lens[b];
        if (L < 0 || L > max_pages * P) {
            err |= 1;
            continue;
        }
        if (L == 0)
            continue;
        int g = h / G, w = wr_per_query_head ? h : g;
        const int32_t *bt_row = block_table + (size_t)b * max_pages;
        double *qr = (double *)malloc(sizeof(double) * (size_t)D);
        double *rows = (double *)malloc(sizeof(double) * (size_t)L * D);
        double *s = (double *)malloc(sizeof(double) * (size_t)L);
        route_row(D, q + ((size_t)b * Hq + h) * D, w_r + (size_t)w * D * D, qr);
        int bad = 0;
        for (int t = 0; t < L && !bad; ++t) {
            int page = bt_row[t / P];
            if (page < 0 || page >= num_pages) {
                bad = 1;
                break;
            }
            size_t row = ((size_t)page * Hkv + g) * P + (size_t)(t % P);
            for (int j = 0; j < D; ++j)
                rows[(size_t)t * D + j] = (double)scales[row] * e4m3_value(codes[row * D + j]);
        }
        if (!bad) {
            double m = -INFINITY;
            for (int t = 0; t < L; ++t) {
                double dot = 0.0;
                for (int j = 0; j < D; ++j)
                    dot += qr[j] * rows[(size_t)t * D + j];
                s[t] = scale * dot;
                if (s[t] > m)
                    m = s[t];
            }
            double l = 0.0;
            for (int t = 0; t < L; ++t) {
                s[t] = exp(s[t] - m);
                l += s[t];
            }
            for (int t = 0; t < L; ++t)
                for (int j = 0; j < D; ++j)
                    o[j] += s[t] / l * rows[(size_t)t * D + j];
        } else {
            err |= 1;
        }
        free(s);
        free(rows);
        free(qr);
    }
    return err ? -1 : 0;
}
