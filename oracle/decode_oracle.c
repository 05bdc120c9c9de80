/*
 * Float64 CPU oracle for paged single-token decode attention and for the
 * paged KV scatter/gather that kv_append and the prefix write perform.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may include, link or
 * call this file: only tests/, __graft_entry__.smoke() and the cpu_baseline
 * leg of bench.py use it.  It shares no code, header, table or helper with the
 * CUDA library; the two meet only through the seeded inputs that the
 * workload generator draws.
 *
 * What it computes (the definition, written out plainly, no blocking, no
 * fusion, no online softmax, no split):
 *
 *   Language decoding streams the KV cache from HBM (HeteroServe, Sec. 2 and
 *   Sec. 5.1); the cache of one request holds s_ctx = N_v + s_text tokens per
 *   layer and KV head (Sec. 4.1, Eq. 1).  One decode step of one layer, for
 *   sequence b, query head h and KV head g = h / G (G = H_q / H_kv, the
 *   contiguous grouping that MHA (G = 1) and GQA (Sec. 5.1 "MHA and GQA
 *   backends", Sec. 6.1 model list) share):
 *
 *       s_t = (q_{b,h} . k_{b,g,t}) * scale             t = 0 .. n_b - 1
 *       w_t = exp(s_t - max_u s_u) / sum_u exp(s_u - max_u s_u)
 *       o_{b,h} = sum_t w_t v_{b,g,t}
 *
 *   over the logical token order (vision prefix first, then text, then the
 *   generated tokens, the newest last).  Inputs are bf16 bit patterns; every
 *   value is widened exactly to float64 by this file's own bf16 decoder and
 *   all arithmetic is float64.
 *
 *   Paged layout (the oracle's own reading of a page table): logical token t
 *   of a sequence lives in physical page page_table_row[t / P], slot t % P;
 *   a pool is laid out [num_pages][H_kv][P][d].
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* bf16 is the upper half of an IEEE-754 binary32: sign, 8 exponent bits,
 * 7 fraction bits.  Widening is exact: shift into the high half, reinterpret,
 * convert to double. */
static double bf16_bits_to_double(uint16_t bits)
{
    uint32_t w = ((uint32_t)bits) << 16;
    float f;
    memcpy(&f, &w, sizeof f);
    return (double)f;
}

void oracle_bf16_to_f64(const uint16_t *in, double *out, int64_t n)
{
    for (int64_t i = 0; i < n; ++i)
        out[i] = bf16_bits_to_double(in[i]);
}

/* Attention of one query vector over n logical tokens.  k and v point at
 * token 0 of this KV head; consecutive tokens are token_stride elements
 * apart.  Writes d outputs and returns sum_t w_t (which must be 1). */
static double attend_one_head(const uint16_t *q, const uint16_t *k,
                              const uint16_t *v, int64_t n,
                              int64_t token_stride, int32_t d, double scale,
                              double *out, double *scores)
{
    for (int64_t t = 0; t < n; ++t) {
        double dot = 0.0;
        for (int32_t i = 0; i < d; ++i)
            dot += bf16_bits_to_double(q[i]) *
                   bf16_bits_to_double(k[t * token_stride + i]);
        scores[t] = dot * scale;
    }
    double mx = -INFINITY;
    for (int64_t t = 0; t < n; ++t)
        if (scores[t] > mx) mx = scores[t];
    double z = 0.0;
    for (int64_t t = 0; t < n; ++t) {
        scores[t] = exp(scores[t] - mx);
        z += scores[t];
    }
    double wsum = 0.0;
    for (int32_t i = 0; i < d; ++i) out[i] = 0.0;
    for (int64_t t = 0; t < n; ++t) {
        double w = scores[t] / z;
        wsum += w;
        for (int32_t i = 0; i < d; ++i)
            out[i] += w * bf16_bits_to_double(v[t * token_stride + i]);
    }
    return wsum;
}

/*
 * Logical-order decode attention.
 *   q        [B][H_q][d]                 bf16 bits
 *   kv_off   [B + 1]                     token offsets into k / v
 *   k, v     [kv_off[B]][H_kv][d]        bf16 bits, logical token order
 *   out      [B][H_q][d]                 float64
 *   wsum     [B][H_q] or NULL            sum of softmax weights per head
 * Returns 0, or -1 on a shape error (H_q not a multiple of H_kv, an empty
 * sequence, a negative size).
 */
int oracle_decode_attention(int32_t B, int32_t H_q, int32_t H_kv, int32_t d,
                            const uint16_t *q, const int64_t *kv_off,
                            const uint16_t *k, const uint16_t *v,
                            double scale, double *out, double *wsum)
{
    if (B < 0 || H_q <= 0 || H_kv <= 0 || d <= 0 || H_q % H_kv != 0)
        return -1;
    for (int32_t b = 0; b < B; ++b)
        if (kv_off[b + 1] - kv_off[b] <= 0) return -1;
    const int32_t G = H_q / H_kv;
    int err = 0;
#pragma omp parallel for schedule(dynamic, 1) reduction(| : err)
    for (int64_t bh = 0; bh < (int64_t)B * H_q; ++bh) {
        const int32_t b = (int32_t)(bh / H_q), h = (int32_t)(bh % H_q);
        const int32_t g = h / G;
        const int64_t n = kv_off[b + 1] - kv_off[b];
        double *scores = (double *)malloc((size_t)n * sizeof(double));
        if (!scores) { err |= 1; continue; }
        const int64_t base = (kv_off[b] * H_kv + g) * d;
        double ws = attend_one_head(q + ((int64_t)b * H_q + h) * d, k + base,
                                    v + base, n, (int64_t)H_kv * d, d, scale,
                                    out + ((int64_t)b * H_q + h) * d, scores);
        if (wsum) wsum[bh] = ws;
        free(scores);
    }
    return err ? -1 : 0;
}

/* Copy logical tokens [first, first + n) of one sequence out of a paged pool
 * into dst[n][H_kv][d].  Returns -1 if a page id is outside the pool. */
int oracle_kv_gather(const uint16_t *pool, int64_t num_pages, int32_t H_kv,
                     int32_t P, int32_t d, const int32_t *page_table_row,
                     int64_t first, int64_t n, uint16_t *dst)
{
    for (int64_t i = 0; i < n; ++i) {
        const int64_t t = first + i;
        const int64_t page = page_table_row[t / P];
        const int64_t slot = t % P;
        if (page < 0 || page >= num_pages) return -1;
        for (int32_t g = 0; g < H_kv; ++g)
            memcpy(dst + (i * H_kv + g) * d,
                   pool + ((page * H_kv + g) * P + slot) * d,
                   (size_t)d * sizeof(uint16_t));
    }
    return 0;
}

/* Write tokens src[n][H_kv][d] into logical positions [first, first + n) of
 * one sequence of a paged pool (what kv_append does for n = 1 at position
 * s_b, and what the prefix write does for the N_v vision tokens plus the
 * prompt).  Returns -1 if a page id is outside the pool. */
int oracle_kv_scatter(uint16_t *pool, int64_t num_pages, int32_t H_kv,
                      int32_t P, int32_t d, const int32_t *page_table_row,
                      int64_t first, int64_t n, const uint16_t *src)
{
    for (int64_t i = 0; i < n; ++i) {
        const int64_t t = first + i;
        const int64_t page = page_table_row[t / P];
        const int64_t slot = t % P;
        if (page < 0 || page >= num_pages) return -1;
        for (int32_t g = 0; g < H_kv; ++g)
            memcpy(pool + ((page * H_kv + g) * P + slot) * d,
                   src + (i * H_kv + g) * d, (size_t)d * sizeof(uint16_t));
    }
    return 0;
}

/*
 * Paged decode attention: gather each sequence's tokens through its own page
 * table row into logical order, then apply the definition above.
 *   q            [B][H_q][d]
 *   lens         [B]            tokens attended per sequence (n_b >= 1)
 *   page_table   [B][max_pages] physical page of each logical page
 *   k_pool/v_pool[num_pages][H_kv][P][d]
 */
int oracle_decode_attention_paged(int32_t B, int32_t H_q, int32_t H_kv,
                                  int32_t d, int32_t P, const uint16_t *q,
                                  const int32_t *lens,
                                  const int32_t *page_table, int32_t max_pages,
                                  const uint16_t *k_pool,
                                  const uint16_t *v_pool, int64_t num_pages,
                                  double scale, double *out)
{
    if (B < 0 || P <= 0 || max_pages <= 0) return -1;
    int64_t total = 0;
    int64_t *off = (int64_t *)malloc((size_t)(B + 1) * sizeof(int64_t));
    if (!off) return -1;
    off[0] = 0;
    for (int32_t b = 0; b < B; ++b) {
        if (lens[b] <= 0 || (lens[b] + P - 1) / P > max_pages) {
            free(off);
            return -1;
        }
        total += lens[b];
        off[b + 1] = total;
    }
    const size_t row = (size_t)H_kv * d;
    uint16_t *k = (uint16_t *)malloc((size_t)total * row * sizeof(uint16_t));
    uint16_t *v = (uint16_t *)malloc((size_t)total * row * sizeof(uint16_t));
    int rc = (k && v) ? 0 : -1;
    for (int32_t b = 0; b < B && rc == 0; ++b) {
        const int32_t *pt = page_table + (int64_t)b * max_pages;
        rc |= oracle_kv_gather(k_pool, num_pages, H_kv, P, d, pt, 0, lens[b],
                               k + off[b] * row);
        rc |= oracle_kv_gather(v_pool, num_pages, H_kv, P, d, pt, 0, lens[b],
                               v + off[b] * row);
    }
    if (rc == 0)
        rc = oracle_decode_attention(B, H_q, H_kv, d, q, off, k, v, scale, out,
                                     NULL);
    free(k);
    free(v);
    free(off);
    return rc;
}
