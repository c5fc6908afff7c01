/*
 * CPU oracle for the three-stage attention hot path -- TEST INFRASTRUCTURE ONLY.
 *
 * Only tests/, the smoke check and the bench's CPU-baseline leg may load this
 * library.  The CUDA path never calls it and shares no code with it.
 *
 * What it computes (arxiv 2607.15865, Section 4; Listings 1-2; Table 1):
 *   every stage applies RoPE to q and k with cos/sin values gathered from a table
 *   precomputed per position (Section 4.6.2), appends the new k/v to a static
 *   maximum-length cache in place (Listing 2 "Concat"; Section 4.6.3), and runs
 *   causal scaled dot-product attention (FAttention, Section 2.2) of every new
 *   query over the history plus the new tokens (prefill: no history; prefill_kv:
 *   Section 4.3; decode: one token per sequence over a length-masked cache,
 *   Section 4.4).  Grouped-query attention: query head h reads kv head
 *   h / (Hq/Hkv).
 *
 * Readings where the paper is silent (kept identical in every caller):
 *   - RoPE pairs element j with element j + D/2 ("rotate half"), inverse
 *     frequency theta^(-2j/D); the table entry is cos/sin of p*theta^(-2j/D)
 *     evaluated in double and rounded to float.
 *   - RoPE arithmetic is float: each product and the difference/sum rounded to
 *     float, no fused multiply-add (build with -ffp-contract=off).
 *   - Rotated q and k are rounded to bf16 (round to nearest even); the cache is
 *     bf16 and holds the rotated k and the unchanged v.
 *   - Scores, softmax and the weighted sum of v are evaluated in double, with
 *     the scale 1/sqrt(D) and the row maximum subtracted; the result is rounded
 *     to float and then to bf16.
 *   - Decode: hist_len[b] valid history tokens; the new token is written to slot
 *     hist_len[b] and attends to slots [0, hist_len[b]].
 *   - Rows i >= chunk of a static chunk buffer are neither computed nor written.
 *
 * Layouts (bf16 bit patterns): q [B,S,Hq,D]; k, v [B,S,Hkv,D];
 * caches [B,Hkv,L,D]; out [B,S,Hq,D]; hist [B] int32.
 * Return value: 0 on success, -1 on an invalid argument (nothing written).
 */
#include <math.h>
#include <stddef.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

typedef struct {
    int batch, n_q_heads, n_kv_heads, head_dim, max_len;
    double rope_theta;
} oracle_cfg;

static float bf16_to_float(uint16_t b) {
    uint32_t u = (uint32_t)b << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return f;
}

static uint16_t float_to_bf16(float f) {
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    if ((u & 0x7fffffffu) > 0x7f800000u) return (uint16_t)((u >> 16) | 0x40u); /* quiet NaN */
    u += 0x7fffu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

static int cfg_ok(const oracle_cfg* c) {
    return c && c->batch > 0 && c->n_q_heads > 0 && c->n_kv_heads > 0 &&
           c->n_q_heads % c->n_kv_heads == 0 && c->head_dim > 0 && c->head_dim % 2 == 0 &&
           c->max_len > 0 && c->rope_theta > 0.0;
}

/* Section 4.6.2: cos/sin of every position 0..max_len-1, D/2 frequencies each. */
int oracle_rope_tables(int max_len, int head_dim, double theta, float* cos_tab, float* sin_tab) {
    if (max_len <= 0 || head_dim <= 0 || head_dim % 2 || theta <= 0.0 || !cos_tab || !sin_tab) return -1;
    int half = head_dim / 2;
    for (int p = 0; p < max_len; ++p) {
        for (int j = 0; j < half; ++j) {
            double inv_freq = pow(theta, -(2.0 * j) / (double)head_dim);
            double angle = (double)p * inv_freq;
            cos_tab[(size_t)p * half + j] = (float)cos(angle);
            sin_tab[(size_t)p * half + j] = (float)sin(angle);
        }
    }
    return 0;
}

/* Listing 1 "Rope": rotate one head vector with the gathered table row of its position. */
void oracle_rope_row(int head_dim, const float* cos_row, const float* sin_row, const uint16_t* x,
                     float* y) {
    int half = head_dim / 2;
    for (int j = 0; j < half; ++j) {
        float a = bf16_to_float(x[j]);
        float b = bf16_to_float(x[j + half]);
        float c = cos_row[j], s = sin_row[j];
        float ac = a * c, bs = b * s, bc = b * c, as = a * s;
        y[j] = ac - bs;
        y[j + half] = bc + as;
    }
}

typedef struct {
    float* cos_tab;
    float* sin_tab;
} tables;

static int make_tables(const oracle_cfg* c, tables* t) {
    size_t n = (size_t)c->max_len * (size_t)(c->head_dim / 2);
    t->cos_tab = (float*)malloc(n * sizeof(float));
    t->sin_tab = (float*)malloc(n * sizeof(float));
    if (!t->cos_tab || !t->sin_tab) {
        free(t->cos_tab);
        free(t->sin_tab);
        return -1;
    }
    return oracle_rope_tables(c->max_len, c->head_dim, c->rope_theta, t->cos_tab, t->sin_tab);
}

static void free_tables(tables* t) {
    free(t->cos_tab);
    free(t->sin_tab);
}

static int hist_ok(const oracle_cfg* c, const int32_t* hist, int chunk) {
    if (!hist || chunk <= 0) return 0;
    for (int b = 0; b < c->batch; ++b)
        if (hist[b] < 0 || (long)hist[b] + chunk > c->max_len) return 0;
    return 1;
}

/*
 * In-place cache append (Listing 2 "Concat"; Section 4.6.3): for every sequence b
 * and new token i < chunk at position p = hist[b] + i, slot p of kv head g gets
 * bf16(rope(k)) and v unchanged.  No other slot is touched.
 */
int oracle_append(const oracle_cfg* c, const uint16_t* k, const uint16_t* v, const int32_t* hist,
                  int chunk, int chunk_stride, uint16_t* k_cache, uint16_t* v_cache) {
    if (!cfg_ok(c) || !k || !v || !k_cache || !v_cache || chunk_stride < chunk || !hist_ok(c, hist, chunk))
        return -1;
    tables t;
    if (make_tables(c, &t)) return -1;
    int D = c->head_dim, Hkv = c->n_kv_heads, L = c->max_len, half = D / 2;
    float* y = (float*)malloc(sizeof(float) * D);
    for (int b = 0; b < c->batch; ++b) {
        for (int i = 0; i < chunk; ++i) {
            int p = hist[b] + i;
            for (int g = 0; g < Hkv; ++g) {
                size_t src = (((size_t)b * chunk_stride + i) * Hkv + g) * D;
                size_t dst = (((size_t)b * Hkv + g) * L + p) * D;
                oracle_rope_row(D, t.cos_tab + (size_t)p * half, t.sin_tab + (size_t)p * half, k + src, y);
                for (int d = 0; d < D; ++d) {
                    k_cache[dst + d] = float_to_bf16(y[d]);
                    v_cache[dst + d] = v[src + d];
                }
            }
        }
    }
    free(y);
    free_tables(&t);
    return 0;
}

/*
 * One output row (FAttention, Section 2.2, with the causal mask of Section 4.6.1):
 * the rotated query at position p of head h attends to slots [0, p] of kv head
 * h / G of its sequence.
 */
static void attend_row(const oracle_cfg* c, const tables* t, const uint16_t* q_row, int b, int h, int p,
                       const uint16_t* k_cache, const uint16_t* v_cache, uint16_t* out_row, float* qr,
                       double* sc, double* acc) {
    int D = c->head_dim, L = c->max_len, half = D / 2;
    int g = h / (c->n_q_heads / c->n_kv_heads);
    oracle_rope_row(D, t->cos_tab + (size_t)p * half, t->sin_tab + (size_t)p * half, q_row, qr);
    for (int d = 0; d < D; ++d) qr[d] = bf16_to_float(float_to_bf16(qr[d]));
    const uint16_t* kb = k_cache + ((size_t)b * c->n_kv_heads + g) * (size_t)L * D;
    const uint16_t* vb = v_cache + ((size_t)b * c->n_kv_heads + g) * (size_t)L * D;
    double scale = 1.0 / sqrt((double)D);
    double m = -INFINITY;
    for (int j = 0; j <= p; ++j) {
        double s = 0.0;
        for (int d = 0; d < D; ++d) s += (double)qr[d] * (double)bf16_to_float(kb[(size_t)j * D + d]);
        s *= scale;
        sc[j] = s;
        if (s > m) m = s;
    }
    double l = 0.0;
    for (int d = 0; d < D; ++d) acc[d] = 0.0;
    for (int j = 0; j <= p; ++j) {
        double w = exp(sc[j] - m);
        l += w;
        for (int d = 0; d < D; ++d) acc[d] += w * (double)bf16_to_float(vb[(size_t)j * D + d]);
    }
    for (int d = 0; d < D; ++d) out_row[d] = float_to_bf16((float)(acc[d] / l));
}

/*
 * Attention of new queries over a cache that already holds their own k/v.
 * rows == NULL: every row (b, i < chunk, h) is written to out [B,chunk_stride,Hq,D].
 * rows != NULL: nrows triples (b, i, h); row r is written to out + r*D.
 */
int oracle_attend(const oracle_cfg* c, const uint16_t* q, const int32_t* hist, int chunk,
                  int chunk_stride, const uint16_t* k_cache, const uint16_t* v_cache, uint16_t* out,
                  int nrows, const int32_t* rows) {
    if (!cfg_ok(c) || !q || !k_cache || !v_cache || !out || chunk_stride < chunk || !hist_ok(c, hist, chunk))
        return -1;
    int D = c->head_dim, Hq = c->n_q_heads;
    if (rows) {
        for (int r = 0; r < nrows; ++r) {
            const int32_t* t3 = rows + 3 * r;
            if (t3[0] < 0 || t3[0] >= c->batch || t3[1] < 0 || t3[1] >= chunk || t3[2] < 0 || t3[2] >= Hq)
                return -1;
        }
    }
    tables t;
    if (make_tables(c, &t)) return -1;
    float* qr = (float*)malloc(sizeof(float) * D);
    double* acc = (double*)malloc(sizeof(double) * D);
    double* sc = (double*)malloc(sizeof(double) * (size_t)c->max_len);
    if (rows) {
        for (int r = 0; r < nrows; ++r) {
            int b = rows[3 * r], i = rows[3 * r + 1], h = rows[3 * r + 2];
            const uint16_t* q_row = q + (((size_t)b * chunk_stride + i) * Hq + h) * D;
            attend_row(c, &t, q_row, b, h, hist[b] + i, k_cache, v_cache, out + (size_t)r * D, qr, sc, acc);
        }
    } else {
        for (int b = 0; b < c->batch; ++b)
            for (int i = 0; i < chunk; ++i)
                for (int h = 0; h < Hq; ++h) {
                    size_t off = (((size_t)b * chunk_stride + i) * Hq + h) * D;
                    attend_row(c, &t, q + off, b, h, hist[b] + i, k_cache, v_cache, out + off, qr, sc, acc);
                }
    }
    free(qr);
    free(acc);
    free(sc);
    free_tables(&t);
    return 0;
}

/* The three stages: append the new tokens, then attend (Listing 2 order). */
static int stage(const oracle_cfg* c, const uint16_t* q, const uint16_t* k, const uint16_t* v,
                 const int32_t* hist, int chunk, uint16_t* k_cache, uint16_t* v_cache, uint16_t* out) {
    if (!cfg_ok(c) || !q || !out || !hist_ok(c, hist, chunk)) return -1;
    if (oracle_append(c, k, v, hist, chunk, chunk, k_cache, v_cache)) return -1;
    return oracle_attend(c, q, hist, chunk, chunk, k_cache, v_cache, out, 0, NULL);
}

/* Prefill (Section 4.2, with_history=False): no history, positions 0..chunk-1. */
int oracle_prefill(const oracle_cfg* c, const uint16_t* q, const uint16_t* k, const uint16_t* v, int chunk,
                   uint16_t* k_cache, uint16_t* v_cache, uint16_t* out) {
    if (!cfg_ok(c)) return -1;
    int32_t* hist = (int32_t*)calloc((size_t)c->batch, sizeof(int32_t));
    int rc = stage(c, q, k, v, hist, chunk, k_cache, v_cache, out);
    free(hist);
    return rc;
}

/* Prefill_kv (Section 4.3, with_history=True): hist_len history tokens shared by the batch. */
int oracle_prefill_kv(const oracle_cfg* c, const uint16_t* q, const uint16_t* k, const uint16_t* v,
                      int hist_len, int chunk, uint16_t* k_cache, uint16_t* v_cache, uint16_t* out) {
    if (!cfg_ok(c)) return -1;
    int32_t* hist = (int32_t*)malloc(sizeof(int32_t) * (size_t)c->batch);
    for (int b = 0; b < c->batch; ++b) hist[b] = hist_len;
    int rc = stage(c, q, k, v, hist, chunk, k_cache, v_cache, out);
    free(hist);
    return rc;
}

/* Decode (Section 4.4): one new token per sequence, hist_len[b] valid history tokens. */
int oracle_decode(const oracle_cfg* c, const uint16_t* q, const uint16_t* k, const uint16_t* v,
                  const int32_t* hist_len, uint16_t* k_cache, uint16_t* v_cache, uint16_t* out) {
    return stage(c, q, k, v, hist_len, 1, k_cache, v_cache, out);
}
