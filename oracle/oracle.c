/*
 * oracle.c - plain CPU oracle for the exact LLM output head.
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the
 * cpu_baseline / reference legs of bench.py may load this library.  It shares
 * no code, header, table or helper with the CUDA path under
 * paper_2608_27460_gb300/csrc and must never be called by that path.
 *
 * What it computes (paper, Section 3 "Vector Index Embedding"):
 *   - the logit vector z = W_out h, one entry per vocabulary row,
 *     z_i = <w_i, h>                                   (Section 3, eq. z = W_out h)
 *   - top-k token selection as exhaustive maximum inner product search:
 *     the k rows with the largest inner product       (Section 2 "MIPS", Section 3)
 *   - the sparse full-vocabulary logit tensor: the k retrieved logits at their
 *     vocabulary indices, -infinity everywhere else   (Section 3, last paragraphs)
 *
 * Precision: W_out is given as raw bf16 bit patterns, h as fp32.  Every
 * element is widened exactly to fp64 and each z_i is one sequential fp64
 * sum over j = 0..d-1 in index order.  No blocking, no reordering.
 *
 * Readings of points the paper leaves open:
 *   - ties between equal logits are broken by ascending vocabulary index;
 *   - the sparse tensor is fp32 with -inf = 0xFF800000;
 *   - within a row of the sparse tensor, indices are expected to be distinct;
 *     if they are not, the later entry j overwrites the earlier one.
 *
 * Rows are independent, so the row loop may run on several OpenMP threads;
 * that changes no arithmetic of any single z_i.
 *
 * Top-k sampling (Section 2: top-k sampling restricts the draw to the k most
 * probable tokens; Section 3: the retrieved logits feed standard logit
 * processors such as top-p and min-p as a second stage; Section 4 samples
 * with k = 50).  The paper names no random generator and no processor order;
 * the readings taken are:
 *   - probabilities are the softmax of z / T over the k candidates;
 *   - top-p and min-p are both defined on that softmax, so each keeps a
 *     prefix of the candidates (they are sorted by logit) and the kept set is
 *     the shorter prefix: the two filters commute;
 *   - the draw is the inverse CDF of the kept probabilities at one uniform u;
 *   - u comes from the counter-based generator Philox4x32-10 (Salmon, Moraes,
 *     Dror, Shaw, "Parallel random numbers: as easy as 1, 2, 3", SC 2011):
 *     counter (step low, step high, query, 0), key (seed low, seed high), the
 *     top 24 bits of the first output word times 2^-24.
 *
 * Quantised output embedding (Section 4 names weight quantisation as a
 * bandwidth-saving technique orthogonal to the method).  Readings: each row
 * of W_out is stored as 8-bit floats of the e4m3 format (1 sign bit, 4
 * exponent bits with bias 7, 3 mantissa bits, subnormals, no infinities,
 * largest finite value 448) times one fp32 scale per row,
 *   scale_i = max_j |w_ij| / 448 in fp32 (1 for an all-zero row),
 *   q_ij = e4m3(w_ij / scale_i), the fp32 quotient rounded to the nearest
 *          e4m3 value, ties to even, magnitudes past 448 saturated;
 * and the head computes z_i = scale_i * sum_j e4m3(q_ij) * h_j.
 *
 * Recall@k (Section 4.3: the share of the exact head's top-k tokens that an
 * approximate search also retrieves, averaged over many hidden states).
 * Readings: the approximate method hands over m candidate indices per query
 * (m may differ from k), taken as a set: a repeated candidate counts once and
 * a negative entry is an empty slot; the hits of a query are the positions
 * j < k of the exact top-k whose index is among the candidates; Recall@k is
 * the sum of the hits over the n queries divided by n k.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORACLE_OK 0
#define ORACLE_EINVAL 1
#define ORACLE_ENOMEM 4

/* A bf16 value is the upper 16 bits of an IEEE binary32 value. */
double oracle_bf16_to_double(uint16_t bits) {
    uint32_t u = ((uint32_t)bits) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* z[b*V + i] = sum_j W[i,j] * h[b,j] in fp64 (Section 3, z_i = <w_i, h>). */
int oracle_logits(const uint16_t *W, int64_t V, int32_t d, const float *h,
                  int32_t batch, double *z, int32_t nthreads) {
    if (!W || !h || !z || V < 1 || d < 1 || batch < 1) return ORACLE_EINVAL;
    if (nthreads < 1) nthreads = 1;
    for (int32_t b = 0; b < batch; ++b) {
        const float *hb = h + (int64_t)b * d;
        double *zb = z + (int64_t)b * V;
#pragma omp parallel for num_threads(nthreads) schedule(static)
        for (int64_t i = 0; i < V; ++i) {
            const uint16_t *wi = W + i * (int64_t)d;
            double acc = 0.0;
            for (int32_t j = 0; j < d; ++j)
                acc += oracle_bf16_to_double(wi[j]) * (double)hb[j];
            zb[i] = acc;
        }
    }
    return ORACLE_OK;
}

typedef struct {
    double z;
    int64_t i;
} scored_row;

/* Descending by logit; equal logits in ascending vocabulary index. */
static int by_logit_desc_index_asc(const void *pa, const void *pb) {
    const scored_row *a = (const scored_row *)pa;
    const scored_row *b = (const scored_row *)pb;
    if (a->z > b->z) return -1;
    if (a->z < b->z) return 1;
    if (a->i < b->i) return -1;
    if (a->i > b->i) return 1;
    return 0;
}

/*
 * Exhaustive MIPS (Section 2, Section 3): compute every z_i, sort all V rows
 * by (z desc, index asc), keep the first k.  idx[b*k + j] is the vocabulary
 * index of rank j, logits[b*k + j] its fp64 logit.
 */
int oracle_topk(const uint16_t *W, int64_t V, int32_t d, const float *h,
                int32_t batch, int32_t k, int32_t *idx, double *logits,
                int32_t nthreads) {
    if (!W || !h || !idx || !logits || V < 1 || d < 1 || batch < 1 || k < 1 ||
        (int64_t)k > V)
        return ORACLE_EINVAL;
    double *z = (double *)malloc(sizeof(double) * (size_t)V);
    scored_row *rows = (scored_row *)malloc(sizeof(scored_row) * (size_t)V);
    if (!z || !rows) {
        free(z);
        free(rows);
        return ORACLE_ENOMEM;
    }
    int rc = ORACLE_OK;
    for (int32_t b = 0; b < batch && rc == ORACLE_OK; ++b) {
        rc = oracle_logits(W, V, d, h + (int64_t)b * d, 1, z, nthreads);
        if (rc != ORACLE_OK) break;
        for (int64_t i = 0; i < V; ++i) {
            rows[i].z = z[i];
            rows[i].i = i;
        }
        qsort(rows, (size_t)V, sizeof(scored_row), by_logit_desc_index_asc);
        for (int32_t j = 0; j < k; ++j) {
            idx[(int64_t)b * k + j] = (int32_t)rows[j].i;
            logits[(int64_t)b * k + j] = rows[j].z;
        }
    }
    free(z);
    free(rows);
    return rc;
}

/*
 * Sparse full-vocabulary logits (Section 3): out[b, v] = -inf for every v,
 * then out[b, idx[b, j]] = logits[b, j] for j = 0..k-1 in order.
 * An index outside [0, V) is skipped and the call returns ORACLE_EINVAL.
 */
int oracle_scatter(const int32_t *idx, const float *logits, int32_t batch,
                   int32_t k, int64_t V, float *out) {
    if (!idx || !logits || !out || batch < 1 || k < 1 || V < 1)
        return ORACLE_EINVAL;
    int rc = ORACLE_OK;
    for (int32_t b = 0; b < batch; ++b) {
        float *row = out + (int64_t)b * V;
        for (int64_t v = 0; v < V; ++v) row[v] = -INFINITY;
        for (int32_t j = 0; j < k; ++j) {
            int32_t t = idx[(int64_t)b * k + j];
            if (t < 0 || (int64_t)t >= V) {
                rc = ORACLE_EINVAL;
                continue;
            }
            row[t] = logits[(int64_t)b * k + j];
        }
    }
    return rc;
}

int oracle_max_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* ------------------------------------------------------------------------ */
/* Philox4x32-10: ten rounds; a round multiplies words 0 and 2 by the two
 * published constants into 64-bit products and mixes the halves with words
 * 1 and 3 and the key; the key is bumped by the two published Weyl
 * constants between rounds. */
void oracle_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) {
    uint32_t c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3];
    uint32_t k0 = key[0], k1 = key[1];
    for (int r = 0; r < 10; ++r) {
        if (r > 0) {
            k0 += 0x9E3779B9u;
            k1 += 0xBB67AE85u;
        }
        const uint64_t p0 = (uint64_t)0xD2511F53u * c0;
        const uint64_t p1 = (uint64_t)0xCD9E8D57u * c2;
        const uint32_t n0 = (uint32_t)(p1 >> 32) ^ c1 ^ k0;
        const uint32_t n1 = (uint32_t)p1;
        const uint32_t n2 = (uint32_t)(p0 >> 32) ^ c3 ^ k1;
        const uint32_t n3 = (uint32_t)p0;
        c0 = n0;
        c1 = n1;
        c2 = n2;
        c3 = n3;
    }
    out[0] = c0;
    out[1] = c1;
    out[2] = c2;
    out[3] = c3;
}

/* The uniform of query q at decode step `step` under `seed`, in [0, 1). */
double oracle_uniform(uint64_t seed, uint64_t step, uint32_t q) {
    const uint32_t ctr[4] = {(uint32_t)step, (uint32_t)(step >> 32), q, 0u};
    const uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
    uint32_t out[4];
    oracle_philox4x32_10(ctr, key, out);
    return (double)(out[0] >> 8) * (1.0 / 16777216.0);
}

/*
 * One draw from the k candidate logits z[0..k), sorted descending:
 *   s_j = z_j / T;  p_j = exp(s_j - s_0) / sum_i exp(s_i - s_0)
 *   top-p: n_p = the smallest n >= 1 with sum_{i<n} p_i >= top_p
 *   min-p: n_m = the number of j with p_j >= min_p * p_0
 *   n = min(n_p, n_m);  M = sum_{i<n} p_i
 *   j* = the smallest j < n with sum_{i<=j} p_i > u * M (n - 1 if none)
 * Writes j*, p_{j*} / M and n.  Requires T > 0, 0 < top_p <= 1,
 * 0 <= min_p <= 1, 0 <= u < 1.
 */
int oracle_sample_sorted(const double *z, int32_t k, double T, double top_p, double min_p,
                         double u, int32_t *j_out, double *prob_out, int32_t *kept_out) {
    if (!z || !j_out || !prob_out || !kept_out || k < 1) return ORACLE_EINVAL;
    if (!(T > 0.0) || !(top_p > 0.0 && top_p <= 1.0) || !(min_p >= 0.0 && min_p <= 1.0) ||
        !(u >= 0.0 && u < 1.0))
        return ORACLE_EINVAL;
    double *p = (double *)malloc(sizeof(double) * (size_t)k);
    if (!p) return ORACLE_ENOMEM;
    const double s0 = z[0] / T;
    double total = 0.0;
    for (int32_t j = 0; j < k; ++j) {
        p[j] = exp(z[j] / T - s0);
        total += p[j];
    }
    for (int32_t j = 0; j < k; ++j) p[j] /= total;
    int32_t n_p = k;
    double run = 0.0;
    for (int32_t n = 1; n <= k; ++n) {
        run += p[n - 1];
        if (run >= top_p) {
            n_p = n;
            break;
        }
    }
    int32_t n_m = 0;
    for (int32_t j = 0; j < k; ++j)
        if (p[j] >= min_p * p[0]) ++n_m;
    const int32_t n = n_p < n_m ? n_p : n_m;
    double M = 0.0;
    for (int32_t j = 0; j < n; ++j) M += p[j];
    const double target = u * M;
    int32_t js = n - 1;
    double cum = 0.0;
    for (int32_t j = 0; j < n; ++j) {
        cum += p[j];
        if (cum > target) {
            js = j;
            break;
        }
    }
    *j_out = js;
    *prob_out = p[js] / M;
    *kept_out = n;
    free(p);
    return ORACLE_OK;
}

/* ------------------------------------------------------------------------ */
/* e4m3 code -> value, exactly.  Code 0x7f / 0xff is NaN. */
double oracle_e4m3_to_double(uint8_t c) {
    const int sgn = (c >> 7) & 1, E = (c >> 3) & 15, M = c & 7;
    double v;
    if (E == 15 && M == 7) return NAN;
    if (E == 0)
        v = ldexp((double)M, -9);              /* subnormal: M * 2^-9 */
    else
        v = ldexp(1.0 + M / 8.0, E - 7);       /* normal: (1 + M/8) * 2^(E-7) */
    return sgn ? -v : v;
}

/* fp32 value -> nearest e4m3 code, ties to even, magnitudes past 448 to 448. */
uint8_t oracle_f32_to_e4m3(float x) {
    const int sgn = signbit(x) ? 1 : 0;
    const double a = fabs((double)x);
    if (a >= 448.0) return (uint8_t)((sgn << 7) | (15 << 3) | 6);
    if (a < ldexp(1.0, -6)) {
        /* subnormal range: a multiple of 2^-9 (8 * 2^-9 is the least normal) */
        const double m = rint(ldexp(a, 9));    /* rint: to nearest, ties to even */
        return (uint8_t)((sgn << 7) | (int)m);  /* m = 8 gives exponent field 1 */
    }
    int e;
    frexp(a, &e);                              /* a = f * 2^e, f in [0.5, 1) */
    e -= 1;                                    /* a = (1 + t) * 2^e, t in [0, 1) */
    double m = rint((ldexp(a, -e) - 1.0) * 8.0);
    if (m == 8.0) {
        m = 0.0;
        e += 1;
    }
    if (e > 8 || (e == 8 && m > 6.0)) return (uint8_t)((sgn << 7) | (15 << 3) | 6);
    return (uint8_t)((sgn << 7) | ((e + 7) << 3) | (int)m);
}

/* Quantise bf16 rows W [V, d] to e4m3 codes q [V, d] and fp32 scales [V]. */
int oracle_quantize_e4m3(const uint16_t *W, int64_t V, int32_t d, uint8_t *q, float *scale) {
    if (!W || !q || !scale || V < 1 || d < 1) return ORACLE_EINVAL;
    for (int64_t i = 0; i < V; ++i) {
        const uint16_t *wi = W + i * (int64_t)d;
        float amax = 0.0f;
        for (int32_t j = 0; j < d; ++j) {
            const float a = fabsf((float)oracle_bf16_to_double(wi[j]));
            if (a > amax) amax = a;
        }
        const float s = amax > 0.0f ? amax / 448.0f : 1.0f;
        scale[i] = s;
        for (int32_t j = 0; j < d; ++j)
            q[i * (int64_t)d + j] = oracle_f32_to_e4m3((float)oracle_bf16_to_double(wi[j]) / s);
    }
    return ORACLE_OK;
}

/* z[b*V + i] = scale_i * sum_j e4m3(q_ij) * h[b, j] in fp64. */
int oracle_logits_e4m3(const uint8_t *q, const float *scale, int64_t V, int32_t d,
                       const float *h, int32_t batch, double *z, int32_t nthreads) {
    if (!q || !scale || !h || !z || V < 1 || d < 1 || batch < 1) return ORACLE_EINVAL;
    if (nthreads < 1) nthreads = 1;
    for (int32_t b = 0; b < batch; ++b) {
        const float *hb = h + (int64_t)b * d;
        double *zb = z + (int64_t)b * V;
#pragma omp parallel for num_threads(nthreads) schedule(static)
        for (int64_t i = 0; i < V; ++i) {
            const uint8_t *qi = q + i * (int64_t)d;
            double acc = 0.0;
            for (int32_t j = 0; j < d; ++j) acc += oracle_e4m3_to_double(qi[j]) * (double)hb[j];
            zb[i] = (double)scale[i] * acc;
        }
    }
    return ORACLE_OK;
}

/* Exhaustive MIPS over the quantised rows: the same full sort as oracle_topk
 * on z_i = scale_i * sum_j e4m3(q_ij) * h_j. */
int oracle_topk_e4m3(const uint8_t *q, const float *scale, int64_t V, int32_t d, const float *h,
                     int32_t batch, int32_t k, int32_t *idx, double *logits, int32_t nthreads) {
    if (!q || !scale || !h || !idx || !logits || V < 1 || d < 1 || batch < 1 || k < 1 ||
        (int64_t)k > V)
        return ORACLE_EINVAL;
    double *z = (double *)malloc(sizeof(double) * (size_t)V);
    scored_row *rows = (scored_row *)malloc(sizeof(scored_row) * (size_t)V);
    if (!z || !rows) {
        free(z);
        free(rows);
        return ORACLE_ENOMEM;
    }
    int rc = ORACLE_OK;
    for (int32_t b = 0; b < batch && rc == ORACLE_OK; ++b) {
        rc = oracle_logits_e4m3(q, scale, V, d, h + (int64_t)b * d, 1, z, nthreads);
        if (rc != ORACLE_OK) break;
        for (int64_t i = 0; i < V; ++i) {
            rows[i].z = z[i];
            rows[i].i = i;
        }
        qsort(rows, (size_t)V, sizeof(scored_row), by_logit_desc_index_asc);
        for (int32_t j = 0; j < k; ++j) {
            idx[(int64_t)b * k + j] = (int32_t)rows[j].i;
            logits[(int64_t)b * k + j] = rows[j].z;
        }
    }
    free(z);
    free(rows);
    return rc;
}

/* ------------------------------------------------------------------------ */
/* hits[q] = #{ j < k : exact[q, j] >= 0 and exact[q, j] in {approx[q, i] : i < m} } */
int oracle_recall_hits(const int32_t *exact, int32_t k, const int32_t *approx, int32_t m, int64_t n,
                       int32_t *hits) {
    if (!exact || !approx || !hits || k < 1 || m < 1 || n < 1) return ORACLE_EINVAL;
    for (int64_t q = 0; q < n; ++q) {
        const int32_t *eq = exact + q * k, *aq = approx + q * m;
        int32_t h = 0;
        for (int32_t j = 0; j < k; ++j) {
            if (eq[j] < 0) continue;
            for (int32_t i = 0; i < m; ++i) {
                if (aq[i] == eq[j]) {
                    ++h;
                    break;
                }
            }
        }
        hits[q] = h;
    }
    return ORACLE_OK;
}
