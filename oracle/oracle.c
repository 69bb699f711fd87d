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
 * Readings of points the paper leaves open (each is listed in the design doc):
 *   - ties between equal logits are broken by ascending vocabulary index;
 *   - the sparse tensor is fp32 with -inf = 0xFF800000;
 *   - within a row of the sparse tensor, indices are expected to be distinct;
 *     if they are not, the later entry j overwrites the earlier one.
 *
 * Rows are independent, so the row loop may run on several OpenMP threads;
 * that changes no arithmetic of any single z_i.
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
