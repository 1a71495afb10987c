/*
 * spike_oracle.c -- plain, slow, single-threaded CPU oracle for the
 * spike-gated INT8 projection of Section 2.3, Eq. (sparse).
 *
 * TEST INFRASTRUCTURE ONLY: used by the test suite, the smoke check and the
 * CPU-baseline leg of the benchmark.  It is never linked into, loaded by or
 * called from the CUDA library, and includes none of its headers.
 *
 * The method reaches exactly the value of the definition (integer sums are
 * order-free and the accumulator never leaves the INT32 range for K <= 2^24
 * / 128), so this file writes the definition out and nothing else:
 *
 *   1. A = { k : x_k = 1 }, ascending                       (Section 2.2)
 *   2. acc_m = sum_{k in A} Q_{m,k},  Q_{m,k} = Q[k*ldq + m] (Eq. sparse,
 *      column-major storage of Section 2.2), in int64, then checked to fit
 *      INT32, the paper's accumulator width (Section 2.3)
 *   3. y_m = s_m * (float)acc_m: one conversion to FP32 and one FP32
 *      multiply per output channel (Section 2.3).  Built with
 *      -ffp-contract=off; there is nothing to contract anyway.
 *
 * Parity pins for this file live in the test suite: dense integer matmul
 * (numpy) on tiny and full shapes, exhaustive masks on tiny K, hand-worked
 * fixtures, invariants (zero, one-hot, additivity, all-ones, permutation,
 * format equivalence) and closed forms.
 */
#include "spike_oracle.h"

#include <math.h>
#include <stdlib.h>

/* Spike x_k of one row: 1 if column k fires, else 0 (Section 1: x in {0,1}^K;
 * any nonzero byte counts as a spike in the U8 format). */
static int spike_at(const void *row, int fmt, int32_t k)
{
    if (fmt == SP_ORACLE_BITS32) {
        const uint32_t *w = (const uint32_t *)row;
        return (int)((w[k / 32] >> (k % 32)) & 1u);
    }
    return ((const uint8_t *)row)[k] != 0;
}

static const void *spike_row(const void *spikes, int fmt, int64_t ld_spikes,
                             int32_t t)
{
    int64_t elem = (fmt == SP_ORACLE_BITS32) ? 4 : 1;
    return (const uint8_t *)spikes + (int64_t)t * ld_spikes * elem;
}

static int check_args(const int8_t *Q, int64_t ldq, int32_t N, int32_t K,
                      const void *spikes, int fmt, int64_t ld_spikes, int32_t T)
{
    if (!Q || !spikes || N < 0 || K < 0 || T < 0 || ldq < N)
        return -1;
    if (fmt != SP_ORACLE_BITS32 && fmt != SP_ORACLE_U8)
        return -1;
    if (T > 1) {
        int64_t need = (fmt == SP_ORACLE_BITS32) ? ((int64_t)K + 31) / 32 : K;
        if (ld_spikes < need)
            return -1;
    }
    return 0;
}

int sp_oracle_active_set(const void *spikes, int fmt, int32_t K,
                         int32_t *idx, int32_t *count)
{
    if (!spikes || !idx || !count || K < 0)
        return -1;
    if (fmt != SP_ORACLE_BITS32 && fmt != SP_ORACLE_U8)
        return -1;
    int32_t n = 0;
    for (int32_t k = 0; k < K; ++k)
        if (spike_at(spikes, fmt, k))
            idx[n++] = k;
    *count = n;
    return 0;
}

/* Steps 2 and 3 for one output channel m, given the active set A. */
static int project_one(const int8_t *Q, int64_t ldq, const float *s,
                       int32_t m, const int32_t *A, int32_t nA,
                       int32_t *acc_out, float *y_out)
{
    int64_t acc = 0;
    for (int32_t i = 0; i < nA; ++i)
        acc += Q[(int64_t)A[i] * ldq + m];
    if (acc > INT32_MAX || acc < INT32_MIN)
        return -2;
    int32_t acc32 = (int32_t)acc;
    if (acc_out)
        *acc_out = acc32;
    if (y_out)
        *y_out = s[m] * (float)acc32;
    return 0;
}

int sp_oracle_project(const int8_t *Q, int64_t ldq, const float *s,
                      int32_t N, int32_t K,
                      const void *spikes, int fmt, int64_t ld_spikes, int32_t T,
                      int32_t *acc, float *y)
{
    int rc = check_args(Q, ldq, N, K, spikes, fmt, ld_spikes, T);
    if (rc)
        return rc;
    if (y && !s)
        return -1;
    int32_t *A = (int32_t *)malloc(sizeof(int32_t) * (size_t)(K > 0 ? K : 1));
    if (!A)
        return -3;
    for (int32_t t = 0; t < T && rc == 0; ++t) {
        int32_t nA = 0;
        sp_oracle_active_set(spike_row(spikes, fmt, ld_spikes, t), fmt, K, A, &nA);
        for (int32_t m = 0; m < N && rc == 0; ++m)
            rc = project_one(Q, ldq, s, m, A, nA,
                             acc ? &acc[(int64_t)t * N + m] : NULL,
                             y ? &y[(int64_t)t * N + m] : NULL);
    }
    free(A);
    return rc;
}

int sp_oracle_project_entries(const int8_t *Q, int64_t ldq, const float *s,
                              int32_t N, int32_t K,
                              const void *spikes, int fmt, int64_t ld_spikes,
                              int32_t T, int64_t count,
                              const int32_t *t_idx, const int32_t *m_idx,
                              int32_t *acc, float *y)
{
    int rc = check_args(Q, ldq, N, K, spikes, fmt, ld_spikes, T);
    if (rc)
        return rc;
    if (count < 0 || (count > 0 && (!t_idx || !m_idx)) || (y && !s))
        return -1;
    int32_t *A = (int32_t *)malloc(sizeof(int32_t) * (size_t)(K > 0 ? K : 1));
    if (!A)
        return -3;
    for (int64_t e = 0; e < count && rc == 0; ++e) {
        int32_t t = t_idx[e], m = m_idx[e];
        if (t < 0 || t >= T || m < 0 || m >= N) {
            rc = -1;
            break;
        }
        int32_t nA = 0;
        sp_oracle_active_set(spike_row(spikes, fmt, ld_spikes, t), fmt, K, A, &nA);
        rc = project_one(Q, ldq, s, m, A, nA,
                         acc ? &acc[e] : NULL, y ? &y[e] : NULL);
    }
    free(A);
    return rc;
}

/* Continuous-input projection, written out as its definition (Section 2.3):
 * for each row t and output m, dot = sum_k Q_{m,k} x_k with Q row-major
 * (Section 2.2), then y = s_m * dot.  See spike_oracle.h for the precision. */
int sp_oracle_dense(const int8_t *Q, int64_t ldq, const float *s,
                    int32_t N, int32_t K, const float *x, int64_t ldx,
                    int32_t T, double *y, double *abs_dot)
{
    if (!Q || !x || N < 0 || K < 0 || T < 0 || ldq < K || (y && !s))
        return -1;
    if (T > 1 && ldx < K)
        return -1;
    for (int32_t t = 0; t < T; ++t) {
        const float *xt = x + (int64_t)t * ldx;
        for (int32_t m = 0; m < N; ++m) {
            const int8_t *q = Q + (int64_t)m * ldq;
            double dot = 0.0, mag = 0.0;
            for (int32_t k = 0; k < K; ++k) {
                double term = (double)q[k] * (double)xt[k];
                dot += term;
                mag += term < 0 ? -term : term;
            }
            if (y)
                y[(int64_t)t * N + m] = (double)s[m] * dot;
            if (abs_dot)
                abs_dot[(int64_t)t * N + m] = mag;
        }
    }
    return 0;
}

/* One LIF step and the spike bits, as stated in spike_oracle.h (a reading:
 * the paper does not give the update). */
int sp_oracle_lif(float *v, const float *I, int32_t K, int32_t T, int64_t ld,
                  float beta, float theta, uint32_t *bits, int64_t ld_bits)
{
    const int64_t words = ((int64_t)K + 31) / 32;
    if (!v || !I || !bits || K < 0 || T < 0 || (T > 1 && (ld < K || ld_bits < words)))
        return -1;
    for (int32_t t = 0; t < T; ++t) {
        float *vt = v + (int64_t)t * ld;
        const float *it = I + (int64_t)t * ld;
        uint32_t *bt = bits + (int64_t)t * ld_bits;
        for (int64_t w = 0; w < words; ++w)
            bt[w] = 0u;
        for (int32_t k = 0; k < K; ++k) {
            float u = fmaf(beta, vt[k], it[k]);
            if (u >= theta) {
                bt[k / 32] |= 1u << (k % 32);
                u = u - theta;
            }
            vt[k] = u;
        }
    }
    return 0;
}

/* Vocabulary head with INT8 activations and candidate-row verification, as
 * stated in spike_oracle.h (Section 5 and Appendix D; the activation quantiser
 * is a reading).  Steps are numbered as there. */
typedef struct {
    float z;
    int32_t m;
} head_entry;

/* z descending, then index ascending */
static int head_order(const void *pa, const void *pb)
{
    const head_entry *a = (const head_entry *)pa, *b = (const head_entry *)pb;
    if (a->z > b->z)
        return -1;
    if (a->z < b->z)
        return 1;
    return a->m < b->m ? -1 : (a->m > b->m ? 1 : 0);
}

int sp_oracle_head(const int8_t *Q, int64_t ldq, const float *s, int32_t V,
                   int32_t K, const float *h, int64_t ldh, int32_t B, float tau,
                   int32_t k_sel, int8_t *codes, float *s_x, float *z,
                   float *gap, int32_t *verified, int32_t *cand, double *r,
                   double *r_abs, int32_t *token)
{
    if (!Q || !s || !h || V < 2 || K < 1 || B < 0 || k_sel < 1 || k_sel > V || ldq < K ||
        (B > 1 && ldh < K))
        return -1;
    int8_t *q = (int8_t *)malloc((size_t)K);
    head_entry *order = (head_entry *)malloc((size_t)V * sizeof(head_entry));
    double *rc = (double *)malloc((size_t)k_sel * sizeof(double));
    if (!q || !order || !rc) {
        free(q);
        free(order);
        free(rc);
        return -3;
    }
    for (int32_t b = 0; b < B; ++b) {
        const float *hb = h + (int64_t)b * ldh;
        /* 1. activation scale and codes */
        float amax = 0.0f;
        for (int32_t k = 0; k < K; ++k)
            if (fabsf(hb[k]) > amax)
                amax = fabsf(hb[k]);
        const float sx = fmaxf(amax, 1e-8f) / 127.0f;
        for (int32_t k = 0; k < K; ++k) {
            float c = rintf(hb[k] / sx);
            if (c > 127.0f)
                c = 127.0f;
            if (c < -127.0f)
                c = -127.0f;
            q[k] = (int8_t)c;
        }
        /* 2. approximate logits */
        for (int32_t m = 0; m < V; ++m) {
            const int8_t *row = Q + (int64_t)m * ldq;
            int64_t a = 0;
            for (int32_t k = 0; k < K; ++k)
                a += (int64_t)row[k] * (int64_t)q[k];
            if (a > INT32_MAX || a < INT32_MIN) {
                free(q);
                free(order);
                free(rc);
                return -2;
            }
            const float t = sx * (float)(int32_t)a;
            order[m].z = s[m] * t;
            order[m].m = m;
            if (z)
                z[(int64_t)b * V + m] = order[m].z;
        }
        /* 3. order and top-two gap; 4. the gate */
        qsort(order, (size_t)V, sizeof(head_entry), head_order);
        const float g = order[0].z - order[1].z;
        const int open = g < tau;
        /* 5. candidates, recomputed with the FP32 activations */
        int32_t best = 0;
        for (int32_t i = 0; i < k_sel; ++i) {
            const int32_t m = order[i].m;
            const int8_t *row = Q + (int64_t)m * ldq;
            double sum = 0.0, abs_sum = 0.0;
            for (int32_t k = 0; k < K; ++k) {
                const double term = (double)row[k] * (double)hb[k];
                sum += term;
                abs_sum += fabs(term);
            }
            rc[i] = (double)s[m] * sum;
            if (rc[i] > rc[best] || (rc[i] == rc[best] && m < order[best].m))
                best = i;
            if (cand)
                cand[(int64_t)b * k_sel + i] = m;
            if (r)
                r[(int64_t)b * k_sel + i] = rc[i];
            if (r_abs)
                r_abs[(int64_t)b * k_sel + i] = abs_sum;
        }
        /* 6. the token */
        if (codes)
            for (int32_t k = 0; k < K; ++k)
                codes[(int64_t)b * K + k] = q[k];
        if (s_x)
            s_x[b] = sx;
        if (gap)
            gap[b] = g;
        if (verified)
            verified[b] = open;
        if (token)
            token[b] = open ? order[best].m : order[0].m;
    }
    free(q);
    free(order);
    free(rc);
    return 0;
}
