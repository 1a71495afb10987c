/*
 * spike_oracle.h -- CPU oracle for the spike-gated INT8 projection.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path links, loads or
 * calls this code: only the test suite, the smoke check and the CPU-baseline
 * leg of the benchmark do.  It shares no source with the CUDA library.
 *
 * What it computes (Section 2.3, Eq. (sparse)):
 *
 *     A   = { k : x_k = 1 }                       (Section 2.2, active set)
 *     y_m = s_m * sum_{k in A} Q_{m,k}             (Eq. sparse)
 *
 * with Q an INT8 matrix of M = N output channels by K input columns, stored
 * column-major (Section 2.2: "each selected column is a contiguous read across
 * output channels"), so element (m, k) lives at Q[k * ldq + m]; s the FP32
 * per-output-channel scale (Section 2.3 quantiser); x a binary spike vector.
 * The sum is held in a 64-bit integer, range-checked and narrowed to INT32
 * (the paper's general accumulator is INT32, Section 2.3), converted to FP32
 * and multiplied by s_m once per output channel (Section 2.3).
 *
 * Spike formats: SP_ORACLE_U8 -- one byte per column, any nonzero byte is a
 * spike; SP_ORACLE_BITS32 -- uint32 words, column k is bit (k % 32) of word
 * (k / 32), bits at or beyond K are ignored.
 *
 * sp_oracle_dense is the paper's other kernel: the continuous-input
 * projection over row-major INT8 weights.  sp_oracle_lif produces spike rows
 * in the BITS32 format from a LIF state.  sp_oracle_head (declared last) is
 * the vocabulary head with INT8 activations and candidate-row verification.
 *
 * All functions are single-threaded, allocate only O(K) scratch, and return
 * 0 on success, a negative code on a bad argument (-1) or an INT32 overflow of
 * the accumulator (-2), and -3 if scratch allocation fails.
 */
#ifndef SPIKE_ORACLE_H
#define SPIKE_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum { SP_ORACLE_BITS32 = 0, SP_ORACLE_U8 = 1 };

/* Active index set A of one spike row, ascending.  idx must hold K entries;
 * *count receives |A|.  ld-free: spikes points at the row itself. */
int sp_oracle_active_set(const void *spikes, int fmt, int32_t K,
                         int32_t *idx, int32_t *count);

/* Eq. (sparse) for T spike rows.  Row t of the spikes starts at
 * (const uint8_t*)spikes + t * ld_spikes * (fmt == BITS32 ? 4 : 1), i.e.
 * ld_spikes counts words for BITS32 and bytes for U8.  Outputs are dense
 * [T][N]: acc[t*N + m], y[t*N + m].  Either output may be NULL. */
int sp_oracle_project(const int8_t *Q, int64_t ldq, const float *s,
                      int32_t N, int32_t K,
                      const void *spikes, int fmt, int64_t ld_spikes, int32_t T,
                      int32_t *acc, float *y);

/* Eq. (sparse) at selected outputs only: entry e is token row t_idx[e],
 * output channel m_idx[e].  For checks at sizes where the full product is
 * too slow for a single CPU thread. */
int sp_oracle_project_entries(const int8_t *Q, int64_t ldq, const float *s,
                              int32_t N, int32_t K,
                              const void *spikes, int fmt, int64_t ld_spikes,
                              int32_t T, int64_t count,
                              const int32_t *t_idx, const int32_t *m_idx,
                              int32_t *acc, float *y);

/* Continuous-input projection (Section 2.3: for continuous inputs the
 * weights are converted to FP32, multiplied with the FP32 activations and
 * accumulated, and the row scale is applied afterwards; Section 2.2: dense
 * projections keep row-major storage, one contiguous dot product per output):
 *
 *     y_m = s_m * sum_k Q_{m,k} x_k
 *
 * with Q INT8 ROW-MAJOR, element (m, k) at Q[m * ldq + k] (ldq >= K), and x
 * FP32 rows, row t at x + t * ldx (ldx >= K when T > 1).  The value is
 * computed in double: every product (double)Q * (double)x is exact (8 + 24
 * significant bits), the K products are summed in ascending k (error at most
 * K * 2^-53 of sum_k |Q_{m,k} x_k|, far below FP32 resolution), and the scale
 * is one double multiply.  Outputs are dense [T][N]: y[t*N + m] and
 * abs_dot[t*N + m] = sum_k |Q_{m,k} x_k| (for error bounds); either may be
 * NULL. */
int sp_oracle_dense(const int8_t *Q, int64_t ldq, const float *s,
                    int32_t N, int32_t K, const float *x, int64_t ldx,
                    int32_t T, double *y, double *abs_dot);

/* Spike producer: one leaky integrate-and-fire step for T rows of K neurons,
 * written straight into the SP_ORACLE_BITS32 format.  The paper names LIF
 * dynamics (Section 1) without stating the update, so this is a reading:
 *
 *     v  <- fmaf(beta, v, I)            one FP32 fused multiply-add
 *     x  =  (v >= theta)                the spike
 *     v  <- v - theta   where x = 1     soft reset, one FP32 subtract
 *
 * Row t of v and I starts at element t * ld; row t of the bits at word
 * t * ld_bits (ceil(K/32) words: bit k % 32 of word k / 32, LSB first, bits at
 * or past K written as 0).  v is updated in place. */
int sp_oracle_lif(float *v, const float *I, int32_t K, int32_t T, int64_t ld,
                  float beta, float theta, uint32_t *bits, int64_t ld_bits);

/* Vocabulary head with INT8 activations and candidate-row verification
 * (Section 5, trace configuration; Appendix D).  The head is a continuous-
 * input projection with row-major INT8 weights Q (element (m, k) at
 * Q[m * ldq + k], V rows of K) and row scales s.  For each hidden state h
 * (row b at h + b * ldh), in the paper's order:
 *
 *   1. INT8 activations.  The paper does not state the activation quantiser;
 *      this reads it as the weight rule of Section 2.3 applied to the vector,
 *      in FP32: s_x = max(max_k |h_k|, 1e-8) / 127,
 *      q_k = clip(round_half_even(h_k / s_x), -127, 127).
 *   2. Approximate logits over the full vocabulary: the integer dot product
 *      a_m = sum_k Q_{m,k} q_k (exact, INT32), then
 *      z_m = s_m * (s_x * float(a_m)), two FP32 multiplies.
 *   3. Order the rows by z descending, equal z by ascending index; the top-two
 *      gap is gap = z_(1) - z_(2) (one FP32 subtraction).
 *   4. The gate: verification runs when gap < tau (0.5 in the trace
 *      configuration, 4.0 in the power configuration).
 *   5. Candidates: the first k_sel rows of that order (K = 16, 32, 64 in the
 *      paper).  Each is recomputed with FP32 activations, the continuous-input
 *      rule of Section 2.3: r_m = s_m * sum_k float(Q_{m,k}) h_k.  Here in
 *      double, as sp_oracle_dense: every product exact, the sum within
 *      K * 2^-53 of sum_k |Q_{m,k} h_k| (returned in r_abs for error bounds).
 *   6. The token: with verification, the candidate with the largest r (equal r
 *      by ascending index); without, the first row of the order.
 *
 * Outputs per row b (any pointer may be NULL): codes[b*K + k] = q_k, s_x[b],
 * z[b*V + m], gap[b], verified[b] (0 / 1), cand[b*k_sel + i] (the order's
 * first k_sel rows), r[b*k_sel + i], r_abs[b*k_sel + i] (for every candidate,
 * whether or not the gate opened), token[b].
 * Requires V >= 2, 1 <= k_sel <= V, ldq >= K, ldh >= K when B > 1; -1 on a bad
 * argument, -3 when scratch allocation fails. */
int sp_oracle_head(const int8_t *Q, int64_t ldq, const float *s, int32_t V,
                   int32_t K, const float *h, int64_t ldh, int32_t B, float tau,
                   int32_t k_sel, int8_t *codes, float *s_x, float *z,
                   float *gap, int32_t *verified, int32_t *cand, double *r,
                   double *r_abs, int32_t *token);

#ifdef __cplusplus
}
#endif

#endif /* SPIKE_ORACLE_H */
