/*
 * Online linear estimators of the global simulator (Sec. 3.3.1 "Transfer &
 * Operator Estimator"): the integer durations and link tables that the
 * what-if simulation (gmgsim.h) consumes, fitted on the GPU from executor
 * feedback.
 *
 *   transfer estimator, one per accelerator pair (d, e):   t = alpha * size + c
 *   operator estimator, one per (accelerator type, template operator):
 *                                                   t = sum_j beta_j * x_j
 *     with shape-derived features x (the paper's example for a batched matmul
 *     (b, m, n, k): x = (bmnk, bmk, bkn, bmn, 1)).
 *
 * "Incorporated online" (Sec. 3.3.1): every estimator keeps running
 * sufficient statistics of all samples it has received -- the Gram matrix
 * X^T X, X^T y and the sample count, in fp64 -- and est_update refits it by
 * least squares after adding a batch: beta = argmin ||X beta - y||^2 over all
 * samples so far, solved from the normal equations by a Cholesky
 * factorisation.  An estimator is "fitted" once it has at least F samples and
 * X^T X is positive definite (every Cholesky pivot above 1e-12 times its own
 * diagonal entry, a test that does not depend on the features' scales);
 * otherwise its coefficients are 0 and it is not used.  The normal equations
 * square the condition number of the column-scaled features: nearly
 * collinear features lose accuracy.
 *
 * All pointers are device pointers unless stated; calls are asynchronous on
 * `stream` and return 0 or a negative GMG_E* code (gmgsim.h) for invalid
 * arguments or a failed launch.  The library allocates nothing.
 */
#ifndef GMGEST_H
#define GMGEST_H

#include <stddef.h>
#include <stdint.h>

#include "gmgsim.h"

#ifdef __cplusplus
extern "C" {
#endif

#define GMG_EST_MAX_FEATURES 8

/* Bytes of device state for E estimators of F features (1 <= F <= 8):
 * per estimator the upper triangle of X^T X, X^T y, the count, the
 * coefficients and the fitted flag.  Caller-owned, 256-byte aligned; 0 on bad
 * arguments. */
size_t est_state_bytes(int32_t n_est, int32_t n_feat);

/* Zero every estimator's statistics, coefficients and fitted flags. */
int est_reset(void* d_state, int32_t n_est, int32_t n_feat, gmg_stream_t stream);

/* Bytes of the caller buffer est_update needs for a batch of n_samples
 * samples (chunk partial sums); 0 on bad arguments. */
size_t est_update_tmp_bytes(int32_t n_est, int32_t n_feat, int64_t n_samples);

/* Add a batch of feedback samples and refit every estimator.
 *   d_off [n_est + 1]  samples of estimator e are rows d_off[e] .. d_off[e+1]
 *                      (non-decreasing, d_off[0] = 0, d_off[n_est] = n_samples;
 *                      an estimator may get none)
 *   d_x   [S * F]      features of each sample, row-major (S = n_samples < 2^31)
 *   d_y   [S]          measured time of each sample (microseconds)
 *   d_tmp              caller buffer of est_update_tmp_bytes bytes, 256-byte
 *                      aligned (GMG_EWS if smaller); scratch, contents lost
 * The coefficients and flags are read back with est_coefficients.  Sums have
 * a fixed order (128-row chunks reduced by a fixed tree, chunks added in
 * order), so results are reproducible run to run. */
int est_update(void* d_state, int32_t n_est, int32_t n_feat, const int32_t* d_off, const double* d_x,
               const double* d_y, int64_t n_samples, void* d_tmp, size_t tmp_bytes, gmg_stream_t stream);

/* Copy the coefficients [n_est * F] (row-major, fp64) and fitted flags
 * [n_est] (int32 0/1) out of the state; either pointer may be NULL. */
int est_coefficients(const void* d_state, int32_t n_est, int32_t n_feat, double* d_beta, int32_t* d_fitted,
                     gmg_stream_t stream);

/* Durations for the simulation (gmg_desc_t.dur_by_type): for op i and
 * accelerator type t, with estimator e = d_est_of[i * n_types + t],
 *   dur[i * n_types + t] = clamp(rint(beta_e . x_i), 1, 2^40)   if e >= 0 and fitted,
 *                          d_dflt[i]                            otherwise.
 *   d_x [n_ops * F] op features (row-major), d_dflt [n_ops] >= 1.
 * rint rounds halves to even. */
int est_predict_durations(const void* d_state, int32_t n_est, int32_t n_feat, int32_t n_ops, int32_t n_types,
                          const int32_t* d_est_of, const double* d_x, const int64_t* d_dflt, int64_t* d_dur,
                          gmg_stream_t stream);

/* Link tables for the simulation (gmg_desc_t.bw_B_per_us / lat_us) from the
 * D*D transfer estimators (estimator d*D + e of a 2-feature state whose
 * features are (size in bytes, 1), so beta = (alpha us/B, c us)): off the
 * diagonal, if fitted,
 *   bw[d*D+e]  = clamp(rint(1 / alpha), 1, 2^40)   (2^40 when alpha <= 0),
 *   lat[d*D+e] = clamp(rint(c), 0, 2^40),
 * else the defaults d_bw_dflt / d_lat_dflt; the diagonal is copied from the
 * defaults. */
int est_links(const void* d_state, int32_t n_dev, const int64_t* d_bw_dflt, const int64_t* d_lat_dflt,
              int64_t* d_bw, int64_t* d_lat, gmg_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* GMGEST_H */
