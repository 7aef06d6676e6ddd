/*
 * Oracle (test infrastructure only): calibration statistics (App. A.3).
 *
 *  omega_i = E_cal[g_{t,i}^2], g_t = A_t^T q_t            (Sec. 4.1)
 *  ell_u   = E_cal[log r_{t,u}], r = alpha (GDN) or d_i (KDA) (Eq. calibration_lifetime)
 *  d_u(b)  = mean over sampled reference states of the per-element squared
 *            reconstruction error of the unit at width b: weighted by w_i^2
 *            for a GDN head (Eq. qwen_calibration_distortion), unweighted per
 *            KDA key row (Eq. kda_calibration_distortion).
 * A candidate reconstruction quantizes the whole head at the uniform width b
 * with the dual-axis codec; FP16 pivot rows (when given) are kept in FP16 and
 * left out of the shared column fit (App. A.3, App. C.2). The last column of
 * each distortion row is the FP16 reconstruction error.
 * These functions return sums; the caller divides by the sample counts.
 */
#include <math.h>
#include <stdlib.h>
#include <omp.h>
#include "oracle.h"

int or_num_threads(void) { return omp_get_max_threads(); }

void or_calib_observe(int n, int Hk, int Hv, int gate_per_row, const float *q,
                      const float *k, const float *beta, const float *gate,
                      double *omega_sum, double *logret_sum)
{
    int grp = Hv / Hk;
#pragma omp parallel for schedule(static)
    for (int h = 0; h < Hv; h++) {
        int hk = h / grp;
        for (int b = 0; b < n; b++) {
            const float *g = gate_per_row ? gate + ((size_t)b * Hv + h) * OR_D
                                          : gate + (size_t)b * Hv + h;
            double gi[OR_D];
            or_row_impact(q + ((size_t)b * Hk + hk) * OR_D, k + ((size_t)b * Hk + hk) * OR_D,
                          beta[(size_t)b * Hv + h], g, gate_per_row, gi);
            for (int i = 0; i < OR_D; i++)
                omega_sum[(size_t)h * OR_D + i] += gi[i] * gi[i];
            if (gate_per_row)
                for (int i = 0; i < OR_D; i++)
                    logret_sum[(size_t)h * OR_D + i] += log((double)g[i]);
            else
                logret_sum[h] += log((double)g[0]);
        }
    }
}

void or_calib_distortion(int n, int Hv, int unit_kind, const float *states, const float *w_layer,
                         int n_cand, const int *cands, const uint8_t *pivot_rows_layer,
                         int fit_iters, double *acc)
{
#pragma omp parallel for schedule(dynamic)
    for (int h = 0; h < Hv; h++) {
        const float *w = w_layer + (size_t)h * OR_D;
        uint8_t *page = malloc((size_t)OR_D * 256 + 512);
        double *R = malloc(sizeof(double) * OR_N);
        for (int s = 0; s < n; s++) {
            const float *S = states + ((size_t)s * Hv + h) * OR_N;
            for (int k = 0; k <= n_cand; k++) {
                int8_t rb[OR_D];
                for (int i = 0; i < OR_D; i++) {
                    int piv = (k == n_cand) || (unit_kind == OR_UNIT_ROW && pivot_rows_layer &&
                                                pivot_rows_layer[(size_t)h * OR_D + i]);
                    rb[i] = piv ? OR_PIVOT_BITS : (int8_t)cands[k];
                }
                if (k == n_cand && unit_kind == OR_UNIT_HEAD) {
                    for (int t = 0; t < OR_N; t++)
                        R[t] = or_fp16_round(S[t]);
                } else {
                    or_encode_head(S, unit_kind, rb, w, fit_iters, page);
                    or_decode_head(page, unit_kind, rb, R);
                }
                if (unit_kind == OR_UNIT_HEAD) {
                    double e = 0.0;
                    for (int i = 0; i < OR_D; i++) {
                        double w2 = (double)w[i] * (double)w[i], ei = 0.0;
                        for (int j = 0; j < OR_D; j++) {
                            double d = R[i * OR_D + j] - (double)S[i * OR_D + j];
                            ei += d * d;
                        }
                        e += w2 * ei;
                    }
                    acc[(size_t)h * (n_cand + 1) + k] += e / OR_N;
                } else {
                    for (int i = 0; i < OR_D; i++) {
                        double ei = 0.0;
                        for (int j = 0; j < OR_D; j++) {
                            double d = R[i * OR_D + j] - (double)S[i * OR_D + j];
                            ei += d * d;
                        }
                        acc[((size_t)h * OR_D + i) * (n_cand + 1) + k] += ei / OR_D;
                    }
                }
            }
        }
        free(page);
        free(R);
    }
}
