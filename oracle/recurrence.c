/*
 * Oracle (test infrastructure only): the gated Delta rule with an FP32 state.
 *
 * Eq. delta_update (Sec. 2.1):
 *   S_t = D_t S_{t-1} + beta_t k_t (v_t^T - k_t^T D_t S_{t-1}),   y_t = S_t^T q_t
 * with D_t = alpha_t I (GDN, scalar gate) or diag(d_t) (KDA, channel gate).
 * The state is kept in FP32 between steps, as in the FP32-state serving
 * baseline (Sec. 5.1); every step is evaluated in fp64 and rounded once.
 */
#include <math.h>
#include <stdlib.h>
#include <string.h>
#include "oracle.h"

/* One step of one head. S: [128][128] fp32 (in/out); gate: 1 value (scalar) or
 * 128 values (per key channel); y: [128] out. */
void or_delta_step_f32(float *S, const float *q, const float *k, const float *v,
                       float beta, const float *gate, int gate_per_row, float *y)
{
    double *P = malloc(sizeof(double) * OR_N);
    double u[OR_D];
    for (int i = 0; i < OR_D; i++) {
        double d = gate_per_row ? gate[i] : gate[0];
        for (int j = 0; j < OR_D; j++)
            P[i * OR_D + j] = d * (double)S[i * OR_D + j];        /* retained state D S */
    }
    for (int j = 0; j < OR_D; j++) {                              /* retrieval k^T D S */
        double acc = 0.0;
        for (int i = 0; i < OR_D; i++)
            acc += (double)k[i] * P[i * OR_D + j];
        u[j] = acc;
    }
    for (int i = 0; i < OR_D; i++)                                /* Delta write */
        for (int j = 0; j < OR_D; j++)
            S[i * OR_D + j] = (float)(P[i * OR_D + j] +
                                      (double)beta * (double)k[i] * ((double)v[j] - u[j]));
    for (int j = 0; j < OR_D; j++) {                              /* readout S^T q */
        double acc = 0.0;
        for (int i = 0; i < OR_D; i++)
            acc += (double)q[i] * (double)S[i * OR_D + j];
        y[j] = (float)acc;
    }
    free(P);
}

/* A batch of heads: S [n][Hv][128][128]; q, k [n][Hk][128]; v [n][Hv][128];
 * beta [n][Hv]; gate [n][Hv] or [n][Hv][128]; y [n][Hv][128]. Value head h
 * reads key head h / (Hv / Hk). */
void or_delta_batch_f32(int n, int Hk, int Hv, int gate_per_row, float *S,
                        const float *q, const float *k, const float *v,
                        const float *beta, const float *gate, float *y)
{
    int grp = Hv / Hk;
#pragma omp parallel for collapse(2) schedule(dynamic)
    for (int b = 0; b < n; b++)
        for (int h = 0; h < Hv; h++) {
            int hk = h / grp;
            const float *g = gate_per_row ? gate + ((size_t)b * Hv + h) * OR_D
                                          : gate + (size_t)b * Hv + h;
            or_delta_step_f32(S + ((size_t)b * Hv + h) * OR_N,
                              q + ((size_t)b * Hk + hk) * OR_D, k + ((size_t)b * Hk + hk) * OR_D,
                              v + ((size_t)b * Hv + h) * OR_D, beta[(size_t)b * Hv + h], g,
                              gate_per_row, y + ((size_t)b * Hv + h) * OR_D);
        }
}

/* The exact-read step of the feedback experiment (App. B.1): only the state
 * inside the Delta residual is replaced by the reference state S_ref,
 *   S_t = D_t S_{t-1} + beta_t k_t (v_t^T - k_t^T D_t S_ref_{t-1}),
 * so that S_t - S_ref_t = D_t (S_{t-1} - S_ref_{t-1}). S is updated in place;
 * S_ref is only read; y = S_t^T q_t. */
void or_delta_step_read_f32(float *S, const float *Sref, const float *q, const float *k,
                            const float *v, float beta, const float *gate, int gate_per_row,
                            float *y)
{
    double u[OR_D];
    for (int j = 0; j < OR_D; j++) {                              /* k^T D S_ref */
        double acc = 0.0;
        for (int i = 0; i < OR_D; i++) {
            double d = gate_per_row ? gate[i] : gate[0];
            acc += (double)k[i] * (d * (double)Sref[i * OR_D + j]);
        }
        u[j] = acc;
    }
    for (int i = 0; i < OR_D; i++) {
        double d = gate_per_row ? gate[i] : gate[0];
        for (int j = 0; j < OR_D; j++)
            S[i * OR_D + j] = (float)(d * (double)S[i * OR_D + j] +
                                      (double)beta * (double)k[i] * ((double)v[j] - u[j]));
    }
    for (int j = 0; j < OR_D; j++) {
        double acc = 0.0;
        for (int i = 0; i < OR_D; i++)
            acc += (double)q[i] * (double)S[i * OR_D + j];
        y[j] = (float)acc;
    }
}

/* Batch form of or_delta_step_read_f32 with the layout of or_delta_batch_f32;
 * Sref has the layout of S. */
void or_delta_batch_read_f32(int n, int Hk, int Hv, int gate_per_row, float *S, const float *Sref,
                             const float *q, const float *k, const float *v,
                             const float *beta, const float *gate, float *y)
{
    int grp = Hv / Hk;
#pragma omp parallel for collapse(2) schedule(dynamic)
    for (int b = 0; b < n; b++)
        for (int h = 0; h < Hv; h++) {
            int hk = h / grp;
            size_t o = ((size_t)b * Hv + h) * OR_N;
            const float *g = gate_per_row ? gate + ((size_t)b * Hv + h) * OR_D
                                          : gate + (size_t)b * Hv + h;
            or_delta_step_read_f32(S + o, Sref + o, q + ((size_t)b * Hk + hk) * OR_D,
                                   k + ((size_t)b * Hk + hk) * OR_D,
                                   v + ((size_t)b * Hv + h) * OR_D, beta[(size_t)b * Hv + h], g,
                                   gate_per_row, y + ((size_t)b * Hv + h) * OR_D);
        }
}

/* Row-impact vector g_t = A_t^T q_t (Sec. 4.1), closed form of Eq.
 * kda_sensitivity: g_i = d_i [q_i - beta k_i (k^T q)]. */
void or_row_impact(const float *q, const float *k, float beta, const float *gate,
                   int gate_per_row, double *g)
{
    double kq = 0.0;
    for (int i = 0; i < OR_D; i++)
        kq += (double)k[i] * (double)q[i];
    for (int i = 0; i < OR_D; i++) {
        double d = gate_per_row ? gate[i] : gate[0];
        g[i] = d * ((double)q[i] - (double)beta * (double)k[i] * kq);
    }
}

/* The same vector from its definition: build A_t = (I - beta k k^T) D_t as a
 * dense matrix (Eq. delta_affine) and multiply its transpose by q. */
void or_row_impact_dense(const float *q, const float *k, float beta, const float *gate,
                         int gate_per_row, double *g)
{
    double *A = malloc(sizeof(double) * OR_N);
    for (int i = 0; i < OR_D; i++)
        for (int j = 0; j < OR_D; j++) {
            double dj = gate_per_row ? gate[j] : gate[0];
            double Pij = (i == j ? 1.0 : 0.0) - (double)beta * (double)k[i] * (double)k[j];
            A[i * OR_D + j] = Pij * dj;                    /* (P D)_{ij} = P_ij d_j */
        }
    for (int j = 0; j < OR_D; j++) {                       /* (A^T q)_j = sum_i A_ij q_i */
        double acc = 0.0;
        for (int i = 0; i < OR_D; i++)
            acc += A[i * OR_D + j] * (double)q[i];
        g[j] = acc;
    }
    free(A);
}
