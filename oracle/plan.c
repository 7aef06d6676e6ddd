/*
 * Oracle (test infrastructure only): the offline plan — row-impact factors,
 * lifetime weights, FP16 pivots, Lifetime-aware Bit Allocation and the packed
 * page layout (Sec. 3.2, Sec. 4.3 footnote, App. A.3, App. C.1-C.2, App. D).
 *
 * Readings where the paper is silent (listed in the design notes):
 *  - omega is floored at 1e-30 before its logarithm;
 *  - the multiple-choice DP works in units of 2 bits per element (all
 *    candidates are even) and resolves exact ties to the wider code;
 *  - the Lagrangian picks the narrower code on ties, bisects 60 times for the
 *    smallest feasible multiplier, then "repairs" by greedily spending the
 *    leftover budget on the upgrade with the largest objective reduction per
 *    bit (ties: lower unit index, then narrower code);
 *  - GDN pivots rank by L_u d_u(b_u) at the pivot-free allocation ("residual
 *    allocation risk"); KDA pivots rank by L_u (d_u(nominal) - d_u(FP16))
 *    ("lifetime-weighted reduction from integer to FP16 error"); ties go to the
 *    lower unit index;
 *  - pivots consume 8 bits per element of the nominal budget (App. D).
 */
#include <math.h>
#include <stdlib.h>
#include <string.h>
#include "oracle.h"

/* Footnote of Sec. 4.3 / Eq. kda_precond: w_i = omega_i^(gamma/2) /
 * GM_k(omega_k^(gamma/2)), gamma = 0.25, per head (n_heads x 128 values). */
void or_row_weights(int n_heads, const float *omega, float *w)
{
    const double half_gamma = 0.125;
    for (int h = 0; h < n_heads; h++) {
        double lw[OR_D], mean = 0.0;
        for (int i = 0; i < OR_D; i++) {
            double om = omega[(size_t)h * OR_D + i];
            if (!(om > 1e-30))
                om = 1e-30;
            lw[i] = half_gamma * log(om);
            mean += lw[i];
        }
        mean /= OR_D;
        for (int i = 0; i < OR_D; i++)
            w[(size_t)h * OR_D + i] = (float)exp(lw[i] - mean);
    }
}

/* Lifetime weight L_u = sum_{j=0}^{H-1} exp(2 j ell_u) (Eq. calibration_lifetime). */
double or_lifetime_weight(double ell, int H)
{
    double L = 0.0;
    for (int j = 0; j < H; j++)
        L += exp(2.0 * j * ell);
    return L;
}

/* Multiple-choice DP (App. C.2): minimise sum_u cost[u][k_u] subject to
 * sum_u cands[k_u]/2 <= capacity. Returns 0, or -1 if infeasible. */
int or_allocate_dp(int n_units, int n_cand, const int *cands, long long capacity,
                   const double *cost, int8_t *choice)
{
    if (capacity < 0)
        return -1;
    long long C = capacity;
    int order[8];
    for (int k = 0; k < n_cand; k++)
        order[k] = k;
    for (int a = 0; a < n_cand; a++)          /* descending width: ties keep the wider code */
        for (int b = a + 1; b < n_cand; b++)
            if (cands[order[b]] > cands[order[a]]) {
                int t = order[a]; order[a] = order[b]; order[b] = t;
            }
    double *Fn = malloc(sizeof(double) * (C + 1));   /* F_{u+1} */
    double *Fc = malloc(sizeof(double) * (C + 1));   /* F_u */
    int8_t *ch = malloc((size_t)n_units * (C + 1));
    for (long long c = 0; c <= C; c++)
        Fn[c] = 0.0;
    for (int u = n_units - 1; u >= 0; u--) {
        for (long long c = 0; c <= C; c++) {
            double best = INFINITY;
            int bk = -1;
            for (int t = 0; t < n_cand; t++) {
                int k = order[t];
                long long a = cands[k] / 2;
                if (a > c)
                    continue;
                double val = cost[(size_t)u * n_cand + k] + Fn[c - a];
                if (val < best) {
                    best = val;
                    bk = k;
                }
            }
            Fc[c] = best;
            ch[(size_t)u * (C + 1) + c] = (int8_t)bk;
        }
        double *t = Fn; Fn = Fc; Fc = t;
    }
    int ok = isfinite(Fn[C]) ? 0 : -1;
    long long c = C;
    for (int u = 0; u < n_units && ok == 0; u++) {
        int k = ch[(size_t)u * (C + 1) + c];
        if (k < 0) { ok = -1; break; }
        choice[u] = (int8_t)k;
        c -= cands[k] / 2;
    }
    free(Fn); free(Fc); free(ch);
    return ok;
}

static long long lagr_pick(int n_units, int n_cand, const int *asc, const int *cands,
                           const double *cost, double lam, int8_t *choice)
{
    long long bits = 0;
    for (int u = 0; u < n_units; u++) {
        double best = INFINITY;
        int bk = asc[0];
        for (int t = 0; t < n_cand; t++) {          /* ascending width: ties keep the narrower */
            int k = asc[t];
            double val = cost[(size_t)u * n_cand + k] + lam * cands[k];
            if (val < best) {
                best = val;
                bk = k;
            }
        }
        choice[u] = (int8_t)bk;
        bits += cands[bk];
    }
    return bits;
}

static void ascending(int n_cand, const int *cands, int *asc)
{
    for (int k = 0; k < n_cand; k++)
        asc[k] = k;
    for (int a = 0; a < n_cand; a++)
        for (int b = a + 1; b < n_cand; b++)
            if (cands[asc[b]] < cands[asc[a]]) {
                int t = asc[a]; asc[a] = asc[b]; asc[b] = t;
            }
}

/* The shared multiplier of the Lagrangian relaxation (App. C.2): 0 if the
 * unconstrained choice fits the budget, else the smallest lambda (bisection,
 * 60 steps in fp64) whose per-unit choices argmin_k cost[u][k] + lambda cands[k]
 * (ties to the narrower code) fit. Returns -1 if no choice fits. */
double or_lagrangian_multiplier(int n_units, int n_cand, const int *cands, long long budget,
                                const double *cost)
{
    int asc[8];
    ascending(n_cand, cands, asc);
    if ((long long)cands[asc[0]] * n_units > budget)
        return -1.0;
    int8_t *choice = malloc((size_t)(n_units > 0 ? n_units : 1));
    double lam = 0.0;
    if (lagr_pick(n_units, n_cand, asc, cands, cost, 0.0, choice) > budget) {
        double lo = 0.0, hi = 1.0;
        int guard = 0;
        while (lagr_pick(n_units, n_cand, asc, cands, cost, hi, choice) > budget) {
            hi *= 2.0;
            if (++guard > 2000 || !isfinite(hi)) {
                free(choice);
                return -1.0;
            }
        }
        for (int it = 0; it < 60; it++) {
            double mid = 0.5 * (lo + hi);
            if (lagr_pick(n_units, n_cand, asc, cands, cost, mid, choice) <= budget)
                hi = mid;
            else
                lo = mid;
        }
        lam = hi;
    }
    free(choice);
    return lam;
}

/* Lagrangian allocation with a shared multiplier and a discrete repair
 * (App. C.2): minimise sum_u cost[u][k_u] s.t. sum_u cands[k_u] <= budget. */
int or_allocate_lagrangian(int n_units, int n_cand, const int *cands, long long budget,
                           const double *cost, int8_t *choice)
{
    int asc[8];
    ascending(n_cand, cands, asc);
    double lam = or_lagrangian_multiplier(n_units, n_cand, cands, budget, cost);
    if (lam < 0.0)
        return -1;
    long long bits = lagr_pick(n_units, n_cand, asc, cands, cost, lam, choice);
    long long slack = budget - bits;
    for (;;) {
        int bu = -1, bk = -1;
        double best_ratio = -1.0;
        for (int u = 0; u < n_units; u++) {
            int cur = choice[u];
            for (int t = 0; t < n_cand; t++) {
                int k = asc[t];
                long long db = cands[k] - cands[cur];
                if (db <= 0 || db > slack)
                    continue;
                double gain = cost[(size_t)u * n_cand + cur] - cost[(size_t)u * n_cand + k];
                if (gain < 0.0)
                    continue;
                double ratio = gain / (double)db;
                if (ratio > best_ratio) {
                    best_ratio = ratio;
                    bu = u;
                    bk = k;
                }
            }
        }
        if (bu < 0)
            break;
        slack -= cands[bk] - cands[choice[bu]];
        choice[bu] = (int8_t)bk;
    }
    return 0;
}

static int cand_index(int n_cand, const int *cands, int b)
{
    for (int k = 0; k < n_cand; k++)
        if (cands[k] == b)
            return k;
    return -1;
}

/* FP16 pivots (Sec. 3.2; Table `config`; App. C.2). dist: [n_units][n_cand + 1],
 * the last column being the FP16 reconstruction distortion. */
int or_select_pivots(int unit_kind, int n_units, int n_cand, const int *cands, int nominal,
                     const double *L, const double *dist, int n_pivots, uint8_t *pivot)
{
    memset(pivot, 0, (size_t)n_units);
    if (n_pivots <= 0)
        return 0;
    if (n_pivots > n_units)
        return -1;
    double *risk = malloc(sizeof(double) * n_units);
    if (unit_kind == OR_UNIT_HEAD) {
        double *cost = malloc(sizeof(double) * (size_t)n_units * n_cand);
        int8_t *ch = malloc((size_t)n_units);
        for (int u = 0; u < n_units; u++)
            for (int k = 0; k < n_cand; k++)
                cost[(size_t)u * n_cand + k] = L[u] * dist[(size_t)u * (n_cand + 1) + k];
        int rc = or_allocate_dp(n_units, n_cand, cands, (long long)nominal / 2 * n_units, cost, ch);
        if (rc == 0)
            for (int u = 0; u < n_units; u++)
                risk[u] = L[u] * dist[(size_t)u * (n_cand + 1) + ch[u]];
        free(cost);
        free(ch);
        if (rc != 0) { free(risk); return -1; }
    } else {
        int kn = cand_index(n_cand, cands, nominal);
        if (kn < 0) { free(risk); return -1; }
        for (int u = 0; u < n_units; u++)
            risk[u] = L[u] * (dist[(size_t)u * (n_cand + 1) + kn] -
                              dist[(size_t)u * (n_cand + 1) + n_cand]);
    }
    for (int p = 0; p < n_pivots; p++) {       /* highest risk first, lower index on ties */
        int best = -1;
        for (int u = 0; u < n_units; u++)
            if (!pivot[u] && (best < 0 || risk[u] > risk[best]))
                best = u;
        pivot[best] = 1;
    }
    free(risk);
    return 0;
}

/* Bit widths per unit: cands[k] for integer units, 16 for pivots. Pivots count
 * as 8-bit replacements against the nominal budget (App. D). */
int or_allocate(int unit_kind, int n_units, int n_cand, const int *cands, int nominal,
                const double *L, const double *dist, const uint8_t *pivot, int8_t *bits)
{
    int n_piv = 0;
    for (int u = 0; u < n_units; u++)
        n_piv += pivot[u] ? 1 : 0;
    int m = n_units - n_piv;
    int *idx = malloc(sizeof(int) * (m > 0 ? m : 1));
    double *cost = malloc(sizeof(double) * (size_t)(m > 0 ? m : 1) * n_cand);
    int8_t *ch = malloc((size_t)(m > 0 ? m : 1));
    int t = 0;
    for (int u = 0; u < n_units; u++)
        if (!pivot[u]) {
            idx[t] = u;
            for (int k = 0; k < n_cand; k++)
                cost[(size_t)t * n_cand + k] = L[u] * dist[(size_t)u * (n_cand + 1) + k];
            t++;
        }
    int rc;
    if (unit_kind == OR_UNIT_HEAD)
        rc = or_allocate_dp(m, n_cand, cands, (long long)nominal / 2 * n_units - 4LL * n_piv,
                            cost, ch);
    else
        rc = or_allocate_lagrangian(m, n_cand, cands, (long long)nominal * n_units - 8LL * n_piv,
                                    cost, ch);
    if (rc == 0) {
        for (int u = 0; u < n_units; u++)
            bits[u] = OR_PIVOT_BITS;
        for (int s = 0; s < m; s++)
            bits[idx[s]] = (int8_t)cands[ch[s]];
    }
    free(idx); free(cost); free(ch);
    return rc;
}

/* Packed slot page: (layer, head) segments in order, each the size of its head
 * page; slot stride rounded up to 256 bytes. */
int or_layout(int unit_kind, int n_layers, int Hv, const int8_t *unit_bits,
              uint64_t *head_off, uint32_t *head_bytes, uint64_t *slot_stride)
{
    uint64_t off = 0;
    for (int lh = 0; lh < n_layers * Hv; lh++) {
        int8_t rb[OR_D];
        for (int i = 0; i < OR_D; i++)
            rb[i] = unit_kind == OR_UNIT_HEAD ? unit_bits[lh] : unit_bits[(size_t)lh * OR_D + i];
        size_t n = or_head_bytes(unit_kind, rb);
        head_off[lh] = off;
        head_bytes[lh] = (uint32_t)n;
        off += n;
    }
    *slot_stride = (off + 255) / 256 * 256;
    return 0;
}
