/*
 * Oracle (test infrastructure only): the compressed state of one head and the
 * persistent decode step (App. C.3, "One persistent STEPQuant decode step").
 *
 * Representation (Sec. 4.3): X_hat_ij = r_i c_j z_ij with FP16 row factors r,
 * FP16 column factors c and integer codes. Head units (GDN) use z = q with
 * |q| <= 2^(b-1)-1 (Eq. uniform_quantization). Row units (KDA) use the
 * normalised codebook z = 2^(8-b_i) q (App. C.1), so rows of different widths
 * share one column vector. FP16 pivots store X directly (Sec. 3.2).
 *
 * Readings where the paper is silent (listed in the design notes):
 *  - r_i = fp16(clamp(m_i^(1/2) w_i^(-1/2), 2^-14, 65504)) with m_i the exact
 *    mean of |X_ij| over the row, the FP16 clamp of the baseline's scale storage
 *    (App. B.5);
 *  - the column fit starts from the clip-free value
 *    c0_j = max_{i in I} |X_ij| / (r_i zs_i qmax_i), then applies `fit_iters`
 *    fixed-code updates c_j = sum w_i^2 v_ij X_ij / sum w_i^2 v_ij^2 (App. C.1),
 *    a zero denominator keeping the current iterate, floor 2^-14, cap 65504;
 *    the iterate is kept exactly (fp64) and rounded once, to FP16, for storage;
 *  - "quantize each scaled entry X_ij / (r_i c_j) to the nearest representable
 *    level" (Sec. 4.3) is taken literally: the nearest integer, ties to even, of
 *    the exact quotient X_ij / (r_i zs_i c_j), then the clip to +-qmax_i. The
 *    paper fixes no precision for this decision, so the oracle takes it on the
 *    exact value; a kernel that evaluates the quotient in fp32 disagrees only
 *    where it lies within a few fp32 ulps of a half-integer;
 *  - codes are stored offset-binary u = q + 2^(b-1), LSB-first per row.
 *
 * Page layout of one head (all pieces 16-byte multiples):
 *   integer head unit: r[128] fp16 | c[128] fp16 | codes: the 16 codes of one
 *                      band of rows (16g..16g+15) in one column form a chunk of
 *                      2b bytes; the four chunks of columns 4t..4t+3 in band g
 *                      form one stream of 2b words, stored as 16-byte pieces
 *                      interleaved over the 32 (band, column quad) streams of
 *                      each group of 16 columns (see bit_addr)
 *   pivot head unit:   the same arrangement of fp16 values (b = 16), no scales
 *   row-unit head:     r[128] fp16 | c[128] fp16 | then the rows, each 16 b_i
 *                      bytes with the codes of columns 0..127 (b_i = 16 marks
 *                      an FP16 pivot row, 256 bytes), stored by decreasing
 *                      width, rows of equal width in index order
 */
#include <math.h>
#include <stdlib.h>
#include <string.h>
#include "oracle.h"

#define F16_MIN_NORMAL (1.0 / 16384.0)   /* 2^-14 */
#define F16_MAX 65504.0

static int is_pivot_head(int unit_kind, const int8_t *rb)
{
    return unit_kind == OR_UNIT_HEAD && rb[0] == OR_PIVOT_BITS;
}

static int qmax_of(int b) { return (1 << (b - 1)) - 1; }

/* codebook spacing: 2^(8-b) for the normalised row-unit codebook, 1 otherwise */
static int zs_of(int unit_kind, int b) { return unit_kind == OR_UNIT_ROW ? 1 << (8 - b) : 1; }

static double clampd(double x, double lo, double hi) { return x < lo ? lo : (x > hi ? hi : x); }

/* fp32 product of two fp32 values (exact in fp64, rounded once) */
static float mul32(float a, float b) { return (float)((double)a * (double)b); }

/* Nearest integer, ties to even, of the exact quotient x / d (d > 0), x an fp32
 * value and d a product of FP16 values and a power of two. The rounded fp64
 * quotient gives a candidate n; the remainder e = x - n d is exact in fp64
 * whenever |n| <= 2^8 (n d has at most 30 significant bits and lies within d/2
 * of x), which covers every code that is not clipped, and it decides the two
 * cases where the rounded quotient lands on the wrong side of a half-integer. */
static double rne_div(double x, double d)
{
    double n = rint(x / d);
    double e = x - n * d;
    if (2.0 * e > d)
        return n + 1.0;
    if (-2.0 * e > d)
        return n - 1.0;
    if (2.0 * fabs(e) == d && fmod(n, 2.0) != 0.0)            /* a tie: the even neighbour */
        return e > 0.0 ? n + 1.0 : n - 1.0;
    return n;
}

/* The level of X_ij at the row scale r_i zs_i and column scale c_j, clipped to
 * +-qmax (Eq. uniform_quantization with the dual-axis scale of Sec. 4.3). */
static double level(float x, double r_zs, double c, int qm)
{
    return clampd(rne_div((double)x, r_zs * c), -qm, qm);
}

size_t or_head_bytes(int unit_kind, const int8_t *rb)
{
    if (is_pivot_head(unit_kind, rb))
        return (size_t)OR_D * 256;
    size_t n = 512;
    for (int i = 0; i < OR_D; i++)
        n += 16 * (size_t)rb[i];
    return n;
}

static void put_u16(uint8_t *p, uint16_t v) { p[0] = v & 0xFF; p[1] = v >> 8; }
static uint16_t get_u16(const uint8_t *p) { return (uint16_t)(p[0] | (p[1] << 8)); }

/* Write code u (b bits) at bit position pos of a little-endian bit stream. */
static void put_bits(uint8_t *row, int pos, int b, unsigned u)
{
    for (int t = 0; t < b; t++) {
        int p = pos + t;
        if ((u >> t) & 1u)
            row[p >> 3] |= (uint8_t)(1u << (p & 7));
        else
            row[p >> 3] &= (uint8_t)~(1u << (p & 7));
    }
}

static unsigned get_bits(const uint8_t *row, int pos, int b)
{
    unsigned u = 0;
    for (int t = 0; t < b; t++) {
        int p = pos + t;
        u |= (unsigned)((row[p >> 3] >> (p & 7)) & 1u) << t;
    }
    return u;
}

/* Byte offset of the payload of row i of a row-unit segment: rows of larger
 * width first, then earlier rows of width b_i (App. D fixes only the sizes). */
static void row_offsets(const int8_t *rb, size_t *off)
{
    for (int i = 0; i < OR_D; i++) {
        int b = rb[i];
        off[i] = 512;
        for (int r = 0; r < OR_D; r++)
            if (rb[r] > b || (rb[r] == b && r < i))
                off[i] += 16 * (size_t)rb[r];
    }
}

/* Byte offset of bit t (0 <= t < b_i) of element (i, j) in a head segment, and
 * that bit's position in the byte. row_off: row_offsets() for row units. */
static size_t bit_addr(int unit_kind, const int8_t *rb, const size_t *row_off, int i, int j, int t,
                       int *bit)
{
    int b = rb[i];
    if (unit_kind == OR_UNIT_HEAD) {
        /* The 16 codes of band g = i / 16 in column j form a chunk of 2b bytes,
         * LSB-first. Column group w = j / 16 and lane l = 8 ((j / 4) % 4) + g own
         * four chunks (columns 4 (j / 4) + 0..3), one stream of 2b 32-bit words;
         * its 16-byte piece k sits at w * 256 b + k * 512 + 16 l. */
        size_t base = is_pivot_head(unit_kind, rb) ? 0 : 512;
        int w = j / 16, l = 8 * ((j / 4) % 4) + i / 16;
        int L = (j % 4) * 16 * b + (i % 16) * b + t;              /* bit of the lane's stream */
        int word = L / 32;
        *bit = L % 8;
        return base + (size_t)w * 256 * b + (size_t)(word / 4) * 512 + 16 * (size_t)l +
               4 * (size_t)(word % 4) + (size_t)(L % 32) / 8;
    }
    *bit = (j * b + t) % 8;
    return row_off[i] + (size_t)(j * b + t) / 8;
}

/* Element (i, j) of a head segment as a b_i-bit value: an offset-binary code,
 * or the binary16 bits of an FP16 pivot (b_i = 16). */
static void put_code(uint8_t *page, int unit_kind, const int8_t *rb, const size_t *row_off, int i,
                     int j, unsigned u)
{
    for (int t = 0; t < rb[i]; t++) {
        int bit;
        uint8_t *p = page + bit_addr(unit_kind, rb, row_off, i, j, t, &bit);
        if ((u >> t) & 1u)
            *p |= (uint8_t)(1u << bit);
        else
            *p &= (uint8_t)~(1u << bit);
    }
}

static unsigned get_code(const uint8_t *page, int unit_kind, const int8_t *rb, const size_t *row_off,
                         int i, int j)
{
    unsigned u = 0;
    for (int t = 0; t < rb[i]; t++) {
        int bit;
        const uint8_t *p = page + bit_addr(unit_kind, rb, row_off, i, j, t, &bit);
        u |= (unsigned)((*p >> bit) & 1u) << t;
    }
    return u;
}

/* Unpack a head page into scales, integer codes and pivot values. For a
 * pivot head r and c are zero and every row is in `piv`. */
void or_unpack_head(const uint8_t *page, int unit_kind, const int8_t *rb,
                    uint16_t *r, uint16_t *c, int8_t *codes, uint16_t *piv)
{
    int ph = is_pivot_head(unit_kind, rb);
    size_t off[OR_D];
    row_offsets(rb, off);
    for (int i = 0; i < OR_D; i++) {
        r[i] = ph ? 0 : get_u16(page + 2 * i);
        c[i] = ph ? 0 : get_u16(page + 256 + 2 * i);
    }
    for (int i = 0; i < OR_D; i++) {
        int b = rb[i];
        for (int j = 0; j < OR_D; j++) {
            unsigned u = get_code(page, unit_kind, rb, off, i, j);
            if (b == OR_PIVOT_BITS) {
                piv[i * OR_D + j] = (uint16_t)u;
                codes[i * OR_D + j] = 0;
            } else {
                codes[i * OR_D + j] = (int8_t)((int)u - (1 << (b - 1)));
                piv[i * OR_D + j] = 0;
            }
        }
    }
}

/* Reconstruction (App. C.3 step 1): S_ij = r_i c_j z_ij, or the FP16 value for
 * pivot units. Exact in fp64. */
void or_decode_head(const uint8_t *page, int unit_kind, const int8_t *rb, double *S)
{
    uint16_t r[OR_D], c[OR_D];
    int8_t *codes = malloc(OR_N);
    uint16_t *piv = malloc(sizeof(uint16_t) * OR_N);
    or_unpack_head(page, unit_kind, rb, r, c, codes, piv);
    for (int i = 0; i < OR_D; i++) {
        int b = rb[i];
        for (int j = 0; j < OR_D; j++) {
            if (b == OR_PIVOT_BITS)
                S[i * OR_D + j] = or_fp16_decode(piv[i * OR_D + j]);
            else
                S[i * OR_D + j] = or_fp16_decode(r[i]) * or_fp16_decode(c[j]) *
                                  (double)zs_of(unit_kind, b) * (double)codes[i * OR_D + j];
        }
    }
    free(codes);
    free(piv);
}

void or_decode_head_f32(const uint8_t *page, int unit_kind, const int8_t *rb, float *S)
{
    double *D = malloc(sizeof(double) * OR_N);
    or_decode_head(page, unit_kind, rb, D);
    for (int t = 0; t < OR_N; t++)
        S[t] = (float)D[t];
    free(D);
}

/* Key-Row-Aware Dual-axis Fitting of an updated tile X (fp32, row-major)
 * (Sec. 4.3; App. C.1; App. C.3 steps 4-5). Outputs the FP16 row factors r,
 * the final column iterate c (exact, before its FP16 rounding) and the codes of
 * the last fixed-code update (for inspection). */
static void fit_head(const float *X, int unit_kind, const int8_t *rb, const float *w,
                     int fit_iters, double *r, double *c, int8_t *z_last)
{
    int in_fit[OR_D];         /* non-pivot integer rows: the set I */
    double rz[OR_D];          /* r_i zs_i */
    for (int i = 0; i < OR_D; i++) {
        int b = rb[i];
        in_fit[i] = (b != OR_PIVOT_BITS);
        if (!in_fit[i]) {
            r[i] = rz[i] = 0.0;
            continue;
        }
        /* Row factors: m_i = (1/d_v) sum_j |X_ij|, r_i = m_i^(1/2) w_i^(-1/2). */
        double s = 0.0;
        for (int j = 0; j < OR_D; j++)
            s += fabs((double)X[i * OR_D + j]);
        double m = s / OR_D;
        double t = sqrt(m) / sqrt((double)w[i]);
        r[i] = or_fp16_round(clampd(t, F16_MIN_NORMAL, F16_MAX));
        rz[i] = r[i] * (double)zs_of(unit_kind, b);
    }
    /* Column factors: clip-free start c0_j = max_{i in I} |X_ij| / (r_i zs_i qmax_i),
     * then fixed-code least-squares updates of
     * min_c sum_{i in I} w_i^2 (X_ij - r_i c_j z_ij)^2 (v_ij = r_i zs_i q_ij). */
    for (int j = 0; j < OR_D; j++) {
        double cmax = 0.0;
        for (int i = 0; i < OR_D; i++)
            if (in_fit[i]) {
                double a = fabs((double)X[i * OR_D + j]) / (rz[i] * qmax_of(rb[i]));
                if (a > cmax)
                    cmax = a;
            }
        c[j] = clampd(cmax, F16_MIN_NORMAL, F16_MAX);
    }
    if (z_last)
        for (int t = 0; t < OR_N; t++)
            z_last[t] = 0;
    for (int it = 0; it < fit_iters; it++) {
        for (int j = 0; j < OR_D; j++) {
            double num = 0.0, den = 0.0;
            for (int i = 0; i < OR_D; i++) {
                if (!in_fit[i])
                    continue;
                double qv = level(X[i * OR_D + j], rz[i], c[j], qmax_of(rb[i]));
                if (z_last)
                    z_last[i * OR_D + j] = (int8_t)qv;
                double v = rz[i] * qv;                                    /* v_ij = r_i z_ij */
                double w2 = (double)w[i] * (double)w[i];
                num += w2 * v * (double)X[i * OR_D + j];
                den += w2 * v * v;
            }
            if (den > 0.0)
                c[j] = clampd(num / den, F16_MIN_NORMAL, F16_MAX);
        }
    }
}

void or_fit_debug(const float *X, int unit_kind, const int8_t *rb, const float *w,
                  int fit_iters, double *r, double *c_iter, int8_t *z_last)
{
    fit_head(X, unit_kind, rb, w, fit_iters, r, c_iter, z_last);
}

/* Fit, then pack with the stored FP16 scales (App. C.3 step 6). */
void or_encode_head(const float *X, int unit_kind, const int8_t *rb, const float *w,
                    int fit_iters, uint8_t *page)
{
    size_t off[OR_D];
    row_offsets(rb, off);
    if (is_pivot_head(unit_kind, rb)) {             /* FP16 pivot head */
        for (int i = 0; i < OR_D; i++)
            for (int j = 0; j < OR_D; j++)
                put_code(page, unit_kind, rb, off, i, j, or_fp16_encode(or_fp16_round(X[i * OR_D + j])));
        return;
    }
    double r[OR_D], c[OR_D];
    fit_head(X, unit_kind, rb, w, fit_iters, r, c, NULL);
    /* Storage precision, then the final codes with the stored scales. */
    double c16[OR_D];
    for (int j = 0; j < OR_D; j++)
        c16[j] = or_fp16_round(c[j]);
    for (int i = 0; i < OR_D; i++) {
        put_u16(page + 2 * i, or_fp16_encode(r[i]));
        put_u16(page + 256 + 2 * i, or_fp16_encode(c16[i]));
    }
    for (int i = 0; i < OR_D; i++) {
        int b = rb[i];
        for (int j = 0; j < OR_D; j++) {
            if (b == OR_PIVOT_BITS) {
                put_code(page, unit_kind, rb, off, i, j, or_fp16_encode(or_fp16_round(X[i * OR_D + j])));
                continue;
            }
            double rz = r[i] * (double)zs_of(unit_kind, b);
            int qv = (int)level(X[i * OR_D + j], rz, c16[j], qmax_of(b));
            put_code(page, unit_kind, rb, off, i, j, (unsigned)(qv + (1 << (b - 1))));
        }
    }
}

/* One persistent decode step of one head (App. C.3 steps 1-7): reconstruct,
 * X = D S + beta k (v^T - k^T D S), y = X^T q, refit, requantize in place.
 * delta (optional, [128]): the residual v_j - u_j of the retrieval. */
void or_step_head(uint8_t *page, int unit_kind, const int8_t *rb, const float *w,
                  int fit_iters, const float *q, const float *k, const float *v,
                  float beta, const float *gate, int gate_per_row, float *y, double *delta)
{
    double *S = malloc(sizeof(double) * OR_N);
    float *X = malloc(sizeof(float) * OR_N);
    double u[OR_D];
    or_decode_head(page, unit_kind, rb, S);
    for (int i = 0; i < OR_D; i++) {
        double d = gate_per_row ? gate[i] : gate[0];
        for (int j = 0; j < OR_D; j++)
            S[i * OR_D + j] *= d;                              /* D S_hat */
    }
    for (int j = 0; j < OR_D; j++) {
        double acc = 0.0;
        for (int i = 0; i < OR_D; i++)
            acc += (double)k[i] * S[i * OR_D + j];
        u[j] = acc;
    }
    for (int i = 0; i < OR_D; i++)
        for (int j = 0; j < OR_D; j++)
            X[i * OR_D + j] = (float)(S[i * OR_D + j] +
                                      (double)beta * (double)k[i] * ((double)v[j] - u[j]));
    for (int j = 0; j < OR_D; j++) {                           /* readout before requantization */
        double acc = 0.0;
        for (int i = 0; i < OR_D; i++)
            acc += (double)q[i] * (double)X[i * OR_D + j];
        y[j] = (float)acc;
    }
    if (delta)                                                 /* v - k^T D S_hat, optional */
        for (int j = 0; j < OR_D; j++)
            delta[j] = (double)v[j] - u[j];
    or_encode_head(X, unit_kind, rb, w, fit_iters, page);
    free(S);
    free(X);
}

/* ---- uniform rowwise-absmax INT-b baseline ----
 * Every key row uses the scale s_i = absmax_i / qmax stored in FP16, clamped
 * to [2^-14, 65504], and nearest-integer codes in [-qmax, qmax] (App. B.5).
 * Page: s[128] fp16 | 128 rows x 16b bytes (offset-binary codes, LSB-first).
 * The code decision uses t = fp32(X * fp32(1/s_i)). */
size_t or_intb_head_bytes(int bits) { return 256 + (size_t)OR_D * 16 * bits; }

void or_intb_encode_head(const float *X, int bits, uint8_t *page)
{
    int qm = qmax_of(bits);
    for (int i = 0; i < OR_D; i++) {
        float amax = 0.0f;
        for (int j = 0; j < OR_D; j++)
            if (fabsf(X[i * OR_D + j]) > amax)
                amax = fabsf(X[i * OR_D + j]);
        float s = (float)((double)amax / qm);
        double s16 = or_fp16_round(clampd(s, F16_MIN_NORMAL, F16_MAX));
        float inv = (float)(1.0 / s16);
        put_u16(page + 2 * i, or_fp16_encode(s16));
        uint8_t *row = page + 256 + (size_t)i * 16 * bits;
        for (int j = 0; j < OR_D; j++) {
            float t = mul32(X[i * OR_D + j], inv);
            int qv = (int)clampd(rint((double)t), -qm, qm);
            put_bits(row, j * bits, bits, (unsigned)(qv + (1 << (bits - 1))));
        }
    }
}

void or_intb_decode_head(const uint8_t *page, int bits, double *S)
{
    for (int i = 0; i < OR_D; i++) {
        double s = or_fp16_decode(get_u16(page + 2 * i));
        const uint8_t *row = page + 256 + (size_t)i * 16 * bits;
        for (int j = 0; j < OR_D; j++)
            S[i * OR_D + j] = s * (double)((int)get_bits(row, j * bits, bits) - (1 << (bits - 1)));
    }
}

void or_intb_step_head(uint8_t *page, int bits, const float *q, const float *k, const float *v,
                       float beta, const float *gate, int gate_per_row, float *y)
{
    double *S = malloc(sizeof(double) * OR_N);
    float *X = malloc(sizeof(float) * OR_N);
    double u[OR_D];
    or_intb_decode_head(page, bits, S);
    for (int i = 0; i < OR_D; i++) {
        double d = gate_per_row ? gate[i] : gate[0];
        for (int j = 0; j < OR_D; j++)
            S[i * OR_D + j] *= d;
    }
    for (int j = 0; j < OR_D; j++) {
        double acc = 0.0;
        for (int i = 0; i < OR_D; i++)
            acc += (double)k[i] * S[i * OR_D + j];
        u[j] = acc;
    }
    for (int i = 0; i < OR_D; i++)
        for (int j = 0; j < OR_D; j++)
            X[i * OR_D + j] = (float)(S[i * OR_D + j] +
                                      (double)beta * (double)k[i] * ((double)v[j] - u[j]));
    for (int j = 0; j < OR_D; j++) {
        double acc = 0.0;
        for (int i = 0; i < OR_D; i++)
            acc += (double)q[i] * (double)X[i * OR_D + j];
        y[j] = (float)acc;
    }
    or_intb_encode_head(X, bits, page);
    free(S);
    free(X);
}

/* ---- "Temporal only" ablation codec (Sec. 5.4) ----
 * The plan's calibrated widths and FP16 pivots, with the uniform baseline's
 * rowwise quantizer (App. B.5) in place of the dual-axis fit: a key row of
 * width b < 16 stores s_i = fp16(clamp(absmax_i / q_b)) and nearest codes of
 * X * fp32(1/s_i) in [-q_b, q_b]; a pivot row (b = 16) stores fp16(X) and s_i = 0.
 * Head segment: s[128] fp16 | row i in index order, 16 b_i bytes (offset-binary
 * codes LSB-first, or 128 fp16 values). rb: the 128 row widths. */
size_t or_temporal_head_bytes(const int8_t *rb)
{
    size_t n = 256;
    for (int i = 0; i < OR_D; i++)
        n += (size_t)16 * rb[i];
    return n;
}

void or_temporal_encode_head(const float *X, const int8_t *rb, uint8_t *page)
{
    uint8_t *row = page + 256;
    for (int i = 0; i < OR_D; i++) {
        int b = rb[i];
        if (b == OR_PIVOT_BITS) {
            put_u16(page + 2 * i, 0);
            for (int j = 0; j < OR_D; j++)
                put_u16(row + 2 * j, or_fp16_encode(or_fp16_round(X[i * OR_D + j])));
        } else {
            int qm = qmax_of(b);
            float amax = 0.0f;
            for (int j = 0; j < OR_D; j++)
                if (fabsf(X[i * OR_D + j]) > amax)
                    amax = fabsf(X[i * OR_D + j]);
            double s16 = or_fp16_round(clampd((float)((double)amax / qm), F16_MIN_NORMAL, F16_MAX));
            float inv = (float)(1.0 / s16);
            put_u16(page + 2 * i, or_fp16_encode(s16));
            for (int j = 0; j < OR_D; j++) {
                int qv = (int)clampd(rint((double)mul32(X[i * OR_D + j], inv)), -qm, qm);
                put_bits(row, j * b, b, (unsigned)(qv + (1 << (b - 1))));
            }
        }
        row += (size_t)16 * b;
    }
}

void or_temporal_decode_head(const uint8_t *page, const int8_t *rb, double *S)
{
    const uint8_t *row = page + 256;
    for (int i = 0; i < OR_D; i++) {
        int b = rb[i];
        if (b == OR_PIVOT_BITS) {
            for (int j = 0; j < OR_D; j++)
                S[i * OR_D + j] = or_fp16_decode(get_u16(row + 2 * j));
        } else {
            double s = or_fp16_decode(get_u16(page + 2 * i));
            for (int j = 0; j < OR_D; j++)
                S[i * OR_D + j] = s * (double)((int)get_bits(row, j * b, b) - (1 << (b - 1)));
        }
        row += (size_t)16 * b;
    }
}
