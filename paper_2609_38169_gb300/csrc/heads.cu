// Head-unit (GDN) kernels: the persistent, bulk-async pipelined decode step and
// the pack/unpack kernels of head pages.
//
// Tile mapping: warp w owns the value columns 16w..16w+15 of the head, all 128
// key rows. Lane l = 8 cg + rg holds the 16 rows 16rg..16rg+15 (band rg) of the
// 4 columns 16w + 4cg .. 16w + 4cg + 3, as eight row pairs (rows 2m, 2m+1 of
// its band) per column, each pair one packed f32x2 register. So every column
// reduction (retrieval, readout, column maximum, least squares) stays inside a
// warp: a three-level shuffle reduce-scatter over the 8 lanes of a column
// group, whose result lane rg holds for column rg >> 1 of its group. Only the
// row reduction of the row factors crosses warps, through shared memory.
//
// Page codes: the 16 codes of band g in column j form a chunk of 2b bytes; a
// thread's four chunks (columns 16w + 4cg + 0..3 of band rg) are one stream of
// 2b words, stored as B/2 16-byte pieces interleaved over the warp's 32 lanes:
// piece k of lane l of warp w at w * 256 B + k * 512 + 16 l. Every 16-byte
// load or store of a warp then covers 512 contiguous bytes, with no bank
// conflicts for any width.
// Per-row constants sit in shared memory with a pad of 4 floats after every
// band of 16 rows, so the 8 bands a warp reads hit distinct banks.
//
// Decode pipeline (App. C.3 steps 1-7 per head): each persistent CTA walks its
// (head, slot) items, head-major; the last warp keeps up to S-1 pages in flight
// (pipeline.cuh), the CTA updates and refits the page in place in shared
// memory, and a bulk store writes it back. CTA barriers per item: one after the
// row constants (which also agrees on the stage's copies), two around the row
// factors, one before the store.
#include <atomic>

#include "async.cuh"
#include "device.cuh"
#include "internal.h"
#include "pipeline.cuh"
#include "tile.cuh"

namespace stepq {
namespace hk {

constexpr int kVecBytes = 5 * 512 + 128;               // q k v w2 wis | gate, beta per stage
constexpr int kPad = 160;                              // padded per-row array: 8 bands x (16 + 4)

// ------------------------------------------------------------ shared layout
constexpr int kOffBars = 0;                            // uint64 [8]
constexpr int kOffRed = 128;                           // float [8][kPad] row partial sums per warp
constexpr int kOffRows = kOffRed + 8 * kPad * 4;       // float [6][kPad] per-row constants
constexpr int kMaxHv = 256;                            // value heads per layer (launch check)
constexpr int kOffHead = kOffRows + 6 * kPad * 4;      // u64 off | u32 bytes | u8 bits | u8 key head
constexpr int kOffStages = (kOffHead + kMaxHv * 14 + 127) / 128 * 128;

// padded index of row i in a per-row array
__host__ __device__ constexpr int prow(int i) { return 20 * (i >> 4) + (i & 15); }

struct Smem {
    uint64_t *bars;
    float *red;
    // per-row constants (padded): kappa_i = k_i a_i, beta k_i / a_i, q_i a_i, a_i,
    // rho_i a_i and the least-squares weight alpha_i = w_i^2 r_i^2
    float *rKap, *rBkp, *rQa, *rA, *rRho, *rAl;
    uint64_t *hoff;
    uint32_t *hbytes;
    uint8_t *hbits, *hkey;
    uint8_t *stages;
    __device__ __forceinline__ explicit Smem(uint8_t *s) {
        bars = (uint64_t *)(s + kOffBars);
        red = (float *)(s + kOffRed);
        rKap = (float *)(s + kOffRows);
        rBkp = rKap + kPad;
        rQa = rKap + 2 * kPad;
        rA = rKap + 3 * kPad;
        rRho = rKap + 4 * kPad;
        rAl = rKap + 5 * kPad;
        hoff = (uint64_t *)(s + kOffHead);
        hbytes = (uint32_t *)(s + kOffHead + kMaxHv * 8);
        hbits = s + kOffHead + kMaxHv * 12;
        hkey = s + kOffHead + kMaxHv * 13;
        stages = s + kOffStages;
    }
};

struct Stage {
    uint8_t *page;
    float *q, *k, *v, *w2, *wis, *gb;
    __device__ __forceinline__ Stage(uint8_t *base, uint32_t page_region) {
        page = base;
        q = (float *)(base + page_region);
        k = q + 128;
        v = q + 256;
        w2 = q + 384;
        wis = q + 512;
        gb = q + 640;
    }
};

struct T {   // thread coordinates
    int tid, w, l, rg, cg;
    __device__ __forceinline__ T() {
        tid = threadIdx.x;
        w = tid >> 5;
        l = tid & 31;
        rg = l & 7;
        cg = l >> 3;
    }
    __device__ __forceinline__ int row(int r) const { return 16 * rg + r; }
    __device__ __forceinline__ int col(int c) const { return 16 * w + 4 * cg + c; }
    // the column whose reduced value this lane holds after a reduce-scatter
    __device__ __forceinline__ int own_col() const { return col(rg >> 1); }
};

// Row-pair constants m = 2p, 2p+1 of the thread's band from one 128-bit load.
__device__ __forceinline__ void row_pairs(const float *v, const T &t, int p, uint64_t &lo, uint64_t &hi) {
    const uint4 q = *(const uint4 *)&v[20 * t.rg + 4 * p];
    lo = u2pair(q.x, q.y);
    hi = u2pair(q.z, q.w);
}

// ---- warp reductions over the 8 lanes of a column group (lane bits 0-2) ----
// Lane rg returns the total over the group of v[rg >> 1].
__device__ __forceinline__ float col_sum_scatter(const float (&v)[4], int rg) {
    const bool b2 = rg & 4, b1 = rg & 2;
    const float a0 = (b2 ? v[2] : v[0]) + __shfl_xor_sync(0xffffffffu, b2 ? v[0] : v[2], 4);
    const float a1 = (b2 ? v[3] : v[1]) + __shfl_xor_sync(0xffffffffu, b2 ? v[1] : v[3], 4);
    const float a = (b1 ? a1 : a0) + __shfl_xor_sync(0xffffffffu, b1 ? a0 : a1, 2);
    return a + __shfl_xor_sync(0xffffffffu, a, 1);
}
__device__ __forceinline__ float col_max_scatter(const float (&v)[4], int rg) {
    const bool b2 = rg & 4, b1 = rg & 2;
    const float a0 = fmaxf(b2 ? v[2] : v[0], __shfl_xor_sync(0xffffffffu, b2 ? v[0] : v[2], 4));
    const float a1 = fmaxf(b2 ? v[3] : v[1], __shfl_xor_sync(0xffffffffu, b2 ? v[1] : v[3], 4));
    const float a = fmaxf(b1 ? a1 : a0, __shfl_xor_sync(0xffffffffu, b1 ? a0 : a1, 2));
    return fmaxf(a, __shfl_xor_sync(0xffffffffu, a, 1));
}
// Two values per column (least-squares numerator and denominator).
__device__ __forceinline__ void col_sum2_scatter(const float (&n)[4], const float (&d)[4], int rg,
                                                 float &no, float &dout) {
    const bool b2 = rg & 4, b1 = rg & 2;
    const float n0 = (b2 ? n[2] : n[0]) + __shfl_xor_sync(0xffffffffu, b2 ? n[0] : n[2], 4);
    const float n1 = (b2 ? n[3] : n[1]) + __shfl_xor_sync(0xffffffffu, b2 ? n[1] : n[3], 4);
    const float d0 = (b2 ? d[2] : d[0]) + __shfl_xor_sync(0xffffffffu, b2 ? d[0] : d[2], 4);
    const float d1 = (b2 ? d[3] : d[1]) + __shfl_xor_sync(0xffffffffu, b2 ? d[1] : d[3], 4);
    const float na = (b1 ? n1 : n0) + __shfl_xor_sync(0xffffffffu, b1 ? n0 : n1, 2);
    const float da = (b1 ? d1 : d0) + __shfl_xor_sync(0xffffffffu, b1 ? d0 : d1, 2);
    no = na + __shfl_xor_sync(0xffffffffu, na, 1);
    dout = da + __shfl_xor_sync(0xffffffffu, da, 1);
}
// The value of column c of the thread's group from the lane that holds it.
__device__ __forceinline__ float col_gather(float v, const T &t, int c) {
    return __shfl_sync(0xffffffffu, v, (t.l & 24) | (2 * c));
}

// ---- row reduction over the 4 lanes of a band (lane bits 3-4) ----
// 16 per-row partials in, 4 out: rows 8 (cg & 1) + 4 (cg >> 1) + t of the band.
__device__ __forceinline__ void row_sum_scatter(const float (&v)[16], int cg, float (&out)[4]) {
    float a8[8];
    const bool b0 = cg & 1, b1 = cg & 2;
#pragma unroll
    for (int t = 0; t < 8; t++)
        a8[t] = (b0 ? v[8 + t] : v[t]) + __shfl_xor_sync(0xffffffffu, b0 ? v[t] : v[8 + t], 8);
#pragma unroll
    for (int t = 0; t < 4; t++)
        out[t] = (b1 ? a8[4 + t] : a8[t]) + __shfl_xor_sync(0xffffffffu, b1 ? a8[t] : a8[4 + t], 16);
}

// ---- page streams: a thread's four chunks as B/2 interleaved 16-byte pieces ----
template <int B>
__device__ __forceinline__ uint8_t *stream_base(uint8_t *page, const T &t) {
    return page + (B == kPivot ? 0 : 512) + t.w * 256 * B + 16 * t.l;
}
template <int B>
__device__ __forceinline__ void load_block(const uint8_t *p, uint32_t (&wd)[2 * B]) {
#pragma unroll
    for (int k = 0; k < B / 2; k++) {
        const uint4 a = *(const uint4 *)(p + 512 * k);
        wd[4 * k] = a.x; wd[4 * k + 1] = a.y; wd[4 * k + 2] = a.z; wd[4 * k + 3] = a.w;
    }
}
template <int B>
__device__ __forceinline__ void store_block(uint8_t *p, const uint32_t (&wd)[2 * B]) {
#pragma unroll
    for (int k = 0; k < B / 2; k++)
        *(uint4 *)(p + 512 * k) = make_uint4(wd[4 * k], wd[4 * k + 1], wd[4 * k + 2], wd[4 * k + 3]);
}

// Scale of the high code of a pair as placed by code_pair (2^B, or 1 for B = 8).
template <int B>
__host__ __device__ constexpr float hi_scale() { return B == 8 ? 1.0f : 1.0f / (float)(1 << B); }

// Codes 2m and 2m+1 of chunk c of a block as the bit patterns of the floats
// 1.5*2^23 + u_lo and 1.5*2^23 + u_hi * 2^B (B = 8: both at the bottom): the
// codes are dropped into the zero low mantissa bits of the constant, one logic
// op each (after at most one shift per pair).
template <int B>
__device__ __forceinline__ uint64_t code_pair(const uint32_t (&wd)[2 * B], int c, int m) {
    constexpr int W = B / 2;                  // words per chunk
    if (B == 8) {
        const uint32_t w = wd[c * W + (m >> 1)];
        const uint32_t sel = 0x7650u + 2u * (uint32_t)(m & 1);
        return u2pair(__byte_perm(w, kMagicBits, sel), __byte_perm(w, kMagicBits, sel + 1u));
    }
    constexpr uint32_t mask = (1u << B) - 1u;
    const int p = 2 * m * B, k = c * W + (p >> 5), s = p & 31;
    uint32_t win;
    if (s == 0)
        win = wd[k];
    else if (s + 2 * B <= 32)
        win = wd[k] >> s;
    else
        win = __funnelshift_r(wd[k], wd[k + 1], s);
    return u2pair(and_or(win, mask, kMagicBits), and_or(win, mask << B, kMagicBits));
}

// Sum over the 16 codes of a chunk of (0x4B400000 << s) and of the parts
// shifted into the next word, i.e. what pack_codes adds besides the codes.
__host__ __device__ constexpr uint32_t pack_bias(int B, int k) {
    uint32_t b = 0;
    for (int r = 0; r < 16; r++) {
        const int p = r * B, kk = p >> 5, s = p & 31;
        if (kk == k) b += kMagicBits << s;
        if (s + B > 32 && kk + 1 == k) b += kMagicBits >> (32 - s);
    }
    return b;
}

// 16 offset-binary codes given as the float bit patterns 0x4B400000 | u_r,
// packed LSB-first into the words of chunk c. The high bits are the same
// constant for every code, so each word is the plain sum of the shifted
// patterns minus the shifted constants (mod 2^32): one shift-add per code.
template <int B>
__device__ __forceinline__ void pack_codes(const uint32_t (&f)[16], uint32_t (&wd)[2 * B], int c) {
    constexpr int W = B / 2;
    if (B == 8) {
#pragma unroll
        for (int t = 0; t < 4; t++) {
            const uint32_t lo = __byte_perm(f[4 * t], f[4 * t + 1], 0x0040);
            const uint32_t hi = __byte_perm(f[4 * t + 2], f[4 * t + 3], 0x0040);
            wd[c * W + t] = __byte_perm(lo, hi, 0x5410);
        }
        return;
    }
    uint32_t acc[W];
#pragma unroll
    for (int k = 0; k < W; k++) acc[k] = 0u - pack_bias(B, k);
#pragma unroll
    for (int r = 0; r < 16; r++) {
        const int p = r * B, k = p >> 5, s = p & 31;
        acc[k] += f[r] << s;
        if (s + B > 32) acc[k + 1] += f[r] >> (32 - s);
    }
#pragma unroll
    for (int k = 0; k < W; k++) wd[c * W + k] = acc[k];
}

// Per-row sums over the thread's 4 columns of |value|, for the row pair's
// low (even) and high (odd) rows.
__device__ __forceinline__ void abs_row_sums(const uint64_t (&x)[4], float &lo, float &hi) {
    lo = (fabsf(f2lo(x[0])) + fabsf(f2lo(x[1]))) + (fabsf(f2lo(x[2])) + fabsf(f2lo(x[3])));
    hi = (fabsf(f2hi(x[0])) + fabsf(f2hi(x[1]))) + (fabsf(f2hi(x[2])) + fabsf(f2hi(x[3])));
}

// Least-squares sums of the thread's columns: n_j += alpha_i z_ij X'_ij and
// d_j += alpha_i z_ij^2 with z_ij = rne(X'_ij gamma_j) (one rounding of the
// product), clamped to +-qmax when CLIP (App. C.1).
template <int B, bool CLIP>
__device__ __forceinline__ void ls_sums(const T &t, const Smem &S, const uint64_t (&x2)[8][4],
                                        const uint64_t (&g)[4], uint64_t (&n)[4], uint64_t (&d)[4]) {
    constexpr float fqm = (float)((1 << (B - 1)) - 1);
    const uint64_t M2 = f2s(kMagic), nM2 = f2s(-kMagic);
#pragma unroll
    for (int p = 0; p < 4; p++) {
        uint64_t alo, ahi;
        row_pairs(S.rAl, t, p, alo, ahi);
#pragma unroll
        for (int h = 0; h < 2; h++) {
            const int m = 2 * p + h;
            const uint64_t al = h ? ahi : alo;
#pragma unroll
            for (int c = 0; c < 4; c++) {
                uint64_t q = fadd2(ffma2(x2[m][c], g[c], M2), nM2);   // rne of the product
                if (CLIP) q = clamp2(q, fqm);
                const uint64_t aq = fmul2(al, q);
                n[c] = ffma2(aq, x2[m][c], n[c]);
                d[c] = ffma2(aq, q, d[c]);
            }
        }
    }
}

// Final codes q_ij = rne(X'_ij gamma_j) with the stored scales (clamped when
// CLIP), packed into the thread's page block.
template <int B, bool CLIP>
__device__ __forceinline__ void final_codes(const T &t, uint8_t *page, const uint64_t (&x2)[8][4],
                                            const uint64_t (&g)[4]) {
    constexpr float fqm = (float)((1 << (B - 1)) - 1);
    constexpr float fmb = kMagic + (float)(1 << (B - 1));
    const uint64_t MB = f2s(fmb), LO = f2s(fmb - fqm), HI = f2s(fmb + fqm);
    uint32_t wd[2 * B];
#pragma unroll
    for (int c = 0; c < 4; c++) {
        uint32_t f[16];
#pragma unroll
        for (int m = 0; m < 8; m++) {
            // one rounding of the product, then the clamp on the biased code
            uint64_t uu = ffma2(x2[m][c], g[c], MB);      // bits: 0x4B400000 | (q + 2^(B-1))
            if (CLIP) uu = clamp2r(uu, LO, HI);
            f[2 * m] = (uint32_t)uu;
            f[2 * m + 1] = (uint32_t)(uu >> 32);
        }
        pack_codes<B>(f, wd, c);
    }
    store_block<B>(stream_base<B>(page, t), wd);
}

// Approximate reciprocal and square root (the SFU's, within about 1 ulp) where
// the result only shapes a scale: the row factor's square root (rounded to FP16
// next), rho_i and the column scale of the first fixed-code pass. The reciprocal
// of the stored FP16 column scale, which takes the final code decisions, stays
// correctly rounded.
__device__ __forceinline__ float rcp_approx(float x) {
    float d;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(d) : "f"(x));
    return d;
}
__device__ __forceinline__ float sqrt_approx(float x) {
    float d;
    asm("sqrt.approx.ftz.f32 %0, %1;" : "=f"(d) : "f"(x));
    return d;
}

// ---------------------------------------------------------------- the fit
// Key-Row-Aware Dual-axis Fitting of the register tile (Sec. 4.3, App. C.1)
// and packing into the page (App. C.3 step 6). The tile holds Z with
// X_ij = a_i Z_ij (a_i > 0 a per-row factor: a_i = alpha r_i in the decode
// step, 1 when packing a dense state, S.rA holds it when `scaled`); rs[r]
// holds the partial sums of |Z| of the thread's rows over its 4 columns.
// `between` runs once the row partials are in shared memory, while threads
// 0..127 derive the row factors (the producer refills a stage there). On
// return the page holds r, c and the codes. Requires every thread to be done
// reading the old page.
template <int B, class Between>
__device__ __forceinline__ void fit_pack(const T &t, const Smem &S, uint8_t *page, const float *w2v,
                                         const float *wisv, bool scaled, uint64_t (&x2)[8][4],
                                         const float (&rs)[16], int fit_iters, const Between &between) {
    constexpr int qm = (1 << (B - 1)) - 1;
    constexpr float fqm = (float)qm;
    uint16_t *page_r = (uint16_t *)page;
    uint16_t *page_c = (uint16_t *)(page + 256);
    // Row factors r_i = m_i^(1/2) w_i^(-1/2), m_i = (1/128) sum_j |X_ij|: the
    // band's 4 lanes reduce-scatter their partials, the 8 warps' sums meet in
    // shared memory.
    {
        float part[4];
        row_sum_scatter(rs, t.cg, part);
        *(float4 *)&S.red[t.w * kPad + prow(t.row(8 * (t.cg & 1) + 4 * (t.cg >> 1)))] =
            make_float4(part[0], part[1], part[2], part[3]);
    }
    __syncthreads();
    between();
    if (t.tid < 128) {
        const int i = t.tid;
        float sz = 0.f;
#pragma unroll
        for (int wv = 0; wv < 8; wv++) sz += S.red[wv * kPad + prow(i)];
        const float a = scaled ? S.rA[prow(i)] : 1.f;
        const float m = (a * sz) * (1.0f / 128.0f);
        const float rf = __half2float(__float2half_rn(
            fminf(fmaxf(__fmul_rn(sqrt_approx(m), wisv[i]), kF16Min), kF16Max)));
        S.rRho[prow(i)] = rcp_approx(rf) * a;             // X' = rho_i X = (rho_i a_i) Z
        S.rAl[prow(i)] = w2v[i] * (rf * rf);              // w_i^2 r_i^2
        page_r[i] = f16_bits(rf);
    }
    __syncthreads();
    // X' = X rho_i (row-normalised state) and the clip-free column start
    // c0_j = max_i |X'_ij| / qmax, reduced inside the warp.
    float cm[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int p = 0; p < 4; p++) {
        uint64_t rlo, rhi;
        row_pairs(S.rRho, t, p, rlo, rhi);
#pragma unroll
        for (int c = 0; c < 4; c++) {
            x2[2 * p][c] = fmul2(x2[2 * p][c], rlo);
            x2[2 * p + 1][c] = fmul2(x2[2 * p + 1][c], rhi);
            cm[c] = fmax3(cm[c], fabsf(f2lo(x2[2 * p][c])), fabsf(f2hi(x2[2 * p][c])));
            cm[c] = fmax3(cm[c], fabsf(f2lo(x2[2 * p + 1][c])), fabsf(f2hi(x2[2 * p + 1][c])));
        }
    }
    // this lane's column (own_col): its max, its current scale, its reciprocal
    const float mx = col_max_scatter(cm, t.rg);
    const float c0 = __fmul_rn(mx, 1.0f / fqm);
    const bool clip0 = __any_sync(0xffffffffu, c0 > kF16Max);   // start capped: codes may clip
    float cc = fminf(fmaxf(c0, kF16Min), kF16Max);
    float gi = rcp_approx(cc);
    uint64_t g[4];
#pragma unroll
    for (int c = 0; c < 4; c++) g[c] = f2s(col_gather(gi, t, c));
    // Fixed-code least-squares updates: c_j = sum alpha_i q_ij X'_ij / sum alpha_i q_ij^2
    // (alpha_i = w_i^2 r_i^2: the w^2-weighted objective in the X' domain).
    bool clip = clip0;
    for (int it = 0; it < fit_iters; it++) {
        uint64_t n[4] = {0, 0, 0, 0}, d[4] = {0, 0, 0, 0};
        // the clip decision is per warp: one branch here, none per element
        if (it > 0 || clip0) ls_sums<B, true>(t, S, x2, g, n, d);
        else ls_sums<B, false>(t, S, x2, g, n, d);
        const float nv[4] = {pair_sum(n[0]), pair_sum(n[1]), pair_sum(n[2]), pair_sum(n[3])};
        const float dv[4] = {pair_sum(d[0]), pair_sum(d[1]), pair_sum(d[2]), pair_sum(d[3])};
        float num, den;
        col_sum2_scatter(nv, dv, t.rg, num, den);
        // num and den carry fp32 summation error already; a 2-ulp quotient adds nothing
        if (den > 0.f) cc = fminf(fmaxf(__fdividef(num, den), kF16Min), kF16Max);
        if (it + 1 < fit_iters) {
            gi = rcp_approx(cc);
        } else {
            // storage precision of c; codes can clip only where max |X'| / c >= qmax + 1/2
            const float cf = __half2float(__float2half_rn(cc));
            gi = __frcp_rn(cf);
            if ((t.rg & 1) == 0) page_c[t.own_col()] = f16_bits(cf);
            clip = __any_sync(0xffffffffu, __fmul_rn(mx, gi) >= fqm + 0.5f);
        }
#pragma unroll
        for (int c = 0; c < 4; c++) g[c] = f2s(col_gather(gi, t, c));
    }
    // Final codes with the stored scales.
    if (clip) final_codes<B, true>(t, page, x2, g);
    else final_codes<B, false>(t, page, x2, g);
}

// FP16 pivot head: store fp16(a_i Z) (saturating) in the chunk order; a row
// pair is one 32-bit word of a chunk.
__device__ __forceinline__ void pack_pivot(const T &t, uint8_t *page, const uint64_t (&x2)[8][4],
                                           float a) {
    uint32_t wd[2 * kPivot];
#pragma unroll
    for (int c = 0; c < 4; c++)
#pragma unroll
        for (int m = 0; m < 8; m++)
            wd[8 * c + m] = (uint32_t)f16_bits(f16_round_sat(a * f2lo(x2[m][c]))) |
                            ((uint32_t)f16_bits(f16_round_sat(a * f2hi(x2[m][c]))) << 16);
    store_block<kPivot>(stream_base<kPivot>(page, t), wd);
}

// Reconstruct the column-scaled codes c_j q_ij (exact in fp32) or the FP16
// values of a pivot head; the row factor stays separate.
template <int B>
__device__ __forceinline__ void load_tile(const T &t, const uint8_t *page, uint64_t (&x2)[8][4]) {
    uint32_t wd[2 * B];
    load_block<B>(stream_base<B>((uint8_t *)page, t), wd);
    if constexpr (B == kPivot) {
#pragma unroll
        for (int c = 0; c < 4; c++)
#pragma unroll
            for (int m = 0; m < 8; m++)
                x2[m][c] = f2(f16_val((uint16_t)(wd[8 * c + m] & 0xFFFFu)), f16_val((uint16_t)(wd[8 * c + m] >> 16)));
        return;
    } else {
    // the thread's 4 column scales: one 8-byte load
    const uint2 c4 = *(const uint2 *)(page + 256 + 2 * t.col(0));
    const uint16_t ch[4] = {(uint16_t)(c4.x & 0xFFFFu), (uint16_t)(c4.x >> 16), (uint16_t)(c4.y & 0xFFFFu),
                            (uint16_t)(c4.y >> 16)};
#pragma unroll
    for (int c = 0; c < 4; c++) {
        // f = 1.5*2^23 + u s (s = 1 or the pair's high scale): fma(f, c/s, -1.5*2^23 c/s)
        // = c u exactly (c fp16 and normal, u < 2^8: 19 significant bits; the
        // offset has 12), and c u - c 2^(B-1) = c q is exact as well.
        const uint64_t cj = f2s(f16_val(ch[c]));
        const uint64_t cc = fmul2(cj, f2(1.0f, hi_scale<B>()));
        const uint64_t oc = fmul2(cc, f2s(-kMagic));
        const uint64_t bc = fmul2(cj, f2s(-(float)(1 << (B - 1))));
#pragma unroll
        for (int m = 0; m < 8; m++) x2[m][c] = fadd2(ffma2(code_pair<B>(wd, c, m), cc, oc), bc);
    }
    }
}

// ------------------------------------------------------------------ decode
// Kernel modes: the fused step, and the two halves of the side-stream split
// (the readout returns y and delta and leaves the page as it is; the writeback
// rebuilds the updated tile from the old page and delta, refits and packs it).
enum : int { kFused = 0, kReadout = 1, kWriteback = 2 };

struct DecodeArgs {
    uint8_t *pool;
    uint64_t stride;
    int pool_slots;
    const int32_t *slots;
    int Hk, Hv, nb, items;     // nb batch entries; item = head * nb + entry
    LayerTables tab;
    const float *q, *k, *v, *beta, *gate;
    float *y;
    float *delta;              // readout: delta_j out; writeback: delta_j in
    unsigned int *err;
    StallKnob stall;
    int n_stages;
    uint32_t page_region, stage_bytes;
    int fit_iters;
};

// Producer warp: start the copies of the item (head h, batch entry b, a valid
// slot) into stage s. The writeback loads delta into the v slot and needs no
// q; the readout needs no w2, wis.
template <int MODE>
__device__ __forceinline__ void issue(const DecodeArgs &a, const Smem &S, int h, int b, int slot, int s,
                                      int lane) {
    uint64_t *bar = &S.bars[s];
    Stage st(S.stages + (size_t)s * a.stage_bytes, a.page_region);
    const int hk = S.hkey[h];
    if (MODE != kWriteback) warp_copy512(st.q, a.q + ((size_t)b * a.Hk + hk) * 128, lane);
    warp_copy512(st.k, a.k + ((size_t)b * a.Hk + hk) * 128, lane);
    warp_copy512(st.v, (MODE != kWriteback ? a.v : a.delta) + ((size_t)b * a.Hv + h) * 128, lane);
    if (MODE != kReadout) {
        warp_copy512(st.w2, a.tab.w2 + (size_t)h * 128, lane);
        warp_copy512(st.wis, a.tab.wis + (size_t)h * 128, lane);
    }
    if (lane == 0) {
        const size_t u = (size_t)b * a.Hv + h;
        cp_async4(st.gb, a.gate + u);
        cp_async4(st.gb + 1, a.beta + u);
    }
    cp_async_mbar_arrive(bar);
    __syncwarp();
    if (lane == 0) {
        const uint32_t nb = S.hbytes[h];
        mbar_arrive_tx(bar, nb);
        bulk_load(st.page, a.pool + (uint64_t)slot * a.stride + S.hoff[h], nb, bar);
    }
}

// One decode step of one head page staged in shared memory (width B).
// `ok` is this thread's verdict on the stage's copies; the first CTA barrier
// takes the OR of the negations, and on a stalled copy every thread returns
// false there (what it read before is discarded). `refill` runs once per item,
// after that barrier; the page itself is rewritten in place afterwards.
//
// With a_i = alpha r_i (> 0) and Z_ij = c_j q_ij + (beta k_i / a_i) delta_j the
// update is X_ij = a_i Z_ij: one fma per element instead of two.
//
// MODE kReadout stops after the readout: it writes y and delta (delta_out) and
// leaves the page untouched. MODE kWriteback takes delta from the stage (the
// readout's, bit for bit), rebuilds Z exactly as the fused step does, and runs
// steps 4-6; its y is not computed.
template <int B, int MODE, class Refill>
__device__ __forceinline__ bool decode_item(const T &t, const Smem &S, const Stage &st, float alpha,
                                            float beta, float *y_out, float *delta_out, int fit_iters,
                                            bool ok, const Refill &refill) {
    const uint16_t *page_r = (const uint16_t *)st.page;
    // Row constants (threads 0..127, one row each).
    if (t.tid < 128) {
        const int i = t.tid, pi = prow(i);
        const float a = fmaxf(B == kPivot ? alpha : alpha * f16_val(page_r[i]), 1e-30f);
        const float ki = st.k[i];
        S.rKap[pi] = ki * a;
        S.rBkp[pi] = __fdividef(beta * ki, a);          // within 2 ulp: Z carries rounding anyway
        if (MODE != kWriteback) S.rQa[pi] = st.q[i] * a;
        S.rA[pi] = a;
    }
    uint64_t x2[8][4];
    load_tile<B>(t, st.page, x2);
    if (__syncthreads_or(!ok)) return false;
    const bool fit = MODE != kReadout && B != kPivot;
    if (!fit) refill();
    uint64_t dl[4];
    if constexpr (MODE == kWriteback) {
        const float4 d4 = *(const float4 *)&st.v[t.col(0)];
        dl[0] = f2s(d4.x); dl[1] = f2s(d4.y); dl[2] = f2s(d4.z); dl[3] = f2s(d4.w);
    } else {
        // Step 2a: retrieval u_j = sum_i k_i a_i (c_j q_ij), reduced over the
        // column group; delta_j = v_j - u_j for the lane's column, gathered.
        uint64_t ua[4] = {0, 0, 0, 0};
#pragma unroll
        for (int p = 0; p < 4; p++) {
            uint64_t klo, khi;
            row_pairs(S.rKap, t, p, klo, khi);
#pragma unroll
            for (int c = 0; c < 4; c++) {
                ua[c] = ffma2(klo, x2[2 * p][c], ua[c]);
                ua[c] = ffma2(khi, x2[2 * p + 1][c], ua[c]);
            }
        }
        const float u4[4] = {pair_sum(ua[0]), pair_sum(ua[1]), pair_sum(ua[2]), pair_sum(ua[3])};
        const float u = col_sum_scatter(u4, t.rg);
        const float dj = st.v[t.own_col()] - u;             // delta_j = v_j - u_j
        if (MODE == kReadout && (t.rg & 1) == 0) delta_out[t.own_col()] = dj;
#pragma unroll
        for (int c = 0; c < 4; c++) dl[c] = f2s(col_gather(dj, t, c));
    }
    // Step 2b-3: Z = c q + (beta k / a) delta; readout partials q_i a_i Z_ij.
    uint64_t ya[4] = {0, 0, 0, 0};
#pragma unroll
    for (int p = 0; p < 4; p++) {
        uint64_t blo, bhi;
        row_pairs(S.rBkp, t, p, blo, bhi);
#pragma unroll
        for (int c = 0; c < 4; c++) {
            x2[2 * p][c] = ffma2(blo, dl[c], x2[2 * p][c]);
            x2[2 * p + 1][c] = ffma2(bhi, dl[c], x2[2 * p + 1][c]);
        }
        if (MODE != kWriteback) {
            uint64_t qlo, qhi;
            row_pairs(S.rQa, t, p, qlo, qhi);
#pragma unroll
            for (int c = 0; c < 4; c++) {
                ya[c] = ffma2(qlo, x2[2 * p][c], ya[c]);
                ya[c] = ffma2(qhi, x2[2 * p + 1][c], ya[c]);
            }
        }
    }
    if (MODE != kWriteback) {
        const float y4[4] = {pair_sum(ya[0]), pair_sum(ya[1]), pair_sum(ya[2]), pair_sum(ya[3])};
        const float yj = col_sum_scatter(y4, t.rg);
        if ((t.rg & 1) == 0) y_out[t.own_col()] = yj;
    }
    if (MODE == kReadout) return true;
    if (B == kPivot) {
        pack_pivot(t, st.page, x2, fmaxf(alpha, 1e-30f));
        return true;
    }
    // Steps 4-6: refit and repack in place.
    float rs[16];
#pragma unroll
    for (int m = 0; m < 8; m++) abs_row_sums(x2[m], rs[2 * m], rs[2 * m + 1]);
    if constexpr (B != kPivot)
        fit_pack<B>(t, S, st.page, st.w2, st.wis, true, x2, rs, fit_iters, refill);
    return true;
}

template <int MODE>
__global__ void __launch_bounds__(kThreads, 2) decode_heads_kernel(DecodeArgs a) {
    extern __shared__ __align__(128) uint8_t smem[];
    const T t;
    const Smem S(smem);
    if ((int)blockIdx.x >= a.items) return;
    const int grp = a.Hv / a.Hk;
    for (int h = t.tid; h < a.Hv; h += kThreads) {
        S.hoff[h] = a.tab.head_off[h];
        S.hbytes[h] = a.tab.head_bytes[h];
        S.hbits[h] = a.tab.head_bits[h];
        S.hkey[h] = (uint8_t)(h / grp);
    }
    if (t.tid == pipe::kProducer) {
        for (int s = 0; s < a.n_stages; s++) mbar_init(&S.bars[s], 1);
        mbar_init_fence();
    }
    __syncthreads();
    const pipe::Shape p{a.items, a.nb, a.n_stages, a.slots, a.pool_slots, a.err, a.stall.wait_cycles,
                        a.stall.withhold_item};
    pipe::run(
        p, S.bars,
        [&](int h, int b, int slot, int s, int lane) { issue<MODE>(a, S, h, b, slot, s, lane); },
        [&](int h, int b, int, int s, bool ok, const auto &refill) {
            const size_t u = (size_t)b * a.Hv + h;
            const Stage st(S.stages + (size_t)s * a.stage_bytes, a.page_region);
            const float2 gb = *(const float2 *)st.gb;     // (gate, beta), staged with the page
            float *y_out = MODE == kWriteback ? nullptr : a.y + u * 128;
            float *d_out = MODE == kReadout ? a.delta + u * 128 : nullptr;
            switch (S.hbits[h]) {
            case 2: return decode_item<2, MODE>(t, S, st, gb.x, gb.y, y_out, d_out, a.fit_iters, ok, refill);
            case 4: return decode_item<4, MODE>(t, S, st, gb.x, gb.y, y_out, d_out, a.fit_iters, ok, refill);
            case 6: return decode_item<6, MODE>(t, S, st, gb.x, gb.y, y_out, d_out, a.fit_iters, ok, refill);
            case 8: return decode_item<8, MODE>(t, S, st, gb.x, gb.y, y_out, d_out, a.fit_iters, ok, refill);
            default: return decode_item<kPivot, MODE>(t, S, st, gb.x, gb.y, y_out, d_out, a.fit_iters, ok, refill);
            }
        },
        [&](int h, int slot, int s) {
            if (MODE != kReadout)
                bulk_store(a.pool + (uint64_t)slot * a.stride + S.hoff[h],
                           S.stages + (size_t)s * a.stage_bytes, S.hbytes[h]);
        });
}

// ---------------------------------------------------------- pack / unpack
struct PoolArgs {
    uint8_t *pool;
    uint64_t stride;
    int pool_slots;
    const int32_t *slots;
    int Hv;
    LayerTables tab;
    float *states;
    size_t state_stride_b;
    unsigned int *err;
    int fit_iters;
};

constexpr int kPageMaxHead = 32768;
constexpr int kPoolSmem = kOffStages + kPageMaxHead + kVecBytes;

template <int B>
__device__ __forceinline__ void quantize_item(const T &t, const Smem &S, uint8_t *page, const float *w2,
                                              const float *wis, const float *X, int fit_iters) {
    uint64_t x2[8][4];
    float rs[16];
#pragma unroll
    for (int m = 0; m < 8; m++) {
        const float4 r0 = *(const float4 *)(X + t.row(2 * m) * 128 + t.col(0));
        const float4 r1 = *(const float4 *)(X + t.row(2 * m + 1) * 128 + t.col(0));
        x2[m][0] = f2(r0.x, r1.x);
        x2[m][1] = f2(r0.y, r1.y);
        x2[m][2] = f2(r0.z, r1.z);
        x2[m][3] = f2(r0.w, r1.w);
        abs_row_sums(x2[m], rs[2 * m], rs[2 * m + 1]);
    }
    if constexpr (B == kPivot) {
        pack_pivot(t, page, x2, 1.f);
    } else {
        fit_pack<B>(t, S, page, w2, wis, false, x2, rs, fit_iters, [] {});
    }
}

__global__ void __launch_bounds__(kThreads, 2) quantize_heads_kernel(PoolArgs a) {
    extern __shared__ __align__(128) uint8_t smem[];
    const T t;
    const Smem S(smem);
    const int b = blockIdx.x / a.Hv, h = blockIdx.x - b * a.Hv;
    const int slot = a.slots[b];
    if (slot < 0 || slot >= a.pool_slots) {
        if (t.tid == 0) raise_error(a.err, STEPQ_ERR_SLOT_RANGE);
        return;
    }
    uint8_t *page = S.stages;
    float *w2 = (float *)(page + kPageMaxHead), *wis = w2 + 128;
    if (t.tid < 128) {
        w2[t.tid] = a.tab.w2[h * 128 + t.tid];
        wis[t.tid] = a.tab.wis[h * 128 + t.tid];
    }
    __syncthreads();
    const float *X = a.states + (size_t)b * a.state_stride_b + (size_t)h * kN;
    switch (a.tab.head_bits[h]) {
    case 2: quantize_item<2>(t, S, page, w2, wis, X, a.fit_iters); break;
    case 4: quantize_item<4>(t, S, page, w2, wis, X, a.fit_iters); break;
    case 6: quantize_item<6>(t, S, page, w2, wis, X, a.fit_iters); break;
    case 8: quantize_item<8>(t, S, page, w2, wis, X, a.fit_iters); break;
    default: quantize_item<kPivot>(t, S, page, w2, wis, X, a.fit_iters); break;
    }
    __syncthreads();
    uint8_t *gpage = a.pool + (uint64_t)slot * a.stride + a.tab.head_off[h];
    const int n16 = (int)a.tab.head_bytes[h] >> 4;
    for (int e = t.tid; e < n16; e += kThreads) ((uint4 *)gpage)[e] = ((const uint4 *)page)[e];
}

template <int B>
__device__ __forceinline__ void dequantize_item(const T &t, const uint8_t *page, float *out) {
    uint64_t x2[8][4];
    load_tile<B>(t, page, x2);      // c_j q_ij (exact) or the FP16 value
    const uint16_t *page_r = (const uint16_t *)page;
#pragma unroll
    for (int m = 0; m < 8; m++) {
        // r_i c_j z_ij rounded once: c_j q_ij is exact in fp32 (fp16 x 8 bits)
        const uint64_t rr = B == kPivot ? 0 : f2(f16_val(page_r[t.row(2 * m)]), f16_val(page_r[t.row(2 * m + 1)]));
        uint64_t v[4];
#pragma unroll
        for (int c = 0; c < 4; c++) v[c] = B == kPivot ? x2[m][c] : fmul2(rr, x2[m][c]);
        *(float4 *)(out + t.row(2 * m) * 128 + t.col(0)) = make_float4(f2lo(v[0]), f2lo(v[1]), f2lo(v[2]), f2lo(v[3]));
        *(float4 *)(out + t.row(2 * m + 1) * 128 + t.col(0)) = make_float4(f2hi(v[0]), f2hi(v[1]), f2hi(v[2]), f2hi(v[3]));
    }
}

__global__ void __launch_bounds__(kThreads, 2) dequantize_heads_kernel(PoolArgs a) {
    extern __shared__ __align__(128) uint8_t smem[];
    const T t;
    const Smem S(smem);
    const int b = blockIdx.x / a.Hv, h = blockIdx.x - b * a.Hv;
    const int slot = a.slots[b];
    if (slot < 0 || slot >= a.pool_slots) {
        if (t.tid == 0) raise_error(a.err, STEPQ_ERR_SLOT_RANGE);
        return;
    }
    uint8_t *page = S.stages;
    const uint8_t *gpage = a.pool + (uint64_t)slot * a.stride + a.tab.head_off[h];
    const int n16 = (int)a.tab.head_bytes[h] >> 4;
    for (int e = t.tid; e < n16; e += kThreads) ((uint4 *)page)[e] = ((const uint4 *)gpage)[e];
    __syncthreads();
    float *out = a.states + (size_t)b * a.state_stride_b + (size_t)h * kN;
    switch (a.tab.head_bits[h]) {
    case 2: dequantize_item<2>(t, page, out); break;
    case 4: dequantize_item<4>(t, page, out); break;
    case 6: dequantize_item<6>(t, page, out); break;
    case 8: dequantize_item<8>(t, page, out); break;
    default: dequantize_item<kPivot>(t, page, out); break;
    }
}

}  // namespace hk

// ------------------------------------------------------------------ launchers
static stepq_status set_attr(const void *fn, int bytes) {
    return cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes) == cudaSuccess
               ? STEPQ_OK
               : STEPQ_ERR_CUDA;
}

static int sm_count() {
    static std::atomic<int> n[64];        // per device; racing first calls store the same value
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev < 0 || dev >= 64) return 1;
    int v = n[dev].load(std::memory_order_relaxed);
    if (!v) {
        cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev);
        n[dev].store(v, std::memory_order_relaxed);
    }
    return v > 0 ? v : 1;
}

stepq_status launch_decode_heads(const stepq_plan *p, int layer, uint8_t *pool, int pool_slots,
                                 const int32_t *slots, int B, const float *q, const float *k,
                                 const float *v, const float *beta, const float *gate, float *y,
                                 cudaStream_t s) {
    return launch_decode_heads_mode(p, layer, pool, pool_slots, slots, B, q, k, v, beta, gate, y,
                                    nullptr, hk::kFused, s);
}

stepq_status launch_decode_heads_mode(const stepq_plan *p, int layer, uint8_t *pool, int pool_slots,
                                      const int32_t *slots, int B, const float *q, const float *k,
                                      const float *v, const float *beta, const float *gate, float *y,
                                      float *delta, int mode, cudaStream_t s) {
    const int Hv = p->cfg.n_value_heads;
    if (Hv > hk::kMaxHv) return STEPQ_ERR_UNSUPPORTED;
    uint32_t maxb = 0;
    for (int h = 0; h < Hv; h++) maxb = p->head_bytes[(size_t)layer * Hv + h] > maxb
                                            ? p->head_bytes[(size_t)layer * Hv + h] : maxb;
    hk::DecodeArgs a{};
    a.pool = pool;
    a.stride = p->slot_stride;
    a.pool_slots = pool_slots;
    a.slots = slots;
    a.Hk = p->cfg.n_key_heads;
    a.Hv = Hv;
    a.nb = B;
    a.items = B * Hv;
    a.tab = p->layer(layer);
    a.q = q; a.k = k; a.v = v; a.beta = beta; a.gate = gate; a.y = y;
    a.delta = delta;
    a.err = device_error_word();
    a.stall = stall_knob();
    a.page_region = (maxb + 127) / 128 * 128;
    a.stage_bytes = a.page_region + hk::kVecBytes;
    // as many stages (2..4) as keep two CTAs per SM
    int stages = (int)((113 * 1024 - hk::kOffStages) / a.stage_bytes);
    stages = stages < 2 ? 2 : (stages > 4 ? 4 : stages);
    a.n_stages = stages;
    a.fit_iters = p->cfg.fit_iters;
    const int smem = hk::kOffStages + stages * (int)a.stage_bytes;
    const void *fn = mode == hk::kReadout     ? (const void *)hk::decode_heads_kernel<hk::kReadout>
                     : mode == hk::kWriteback ? (const void *)hk::decode_heads_kernel<hk::kWriteback>
                                              : (const void *)hk::decode_heads_kernel<hk::kFused>;
    if (set_attr(fn, smem) != STEPQ_OK) return STEPQ_ERR_CUDA;
    int grid = 2 * sm_count();
    if (grid > a.items) grid = a.items;
    if (mode == hk::kReadout) hk::decode_heads_kernel<hk::kReadout><<<grid, kThreads, smem, s>>>(a);
    else if (mode == hk::kWriteback) hk::decode_heads_kernel<hk::kWriteback><<<grid, kThreads, smem, s>>>(a);
    else hk::decode_heads_kernel<hk::kFused><<<grid, kThreads, smem, s>>>(a);
    return cudaGetLastError() == cudaSuccess ? STEPQ_OK : STEPQ_ERR_CUDA;
}

static hk::PoolArgs pool_args(const stepq_plan *p, int layer, uint8_t *pool, int pool_slots,
                              const int32_t *slots, float *states, size_t stride_b) {
    hk::PoolArgs a{};
    a.pool = pool;
    a.stride = p->slot_stride;
    a.pool_slots = pool_slots;
    a.slots = slots;
    a.Hv = p->cfg.n_value_heads;
    a.tab = p->layer(layer);
    a.states = states;
    a.state_stride_b = stride_b;
    a.err = device_error_word();
    a.fit_iters = p->cfg.fit_iters;
    return a;
}

stepq_status launch_quantize_heads(const stepq_plan *p, int layer, const float *states,
                                   size_t stride_b, const int32_t *slots, int B, uint8_t *pool,
                                   int pool_slots, cudaStream_t s) {
    if (set_attr((const void *)hk::quantize_heads_kernel, hk::kPoolSmem) != STEPQ_OK) return STEPQ_ERR_CUDA;
    hk::PoolArgs a = pool_args(p, layer, pool, pool_slots, slots, (float *)states, stride_b);
    hk::quantize_heads_kernel<<<(unsigned)B * a.Hv, kThreads, hk::kPoolSmem, s>>>(a);
    return cudaGetLastError() == cudaSuccess ? STEPQ_OK : STEPQ_ERR_CUDA;
}

stepq_status launch_dequantize_heads(const stepq_plan *p, int layer, const uint8_t *pool,
                                     int pool_slots, const int32_t *slots, int B, float *states,
                                     size_t stride_b, cudaStream_t s) {
    if (set_attr((const void *)hk::dequantize_heads_kernel, hk::kPoolSmem) != STEPQ_OK) return STEPQ_ERR_CUDA;
    hk::PoolArgs a = pool_args(p, layer, (uint8_t *)pool, pool_slots, slots, states, stride_b);
    hk::dequantize_heads_kernel<<<(unsigned)B * a.Hv, kThreads, hk::kPoolSmem, s>>>(a);
    return cudaGetLastError() == cudaSuccess ? STEPQ_OK : STEPQ_ERR_CUDA;
}

}  // namespace stepq
