// Row-unit (KDA, per-key-channel gate) decode step: the persistent, bulk-async
// pipelined kernel over row-major pages with one width per key row.
//
// Rows are stored by decreasing width, so the kernel works in storage order:
// warp w owns the stored rows (slots) 16w..16w+15 and lane l the value columns
// 4l..4l+3. All lanes of a warp read the same row at a time, so a row's width
// is uniform across the warp and a lane's 4 codes are one contiguous 4b-bit
// segment of the row. A thread holds 8 slot pairs x 4 columns as packed f32x2
// registers: per-row constants of a pair are adjacent in shared memory (one
// 128-bit load serves two pairs), column constants are duplicated pairs kept
// in registers. Widths are handled with runtime shifts and masks (one funnel
// shift per row segment), which keeps the unrolled code small; FP16 pivot rows
// take an out-of-line path.
//
// Per row i the tile holds Z with X_ij = a_i Z_ij: a_i = d_i r_i zs_i and
// Z = c_j q_ij for an integer row (zs_i = 2^(8 - b_i), the normalised codebook
// of App. C.1), a_i = d_i and Z = the FP16 value for a pivot row. Pivot rows
// stay out of the column fit (rho a = 1, mu = alpha = qmax = 0).
#include "async.cuh"
#include "device.cuh"
#include "internal.h"
#include "pipeline.cuh"
#include "tile.cuh"

namespace stepq {
namespace rk {

constexpr int kVecBytes = 7 * 512 + 128;               // q k v gate w2 wis | row slots | beta

// ------------------------------------------------------------ shared layout
constexpr int kOffBars = 0;                            // uint64 [8]
constexpr int kOffFlags = 64;                          // int [16]
constexpr int kOffRed = 128;                           // float [3][8][128] cross-warp partials
constexpr int kOffColC = kOffRed + 3 * 8 * 128 * 4;    // float [128] c_j (start / iterate)
constexpr int kOffColM = kOffColC + 512;               // u32 [128] bits of max_i fp32(|X'_ij| mu_i)
constexpr int kOffColD = kOffColM + 512;               // float [128] delta_j
constexpr int kOffColG = kOffColD + 512;               // float [128] 1/c_j
constexpr int kNRowVec = 10;                           // per-row float vectors
constexpr int kOffRows = kOffColG + 512;               // float [kNRowVec][128]
constexpr int kOffInfo = kOffRows + kNRowVec * 512;    // uint2 [128]: (row slot, pack bias)
constexpr int kMaxHv = 256;                            // value heads per layer (launch check)
constexpr int kOffHead = kOffInfo + 128 * 8;           // u64 off | u32 bytes | u8 key head
constexpr int kOffStages = (kOffHead + kMaxHv * 13 + 127) / 128 * 128;

struct Smem {
    uint64_t *bars;
    int *flags;
    float *red, *colC, *colD, *colG;
    uint32_t *colM;
    // per-row constants: kappa = k a, beta k / a, q a, a, rho a, alpha = w^2 (r zs)^2,
    // mu = 1/qmax, qmax, the decode offset -(1.5*2^23 + 2^(b-1)) and 1.5*2^23 + 2^(b-1)
    float *rKap, *rBkp, *rQa, *rA, *rRho, *rAl, *rMu, *rQm, *rOff, *rMb;
    uint2 *rInfo;
    uint64_t *hoff;
    uint32_t *hbytes;
    uint8_t *hkey;
    uint8_t *stages;
    __device__ __forceinline__ explicit Smem(uint8_t *s) {
        bars = (uint64_t *)(s + kOffBars);
        flags = (int *)(s + kOffFlags);
        red = (float *)(s + kOffRed);
        colC = (float *)(s + kOffColC);
        colM = (uint32_t *)(s + kOffColM);
        colD = (float *)(s + kOffColD);
        colG = (float *)(s + kOffColG);
        float *r = (float *)(s + kOffRows);
        rKap = r; rBkp = r + 128; rQa = r + 256; rA = r + 384; rRho = r + 512;
        rAl = r + 640; rMu = r + 768; rQm = r + 896; rOff = r + 1024; rMb = r + 1152;
        rInfo = (uint2 *)(s + kOffInfo);
        hoff = (uint64_t *)(s + kOffHead);
        hbytes = (uint32_t *)(s + kOffHead + kMaxHv * 8);
        hkey = s + kOffHead + kMaxHv * 12;
        stages = s + kOffStages;
    }
};

struct Stage {
    uint8_t *page;
    float *q, *k, *v, *gate, *w2, *wis;
    uint32_t *slot;     // s-th stored row of the head: offset | width << 16 | row << 24
    float *beta;
    __device__ __forceinline__ Stage(uint8_t *base, uint32_t page_region) {
        page = base;
        q = (float *)(base + page_region);
        k = q + 128;
        v = q + 256;
        gate = q + 384;
        w2 = q + 512;
        wis = q + 640;
        slot = (uint32_t *)(q + 768);
        beta = q + 896;
    }
};

struct T {   // thread coordinates
    int tid, w, l;
    __device__ __forceinline__ T() {
        tid = threadIdx.x;
        w = tid >> 5;
        l = tid & 31;
    }
    __device__ __forceinline__ int row(int r) const { return 16 * w + r; }
};

// Row-pair constants m = 2p, 2p+1 of the warp's band from one 128-bit load.
__device__ __forceinline__ void row_pairs(const float *v, const T &t, int p, uint64_t &lo, uint64_t &hi) {
    const uint4 q = *(const uint4 *)&v[t.row(4 * p)];
    lo = u2pair(q.x, q.y);
    hi = u2pair(q.z, q.w);
}
__device__ __forceinline__ uint64_t row_pair(const float *v, const T &t, int m) {
    return *(const uint64_t *)&v[t.row(2 * m)];
}
// The lane's 4 columns of a per-column vector as duplicated pairs.
__device__ __forceinline__ void col_dup(const float *v, int l, uint64_t (&d)[4]) {
    const float4 q = *(const float4 *)&v[4 * l];
    d[0] = f2s(q.x);
    d[1] = f2s(q.y);
    d[2] = f2s(q.z);
    d[3] = f2s(q.w);
}
__device__ __forceinline__ void cols_to_red(const T &t, float *red, int reg, const float (&v)[4]) {
    *(float4 *)&red[(reg * 8 + t.w) * 128 + 4 * t.l] = make_float4(v[0], v[1], v[2], v[3]);
}
// (lo, hi) clamped to +-lim_lo and +-lim_hi.
__device__ __forceinline__ uint64_t clamp2p(uint64_t v, uint64_t lim) {
    const float a = f2lo(lim), b = f2hi(lim);
    return f2(fminf(fmaxf(f2lo(v), -a), a), fminf(fmaxf(f2hi(v), -b), b));
}

// The lane's 4b-bit code segment of a row of width b (columns 4l..4l+3),
// right-aligned. The second word may lie past the row; it stays inside the
// stage and its bits beyond the segment are masked off by the callers.
__device__ __forceinline__ uint32_t lane_segment(const uint8_t *row, int b, int l) {
    const uint32_t *wp = (const uint32_t *)row;
    const int bit = 4 * l * b;
    return __funnelshift_r(wp[bit >> 5], wp[(bit >> 5) + 1], bit & 31);
}

// Write the lane's 4b-bit segment v (b in {2, 4, 6, 8}) into the row: b/2
// bytes from byte l b/2, as byte stores under warp-uniform conditions (no
// branches; the lanes never share a byte).
__device__ __forceinline__ void store_segment(uint8_t *row, int b, int l, uint32_t v) {
    uint8_t *p = row + ((l * b) >> 1);
    p[0] = (uint8_t)v;
    if (b >= 4) p[1] = (uint8_t)(v >> 8);
    if (b >= 6) p[2] = (uint8_t)(v >> 16);
    if (b >= 8) p[3] = (uint8_t)(v >> 24);
}

// Sum over the 4 codes of a lane segment of (0x4B400000 << k b): what the
// packing adds besides the codes.
__device__ __forceinline__ uint32_t pack_bias4(int b) {
    return kMagicBits + (kMagicBits << b) + (kMagicBits << (2 * b)) + (kMagicBits << (3 * b));
}

// FP16 pivot rows (rare): kept out of line so the unrolled tile loops stay small.
__device__ __noinline__ float4 pivot_values(const uint8_t *row, int l) {
    const uint2 p = ((const uint2 *)row)[l];
    return make_float4(f16_val((uint16_t)(p.x & 0xFFFFu)), f16_val((uint16_t)(p.x >> 16)),
                       f16_val((uint16_t)(p.y & 0xFFFFu)), f16_val((uint16_t)(p.y >> 16)));
}
__device__ __noinline__ void store_pivot(uint8_t *row, int l, float a, float4 z) {
    const uint32_t w0 = (uint32_t)f16_bits(f16_round_sat(a * z.x)) |
                        ((uint32_t)f16_bits(f16_round_sat(a * z.y)) << 16);
    const uint32_t w1 = (uint32_t)f16_bits(f16_round_sat(a * z.z)) |
                        ((uint32_t)f16_bits(f16_round_sat(a * z.w)) << 16);
    ((uint2 *)row)[l] = make_uint2(w0, w1);
}

// ------------------------------------------------------------------ decode
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

// Kernel modes as for the head-unit kernel: the fused step, the readout (y and
// delta, page untouched) and the writeback (delta in; refit and pack).
enum : int { kFused = 0, kReadout = 1, kWriteback = 2 };

template <int MODE>
__device__ __forceinline__ void issue(const DecodeArgs &a, const Smem &S, int h, int b, int slot, int s,
                                      int lane) {
    uint64_t *bar = &S.bars[s];
    Stage st(S.stages + (size_t)s * a.stage_bytes, a.page_region);
    const int hk = S.hkey[h];
    const size_t u = (size_t)b * a.Hv + h;
    if (MODE != kWriteback) warp_copy512(st.q, a.q + ((size_t)b * a.Hk + hk) * 128, lane);
    warp_copy512(st.k, a.k + ((size_t)b * a.Hk + hk) * 128, lane);
    warp_copy512(st.v, (MODE != kWriteback ? a.v : a.delta) + u * 128, lane);
    warp_copy512(st.gate, a.gate + u * 128, lane);
    if (MODE != kReadout) {
        warp_copy512(st.w2, a.tab.w2 + (size_t)h * 128, lane);
        warp_copy512(st.wis, a.tab.wis + (size_t)h * 128, lane);
    }
    warp_copy512(st.slot, a.tab.row_slot + (size_t)h * 128, lane);
    if (lane == 0) cp_async4(st.beta, a.beta + u);
    cp_async_mbar_arrive(bar);
    __syncwarp();
    if (lane == 0) {
        const uint32_t nb = S.hbytes[h];
        mbar_arrive_tx(bar, nb);
        bulk_load(st.page, a.pool + (uint64_t)slot * a.stride + S.hoff[h], nb, bar);
    }
}

// Z of row pair m (columns 4l..4l+3): c_j q_ij (exact) for integer rows, the
// FP16 value for pivot rows.
__device__ __forceinline__ void load_pair(const T &t, const Smem &S, const uint8_t *page, int m,
                                          const uint64_t (&cd)[4], uint64_t (&x)[4]) {
    const uint4 inf = *(const uint4 *)&S.rInfo[t.row(2 * m)];
    const int b0 = (int)((inf.x >> 16) & 0xFFu), b1 = (int)((inf.z >> 16) & 0xFFu);
    const uint8_t *r0 = page + (inf.x & 0xFFFFu), *r1 = page + (inf.z & 0xFFFFu);
    if (b0 != kPivot && b1 != kPivot) {                  // two integer rows: paired arithmetic
        const uint32_t s0 = lane_segment(r0, b0, t.l), s1 = lane_segment(r1, b1, t.l);
        const uint32_t k0 = (1u << b0) - 1u, k1 = (1u << b1) - 1u;
        const uint64_t off = row_pair(S.rOff, t, m);
#pragma unroll
        for (int c = 0; c < 4; c++)
            x[c] = fmul2(fadd2(u2pair(and_or(s0 >> (c * b0), k0, kMagicBits), and_or(s1 >> (c * b1), k1, kMagicBits)),
                               off),
                         cd[c]);
        return;
    }
    float v[2][4];
#pragma unroll
    for (int h = 0; h < 2; h++) {
        const int b = h ? b1 : b0;
        const uint8_t *row = h ? r1 : r0;
        if (b == kPivot) {
            const float4 p = pivot_values(row, t.l);
            v[h][0] = p.x;
            v[h][1] = p.y;
            v[h][2] = p.z;
            v[h][3] = p.w;
        } else {
            const uint32_t s = lane_segment(row, b, t.l), k = (1u << b) - 1u;
            const float off = S.rOff[t.row(2 * m + h)];
#pragma unroll
            for (int c = 0; c < 4; c++)
                v[h][c] = __fmul_rn(__uint_as_float(and_or(s >> (c * b), k, kMagicBits)) + off,
                                    f2lo(cd[c]));
        }
    }
#pragma unroll
    for (int c = 0; c < 4; c++) x[c] = f2(v[0][c], v[1][c]);
}

// Final codes of row pair m: q = rne(X' / c_j) (clamped to +-qmax when CLIP),
// or fp16(a Z) for a pivot row, written into the page.
template <bool CLIP>
__device__ __forceinline__ void store_pair(const T &t, const Smem &S, uint8_t *page, int m,
                                           const uint64_t (&x)[4], const uint64_t (&gd)[4]) {
    const uint4 inf = *(const uint4 *)&S.rInfo[t.row(2 * m)];
    const int b0 = (int)((inf.x >> 16) & 0xFFu), b1 = (int)((inf.z >> 16) & 0xFFu);
    uint8_t *r0 = page + (inf.x & 0xFFFFu), *r1 = page + (inf.z & 0xFFFFu);
    const uint64_t mb = row_pair(S.rMb, t, m);
    uint64_t lo = 0, hi = 0;
    if (CLIP) {
        const uint64_t qm = row_pair(S.rQm, t, m);
        lo = f2(f2lo(mb) - f2lo(qm), f2hi(mb) - f2hi(qm));
        hi = f2(f2lo(mb) + f2lo(qm), f2hi(mb) + f2hi(qm));
    }
    uint32_t f[2][4];
#pragma unroll
    for (int c = 0; c < 4; c++) {
        // one rounding of the exact product, then the clamp on the biased code
        uint64_t uu = ffma2(x[c], gd[c], mb);           // bits: 0x4B400000 | (q + 2^(b-1))
        if (CLIP) uu = clamp2r(uu, lo, hi);
        f[0][c] = (uint32_t)uu;
        f[1][c] = (uint32_t)(uu >> 32);
    }
#pragma unroll
    for (int h = 0; h < 2; h++) {
        const int b = h ? b1 : b0;
        uint8_t *row = h ? r1 : r0;
        if (b == kPivot) {
            store_pivot(row, t.l, S.rA[t.row(2 * m + h)],
                        make_float4(h ? f2hi(x[0]) : f2lo(x[0]), h ? f2hi(x[1]) : f2lo(x[1]),
                                    h ? f2hi(x[2]) : f2lo(x[2]), h ? f2hi(x[3]) : f2lo(x[3])));
        } else {
            const uint32_t K = h ? inf.w : inf.y;
            const uint32_t v = f[h][0] + (f[h][1] << b) + (f[h][2] << (2 * b)) + (f[h][3] << (3 * b)) - K;
            store_segment(row, b, t.l, v);
        }
    }
}

template <bool CLIP>
__device__ __forceinline__ void ls_sums(const T &t, const Smem &S, const uint64_t (&x2)[8][4],
                                        const uint64_t (&g)[4], uint64_t (&n)[4], uint64_t (&d)[4]) {
    const uint64_t M2 = f2s(kMagic), nM2 = f2s(-kMagic);
#pragma unroll
    for (int p = 0; p < 4; p++) {
        uint64_t alo, ahi, qlo = 0, qhi = 0;
        row_pairs(S.rAl, t, p, alo, ahi);
        if (CLIP) row_pairs(S.rQm, t, p, qlo, qhi);
#pragma unroll
        for (int h = 0; h < 2; h++) {
            const int m = 2 * p + h;
            const uint64_t al = h ? ahi : alo;
#pragma unroll
            for (int c = 0; c < 4; c++) {
                uint64_t q = fadd2(ffma2(x2[m][c], g[c], M2), nM2);   // rne of the exact product
                if (CLIP) q = clamp2p(q, h ? qhi : qlo);
                const uint64_t aq = fmul2(al, q);
                n[c] = ffma2(aq, x2[m][c], n[c]);
                d[c] = ffma2(aq, q, d[c]);
            }
        }
    }
}

// One decode step of one row-unit head page staged in shared memory
// (App. C.3 steps 1-7; the Key-Row-Aware Dual-axis Fitting of Sec. 4.3 over
// the non-pivot rows). `ok` and `refill` as for the pipeline's process().
//
// MODE kReadout stops after the readout: it writes y and delta (delta_out) and
// leaves the page untouched. MODE kWriteback takes delta from the stage (the
// readout's, bit for bit), rebuilds Z exactly as the fused step does, and runs
// steps 4-6; its y is not computed.
template <int MODE, class Refill>
__device__ __forceinline__ bool decode_item(const T &t, const Smem &S, const Stage &st, float beta,
                                            float *y_out, float *delta_out, int fit_iters, bool ok,
                                            const Refill &refill) {
    uint16_t *page_r = (uint16_t *)st.page;
    uint16_t *page_c = (uint16_t *)(st.page + 256);
    // Row constants of the warp's band (warp-local).
    if (t.l < 16) {
        const int sl = t.row(t.l);                         // stored slot; i = its key row
        // The row table arrives with the page; a stage whose copies did not
        // complete still holds whatever it held, and the first CTA barrier ends
        // the item then. Offset and width are capped first, and the offset
        // rounded down to the 32 bytes every row start has, so that the page
        // reads before that barrier stay inside the stage and aligned whatever
        // the table holds.
        const uint32_t raw = st.slot[sl];
        const uint32_t region = (uint32_t)((const uint8_t *)st.q - st.page);
        const uint32_t off = min(raw & 0xFFFFu, region) & ~31u, bw = min((raw >> 16) & 0xFFu, (uint32_t)kPivot);
        const uint32_t info = off | (bw << 16) | (raw & 0xFF000000u);
        const int b = (int)bw, i = (int)(info >> 24);
        const float dg = st.gate[i];
        float a = dg, mu = 0.f, qm = 0.f, mb = 0.f;
        uint32_t K = 0;
        if (b != kPivot) {
            a = dg * (f16_val(page_r[i]) * (float)(1 << (8 - b)));
            qm = (float)((1 << (b - 1)) - 1);
            mu = __frcp_rn(qm);
            mb = kMagic + (float)(1 << (b - 1));
            K = pack_bias4(b);
        }
        a = fmaxf(a, 1e-30f);
        const float ki = st.k[i];
        S.rKap[sl] = ki * a;
        S.rBkp[sl] = __fdividef(beta * ki, a);
        if (MODE != kWriteback) S.rQa[sl] = st.q[i] * a;
        S.rA[sl] = a;
        S.rMu[sl] = mu;
        S.rQm[sl] = qm;
        S.rOff[sl] = -mb;
        S.rMb[sl] = mb;
        S.rInfo[sl] = make_uint2(info, K);
    }
    if (MODE != kReadout && t.tid < 128) S.colM[t.tid] = 0u;
    __syncwarp();
    // Step 1: Z = c_j q_ij (exact) or the FP16 value.
    uint64_t x2[8][4];
    {
        uint64_t cd[4];
        const uint2 cb = ((const uint2 *)page_c)[t.l];
        cd[0] = f2s(f16_val((uint16_t)(cb.x & 0xFFFFu)));
        cd[1] = f2s(f16_val((uint16_t)(cb.x >> 16)));
        cd[2] = f2s(f16_val((uint16_t)(cb.y & 0xFFFFu)));
        cd[3] = f2s(f16_val((uint16_t)(cb.y >> 16)));
#pragma unroll
        for (int m = 0; m < 8; m++) load_pair(t, S, st.page, m, cd, x2[m]);
    }
    float rs[16];
    if constexpr (MODE == kWriteback) {
        if (__syncthreads_or(!ok)) return false;
        refill();
        // Z += (beta k_i / a_i) delta_j with the readout's delta; row sums of |Z|.
        uint64_t dl[4];
        col_dup(st.v, t.l, dl);
#pragma unroll
        for (int p = 0; p < 4; p++) {
            uint64_t blo, bhi;
            row_pairs(S.rBkp, t, p, blo, bhi);
#pragma unroll
            for (int c = 0; c < 4; c++) {
                x2[2 * p][c] = ffma2(blo, dl[c], x2[2 * p][c]);
                x2[2 * p + 1][c] = ffma2(bhi, dl[c], x2[2 * p + 1][c]);
            }
#pragma unroll
            for (int h = 0; h < 2; h++) {
                const uint64_t(&xm)[4] = x2[2 * p + h];
                rs[4 * p + 2 * h] = (fabsf(f2lo(xm[0])) + fabsf(f2lo(xm[1]))) +
                                    (fabsf(f2lo(xm[2])) + fabsf(f2lo(xm[3])));
                rs[4 * p + 2 * h + 1] = (fabsf(f2hi(xm[0])) + fabsf(f2hi(xm[1]))) +
                                        (fabsf(f2hi(xm[2])) + fabsf(f2hi(xm[3])));
            }
        }
    } else {
    // Step 2a: retrieval u_j = sum_i k_i a_i Z_ij.
    {
        uint64_t ua[4] = {0, 0, 0, 0}, ub[4] = {0, 0, 0, 0};
#pragma unroll
        for (int p = 0; p < 4; p++) {
            uint64_t klo, khi;
            row_pairs(S.rKap, t, p, klo, khi);
#pragma unroll
            for (int c = 0; c < 4; c++) {
                ua[c] = ffma2(klo, x2[2 * p][c], ua[c]);
                ub[c] = ffma2(khi, x2[2 * p + 1][c], ub[c]);
            }
        }
        const float v[4] = {pair_sum(fadd2(ua[0], ub[0])), pair_sum(fadd2(ua[1], ub[1])),
                            pair_sum(fadd2(ua[2], ub[2])), pair_sum(fadd2(ua[3], ub[3]))};
        cols_to_red(t, S.red, 0, v);
    }
    if (__syncthreads_or(!ok)) return false;
    if (t.tid < 128) {
        float s = 0.f;
#pragma unroll
        for (int wv = 0; wv < 8; wv++) s += S.red[wv * 128 + t.tid];
        S.colD[t.tid] = st.v[t.tid] - s;                   // delta_j = v_j - u_j
        if (MODE == kReadout) delta_out[t.tid] = S.colD[t.tid];
    }
    refill();
    __syncthreads();
    // Step 2b-3: Z += (beta k_i / a_i) delta_j; readout partials q_i a_i Z_ij.
    {
        uint64_t dl[4];
        col_dup(S.colD, t.l, dl);
        uint64_t ya[4] = {0, 0, 0, 0}, yb[4] = {0, 0, 0, 0};
#pragma unroll
        for (int p = 0; p < 4; p++) {
            uint64_t blo, bhi, qlo, qhi;
            row_pairs(S.rBkp, t, p, blo, bhi);
            row_pairs(S.rQa, t, p, qlo, qhi);
#pragma unroll
            for (int c = 0; c < 4; c++) {
                x2[2 * p][c] = ffma2(blo, dl[c], x2[2 * p][c]);
                x2[2 * p + 1][c] = ffma2(bhi, dl[c], x2[2 * p + 1][c]);
                ya[c] = ffma2(qlo, x2[2 * p][c], ya[c]);
                yb[c] = ffma2(qhi, x2[2 * p + 1][c], yb[c]);
            }
            if (MODE == kFused) {
#pragma unroll
                for (int h = 0; h < 2; h++) {
                    const uint64_t(&xm)[4] = x2[2 * p + h];
                    rs[4 * p + 2 * h] = (fabsf(f2lo(xm[0])) + fabsf(f2lo(xm[1]))) +
                                        (fabsf(f2lo(xm[2])) + fabsf(f2lo(xm[3])));
                    rs[4 * p + 2 * h + 1] = (fabsf(f2hi(xm[0])) + fabsf(f2hi(xm[1]))) +
                                            (fabsf(f2hi(xm[2])) + fabsf(f2hi(xm[3])));
                }
            }
        }
        const float v[4] = {pair_sum(fadd2(ya[0], yb[0])), pair_sum(fadd2(ya[1], yb[1])),
                            pair_sum(fadd2(ya[2], yb[2])), pair_sum(fadd2(ya[3], yb[3]))};
        cols_to_red(t, S.red, 2, v);
    }
    if (MODE == kReadout) {
        __syncthreads();
        if (t.tid < 128) {                              // the fused step's summation order
            float s = S.red[(2 * 8) * 128 + t.tid];
#pragma unroll
            for (int wv = 1; wv < 8; wv++) s += S.red[(2 * 8 + wv) * 128 + t.tid];
            y_out[t.tid] = s;
        }
        return true;
    }
    }
    // Step 4: row factors r_i = m_i^(1/2) w_i^(-1/2) of the integer rows.
    {
        int rr;
        const float sz = warp_row_sums(rs, t.l, rr);
        const int sl = t.row(rr);
        if ((t.l & 1) == 0) {
            const uint32_t info = S.rInfo[sl].x;
            const int b = (int)((info >> 16) & 0xFFu), i = (int)(info >> 24);
            if (b == kPivot) {
                S.rRho[sl] = 1.f;
                S.rAl[sl] = 0.f;
                page_r[i] = 0;
            } else {
                const float a = S.rA[sl];
                const float m = (a * sz) * (1.0f / 128.0f);
                const float rf = __half2float(__float2half_rn(
                    fminf(fmaxf(__fmul_rn(sqrtf(m), st.wis[i]), kF16Min), kF16Max)));
                const float rz = rf * (float)(1 << (8 - b));          // r_i zs_i, exact
                S.rRho[sl] = __frcp_rn(rz) * a;                       // X' = rho_i X = (rho_i a_i) Z
                S.rAl[sl] = st.w2[i] * (rz * rz);                     // w_i^2 (r_i zs_i)^2
                page_r[i] = f16_bits(rf);
            }
        }
    }
    __syncwarp();
    // X' = rho_i X; clip-free column start max_i fp32(|X'_ij| mu_i) (order-free
    // atomic max on the non-negative float bits; pivot rows have mu = 0).
    {
        float cm[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int p = 0; p < 4; p++) {
            uint64_t rlo, rhi, mlo, mhi;
            row_pairs(S.rRho, t, p, rlo, rhi);
            row_pairs(S.rMu, t, p, mlo, mhi);
#pragma unroll
            for (int c = 0; c < 4; c++) {
                x2[2 * p][c] = fmul2(x2[2 * p][c], rlo);
                x2[2 * p + 1][c] = fmul2(x2[2 * p + 1][c], rhi);
                const uint64_t e0 = fmul2(x2[2 * p][c], mlo), e1 = fmul2(x2[2 * p + 1][c], mhi);
                cm[c] = fmax3(cm[c], fabsf(f2lo(e0)), fabsf(f2hi(e0)));
                cm[c] = fmax3(cm[c], fabsf(f2lo(e1)), fabsf(f2hi(e1)));
            }
        }
#pragma unroll
        for (int c = 0; c < 4; c++) atomicMax(&S.colM[4 * t.l + c], __float_as_uint(cm[c]));
    }
    if (t.tid == 0) {
        S.flags[1] = 0;
        S.flags[2] = 0;
    }
    __syncthreads();
    // Column start (threads 0..127) beside the readout sums (threads 128..255).
    if (t.tid < 128) {
        const float c0 = __uint_as_float(S.colM[t.tid]);
        if (c0 > kF16Max) S.flags[1] = 1;                 // start capped: codes may clip
        const float cc = fminf(fmaxf(c0, kF16Min), kF16Max);
        S.colC[t.tid] = cc;
        S.colG[t.tid] = __frcp_rn(cc);
    } else if (MODE == kFused) {
        const int j = t.tid - 128;
        float s = S.red[(2 * 8) * 128 + j];
#pragma unroll
        for (int wv = 1; wv < 8; wv++) s += S.red[(2 * 8 + wv) * 128 + j];
        y_out[j] = s;
    }
    __syncthreads();
    // Step 5: fixed-code least-squares updates of c over the integer rows.
    const bool clip0 = S.flags[1] != 0;
    for (int it = 0; it < fit_iters; it++) {
        uint64_t g[4];
        col_dup(S.colG, t.l, g);
        uint64_t n[4] = {0, 0, 0, 0}, d[4] = {0, 0, 0, 0};
        if (it > 0 || clip0) ls_sums<true>(t, S, x2, g, n, d);
        else ls_sums<false>(t, S, x2, g, n, d);
        {
            const float vn[4] = {pair_sum(n[0]), pair_sum(n[1]), pair_sum(n[2]), pair_sum(n[3])};
            const float vd[4] = {pair_sum(d[0]), pair_sum(d[1]), pair_sum(d[2]), pair_sum(d[3])};
            cols_to_red(t, S.red, 0, vn);
            cols_to_red(t, S.red, 1, vd);
        }
        __syncthreads();
        if (t.tid < 128) {
            float num = 0.f, den = 0.f;
#pragma unroll
            for (int wv = 0; wv < 8; wv++) {
                num += S.red[wv * 128 + t.tid];
                den += S.red[(8 + wv) * 128 + t.tid];
            }
            float c = S.colC[t.tid];
            if (den > 0.f) c = fminf(fmaxf(__fdividef(num, den), kF16Min), kF16Max);
            if (it + 1 < fit_iters) {
                S.colC[t.tid] = c;
                S.colG[t.tid] = __frcp_rn(c);
            } else {
                const float cf = __half2float(__float2half_rn(c));
                const float gi = __frcp_rn(cf);
                page_c[t.tid] = f16_bits(cf);
                S.colG[t.tid] = gi;
                // a code can clip only if |X'_ij| / c_j >= qmax_i + 1/2 for some i,
                // i.e. max_i |X'_ij| mu_i / c_j >= 1 + 1/(2 qmax_i) >= 1 + 1/254
                if (__fmul_rn(__uint_as_float(S.colM[t.tid]), gi) >= (1.0f + 0.5f / 127.0f) * 0.999999f)
                    S.flags[2] = 1;
            }
        }
        __syncthreads();
    }
    // Step 6: final codes with the stored scales, written in place.
    {
        uint64_t gd[4];
        col_dup(S.colG, t.l, gd);
        if (S.flags[2]) {
#pragma unroll
            for (int m = 0; m < 8; m++) store_pair<true>(t, S, st.page, m, x2[m], gd);
        } else {
#pragma unroll
            for (int m = 0; m < 8; m++) store_pair<false>(t, S, st.page, m, x2[m], gd);
        }
    }
    return true;
}

template <int MODE>
__global__ void __launch_bounds__(kThreads, 2) decode_rows_kernel(DecodeArgs a) {
    extern __shared__ __align__(128) uint8_t smem[];
    const T t;
    const Smem S(smem);
    if ((int)blockIdx.x >= a.items) return;
    const int grp = a.Hv / a.Hk;
    for (int h = t.tid; h < a.Hv; h += kThreads) {
        S.hoff[h] = a.tab.head_off[h];
        S.hbytes[h] = a.tab.head_bytes[h];
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
        p, S.bars, [&](int h, int b, int slot, int s, int lane) { issue<MODE>(a, S, h, b, slot, s, lane); },
        [&](int h, int b, int, int s, bool ok, const auto &refill) {
            const size_t u = (size_t)b * a.Hv + h;
            const Stage st(S.stages + (size_t)s * a.stage_bytes, a.page_region);
            const float beta = *st.beta;                   // staged with the page
            return decode_item<MODE>(t, S, st, beta, MODE == kWriteback ? nullptr : a.y + u * 128,
                                     MODE == kReadout ? a.delta + u * 128 : nullptr, a.fit_iters, ok,
                                     refill);
        },
        [&](int h, int slot, int s) {
            if (MODE != kReadout)
                bulk_store(a.pool + (uint64_t)slot * a.stride + S.hoff[h],
                           S.stages + (size_t)s * a.stage_bytes, S.hbytes[h]);
        });
}

}  // namespace rk

stepq_status launch_decode_rows(const stepq_plan *p, int layer, uint8_t *pool, int pool_slots,
                                const int32_t *slots, int B, const float *q, const float *k,
                                const float *v, const float *beta, const float *gate, float *y,
                                cudaStream_t s) {
    return launch_decode_rows_mode(p, layer, pool, pool_slots, slots, B, q, k, v, beta, gate, y,
                                   nullptr, rk::kFused, s);
}

stepq_status launch_decode_rows_mode(const stepq_plan *p, int layer, uint8_t *pool, int pool_slots,
                                     const int32_t *slots, int B, const float *q, const float *k,
                                     const float *v, const float *beta, const float *gate, float *y,
                                     float *delta, int mode, cudaStream_t s) {
    const int Hv = p->cfg.n_value_heads;
    if (Hv > rk::kMaxHv) return STEPQ_ERR_UNSUPPORTED;
    uint32_t maxb = 0;
    for (int h = 0; h < Hv; h++) maxb = p->head_bytes[(size_t)layer * Hv + h] > maxb
                                            ? p->head_bytes[(size_t)layer * Hv + h] : maxb;
    rk::DecodeArgs a{};
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
    a.stage_bytes = a.page_region + rk::kVecBytes;
    // as many stages (2..4) as keep two CTAs per SM
    int stages = (int)((113 * 1024 - rk::kOffStages) / a.stage_bytes);
    stages = stages < 2 ? 2 : (stages > 4 ? 4 : stages);
    a.n_stages = stages;
    a.fit_iters = p->cfg.fit_iters;
    const int smem = rk::kOffStages + stages * (int)a.stage_bytes;
    const void *fn = mode == rk::kReadout     ? (const void *)rk::decode_rows_kernel<rk::kReadout>
                     : mode == rk::kWriteback ? (const void *)rk::decode_rows_kernel<rk::kWriteback>
                                              : (const void *)rk::decode_rows_kernel<rk::kFused>;
    if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
        return STEPQ_ERR_CUDA;
    int dev = 0, sms = 1;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    int grid = 2 * (sms > 0 ? sms : 1);
    if (grid > a.items) grid = a.items;
    if (mode == rk::kReadout) rk::decode_rows_kernel<rk::kReadout><<<grid, kThreads, smem, s>>>(a);
    else if (mode == rk::kWriteback) rk::decode_rows_kernel<rk::kWriteback><<<grid, kThreads, smem, s>>>(a);
    else rk::decode_rows_kernel<rk::kFused><<<grid, kThreads, smem, s>>>(a);
    return cudaGetLastError() == cudaSuccess ? STEPQ_OK : STEPQ_ERR_CUDA;
}

}  // namespace stepq
