// Row-unit (KDA, per-key-channel gate) decode step: the persistent, bulk-async
// pipelined kernel over row-major pages with one width per key row.
//
// Tile mapping: warp w owns key rows 16w..16w+15; lane l owns the value
// columns 4l..4l+3. All lanes of a warp work on the same row at a time, so the
// row's width is uniform across the warp (no divergence) and a lane's 4 codes
// are one word (8-bit), half-word (4-bit), byte (2-bit), three bytes (6-bit,
// assembled from two words) or four FP16 values (pivot row). A thread holds its
// 16 rows x 2 column pairs as packed f32x2 registers: column constants of a lane
// are adjacent in shared memory, per-row constants are stored as duplicated
// pairs and read with broadcast loads.
//
// Per row i the tile holds Z with X_ij = a_i Z_ij: a_i = d_i r_i zs_i and
// Z = c_j q_ij for an integer row (zs_i = 2^(8 - b_i), the normalised codebook
// of App. C.1), a_i = d_i and Z = the FP16 value for a pivot row. Pivot rows
// stay out of the column fit (rho a = 1, mu = alpha = 0).
#include "async.cuh"
#include "device.cuh"
#include "internal.h"
#include "pipeline.cuh"
#include "tile.cuh"

namespace stepq {
namespace rk {

constexpr int kVecBytes = 6 * 512 + 512 + 128;         // q k v gate w2 wis | row_off | row_bits

// ------------------------------------------------------------ shared layout
constexpr int kOffBars = 0;                            // uint64 [8]
constexpr int kOffFlags = 64;                          // int [16]
constexpr int kOffRed = 128;                           // float [3][8][128] cross-warp partials
constexpr int kOffColC = kOffRed + 3 * 8 * 128 * 4;    // float [128] c_j (start / iterate)
constexpr int kOffColM = kOffColC + 512;               // u32 [128] bits of max_i fp32(|X'_ij| mu_i)
constexpr int kOffColD = kOffColM + 512;               // float [128] delta_j
constexpr int kOffColG = kOffColD + 512;               // float [128] 1/c_j
constexpr int kOffRows = kOffColG + 512;               // float4 [4][128] per-row constants
constexpr int kMaxHv = 256;                            // value heads per layer (launch check)
constexpr int kOffHead = kOffRows + 4 * 128 * 16;      // u64 off | u32 bytes | u8 key head
constexpr int kOffStages = (kOffHead + kMaxHv * 13 + 127) / 128 * 128;

struct Smem {
    uint64_t *bars;
    int *flags;
    float *red, *colC, *colD, *colG;
    uint32_t *colM;
    float4 *rowK;   // (kappa, kappa, beta k / a, beta k / a), kappa = k a
    float4 *rowQ;   // (q a, q a, a, a)
    float4 *rowF;   // (rho a, rho a, alpha, alpha), alpha = w^2 (r zs)^2
    float4 *rowM;   // (mu, mu, qmax, qmax): 1/qmax of the row's width (0 for pivots)
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
        rowK = (float4 *)(s + kOffRows);
        rowQ = rowK + 128;
        rowF = rowK + 256;
        rowM = rowK + 384;
        hoff = (uint64_t *)(s + kOffHead);
        hbytes = (uint32_t *)(s + kOffHead + kMaxHv * 8);
        hkey = s + kOffHead + kMaxHv * 12;
        stages = s + kOffStages;
    }
};

struct Stage {
    uint8_t *page;
    float *q, *k, *v, *gate, *w2, *wis;
    uint32_t *roff;
    uint8_t *rbits;
    __device__ __forceinline__ Stage(uint8_t *base, uint32_t page_region) {
        page = base;
        q = (float *)(base + page_region);
        k = q + 128;
        v = q + 256;
        gate = q + 384;
        w2 = q + 512;
        wis = q + 640;
        roff = (uint32_t *)(q + 768);
        rbits = (uint8_t *)(q + 896);
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

// Duplicated row constants of row i: the (x, x) and (z, z) pairs of a float4.
__device__ __forceinline__ void row_dup(const float4 *v, int i, uint64_t &xx, uint64_t &zz) {
    const uint4 q = *(const uint4 *)&v[i];
    xx = u2pair(q.x, q.y);
    zz = u2pair(q.z, q.w);
}
// The lane's two column pairs of a per-column vector.
__device__ __forceinline__ void col_pairs(const float *v, int l, uint64_t &p0, uint64_t &p1) {
    const uint4 q = *(const uint4 *)&v[4 * l];
    p0 = u2pair(q.x, q.y);
    p1 = u2pair(q.z, q.w);
}
__device__ __forceinline__ void cols_to_red(const T &t, float *red, int reg, const float (&v)[4]) {
    *(float4 *)&red[(reg * 8 + t.w) * 128 + 4 * t.l] = make_float4(v[0], v[1], v[2], v[3]);
}

// Row widths of the warp's band, one byte each in four registers.
struct Widths {
    uint32_t w[4];
    __device__ __forceinline__ Widths(const uint8_t *rbits, int band) {
        const uint4 q = *(const uint4 *)&rbits[16 * band];
        w[0] = q.x; w[1] = q.y; w[2] = q.z; w[3] = q.w;
    }
    __device__ __forceinline__ int operator[](int r) const { return (w[r >> 2] >> (8 * (r & 3))) & 0xFF; }
};

// The lane's 4 codes of a row of width B (B < 8), right-aligned in one word.
template <int B>
__device__ __forceinline__ uint32_t lane_codes(const uint8_t *row, int l) {
    if (B == 2) return row[l];
    if (B == 4) return ((const uint16_t *)row)[l];
    // B == 6: bytes 3l..3l+2 of the row (the next word may lie past the row;
    // it stays inside the stage and its bits are masked off)
    const uint32_t *wp = (const uint32_t *)row;
    const int byte = 3 * l;
    return __funnelshift_r(wp[byte >> 2], wp[(byte >> 2) + 1], 8 * (byte & 3)) & 0xFFFFFFu;
}

// Decode the lane's 4 codes of one integer row into (c q) pairs: each code is
// dropped into the zero mantissa bits of 1.5*2^23 (one logic op), the offset
// 1.5*2^23 + 2^(B-1) comes off exactly and c_j q_ij is exact in fp32.
template <int B>
__device__ __forceinline__ void decode_row(const uint8_t *row, int l, uint64_t c01, uint64_t c23,
                                           uint64_t &x0, uint64_t &x1) {
    uint32_t f0, f1, f2, f3;
    if (B == 8) {
        const uint32_t w = ((const uint32_t *)row)[l];
        f0 = __byte_perm(w, kMagicBits, 0x7650);
        f1 = __byte_perm(w, kMagicBits, 0x7651);
        f2 = __byte_perm(w, kMagicBits, 0x7652);
        f3 = __byte_perm(w, kMagicBits, 0x7653);
    } else {
        constexpr uint32_t mask = (1u << B) - 1u;
        const uint32_t x = lane_codes<B>(row, l);
        f0 = and_or(x, mask, kMagicBits);
        f1 = and_or(x >> B, mask, kMagicBits);
        f2 = and_or(x >> (2 * B), mask, kMagicBits);
        f3 = and_or(x >> (3 * B), mask, kMagicBits);
    }
    const uint64_t off = f2s(-(kMagic + (float)(1 << (B - 1))));
    x0 = fmul2(fadd2(u2pair(f0, f1), off), c01);
    x1 = fmul2(fadd2(u2pair(f2, f3), off), c23);
}

// Pack the lane's 4 codes (float bit patterns 0x4B400000 | u) of a row of
// width B into the row: the known high bits are summed and subtracted once.
template <int B>
__device__ __forceinline__ void store_row(uint8_t *row, int l, uint32_t f0, uint32_t f1, uint32_t f2,
                                          uint32_t f3) {
    if (B == 8) {
        const uint32_t lo = __byte_perm(f0, f1, 0x0040), hi = __byte_perm(f2, f3, 0x0040);
        ((uint32_t *)row)[l] = __byte_perm(lo, hi, 0x5410);
        return;
    }
    constexpr uint32_t K = kMagicBits + (kMagicBits << B) + (kMagicBits << (2 * B)) + (kMagicBits << (3 * B));
    const uint32_t v = f0 + (f1 << B) + (f2 << (2 * B)) + (f3 << (3 * B)) - K;   // 4B bits
    if (B == 2) {
        row[l] = (uint8_t)v;
    } else if (B == 4) {
        ((uint16_t *)row)[l] = (uint16_t)v;
    } else {
        // 24 bits per lane: lanes 4g..4g+2 each store one of the words 3g..3g+2
        const uint32_t nb = __shfl_down_sync(0xffffffffu, v, 1);
        const int j = l & 3;
        if (j < 3) ((uint32_t *)row)[3 * (l >> 2) + j] = (v >> (8 * j)) | (nb << (24 - 8 * j));
    }
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
    unsigned int *err;
    int n_stages;
    uint32_t page_region, stage_bytes;
    int fit_iters;
};

__device__ __forceinline__ void issue(const DecodeArgs &a, const Smem &S, int h, int b, int slot, int s) {
    uint64_t *bar = &S.bars[s];
    Stage st(S.stages + (size_t)s * a.stage_bytes, a.page_region);
    const uint32_t nb = S.hbytes[h];
    const int hk = S.hkey[h];
    mbar_arrive_tx(bar, nb + kVecBytes);
    bulk_load(st.page, a.pool + (uint64_t)slot * a.stride + S.hoff[h], nb, bar);
    bulk_load(st.q, a.q + ((size_t)b * a.Hk + hk) * 128, 512, bar);
    bulk_load(st.k, a.k + ((size_t)b * a.Hk + hk) * 128, 512, bar);
    bulk_load(st.v, a.v + ((size_t)b * a.Hv + h) * 128, 512, bar);
    bulk_load(st.gate, a.gate + ((size_t)b * a.Hv + h) * 128, 512, bar);
    bulk_load(st.w2, a.tab.w2 + (size_t)h * 128, 512, bar);
    bulk_load(st.wis, a.tab.wis + (size_t)h * 128, 512, bar);
    bulk_load(st.roff, a.tab.row_off + (size_t)h * 128, 512, bar);
    bulk_load(st.rbits, a.tab.row_bits + (size_t)h * 128, 128, bar);
}

// Decode of one row r of the thread's band at its width.
__device__ __forceinline__ void load_row(const T &t, const Stage &st, int B, int r, uint64_t c01,
                                         uint64_t c23, uint64_t &x0, uint64_t &x1) {
    const uint8_t *row = st.page + st.roff[t.row(r)];
    switch (B) {
    case 2: decode_row<2>(row, t.l, c01, c23, x0, x1); break;
    case 4: decode_row<4>(row, t.l, c01, c23, x0, x1); break;
    case 6: decode_row<6>(row, t.l, c01, c23, x0, x1); break;
    case 8: decode_row<8>(row, t.l, c01, c23, x0, x1); break;
    default: {
        const uint2 v = ((const uint2 *)row)[t.l];
        x0 = f2(f16_val((uint16_t)(v.x & 0xFFFFu)), f16_val((uint16_t)(v.x >> 16)));
        x1 = f2(f16_val((uint16_t)(v.y & 0xFFFFu)), f16_val((uint16_t)(v.y >> 16)));
    } break;
    }
}

// Final codes of one row: q = rne(X' / c_j) (clamped to +-qmax when CLIP), or
// fp16(a Z) for a pivot row.
template <bool CLIP>
__device__ __forceinline__ void store_final(const T &t, const Smem &S, const Stage &st, int B, int r,
                                            uint64_t x0, uint64_t x1, uint64_t g01, uint64_t g23) {
    const int i = t.row(r);
    uint8_t *row = st.page + st.roff[i];
    if (B == kPivot) {
        const float a = S.rowQ[i].z;
        const uint32_t w0 = (uint32_t)f16_bits(f16_round_sat(a * f2lo(x0))) |
                            ((uint32_t)f16_bits(f16_round_sat(a * f2hi(x0))) << 16);
        const uint32_t w1 = (uint32_t)f16_bits(f16_round_sat(a * f2lo(x1))) |
                            ((uint32_t)f16_bits(f16_round_sat(a * f2hi(x1))) << 16);
        ((uint2 *)row)[t.l] = make_uint2(w0, w1);
        return;
    }
    uint64_t t0 = fmul2(x0, g01), t1 = fmul2(x1, g23);
    if (CLIP) {
        const float qm = S.rowM[i].z;
        t0 = clamp2(t0, qm);
        t1 = clamp2(t1, qm);
    }
    const uint64_t mb = f2s(kMagic + (float)(1 << (B - 1)));
    const uint64_t u0 = fadd2(t0, mb), u1 = fadd2(t1, mb);   // bits: 0x4B400000 | (q + 2^(B-1))
    const uint32_t f0 = (uint32_t)u0, f1 = (uint32_t)(u0 >> 32), f2v = (uint32_t)u1, f3 = (uint32_t)(u1 >> 32);
    switch (B) {
    case 2: store_row<2>(row, t.l, f0, f1, f2v, f3); break;
    case 4: store_row<4>(row, t.l, f0, f1, f2v, f3); break;
    case 6: store_row<6>(row, t.l, f0, f1, f2v, f3); break;
    default: store_row<8>(row, t.l, f0, f1, f2v, f3); break;
    }
}

template <bool CLIP>
__device__ __forceinline__ void ls_sums(const T &t, const Smem &S, const uint64_t (&x2)[16][2], uint64_t g01,
                                        uint64_t g23, uint64_t (&n)[2], uint64_t (&d)[2]) {
    const uint64_t M2 = f2s(kMagic), nM2 = f2s(-kMagic);
#pragma unroll
    for (int r = 0; r < 16; r++) {
        uint64_t rho, al;
        row_dup(S.rowF, t.row(r), rho, al);
        uint64_t q0 = fadd2(fadd2(fmul2(x2[r][0], g01), M2), nM2);
        uint64_t q1 = fadd2(fadd2(fmul2(x2[r][1], g23), M2), nM2);
        if (CLIP) {
            const float qm = S.rowM[t.row(r)].z;
            q0 = clamp2(q0, qm);
            q1 = clamp2(q1, qm);
        }
        const uint64_t a0 = fmul2(al, q0), a1 = fmul2(al, q1);
        n[0] = ffma2(a0, x2[r][0], n[0]);
        n[1] = ffma2(a1, x2[r][1], n[1]);
        d[0] = ffma2(a0, q0, d[0]);
        d[1] = ffma2(a1, q1, d[1]);
    }
}

template <bool CLIP>
__device__ __forceinline__ void final_codes(const T &t, const Smem &S, const Stage &st, const Widths &wd,
                                            const uint64_t (&x2)[16][2]) {
    uint64_t g01, g23;
    col_pairs(S.colG, t.l, g01, g23);
#pragma unroll
    for (int r = 0; r < 16; r++) store_final<CLIP>(t, S, st, wd[r], r, x2[r][0], x2[r][1], g01, g23);
}

// One decode step of one row-unit head page staged in shared memory
// (App. C.3 steps 1-7; the Key-Row-Aware Dual-axis Fitting of Sec. 4.3 over
// the non-pivot rows). `ok` and `refill` as for the pipeline's process().
template <class Refill>
__device__ __forceinline__ bool decode_item(const T &t, const Smem &S, const Stage &st, float beta,
                                            float *y_out, int fit_iters, bool ok, const Refill &refill) {
    uint16_t *page_r = (uint16_t *)st.page;
    uint16_t *page_c = (uint16_t *)(st.page + 256);
    // Row constants of the warp's band (warp-local).
    if (t.l < 16) {
        const int i = t.row(t.l);
        const int b = st.rbits[i];
        const float dg = st.gate[i];
        float a = dg, mu = 0.f, qm = 0.f;
        if (b != kPivot) {
            a = dg * (f16_val(page_r[i]) * (float)(1 << (8 - b)));
            qm = (float)((1 << (b - 1)) - 1);
            mu = __frcp_rn(qm);
        }
        a = fmaxf(a, 1e-30f);
        const float ki = st.k[i], kap = ki * a, bkp = __fdividef(beta * ki, a), qa = st.q[i] * a;
        S.rowK[i] = make_float4(kap, kap, bkp, bkp);
        S.rowQ[i] = make_float4(qa, qa, a, a);
        S.rowM[i] = make_float4(mu, mu, qm, qm);
    }
    if (t.tid < 128) S.colM[t.tid] = 0u;
    // Step 1: Z = c_j q_ij (exact) or the FP16 value.
    uint64_t x2[16][2];
    {
        const uint2 cb = ((const uint2 *)page_c)[t.l];
        const uint64_t c01 = f2(f16_val((uint16_t)(cb.x & 0xFFFFu)), f16_val((uint16_t)(cb.x >> 16)));
        const uint64_t c23 = f2(f16_val((uint16_t)(cb.y & 0xFFFFu)), f16_val((uint16_t)(cb.y >> 16)));
#pragma unroll
        const Widths wd(st.rbits, t.w);
#pragma unroll
        for (int r = 0; r < 16; r++) load_row(t, st, wd[r], r, c01, c23, x2[r][0], x2[r][1]);
    }
    __syncwarp();
    // Step 2a: retrieval u_j = sum_i k_i a_i Z_ij.
    {
        uint64_t ua[2] = {0, 0}, ub[2] = {0, 0};
#pragma unroll
        for (int r = 0; r < 16; r += 2) {
            uint64_t k0, k1, z;
            row_dup(S.rowK, t.row(r), k0, z);
            row_dup(S.rowK, t.row(r + 1), k1, z);
            ua[0] = ffma2(k0, x2[r][0], ua[0]);
            ua[1] = ffma2(k0, x2[r][1], ua[1]);
            ub[0] = ffma2(k1, x2[r + 1][0], ub[0]);
            ub[1] = ffma2(k1, x2[r + 1][1], ub[1]);
        }
        const uint64_t s0 = fadd2(ua[0], ub[0]), s1 = fadd2(ua[1], ub[1]);
        const float v[4] = {f2lo(s0), f2hi(s0), f2lo(s1), f2hi(s1)};
        cols_to_red(t, S.red, 0, v);
    }
    if (__syncthreads_or(!ok)) return false;
    if (t.tid < 128) {
        float s = 0.f;
#pragma unroll
        for (int wv = 0; wv < 8; wv++) s += S.red[wv * 128 + t.tid];
        S.colD[t.tid] = st.v[t.tid] - s;                   // delta_j = v_j - u_j
    }
    refill();
    __syncthreads();
    // Step 2b-3: Z += (beta k_i / a_i) delta_j; readout partials q_i a_i Z_ij.
    float rs[16];
    {
        uint64_t d01, d23;
        col_pairs(S.colD, t.l, d01, d23);
        uint64_t ya[2] = {0, 0}, yb[2] = {0, 0};
#pragma unroll
        for (int r = 0; r < 16; r++) {
            uint64_t z, bk, qa;
            row_dup(S.rowK, t.row(r), z, bk);
            row_dup(S.rowQ, t.row(r), qa, z);
            x2[r][0] = ffma2(bk, d01, x2[r][0]);
            x2[r][1] = ffma2(bk, d23, x2[r][1]);
            if (r & 1) {
                yb[0] = ffma2(qa, x2[r][0], yb[0]);
                yb[1] = ffma2(qa, x2[r][1], yb[1]);
            } else {
                ya[0] = ffma2(qa, x2[r][0], ya[0]);
                ya[1] = ffma2(qa, x2[r][1], ya[1]);
            }
            rs[r] = (fabsf(f2lo(x2[r][0])) + fabsf(f2hi(x2[r][0]))) +
                    (fabsf(f2lo(x2[r][1])) + fabsf(f2hi(x2[r][1])));
        }
        const uint64_t s0 = fadd2(ya[0], yb[0]), s1 = fadd2(ya[1], yb[1]);
        const float v[4] = {f2lo(s0), f2hi(s0), f2lo(s1), f2hi(s1)};
        cols_to_red(t, S.red, 2, v);
    }
    // Step 4: row factors r_i = m_i^(1/2) w_i^(-1/2) of the integer rows.
    {
        int rr;
        const float sz = warp_row_sums(rs, t.l, rr);
        const int i = t.row(rr);
        const int b = st.rbits[i];
        if ((t.l & 1) == 0) {
            if (b == kPivot) {
                S.rowF[i] = make_float4(1.f, 1.f, 0.f, 0.f);
                page_r[i] = 0;
            } else {
                const float a = S.rowQ[i].z;
                const float m = (a * sz) * (1.0f / 128.0f);
                const float rf = __half2float(__float2half_rn(
                    fminf(fmaxf(__fmul_rn(sqrtf(m), st.wis[i]), kF16Min), kF16Max)));
                const float rz = rf * (float)(1 << (8 - b));          // r_i zs_i, exact
                const float rho_a = __frcp_rn(rz) * a;                // X' = rho_i X = (rho_i a_i) Z
                const float al = st.w2[i] * (rz * rz);                // w_i^2 (r_i zs_i)^2
                S.rowF[i] = make_float4(rho_a, rho_a, al, al);
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
        for (int r = 0; r < 16; r += 2) {
            uint64_t rho0, rho1, mu0, mu1, z;
            row_dup(S.rowF, t.row(r), rho0, z);
            row_dup(S.rowF, t.row(r + 1), rho1, z);
            row_dup(S.rowM, t.row(r), mu0, z);
            row_dup(S.rowM, t.row(r + 1), mu1, z);
#pragma unroll
            for (int p = 0; p < 2; p++) {
                x2[r][p] = fmul2(x2[r][p], rho0);
                x2[r + 1][p] = fmul2(x2[r + 1][p], rho1);
                const uint64_t m0 = fmul2(x2[r][p], mu0), m1 = fmul2(x2[r + 1][p], mu1);
                cm[2 * p] = fmax3(cm[2 * p], fabsf(f2lo(m0)), fabsf(f2lo(m1)));
                cm[2 * p + 1] = fmax3(cm[2 * p + 1], fabsf(f2hi(m0)), fabsf(f2hi(m1)));
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
    } else {
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
        uint64_t g01, g23;
        col_pairs(S.colG, t.l, g01, g23);
        uint64_t n[2] = {0, 0}, d[2] = {0, 0};
        if (it > 0 || clip0) ls_sums<true>(t, S, x2, g01, g23, n, d);
        else ls_sums<false>(t, S, x2, g01, g23, n, d);
        {
            const float vn[4] = {f2lo(n[0]), f2hi(n[0]), f2lo(n[1]), f2hi(n[1])};
            const float vd[4] = {f2lo(d[0]), f2hi(d[0]), f2lo(d[1]), f2hi(d[1])};
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
    const Widths wd(st.rbits, t.w);
    if (S.flags[2]) final_codes<true>(t, S, st, wd, x2);
    else final_codes<false>(t, S, st, wd, x2);
    return true;
}

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
    const pipe::Shape p{a.items, a.nb, a.n_stages, a.slots, a.pool_slots, a.err};
    pipe::run(
        p, S.bars, [&](int h, int b, int slot, int s) { issue(a, S, h, b, slot, s); },
        [&](int h, int b, int, int s, bool ok, const auto &refill) {
            const float beta = a.beta[(size_t)b * a.Hv + h];
            const Stage st(S.stages + (size_t)s * a.stage_bytes, a.page_region);
            return decode_item(t, S, st, beta, a.y + ((size_t)b * a.Hv + h) * 128, a.fit_iters, ok,
                               refill);
        },
        [&](int h, int slot, int s) {
            bulk_store(a.pool + (uint64_t)slot * a.stride + S.hoff[h],
                       S.stages + (size_t)s * a.stage_bytes, S.hbytes[h]);
        });
}

}  // namespace rk

static int sm_count_rows() {
    static int n[64];
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev < 0 || dev >= 64) return 1;
    if (!n[dev]) cudaDeviceGetAttribute(&n[dev], cudaDevAttrMultiProcessorCount, dev);
    return n[dev] > 0 ? n[dev] : 1;
}

stepq_status launch_decode_rows(const stepq_plan *p, int layer, uint8_t *pool, int pool_slots,
                                const int32_t *slots, int B, const float *q, const float *k,
                                const float *v, const float *beta, const float *gate, float *y,
                                cudaStream_t s) {
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
    a.err = device_error_word();
    a.page_region = (maxb + 127) / 128 * 128;
    a.stage_bytes = a.page_region + rk::kVecBytes;
    // as many stages (2..4) as keep two CTAs per SM
    int stages = (int)((113 * 1024 - rk::kOffStages) / a.stage_bytes);
    stages = stages < 2 ? 2 : (stages > 4 ? 4 : stages);
    a.n_stages = stages;
    a.fit_iters = p->cfg.fit_iters;
    const int smem = rk::kOffStages + stages * (int)a.stage_bytes;
    if (cudaFuncSetAttribute((const void *)rk::decode_rows_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             smem) != cudaSuccess)
        return STEPQ_ERR_CUDA;
    int grid = 2 * sm_count_rows();
    if (grid > a.items) grid = a.items;
    rk::decode_rows_kernel<<<grid, kThreads, smem, s>>>(a);
    return cudaGetLastError() == cudaSuccess ? STEPQ_OK : STEPQ_ERR_CUDA;
}

}  // namespace stepq
