// Head-unit (GDN) kernels: the persistent, bulk-async pipelined decode step and
// the pack/unpack kernels for head pages stored in band-major order.
//
// Tile mapping: warp w owns the band of key rows 16w..16w+15; lane l owns the
// value columns l, l+32, l+64, l+96. A thread holds a 16 x 4 register tile, so
// every column reduction needs only one cross-warp step and the single row
// reduction (m_i) stays inside a warp. In the band-major page a thread's 16
// codes of one column are one 2b-byte chunk, and consecutive lanes read
// consecutive chunks (no shared-memory bank conflicts).
//
// Decode pipeline (App. C.3 steps 1-7 per head): each persistent CTA walks its
// (slot, head) items; one thread keeps up to S-1 pages in flight with bulk
// copies completing on per-stage mbarriers, the CTA updates and refits the
// page in place in shared memory, and a bulk store writes it back. Every wait
// is bounded: a stalled copy raises STEPQ_ERR_TIMEOUT and the CTA drains its
// own copies before returning.
#include "async.cuh"
#include "device.cuh"
#include "internal.h"

namespace stepq {
namespace hk {

constexpr long long kWaitCycles = 2000000000LL;      // ~1 s at 2 GHz
constexpr float kMagic = 12582912.0f;                  // 1.5 * 2^23: rint by addition
constexpr int kVecBytes = 5 * 512;                     // q k v w2 wis per stage

// ------------------------------------------------------------ shared layout
constexpr int kOffBars = 0;                            // uint64 [8]
constexpr int kOffFlags = 64;                          // int [16]
constexpr int kOffRed = 128;                           // float [2][8][128]
constexpr int kOffCol = kOffRed + 2 * 8 * 128 * 4;     // float [4][128] (colX and paired G, D)
constexpr int kOffRowC = kOffCol + 4 * 128 * 4;        // float4 [2][128]: kappa,kappa,bk',bk' | qa,qa,a,a
constexpr int kOffRowF = kOffRowC + 256 * 16;          // float4 [128]: rho a, rho a, alpha_ls, alpha_ls
constexpr int kOffRowA = kOffRowF + 128 * 16;          // float [128]: a_i
constexpr int kMaxHv = 256;                            // value heads per layer (launch check)
constexpr int kOffHead = kOffRowA + 128 * 4;           // u64 off[256] | u32 bytes[256] | u8 bits[256]
constexpr int kOffStages = (kOffHead + kMaxHv * 13 + 127) / 128 * 128;

struct Smem {
    uint64_t *bars;
    int *flags;
    float *red, *colC, *colG, *colD, *colX;
    float4 *rowc;
    float4 *rowf;
    float *rowa;
    uint64_t *hoff;
    uint32_t *hbytes;
    uint8_t *hbits;
    uint8_t *stages;
    __device__ __forceinline__ explicit Smem(uint8_t *s) {
        bars = (uint64_t *)(s + kOffBars);
        flags = (int *)(s + kOffFlags);
        red = (float *)(s + kOffRed);
        colC = (float *)(s + kOffCol);
        colG = colC + 128;
        colD = colC + 256;
        colX = colC + 384;
        rowc = (float4 *)(s + kOffRowC);
        rowf = (float4 *)(s + kOffRowF);
        rowa = (float *)(s + kOffRowA);
        hoff = (uint64_t *)(s + kOffHead);
        hbytes = (uint32_t *)(s + kOffHead + kMaxHv * 8);
        hbits = s + kOffHead + kMaxHv * 12;
        stages = s + kOffStages;
    }
};

struct Stage {
    uint8_t *page;
    float *q, *k, *v, *w2, *wis;
    __device__ __forceinline__ Stage(uint8_t *base, uint32_t page_region) {
        page = base;
        q = (float *)(base + page_region);
        k = q + 128;
        v = q + 256;
        w2 = q + 384;
        wis = q + 512;
    }
};

constexpr int kProducer = kThreads - 32;              // lane 0 of the last warp issues copies

struct T {   // thread coordinates
    int tid, w, l;
    __device__ __forceinline__ T() {
        tid = threadIdx.x;
        w = tid >> 5;
        l = tid & 31;
    }
    __device__ __forceinline__ int row(int r) const { return 16 * w + r; }
    __device__ __forceinline__ int col(int c) const { return l + 32 * c; }
};

// Byte offset of the band-major chunk (band w, column j) in a head page.
template <int B>
__device__ __forceinline__ int chunk_off(int w, int j) {
    return (B == kPivot ? 0 : 512) + (w * 128 + j) * 2 * B;
}

// ---- chunk (un)packing: 16 codes (rows of one band) of one column ----
template <int B>
__device__ __forceinline__ void load_chunk(const uint8_t *p, uint32_t (&wd)[8]) {
    if (B == 2) {
        wd[0] = *(const uint32_t *)p;
    } else if (B == 4) {
        uint2 a = *(const uint2 *)p;
        wd[0] = a.x; wd[1] = a.y;
    } else if (B == 6) {
        const uint32_t *q = (const uint32_t *)p;
        wd[0] = q[0]; wd[1] = q[1]; wd[2] = q[2];
    } else if (B == 8) {
        uint4 a = *(const uint4 *)p;
        wd[0] = a.x; wd[1] = a.y; wd[2] = a.z; wd[3] = a.w;
    } else {
        uint4 a = ((const uint4 *)p)[0], b = ((const uint4 *)p)[1];
        wd[0] = a.x; wd[1] = a.y; wd[2] = a.z; wd[3] = a.w;
        wd[4] = b.x; wd[5] = b.y; wd[6] = b.z; wd[7] = b.w;
    }
}

template <int B>
__device__ __forceinline__ uint32_t code_at(const uint32_t (&wd)[8], int r) {
    const int bit = r * B, wi = bit >> 5, sh = bit & 31;
    constexpr uint32_t mask = (1u << B) - 1u;
    if (sh + B <= 32) return (wd[wi] >> sh) & mask;
    return __funnelshift_r(wd[wi], wd[wi + 1], sh) & mask;
}

template <int B>
__device__ __forceinline__ void store_chunk(uint8_t *p, const uint32_t (&wd)[8]) {
    if (B == 2) {
        *(uint32_t *)p = wd[0];
    } else if (B == 4) {
        *(uint2 *)p = make_uint2(wd[0], wd[1]);
    } else if (B == 6) {
        uint32_t *q = (uint32_t *)p;
        q[0] = wd[0]; q[1] = wd[1]; q[2] = wd[2];
    } else if (B == 8) {
        *(uint4 *)p = make_uint4(wd[0], wd[1], wd[2], wd[3]);
    } else {
        ((uint4 *)p)[0] = make_uint4(wd[0], wd[1], wd[2], wd[3]);
        ((uint4 *)p)[1] = make_uint4(wd[4], wd[5], wd[6], wd[7]);
    }
}

// 16 offset-binary codes (low B bits of u[r]) into the chunk words.
template <int B>
__device__ __forceinline__ void pack16(const uint32_t (&u)[16], uint32_t (&wd)[8]) {
    if (B == 8) {
#pragma unroll
        for (int t = 0; t < 4; t++) {
            const uint32_t lo = __byte_perm(u[4 * t], u[4 * t + 1], 0x0040);
            const uint32_t hi = __byte_perm(u[4 * t + 2], u[4 * t + 3], 0x0040);
            wd[t] = __byte_perm(lo, hi, 0x5410);
        }
        return;
    }
    constexpr uint32_t mask = (1u << B) - 1u;
#pragma unroll
    for (int t = 0; t < B / 2; t++) wd[t] = 0u;
#pragma unroll
    for (int r = 0; r < 16; r++) {
        const uint32_t v = u[r] & mask;
        const int bit = r * B, wi = bit >> 5, sh = bit & 31;
        wd[wi] |= v << sh;
        if (sh + B > 32) wd[wi + 1] |= v >> (32 - sh);
    }
}

// Sum of 16 per-row partials over the 32 lanes of a warp (reduce-scatter): lane
// l returns the full sum of row 8*b4 + 4*b3 + 2*b2 + b1 (b_k = bit k of l).
__device__ __forceinline__ float warp_row_sums(float (&v)[16], int l, int &row_out) {
    float a8[8];
    const bool h16 = l & 16;
#pragma unroll
    for (int t = 0; t < 8; t++) {
        const float keep = h16 ? v[8 + t] : v[t], send = h16 ? v[t] : v[8 + t];
        a8[t] = keep + __shfl_xor_sync(0xffffffffu, send, 16);
    }
    float a4[4];
    const bool h8 = l & 8;
#pragma unroll
    for (int t = 0; t < 4; t++) {
        const float keep = h8 ? a8[4 + t] : a8[t], send = h8 ? a8[t] : a8[4 + t];
        a4[t] = keep + __shfl_xor_sync(0xffffffffu, send, 8);
    }
    float a2[2];
    const bool h4 = l & 4;
#pragma unroll
    for (int t = 0; t < 2; t++) {
        const float keep = h4 ? a4[2 + t] : a4[t], send = h4 ? a4[t] : a4[2 + t];
        a2[t] = keep + __shfl_xor_sync(0xffffffffu, send, 4);
    }
    const bool h2 = l & 2;
    float a1 = (h2 ? a2[1] : a2[0]) + __shfl_xor_sync(0xffffffffu, h2 ? a2[0] : a2[1], 2);
    a1 += __shfl_xor_sync(0xffffffffu, a1, 1);
    row_out = 8 * ((l >> 4) & 1) + 4 * ((l >> 3) & 1) + 2 * ((l >> 2) & 1) + ((l >> 1) & 1);
    return a1;
}

// Column vectors are kept in "pair" order so a thread loads the values of its
// column pairs (l, l+32) and (l+64, l+96) as one 64-bit word each.
__device__ __forceinline__ int pair_idx(int j) {      // column j -> float index in the pair array
    const int m = j >> 6, rem = j & 63;                 // rem = l or l + 32
    return (m * 32 + (rem & 31)) * 2 + (rem >> 5);
}
__device__ __forceinline__ uint64_t load_pair(const float *v, int l, int m) {
    return *(const uint64_t *)&v[(m * 32 + l) * 2];
}

// Cross-warp column reduction of NR values per thread column (4 columns per
// thread, 8 warps); results land in out[k][128] for threads 0..127 to use.
template <int NR>
__device__ __forceinline__ void cols_to_red(const T &t, float *red, const float (&v)[NR][4]) {
#pragma unroll
    for (int k = 0; k < NR; k++)
#pragma unroll
        for (int c = 0; c < 4; c++) red[(k * 8 + t.w) * 128 + t.col(c)] = v[k][c];
}

// ---------------------------------------------------------------- the fit
// Key-Row-Aware Dual-axis Fitting of the register tile (Sec. 4.3, App. C.1)
// and packing into the page (App. C.3 step 6). The tile holds Z with
// X_ij = a_i Z_ij (a_i > 0 a per-row factor: a_i = alpha r_i in the decode
// step, 1 when packing a dense state); rs[r] holds the partial sums of |Z| of
// the thread's rows over its 4 columns. Readout partials (y_part), when given,
// ride on the column-start reduction round. On return the page holds r, c and
// the codes. Requires the old page to be fully consumed by every thread.
template <int B>
__device__ __forceinline__ void fit_pack(const T &t, const Smem &S, uint8_t *page, const float *w2v,
                                         const float *wisv, const float *a_row, uint64_t (&x2)[16][2],
                                         float (&rs)[16], const float (&y_part)[4], bool with_y,
                                         float *y_out, int fit_iters) {
    constexpr int qm = (1 << (B - 1)) - 1;
    constexpr float fqm = (float)qm;
    const float mu = __frcp_rn(fqm);
    uint16_t *page_r = (uint16_t *)page;
    uint16_t *page_c = (uint16_t *)(page + 256);
    // Row factors r_i = m_i^(1/2) w_i^(-1/2), m_i = (1/128) sum_j |X_ij|.
    {
        int rr;
        const float sz = warp_row_sums(rs, t.l, rr);
        const int i = t.row(rr);
        const float a = a_row ? a_row[i] : 1.f;
        const float m = (a * sz) * (1.0f / 128.0f);
        const float rf = __half2float(__float2half_rn(
            fminf(fmaxf(__fmul_rn(sqrtf(m), wisv[i]), kF16Min), kF16Max)));
        if ((t.l & 1) == 0) {
            const float rho_a = __frcp_rn(rf) * a;                 // X' = rho_i X = (rho_i a_i) Z
            const float al = w2v[i] * (rf * rf);                   // w_i^2 r_i^2
            S.rowf[i] = make_float4(rho_a, rho_a, al, al);
            page_r[i] = f16_bits(rf);
        }
    }
    __syncwarp();
    // X' = X rho_i (row-normalised state) and the clip-free column start.
    float cm[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int r = 0; r < 16; r++) {
        const uint4 rf = *(const uint4 *)&S.rowf[t.row(r)];
        const uint64_t rho = ((uint64_t)rf.y << 32) | rf.x;
        x2[r][0] = fmul2(x2[r][0], rho);
        x2[r][1] = fmul2(x2[r][1], rho);
        cm[0] = fmaxf(cm[0], fabsf(f2lo(x2[r][0])));
        cm[1] = fmaxf(cm[1], fabsf(f2hi(x2[r][0])));
        cm[2] = fmaxf(cm[2], fabsf(f2lo(x2[r][1])));
        cm[3] = fmaxf(cm[3], fabsf(f2hi(x2[r][1])));
    }
    {
        float v[2][4];
#pragma unroll
        for (int c = 0; c < 4; c++) {
            v[0][c] = cm[c];
            v[1][c] = with_y ? y_part[c] : 0.f;
        }
        cols_to_red<2>(t, S.red, v);
    }
    if (t.tid == 0) {
        S.flags[1] = 0;
        S.flags[2] = 0;
    }
    __syncthreads();
    if (t.tid < 128) {
        float mx = S.red[t.tid];
#pragma unroll
        for (int wv = 1; wv < 8; wv++) mx = fmaxf(mx, S.red[wv * 128 + t.tid]);
        const float c0 = __fmul_rn(mx, mu);
        if (c0 > kF16Max) S.flags[1] = 1;                 // start capped: codes may clip
        const float c = fminf(fmaxf(c0, kF16Min), kF16Max);
        S.colC[t.tid] = c;
        S.colG[pair_idx(t.tid)] = __frcp_rn(c);
        S.colX[t.tid] = mx;                               // max_i |X'_ij|
    } else if (with_y) {
        const int j = t.tid - 128;
        float s = S.red[8 * 128 + j];
#pragma unroll
        for (int wv = 1; wv < 8; wv++) s += S.red[(8 + wv) * 128 + j];
        y_out[j] = s;
    }
    __syncthreads();
    // Fixed-code least-squares updates: c_j = sum alpha_i q_ij X'_ij / sum alpha_i q_ij^2
    // (alpha_i = w_i^2 r_i^2: the w^2-weighted objective in the X' domain).
    const uint64_t M2 = f2s(kMagic), nM2 = f2s(-kMagic);
    for (int it = 0; it < fit_iters; it++) {
        const bool clip = it > 0 || S.flags[1];
        const uint64_t g01 = load_pair(S.colG, t.l, 0);
        const uint64_t g23 = load_pair(S.colG, t.l, 1);
        uint64_t n01 = 0, n23 = 0, d01 = 0, d23 = 0, e01 = 0, e23 = 0, h01 = 0, h23 = 0;
#pragma unroll
        for (int r = 0; r < 16; r++) {
            const uint4 rf = *(const uint4 *)&S.rowf[t.row(r)];
            const uint64_t al = ((uint64_t)rf.w << 32) | rf.z;
            uint64_t q01 = fadd2(fadd2(fmul2(x2[r][0], g01), M2), nM2);
            uint64_t q23 = fadd2(fadd2(fmul2(x2[r][1], g23), M2), nM2);
            if (clip) {
                q01 = f2(fminf(fmaxf(f2lo(q01), -fqm), fqm), fminf(fmaxf(f2hi(q01), -fqm), fqm));
                q23 = f2(fminf(fmaxf(f2lo(q23), -fqm), fqm), fminf(fmaxf(f2hi(q23), -fqm), fqm));
            }
            const uint64_t a01 = fmul2(al, q01), a23 = fmul2(al, q23);
            if (r & 1) {
                e01 = ffma2(a01, x2[r][0], e01);
                e23 = ffma2(a23, x2[r][1], e23);
                h01 = ffma2(a01, q01, h01);
                h23 = ffma2(a23, q23, h23);
            } else {
                n01 = ffma2(a01, x2[r][0], n01);
                n23 = ffma2(a23, x2[r][1], n23);
                d01 = ffma2(a01, q01, d01);
                d23 = ffma2(a23, q23, d23);
            }
        }
        n01 = fadd2(n01, e01);
        n23 = fadd2(n23, e23);
        d01 = fadd2(d01, h01);
        d23 = fadd2(d23, h23);
        {
            float v[2][4] = {{f2lo(n01), f2hi(n01), f2lo(n23), f2hi(n23)},
                             {f2lo(d01), f2hi(d01), f2lo(d23), f2hi(d23)}};
            cols_to_red<2>(t, S.red, v);
        }
        __syncthreads();
        if (t.tid < 128) {
            float num = 0.f, den = 0.f;
#pragma unroll
            for (int wv = 0; wv < 8; wv++) {
                num += S.red[wv * 128 + t.tid];
                den += S.red[(8 + wv) * 128 + t.tid];
            }
            // num and den carry fp32 summation error already; a 2-ulp quotient adds nothing
            float c = S.colC[t.tid];
            if (den > 0.f) c = fminf(fmaxf(__fdividef(num, den), kF16Min), kF16Max);
            if (it + 1 < fit_iters) {
                S.colC[t.tid] = c;
                S.colG[pair_idx(t.tid)] = __frcp_rn(c);
            } else {
                // storage precision of c; codes can clip only where max |X'| / c >= qmax + 1/2
                const float cf = __half2float(__float2half_rn(c));
                const float g = __frcp_rn(cf);
                page_c[t.tid] = f16_bits(cf);
                S.colG[pair_idx(t.tid)] = g;
                if (__fmul_rn(S.colX[t.tid], g) >= fqm + 0.5f) S.flags[2] = 1;
            }
        }
        __syncthreads();
    }
    // Final codes with the stored scales.
    const bool clip = S.flags[2] != 0;
    const uint64_t MB = f2s(kMagic + (float)(1 << (B - 1)));
#pragma unroll
    for (int c = 0; c < 4; c += 2) {
        const uint64_t g = load_pair(S.colG, t.l, c >> 1);
        uint32_t ua[16], ub[16];
#pragma unroll
        for (int r = 0; r < 16; r++) {
            uint64_t tq = fmul2(x2[r][c >> 1], g);
            if (clip)
                tq = f2(fminf(fmaxf(f2lo(tq), -fqm), fqm), fminf(fmaxf(f2hi(tq), -fqm), fqm));
            const uint64_t uu = fadd2(tq, MB);              // bits: 0x4B400000 + (q + 2^(B-1))
            ua[r] = (uint32_t)uu;
            ub[r] = (uint32_t)(uu >> 32);
        }
        uint32_t wd[8];
        pack16<B>(ua, wd);
        store_chunk<B>(page + chunk_off<B>(t.w, t.col(c)), wd);
        pack16<B>(ub, wd);
        store_chunk<B>(page + chunk_off<B>(t.w, t.col(c + 1)), wd);
    }
}

// FP16 pivot head: store fp16(a_i Z) (saturating) in band-major order.
__device__ __forceinline__ void pack_pivot(const T &t, uint8_t *page, const uint64_t (&x2)[16][2],
                                           float a) {
#pragma unroll
    for (int c = 0; c < 4; c++) {
        uint32_t wd[8];
#pragma unroll
        for (int r = 0; r < 16; r += 2) {
            const float za = (c & 1) ? f2hi(x2[r][c >> 1]) : f2lo(x2[r][c >> 1]);
            const float zb = (c & 1) ? f2hi(x2[r + 1][c >> 1]) : f2lo(x2[r + 1][c >> 1]);
            wd[r >> 1] = (uint32_t)f16_bits(f16_round_sat(a * za)) |
                         ((uint32_t)f16_bits(f16_round_sat(a * zb)) << 16);
        }
        store_chunk<kPivot>(page + chunk_off<kPivot>(t.w, t.col(c)), wd);
    }
}

// Reconstruct the column-scaled codes c_j q_ij (exact in fp32) or the FP16
// values of a pivot head; the row factor stays separate.
template <int B>
__device__ __forceinline__ void load_tile(const T &t, const uint8_t *page, uint64_t (&x2)[16][2]) {
    const uint16_t *page_c = (const uint16_t *)(page + 256);
#pragma unroll
    for (int c = 0; c < 4; c += 2) {
        uint32_t wa[8], wb[8];
        load_chunk<B>(page + chunk_off<B>(t.w, t.col(c)), wa);
        load_chunk<B>(page + chunk_off<B>(t.w, t.col(c + 1)), wb);
        if (B == kPivot) {
#pragma unroll
            for (int r = 0; r < 16; r++) {
                const float a = f16_val((uint16_t)(wa[r >> 1] >> (16 * (r & 1))));
                const float b = f16_val((uint16_t)(wb[r >> 1] >> (16 * (r & 1))));
                x2[r][c >> 1] = f2(a, b);
            }
        } else {
            const float ca = f16_val(page_c[t.col(c)]), cb = f16_val(page_c[t.col(c + 1)]);
            // 0x4B400000 + u - 2^(B-1) is the float 1.5*2^23 + q; fma(f, c, -1.5*2^23 c)
            // = c q exactly (c fp16, |q| <= 127: 19 significant bits; 1.5*2^23 c exact).
            constexpr uint32_t kBias = 0x4B400000u - (1u << (B - 1));
            const uint64_t cc = f2(ca, cb), oc = f2(-kMagic * ca, -kMagic * cb);
#pragma unroll
            for (int r = 0; r < 16; r++) {
                const uint64_t fq = ((uint64_t)(code_at<B>(wb, r) + kBias) << 32) |
                                    (uint64_t)(code_at<B>(wa, r) + kBias);
                x2[r][c >> 1] = ffma2(fq, cc, oc);
            }
        }
    }
}

// ------------------------------------------------------------------ decode
struct DecodeArgs {
    uint8_t *pool;
    uint64_t stride;
    int pool_slots;
    const int32_t *slots;
    int Hk, Hv, items;
    LayerTables tab;
    const float *q, *k, *v, *beta, *gate;
    float *y;
    unsigned int *err;
    int n_stages;
    uint32_t page_region, stage_bytes;
    int fit_iters;
};

__device__ __forceinline__ bool slot_ok(const DecodeArgs &a, int slot) {
    return slot >= 0 && slot < a.pool_slots;
}

// Producer: start the copies of `item` (batch entry b = item / Hv, head h) into
// stage s (thread 0 only). An invalid slot completes the phase without data.
__device__ __forceinline__ void issue(const DecodeArgs &a, const Smem &S, int item, int slot, int s) {
    const int b = item / a.Hv, h = item - b * a.Hv;
    uint64_t *bar = &S.bars[s];
    if (!slot_ok(a, slot)) {
        mbar_arrive(bar);
        return;
    }
    Stage st(S.stages + (size_t)s * a.stage_bytes, a.page_region);
    const uint32_t nb = S.hbytes[h];
    const int hk = h / (a.Hv / a.Hk);
    mbar_arrive_tx(bar, nb + kVecBytes);
    bulk_load(st.page, a.pool + (uint64_t)slot * a.stride + S.hoff[h], nb, bar);
    bulk_load(st.q, a.q + ((size_t)b * a.Hk + hk) * 128, 512, bar);
    bulk_load(st.k, a.k + ((size_t)b * a.Hk + hk) * 128, 512, bar);
    bulk_load(st.v, a.v + ((size_t)b * a.Hv + h) * 128, 512, bar);
    bulk_load(st.w2, a.tab.w2 + (size_t)h * 128, 512, bar);
    bulk_load(st.wis, a.tab.wis + (size_t)h * 128, 512, bar);
}

// One decode step of one head page staged in shared memory (width B).
// `refill` runs once the stage's inputs are fully consumed (after the retrieval
// reduction); the page itself is rewritten in place afterwards.
//
// With a_i = alpha r_i (> 0) and Z_ij = c_j q_ij + (beta k_i / a_i) delta_j the
// update is X_ij = a_i Z_ij: one fma per element instead of two.
template <int B, class Refill>
__device__ __forceinline__ void decode_item(const T &t, const Smem &S, const Stage &st, float alpha,
                                            float beta, float *y_out, int fit_iters,
                                            const Refill &refill) {
    const uint16_t *page_r = (const uint16_t *)st.page;
    // Row constants of the warp's band (warp-local): a_i, kappa_i = k_i a_i,
    // beta k_i / a_i, q_i a_i, as duplicated fp32 pairs.
    if (t.l < 16) {
        const int i = t.row(t.l);
        const float a = fmaxf(B == kPivot ? alpha : alpha * f16_val(page_r[i]), 1e-30f);
        const float ki = st.k[i];
        const float kap = ki * a, bkp = __fdiv_rn(beta * ki, a), qa = st.q[i] * a;
        S.rowc[2 * i] = make_float4(kap, kap, bkp, bkp);
        S.rowc[2 * i + 1] = make_float4(qa, qa, a, a);
        S.rowa[i] = a;
    }
    uint64_t x2[16][2];
    load_tile<B>(t, st.page, x2);
    __syncwarp();
    // Step 2a: retrieval u_j = sum_i k_i a_i (c_j q_ij).
    uint64_t u01 = 0, u23 = 0, v01 = 0, v23 = 0;
#pragma unroll
    for (int r = 0; r < 16; r++) {
        const uint4 rc = *(const uint4 *)&S.rowc[2 * t.row(r)];
        const uint64_t kap = ((uint64_t)rc.y << 32) | rc.x;
        if (r & 1) {
            v01 = ffma2(kap, x2[r][0], v01);
            v23 = ffma2(kap, x2[r][1], v23);
        } else {
            u01 = ffma2(kap, x2[r][0], u01);
            u23 = ffma2(kap, x2[r][1], u23);
        }
    }
    u01 = fadd2(u01, v01);
    u23 = fadd2(u23, v23);
    {
        float v[1][4] = {{f2lo(u01), f2hi(u01), f2lo(u23), f2hi(u23)}};
        cols_to_red<1>(t, S.red, v);
    }
    __syncthreads();
    if (t.tid < 128) {
        float s = 0.f;
#pragma unroll
        for (int wv = 0; wv < 8; wv++) s += S.red[wv * 128 + t.tid];
        S.colD[pair_idx(t.tid)] = st.v[t.tid] - s;          // delta_j = v_j - u_j
    }
    refill();
    __syncthreads();
    // Step 2b-3: Z = c q + (beta k / a) delta; readout partials q_i a_i Z_ij.
    const uint64_t dl01 = load_pair(S.colD, t.l, 0);
    const uint64_t dl23 = load_pair(S.colD, t.l, 1);
    uint64_t y01 = 0, y23 = 0, z01 = 0, z23 = 0;
    float rs[16];
#pragma unroll
    for (int r = 0; r < 16; r++) {
        const uint4 rc = *(const uint4 *)&S.rowc[2 * t.row(r)];
        const uint4 rq = *(const uint4 *)&S.rowc[2 * t.row(r) + 1];
        const uint64_t bkp = ((uint64_t)rc.w << 32) | rc.z;
        const uint64_t qa = ((uint64_t)rq.y << 32) | rq.x;
        x2[r][0] = ffma2(bkp, dl01, x2[r][0]);
        x2[r][1] = ffma2(bkp, dl23, x2[r][1]);
        if (r & 1) {
            z01 = ffma2(qa, x2[r][0], z01);
            z23 = ffma2(qa, x2[r][1], z23);
        } else {
            y01 = ffma2(qa, x2[r][0], y01);
            y23 = ffma2(qa, x2[r][1], y23);
        }
        rs[r] = (fabsf(f2lo(x2[r][0])) + fabsf(f2hi(x2[r][0]))) +
                (fabsf(f2lo(x2[r][1])) + fabsf(f2hi(x2[r][1])));
    }
    y01 = fadd2(y01, z01);
    y23 = fadd2(y23, z23);
    const float yp[4] = {f2lo(y01), f2hi(y01), f2lo(y23), f2hi(y23)};
    if (B == kPivot) {
        float v[1][4] = {{yp[0], yp[1], yp[2], yp[3]}};
        cols_to_red<1>(t, S.red, v);
        __syncthreads();
        if (t.tid < 128) {
            float s = 0.f;
#pragma unroll
            for (int wv = 0; wv < 8; wv++) s += S.red[wv * 128 + t.tid];
            y_out[t.tid] = s;
        }
        pack_pivot(t, st.page, x2, fmaxf(alpha, 1e-30f));
        return;
    }
    // Steps 4-6: refit and repack in place.
    fit_pack<B>(t, S, st.page, st.w2, st.wis, S.rowa, x2, rs, yp, true, y_out, fit_iters);
}

__global__ void __launch_bounds__(kThreads, 2) decode_heads_kernel(DecodeArgs a) {
    extern __shared__ __align__(128) uint8_t smem[];
    const T t;
    const Smem S(smem);
    const int G = gridDim.x, S_n = a.n_stages;
    const int first = blockIdx.x;
    if (first >= a.items) return;
    for (int h = t.tid; h < a.Hv; h += kThreads) {
        S.hoff[h] = a.tab.head_off[h];
        S.hbytes[h] = a.tab.head_bytes[h];
        S.hbits[h] = a.tab.head_bits[h];
    }
    if (t.tid == kProducer) {
        for (int s = 0; s < S_n; s++) mbar_init(&S.bars[s], 1);
        mbar_init_fence();
    }
    __syncthreads();
    if (t.tid == kProducer) {
        for (int s = 0; s < S_n; s++) {
            const int item = first + s * G;
            if (item < a.items) issue(a, S, item, a.slots[item / a.Hv], s);
        }
    }
    // With three or more stages a stage is refilled two items after its own item
    // (its store has long finished reading it); with two stages, one item after.
    const int lag = S_n >= 3 ? 2 : 1;
    // scalars of the current item; the next item's are fetched one iteration ahead
    int b = first / a.Hv, h = first - b * a.Hv;
    int slot = a.slots[b];
    float alpha = a.gate[(size_t)b * a.Hv + h], beta = a.beta[(size_t)b * a.Hv + h];
    int n = 0;
    for (int item = first; item < a.items; item += G, n++) {
        const int s = n % S_n;
        const uint32_t parity = (uint32_t)(n / S_n) & 1u;
        // prefetch: next item's scalars (all threads), and the slot of the item
        // this iteration will issue (thread 0)
        const int nitem = item + G;
        int nb = 0, nh = 0, nslot = -1;
        float nalpha = 0.f, nbeta = 0.f;
        if (nitem < a.items) {
            nb = nitem / a.Hv;
            nh = nitem - nb * a.Hv;
            nslot = a.slots[nb];
            nalpha = a.gate[(size_t)nb * a.Hv + nh];
            nbeta = a.beta[(size_t)nb * a.Hv + nh];
        }
        const int iitem = first + (n - lag + S_n) * G;
        int islot = -1;
        if (t.tid == kProducer && n >= lag && iitem < a.items) islot = a.slots[iitem / a.Hv];

        const bool ok = mbar_wait(&S.bars[s], parity, kWaitCycles);
        if (__syncthreads_or(!ok)) {
            if (t.tid == kProducer) {
                raise_error(a.err, STEPQ_ERR_TIMEOUT);
                // drain this CTA's copies still in flight (items n .. issued), with a bound
                const int last = n < lag ? S_n - 1 : n - 1 - lag + S_n;
                for (int m = n; m <= last; m++) {
                    if (first + m * G >= a.items) break;
                    mbar_wait(&S.bars[m % S_n], (uint32_t)(m / S_n) & 1u, kWaitCycles);
                }
                bulk_wait_all();
            }
            return;
        }
        const bool valid = slot_ok(a, slot);
        if (!valid && t.tid == 0) raise_error(a.err, STEPQ_ERR_SLOT_RANGE);
        const Stage st(S.stages + (size_t)s * a.stage_bytes, a.page_region);
        // Refill the stage of the previous item (its store was committed one item
        // ago) with the item S-1 ahead of it: S-1 items stay in flight.
        const auto refill = [&]() {
            if (t.tid == kProducer && n >= lag && iitem < a.items) {
                if (lag == 2) bulk_wait_read_all_but_one();
                else bulk_wait_read_all();
                issue(a, S, iitem, islot, (n - lag) % S_n);
            }
        };
        if (valid) {
            float *y_out = a.y + ((size_t)b * a.Hv + h) * 128;
            switch (S.hbits[h]) {
            case 2: decode_item<2>(t, S, st, alpha, beta, y_out, a.fit_iters, refill); break;
            case 4: decode_item<4>(t, S, st, alpha, beta, y_out, a.fit_iters, refill); break;
            case 6: decode_item<6>(t, S, st, alpha, beta, y_out, a.fit_iters, refill); break;
            case 8: decode_item<8>(t, S, st, alpha, beta, y_out, a.fit_iters, refill); break;
            default: decode_item<kPivot>(t, S, st, alpha, beta, y_out, a.fit_iters, refill); break;
            }
        } else {
            refill();
        }
        __syncthreads();                                 // the page in stage s is final
        if (t.tid == kProducer) {
            if (valid) {
                fence_async_smem();
                bulk_store(a.pool + (uint64_t)slot * a.stride + S.hoff[h], st.page, S.hbytes[h]);
            }
            bulk_commit();
        }
        b = nb; h = nh; slot = nslot; alpha = nalpha; beta = nbeta;
    }
    if (t.tid == kProducer) bulk_wait_all();
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
    uint64_t x2[16][2];
    float rs[16];
#pragma unroll
    for (int r = 0; r < 16; r++) {
        const float *row = X + t.row(r) * 128;
        const float a = row[t.col(0)], b = row[t.col(1)], c = row[t.col(2)], d = row[t.col(3)];
        x2[r][0] = f2(a, b);
        x2[r][1] = f2(c, d);
        rs[r] = fabsf(a) + fabsf(b) + fabsf(c) + fabsf(d);
    }
    if (B == kPivot) {
        pack_pivot(t, page, x2, 1.f);
        return;
    }
    const float none[4] = {0.f, 0.f, 0.f, 0.f};
    fit_pack<B>(t, S, page, w2, wis, nullptr, x2, rs, none, false, nullptr, fit_iters);
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
    if (t.tid == 0) S.flags[1] = 0;
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
    uint64_t x2[16][2];
    load_tile<B>(t, page, x2);      // c_j q_ij (rounded once) or the FP16 value
    const uint16_t *page_r = (const uint16_t *)page;
#pragma unroll
    for (int r = 0; r < 16; r++) {
        float *row = out + t.row(r) * 128;
#pragma unroll
        for (int c = 0; c < 4; c++) {
            float v;
            if (B == kPivot) {
                v = (c & 1) ? f2hi(x2[r][c >> 1]) : f2lo(x2[r][c >> 1]);
            } else {
                // r_i c_j z_ij rounded once: c_j q_ij is exact in fp32 (fp16 x 8 bits)
                const float cq = (c & 1) ? f2hi(x2[r][c >> 1]) : f2lo(x2[r][c >> 1]);
                v = __fmul_rn(f16_val(page_r[t.row(r)]), cq);
            }
            row[t.col(c)] = v;
        }
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
    static int n[64];
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev < 0 || dev >= 64) return 1;
    if (!n[dev]) cudaDeviceGetAttribute(&n[dev], cudaDevAttrMultiProcessorCount, dev);
    return n[dev] > 0 ? n[dev] : 1;
}

stepq_status launch_decode_heads(const stepq_plan *p, int layer, uint8_t *pool, int pool_slots,
                                 const int32_t *slots, int B, const float *q, const float *k,
                                 const float *v, const float *beta, const float *gate, float *y,
                                 cudaStream_t s) {
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
    a.items = B * Hv;
    a.tab = p->layer(layer);
    a.q = q; a.k = k; a.v = v; a.beta = beta; a.gate = gate; a.y = y;
    a.err = device_error_word();
    a.page_region = (maxb + 127) / 128 * 128;
    a.stage_bytes = a.page_region + hk::kVecBytes;
    // as many stages (2..4) as keep two CTAs per SM
    int stages = (int)((113 * 1024 - hk::kOffStages) / a.stage_bytes);
    stages = stages < 2 ? 2 : (stages > 4 ? 4 : stages);
    a.n_stages = stages;
    a.fit_iters = p->cfg.fit_iters;
    const int smem = hk::kOffStages + stages * (int)a.stage_bytes;
    if (set_attr((const void *)hk::decode_heads_kernel, smem) != STEPQ_OK) return STEPQ_ERR_CUDA;
    int grid = 2 * sm_count();
    if (grid > a.items) grid = a.items;
    hk::decode_heads_kernel<<<grid, kThreads, smem, s>>>(a);
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
