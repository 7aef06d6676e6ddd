// Uniform rowwise-absmax INT-b comparison decode (App. B.5: per key row an FP16
// scale s_i = absmax_i / q_b in [2^-14, 65504], nearest codes in [-q_b, q_b]),
// on the same persistent bulk-async pipeline and tile as the row-unit STEPQuant
// kernel, so that the comparison measures the codecs and not the plumbing.
//
// Tile mapping: warp w owns key rows 16w..16w+15, lane l the value columns
// 4l..4l+3; a lane's 4 codes of a row are one word (8-bit), three bytes at
// byte 3l (6-bit) or a half-word (4-bit). A thread holds its 16 rows as eight
// row pairs per column, each pair one packed f32x2 register, so one 128-bit
// load of a per-row constant serves two pairs.
// Per row the tile holds Z = q with X_ij = a_i Z_ij, a_i = s_i d_i (d_i the
// gate), so the decode is the code itself. Every column reduction needs one
// cross-warp step; the row absmax is a warp reduce-scatter.
#include "async.cuh"
#include "device.cuh"
#include "internal.h"
#include "pipeline.cuh"
#include "tile.cuh"

namespace stepq {
namespace ib {

// ------------------------------------------------------------ shared layout
constexpr int kOffBars = 0;                            // uint64 [8]
constexpr int kOffRed = 64;                            // float [2][8][128]: retrieval, readout
constexpr int kOffColD = kOffRed + 2 * 8 * 128 * 4;    // float [128] delta_j
constexpr int kOffRows = kOffColD + 512;               // float [6][128] per-row constants
constexpr int kOffStages = (kOffRows + 6 * 128 * 4 + 127) / 128 * 128;

struct Smem {
    uint64_t *bars;
    float *red, *colD;
    // per-row constants: kappa = k a, beta k / a, q a, a, a / s_new and the
    // clamp limit (q_b where the new scale was capped, else no limit)
    float *rKap, *rBkp, *rQa, *rA, *rTs, *rLim;
    uint8_t *stages;
    __device__ __forceinline__ explicit Smem(uint8_t *s) {
        bars = (uint64_t *)(s + kOffBars);
        red = (float *)(s + kOffRed);
        colD = (float *)(s + kOffColD);
        rKap = (float *)(s + kOffRows);
        rBkp = rKap + 128;
        rQa = rKap + 256;
        rA = rKap + 384;
        rTs = rKap + 512;
        rLim = rKap + 640;
        stages = s + kOffStages;
    }
};

struct DecodeArgs {
    uint8_t *pool;
    uint64_t slot_bytes, layer_off, head_bytes;
    int pool_slots;
    const int32_t *slots;
    int Hk, Hv, nb, items, gate_per_row;
    const float *q, *k, *v, *beta, *gate;
    float *y;
    unsigned int *err;
    StallKnob stall;
    int n_stages;
    uint32_t page_region, stage_bytes, vec_bytes;
};

struct Stage {
    uint8_t *page;
    float *q, *k, *v, *gate, *gb;
    __device__ __forceinline__ Stage(uint8_t *base, uint32_t page_region) {
        page = base;
        q = (float *)(base + page_region);
        k = q + 128;
        v = q + 256;
        gate = q + 384;
        gb = q + 512;       // scalar gate, beta
    }
};

struct T {
    int tid, w, l;
    __device__ __forceinline__ T() {
        tid = threadIdx.x;
        w = tid >> 5;
        l = tid & 31;
    }
    __device__ __forceinline__ int row(int r) const { return 16 * w + r; }
};

// Row-pair constants (rows 4p, 4p+1) and (4p+2, 4p+3) of the warp's band.
__device__ __forceinline__ void row_pairs(const float *v, const T &t, int p, uint64_t &lo, uint64_t &hi) {
    const uint4 q = *(const uint4 *)&v[t.row(4 * p)];
    lo = u2pair(q.x, q.y);
    hi = u2pair(q.z, q.w);
}

// Warp reduce-scatter of 16 per-row maxima (as warp_row_sums, with max).
__device__ __forceinline__ float warp_row_max(float (&v)[16], int l, int &row_out) {
    float a8[8];
    const bool h16 = l & 16;
#pragma unroll
    for (int t = 0; t < 8; t++) {
        const float keep = h16 ? v[8 + t] : v[t], send = h16 ? v[t] : v[8 + t];
        a8[t] = fmaxf(keep, __shfl_xor_sync(0xffffffffu, send, 16));
    }
    float a4[4];
    const bool h8 = l & 8;
#pragma unroll
    for (int t = 0; t < 4; t++) {
        const float keep = h8 ? a8[4 + t] : a8[t], send = h8 ? a8[t] : a8[4 + t];
        a4[t] = fmaxf(keep, __shfl_xor_sync(0xffffffffu, send, 8));
    }
    float a2[2];
    const bool h4 = l & 4;
#pragma unroll
    for (int t = 0; t < 2; t++) {
        const float keep = h4 ? a4[2 + t] : a4[t], send = h4 ? a4[t] : a4[2 + t];
        a2[t] = fmaxf(keep, __shfl_xor_sync(0xffffffffu, send, 4));
    }
    const bool h2 = l & 2;
    float a1 = fmaxf(h2 ? a2[1] : a2[0], __shfl_xor_sync(0xffffffffu, h2 ? a2[0] : a2[1], 2));
    a1 = fmaxf(a1, __shfl_xor_sync(0xffffffffu, a1, 1));
    row_out = 8 * ((l >> 4) & 1) + 4 * ((l >> 3) & 1) + 2 * ((l >> 2) & 1) + ((l >> 1) & 1);
    return a1;
}

// The lane's 4 codes of a row as the bit patterns 1.5*2^23 + u (one logic
// op or byte permute each).
template <int B>
__device__ __forceinline__ void row_codes(const uint8_t *row, int l, uint32_t (&f)[4]) {
    if (B == 8) {
        const uint32_t w = ((const uint32_t *)row)[l];
#pragma unroll
        for (int c = 0; c < 4; c++) f[c] = __byte_perm(w, kMagicBits, 0x7650u + (uint32_t)c);
    } else if (B == 6) {
        // 24 bits at bit 24 l: a funnel shift of the two words that hold them
        // (the last lane's upper word is clamped into the row; it is unused).
        const uint32_t *wd = (const uint32_t *)row;
        const int wi = (3 * l) >> 2;
        const uint32_t x = __funnelshift_r(wd[wi], wd[min(wi + 1, 23)], 8 * ((3 * l) & 3));
#pragma unroll
        for (int c = 0; c < 4; c++) f[c] = and_or(x >> (6 * c), 0x3Fu, kMagicBits);
    } else {
        const uint32_t x = ((const uint16_t *)row)[l];
#pragma unroll
        for (int c = 0; c < 4; c++) f[c] = and_or(x >> (4 * c), 0xFu, kMagicBits);
    }
}

template <int B>
__device__ __forceinline__ void store_row(uint8_t *row, int l, uint32_t f0, uint32_t f1, uint32_t f2,
                                          uint32_t f3) {
    if (B == 8) {
        const uint32_t lo = __byte_perm(f0, f1, 0x0040), hi = __byte_perm(f2, f3, 0x0040);
        ((uint32_t *)row)[l] = __byte_perm(lo, hi, 0x5410);
    } else if (B == 6) {
        // Lane l writes its 24 bits as bytes 3l .. 3l + 2 of the row: one aligned
        // 16-bit store and one byte store (which is which depends on l's parity).
        constexpr uint32_t K = kMagicBits + (kMagicBits << 6) + (kMagicBits << 12) + (kMagicBits << 18);
        const uint32_t v = (f0 + (f1 << 6) + (f2 << 12) + (f3 << 18) - K) & 0xFFFFFFu;
        const int odd = l & 1;
        uint8_t *p = row + 3 * l;
        *(uint16_t *)(p + odd) = (uint16_t)(odd ? v >> 8 : v);
        p[odd ? 0 : 2] = (uint8_t)(odd ? v : v >> 16);
    } else {
        constexpr uint32_t K = kMagicBits + (kMagicBits << 4) + (kMagicBits << 8) + (kMagicBits << 12);
        ((uint16_t *)row)[l] = (uint16_t)(f0 + (f1 << 4) + (f2 << 8) + (f3 << 12) - K);
    }
}

// Codes rne(X / s_i) of the warp's 16 rows, written in place; CLIP clamps each
// row to its limit (q_b where the row's scale was capped, else none).
template <int B, bool CLIP>
__device__ __forceinline__ void requant_rows(const T &t, const Smem &S, uint8_t *codes,
                                             const uint64_t (&x2)[8][4]) {
    const uint64_t mb = f2s(kMagic + (float)(1 << (B - 1)));
#pragma unroll
    for (int p = 0; p < 4; p++) {
        uint64_t tlo, thi, llo = 0, lhi = 0;
        row_pairs(S.rTs, t, p, tlo, thi);
        if (CLIP) row_pairs(S.rLim, t, p, llo, lhi);
#pragma unroll
        for (int h = 0; h < 2; h++) {
            const int m = 2 * p + h;
            const uint64_t ts = h ? thi : tlo, lim = h ? lhi : llo;
            uint32_t f0[4], f1[4];
#pragma unroll
            for (int c = 0; c < 4; c++) {
                uint64_t tt = fmul2(x2[m][c], ts);
                if (CLIP) tt = f2(fminf(fmaxf(f2lo(tt), -f2lo(lim)), f2lo(lim)),
                                  fminf(fmaxf(f2hi(tt), -f2hi(lim)), f2hi(lim)));
                const uint64_t u = fadd2(tt, mb);
                f0[c] = (uint32_t)u;
                f1[c] = (uint32_t)(u >> 32);
            }
            store_row<B>(codes + t.row(2 * m) * 16 * B, t.l, f0[0], f0[1], f0[2], f0[3]);
            store_row<B>(codes + t.row(2 * m + 1) * 16 * B, t.l, f1[0], f1[1], f1[2], f1[3]);
        }
    }
}

// One INT-b decode step of a head page staged in shared memory.
template <int B, class Refill>
__device__ __forceinline__ bool decode_item(const T &t, const Smem &S, const Stage &st, float gate_s,
                                            bool per_row, float beta, float *y_out, bool ok,
                                            const Refill &refill) {
    constexpr int qm = (1 << (B - 1)) - 1;
    uint16_t *page_s = (uint16_t *)st.page;
    uint8_t *codes = st.page + 256;
    if (t.l < 16) {
        const int i = t.row(t.l);
        const float dg = per_row ? st.gate[i] : gate_s;
        const float a = fmaxf(f16_val(page_s[i]) * dg, 1e-30f);
        const float ki = st.k[i];
        S.rKap[i] = ki * a;
        S.rBkp[i] = __fdividef(beta * ki, a);
        S.rQa[i] = st.q[i] * a;
        S.rA[i] = a;
    }
    // Z = q: rows 2m, 2m+1 of column 4l + c as one pair
    uint64_t x2[8][4];
    {
        const uint64_t off = f2s(-(kMagic + (float)(1 << (B - 1))));
#pragma unroll
        for (int m = 0; m < 8; m++) {
            uint32_t f0[4], f1[4];
            row_codes<B>(codes + t.row(2 * m) * 16 * B, t.l, f0);
            row_codes<B>(codes + t.row(2 * m + 1) * 16 * B, t.l, f1);
#pragma unroll
            for (int c = 0; c < 4; c++) x2[m][c] = fadd2(u2pair(f0[c], f1[c]), off);
        }
    }
    __syncwarp();
    {
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
        *(float4 *)&S.red[t.w * 128 + 4 * t.l] =
            make_float4(pair_sum(ua[0]), pair_sum(ua[1]), pair_sum(ua[2]), pair_sum(ua[3]));
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
    // Z += (beta k_i / a_i) delta_j; readout partials; per-row max |Z|.
    float rm[16];
    {
        const float4 dq = *(const float4 *)&S.colD[4 * t.l];
        const uint64_t dl[4] = {f2s(dq.x), f2s(dq.y), f2s(dq.z), f2s(dq.w)};
        uint64_t ya[4] = {0, 0, 0, 0};
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
                ya[c] = ffma2(qhi, x2[2 * p + 1][c], ya[c]);
            }
#pragma unroll
            for (int h = 0; h < 2; h++) {
                const uint64_t(&xm)[4] = x2[2 * p + h];
                rm[4 * p + 2 * h] = fmax3(fmax3(0.f, fabsf(f2lo(xm[0])), fabsf(f2lo(xm[1]))),
                                          fabsf(f2lo(xm[2])), fabsf(f2lo(xm[3])));
                rm[4 * p + 2 * h + 1] = fmax3(fmax3(0.f, fabsf(f2hi(xm[0])), fabsf(f2hi(xm[1]))),
                                              fabsf(f2hi(xm[2])), fabsf(f2hi(xm[3])));
            }
        }
        *(float4 *)&S.red[(8 + t.w) * 128 + 4 * t.l] =
            make_float4(pair_sum(ya[0]), pair_sum(ya[1]), pair_sum(ya[2]), pair_sum(ya[3]));
    }
    // Row scale s_i = fp16(clamp(absmax_i / q_b)), absmax_i = a_i max_j |Z_ij|
    // (lanes l and l ^ 1 hold the same row; the even one writes it).
    bool capped;                                            // a row of the warp's band was capped
    {
        int rr;
        const float zmax = warp_row_max(rm, t.l, rr);
        const int i = t.row(rr);
        const float a = S.rA[i];
        const float q = __fdiv_rn(a * zmax, (float)qm);
        capped = __any_sync(0xffffffffu, q > kF16Max);
        if ((t.l & 1) == 0) {
            const float s = __half2float(__float2half_rn(fminf(fmaxf(q, kF16Min), kF16Max)));
            S.rTs[i] = a * __frcp_rn(s);                      // t = Z (a / s)
            S.rLim[i] = q > kF16Max ? (float)qm : 3.0e38f;
            page_s[i] = f16_bits(s);
        }
    }
    __syncthreads();
    if (t.tid < 128) {                                      // readout sums
        float s = S.red[8 * 128 + t.tid];
#pragma unroll
        for (int wv = 1; wv < 8; wv++) s += S.red[(8 + wv) * 128 + t.tid];
        y_out[t.tid] = s;
    }
    // Codes rne(X / s_i) (clamped only in warps with a capped row), in place.
    if (capped) requant_rows<B, true>(t, S, codes, x2);
    else requant_rows<B, false>(t, S, codes, x2);
    return true;
}

__global__ void __launch_bounds__(kThreads, 2) decode_kernel(DecodeArgs a, int bits) {
    extern __shared__ __align__(128) uint8_t smem[];
    const T t;
    const Smem S(smem);
    if ((int)blockIdx.x >= a.items) return;
    if (t.tid == pipe::kProducer) {
        for (int s = 0; s < a.n_stages; s++) mbar_init(&S.bars[s], 1);
        mbar_init_fence();
    }
    __syncthreads();
    const int grp = a.Hv / a.Hk;
    const auto page_of = [&](int h, int slot) {
        return a.pool + (uint64_t)slot * a.slot_bytes + a.layer_off + (uint64_t)h * a.head_bytes;
    };
    const pipe::Shape p{a.items, a.nb, a.n_stages, a.slots, a.pool_slots, a.err, a.stall.wait_cycles,
                        a.stall.withhold_item};
    pipe::run(
        p, S.bars,
        [&](int h, int b, int slot, int s, int lane) {
            uint64_t *bar = &S.bars[s];
            const Stage st(S.stages + (size_t)s * a.stage_bytes, a.page_region);
            const int hk = h / grp;
            const size_t u = (size_t)b * a.Hv + h;
            warp_copy512(st.q, a.q + ((size_t)b * a.Hk + hk) * 128, lane);
            warp_copy512(st.k, a.k + ((size_t)b * a.Hk + hk) * 128, lane);
            warp_copy512(st.v, a.v + u * 128, lane);
            if (a.gate_per_row) warp_copy512(st.gate, a.gate + u * 128, lane);
            else if (lane == 1) cp_async4(st.gb, a.gate + u);
            if (lane == 0) cp_async4(st.gb + 1, a.beta + u);
            cp_async_mbar_arrive(bar);
            __syncwarp();
            if (lane == 0) {
                mbar_arrive_tx(bar, (uint32_t)a.head_bytes);
                bulk_load(st.page, page_of(h, slot), (uint32_t)a.head_bytes, bar);
            }
        },
        [&](int h, int b, int, int s, bool ok, const auto &refill) {
            const size_t u = (size_t)b * a.Hv + h;
            const Stage st(S.stages + (size_t)s * a.stage_bytes, a.page_region);
            const float beta = st.gb[1], gs = a.gate_per_row ? 0.f : st.gb[0];    // staged
            float *y_out = a.y + u * 128;
            if (bits == 8) return decode_item<8>(t, S, st, gs, a.gate_per_row, beta, y_out, ok, refill);
            if (bits == 6) return decode_item<6>(t, S, st, gs, a.gate_per_row, beta, y_out, ok, refill);
            return decode_item<4>(t, S, st, gs, a.gate_per_row, beta, y_out, ok, refill);
        },
        [&](int h, int slot, int s) {
            bulk_store(page_of(h, slot), S.stages + (size_t)s * a.stage_bytes, (uint32_t)a.head_bytes);
        });
}

}  // namespace ib

stepq_status launch_intb_decode(const stepq_config *cfg, int bits, int layer, uint8_t *pool,
                                int pool_slots, const int32_t *slots, int B, const float *q,
                                const float *k, const float *v, const float *beta,
                                const float *gate, float *y, cudaStream_t s) {
    if (bits != 4 && bits != 6 && bits != 8) return STEPQ_ERR_ARG;
    ib::DecodeArgs a{};
    const uint64_t hb = intb_head_bytes(bits);
    const uint64_t per_layer = hb * (uint64_t)cfg->n_value_heads;
    a.pool = pool;
    a.slot_bytes = (per_layer * (uint64_t)cfg->n_layers + 255) / 256 * 256;
    a.layer_off = per_layer * (uint64_t)layer;
    a.head_bytes = hb;
    a.pool_slots = pool_slots;
    a.slots = slots;
    a.Hk = cfg->n_key_heads;
    a.Hv = cfg->n_value_heads;
    a.nb = B;
    a.items = B * a.Hv;
    a.gate_per_row = cfg->gate_kind == STEPQ_GATE_CHANNEL;
    a.q = q; a.k = k; a.v = v; a.beta = beta; a.gate = gate; a.y = y;
    a.err = device_error_word();
    a.stall = stall_knob();
    a.page_region = (uint32_t)((hb + 127) / 128 * 128);
    a.vec_bytes = a.gate_per_row ? 2048 : 1536;
    a.stage_bytes = a.page_region + 2048 + 128;
    int stages = (int)((113 * 1024 - ib::kOffStages) / a.stage_bytes);
    stages = stages < 2 ? 2 : (stages > 4 ? 4 : stages);
    a.n_stages = stages;
    const int smem = ib::kOffStages + stages * (int)a.stage_bytes;
    if (cudaFuncSetAttribute((const void *)ib::decode_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             smem) != cudaSuccess)
        return STEPQ_ERR_CUDA;
    int dev = 0, sms = 1;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    int grid = 2 * (sms > 0 ? sms : 1);
    if (grid > a.items) grid = a.items;
    ib::decode_kernel<<<grid, kThreads, smem, s>>>(a, bits);
    return cudaGetLastError() == cudaSuccess ? STEPQ_OK : STEPQ_ERR_CUDA;
}

}  // namespace stepq
