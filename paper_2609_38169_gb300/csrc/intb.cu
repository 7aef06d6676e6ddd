// Uniform rowwise-absmax INT-b comparison decode (App. B.5: per key row an FP16
// scale s_i = absmax_i / q_b in [2^-14, 65504], nearest codes in [-q_b, q_b]),
// on the same persistent bulk-async pipeline and tile as the row-unit STEPQuant
// kernel, so that the comparison measures the codecs and not the plumbing.
//
// Tile mapping: warp w owns key rows 16w..16w+15, lane l the value columns
// 4l..4l+3; a lane's 4 codes of a row are one word (8-bit), three bytes at
// byte 3l (6-bit) or a half-word (4-bit).
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
constexpr int kOffRows = kOffColD + 512;               // float4 [3][128] per-row constants
constexpr int kOffStages = (kOffRows + 3 * 128 * 16 + 127) / 128 * 128;

struct Smem {
    uint64_t *bars;
    float *red, *colD;
    float4 *rowK;   // (kappa, kappa, beta k / a, beta k / a), kappa = k a
    float4 *rowQ;   // (q a, q a, a, a)
    float4 *rowT;   // (a / s_new, a / s_new, clamp limit or 0, -)
    uint8_t *stages;
    __device__ __forceinline__ explicit Smem(uint8_t *s) {
        bars = (uint64_t *)(s + kOffBars);
        red = (float *)(s + kOffRed);
        colD = (float *)(s + kOffColD);
        rowK = (float4 *)(s + kOffRows);
        rowQ = rowK + 128;
        rowT = rowK + 256;
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

__device__ __forceinline__ void row_dup(const float4 *v, int i, uint64_t &xx, uint64_t &zz) {
    const uint4 q = *(const uint4 *)&v[i];
    xx = u2pair(q.x, q.y);
    zz = u2pair(q.z, q.w);
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

template <int B>
__device__ __forceinline__ void decode_row(const uint8_t *row, int l, uint64_t &x0, uint64_t &x1) {
    uint32_t f0, f1, f2, f3;
    if (B == 8) {
        const uint32_t w = ((const uint32_t *)row)[l];
        f0 = __byte_perm(w, kMagicBits, 0x7650);
        f1 = __byte_perm(w, kMagicBits, 0x7651);
        f2 = __byte_perm(w, kMagicBits, 0x7652);
        f3 = __byte_perm(w, kMagicBits, 0x7653);
    } else if (B == 6) {
        // 24 bits at bit 24 l: a funnel shift of the two words that hold them
        // (the last lane's upper word is clamped into the row; it is unused).
        const uint32_t *wd = (const uint32_t *)row;
        const int wi = (3 * l) >> 2;
        const uint32_t x = __funnelshift_r(wd[wi], wd[min(wi + 1, 23)], 8 * ((3 * l) & 3));
        f0 = and_or(x, 0x3Fu, kMagicBits);
        f1 = and_or(x >> 6, 0x3Fu, kMagicBits);
        f2 = and_or(x >> 12, 0x3Fu, kMagicBits);
        f3 = and_or(x >> 18, 0x3Fu, kMagicBits);
    } else {
        const uint32_t x = ((const uint16_t *)row)[l];
        f0 = and_or(x, 0xFu, kMagicBits);
        f1 = and_or(x >> 4, 0xFu, kMagicBits);
        f2 = and_or(x >> 8, 0xFu, kMagicBits);
        f3 = and_or(x >> 12, 0xFu, kMagicBits);
    }
    const uint64_t off = f2s(-(kMagic + (float)(1 << (B - 1))));
    x0 = fadd2(u2pair(f0, f1), off);
    x1 = fadd2(u2pair(f2, f3), off);
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
        const float ki = st.k[i], kap = ki * a, bkp = __fdividef(beta * ki, a), qa = st.q[i] * a;
        S.rowK[i] = make_float4(kap, kap, bkp, bkp);
        S.rowQ[i] = make_float4(qa, qa, a, a);
    }
    uint64_t x2[16][2];
#pragma unroll
    for (int r = 0; r < 16; r++) decode_row<B>(codes + t.row(r) * 16 * B, t.l, x2[r][0], x2[r][1]);
    __syncwarp();
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
        *(float4 *)&S.red[t.w * 128 + 4 * t.l] = make_float4(f2lo(s0), f2hi(s0), f2lo(s1), f2hi(s1));
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
        const uint4 dq = *(const uint4 *)&S.colD[4 * t.l];
        const uint64_t d01 = u2pair(dq.x, dq.y), d23 = u2pair(dq.z, dq.w);
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
            rm[r] = fmax3(fmax3(0.f, fabsf(f2lo(x2[r][0])), fabsf(f2hi(x2[r][0]))),
                          fabsf(f2lo(x2[r][1])), fabsf(f2hi(x2[r][1])));
        }
        const uint64_t s0 = fadd2(ya[0], yb[0]), s1 = fadd2(ya[1], yb[1]);
        *(float4 *)&S.red[(8 + t.w) * 128 + 4 * t.l] = make_float4(f2lo(s0), f2hi(s0), f2lo(s1), f2hi(s1));
    }
    // Row scale s_i = fp16(clamp(absmax_i / q_b)), absmax_i = a_i max_j |Z_ij|.
    {
        int rr;
        const float zmax = warp_row_max(rm, t.l, rr);
        const int i = t.row(rr);
        if ((t.l & 1) == 0) {
            const float a = S.rowQ[i].z;
            const float q = __fdiv_rn(a * zmax, (float)qm);
            const float s = __half2float(__float2half_rn(fminf(fmaxf(q, kF16Min), kF16Max)));
            const float ts = a * __frcp_rn(s);                // t = Z (a / s)
            S.rowT[i] = make_float4(ts, ts, q > kF16Max ? (float)qm : 0.f, 0.f);
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
    // Codes rne(X / s_i) (clamped only where the scale was capped), in place.
    const uint64_t mb = f2s(kMagic + (float)(1 << (B - 1)));
#pragma unroll
    for (int r = 0; r < 16; r++) {
        uint64_t ts, lim;
        row_dup(S.rowT, t.row(r), ts, lim);
        uint64_t t0 = fmul2(x2[r][0], ts), t1 = fmul2(x2[r][1], ts);
        const float cl = f2lo(lim);
        if (cl != 0.f) {
            t0 = clamp2(t0, cl);
            t1 = clamp2(t1, cl);
        }
        const uint64_t u0 = fadd2(t0, mb), u1 = fadd2(t1, mb);
        store_row<B>(codes + t.row(r) * 16 * B, t.l, (uint32_t)u0, (uint32_t)(u0 >> 32), (uint32_t)u1,
                     (uint32_t)(u1 >> 32));
    }
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
