// Device building blocks of the decode-step kernels: the head tile mapping,
// sub-byte code (un)packing, fp16 helpers and the column/row reductions.
//
// Tile mapping (one 128 x 128 head per 256-thread CTA): warp w owns key rows
// 16w..16w+15; lane = 8*rs + cg; a thread holds 4 rows (16w + 4t + rs, t = 0..3)
// by 16 consecutive value columns (16cg..16cg+15), i.e. 64 fp32 values in
// registers. Sixteen codes of one row occupy 2b bytes (a whole number of
// 32-bit words for every b in {2,4,6,8}), so each thread reads and writes its
// codes with aligned word accesses.
#pragma once

#include <cstdint>
#include <cuda_fp16.h>

namespace stepq {

constexpr int kThreads = 256;
constexpr float kF16Min = 6.103515625e-05f;   // 2^-14
constexpr float kF16Max = 65504.0f;

// Sticky device error word (see errors.cu): the first status raised wins.
__device__ __forceinline__ void raise_error(unsigned int *err, unsigned int code) {
    atomicCAS(err, 0u, code);
}

struct Lane {
    int tid, warp, lane, cg, rs;
    __device__ __forceinline__ Lane() {
        tid = threadIdx.x;
        warp = tid >> 5;
        lane = tid & 31;
        cg = lane & 7;
        rs = lane >> 3;
    }
    __device__ __forceinline__ int row(int t) const { return 16 * warp + 4 * t + rs; }
    __device__ __forceinline__ int col0() const { return 16 * cg; }
};

__device__ __forceinline__ float f16_round_sat(float x) {      // binary16 RNE, saturating
    return __half2float(__float2half_rn(fminf(fmaxf(x, -kF16Max), kF16Max)));
}
__device__ __forceinline__ uint16_t f16_bits(float x) {        // x already representable
    return __half_as_ushort(__float2half_rn(x));
}
__device__ __forceinline__ float f16_val(uint16_t h) { return __half2float(__ushort_as_half(h)); }

// ---- code (un)packing: 16 codes of width B, LSB-first, offset binary ----

template <int B>
__device__ __forceinline__ void unpack16(const uint32_t *wd, float q[16]) {
    constexpr uint32_t mask = (1u << B) - 1u;
    constexpr int off = 1 << (B - 1);
#pragma unroll
    for (int j = 0; j < 16; j++) {
        const int bit = j * B, wi = bit >> 5, sh = bit & 31;
        uint32_t u;
        if (sh + B <= 32)
            u = (wd[wi] >> sh) & mask;
        else
            u = __funnelshift_r(wd[wi], wd[wi + 1], sh) & mask;
        q[j] = (float)((int)u - off);
    }
}

template <int B>
__device__ __forceinline__ void pack16(const int q[16], uint32_t *wd) {
    constexpr int W = B / 2;
    constexpr int off = 1 << (B - 1);
#pragma unroll
    for (int t = 0; t < W; t++) wd[t] = 0u;
#pragma unroll
    for (int j = 0; j < 16; j++) {
        const uint32_t u = (uint32_t)(q[j] + off);
        const int bit = j * B, wi = bit >> 5, sh = bit & 31;
        wd[wi] |= u << sh;
        if (sh + B > 32) wd[wi + 1] |= u >> (32 - sh);
    }
}

// Load 16 values of row payload `row` for column group cg: integer codes as
// floats (q), or FP16 pivot values.
__device__ __forceinline__ void load_row16(const uint8_t *row, int bits, int cg, float out[16]) {
    switch (bits) {
    case 2: {
        uint32_t wd[1] = {*(const uint32_t *)(row + 4 * cg)};
        unpack16<2>(wd, out);
    } break;
    case 4: {
        uint2 a = *(const uint2 *)(row + 8 * cg);
        uint32_t wd[2] = {a.x, a.y};
        unpack16<4>(wd, out);
    } break;
    case 6: {
        const uint32_t *p = (const uint32_t *)(row + 12 * cg);
        uint32_t wd[3] = {p[0], p[1], p[2]};
        unpack16<6>(wd, out);
    } break;
    case 8: {
        uint4 a = *(const uint4 *)(row + 16 * cg);
        uint32_t wd[4] = {a.x, a.y, a.z, a.w};
        unpack16<8>(wd, out);
    } break;
    default: {   // FP16 pivot row
        const uint4 *p = (const uint4 *)(row + 32 * cg);
        uint4 a = p[0], b = p[1];
        uint32_t wd[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
#pragma unroll
        for (int t = 0; t < 8; t++) {
            out[2 * t] = f16_val((uint16_t)(wd[t] & 0xFFFFu));
            out[2 * t + 1] = f16_val((uint16_t)(wd[t] >> 16));
        }
    } break;
    }
}

__device__ __forceinline__ void store_codes16(uint8_t *row, int bits, int cg, const int q[16]) {
    switch (bits) {
    case 2: {
        uint32_t wd[1];
        pack16<2>(q, wd);
        *(uint32_t *)(row + 4 * cg) = wd[0];
    } break;
    case 4: {
        uint32_t wd[2];
        pack16<4>(q, wd);
        *(uint2 *)(row + 8 * cg) = make_uint2(wd[0], wd[1]);
    } break;
    case 6: {
        uint32_t wd[3];
        pack16<6>(q, wd);
        uint32_t *p = (uint32_t *)(row + 12 * cg);
        p[0] = wd[0];
        p[1] = wd[1];
        p[2] = wd[2];
    } break;
    default: {
        uint32_t wd[4];
        pack16<8>(q, wd);
        *(uint4 *)(row + 16 * cg) = make_uint4(wd[0], wd[1], wd[2], wd[3]);
    } break;
    }
}

__device__ __forceinline__ void store_f16_row16(uint8_t *row, int cg, const float x[16]) {
    uint32_t wd[8];
#pragma unroll
    for (int t = 0; t < 8; t++)
        wd[t] = (uint32_t)f16_bits(f16_round_sat(x[2 * t])) |
                ((uint32_t)f16_bits(f16_round_sat(x[2 * t + 1])) << 16);
    uint4 *p = (uint4 *)(row + 32 * cg);
    p[0] = make_uint4(wd[0], wd[1], wd[2], wd[3]);
    p[1] = make_uint4(wd[4], wd[5], wd[6], wd[7]);
}

// ---- reductions over the head tile ----

// Column reduction of NR partial vectors acc[r][16] (each over the thread's 4
// rows) into out[r][128] in shared memory. red: shared [NR][8][128] floats.
// Reduce-scatter over the 4 rs lanes, then a sum over the 8 warps.
template <int NR, bool MAX>
__device__ __forceinline__ void column_reduce(const Lane &L, float (&acc)[NR][16], float *red,
                                              float *out) {
#pragma unroll
    for (int r = 0; r < NR; r++) {
        float h8[8];
        const bool hi16 = (L.rs & 2) != 0;
#pragma unroll
        for (int t = 0; t < 8; t++) {
            float keep = hi16 ? acc[r][8 + t] : acc[r][t];
            float send = hi16 ? acc[r][t] : acc[r][8 + t];
            float got = __shfl_xor_sync(0xffffffffu, send, 16);
            h8[t] = MAX ? fmaxf(keep, got) : keep + got;
        }
        float h4[4];
        const bool hi8 = (L.rs & 1) != 0;
#pragma unroll
        for (int t = 0; t < 4; t++) {
            float keep = hi8 ? h8[4 + t] : h8[t];
            float send = hi8 ? h8[t] : h8[4 + t];
            float got = __shfl_xor_sync(0xffffffffu, send, 8);
            h4[t] = MAX ? fmaxf(keep, got) : keep + got;
        }
        const int col = L.col0() + 8 * (L.rs >> 1) + 4 * (L.rs & 1);
        *(float4 *)&red[(r * 8 + L.warp) * 128 + col] = make_float4(h4[0], h4[1], h4[2], h4[3]);
    }
    __syncthreads();
    for (int e = L.tid; e < NR * 128; e += kThreads) {
        const int r = e >> 7, c = e & 127;
        float s = red[(r * 8) * 128 + c];
#pragma unroll
        for (int wv = 1; wv < 8; wv++) {
            float x = red[(r * 8 + wv) * 128 + c];
            s = MAX ? fmaxf(s, x) : s + x;
        }
        out[r * 128 + c] = s;
    }
    __syncthreads();
}

// Sum over the 16 columns a thread holds and the 8 cg lanes of its row group:
// every lane of the group receives the full row sum.
__device__ __forceinline__ float row_allreduce(float s) {
    s += __shfl_xor_sync(0xffffffffu, s, 1);
    s += __shfl_xor_sync(0xffffffffu, s, 2);
    s += __shfl_xor_sync(0xffffffffu, s, 4);
    return s;
}

}  // namespace stepq
