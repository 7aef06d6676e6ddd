// Register-tile helpers shared by the fused decode kernels: the magic-number
// rounding constant, f32x2 pair sums and clamps, and the warp reduce-scatter
// of per-row partial sums.
#pragma once

#include <cstdint>

#include "async.cuh"

namespace stepq {

constexpr float kMagic = 12582912.0f;                  // 1.5 * 2^23: rint by addition
constexpr uint32_t kMagicBits = 0x4B400000u;           // its bit pattern (low 22 bits zero)

__device__ __forceinline__ float pair_sum(uint64_t v) { return f2lo(v) + f2hi(v); }

__device__ __forceinline__ uint64_t clamp2(uint64_t v, float lim) {
    return f2(fminf(fmaxf(f2lo(v), -lim), lim), fminf(fmaxf(f2hi(v), -lim), lim));
}

// Clamp of a pair to [lo, hi] per half (used on magic-biased codes).
__device__ __forceinline__ uint64_t clamp2r(uint64_t v, uint64_t lo, uint64_t hi) {
    return f2(fminf(fmaxf(f2lo(v), f2lo(lo)), f2lo(hi)), fminf(fmaxf(f2hi(v), f2hi(lo)), f2hi(hi)));
}

// Nearest integer (ties to even) of the exact product a * b for |a b| < 2^22:
// one fused multiply-add with 1.5 * 2^23 rounds it once. Larger products come
// out within a few units of a b, which every caller clamps to +-qmax anyway.
__device__ __forceinline__ float rne_prod(float a, float b) {
    return __fmaf_rn(a, b, 12582912.0f) - 12582912.0f;
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

}  // namespace stepq
