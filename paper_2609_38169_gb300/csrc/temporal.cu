// Pack/unpack of the "Temporal only" ablation state (Sec. 5.4): the plan's
// calibrated widths and FP16 pivots, with the uniform baseline's rowwise
// quantizer (App. B.5: s_i = fp16(clamp(absmax_i / q_b)), nearest codes of
// X * fp32(1/s_i)) in place of the dual-axis fit. A pivot row stores fp16(X)
// and s_i = 0. Head segment: s[128] fp16, then row i in index order, 16 b_i
// bytes; segments in (layer, head) order (plan tables t_head_off, t_row_off).
//
// One CTA per (slot, value head); lane (warp, rs) owns key rows 16w + 4t + rs
// and the 16 columns of group cg. The row absmax is reduced over the 8 lanes of
// a row before any branch on the row's width, so every shuffle is warp-uniform.
#include "device.cuh"
#include "internal.h"

namespace stepq {
namespace tq {

struct Args {
    uint8_t *pool;
    uint64_t slot_bytes;
    const uint64_t *head_off;   // [Hv] of this layer
    const uint32_t *row_off;    // [Hv][128] of this layer
    const uint8_t *row_bits;    // [Hv][128] of this layer (16 = pivot)
    int pool_slots, Hv;
    const int32_t *slots;
    float *states;
    size_t state_stride_b;
    unsigned int *err;
};

__device__ __forceinline__ int unit_slot(const Args &a, int &b, int &h) {
    b = blockIdx.x / a.Hv;
    h = blockIdx.x - b * a.Hv;
    const int slot = a.slots[b];
    if (slot < 0 || slot >= a.pool_slots) {
        if (threadIdx.x == 0) raise_error(a.err, STEPQ_ERR_SLOT_RANGE);
        return -1;
    }
    return slot;
}

__global__ void __launch_bounds__(kThreads) quantize_kernel(Args a) {
    const Lane L;
    int b, h;
    const int slot = unit_slot(a, b, h);
    if (slot < 0) return;
    uint8_t *seg = a.pool + (uint64_t)slot * a.slot_bytes + a.head_off[h];
    const float *X = a.states + (size_t)b * a.state_stride_b + (size_t)h * kN;
#pragma unroll
    for (int t = 0; t < 4; t++) {
        const int i = L.row(t);
        float x[16];
        const float4 *src = (const float4 *)(X + i * 128 + L.col0());
#pragma unroll
        for (int e = 0; e < 4; e++) {
            const float4 f = src[e];
            x[4 * e] = f.x;
            x[4 * e + 1] = f.y;
            x[4 * e + 2] = f.z;
            x[4 * e + 3] = f.w;
        }
        float amax = 0.f;
#pragma unroll
        for (int j = 0; j < 16; j++) amax = fmaxf(amax, fabsf(x[j]));
        amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, 1));
        amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, 2));
        amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, 4));
        const int bits = a.row_bits[h * kD + i];
        uint8_t *row = seg + a.row_off[h * kD + i];
        if (bits == 16) {
            if (L.cg == 0) ((uint16_t *)seg)[i] = 0;
            store_f16_row16(row, L.cg, x);
            continue;
        }
        const int qm = (1 << (bits - 1)) - 1;
        const float lim = (float)qm;
        const float s = __half2float(__float2half_rn(
            fminf(fmaxf(__fdiv_rn(amax, (float)qm), kF16Min), kF16Max)));
        const float inv = __frcp_rn(s);
        if (L.cg == 0) ((uint16_t *)seg)[i] = f16_bits(s);
        int q[16];
#pragma unroll
        for (int j = 0; j < 16; j++) q[j] = (int)fminf(fmaxf(rintf(__fmul_rn(x[j], inv)), -lim), lim);
        store_codes16(row, bits, L.cg, q);
    }
}

__global__ void __launch_bounds__(kThreads) dequantize_kernel(Args a) {
    const Lane L;
    int b, h;
    const int slot = unit_slot(a, b, h);
    if (slot < 0) return;
    const uint8_t *seg = a.pool + (uint64_t)slot * a.slot_bytes + a.head_off[h];
    float *out = a.states + (size_t)b * a.state_stride_b + (size_t)h * kN;
#pragma unroll
    for (int t = 0; t < 4; t++) {
        const int i = L.row(t);
        const int bits = a.row_bits[h * kD + i];
        float v[16];
        load_row16(seg + a.row_off[h * kD + i], bits, L.cg, v);
        if (bits != 16) {
            const float s = f16_val(((const uint16_t *)seg)[i]);
#pragma unroll
            for (int j = 0; j < 16; j++) v[j] = __fmul_rn(s, v[j]);
        }
        float4 *dst = (float4 *)(out + i * 128 + L.col0());
#pragma unroll
        for (int e = 0; e < 4; e++) dst[e] = make_float4(v[4 * e], v[4 * e + 1], v[4 * e + 2], v[4 * e + 3]);
    }
}

static Args args(const stepq_plan *p, int layer, uint8_t *pool, int pool_slots, const int32_t *slots,
                 float *states, size_t state_stride_b) {
    const size_t Hv = (size_t)p->cfg.n_value_heads;
    Args a{};
    a.pool = pool;
    a.slot_bytes = p->t_slot_stride;
    a.head_off = p->d_t_head_off + layer * Hv;
    a.row_off = p->d_t_row_off + layer * Hv * kD;
    a.row_bits = p->d_row_bits + layer * Hv * kD;
    a.pool_slots = pool_slots;
    a.Hv = (int)Hv;
    a.slots = slots;
    a.states = states;
    a.state_stride_b = state_stride_b;
    a.err = device_error_word();
    return a;
}

}  // namespace tq

stepq_status launch_temporal_quantize(const stepq_plan *p, int layer, const float *states,
                                      size_t state_stride_b, const int32_t *slots, int B,
                                      uint8_t *pool, int pool_slots, cudaStream_t s) {
    tq::Args a = tq::args(p, layer, pool, pool_slots, slots, (float *)states, state_stride_b);
    tq::quantize_kernel<<<(unsigned)B * p->cfg.n_value_heads, kThreads, 0, s>>>(a);
    return cudaGetLastError() == cudaSuccess ? STEPQ_OK : STEPQ_ERR_CUDA;
}

stepq_status launch_temporal_dequantize(const stepq_plan *p, int layer, const uint8_t *pool,
                                        int pool_slots, const int32_t *slots, int B, float *states,
                                        size_t state_stride_b, cudaStream_t s) {
    tq::Args a = tq::args(p, layer, (uint8_t *)pool, pool_slots, slots, states, state_stride_b);
    tq::dequantize_kernel<<<(unsigned)B * p->cfg.n_value_heads, kThreads, 0, s>>>(a);
    return cudaGetLastError() == cudaSuccess ? STEPQ_OK : STEPQ_ERR_CUDA;
}

}  // namespace stepq
