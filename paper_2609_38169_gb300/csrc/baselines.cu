// Pack/unpack of the uniform rowwise-absmax INT-b comparison state (App. B.5:
// per key row an FP16 scale absmax/q_b in [2^-14, 65504], nearest codes in
// [-q_b, q_b]). One CTA per (slot, value head); the pipelined INT-b decode step
// is in intb.cu and the FP32-state step in fp32.cu.
#include "device.cuh"
#include "internal.h"

namespace stepq {

size_t intb_head_bytes(int bits) { return 256 + (size_t)kD * 16 * bits; }

struct BaseArgs {
    uint8_t *pool;              // INT-b pool
    uint64_t slot_bytes;        // bytes per slot page
    uint64_t layer_off;         // byte offset of the layer inside a page
    uint64_t head_bytes;        // bytes per head segment
    int pool_slots;
    const int32_t *slots;
    int Hk, Hv, gate_per_row, bits;
    const float *q, *k, *v, *beta, *gate;
    float *y;
    float *states;              // dense states for quantize / dequantize
    size_t state_stride_b;
    unsigned int *err;
};

__device__ __forceinline__ int unit_slot(const BaseArgs &a, int &b, int &h) {
    b = blockIdx.x / a.Hv;
    h = blockIdx.x - b * a.Hv;
    const int slot = a.slots[b];
    if (slot < 0 || slot >= a.pool_slots) {
        if (threadIdx.x == 0) raise_error(a.err, STEPQ_ERR_SLOT_RANGE);
        return -1;
    }
    return slot;
}

// ---------------------------------------------------------------- INT-b state
// Row scale s_i = fp16(clamp(absmax_i / q_b)) and codes rint(fp32(X * fp32(1/s_i))).
__device__ __forceinline__ void intb_pack(const Lane &L, float (&x)[4][16], uint8_t *page,
                                          int bits) {
    const int qm = (1 << (bits - 1)) - 1;
    const float lim = (float)qm;
#pragma unroll
    for (int t = 0; t < 4; t++) {
        float amax = 0.f;
#pragma unroll
        for (int j = 0; j < 16; j++) amax = fmaxf(amax, fabsf(x[t][j]));
        amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, 1));
        amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, 2));
        amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, 4));
        const float s = __half2float(__float2half_rn(
            fminf(fmaxf(__fdiv_rn(amax, (float)qm), kF16Min), kF16Max)));
        const float inv = __frcp_rn(s);
        const int i = L.row(t);
        if (L.cg == 0) ((uint16_t *)page)[i] = f16_bits(s);
        int q[16];
#pragma unroll
        for (int j = 0; j < 16; j++)
            q[j] = (int)fminf(fmaxf(rintf(__fmul_rn(x[t][j], inv)), -lim), lim);
        store_codes16(page + 256 + (size_t)i * 16 * bits, bits, L.cg, q);
    }
}

__device__ __forceinline__ void intb_unpack(const Lane &L, const uint8_t *page, int bits,
                                            float (&x)[4][16]) {
#pragma unroll
    for (int t = 0; t < 4; t++) {
        const int i = L.row(t);
        const float s = f16_val(((const uint16_t *)page)[i]);
        float vals[16];
        load_row16(page + 256 + (size_t)i * 16 * bits, bits, L.cg, vals);
#pragma unroll
        for (int j = 0; j < 16; j++) x[t][j] = __fmul_rn(s, vals[j]);
    }
}

__global__ void __launch_bounds__(kThreads, 2) intb_quantize_kernel(BaseArgs a) {
    extern __shared__ __align__(16) uint8_t smem[];
    uint8_t *page = smem;
    const Lane L;
    int b, h;
    const int slot = unit_slot(a, b, h);
    if (slot < 0) return;
    const float *X = a.states + (size_t)b * a.state_stride_b + (size_t)h * kN;
    float x[4][16];
#pragma unroll
    for (int t = 0; t < 4; t++) {
        const float4 *src = (const float4 *)(X + L.row(t) * 128 + L.col0());
#pragma unroll
        for (int e = 0; e < 4; e++) {
            const float4 f = src[e];
            x[t][4 * e] = f.x;
            x[t][4 * e + 1] = f.y;
            x[t][4 * e + 2] = f.z;
            x[t][4 * e + 3] = f.w;
        }
    }
    intb_pack(L, x, page, a.bits);
    __syncthreads();
    uint8_t *gpage = a.pool + (uint64_t)slot * a.slot_bytes + a.layer_off + h * a.head_bytes;
    for (int e = L.tid; e < (int)(a.head_bytes >> 4); e += kThreads)
        ((uint4 *)gpage)[e] = ((const uint4 *)page)[e];
}

__global__ void __launch_bounds__(kThreads, 2) intb_dequantize_kernel(BaseArgs a) {
    const Lane L;
    int b, h;
    const int slot = unit_slot(a, b, h);
    if (slot < 0) return;
    const uint8_t *gpage = a.pool + (uint64_t)slot * a.slot_bytes + a.layer_off + h * a.head_bytes;
    float x[4][16];
    intb_unpack(L, gpage, a.bits, x);
    float *out = a.states + (size_t)b * a.state_stride_b + (size_t)h * kN;
#pragma unroll
    for (int t = 0; t < 4; t++) {
        float4 *dst = (float4 *)(out + L.row(t) * 128 + L.col0());
#pragma unroll
        for (int e = 0; e < 4; e++)
            dst[e] = make_float4(x[t][4 * e], x[t][4 * e + 1], x[t][4 * e + 2], x[t][4 * e + 3]);
    }
}

// ------------------------------------------------------------------ launchers
static BaseArgs base_args(const stepq_config *cfg, int bits, int layer, uint8_t *pool,
                          int pool_slots, const int32_t *slots) {
    BaseArgs a{};
    const uint64_t hb = intb_head_bytes(bits);
    const uint64_t per_layer = hb * (uint64_t)cfg->n_value_heads;
    const uint64_t page = per_layer * (uint64_t)cfg->n_layers;
    a.pool = pool;
    a.slot_bytes = (page + 255) / 256 * 256;
    a.layer_off = per_layer * (uint64_t)layer;
    a.head_bytes = hb;
    a.pool_slots = pool_slots;
    a.slots = slots;
    a.Hk = cfg->n_key_heads;
    a.Hv = cfg->n_value_heads;
    a.gate_per_row = cfg->gate_kind == STEPQ_GATE_CHANNEL;
    a.bits = bits;
    a.err = device_error_word();
    return a;
}

stepq_status launch_intb_quantize(const stepq_config *cfg, int bits, int layer,
                                  const float *states, size_t state_stride_b,
                                  const int32_t *slots, int B, uint8_t *pool, int pool_slots,
                                  cudaStream_t s) {
    BaseArgs a = base_args(cfg, bits, layer, pool, pool_slots, slots);
    a.states = (float *)states;
    a.state_stride_b = state_stride_b;
    intb_quantize_kernel<<<(unsigned)B * cfg->n_value_heads, kThreads, (int)intb_head_bytes(bits), s>>>(a);
    return cudaGetLastError() == cudaSuccess ? STEPQ_OK : STEPQ_ERR_CUDA;
}

stepq_status launch_intb_dequantize(const stepq_config *cfg, int bits, int layer,
                                    const uint8_t *pool, int pool_slots, const int32_t *slots,
                                    int B, float *states, size_t state_stride_b, cudaStream_t s) {
    BaseArgs a = base_args(cfg, bits, layer, (uint8_t *)pool, pool_slots, slots);
    a.states = states;
    a.state_stride_b = state_stride_b;
    intb_dequantize_kernel<<<(unsigned)B * cfg->n_value_heads, kThreads, 0, s>>>(a);
    return cudaGetLastError() == cudaSuccess ? STEPQ_OK : STEPQ_ERR_CUDA;
}

}  // namespace stepq
