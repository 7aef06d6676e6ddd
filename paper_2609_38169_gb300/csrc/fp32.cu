// FP32-state comparison decode (the serving default the paper measures against,
// Sec. 5.1): X = D S + beta k (v - k^T D S)^T and y = X^T q with the state kept
// in fp32, on the same persistent bulk-async pipeline and tile as the
// compressed kernels. A head page is the 64 KB fp32 state, so one CTA per SM
// keeps three pages staged (two in flight while it updates the third).
//
// Tile mapping: warp w owns key rows 16w..16w+15, lane l the value columns
// 4l..4l+3 (one 128-bit shared-memory access per row); the updated state is
// written back into the stage and leaves with the page's bulk store.
#include "async.cuh"
#include "device.cuh"
#include "internal.h"
#include "pipeline.cuh"
#include "tile.cuh"

namespace stepq {
namespace fk {

constexpr int kPage = kN * 4;                          // 65,536 B
constexpr int kVecBytes = 4 * 512 + 128;               // q k v | gate (channel gates) | scalar gate, beta
constexpr int kOffBars = 0;                            // uint64 [8]
constexpr int kOffRed = 64;                            // float [2][8][128]: retrieval, readout
constexpr int kOffColD = kOffRed + 2 * 8 * 128 * 4;    // float [128] delta_j
constexpr int kOffRows = kOffColD + 512;               // float4 [2][128]
constexpr int kOffStages = (kOffRows + 2 * 128 * 16 + 127) / 128 * 128;
constexpr int kStage = kPage + kVecBytes;

struct DecodeArgs {
    uint8_t *pool;
    const uint8_t *read_pool;   // exact-read variant: the states the retrieval reads
    uint64_t slot_bytes, layer_off;
    int pool_slots;
    const int32_t *slots;
    int Hk, Hv, nb, items, gate_per_row, n_stages;
    const float *q, *k, *v, *beta, *gate;
    float *y;
    unsigned int *err;
    StallKnob stall;
};

__device__ __forceinline__ void row_dup(const float4 *v, int i, uint64_t &xx, uint64_t &zz) {
    const uint4 q = *(const uint4 *)&v[i];
    xx = u2pair(q.x, q.y);
    zz = u2pair(q.z, q.w);
}

// READ: the retrieval reads u = k^T D S_ref from read_pool (same layout)
// instead of the page's own state; the update still writes D S + beta k (v - u)^T.
template <bool READ>
__global__ void __launch_bounds__(kThreads, 1) decode_kernel(DecodeArgs a) {
    extern __shared__ __align__(128) uint8_t smem[];
    uint64_t *bars = (uint64_t *)(smem + kOffBars);
    float *red = (float *)(smem + kOffRed), *colD = (float *)(smem + kOffColD);
    float4 *rowA = (float4 *)(smem + kOffRows), *rowB = rowA + 128;   // (d d k k), (bk bk q q)
    uint8_t *stages = smem + kOffStages;
    const int tid = threadIdx.x, w = tid >> 5, l = tid & 31;
    if ((int)blockIdx.x >= a.items) return;
    if (tid == pipe::kProducer) {
        for (int s = 0; s < a.n_stages; s++) mbar_init(&bars[s], 1);
        mbar_init_fence();
    }
    __syncthreads();
    const int grp = a.Hv / a.Hk;
    const auto page_of = [&](int h, int slot) {
        return a.pool + (uint64_t)slot * a.slot_bytes + a.layer_off + (uint64_t)h * kPage;
    };
    const pipe::Shape p{a.items, a.nb, a.n_stages, a.slots, a.pool_slots, a.err, a.stall.wait_cycles,
                        a.stall.withhold_item};
    pipe::run(
        p, bars,
        [&](int h, int b, int slot, int s, int lane) {
            uint8_t *st = stages + (size_t)s * kStage;
            float *vec = (float *)(st + kPage);
            const int hk = h / grp;
            const size_t u = (size_t)b * a.Hv + h;
            warp_copy512(vec, a.q + ((size_t)b * a.Hk + hk) * 128, lane);
            warp_copy512(vec + 128, a.k + ((size_t)b * a.Hk + hk) * 128, lane);
            warp_copy512(vec + 256, a.v + u * 128, lane);
            if (a.gate_per_row) warp_copy512(vec + 384, a.gate + u * 128, lane);
            else if (lane == 1) cp_async4(vec + 512, a.gate + u);
            if (lane == 0) cp_async4(vec + 513, a.beta + u);
            cp_async_mbar_arrive(&bars[s]);
            __syncwarp();
            if (lane == 0) {
                mbar_arrive_tx(&bars[s], kPage);
                bulk_load(st, page_of(h, slot), kPage, &bars[s]);
            }
        },
        [&](int h, int b, int slot, int s, bool ok, const auto &refill) {
            const size_t u = (size_t)b * a.Hv + h;
            float *S = (float *)(stages + (size_t)s * kStage);
            const float *sv = S + kN;
            const float beta = sv[513], gs = a.gate_per_row ? 0.f : sv[512];       // staged
            const float *q = S + kN, *k = q + 128, *v = q + 256, *gv = q + 384;
            if (l < 16) {
                const int i = 16 * w + l;
                const float d = a.gate_per_row ? gv[i] : gs, ki = k[i];
                rowA[i] = make_float4(d, d, ki, ki);
                rowB[i] = make_float4(beta * ki, beta * ki, q[i], q[i]);
            }
            __syncwarp();
            // P = D S (fp32) and the retrieval u_j = sum_i k_i P_ij.
            uint64_t x2[16][2];
            uint64_t ua[2] = {0, 0}, ub[2] = {0, 0};
#pragma unroll
            for (int r = 0; r < 16; r++) {
                uint64_t dd, kk;
                row_dup(rowA, 16 * w + r, dd, kk);
                const uint4 sv = *(const uint4 *)&S[(16 * w + r) * 128 + 4 * l];
                x2[r][0] = fmul2(u2pair(sv.x, sv.y), dd);
                x2[r][1] = fmul2(u2pair(sv.z, sv.w), dd);
                uint64_t(&acc)[2] = (r & 1) ? ub : ua;
                if (READ) {
                    const float *Sr = (const float *)(a.read_pool + (page_of(h, slot) - a.pool));
                    const float4 rv = *(const float4 *)&Sr[(16 * w + r) * 128 + 4 * l];
                    acc[0] = ffma2(kk, fmul2(f2(rv.x, rv.y), dd), acc[0]);
                    acc[1] = ffma2(kk, fmul2(f2(rv.z, rv.w), dd), acc[1]);
                } else {
                    acc[0] = ffma2(kk, x2[r][0], acc[0]);
                    acc[1] = ffma2(kk, x2[r][1], acc[1]);
                }
            }
            {
                const uint64_t s0 = fadd2(ua[0], ub[0]), s1 = fadd2(ua[1], ub[1]);
                *(float4 *)&red[w * 128 + 4 * l] = make_float4(f2lo(s0), f2hi(s0), f2lo(s1), f2hi(s1));
            }
            if (__syncthreads_or(!ok)) return false;
            if (tid < 128) {
                float sum = 0.f;
#pragma unroll
                for (int wv = 0; wv < 8; wv++) sum += red[wv * 128 + tid];
                colD[tid] = v[tid] - sum;                      // delta_j = v_j - u_j
            }
            refill();
            __syncthreads();
            // X = P + beta k_i delta_j, written back in place; readout y = X^T q.
            const uint4 dq = *(const uint4 *)&colD[4 * l];
            const uint64_t d01 = u2pair(dq.x, dq.y), d23 = u2pair(dq.z, dq.w);
            uint64_t ya[2] = {0, 0}, yb[2] = {0, 0};
#pragma unroll
            for (int r = 0; r < 16; r++) {
                uint64_t bk, qq;
                row_dup(rowB, 16 * w + r, bk, qq);
                const uint64_t x0 = ffma2(bk, d01, x2[r][0]), x1 = ffma2(bk, d23, x2[r][1]);
                uint64_t(&acc)[2] = (r & 1) ? yb : ya;
                acc[0] = ffma2(qq, x0, acc[0]);
                acc[1] = ffma2(qq, x1, acc[1]);
                *(uint4 *)&S[(16 * w + r) * 128 + 4 * l] =
                    make_uint4((uint32_t)x0, (uint32_t)(x0 >> 32), (uint32_t)x1, (uint32_t)(x1 >> 32));
            }
            {
                const uint64_t s0 = fadd2(ya[0], yb[0]), s1 = fadd2(ya[1], yb[1]);
                *(float4 *)&red[(8 + w) * 128 + 4 * l] = make_float4(f2lo(s0), f2hi(s0), f2lo(s1), f2hi(s1));
            }
            __syncthreads();
            if (tid < 128) {
                float sum = red[8 * 128 + tid];
#pragma unroll
                for (int wv = 1; wv < 8; wv++) sum += red[(8 + wv) * 128 + tid];
                a.y[u * 128 + tid] = sum;
            }
            return true;
        },
        [&](int h, int slot, int s) { bulk_store(page_of(h, slot), stages + (size_t)s * kStage, kPage); });
}

}  // namespace fk

stepq_status launch_fp32_decode(const stepq_config *cfg, int layer, float *pool,
                                const float *read_pool, int pool_slots, const int32_t *slots, int B,
                                const float *q, const float *k, const float *v, const float *beta,
                                const float *gate, float *y, cudaStream_t s) {
    fk::DecodeArgs a{};
    a.read_pool = (const uint8_t *)read_pool;
    const uint64_t per_layer = (uint64_t)fk::kPage * (uint64_t)cfg->n_value_heads;
    a.pool = (uint8_t *)pool;
    a.slot_bytes = per_layer * (uint64_t)cfg->n_layers;
    a.layer_off = per_layer * (uint64_t)layer;
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
    int dev = 0, sms = 1, max_smem = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    cudaDeviceGetAttribute(&max_smem, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    int stages = (max_smem - fk::kOffStages) / fk::kStage;
    stages = stages < 2 ? 2 : (stages > 3 ? 3 : stages);
    a.n_stages = stages;
    const int smem = fk::kOffStages + stages * fk::kStage;
    const void *fn = read_pool ? (const void *)fk::decode_kernel<true> : (const void *)fk::decode_kernel<false>;
    if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
        return STEPQ_ERR_CUDA;
    int grid = sms > 0 ? sms : 1;
    if (grid > a.items) grid = a.items;
    if (read_pool) fk::decode_kernel<true><<<grid, kThreads, smem, s>>>(a);
    else fk::decode_kernel<false><<<grid, kThreads, smem, s>>>(a);
    return cudaGetLastError() == cudaSuccess ? STEPQ_OK : STEPQ_ERR_CUDA;
}

}  // namespace stepq
