// Chunked FP32-state prefill: the gated Delta rule (Eq. delta_update) over T
// tokens, 32 tokens at a time, producing the boundary state that
// stepq_quantize_pool packs (the prefill side of App. C.3 / App. F.1: the
// native chunk computation runs on an uncompressed state, and the state is
// packed once at the boundary).
//
// Within a chunk with cumulative gates g_t = d_1 ... d_t (per key channel; a
// scalar gate is the same value in every channel) and S_0 the state before it:
//   S_t = G_t S_0 + sum_{s<=t} G_t G_s^-1 k_s w_s^T,
//   w_t = beta_t (v_t - S_0^T g_t k_t - sum_{s<t} (k_s/g_s . g_t k_t) w_s),
// i.e. (I + A) W = diag(beta) (V - K~ S_0) with K~ = G K, K^ = G^-1 K and
// A_ts = beta_t (K~_t . K^_s) for s < t; the outputs are
//   Y = Q~ S_0 + tril(Q~ K^T) W   (Q~ = G Q, lower triangle with the diagonal),
// and the state after the chunk is S_C = G_C S_0 + K_bar^T W, K_bar = K g_C / g.
//
// The two large products run on the tensor cores (tcgen05, kind::tf32) with
// the state resident in tensor memory as S^T (lane j = value column, column i
// = key row), in split precision: every fp32 operand is a TF32 head plus its
// remainder, and a product is head*head + head*rest + rest*head (the rest*rest
// term is below fp32 rounding of the accumulation), so the chunk keeps fp32
// accuracy:
//   P1  [K~ S_0 ; Q~ S_0]^T = S_0^T [K~ ; Q~]^T   M = 128 (j), N = 64, K = 128
//   P2  S^T += W^T K_bar                            M = 128 (j), N = 128, K = 32
// with A (S^T or W^T) in tensor memory and B ([K~ ; Q~] or K_bar^T) in shared
// memory as K-major core matrices. The 32 x 32 products A and Q~ K^T, the
// triangular solve (one value column per thread) and the readout
// Y = Q~ S_0 + tril(Q~ K^T) W stay on the FMA pipe.
//
// One CTA (256 threads, 8 warps) per SM, persistent over (slot, value head)
// items; it owns all 512 tensor-memory columns:
//   [0, 128) S^T fp32 | [128, 256) S^T head | [256, 384) S^T rest |
//   [384, 448) P1 result | [448, 480) W^T head | [480, 512) W^T rest.
// Warps w and w + 4 share tensor-memory lanes 32 (w % 4) ..: the first four
// warps solve for W, the last four scale the state by g_C, and both halves
// split the column ranges of the loads and stores.
#include "async.cuh"
#include "device.cuh"
#include "internal.h"
#include "pipeline.cuh"
#include "tcgen05.cuh"

namespace stepq {
namespace pf {

constexpr int C = 32;                                  // tokens per chunk
constexpr uint32_t kColS = 0, kColSh = 128, kColSl = 256, kColX = 384, kColWh = 448, kColWl = 480;
constexpr uint32_t kCols = 512;
constexpr uint32_t kIdesc1 = tc::idesc_tf32(128, 64);
constexpr uint32_t kIdesc2 = tc::idesc_tf32(128, 128);

// shared memory (bytes); the MMA operands first, 1024-byte aligned
constexpr int kOffB1h = 0;                             // [K~ ; Q~] head: 64 rows x K 128 (32 KB)
constexpr int kOffB1l = kOffB1h + 32768;               // rest
constexpr int kOffB2h = kOffB1l + 32768;               // K_bar^T head: 128 rows (i) x K 32 (t) (16 KB)
constexpr int kOffB2l = kOffB2h + 16384;
constexpr int kOffKt = kOffB2l + 16384;                // float [C][128] G K
constexpr int kOffKh = kOffKt + C * 128 * 4;           // float [C][128] G^-1 K
constexpr int kOffQt = kOffKh + C * 128 * 4;           // float [C][128] G Q
constexpr int kOffV = kOffQt + C * 128 * 4;            // float [C][128] V
constexpr int kOffG = kOffV + C * 128 * 4;             // float [C][128] cumulative gates
constexpr int kOffW = kOffG + C * 128 * 4;             // float [C][128] W
constexpr int kOffA = kOffW + C * 128 * 4;             // float [C][C] A (strict lower)
constexpr int kOffB = kOffA + C * C * 4;               // float [C][C] Q~ K^T (lower, with diagonal)
constexpr int kOffBeta = kOffB + C * C * 4;            // float [C]
constexpr int kOffBar = kOffBeta + C * 4;              // uint64 mbarrier
constexpr int kOffTmem = kOffBar + 8;                  // u32 tensor-memory base
constexpr int kSmem = kOffTmem + 8;

// Element (row r, k) of a K-major operand stored as core matrices of 8 rows x
// 4 fp32: the matrix (r / 8, k / 4) sits at (r / 8) * sbo + (k / 4) * 128.
__device__ __forceinline__ int core_off(int r, int k, int sbo) {
    return (r >> 3) * sbo + (k >> 2) * 128 + (r & 7) * 16 + (k & 3) * 4;
}

struct Args {
    const float *q, *k, *v, *beta, *gate;
    float *states, *y;
    int B, T, Hk, Hv, gate_per_row, items;
    unsigned int *err;
};

__global__ void __launch_bounds__(kThreads, 1) prefill_kernel(Args a) {
    extern __shared__ __align__(1024) uint8_t smem[];
    uint8_t *B1h = smem + kOffB1h, *B1l = smem + kOffB1l, *B2h = smem + kOffB2h, *B2l = smem + kOffB2l;
    float *Kt = (float *)(smem + kOffKt), *Kh = (float *)(smem + kOffKh), *Qt = (float *)(smem + kOffQt);
    float *V = (float *)(smem + kOffV), *G = (float *)(smem + kOffG), *Wm = (float *)(smem + kOffW);
    float *A = (float *)(smem + kOffA), *Bm = (float *)(smem + kOffB), *bet = (float *)(smem + kOffBeta);
    uint64_t *bar = (uint64_t *)(smem + kOffBar);
    uint32_t *tbase = (uint32_t *)(smem + kOffTmem);
    const int tid = threadIdx.x, w = tid >> 5, l = tid & 31;
    const int quad = w & 3, half = w >> 2;
    const int j = 32 * quad + l;                           // tensor-memory lane = value column
    if (w == 0) {
        tc::tmem_alloc(tbase, kCols);
        tc::tmem_relinquish();
    }
    if (tid == 0) {
        mbar_init(bar, 1);
        mbar_init_fence();
    }
    tc::fence_before();
    __syncthreads();
    tc::fence_after();
    const uint32_t tm = *tbase;                            // lane 0, first column
    const uint32_t tl = tm + ((uint32_t)(32 * quad) << 16);   // this warp's lanes
    uint32_t parity = 0;
    bool alive = true;
    const int grp = a.Hv / a.Hk;
    for (int item = blockIdx.x; alive && item < a.items; item += gridDim.x) {
        const int b = item / a.Hv, h = item - b * a.Hv, hk = h / grp;
        float *Sg = a.states + (size_t)item * kN;
        // S^T into tensor memory: this thread's lane j, the 64 key rows of its half.
        for (int c = 0; c < 2; c++) {
            const int i0 = 64 * half + 32 * c;
            float s[32], hi[32], lo[32];
#pragma unroll
            for (int e = 0; e < 32; e++) {
                s[e] = Sg[(size_t)(i0 + e) * 128 + j];
                tc::split_tf32(s[e], hi[e], lo[e]);
            }
            tc::st32(tl + kColS + i0, s);
            tc::st32(tl + kColSh + i0, hi);
            tc::st32(tl + kColSl + i0, lo);
        }
        tc::wait_st();
        for (int t0 = 0; alive && t0 < a.T; t0 += C) {
            const int n = min(C, a.T - t0);               // tokens in this chunk (ragged tail)
            tc::fence_before();
            __syncthreads();                              // the previous chunk is done with every buffer
            // Chunk operands; missing tokens of the tail are the identity step
            // (gate 1, beta 0, zero k, q, v).
#pragma unroll
            for (int e = tid; e < C * 32; e += kThreads) {
                const int t = e >> 5, c4 = e & 31;
                float4 kq = make_float4(0.f, 0.f, 0.f, 0.f), qq = kq, vv = kq;
                if (t < n) {
                    const size_t tok = (size_t)b * a.T + t0 + t;
                    kq = ((const float4 *)(a.k + (tok * a.Hk + hk) * 128))[c4];
                    qq = ((const float4 *)(a.q + (tok * a.Hk + hk) * 128))[c4];
                    vv = ((const float4 *)(a.v + (tok * a.Hv + h) * 128))[c4];
                }
                ((float4 *)Kt)[e] = kq;                   // raw k until the gates are known
                ((float4 *)Qt)[e] = qq;
                ((float4 *)V)[e] = vv;
            }
            if (tid < C) {
                const size_t tok = (size_t)b * a.T + t0 + tid;
                bet[tid] = tid < n ? a.beta[tok * a.Hv + h] : 0.f;
            }
            // Cumulative gates g_t per key channel: the chunk's 32 gates are loaded
            // at once (independent loads), then multiplied in token order.
            if (tid < 128) {
                float d[C];
#pragma unroll
                for (int t = 0; t < C; t++) {
                    const size_t tok = (size_t)b * a.T + t0 + t;
                    float dv = 1.f;
                    if (t < n) dv = a.gate_per_row ? a.gate[(tok * a.Hv + h) * 128 + tid] : a.gate[tok * a.Hv + h];
                    d[t] = dv;
                }
                float g = 1.f;
#pragma unroll
                for (int t = 0; t < C; t++) {
                    g = fmaxf(g * d[t], 1e-30f);          // keeps K / g finite
                    G[t * 128 + tid] = g;
                }
            }
            __syncthreads();
            // K~ = G K, K^ = K / G, Q~ = G Q (fp32), and the split MMA operands
            // [K~ ; Q~] and K_bar^T with K_bar = K g_C / g.
            for (int e = tid; e < C * 128; e += kThreads) {
                const int t = e >> 7, i = e & 127;
                const float g = G[e], kv = Kt[e];
                const float kt = g * kv, qt = Qt[e] * g, kb = kv * (G[(C - 1) * 128 + i] / g);
                Kt[e] = kt;
                Kh[e] = kv / g;
                Qt[e] = qt;
                float hi, lo;
                tc::split_tf32(kt, hi, lo);
                *(float *)(B1h + core_off(t, i, 4096)) = hi;
                *(float *)(B1l + core_off(t, i, 4096)) = lo;
                tc::split_tf32(qt, hi, lo);
                *(float *)(B1h + core_off(C + t, i, 4096)) = hi;
                *(float *)(B1l + core_off(C + t, i, 4096)) = lo;
                tc::split_tf32(kb, hi, lo);
                *(float *)(B2h + core_off(i, t, 1024)) = hi;
                *(float *)(B2l + core_off(i, t, 1024)) = lo;
            }
            fence_async_smem();                           // operands visible to the tensor cores
            __syncthreads();
            // P1: [K~ S_0 ; Q~ S_0]^T into columns [384, 448), 16 steps of K = 8.
            if (tid == 0) {
                tc::fence_after();
#pragma unroll 1
                for (int s = 0; s < 16; s++) {
                    const uint64_t bh = tc::sdesc(B1h + 256 * s, 128, 4096);
                    const uint64_t bl = tc::sdesc(B1l + 256 * s, 128, 4096);
                    tc::mma_tf32_ts(tm + kColX, tm + kColSh + 8 * s, bh, kIdesc1, s > 0 ? 1u : 0u);
                    tc::mma_tf32_ts(tm + kColX, tm + kColSh + 8 * s, bl, kIdesc1, 1u);
                    tc::mma_tf32_ts(tm + kColX, tm + kColSl + 8 * s, bh, kIdesc1, 1u);
                }
                tc::commit(bar);
            }
            __syncwarp();                                 // warp 0 converged again
            // Meanwhile on the FMA pipe: A = strict lower of diag(beta) K~ K^T,
            // Bm = lower (with diagonal) of Q~ K^T.
            {
                const int t = tid >> 3, s0 = (tid & 7) * 4;
                float ac[4] = {0.f, 0.f, 0.f, 0.f}, bc[4] = {0.f, 0.f, 0.f, 0.f};
                for (int i4 = 0; i4 < 32; i4++) {
                    const float4 kt = ((const float4 *)(Kt + t * 128))[i4];
                    const float4 qt = ((const float4 *)(Qt + t * 128))[i4];
#pragma unroll
                    for (int c = 0; c < 4; c++) {
                        const float4 kh = ((const float4 *)(Kh + (s0 + c) * 128))[i4];
                        ac[c] += kt.x * kh.x + kt.y * kh.y + kt.z * kh.z + kt.w * kh.w;
                        bc[c] += qt.x * kh.x + qt.y * kh.y + qt.z * kh.z + qt.w * kh.w;
                    }
                }
#pragma unroll
                for (int c = 0; c < 4; c++) {
                    const int s = s0 + c;
                    A[t * C + s] = s < t ? bet[t] * ac[c] : 0.f;
                    Bm[t * C + s] = s <= t ? bc[c] : 0.f;
                }
            }
            {
                const bool ok = mbar_wait(bar, parity, pipe::kWaitCycles);
                parity ^= 1u;
                if (__syncthreads_or(!ok)) {              // A, Bm visible as well
                    alive = false;
                    break;
                }
            }
            tc::fence_after();
            if (half == 0) {
                // W = (I + A)^-1 diag(beta) (V - K~ S_0), value column j.
                float x[32], wv[32];
                tc::ld32(tl + kColX, x);
#pragma unroll
                for (int t = 0; t < C; t++) {
                    float acc = bet[t] * (V[t * 128 + j] - x[t]);
#pragma unroll
                    for (int s = 0; s < t; s++) acc -= A[t * C + s] * wv[s];
                    wv[t] = acc;
                }
                float hi[32], lo[32];
#pragma unroll
                for (int t = 0; t < C; t++) {
                    Wm[t * 128 + j] = wv[t];
                    tc::split_tf32(wv[t], hi[t], lo[t]);
                }
                tc::st32(tl + kColWh, hi);
                tc::st32(tl + kColWl, lo);
            } else {
                // S^T <- S^T diag(g_C): key row i scaled by its cumulative gate.
#pragma unroll 1
                for (int c = 0; c < 4; c++) {
                    float s[32];
                    tc::ld32(tl + kColS + 32 * c, s);
#pragma unroll
                    for (int e = 0; e < 32; e++) s[e] *= G[(C - 1) * 128 + 32 * c + e];
                    tc::st32(tl + kColS + 32 * c, s);
                }
            }
            tc::wait_st();
            tc::fence_before();
            __syncthreads();
            // P2: S^T += W^T K_bar, 4 steps of K = 8.
            if (tid == 0) {
                tc::fence_after();
#pragma unroll 1
                for (int s = 0; s < 4; s++) {
                    const uint64_t bh = tc::sdesc(B2h + 256 * s, 128, 1024);
                    const uint64_t bl = tc::sdesc(B2l + 256 * s, 128, 1024);
                    tc::mma_tf32_ts(tm + kColS, tm + kColWh + 8 * s, bh, kIdesc2, 1u);
                    tc::mma_tf32_ts(tm + kColS, tm + kColWh + 8 * s, bl, kIdesc2, 1u);
                    tc::mma_tf32_ts(tm + kColS, tm + kColWl + 8 * s, bh, kIdesc2, 1u);
                }
                tc::commit(bar);
            }
            __syncwarp();                                 // warp 0 converged before tcgen05.ld
            // Meanwhile: Y = Q~ S_0 + Bm W, tokens 16 half .. 16 half + 15 of column j.
            {
                float yo[16];
                tc::ld16(tl + kColX + 32 + 16 * half, yo);
#pragma unroll 4
                for (int u = 0; u < 16; u++) {
                    const int t = 16 * half + u;
                    float acc = yo[u];
                    for (int s = 0; s <= t; s++) acc += Bm[t * C + s] * Wm[s * 128 + j];
                    if (t < n) a.y[(((size_t)b * a.T + t0 + t) * a.Hv + h) * 128 + j] = acc;
                }
            }
            {
                const bool ok = mbar_wait(bar, parity, pipe::kWaitCycles);
                parity ^= 1u;
                if (__syncthreads_or(!ok)) {
                    alive = false;
                    break;
                }
            }
            tc::fence_after();
            // Heads and rests of the new state for the next chunk's P1.
            for (int c = 0; c < 2; c++) {
                const int i0 = 64 * half + 32 * c;
                float s[32], hi[32], lo[32];
                tc::ld32(tl + kColS + i0, s);
#pragma unroll
                for (int e = 0; e < 32; e++) tc::split_tf32(s[e], hi[e], lo[e]);
                tc::st32(tl + kColSh + i0, hi);
                tc::st32(tl + kColSl + i0, lo);
            }
            tc::wait_st();
        }
        if (!alive) break;
        // The boundary state back to global memory.
        for (int c = 0; c < 2; c++) {
            const int i0 = 64 * half + 32 * c;
            float s[32];
            tc::ld32(tl + kColS + i0, s);
#pragma unroll
            for (int e = 0; e < 32; e++) Sg[(size_t)(i0 + e) * 128 + j] = s[e];
        }
    }
    if (!alive && tid == 0) {
        raise_error(a.err, STEPQ_ERR_TIMEOUT);
        mbar_wait(bar, parity ^ 1u, pipe::kWaitCycles);  // the stalled MMAs, once more with a bound
    }
    tc::fence_before();
    __syncthreads();
    if (w == 0) {
        tc::fence_after();
        tc::tmem_dealloc(tm, kCols);
    }
}

}  // namespace pf

stepq_status launch_prefill(const stepq_config *cfg, const float *q, const float *k, const float *v,
                            const float *beta, const float *gate, int B, int T, float *states, float *y,
                            cudaStream_t s) {
    pf::Args a{};
    a.q = q; a.k = k; a.v = v; a.beta = beta; a.gate = gate;
    a.states = states; a.y = y;
    a.B = B; a.T = T;
    a.Hk = cfg->n_key_heads;
    a.Hv = cfg->n_value_heads;
    a.gate_per_row = cfg->gate_kind == STEPQ_GATE_CHANNEL;
    a.items = B * a.Hv;
    a.err = device_error_word();
    if (cudaFuncSetAttribute((const void *)pf::prefill_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             pf::kSmem) != cudaSuccess)
        return STEPQ_ERR_CUDA;
    int dev = 0, sms = 1;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    int grid = sms > 0 ? sms : 1;
    if (grid > a.items) grid = a.items;
    pf::prefill_kernel<<<grid, kThreads, pf::kSmem, s>>>(a);
    return cudaGetLastError() == cudaSuccess ? STEPQ_OK : STEPQ_ERR_CUDA;
}

}  // namespace stepq
