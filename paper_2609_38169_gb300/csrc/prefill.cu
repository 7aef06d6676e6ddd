// Chunked FP32-state prefill: the gated Delta rule (Eq. delta_update) over T
// tokens, 32 tokens at a time, producing the boundary state that
// stepq_quantize_pool packs (the prefill side of App. C.3 / App. F: the
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
// and the state after the chunk is S_C = G_C S_0 + (K (g_C/g))^T W.
// These are five small dense products and one triangular solve per chunk;
// this build evaluates them in fp32 on the FMA pipe (the reference the
// parity tests use is the oracle's token-by-token recurrence).
//
// One CTA (256 threads) per (slot, value head) item, persistent over items;
// the state, the chunk's operands and the two 32 x 32 matrices live in
// shared memory (about 170 KB, one CTA per SM).
#include "device.cuh"
#include "internal.h"

namespace stepq {
namespace pf {

constexpr int C = 32;                                  // tokens per chunk
constexpr int kOffS = 0;                               // float [128][128] state
constexpr int kOffKt = kOffS + kN * 4;                 // float [C][128] G K
constexpr int kOffKh = kOffKt + C * 128 * 4;           // float [C][128] G^-1 K
constexpr int kOffKb = kOffKh + C * 128 * 4;           // float [C][128] K g_C / g
constexpr int kOffQt = kOffKb + C * 128 * 4;           // float [C][128] G Q
constexpr int kOffV = kOffQt + C * 128 * 4;            // float [C][128] V, then R, then W
constexpr int kOffA = kOffV + C * 128 * 4;             // float [C][C] A (strict lower)
constexpr int kOffB = kOffA + C * C * 4;               // float [C][C] Q~ K^T (lower, with diagonal)
constexpr int kOffG = kOffB + C * C * 4;               // float [C][128] cumulative gates
constexpr int kOffBeta = kOffG + C * 128 * 4;          // float [C]
constexpr int kSmem = kOffBeta + C * 4;

struct Args {
    const float *q, *k, *v, *beta, *gate;
    float *states, *y;
    int B, T, Hk, Hv, gate_per_row, items;
};

__global__ void __launch_bounds__(kThreads, 1) prefill_kernel(Args a) {
    extern __shared__ __align__(16) uint8_t smem[];
    float *S = (float *)(smem + kOffS), *Kt = (float *)(smem + kOffKt), *Kh = (float *)(smem + kOffKh);
    float *Kb = (float *)(smem + kOffKb), *Qt = (float *)(smem + kOffQt), *V = (float *)(smem + kOffV);
    float *A = (float *)(smem + kOffA), *Bm = (float *)(smem + kOffB), *G = (float *)(smem + kOffG);
    float *bet = (float *)(smem + kOffBeta);
    const int tid = threadIdx.x, w = tid >> 5, l = tid & 31;
    const int grp = a.Hv / a.Hk;
    for (int item = blockIdx.x; item < a.items; item += gridDim.x) {
        const int b = item / a.Hv, h = item - b * a.Hv, hk = h / grp;
        float *Sg = a.states + (size_t)item * kN;
        for (int e = tid; e < kN / 4; e += kThreads) ((float4 *)S)[e] = ((const float4 *)Sg)[e];
        for (int t0 = 0; t0 < a.T; t0 += C) {
            const int n = min(C, a.T - t0);               // tokens in this chunk (ragged tail)
            __syncthreads();                              // previous chunk done with the buffers
            // Chunk operands; missing tokens of the tail are the identity step
            // (gate 1, beta 0, zero k, q, v).
            for (int e = tid; e < C * 32; e += kThreads) {
                const int t = e >> 5, c4 = e & 31;
                float4 kq = make_float4(0.f, 0.f, 0.f, 0.f), qq = kq, vv = kq;
                if (t < n) {
                    const size_t tok = (size_t)b * a.T + t0 + t;
                    kq = ((const float4 *)(a.k + (tok * a.Hk + hk) * 128))[c4];
                    qq = ((const float4 *)(a.q + (tok * a.Hk + hk) * 128))[c4];
                    vv = ((const float4 *)(a.v + (tok * a.Hv + h) * 128))[c4];
                }
                ((float4 *)Kb)[e] = kq;                   // raw k until the gates are known
                ((float4 *)Qt)[e] = qq;
                ((float4 *)V)[e] = vv;
            }
            if (tid < C) {
                const size_t tok = (size_t)b * a.T + t0 + tid;
                bet[tid] = tid < n ? a.beta[tok * a.Hv + h] : 0.f;
            }
            // Cumulative gates g_t per key channel (a sequential product over the chunk).
            if (tid < 128) {
                float g = 1.f;
                for (int t = 0; t < C; t++) {
                    float d = 1.f;
                    if (t < n) {
                        const size_t tok = (size_t)b * a.T + t0 + t;
                        d = a.gate_per_row ? a.gate[(tok * a.Hv + h) * 128 + tid] : a.gate[tok * a.Hv + h];
                    }
                    g = fmaxf(g * d, 1e-30f);             // keeps K / g finite
                    G[t * 128 + tid] = g;
                }
            }
            __syncthreads();
            // K~ = G K, K^ = K / G, K_bar = K g_C / g, Q~ = G Q.
            for (int e = tid; e < C * 128; e += kThreads) {
                const int i = e & 127;
                const float g = G[e], kv = Kb[e];
                Kt[e] = g * kv;
                Kh[e] = kv / g;
                Kb[e] = kv * (G[(C - 1) * 128 + i] / g);
                Qt[e] = Qt[e] * g;
            }
            __syncthreads();
            // A = strict lower of diag(beta) K~ K^T, Bm = lower (with diagonal) of Q~ K^T.
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
            // R = diag(beta) (V - K~ S_0) and the state part of the output Q~ S_0:
            // thread = tokens 4tg..4tg+3 x columns 4cg..4cg+3.
            const int tg = tid >> 5, cg = tid & 31;
            float r[4][4], yo[4][4];
#pragma unroll
            for (int u = 0; u < 4; u++)
#pragma unroll
                for (int c = 0; c < 4; c++) r[u][c] = yo[u][c] = 0.f;
            for (int i = 0; i < 128; i++) {
                const float4 sv = ((const float4 *)(S + i * 128))[cg];
#pragma unroll
                for (int u = 0; u < 4; u++) {
                    const float kt = Kt[(4 * tg + u) * 128 + i], qt = Qt[(4 * tg + u) * 128 + i];
                    r[u][0] += kt * sv.x; r[u][1] += kt * sv.y; r[u][2] += kt * sv.z; r[u][3] += kt * sv.w;
                    yo[u][0] += qt * sv.x; yo[u][1] += qt * sv.y; yo[u][2] += qt * sv.z; yo[u][3] += qt * sv.w;
                }
            }
            __syncthreads();                              // A, Bm complete; V still unread
#pragma unroll
            for (int u = 0; u < 4; u++) {
                const int t = 4 * tg + u;
                float4 vv = ((float4 *)(V + t * 128))[cg];
                vv.x = bet[t] * (vv.x - r[u][0]);
                vv.y = bet[t] * (vv.y - r[u][1]);
                vv.z = bet[t] * (vv.z - r[u][2]);
                vv.w = bet[t] * (vv.w - r[u][3]);
                ((float4 *)(V + t * 128))[cg] = vv;       // R
            }
            __syncthreads();
            // W = (I + A)^-1 R by forward substitution, one column per thread.
            if (tid < 128) {
                float wcol[C];
#pragma unroll
                for (int t = 0; t < C; t++) {
                    float acc = V[t * 128 + tid];
#pragma unroll
                    for (int s = 0; s < t; s++) acc -= A[t * C + s] * wcol[s];
                    wcol[t] = acc;
                }
#pragma unroll
                for (int t = 0; t < C; t++) V[t * 128 + tid] = wcol[t];   // W
            }
            __syncthreads();
            // Y = Q~ S_0 + Bm W for the chunk's tokens.
            {
#pragma unroll 4
                for (int s = 0; s < C; s++) {
                    const float4 wv = ((const float4 *)(V + s * 128))[cg];
#pragma unroll
                    for (int u = 0; u < 4; u++) {
                        const float bm = Bm[(4 * tg + u) * C + s];
                        yo[u][0] += bm * wv.x; yo[u][1] += bm * wv.y; yo[u][2] += bm * wv.z; yo[u][3] += bm * wv.w;
                    }
                }
#pragma unroll
                for (int u = 0; u < 4; u++) {
                    const int t = 4 * tg + u;
                    if (t < n) {
                        const size_t tok = (size_t)b * a.T + t0 + t;
                        ((float4 *)(a.y + (tok * a.Hv + h) * 128))[cg] =
                            make_float4(yo[u][0], yo[u][1], yo[u][2], yo[u][3]);
                    }
                }
            }
            // S = G_C S_0 + K_bar^T W: thread = rows 16w..16w+15 x columns 4l..4l+3.
            {
                float acc[16][4];
#pragma unroll
                for (int rr = 0; rr < 16; rr++)
#pragma unroll
                    for (int c = 0; c < 4; c++) acc[rr][c] = 0.f;
                for (int t = 0; t < C; t++) {
                    const float4 wv = ((const float4 *)(V + t * 128))[l];
#pragma unroll
                    for (int q4 = 0; q4 < 4; q4++) {
                        const float4 kb = ((const float4 *)(Kb + t * 128 + 16 * w))[q4];
                        const float kk[4] = {kb.x, kb.y, kb.z, kb.w};
#pragma unroll
                        for (int e = 0; e < 4; e++) {
                            acc[4 * q4 + e][0] += kk[e] * wv.x;
                            acc[4 * q4 + e][1] += kk[e] * wv.y;
                            acc[4 * q4 + e][2] += kk[e] * wv.z;
                            acc[4 * q4 + e][3] += kk[e] * wv.w;
                        }
                    }
                }
#pragma unroll
                for (int rr = 0; rr < 16; rr++) {
                    const int i = 16 * w + rr;
                    const float gC = G[(C - 1) * 128 + i];
                    float4 sv = ((float4 *)(S + i * 128))[l];
                    sv.x = fmaf(gC, sv.x, acc[rr][0]);
                    sv.y = fmaf(gC, sv.y, acc[rr][1]);
                    sv.z = fmaf(gC, sv.z, acc[rr][2]);
                    sv.w = fmaf(gC, sv.w, acc[rr][3]);
                    ((float4 *)(S + i * 128))[l] = sv;
                }
            }
        }
        __syncthreads();
        for (int e = tid; e < kN / 4; e += kThreads) ((float4 *)Sg)[e] = ((const float4 *)S)[e];
        __syncthreads();
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
