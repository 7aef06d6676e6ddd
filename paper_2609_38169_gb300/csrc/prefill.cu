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
//   Y = Q~ S_0 + Bm W,  Bm = tril(Q~ K^T) (Q~ = G Q, lower triangle with the diagonal),
// and the state after the chunk is S_C = G_C S_0 + K_bar^T W, K_bar = K g_C / g.
//
// Every product runs on the tensor cores (tcgen05, kind::tf32) in split
// precision: an fp32 operand is a TF32 head plus its remainder, and a product
// is head*head + head*rest + rest*head (the rest*rest term is below fp32
// rounding of the accumulation), which keeps fp32 accuracy. The state stays
// in tensor memory as S^T (lane j = value column, column i = key row):
//   P0  [K~ ; Q~] K^T        -> A, Bm      M = 128 (64 used), N = 32, K = 128, A, B in smem
//   P1  S_0^T [K~ ; Q~]^T    -> [K~ S_0 ; Q~ S_0]^T    M = 128, N = 64, K = 128, A in tmem
//   P2  S^T += W^T K_bar                               M = 128, N = 128, K = 32, A in tmem
//   P3  (Q~ S_0)^T += W^T Bm^T  -> Y^T                 M = 128, N = 32, K = 32, A in tmem
// Shared-memory operands are K-major core matrices (8 rows x 16 bytes). The
// FMA pipe keeps the element-wise work, the triangular solve (I + A) W = R
// (one value column per thread) and the scaling of S by g_C.
//
// One CTA (256 threads, 8 warps) per SM, persistent over (slot, value head)
// items; it owns all 512 tensor-memory columns:
//   [0, 128) S^T fp32 | [128, 256) S^T head | [256, 384) S^T rest |
//   [384, 416) (K~ S_0)^T | [416, 448) (Q~ S_0)^T, then Y^T |
//   [448, 480) P0 result, then W^T head | [480, 512) W^T rest.
// Warps w and w + 4 share tensor-memory lanes 32 (w % 4) ..: the first four
// warps solve for W while the last four scale the state by g_C. While P2 and
// P3 run, all warps prepare the next chunk's operands.
#include "async.cuh"
#include "device.cuh"
#include "internal.h"
#include "pipeline.cuh"
#include "tcgen05.cuh"

namespace stepq {
namespace pf {

constexpr int C = 32;                                  // tokens per chunk
constexpr uint32_t kColS = 0, kColSh = 128, kColSl = 256, kColX = 384, kColY = 416, kColP0 = 448,
                   kColWh = 448, kColWl = 480;
constexpr uint32_t kCols = 512;
constexpr uint32_t kIdescP0 = tc::idesc_tf32(128, 32);
constexpr uint32_t kIdescP1 = tc::idesc_tf32(128, 64);
constexpr uint32_t kIdescP2 = tc::idesc_tf32(128, 128);
constexpr uint32_t kIdescP3 = tc::idesc_tf32(128, 32);

// Shared-memory operands: K-major core matrices of 8 rows x 4 fp32 (128 B),
// the core matrices of one row group 144 B apart along K (16 B of padding each,
// so that a warp storing 32 consecutive K elements of one row hits 32 banks),
// row groups kSbo128 / kSbo32 apart for K = 128 / 32.
constexpr int kLbo = 144;
constexpr int kSbo128 = 32 * kLbo;                     // 4608
constexpr int kSbo32 = 8 * kLbo + 16;                  // 1168: 16-byte rows of 8 row groups in distinct banks
// P0 reads 128 rows of A from B1: rows 64..127 fall on B1l and B3 (valid
// memory; their results are unused).
constexpr int kOffB1h = 0;                             // [K~ ; Q~] head: 64 rows x K 128
constexpr int kOffB1l = kOffB1h + 8 * kSbo128;         // rest
constexpr int kOffB3h = kOffB1l + 8 * kSbo128;         // K^ head: 32 rows (s) x K 128
constexpr int kOffB3l = kOffB3h + 4 * kSbo128;
constexpr int kOffB2h = kOffB3l + 4 * kSbo128;         // K_bar^T head: 128 rows (i) x K 32 (t)
constexpr int kOffB2l = kOffB2h + 16 * kSbo32;
constexpr int kOffB4h = kOffB2l + 16 * kSbo32;         // Bm head: 32 rows (t) x K 32 (s)
constexpr int kOffB4l = kOffB4h + 4 * kSbo32;
constexpr int kOffV = kOffB4l + 4 * kSbo32;            // float [C][128] V
constexpr int kOffG = kOffV + C * 128 * 4;             // float [C][128] cumulative gates
constexpr int kOffA = kOffG + C * 128 * 4;             // float [C][C] A^T: row s holds A_ts over t (t > s)
constexpr int kOffBeta = kOffA + C * C * 4;            // float [C]
constexpr int kOffBar = kOffBeta + C * 4;              // uint64 mbarrier
constexpr int kOffTmem = kOffBar + 8;                  // u32 tensor-memory base
constexpr int kSmem = kOffTmem + 8;
static_assert(kOffB1l + 16 * kSbo128 <= kSmem, "P0's unused A rows must stay inside shared memory");

// Byte offset of element (row r, k) of a K-major operand with row groups `sbo` apart.
__device__ __forceinline__ int core_off(int r, int k, int sbo) {
    return (r >> 3) * sbo + (k >> 2) * kLbo + (r & 7) * 16 + (k & 3) * 4;
}

__device__ __forceinline__ void put_split(uint8_t *hi_base, uint8_t *lo_base, int off, float x) {
    float hi, lo;
    tc::split_tf32(x, hi, lo);
    *(float *)(hi_base + off) = hi;
    *(float *)(lo_base + off) = lo;
}
// Four consecutive K elements of one row (off 16-byte aligned).
__device__ __forceinline__ void put_split4(uint8_t *hi_base, uint8_t *lo_base, int off, float4 x) {
    float4 hi, lo;
    tc::split_tf32(x.x, hi.x, lo.x);
    tc::split_tf32(x.y, hi.y, lo.y);
    tc::split_tf32(x.z, hi.z, lo.z);
    tc::split_tf32(x.w, hi.w, lo.w);
    *(float4 *)(hi_base + off) = hi;
    *(float4 *)(lo_base + off) = lo;
}
__device__ __forceinline__ float4 mul4(float4 a, float4 b) {
    return make_float4(a.x * b.x, a.y * b.y, a.z * b.z, a.w * b.w);
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
    uint8_t *B3h = smem + kOffB3h, *B3l = smem + kOffB3l, *B4h = smem + kOffB4h, *B4l = smem + kOffB4l;
    float *V = (float *)(smem + kOffV), *G = (float *)(smem + kOffG), *A = (float *)(smem + kOffA);
    float *bet = (float *)(smem + kOffBeta);
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
    // a CTA-wide bounded wait on the commit barrier; false if any thread gave up
    const auto wait_mma = [&]() {
        const bool ok = mbar_wait(bar, parity, pipe::kWaitCycles);
        parity ^= 1u;
        const bool stalled = __syncthreads_or(!ok);
        tc::fence_after();
        return !stalled;
    };
    // This thread's share of a chunk's operands, loaded one chunk ahead (their
    // global-memory latency overlaps the previous chunk's tensor-core work):
    // key channels 4 cq .. 4 cq + 3 at tokens 4 tq .. 4 tq + 3 of k, q, v (one
    // 16-byte load each); threads 0..127 the chunk's gates of channel ci,
    // threads 128..159 one beta each. Missing tokens of a ragged tail are the
    // identity step (gate 1, beta 0, zero k, q, v).
    const int ci = tid & 127, cq = tid & 31, tq = tid >> 5;
    float4 kv[4], qv[4], vv[4];
    float dg[C], bt = 0.f;
    const auto fetch = [&](int it, int c0) {
        const int fb = it / a.Hv, fh = it - fb * a.Hv, fhk = fh / grp, fn = min(C, a.T - c0);
#pragma unroll
        for (int m = 0; m < 4; m++) {
            const int t = 4 * tq + m;
            kv[m] = qv[m] = vv[m] = make_float4(0.f, 0.f, 0.f, 0.f);
            if (t < fn) {
                const size_t tok = (size_t)fb * a.T + c0 + t;
                kv[m] = *(const float4 *)&a.k[(tok * a.Hk + fhk) * 128 + 4 * cq];
                qv[m] = *(const float4 *)&a.q[(tok * a.Hk + fhk) * 128 + 4 * cq];
                vv[m] = *(const float4 *)&a.v[(tok * a.Hv + fh) * 128 + 4 * cq];
            }
        }
        if (tid < 128) {
#pragma unroll
            for (int t = 0; t < C; t++) {
                const size_t tok = (size_t)fb * a.T + c0 + t;
                float dv = 1.f;
                if (t < fn) dv = a.gate_per_row ? a.gate[(tok * a.Hv + fh) * 128 + ci] : a.gate[tok * a.Hv + fh];
                dg[t] = dv;
            }
        } else if (tid < 128 + C) {
            const int t = tid - 128;
            bt = t < fn ? a.beta[((size_t)fb * a.T + c0 + t) * a.Hv + fh] : 0.f;
        }
    };
    // One chunk's cumulative gates g_t per key channel (multiplied in token
    // order), beta, V and the split operands [K~ ; Q~] and K^, from the fetched
    // registers, four consecutive K elements per store. K_bar^T, P2's operand,
    // stays in kb until put_kbar (the previous chunk's P2 may still read it).
    float kb[4][4];                                        // K_bar^T: [channel][token]
    const auto prep = [&]() {
        if (tid < 128) {
            float g = 1.f;
#pragma unroll
            for (int t = 0; t < C; t++) {
                g = fmaxf(g * dg[t], 1e-30f);             // keeps K / g finite
                G[t * 128 + tid] = g;
            }
        } else if (tid < 128 + C) {
            bet[tid - 128] = bt;
        }
        __syncthreads();
        const int c4 = 4 * cq;
        const float4 gC = *(const float4 *)&G[(C - 1) * 128 + c4];
#pragma unroll
        for (int m = 0; m < 4; m++) {
            const int t = 4 * tq + m;
            const float4 g = *(const float4 *)&G[t * 128 + c4];
            const float4 rg = make_float4(__fdividef(1.0f, g.x), __fdividef(1.0f, g.y),   // within 2 ulp
                                          __fdividef(1.0f, g.z), __fdividef(1.0f, g.w));
            *(float4 *)&V[t * 128 + c4] = vv[m];
            put_split4(B1h, B1l, core_off(t, c4, kSbo128), mul4(g, kv[m]));        // K~
            put_split4(B1h, B1l, core_off(C + t, c4, kSbo128), mul4(g, qv[m]));    // Q~
            put_split4(B3h, B3l, core_off(t, c4, kSbo128), mul4(kv[m], rg));       // K^
            kb[0][m] = kv[m].x * (gC.x * rg.x);
            kb[1][m] = kv[m].y * (gC.y * rg.y);
            kb[2][m] = kv[m].z * (gC.z * rg.z);
            kb[3][m] = kv[m].w * (gC.w * rg.w);
        }
    };
    const auto put_kbar = [&]() {
#pragma unroll
        for (int e = 0; e < 4; e++)
            put_split4(B2h, B2l, core_off(4 * cq + e, 4 * tq, kSbo32),
                       make_float4(kb[e][0], kb[e][1], kb[e][2], kb[e][3]));
    };
    // This CTA's chunks in order: (item, first token); fi, fc is the chunk
    // whose inputs the registers hold.
    int fi = blockIdx.x, fc = 0;
    const auto advance = [&]() {
        fc += C;
        if (fc >= a.T) {
            fi += gridDim.x;
            fc = 0;
        }
    };
    // Prologue: the first chunk prepared, the second fetched.
    if (fi < a.items) {
        fetch(fi, fc);
        prep();
        put_kbar();
        advance();
        if (fi < a.items) fetch(fi, fc);
    }
    for (int item = blockIdx.x; alive && item < a.items; item += gridDim.x) {
        const int b = item / a.Hv, h = item - b * a.Hv;
        float *Sg = a.states + (size_t)item * kN;
        // S^T into tensor memory: this thread's lane j, the 64 key rows of its half.
        for (int c = 0; c < 2; c++) {
            const int i0 = 64 * half + 32 * c;
            float sv[32], hi[32], lo[32];
#pragma unroll
            for (int e = 0; e < 32; e++) {
                sv[e] = Sg[(size_t)(i0 + e) * 128 + j];
                tc::split_tf32(sv[e], hi[e], lo[e]);
            }
            tc::st32(tl + kColS + i0, sv);
            tc::st32(tl + kColSh + i0, hi);
            tc::st32(tl + kColSl + i0, lo);
        }
        tc::wait_st();
        for (int t0 = 0; alive && t0 < a.T; t0 += C) {
            const int n = min(C, a.T - t0);               // tokens in this chunk (ragged tail)
            fence_async_smem();                           // this chunk's operands visible to the tensor cores
            tc::fence_before();
            __syncthreads();                              // the previous chunk is done with every buffer
            // P0: [K~ ; Q~] K^T into columns [448, 480); P1: [K~ S_0 ; Q~ S_0]^T into [384, 448).
            if (tid == 0) {
                tc::fence_after();
#pragma unroll 1
                for (int s = 0; s < 16; s++) {
                    const uint64_t ah = tc::sdesc(B1h + 2 * kLbo * s, kLbo, kSbo128), al = tc::sdesc(B1l + 2 * kLbo * s, kLbo, kSbo128);
                    const uint64_t kh = tc::sdesc(B3h + 2 * kLbo * s, kLbo, kSbo128), kl = tc::sdesc(B3l + 2 * kLbo * s, kLbo, kSbo128);
                    const uint32_t acc = s > 0 ? 1u : 0u;
                    tc::mma_tf32_ss(tm + kColP0, ah, kh, kIdescP0, acc);
                    tc::mma_tf32_ss(tm + kColP0, ah, kl, kIdescP0, 1u);
                    tc::mma_tf32_ss(tm + kColP0, al, kh, kIdescP0, 1u);
                    tc::mma_tf32_ts(tm + kColX, tm + kColSh + 8 * s, ah, kIdescP1, acc);
                    tc::mma_tf32_ts(tm + kColX, tm + kColSh + 8 * s, al, kIdescP1, 1u);
                    tc::mma_tf32_ts(tm + kColX, tm + kColSl + 8 * s, ah, kIdescP1, 1u);
                }
                tc::commit(bar);
            }
            __syncwarp();
            if (!wait_mma()) {
                alive = false;
                break;
            }
            // A = strict lower of diag(beta) K~ K^T (row t = lane t), stored
            // transposed (a warp's store is one row of A^T: no bank conflicts), and
            // Bm = lower (with diagonal) of Q~ K^T (row t = lane 32 + t), Bm split
            // as an operand.
            if (w < 2) {
                float d[32];
                tc::ld32(tl + kColP0, d);
                if (w == 0) {
                    const float bt = bet[l];
#pragma unroll
                    for (int s = 0; s < C; s++) A[s * C + l] = s < l ? bt * d[s] : 0.f;
                } else {
#pragma unroll
                    for (int s = 0; s < C; s++) put_split(B4h, B4l, core_off(l, s, kSbo32), s <= l ? d[s] : 0.f);
                    fence_async_smem();
                }
            }
            __syncthreads();                              // A visible; P0's columns free for W
            if (half == 0) {
                // W = (I + A)^-1 diag(beta) (V - K~ S_0), value column j, by forward
                // substitution in column order: once w_s is final it is taken out
                // of every later row (independent updates, so the dependent chain
                // is one fma per token).
                float wv[32];
                tc::ld32(tl + kColX, wv);
#pragma unroll
                for (int t = 0; t < C; t++) wv[t] = bet[t] * (V[t * 128 + j] - wv[t]);
#pragma unroll
                for (int s = 0; s < C - 1; s++) {
                    const float ws = wv[s];
#pragma unroll
                    for (int t4 = (s + 1) / 4; t4 < C / 4; t4++) {    // row s of A^T, four at a time
                        const float4 a4 = ((const float4 *)(A + s * C))[t4];
                        const float av[4] = {a4.x, a4.y, a4.z, a4.w};
#pragma unroll
                        for (int e = 0; e < 4; e++)
                            if (4 * t4 + e > s) wv[4 * t4 + e] = fmaf(-av[e], ws, wv[4 * t4 + e]);
                    }
                }
                float hi[32], lo[32];
#pragma unroll
                for (int t = 0; t < C; t++) tc::split_tf32(wv[t], hi[t], lo[t]);
                tc::st32(tl + kColWh, hi);
                tc::st32(tl + kColWl, lo);
            } else {
                // S^T <- S^T diag(g_C): key row i scaled by its cumulative gate.
#pragma unroll 1
                for (int c = 0; c < 4; c++) {
                    float sv[32];
                    tc::ld32(tl + kColS + 32 * c, sv);
#pragma unroll
                    for (int e = 0; e < 32; e++) sv[e] *= G[(C - 1) * 128 + 32 * c + e];
                    tc::st32(tl + kColS + 32 * c, sv);
                }
            }
            tc::wait_st();
            tc::fence_before();
            __syncthreads();
            // P2: S^T += W^T K_bar; P3: Y^T = (Q~ S_0)^T + W^T Bm^T.
            if (tid == 0) {
                tc::fence_after();
#pragma unroll 1
                for (int s = 0; s < 4; s++) {
                    const uint64_t bh = tc::sdesc(B2h + 2 * kLbo * s, kLbo, kSbo32), bl = tc::sdesc(B2l + 2 * kLbo * s, kLbo, kSbo32);
                    const uint64_t mh = tc::sdesc(B4h + 2 * kLbo * s, kLbo, kSbo32), ml = tc::sdesc(B4l + 2 * kLbo * s, kLbo, kSbo32);
                    tc::mma_tf32_ts(tm + kColS, tm + kColWh + 8 * s, bh, kIdescP2, 1u);
                    tc::mma_tf32_ts(tm + kColS, tm + kColWh + 8 * s, bl, kIdescP2, 1u);
                    tc::mma_tf32_ts(tm + kColS, tm + kColWl + 8 * s, bh, kIdescP2, 1u);
                    tc::mma_tf32_ts(tm + kColY, tm + kColWh + 8 * s, mh, kIdescP3, 1u);
                    tc::mma_tf32_ts(tm + kColY, tm + kColWh + 8 * s, ml, kIdescP3, 1u);
                    tc::mma_tf32_ts(tm + kColY, tm + kColWl + 8 * s, mh, kIdescP3, 1u);
                }
                tc::commit(bar);
            }
            __syncwarp();
            // While P2 and P3 run: the next chunk's operands (this item's next
            // chunk or the next item's first), and the inputs of the one after.
            const bool more = fi < a.items;
            if (more) {
                prep();
                advance();
                if (fi < a.items) fetch(fi, fc);
            }
            if (!wait_mma()) {
                alive = false;
                break;
            }
            if (more) put_kbar();                         // P2 is done with K_bar^T
            // Outputs: tokens 16 half .. 16 half + 15 of column j.
            {
                float yv[16];
                tc::ld16(tl + kColY + 16 * half, yv);
#pragma unroll
                for (int e = 0; e < 16; e++) {
                    const int t = 16 * half + e;
                    if (t < n) a.y[(((size_t)b * a.T + t0 + t) * a.Hv + h) * 128 + j] = yv[e];
                }
            }
            // Heads and rests of the new state for the next chunk's P1.
            for (int c = 0; c < 2; c++) {
                const int i0 = 64 * half + 32 * c;
                float sv[32], hi[32], lo[32];
                tc::ld32(tl + kColS + i0, sv);
#pragma unroll
                for (int e = 0; e < 32; e++) tc::split_tf32(sv[e], hi[e], lo[e]);
                tc::st32(tl + kColSh + i0, hi);
                tc::st32(tl + kColSl + i0, lo);
            }
            tc::wait_st();
        }
        if (!alive) break;
        // The boundary state back to global memory.
        for (int c = 0; c < 2; c++) {
            const int i0 = 64 * half + 32 * c;
            float sv[32];
            tc::ld32(tl + kColS + i0, sv);
#pragma unroll
            for (int e = 0; e < 32; e++) Sg[(size_t)(i0 + e) * 128 + j] = sv[e];
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
