// Row-unit (KDA) pool pack/unpack and the calibration distortion kernel
// (sm_103a), and the dispatch of the decode step: head units (GDN) run the
// pipelined kernel of heads.cu, row units the one of rows.cu.
//
// One 256-thread CTA owns one (slot, value head) page: it stages the head
// segment in shared memory with 128-bit loads, holds the tile in registers,
// fits the dual-axis scales and writes the packed segment (App. C.3 steps 4-6).
//
// Numerical contract (shared with the CPU oracle, which restates it in fp64):
// the tile X is fp32; r_i = fp16(clamp(sqrt(m_i) * w_i^(-1/2), 2^-14, 65504));
// rho_i = fp32(1/(r_i zs_i)); every code decision is the nearest integer to the
// exact product fp32(X rho_i) gamma_j with gamma_j = fp32(1/c_j) (rne_prod);
// c is fitted from the clip-free start
// max_i fp32(fp32(|X_ij| rho_i) / qmax_i) by `fit_iters` fixed-code
// least-squares updates.
#include <atomic>
#include <cstdio>

#include "device.cuh"
#include "internal.h"
#include "tile.cuh"

namespace stepq {

// ---------------------------------------------------------------- smem layout
constexpr int kPageBytes = (int)kMaxHeadBytes;             // 33,280
constexpr int kOffRed = kPageBytes;                          // float [2][8][128]
constexpr int kOffCol = kOffRed + 2 * 8 * 128 * 4;           // float [6][128]
constexpr int kOffRowF = kOffCol + 6 * 128 * 4;              // float [5][128]: q k gate w2 wis
constexpr int kOffRowI = kOffRowF + 5 * 128 * 4;             // int [2][128]: bits, offset
constexpr int kSmemBytes = kOffRowI + 2 * 128 * 4;

struct TileSmem {
    uint8_t *page;
    float *red, *col, *qv, *kv, *gv, *w2, *wis;
    int *rbits, *roff;
    __device__ __forceinline__ explicit TileSmem(uint8_t *s) {
        page = s;
        red = (float *)(s + kOffRed);
        col = (float *)(s + kOffCol);
        float *rf = (float *)(s + kOffRowF);
        qv = rf;
        kv = rf + 128;
        gv = rf + 256;
        w2 = rf + 384;
        wis = rf + 512;
        int *ri = (int *)(s + kOffRowI);
        rbits = ri;
        roff = ri + 128;
    }
};

__device__ __forceinline__ int qmax_of(int b) { return (1 << (b - 1)) - 1; }

// Per-thread results of the row-factor fit for its 4 rows.
struct RowFit {
    float rr[4], rho[4], zsv[4];
    int qm[4], bits[4];
};

// Key-Row-Aware Dual-axis Fitting of the register tile x (Sec. 4.3, App. C.1).
// msum[t]: sum_j |X_ij| of the thread's rows; row widths come from S.rbits.
// On return S.col[0..128) holds the stored (FP16-rounded) column factors and
// S.col[128..256) their reciprocals; with write_scales the FP16 r and c are
// written into the staged page. Requires every thread to be done reading the
// old page.
__device__ __forceinline__ void fit_scales(const Lane &L, const TileSmem &S, const float (&x)[4][16],
                                           const float (&msum)[4], int unit_rows,
                                           int write_scales, int fit_iters, RowFit &f) {
    uint16_t *page_r = (uint16_t *)S.page;
    uint16_t *page_c = (uint16_t *)(S.page + 256);
    float *colC = S.col;           // current column iterate
    float *colG = S.col + 128;     // its reciprocal
    float *colND = S.col + 256;    // [2][128] numerator / denominator
    float mu[4];                   // fp32(1 / qmax_i)
    // Row factors r_i = m_i^(1/2) w_i^(-1/2).
#pragma unroll
    for (int t = 0; t < 4; t++) {
        const int i = L.row(t);
        f.bits[t] = S.rbits[i];
        if (f.bits[t] == kPivot) {
            f.rr[t] = f.rho[t] = mu[t] = f.zsv[t] = 0.f;
            f.qm[t] = 0;
            if (write_scales && L.cg == 0) page_r[i] = 0;
            continue;
        }
        const float m = msum[t] * (1.0f / 128.0f);
        const float rf = __half2float(__float2half_rn(
            fminf(fmaxf(__fmul_rn(sqrtf(m), S.wis[i]), kF16Min), kF16Max)));
        const float zs = unit_rows ? (float)(1 << (8 - f.bits[t])) : 1.0f;
        f.qm[t] = qmax_of(f.bits[t]);
        f.rr[t] = rf;
        f.zsv[t] = zs;
        f.rho[t] = __frcp_rn(rf * zs);
        mu[t] = __frcp_rn((float)f.qm[t]);
        if (write_scales && L.cg == 0) page_r[i] = f16_bits(rf);
    }
    // Clip-free column start: c0_j = max_i |X_ij| / (r_i zs_i qmax_i), as
    // max_i fp32(fp32(|X_ij| rho_i) mu_i).
    {
        float acc[1][16];
#pragma unroll
        for (int j = 0; j < 16; j++) acc[0][j] = 0.f;
#pragma unroll
        for (int t = 0; t < 4; t++)
#pragma unroll
            for (int j = 0; j < 16; j++)
                acc[0][j] = fmaxf(acc[0][j], __fmul_rn(__fmul_rn(fabsf(x[t][j]), f.rho[t]), mu[t]));
        column_reduce<1, true>(L, acc, S.red, colC);
        if (L.tid < 128) {
            const float c = fminf(fmaxf(colC[L.tid], kF16Min), kF16Max);
            colC[L.tid] = c;
            colG[L.tid] = __frcp_rn(c);
        }
        __syncthreads();
    }
    // Fixed-code least-squares updates (App. C.1) over the non-pivot rows.
    for (int it = 0; it < fit_iters; it++) {
        float g[16];
#pragma unroll
        for (int j = 0; j < 16; j++) g[j] = colG[L.col0() + j];
        float acc[2][16];
#pragma unroll
        for (int j = 0; j < 16; j++) acc[0][j] = acc[1][j] = 0.f;
#pragma unroll
        for (int t = 0; t < 4; t++) {
            if (f.bits[t] == kPivot) continue;
            const float w2 = S.w2[L.row(t)], rz = f.rr[t] * f.zsv[t], lim = (float)f.qm[t];
#pragma unroll
            for (int j = 0; j < 16; j++) {
                const float qv = fminf(fmaxf(rne_prod(__fmul_rn(x[t][j], f.rho[t]), g[j]), -lim), lim);
                const float v = rz * qv;                      // v_ij = r_i z_ij
                acc[0][j] += w2 * (v * x[t][j]);
                acc[1][j] += w2 * (v * v);
            }
        }
        column_reduce<2, false>(L, acc, S.red, colND);
        if (L.tid < 128) {
            const float num = colND[L.tid], den = colND[128 + L.tid];
            float c = colC[L.tid];
            if (den > 0.f) c = fminf(fmaxf(__fdiv_rn(num, den), kF16Min), kF16Max);
            colC[L.tid] = c;
            colG[L.tid] = __frcp_rn(c);
        }
        __syncthreads();
    }
    // Storage precision of c.
    if (L.tid < 128) {
        const float cf = __half2float(__float2half_rn(colC[L.tid]));
        colC[L.tid] = cf;
        colG[L.tid] = __frcp_rn(cf);
        if (write_scales) page_c[L.tid] = f16_bits(cf);
    }
    __syncthreads();
}

// Final codes with the stored scales, packed into the staged page (App. C.3 step 6).
__device__ __forceinline__ void pack_codes(const Lane &L, const TileSmem &S, const float (&x)[4][16],
                                           const RowFit &f) {
    float g[16];
#pragma unroll
    for (int j = 0; j < 16; j++) g[j] = S.col[128 + L.col0() + j];
#pragma unroll
    for (int t = 0; t < 4; t++) {
        const int i = L.row(t);
        uint8_t *row = S.page + S.roff[i];
        if (f.bits[t] == kPivot) {
            store_f16_row16(row, L.cg, x[t]);
            continue;
        }
        const float lim = (float)f.qm[t];
        int q[16];
#pragma unroll
        for (int j = 0; j < 16; j++)
            q[j] = (int)fminf(fmaxf(rne_prod(__fmul_rn(x[t][j], f.rho[t]), g[j]), -lim), lim);
        store_codes16(row, f.bits[t], L.cg, q);
    }
    __syncthreads();
}

__device__ __forceinline__ void fit_and_pack(const Lane &L, const TileSmem &S, const float (&x)[4][16],
                                             const float (&msum)[4], int unit_rows,
                                             int has_scales, int fit_iters) {
    RowFit f;
    fit_scales(L, S, x, msum, unit_rows, has_scales, fit_iters, f);
    pack_codes(L, S, x, f);
}

// Per-row metadata of head h into shared memory (threads 0..127).
__device__ __forceinline__ void load_row_meta(const Lane &L, const TileSmem &S,
                                              const LayerTables &tab, int h) {
    if (L.tid < 128) {
        S.rbits[L.tid] = tab.row_bits[h * 128 + L.tid];
        S.roff[L.tid] = (int)tab.row_off[h * 128 + L.tid];
        S.w2[L.tid] = tab.w2[h * 128 + L.tid];
        S.wis[L.tid] = tab.wis[h * 128 + L.tid];
    }
}

__device__ __forceinline__ void copy16(uint4 *dst, const uint4 *src, int n16, int tid) {
    for (int e = tid; e < n16; e += kThreads) dst[e] = src[e];
}

// ---------------------------------------------------------- quantize / dequantize
struct PoolArgs {
    uint8_t *pool;
    uint64_t stride;
    int pool_slots;
    const int32_t *slots;
    LayerTables tab;
    Shape sh;
    float *states;            // [B][..][Hv][128][128]
    size_t state_stride_b;    // floats between consecutive batch entries
    unsigned int *err;
};

__global__ void __launch_bounds__(kThreads, 2) quantize_kernel(PoolArgs a) {
    extern __shared__ __align__(16) uint8_t smem[];
    const Lane L;
    const TileSmem S(smem);
    const int Hv = a.sh.Hv;
    const int b = blockIdx.x / Hv, h = blockIdx.x - b * Hv;
    const int slot = a.slots[b];
    if (slot < 0 || slot >= a.pool_slots) {
        if (L.tid == 0) raise_error(a.err, STEPQ_ERR_SLOT_RANGE);
        return;
    }
    load_row_meta(L, S, a.tab, h);
    const float *X = a.states + (size_t)b * a.state_stride_b + (size_t)h * kN;
    float x[4][16], msum[4];
#pragma unroll
    for (int t = 0; t < 4; t++) {
        const float4 *src = (const float4 *)(X + L.row(t) * 128 + L.col0());
        float s = 0.f;
#pragma unroll
        for (int e = 0; e < 4; e++) {
            float4 f = src[e];
            x[t][4 * e] = f.x;
            x[t][4 * e + 1] = f.y;
            x[t][4 * e + 2] = f.z;
            x[t][4 * e + 3] = f.w;
            s += fabsf(f.x) + fabsf(f.y) + fabsf(f.z) + fabsf(f.w);
        }
        msum[t] = row_allreduce(s);
    }
    __syncthreads();
    fit_and_pack(L, S, x, msum, a.sh.unit_kind, a.tab.head_bits[h] != kPivot, a.sh.fit_iters);
    uint8_t *gpage = a.pool + (uint64_t)slot * a.stride + a.tab.head_off[h];
    copy16((uint4 *)gpage, (const uint4 *)S.page, (int)a.tab.head_bytes[h] >> 4, L.tid);
}

__global__ void __launch_bounds__(kThreads, 2) dequantize_kernel(PoolArgs a) {
    extern __shared__ __align__(16) uint8_t smem[];
    const Lane L;
    const TileSmem S(smem);
    const int Hv = a.sh.Hv;
    const int b = blockIdx.x / Hv, h = blockIdx.x - b * Hv;
    const int slot = a.slots[b];
    if (slot < 0 || slot >= a.pool_slots) {
        if (L.tid == 0) raise_error(a.err, STEPQ_ERR_SLOT_RANGE);
        return;
    }
    const uint8_t *gpage = a.pool + (uint64_t)slot * a.stride + a.tab.head_off[h];
    copy16((uint4 *)S.page, (const uint4 *)gpage, (int)a.tab.head_bytes[h] >> 4, L.tid);
    load_row_meta(L, S, a.tab, h);
    __syncthreads();
    const int has_scales = a.tab.head_bits[h] != kPivot;
    const uint16_t *page_r = (const uint16_t *)S.page;
    const uint16_t *page_c = (const uint16_t *)(S.page + 256);
    float *out = a.states + (size_t)b * a.state_stride_b + (size_t)h * kN;
#pragma unroll
    for (int t = 0; t < 4; t++) {
        const int i = L.row(t);
        const int bits = S.rbits[i];
        float vals[16];
        load_row16(S.page + S.roff[i], bits, L.cg, vals);
        if (bits != kPivot) {
            const float r = f16_val(page_r[i]);
            const float zs = a.sh.unit_kind ? (float)(1 << (8 - bits)) : 1.f;
#pragma unroll
            for (int j = 0; j < 16; j++) {
                const float rc = r * (has_scales ? f16_val(page_c[L.col0() + j]) : 1.f);
                vals[j] = __fmul_rn(rc, zs * vals[j]);       // one rounding of r c z
            }
        }
        float4 *dst = (float4 *)(out + i * 128 + L.col0());
#pragma unroll
        for (int e = 0; e < 4; e++)
            dst[e] = make_float4(vals[4 * e], vals[4 * e + 1], vals[4 * e + 2], vals[4 * e + 3]);
    }
}

// ------------------------------------------------------ calibration distortion
// One CTA per (sample, head): the reference state is fitted at every candidate
// width with the codec above (uniform over the head; pivot rows kept in FP16
// and out of the column fit) and its reconstruction error accumulated
// (Eqs. qwen_calibration_distortion, kda_calibration_distortion).
struct DistArgs {
    const float *states;          // [n][Hv][128][128]
    const float *w;               // [Hv][128] of the layer
    const uint8_t *pivot_rows;    // [Hv][128] of the layer, or null
    double *acc;                  // head: [Hv][K+1]; row: [Hv*128][K+1] (layer slice)
    int Hv, unit_rows, n_cand, fit_iters;
    int cands[4];
};

__global__ void __launch_bounds__(kThreads, 2) distortion_kernel(DistArgs a) {
    extern __shared__ __align__(16) uint8_t smem[];
    const Lane L;
    const TileSmem S(smem);
    const int s = blockIdx.x / a.Hv, h = blockIdx.x - s * a.Hv;
    const int K1 = a.n_cand + 1;
    if (L.tid < 128) {
        const float wv = a.w[h * 128 + L.tid];
        S.w2[L.tid] = __fmul_rn(wv, wv);
        S.wis[L.tid] = __frsqrt_rn(wv);
    }
    const float *X = a.states + ((size_t)s * a.Hv + h) * kN;
    float x[4][16], msum[4];
#pragma unroll
    for (int t = 0; t < 4; t++) {
        const float4 *src = (const float4 *)(X + L.row(t) * 128 + L.col0());
        float sm = 0.f;
#pragma unroll
        for (int e = 0; e < 4; e++) {
            const float4 v = src[e];
            x[t][4 * e] = v.x;
            x[t][4 * e + 1] = v.y;
            x[t][4 * e + 2] = v.z;
            x[t][4 * e + 3] = v.w;
            sm += fabsf(v.x) + fabsf(v.y) + fabsf(v.z) + fabsf(v.w);
        }
        msum[t] = row_allreduce(sm);
    }
    float *blk = S.col + 512;
    for (int k = 0; k < K1; k++) {
        const bool fp16_col = (k == a.n_cand);
        if (L.tid < 128) {
            const bool piv = fp16_col ||
                             (a.unit_rows && a.pivot_rows && a.pivot_rows[h * 128 + L.tid]);
            S.rbits[L.tid] = piv ? kPivot : a.cands[k];
        }
        __syncthreads();
        RowFit f;
        if (!fp16_col) fit_scales(L, S, x, msum, a.unit_rows, 0, a.fit_iters, f);
        float head_err = 0.f;
#pragma unroll
        for (int t = 0; t < 4; t++) {
            const int i = L.row(t);
            const int bits = S.rbits[i];
            float e = 0.f;
            if (bits == kPivot) {
#pragma unroll
                for (int j = 0; j < 16; j++) {
                    const float d = f16_round_sat(x[t][j]) - x[t][j];
                    e += d * d;
                }
            } else {
                const float lim = (float)f.qm[t];
#pragma unroll
                for (int j = 0; j < 16; j++) {
                    const float cj = S.col[L.col0() + j], gj = S.col[128 + L.col0() + j];
                    const float qv = fminf(fmaxf(rne_prod(__fmul_rn(x[t][j], f.rho[t]), gj), -lim), lim);
                    const float rec = __fmul_rn(f.rr[t] * cj, f.zsv[t] * qv);
                    const float d = rec - x[t][j];
                    e += d * d;
                }
            }
            e = row_allreduce(e);
            if (a.unit_rows) {
                if (L.cg == 0)
                    atomicAdd(&a.acc[((size_t)h * 128 + i) * K1 + k], (double)e / 128.0);
            } else {
                head_err += S.w2[i] * e;
            }
        }
        if (!a.unit_rows) {
            // rows of one lane group share head_err; take it once per group
            float v = (L.cg == 0) ? head_err : 0.f;
            for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
            if (L.lane == 0) blk[L.warp] = v;
            __syncthreads();
            if (L.tid == 0) {
                double sum = 0.0;
                for (int wv = 0; wv < 8; wv++) sum += blk[wv];
                atomicAdd(&a.acc[(size_t)h * K1 + k], sum / (double)kN);
            }
        }
        __syncthreads();
    }
}

// ------------------------------------------------------------------ launchers
static std::atomic<bool> g_attr_set[64];   // per device; setting the attributes twice is harmless

static stepq_status prepare(int dev) {
    if (dev < 0) cudaGetDevice(&dev);
    if (dev < 0 || dev >= 64) return STEPQ_ERR_CUDA;
    if (!g_attr_set[dev]) {
        if (cudaFuncSetAttribute(quantize_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 kSmemBytes) != cudaSuccess ||
            cudaFuncSetAttribute(dequantize_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 kSmemBytes) != cudaSuccess ||
            cudaFuncSetAttribute(distortion_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 kSmemBytes) != cudaSuccess)
            return STEPQ_ERR_CUDA;
        g_attr_set[dev] = true;
    }
    return STEPQ_OK;
}

static stepq_status launched() {
    return cudaGetLastError() == cudaSuccess ? STEPQ_OK : STEPQ_ERR_CUDA;
}

stepq_status launch_decode(const stepq_plan *p, int layer, uint8_t *pool, int pool_slots,
                           const int32_t *slots, int B, const float *q, const float *k,
                           const float *v, const float *beta, const float *gate, float *y,
                           cudaStream_t s) {
    if (p->cfg.gate_kind == STEPQ_GATE_SCALAR)
        return launch_decode_heads(p, layer, pool, pool_slots, slots, B, q, k, v, beta, gate, y, s);
    return launch_decode_rows(p, layer, pool, pool_slots, slots, B, q, k, v, beta, gate, y, s);
}

stepq_status launch_quantize(const stepq_plan *p, int layer, const float *states,
                             size_t state_stride_b, const int32_t *slots, int B, uint8_t *pool,
                             int pool_slots, cudaStream_t s) {
    if (p->cfg.gate_kind == STEPQ_GATE_SCALAR)
        return launch_quantize_heads(p, layer, states, state_stride_b, slots, B, pool, pool_slots, s);
    stepq_status st = prepare(p->device);
    if (st != STEPQ_OK) return st;
    PoolArgs a{pool, p->slot_stride, pool_slots, slots, p->layer(layer), p->shape(),
               (float *)states, state_stride_b, device_error_word()};
    quantize_kernel<<<(unsigned)B * p->cfg.n_value_heads, kThreads, kSmemBytes, s>>>(a);
    return launched();
}

stepq_status launch_dequantize(const stepq_plan *p, int layer, const uint8_t *pool, int pool_slots,
                               const int32_t *slots, int B, float *states, size_t state_stride_b,
                               cudaStream_t s) {
    if (p->cfg.gate_kind == STEPQ_GATE_SCALAR)
        return launch_dequantize_heads(p, layer, pool, pool_slots, slots, B, states, state_stride_b, s);
    stepq_status st = prepare(p->device);
    if (st != STEPQ_OK) return st;
    PoolArgs a{(uint8_t *)pool, p->slot_stride, pool_slots, slots, p->layer(layer), p->shape(),
               states, state_stride_b, device_error_word()};
    dequantize_kernel<<<(unsigned)B * p->cfg.n_value_heads, kThreads, kSmemBytes, s>>>(a);
    return launched();
}

stepq_status launch_calib_distortion(const stepq_config *cfg, int layer, const float *w,
                                     const uint8_t *pivot_rows, const float *states, int n,
                                     double *acc, cudaStream_t s) {
    stepq_status st = prepare(-1);
    if (st != STEPQ_OK) return st;
    const size_t Hv = (size_t)cfg->n_value_heads;
    const bool rows = cfg->gate_kind == STEPQ_GATE_CHANNEL;
    const size_t K1 = (size_t)cfg->n_candidates + 1;
    DistArgs a{};
    a.states = states;
    a.w = w + (size_t)layer * Hv * kD;
    a.pivot_rows = (rows && pivot_rows) ? pivot_rows + (size_t)layer * Hv * kD : nullptr;
    a.acc = acc + (size_t)layer * Hv * (rows ? kD : 1) * K1;
    a.Hv = (int)Hv;
    a.unit_rows = rows;
    a.n_cand = cfg->n_candidates;
    a.fit_iters = cfg->fit_iters;
    for (int k = 0; k < cfg->n_candidates; k++) a.cands[k] = cfg->candidates[k];
    distortion_kernel<<<(unsigned)(n * Hv), kThreads, kSmemBytes, s>>>(a);
    return launched();
}

}  // namespace stepq
