// The calibration protocol of App. A.3 behind one C entry point: it drives the
// observe, FP32-state replay and candidate-distortion kernels over a recorded
// trace, forms the means, chooses the FP16 pivots and, for row units, repeats
// the distortion pass with the pivot rows held out of the column fit (App. C.2).
#include <cstring>
#include <vector>

#include "internal.h"

using namespace stepq;

namespace {

size_t up256(size_t n) { return (n + 255) / 256 * 256; }

// Regions of the caller's workspace, each 256-byte aligned.
struct Workspace {
    double *omega_sum, *logret_sum, *acc;
    float *w, *S, *y;
    uint8_t *pivot;
    int32_t *slots;
    size_t bytes;

    Workspace(const stepq_config *cfg, int n, uint8_t *base) {
        const size_t heads = (size_t)cfg->n_layers * cfg->n_value_heads;
        const size_t U = stepq_num_units(cfg), K1 = (size_t)cfg->n_candidates + 1;
        size_t o = 0;
        const auto take = [&](size_t nb) {
            uint8_t *p = base ? base + o : nullptr;
            o += up256(nb);
            return p;
        };
        omega_sum = (double *)take(heads * kD * sizeof(double));
        logret_sum = (double *)take(U * sizeof(double));
        acc = (double *)take(U * K1 * sizeof(double));
        w = (float *)take(heads * kD * sizeof(float));
        pivot = take(U);
        slots = (int32_t *)take((size_t)n * sizeof(int32_t));
        S = (float *)take((size_t)n * cfg->n_value_heads * kN * sizeof(float));
        y = (float *)take((size_t)n * cfg->n_value_heads * kD * sizeof(float));
        bytes = o;
    }
};

__global__ void iota_kernel(int32_t *out, int n) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i < n) out[i] = i;
}

stepq_status cuda_ok(cudaError_t e) { return e == cudaSuccess ? STEPQ_OK : STEPQ_ERR_CUDA; }

}  // namespace

extern "C" size_t stepq_calib_workspace_bytes(const stepq_config *cfg, int n) {
    if (validate_config(cfg, true) != STEPQ_OK || n <= 0) return 0;
    return Workspace(cfg, n, nullptr).bytes;
}

extern "C" stepq_status stepq_calibrate_from_trace(const stepq_config *cfg, int n, int T, int every,
                                                   const float *q, const float *k, const float *v,
                                                   const float *beta, const float *gate,
                                                   void *workspace, size_t workspace_bytes,
                                                   stepq_calib_result *out, stepq_stream_t stream) {
    stepq_status st = validate_config(cfg, true);
    if (st != STEPQ_OK) return st;
    if (n <= 0 || T <= 0 || every <= 0 || !q || !k || !v || !beta || !gate || !workspace || !out ||
        !out->omega || !out->mean_log_ret || !out->distortion || !out->pivot_mask)
        return STEPQ_ERR_ARG;
    if (((uintptr_t)workspace & 255) || ((uintptr_t)q & 15) || ((uintptr_t)k & 15) ||
        ((uintptr_t)v & 15) || ((uintptr_t)beta & 3) || ((uintptr_t)gate & 15))
        return STEPQ_ERR_ALIGN;
    Workspace ws(cfg, n, (uint8_t *)workspace);
    if (workspace_bytes < ws.bytes) return STEPQ_ERR_ARG;
    cudaStream_t s = (cudaStream_t)stream;
    const int L = cfg->n_layers, Hv = cfg->n_value_heads, Hk = cfg->n_key_heads;
    const bool rows = cfg->gate_kind == STEPQ_GATE_CHANNEL;
    const size_t heads = (size_t)L * Hv, U = stepq_num_units(cfg), K1 = (size_t)cfg->n_candidates + 1;
    // trace strides per token step of one layer
    const size_t sq = (size_t)n * Hk * kD, sv = (size_t)n * Hv * kD, sb = (size_t)n * Hv;
    const size_t sg = rows ? sv : sb;
    const auto at = [&](const float *base, size_t stride, int layer, int t) {
        return base + ((size_t)layer * T + t) * stride;
    };

    // Pass A: sums of g_{t,i}^2 (Sec. 4.1) and of log retention (Eq. calibration_lifetime).
    if ((st = cuda_ok(cudaMemsetAsync(ws.omega_sum, 0, heads * kD * sizeof(double), s))) != STEPQ_OK ||
        (st = cuda_ok(cudaMemsetAsync(ws.logret_sum, 0, U * sizeof(double), s))) != STEPQ_OK)
        return st;
    for (int t = 0; t < T; t++)
        for (int l = 0; l < L; l++)
            if ((st = launch_calib_observe(cfg, l, at(q, sq, l, t), at(k, sq, l, t), at(beta, sb, l, t),
                                           at(gate, sg, l, t), n, ws.omega_sum, ws.logret_sum, s)) != STEPQ_OK)
                return st;
    std::vector<double> osum(heads * kD), lsum(U);
    if ((st = cuda_ok(cudaMemcpyAsync(osum.data(), ws.omega_sum, osum.size() * sizeof(double),
                                      cudaMemcpyDeviceToHost, s))) != STEPQ_OK ||
        (st = cuda_ok(cudaMemcpyAsync(lsum.data(), ws.logret_sum, lsum.size() * sizeof(double),
                                      cudaMemcpyDeviceToHost, s))) != STEPQ_OK ||
        (st = cuda_ok(cudaStreamSynchronize(s))) != STEPQ_OK)
        return st;
    const double n_tok = (double)n * T;
    for (size_t e = 0; e < osum.size(); e++) out->omega[e] = (float)(osum[e] / n_tok);
    for (size_t u = 0; u < U; u++) out->mean_log_ret[u] = lsum[u] / n_tok;
    out->n_tokens = n * T;

    // Row-impact factors of the fit weights (footnote of Sec. 4.3).
    std::vector<float> w(heads * kD);
    if ((st = stepq_row_weights(cfg, out->omega, w.data())) != STEPQ_OK) return st;
    if ((st = cuda_ok(cudaMemcpyAsync(ws.w, w.data(), w.size() * sizeof(float), cudaMemcpyHostToDevice, s))) !=
        STEPQ_OK)
        return st;
    iota_kernel<<<(n + 255) / 256, 256, 0, s>>>(ws.slots, n);
    if ((st = cuda_ok(cudaGetLastError())) != STEPQ_OK) return st;

    // Pass B: replay the FP32-state recurrence from zero per layer and fit every
    // `every`-th state at each candidate width (Eqs. qwen_calibration_distortion,
    // kda_calibration_distortion); each sequence is one sample.
    stepq_config one = *cfg;
    one.n_layers = 1;
    const auto distortion_pass = [&](const uint8_t *pivot_rows, double *dist) -> stepq_status {
        stepq_status e;
        if ((e = cuda_ok(cudaMemsetAsync(ws.acc, 0, U * K1 * sizeof(double), s))) != STEPQ_OK) return e;
        int n_samp = 0;
        for (int l = 0; l < L; l++) {
            if ((e = cuda_ok(cudaMemsetAsync(ws.S, 0, (size_t)n * Hv * kN * sizeof(float), s))) != STEPQ_OK)
                return e;
            for (int t = 0; t < T; t++) {
                if ((e = launch_fp32_decode(&one, 0, ws.S, nullptr, n, ws.slots, n, at(q, sq, l, t),
                                            at(k, sq, l, t), at(v, sv, l, t), at(beta, sb, l, t),
                                            at(gate, sg, l, t), ws.y, s)) != STEPQ_OK)
                    return e;
                if ((t + 1) % every == 0) {
                    if ((e = launch_calib_distortion(cfg, l, ws.w, pivot_rows, ws.S, n, ws.acc, s)) != STEPQ_OK)
                        return e;
                    if (l == 0) n_samp += n;
                }
            }
        }
        std::vector<double> acc(U * K1);
        if ((e = cuda_ok(cudaMemcpyAsync(acc.data(), ws.acc, acc.size() * sizeof(double),
                                         cudaMemcpyDeviceToHost, s))) != STEPQ_OK ||
            (e = cuda_ok(cudaStreamSynchronize(s))) != STEPQ_OK)
            return e;
        const double ns = n_samp > 0 ? n_samp : 1;
        for (size_t x = 0; x < acc.size(); x++) dist[x] = acc[x] / ns;
        out->n_samples = n_samp;
        return STEPQ_OK;
    };
    std::vector<double> d1(U * K1);
    if ((st = distortion_pass(nullptr, d1.data())) != STEPQ_OK) return st;
    if (out->distortion_stage1) std::memcpy(out->distortion_stage1, d1.data(), d1.size() * sizeof(double));
    if ((st = stepq_select_pivots(cfg, out->mean_log_ret, d1.data(), out->pivot_mask)) != STEPQ_OK) return st;
    bool any = false;
    for (size_t u = 0; u < U; u++) any = any || out->pivot_mask[u];
    if (rows && any) {
        // row units: measure again with the chosen pivot rows kept in FP16
        if ((st = cuda_ok(cudaMemcpyAsync(ws.pivot, out->pivot_mask, U, cudaMemcpyHostToDevice, s))) != STEPQ_OK)
            return st;
        return distortion_pass(ws.pivot, out->distortion);
    }
    std::memcpy(out->distortion, d1.data(), d1.size() * sizeof(double));
    return STEPQ_OK;
}
