// Calibration statistics on the device (App. A.3): row-impact scores
// omega_i = E[g_{t,i}^2] with g_t = A_t^T q_t = D_t (q_t - beta_t k_t (k_t^T q_t))
// (Sec. 4.1, Eq. kda_sensitivity) and the mean log retention ell_u
// (Eq. calibration_lifetime). Sums are kept in fp64; the caller divides.
#include "device.cuh"
#include "internal.h"

namespace stepq {

struct ObsArgs {
    const float *q, *k, *beta, *gate;
    int n, Hk, Hv, gate_per_row;
    double *omega;     // [Hv][128] slice of the layer
    double *logret;    // [Hv] (scalar gate) or [Hv][128] slice of the layer
};

// One 128-thread CTA per value head; thread i owns key row i.
__global__ void __launch_bounds__(128) observe_kernel(ObsArgs a) {
    __shared__ double part[4];
    const int h = blockIdx.x, i = threadIdx.x;
    const int hk = h / (a.Hv / a.Hk);
    double om = 0.0, lr = 0.0;
    for (int b = 0; b < a.n; b++) {
        const double qi = a.q[((size_t)b * a.Hk + hk) * 128 + i];
        const double ki = a.k[((size_t)b * a.Hk + hk) * 128 + i];
        double p = qi * ki;
        for (int o = 16; o > 0; o >>= 1) p += __shfl_xor_sync(0xffffffffu, p, o);
        if ((i & 31) == 0) part[i >> 5] = p;
        __syncthreads();
        const double kq = part[0] + part[1] + part[2] + part[3];
        __syncthreads();
        const double d = a.gate_per_row ? (double)a.gate[((size_t)b * a.Hv + h) * 128 + i]
                                        : (double)a.gate[(size_t)b * a.Hv + h];
        const double g = d * (qi - (double)a.beta[(size_t)b * a.Hv + h] * ki * kq);
        om += g * g;
        lr += log(d);
    }
    a.omega[h * 128 + i] += om;
    if (a.gate_per_row) a.logret[h * 128 + i] += lr;
    else if (i == 0) a.logret[h] += lr;
}

stepq_status launch_calib_observe(const stepq_config *cfg, int layer, const float *q,
                                  const float *k, const float *beta, const float *gate, int n,
                                  double *omega_sum, double *logret_sum, cudaStream_t s) {
    ObsArgs a{};
    const size_t Hv = (size_t)cfg->n_value_heads;
    a.q = q; a.k = k; a.beta = beta; a.gate = gate;
    a.n = n;
    a.Hk = cfg->n_key_heads;
    a.Hv = (int)Hv;
    a.gate_per_row = cfg->gate_kind == STEPQ_GATE_CHANNEL;
    a.omega = omega_sum + (size_t)layer * Hv * kD;
    a.logret = logret_sum + (size_t)layer * Hv * (a.gate_per_row ? kD : 1);
    observe_kernel<<<(unsigned)Hv, 128, 0, s>>>(a);
    return cudaGetLastError() == cudaSuccess ? STEPQ_OK : STEPQ_ERR_CUDA;
}

}  // namespace stepq
