// C-ABI entry points of the device path: argument checks, then one launch.
// No entry point here synchronises or allocates except stepq_device_error() and
// stepq_stream_status(), which read the sticky device error.
#include <cstdint>

#include "internal.h"

using namespace stepq;

namespace {

bool aligned(const void *p, uintptr_t a) { return ((uintptr_t)p % a) == 0; }

stepq_status check_plan_call(const stepq_plan *p, int layer, bool allow_all, const void *pool,
                             int pool_slots, const int32_t *slots, int B) {
    if (!p || !pool || (B > 0 && !slots) || B < 0 || pool_slots <= 0) return STEPQ_ERR_ARG;
    if (layer < (allow_all ? -1 : 0) || layer >= p->cfg.n_layers) return STEPQ_ERR_ARG;
    if (!aligned(pool, 256) || !aligned(slots, 4)) return STEPQ_ERR_ALIGN;
    if (!p->dev_mem) return STEPQ_ERR_CUDA;      // plan built without a CUDA device
    return STEPQ_OK;
}

stepq_status check_inputs(const stepq_config *cfg, const float *q, const float *k, const float *v,
                          const float *beta, const float *gate, const float *y) {
    if (!q || !k || !beta || !gate || (v == nullptr) != (y == nullptr)) return STEPQ_ERR_ARG;
    if (!aligned(q, 16) || !aligned(k, 16) || (v && !aligned(v, 16)) || (y && !aligned(y, 16)) ||
        !aligned(beta, 4) || !aligned(gate, cfg->gate_kind == STEPQ_GATE_CHANNEL ? 16 : 4))
        return STEPQ_ERR_ALIGN;
    return STEPQ_OK;
}

}  // namespace

extern "C" stepq_status stepq_quantize_pool(const stepq_plan *p, int layer, const float *states,
                                            const int32_t *slots, int B, void *pool,
                                            int pool_slots, stepq_stream_t stream) {
    stepq_status st = check_plan_call(p, layer, true, pool, pool_slots, slots, B);
    if (st != STEPQ_OK) return st;
    if (!states) return STEPQ_ERR_ARG;
    if (!aligned(states, 16)) return STEPQ_ERR_ALIGN;
    if (B == 0) return STEPQ_OK;
    const size_t per_layer = (size_t)p->cfg.n_value_heads * kN;
    cudaStream_t s = (cudaStream_t)stream;
    if (layer >= 0) return launch_quantize(p, layer, states, per_layer, slots, B, (uint8_t *)pool, pool_slots, s);
    for (int l = 0; l < p->cfg.n_layers; l++) {
        st = launch_quantize(p, l, states + l * per_layer, per_layer * p->cfg.n_layers, slots, B,
                             (uint8_t *)pool, pool_slots, s);
        if (st != STEPQ_OK) return st;
    }
    return STEPQ_OK;
}

extern "C" stepq_status stepq_dequantize_pool(const stepq_plan *p, int layer, const void *pool,
                                              int pool_slots, const int32_t *slots, int B,
                                              float *states, stepq_stream_t stream) {
    stepq_status st = check_plan_call(p, layer, true, pool, pool_slots, slots, B);
    if (st != STEPQ_OK) return st;
    if (!states) return STEPQ_ERR_ARG;
    if (!aligned(states, 16)) return STEPQ_ERR_ALIGN;
    if (B == 0) return STEPQ_OK;
    const size_t per_layer = (size_t)p->cfg.n_value_heads * kN;
    cudaStream_t s = (cudaStream_t)stream;
    if (layer >= 0) return launch_dequantize(p, layer, (const uint8_t *)pool, pool_slots, slots, B, states, per_layer, s);
    for (int l = 0; l < p->cfg.n_layers; l++) {
        st = launch_dequantize(p, l, (const uint8_t *)pool, pool_slots, slots, B,
                               states + l * per_layer, per_layer * p->cfg.n_layers, s);
        if (st != STEPQ_OK) return st;
    }
    return STEPQ_OK;
}

extern "C" size_t stepq_temporal_slot_bytes(const stepq_plan *p) { return p ? p->t_slot_stride : 0; }

extern "C" stepq_status stepq_temporal_quantize_pool(const stepq_plan *p, int layer,
                                                     const float *states, const int32_t *slots,
                                                     int B, void *pool, int pool_slots,
                                                     stepq_stream_t stream) {
    stepq_status st = check_plan_call(p, layer, true, pool, pool_slots, slots, B);
    if (st != STEPQ_OK) return st;
    if (!states) return STEPQ_ERR_ARG;
    if (!aligned(states, 16)) return STEPQ_ERR_ALIGN;
    if (B == 0) return STEPQ_OK;
    const size_t per_layer = (size_t)p->cfg.n_value_heads * kN;
    cudaStream_t s = (cudaStream_t)stream;
    if (layer >= 0)
        return launch_temporal_quantize(p, layer, states, per_layer, slots, B, (uint8_t *)pool, pool_slots, s);
    for (int l = 0; l < p->cfg.n_layers; l++)
        if ((st = launch_temporal_quantize(p, l, states + l * per_layer, per_layer * p->cfg.n_layers,
                                           slots, B, (uint8_t *)pool, pool_slots, s)) != STEPQ_OK)
            return st;
    return STEPQ_OK;
}

extern "C" stepq_status stepq_temporal_dequantize_pool(const stepq_plan *p, int layer,
                                                       const void *pool, int pool_slots,
                                                       const int32_t *slots, int B, float *states,
                                                       stepq_stream_t stream) {
    stepq_status st = check_plan_call(p, layer, true, pool, pool_slots, slots, B);
    if (st != STEPQ_OK) return st;
    if (!states) return STEPQ_ERR_ARG;
    if (!aligned(states, 16)) return STEPQ_ERR_ALIGN;
    if (B == 0) return STEPQ_OK;
    const size_t per_layer = (size_t)p->cfg.n_value_heads * kN;
    cudaStream_t s = (cudaStream_t)stream;
    if (layer >= 0)
        return launch_temporal_dequantize(p, layer, (const uint8_t *)pool, pool_slots, slots, B, states,
                                          per_layer, s);
    for (int l = 0; l < p->cfg.n_layers; l++)
        if ((st = launch_temporal_dequantize(p, l, (const uint8_t *)pool, pool_slots, slots, B,
                                             states + l * per_layer, per_layer * p->cfg.n_layers,
                                             s)) != STEPQ_OK)
            return st;
    return STEPQ_OK;
}

extern "C" stepq_status stepq_decode_step(const stepq_plan *p, int layer, void *pool,
                                          int pool_slots, const int32_t *slots, int B,
                                          const float *q, const float *k, const float *v,
                                          const float *beta, const float *gate, float *y,
                                          stepq_stream_t stream) {
    stepq_status st = check_plan_call(p, layer, false, pool, pool_slots, slots, B);
    if (st != STEPQ_OK) return st;
    if (!v || !y) return STEPQ_ERR_ARG;
    if ((st = check_inputs(&p->cfg, q, k, v, beta, gate, y)) != STEPQ_OK) return st;
    if (B == 0) return STEPQ_OK;
    return launch_decode(p, layer, (uint8_t *)pool, pool_slots, slots, B, q, k, v, beta, gate, y,
                         (cudaStream_t)stream);
}

extern "C" stepq_status stepq_decode_readout(const stepq_plan *p, int layer, const void *pool,
                                             int pool_slots, const int32_t *slots, int B,
                                             const float *q, const float *k, const float *v,
                                             const float *beta, const float *gate, float *y,
                                             float *delta, stepq_stream_t stream) {
    stepq_status st = check_plan_call(p, layer, false, pool, pool_slots, slots, B);
    if (st != STEPQ_OK) return st;
    if (!v || !y || !delta) return STEPQ_ERR_ARG;
    if ((st = check_inputs(&p->cfg, q, k, v, beta, gate, y)) != STEPQ_OK) return st;
    if (!aligned(delta, 16)) return STEPQ_ERR_ALIGN;
    if (B == 0) return STEPQ_OK;
    if (p->cfg.gate_kind == STEPQ_GATE_CHANNEL)
        return launch_decode_rows_mode(p, layer, (uint8_t *)pool, pool_slots, slots, B, q, k, v, beta,
                                       gate, y, delta, 1, (cudaStream_t)stream);
    return launch_decode_heads_mode(p, layer, (uint8_t *)pool, pool_slots, slots, B, q, k, v, beta,
                                    gate, y, delta, 1, (cudaStream_t)stream);
}

extern "C" stepq_status stepq_decode_writeback(const stepq_plan *p, int layer, void *pool,
                                               int pool_slots, const int32_t *slots, int B,
                                               const float *k, const float *beta,
                                               const float *gate, const float *delta,
                                               stepq_stream_t stream) {
    stepq_status st = check_plan_call(p, layer, false, pool, pool_slots, slots, B);
    if (st != STEPQ_OK) return st;
    if (!k || !beta || !gate || !delta) return STEPQ_ERR_ARG;
    if (!aligned(k, 16) || !aligned(delta, 16) || !aligned(beta, 4) ||
        !aligned(gate, p->cfg.gate_kind == STEPQ_GATE_CHANNEL ? 16 : 4))
        return STEPQ_ERR_ALIGN;
    if (B == 0) return STEPQ_OK;
    if (p->cfg.gate_kind == STEPQ_GATE_CHANNEL)
        return launch_decode_rows_mode(p, layer, (uint8_t *)pool, pool_slots, slots, B, nullptr, k,
                                       nullptr, beta, gate, nullptr, (float *)delta, 2,
                                       (cudaStream_t)stream);
    return launch_decode_heads_mode(p, layer, (uint8_t *)pool, pool_slots, slots, B, nullptr, k,
                                    nullptr, beta, gate, nullptr, (float *)delta, 2,
                                    (cudaStream_t)stream);
}

extern "C" stepq_status stepq_fp32_decode_step(const stepq_config *cfg, int layer, float *pool,
                                               int pool_slots, const int32_t *slots, int B,
                                               const float *q, const float *k, const float *v,
                                               const float *beta, const float *gate, float *y,
                                               stepq_stream_t stream) {
    stepq_status st = validate_config(cfg, false);
    if (st != STEPQ_OK) return st;
    if (!pool || (B > 0 && !slots) || B < 0 || pool_slots <= 0 || layer < 0 || layer >= cfg->n_layers || !v || !y)
        return STEPQ_ERR_ARG;
    if (!aligned(pool, 16)) return STEPQ_ERR_ALIGN;
    if ((st = check_inputs(cfg, q, k, v, beta, gate, y)) != STEPQ_OK) return st;
    if (B == 0) return STEPQ_OK;
    return launch_fp32_decode(cfg, layer, pool, nullptr, pool_slots, slots, B, q, k, v, beta, gate,
                              y, (cudaStream_t)stream);
}

extern "C" stepq_status stepq_fp32_exact_read_step(const stepq_config *cfg, int layer, float *pool,
                                                   const float *read_pool, int pool_slots,
                                                   const int32_t *slots, int B, const float *q,
                                                   const float *k, const float *v, const float *beta,
                                                   const float *gate, float *y,
                                                   stepq_stream_t stream) {
    stepq_status st = validate_config(cfg, false);
    if (st != STEPQ_OK) return st;
    if (!pool || !read_pool || (B > 0 && !slots) || B < 0 || pool_slots <= 0 || layer < 0 ||
        layer >= cfg->n_layers || !v || !y)
        return STEPQ_ERR_ARG;
    if (!aligned(pool, 16) || !aligned(read_pool, 16)) return STEPQ_ERR_ALIGN;
    if ((st = check_inputs(cfg, q, k, v, beta, gate, y)) != STEPQ_OK) return st;
    if (B == 0) return STEPQ_OK;
    return launch_fp32_decode(cfg, layer, pool, read_pool, pool_slots, slots, B, q, k, v, beta, gate,
                              y, (cudaStream_t)stream);
}

extern "C" stepq_status stepq_prefill_fp32(const stepq_config *cfg, int B, int T, float *states,
                                           const float *q, const float *k, const float *v,
                                           const float *beta, const float *gate, float *y,
                                           stepq_stream_t stream) {
    stepq_status st = validate_config(cfg, false);
    if (st != STEPQ_OK) return st;
    if (B < 0 || T < 0 || (B > 0 && T > 0 && (!states || !v || !y))) return STEPQ_ERR_ARG;
    if (B == 0 || T == 0) return STEPQ_OK;
    if (!aligned(states, 16)) return STEPQ_ERR_ALIGN;
    if ((st = check_inputs(cfg, q, k, v, beta, gate, y)) != STEPQ_OK) return st;
    return launch_prefill(cfg, q, k, v, beta, gate, B, T, states, y, (cudaStream_t)stream);
}

extern "C" size_t stepq_intb_slot_bytes(const stepq_config *cfg, int bits) {
    if (validate_config(cfg, false) != STEPQ_OK || (bits != 4 && bits != 6 && bits != 8)) return 0;
    size_t page = intb_head_bytes(bits) * cfg->n_value_heads * cfg->n_layers;
    return (page + 255) / 256 * 256;
}

static stepq_status check_intb(const stepq_config *cfg, int bits, int layer, bool allow_all,
                               const void *pool, int pool_slots, const int32_t *slots, int B) {
    stepq_status st = validate_config(cfg, false);
    if (st != STEPQ_OK) return st;
    if (bits != 4 && bits != 6 && bits != 8) return STEPQ_ERR_UNSUPPORTED;
    if (!pool || (B > 0 && !slots) || B < 0 || pool_slots <= 0) return STEPQ_ERR_ARG;
    if (layer < (allow_all ? -1 : 0) || layer >= cfg->n_layers) return STEPQ_ERR_ARG;
    if (!aligned(pool, 256)) return STEPQ_ERR_ALIGN;
    return STEPQ_OK;
}

extern "C" stepq_status stepq_intb_quantize_pool(const stepq_config *cfg, int bits, int layer,
                                                 const float *states, const int32_t *slots, int B,
                                                 void *pool, int pool_slots, stepq_stream_t stream) {
    stepq_status st = check_intb(cfg, bits, layer, true, pool, pool_slots, slots, B);
    if (st != STEPQ_OK) return st;
    if (!states) return STEPQ_ERR_ARG;
    if (!aligned(states, 16)) return STEPQ_ERR_ALIGN;
    if (B == 0) return STEPQ_OK;
    const size_t per_layer = (size_t)cfg->n_value_heads * kN;
    cudaStream_t s = (cudaStream_t)stream;
    if (layer >= 0) return launch_intb_quantize(cfg, bits, layer, states, per_layer, slots, B, (uint8_t *)pool, pool_slots, s);
    for (int l = 0; l < cfg->n_layers; l++)
        if ((st = launch_intb_quantize(cfg, bits, l, states + l * per_layer, per_layer * cfg->n_layers,
                                       slots, B, (uint8_t *)pool, pool_slots, s)) != STEPQ_OK)
            return st;
    return STEPQ_OK;
}

extern "C" stepq_status stepq_intb_dequantize_pool(const stepq_config *cfg, int bits, int layer,
                                                   const void *pool, int pool_slots,
                                                   const int32_t *slots, int B, float *states,
                                                   stepq_stream_t stream) {
    stepq_status st = check_intb(cfg, bits, layer, true, pool, pool_slots, slots, B);
    if (st != STEPQ_OK) return st;
    if (!states) return STEPQ_ERR_ARG;
    if (!aligned(states, 16)) return STEPQ_ERR_ALIGN;
    if (B == 0) return STEPQ_OK;
    const size_t per_layer = (size_t)cfg->n_value_heads * kN;
    cudaStream_t s = (cudaStream_t)stream;
    if (layer >= 0) return launch_intb_dequantize(cfg, bits, layer, (const uint8_t *)pool, pool_slots, slots, B, states, per_layer, s);
    for (int l = 0; l < cfg->n_layers; l++)
        if ((st = launch_intb_dequantize(cfg, bits, l, (const uint8_t *)pool, pool_slots, slots, B,
                                         states + l * per_layer, per_layer * cfg->n_layers, s)) != STEPQ_OK)
            return st;
    return STEPQ_OK;
}

extern "C" stepq_status stepq_intb_decode_step(const stepq_config *cfg, int bits, int layer,
                                               void *pool, int pool_slots, const int32_t *slots,
                                               int B, const float *q, const float *k,
                                               const float *v, const float *beta,
                                               const float *gate, float *y, stepq_stream_t stream) {
    stepq_status st = check_intb(cfg, bits, layer, false, pool, pool_slots, slots, B);
    if (st != STEPQ_OK) return st;
    if (!v || !y) return STEPQ_ERR_ARG;
    if ((st = check_inputs(cfg, q, k, v, beta, gate, y)) != STEPQ_OK) return st;
    if (B == 0) return STEPQ_OK;
    return launch_intb_decode(cfg, bits, layer, (uint8_t *)pool, pool_slots, slots, B, q, k, v,
                              beta, gate, y, (cudaStream_t)stream);
}

extern "C" stepq_status stepq_calib_observe(const stepq_config *cfg, int layer, const float *q,
                                            const float *k, const float *beta, const float *gate,
                                            int n, double *omega_sum, double *logret_sum,
                                            stepq_stream_t stream) {
    stepq_status st = validate_config(cfg, false);
    if (st != STEPQ_OK) return st;
    if (layer < 0 || layer >= cfg->n_layers || n < 0 || !omega_sum || !logret_sum) return STEPQ_ERR_ARG;
    if ((st = check_inputs(cfg, q, k, nullptr, beta, gate, nullptr)) != STEPQ_OK) return st;
    if (n == 0) return STEPQ_OK;
    return launch_calib_observe(cfg, layer, q, k, beta, gate, n, omega_sum, logret_sum,
                                (cudaStream_t)stream);
}

extern "C" stepq_status stepq_calib_distortion(const stepq_config *cfg, int layer, const float *w,
                                               const uint8_t *pivot_rows, const float *states,
                                               int n, double *acc, stepq_stream_t stream) {
    stepq_status st = validate_config(cfg, true);
    if (st != STEPQ_OK) return st;
    if (layer < 0 || layer >= cfg->n_layers || n < 0 || !w || !states || !acc) return STEPQ_ERR_ARG;
    if (!aligned(states, 16) || !aligned(w, 4) || !aligned(acc, 8)) return STEPQ_ERR_ALIGN;
    if (n == 0) return STEPQ_OK;
    return launch_calib_distortion(cfg, layer, w, pivot_rows, states, n, acc, (cudaStream_t)stream);
}

extern "C" stepq_status stepq_validate_slots(const int32_t *slots, int B, int pool_slots,
                                             uint32_t *scratch, int32_t *status_out,
                                             stepq_stream_t stream) {
    if ((B > 0 && !slots) || B < 0 || pool_slots <= 0 || !scratch || !status_out) return STEPQ_ERR_ARG;
    return launch_validate_slots(slots, B, pool_slots, scratch, status_out, (cudaStream_t)stream);
}

extern "C" stepq_status stepq_validate_slots_noalloc(const int32_t *slots, int B, int pool_slots,
                                                     int32_t *status_out, stepq_stream_t stream) {
    if ((B > 0 && !slots) || B < 0 || pool_slots <= 0 || !status_out) return STEPQ_ERR_ARG;
    return launch_validate_slots_static(slots, B, pool_slots, status_out, (cudaStream_t)stream);
}

extern "C" stepq_status stepq_device_error(stepq_stream_t stream) {
    return read_device_error((cudaStream_t)stream);
}

extern "C" stepq_status stepq_stream_status(stepq_stream_t stream) {
    return read_device_error((cudaStream_t)stream);
}

extern "C" const char *stepq_status_str(stepq_status s) {
    switch (s) {
    case STEPQ_OK: return "ok";
    case STEPQ_ERR_ARG: return "invalid argument";
    case STEPQ_ERR_SLOT_RANGE: return "slot id out of range";
    case STEPQ_ERR_DUP_SLOT: return "slot id repeated within one call";
    case STEPQ_ERR_ALIGN: return "misaligned buffer";
    case STEPQ_ERR_CUDA: return "CUDA runtime error";
    case STEPQ_ERR_BUDGET: return "bit budget cannot be met by the candidates";
    case STEPQ_ERR_UNSUPPORTED: return "unsupported configuration";
    case STEPQ_ERR_TIMEOUT: return "a device-side wait exceeded its bound";
    }
    return "unknown status";
}

extern "C" const char *stepq_version(void) { return "stepq 0.1 (sm_103a)"; }

extern "C" stepq_status stepq_debug_stall(long long wait_cycles, int withhold_item) {
    return set_stall_knob(wait_cycles, withhold_item);
}
