// Internal definitions shared by the library's translation units (not part of the ABI).
#pragma once

#include <cstddef>
#include <cstdint>
#include <vector>

#include <cuda_runtime.h>

#include "stepq.h"

namespace stepq {

constexpr int kD = 128;                    // d_k = d_v
constexpr int kN = kD * kD;
constexpr int kPivot = STEPQ_PIVOT_BITS;
constexpr uint32_t kMaxHeadBytes = 512 + kD * 16 * kPivot;   // a row-unit head of FP16 rows

// Device-side view of a plan for one layer. Per-row tables cover both unit
// kinds: a head unit repeats its width on every row.
struct LayerTables {
    const float *w2;          // [Hv][128] fp32(w_i^2)
    const float *wis;         // [Hv][128] fp32(w_i^(-1/2))
    const uint64_t *head_off; // [Hv] byte offset of the head segment in a slot page
    const uint32_t *head_bytes;
    const uint8_t *head_bits; // [Hv] head width, 16 for a pivot head, 0 for row units
    const uint8_t *row_bits;  // [Hv][128]
    const uint32_t *row_off;  // [Hv][128] payload offset of row i within the head segment
    const uint32_t *row_slot; // [Hv][128] s-th stored row: offset | width << 16 | row << 24
};

struct Shape {
    int Hk, Hv, n_layers;
    int gate_per_row;         // 1 for the channel gate (KDA)
    int unit_kind;            // 0 head units, 1 row units
    int fit_iters;
};

}  // namespace stepq

struct stepq_plan {
    stepq_config cfg;
    size_t n_units = 0;
    std::vector<int8_t> unit_bits;
    std::vector<uint8_t> pivot;
    std::vector<float> w;
    std::vector<double> life;
    std::vector<uint64_t> head_off;
    std::vector<uint32_t> head_bytes;
    size_t slot_stride = 0;
    uint32_t max_head_bytes = 0;
    int device = 0;
    // device tables (one allocation)
    void *dev_mem = nullptr;
    float *d_w2 = nullptr, *d_wis = nullptr;
    uint64_t *d_head_off = nullptr;
    uint32_t *d_head_bytes = nullptr;
    uint8_t *d_head_bits = nullptr;
    uint8_t *d_row_bits = nullptr;
    uint32_t *d_row_off = nullptr;
    uint32_t *d_row_slot = nullptr;
    // layout of the "Temporal only" ablation codec (rowwise absmax at the plan's
    // widths): head segments in (layer, head) order, rows in index order
    std::vector<uint64_t> t_head_off;
    size_t t_slot_stride = 0;
    uint64_t *d_t_head_off = nullptr;
    uint32_t *d_t_row_off = nullptr;   // [heads][128] row payload offset within the head segment

    stepq::LayerTables layer(int l) const {
        const size_t Hv = (size_t)cfg.n_value_heads;
        return {d_w2 + l * Hv * stepq::kD, d_wis + l * Hv * stepq::kD, d_head_off + l * Hv,
                d_head_bytes + l * Hv, d_head_bits + l * Hv, d_row_bits + l * Hv * stepq::kD,
                d_row_off + l * Hv * stepq::kD, d_row_slot + l * Hv * stepq::kD};
    }
    stepq::Shape shape() const {
        return {cfg.n_key_heads, cfg.n_value_heads, cfg.n_layers,
                cfg.gate_kind == STEPQ_GATE_CHANNEL ? 1 : 0,
                cfg.gate_kind == STEPQ_GATE_CHANNEL ? 1 : 0, cfg.fit_iters};
    }
};

namespace stepq {

// plan.cpp
stepq_status validate_config(const stepq_config *cfg, bool need_quant_fields);

// kernels (stepq_kernels.cu)
stepq_status launch_decode(const stepq_plan *p, int layer, uint8_t *pool, int pool_slots,
                           const int32_t *slots, int B, const float *q, const float *k,
                           const float *v, const float *beta, const float *gate, float *y,
                           cudaStream_t s);
stepq_status launch_quantize(const stepq_plan *p, int layer, const float *states,
                             size_t state_stride_b, const int32_t *slots, int B, uint8_t *pool,
                             int pool_slots, cudaStream_t s);
stepq_status launch_dequantize(const stepq_plan *p, int layer, const uint8_t *pool, int pool_slots,
                               const int32_t *slots, int B, float *states, size_t state_stride_b,
                               cudaStream_t s);
// prefill.cu (chunked FP32-state prefill)
stepq_status launch_prefill(const stepq_config *cfg, const float *q, const float *k, const float *v,
                            const float *beta, const float *gate, int B, int T, float *states, float *y,
                            cudaStream_t s);
// rows.cu (row units, row-major pages with per-row widths)
stepq_status launch_decode_rows(const stepq_plan *p, int layer, uint8_t *pool, int pool_slots,
                                const int32_t *slots, int B, const float *q, const float *k,
                                const float *v, const float *beta, const float *gate, float *y,
                                cudaStream_t s);
stepq_status launch_decode_rows_mode(const stepq_plan *p, int layer, uint8_t *pool, int pool_slots,
                                     const int32_t *slots, int B, const float *q, const float *k,
                                     const float *v, const float *beta, const float *gate, float *y,
                                     float *delta, int mode, cudaStream_t s);
// heads.cu (head units, band-major pages)
stepq_status launch_decode_heads(const stepq_plan *p, int layer, uint8_t *pool, int pool_slots,
                                 const int32_t *slots, int B, const float *q, const float *k,
                                 const float *v, const float *beta, const float *gate, float *y,
                                 cudaStream_t s);
// mode 0 fused, 1 readout (y and delta out, pages untouched), 2 writeback (delta in)
stepq_status launch_decode_heads_mode(const stepq_plan *p, int layer, uint8_t *pool, int pool_slots,
                                      const int32_t *slots, int B, const float *q, const float *k,
                                      const float *v, const float *beta, const float *gate, float *y,
                                      float *delta, int mode, cudaStream_t s);
stepq_status launch_quantize_heads(const stepq_plan *p, int layer, const float *states,
                                   size_t stride_b, const int32_t *slots, int B, uint8_t *pool,
                                   int pool_slots, cudaStream_t s);
stepq_status launch_dequantize_heads(const stepq_plan *p, int layer, const uint8_t *pool,
                                     int pool_slots, const int32_t *slots, int B, float *states,
                                     size_t stride_b, cudaStream_t s);
// baselines.cu
stepq_status launch_fp32_decode(const stepq_config *cfg, int layer, float *pool,
                                const float *read_pool, int pool_slots, const int32_t *slots, int B,
                                const float *q, const float *k, const float *v, const float *beta,
                                const float *gate, float *y, cudaStream_t s);
stepq_status launch_temporal_quantize(const stepq_plan *p, int layer, const float *states,
                                      size_t state_stride_b, const int32_t *slots, int B,
                                      uint8_t *pool, int pool_slots, cudaStream_t s);
stepq_status launch_temporal_dequantize(const stepq_plan *p, int layer, const uint8_t *pool,
                                        int pool_slots, const int32_t *slots, int B, float *states,
                                        size_t state_stride_b, cudaStream_t s);
stepq_status launch_intb_quantize(const stepq_config *cfg, int bits, int layer,
                                  const float *states, size_t state_stride_b,
                                  const int32_t *slots, int B, uint8_t *pool, int pool_slots,
                                  cudaStream_t s);
stepq_status launch_intb_dequantize(const stepq_config *cfg, int bits, int layer,
                                    const uint8_t *pool, int pool_slots, const int32_t *slots,
                                    int B, float *states, size_t state_stride_b, cudaStream_t s);
stepq_status launch_intb_decode(const stepq_config *cfg, int bits, int layer, uint8_t *pool,
                                int pool_slots, const int32_t *slots, int B, const float *q,
                                const float *k, const float *v, const float *beta,
                                const float *gate, float *y, cudaStream_t s);
// calib.cu
stepq_status launch_calib_observe(const stepq_config *cfg, int layer, const float *q,
                                  const float *k, const float *beta, const float *gate, int n,
                                  double *omega_sum, double *logret_sum, cudaStream_t s);
stepq_status launch_calib_distortion(const stepq_config *cfg, int layer, const float *w,
                                     const uint8_t *pivot_rows, const float *states, int n,
                                     double *acc, cudaStream_t s);
stepq_status launch_validate_slots(const int32_t *slots, int B, int pool_slots,
                                   uint32_t *scratch, int32_t *status, cudaStream_t s);
stepq_status launch_validate_slots_static(const int32_t *slots, int B, int pool_slots,
                                          int32_t *status, cudaStream_t s);
stepq_status read_device_error(cudaStream_t s);
unsigned int *device_error_word();   // address of the current device's sticky error word
// Test switch of the pipelined decode kernels (stepq_debug_stall): the bound of
// every wait in SM cycles and an item whose copies never start (-1: none).
struct StallKnob {
    long long wait_cycles;
    int withhold_item;
};
StallKnob stall_knob();
stepq_status set_stall_knob(long long wait_cycles, int withhold_item);

size_t intb_head_bytes(int bits);

}  // namespace stepq
