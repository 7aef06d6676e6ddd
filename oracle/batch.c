/*
 * Oracle (test infrastructure only): pool-level drivers. A slot page holds
 * every (layer, head) segment of one request; a decode step of one layer
 * touches the segment of each (slot, head) independently (App. F.1), so these
 * loops run those units in parallel with OpenMP and nothing else.
 *
 * Per-layer arguments: layer_row_bits [Hv][128] (a head unit repeats its width
 * on every row), layer_w [Hv][128], layer_head_off [Hv] (byte offset of the
 * head segment inside a slot page).
 */
#include <stdlib.h>
#include "oracle.h"

static uint8_t *page_of(uint8_t *pool, const int32_t *slots, int b, uint64_t stride,
                        const uint64_t *head_off, int h)
{
    return pool + (uint64_t)slots[b] * stride + head_off[h];
}

void or_pool_encode(int unit_kind, int Hv, const int8_t *layer_row_bits, const float *layer_w,
                    int fit_iters, const uint64_t *layer_head_off, uint64_t slot_stride,
                    uint8_t *pool, const int32_t *slots, int B, const float *states)
{
#pragma omp parallel for collapse(2) schedule(dynamic)
    for (int b = 0; b < B; b++)
        for (int h = 0; h < Hv; h++)
            or_encode_head(states + ((size_t)b * Hv + h) * OR_N, unit_kind,
                           layer_row_bits + (size_t)h * OR_D, layer_w + (size_t)h * OR_D,
                           fit_iters, page_of(pool, slots, b, slot_stride, layer_head_off, h));
}

void or_pool_decode(int unit_kind, int Hv, const int8_t *layer_row_bits,
                    const uint64_t *layer_head_off, uint64_t slot_stride,
                    const uint8_t *pool, const int32_t *slots, int B, float *states)
{
#pragma omp parallel for collapse(2) schedule(dynamic)
    for (int b = 0; b < B; b++)
        for (int h = 0; h < Hv; h++)
            or_decode_head_f32(page_of((uint8_t *)pool, slots, b, slot_stride, layer_head_off, h),
                               unit_kind, layer_row_bits + (size_t)h * OR_D,
                               states + ((size_t)b * Hv + h) * OR_N);
}

static void step_one(int unit_kind, int Hk, int Hv, int gate_per_row,
                     const int8_t *layer_row_bits, const float *layer_w, int fit_iters,
                     const uint64_t *layer_head_off, uint64_t slot_stride, uint8_t *pool,
                     const int32_t *slots, int b, int h, const float *q, const float *k,
                     const float *v, const float *beta, const float *gate, float *y, double *delta)
{
    int hk = h / (Hv / Hk);
    const float *g = gate_per_row ? gate + ((size_t)b * Hv + h) * OR_D : gate + (size_t)b * Hv + h;
    or_step_head(page_of(pool, slots, b, slot_stride, layer_head_off, h), unit_kind,
                 layer_row_bits + (size_t)h * OR_D, layer_w + (size_t)h * OR_D, fit_iters,
                 q + ((size_t)b * Hk + hk) * OR_D, k + ((size_t)b * Hk + hk) * OR_D,
                 v + ((size_t)b * Hv + h) * OR_D, beta[(size_t)b * Hv + h], g, gate_per_row,
                 y + ((size_t)b * Hv + h) * OR_D, delta ? delta + ((size_t)b * Hv + h) * OR_D : NULL);
}

void or_pool_step(int unit_kind, int Hk, int Hv, int gate_per_row, const int8_t *layer_row_bits,
                  const float *layer_w, int fit_iters, const uint64_t *layer_head_off,
                  uint64_t slot_stride, uint8_t *pool, const int32_t *slots, int B,
                  const float *q, const float *k, const float *v, const float *beta,
                  const float *gate, float *y, double *delta)
{
#pragma omp parallel for collapse(2) schedule(dynamic)
    for (int b = 0; b < B; b++)
        for (int h = 0; h < Hv; h++)
            step_one(unit_kind, Hk, Hv, gate_per_row, layer_row_bits, layer_w, fit_iters,
                     layer_head_off, slot_stride, pool, slots, b, h, q, k, v, beta, gate, y, delta);
}

/* Only the listed (batch index, head) units; the rest of the pool is untouched. */
void or_pool_step_units(int unit_kind, int Hk, int Hv, int gate_per_row,
                        const int8_t *layer_row_bits, const float *layer_w, int fit_iters,
                        const uint64_t *layer_head_off, uint64_t slot_stride, uint8_t *pool,
                        const int32_t *slots, int n_units, const int32_t *unit_b,
                        const int32_t *unit_h, const float *q, const float *k, const float *v,
                        const float *beta, const float *gate, float *y)
{
#pragma omp parallel for schedule(dynamic)
    for (int t = 0; t < n_units; t++)
        step_one(unit_kind, Hk, Hv, gate_per_row, layer_row_bits, layer_w, fit_iters,
                 layer_head_off, slot_stride, pool, slots, unit_b[t], unit_h[t], q, k, v, beta,
                 gate, y, NULL);
}

/* Uniform INT-b pool: head h of the layer at layer_off + h * head_bytes. */
void or_intb_pool_step(int bits, int Hk, int Hv, int gate_per_row, uint64_t layer_off,
                       uint64_t slot_stride, uint8_t *pool, const int32_t *slots, int B,
                       const float *q, const float *k, const float *v, const float *beta,
                       const float *gate, float *y)
{
    size_t hb = or_intb_head_bytes(bits);
#pragma omp parallel for collapse(2) schedule(dynamic)
    for (int b = 0; b < B; b++)
        for (int h = 0; h < Hv; h++) {
            int hk = h / (Hv / Hk);
            const float *g = gate_per_row ? gate + ((size_t)b * Hv + h) * OR_D
                                          : gate + (size_t)b * Hv + h;
            or_intb_step_head(pool + (uint64_t)slots[b] * slot_stride + layer_off + h * hb, bits,
                              q + ((size_t)b * Hk + hk) * OR_D, k + ((size_t)b * Hk + hk) * OR_D,
                              v + ((size_t)b * Hv + h) * OR_D, beta[(size_t)b * Hv + h], g,
                              gate_per_row, y + ((size_t)b * Hv + h) * OR_D);
        }
}
