/*
 * STEPQuant CPU oracle — TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow restatement of the paper's decode-step method (arxiv
 * 2609.38169, "STEPQuant: When and Where Errors Matter in Delta-Rule Recurrent
 * State Quantization"), used to check the CUDA library. Only the tests, the
 * package's smoke check and the timing script's CPU-baseline leg may load it.
 * It shares no code with the CUDA library.
 *
 * Arithmetic is fp64 (scalar loops, no blocking or fusion). Quantities the
 * method stores or decides on are rounded at the points where the state format
 * materialises them: the updated state tile X in fp32, the readout y in fp32,
 * the row/column scales and FP16 pivots in binary16, and each quantization
 * decision taken on fp32 operands (the precision of the GPU tile).
 *
 * State orientation (Sec. 2.1): S is d_k x d_v, row i = key channel, column j =
 * value channel, stored row-major.
 *
 * Parity pins: every function here is pinned by tests under tests/ (closed
 * forms, identities of Sec. 2.1 / Prop. 1 / App. B.1 / App. B.3, brute force on
 * tiny inputs, the byte counts of App. D). The paper prints no fitted scale
 * value; the fit is pinned step by step (the smallest clip-free column start,
 * nearest codes, the fixed-code update as the 1-D minimiser of the weighted
 * error, the row factors' scaling laws).
 */
#ifndef STEPQ_ORACLE_H
#define STEPQ_ORACLE_H

#include <stddef.h>
#include <stdint.h>

#define OR_D 128              /* d_k = d_v = 128 (Table `config`) */
#define OR_N (OR_D * OR_D)
#define OR_PIVOT_BITS 16      /* bit-width code meaning "stored in FP16" */

/* unit kinds: a whole head (GDN / Qwen) or a key row (KDA), Sec. 3.2 */
#define OR_UNIT_HEAD 0
#define OR_UNIT_ROW 1

#ifdef __cplusplus
extern "C" {
#endif

/* ---- numerics.c: binary16 ---- */
double or_fp16_round(double x);          /* RNE to binary16, saturating at +-65504 */
uint16_t or_fp16_encode(double v);       /* bits of a binary16-representable value */
double or_fp16_decode(uint16_t h);

/* ---- recurrence.c: Eq. delta_update (FP32-state reference) ---- */
void or_delta_step_f32(float *S, const float *q, const float *k, const float *v,
                       float beta, const float *gate, int gate_per_row, float *y);
void or_delta_batch_f32(int n, int Hk, int Hv, int gate_per_row, float *S,
                        const float *q, const float *k, const float *v,
                        const float *beta, const float *gate, float *y);
void or_delta_step_read_f32(float *S, const float *Sref, const float *q, const float *k,
                            const float *v, float beta, const float *gate, int gate_per_row,
                            float *y);
void or_delta_batch_read_f32(int n, int Hk, int Hv, int gate_per_row, float *S, const float *Sref,
                             const float *q, const float *k, const float *v,
                             const float *beta, const float *gate, float *y);
void or_row_impact(const float *q, const float *k, float beta, const float *gate,
                   int gate_per_row, double *g);
void or_row_impact_dense(const float *q, const float *k, float beta, const float *gate,
                         int gate_per_row, double *g);

/* ---- codec.c: Key-Row-Aware Dual-axis Fitting (Sec. 4.3, App. C.1/C.3) ---- */
size_t or_head_bytes(int unit_kind, const int8_t *row_bits);
void or_encode_head(const float *X, int unit_kind, const int8_t *row_bits,
                    const float *w, int fit_iters, uint8_t *page);
void or_decode_head(const uint8_t *page, int unit_kind, const int8_t *row_bits, double *S);
void or_decode_head_f32(const uint8_t *page, int unit_kind, const int8_t *row_bits, float *S);
void or_step_head(uint8_t *page, int unit_kind, const int8_t *row_bits, const float *w,
                  int fit_iters, const float *q, const float *k, const float *v,
                  float beta, const float *gate, int gate_per_row, float *y, double *delta);
void or_fit_debug(const float *X, int unit_kind, const int8_t *row_bits, const float *w,
                  int fit_iters, double *r, double *c_iter, int8_t *z_last);
void or_unpack_head(const uint8_t *page, int unit_kind, const int8_t *row_bits,
                    uint16_t *r, uint16_t *c, int8_t *codes, uint16_t *piv);

/* uniform rowwise-absmax INT-b baseline (App. B.5 / Sec. 5.1) */
size_t or_intb_head_bytes(int bits);
void or_intb_encode_head(const float *X, int bits, uint8_t *page);
void or_intb_decode_head(const uint8_t *page, int bits, double *S);
size_t or_temporal_head_bytes(const int8_t *rb);
void or_temporal_encode_head(const float *X, const int8_t *rb, uint8_t *page);
void or_temporal_decode_head(const uint8_t *page, const int8_t *rb, double *S);
void or_intb_step_head(uint8_t *page, int bits, const float *q, const float *k, const float *v,
                       float beta, const float *gate, int gate_per_row, float *y);

/* ---- plan.c: Lifetime-aware Bit Allocation (Sec. 3.2, App. C.2, App. D) ---- */
void or_row_weights(int n_heads, const float *omega, float *w);
double or_lifetime_weight(double ell, int H);
int or_allocate_dp(int n_units, int n_cand, const int *cands, long long capacity_half_bits,
                   const double *cost, int8_t *choice);
int or_allocate_lagrangian(int n_units, int n_cand, const int *cands, long long budget_bits,
                           const double *cost, int8_t *choice);
double or_lagrangian_multiplier(int n_units, int n_cand, const int *cands, long long budget_bits,
                                const double *cost);
int or_select_pivots(int unit_kind, int n_units, int n_cand, const int *cands, int nominal,
                     const double *L, const double *dist, int n_pivots, uint8_t *pivot);
int or_allocate(int unit_kind, int n_units, int n_cand, const int *cands, int nominal,
                const double *L, const double *dist, const uint8_t *pivot, int8_t *bits);
int or_layout(int unit_kind, int n_layers, int Hv, const int8_t *unit_bits,
              uint64_t *head_off, uint32_t *head_bytes, uint64_t *slot_stride);

/* ---- batch.c: pool-level drivers (OpenMP over independent (slot, head) units) ---- */
void or_pool_encode(int unit_kind, int Hv, const int8_t *layer_row_bits, const float *layer_w,
                    int fit_iters, const uint64_t *layer_head_off, uint64_t slot_stride,
                    uint8_t *pool, const int32_t *slots, int B, const float *states);
void or_pool_decode(int unit_kind, int Hv, const int8_t *layer_row_bits,
                    const uint64_t *layer_head_off, uint64_t slot_stride,
                    const uint8_t *pool, const int32_t *slots, int B, float *states);
void or_pool_step(int unit_kind, int Hk, int Hv, int gate_per_row, const int8_t *layer_row_bits,
                  const float *layer_w, int fit_iters, const uint64_t *layer_head_off,
                  uint64_t slot_stride, uint8_t *pool, const int32_t *slots, int B,
                  const float *q, const float *k, const float *v, const float *beta,
                  const float *gate, float *y,
                  double *delta);
void or_pool_step_units(int unit_kind, int Hk, int Hv, int gate_per_row,
                        const int8_t *layer_row_bits, const float *layer_w, int fit_iters,
                        const uint64_t *layer_head_off, uint64_t slot_stride, uint8_t *pool,
                        const int32_t *slots, int n_units, const int32_t *unit_b,
                        const int32_t *unit_h, const float *q, const float *k, const float *v,
                        const float *beta, const float *gate, float *y);
void or_intb_pool_step(int bits, int Hk, int Hv, int gate_per_row, uint64_t layer_off,
                       uint64_t slot_stride, uint8_t *pool, const int32_t *slots, int B,
                       const float *q, const float *k, const float *v, const float *beta,
                       const float *gate, float *y);

/* ---- calib.c: calibration statistics (App. A.3) ---- */
void or_calib_observe(int n, int Hk, int Hv, int gate_per_row, const float *q,
                      const float *k, const float *beta, const float *gate,
                      double *omega_sum, double *logret_sum);
void or_calib_distortion(int n, int Hv, int unit_kind, const float *states, const float *w_layer,
                         int n_cand, const int *cands, const uint8_t *pivot_rows_layer,
                         int fit_iters, double *acc);
int or_num_threads(void);

#ifdef __cplusplus
}
#endif
#endif
