/*
 * stepq.h — C ABI of the STEPQuant decode-step library for one NVIDIA GB300
 * (sm_103a).
 *
 * The library implements the serving hot path of STEPQuant (arxiv 2609.38169):
 * the per-token gated Delta-rule decode step over a slot-indexed pool of
 * low-bit, mixed-precision, dual-axis-scaled recurrent states, together with
 * the offline plan (row-impact factors, lifetime-aware bit allocation, FP16
 * pivots, packed layout) and the calibration statistics that feed it.
 *
 * Conventions for every entry point
 *  - Orientation (Sec. 2.1): the state of one (layer, value head) is S in
 *    R^{d_k x d_v}; row i is key channel i, column j value channel j; dense
 *    states are row-major fp32. d_k = d_v = 128 (Table `config`).
 *  - GQA: value head h reads key head h / (n_value_heads / n_key_heads).
 *  - Device buffers are allocated and owned by the caller. Device calls are
 *    asynchronous on the given stream (NULL = legacy default stream), never
 *    synchronise and never allocate, so they can be captured in a CUDA graph
 *    (on a capturing stream) and replayed. Argument errors return before
 *    anything is launched. Slot ids found out of range by a kernel skip that unit and raise
 *    a sticky error readable with stepq_device_error().
 *  - Within one call slot ids must be distinct (two units writing one page race);
 *    stepq_validate_slots() checks a slot list on the device.
 *  - Plans are created on, and used with, the CUDA device current at creation.
 *  - Host arrays passed in are read during the call only.
 */
#ifndef STEPQ_H
#define STEPQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st *stepq_stream_t;   /* a cudaStream_t */

typedef enum {
    STEPQ_OK = 0,
    STEPQ_ERR_ARG = 1,          /* null pointer, bad size, enum or layer index */
    STEPQ_ERR_SLOT_RANGE = 2,   /* a slot id outside [0, pool_slots) (device-detected) */
    STEPQ_ERR_DUP_SLOT = 3,     /* a slot id repeated within one call */
    STEPQ_ERR_ALIGN = 4,        /* a buffer not aligned as documented */
    STEPQ_ERR_CUDA = 5,         /* a CUDA runtime call failed */
    STEPQ_ERR_BUDGET = 6,       /* the candidates cannot meet the bit budget */
    STEPQ_ERR_UNSUPPORTED = 7,  /* a configuration the library does not implement */
    STEPQ_ERR_TIMEOUT = 8       /* a bounded device-side wait gave up (device-detected) */
} stepq_status;

/* Gate kinds (Sec. 2.1): GDN's scalar gate D_t = alpha_t I, allocated per head;
 * KDA's channel-wise gate D_t = diag(d_t), allocated per key row (Sec. 3.2). */
#define STEPQ_GATE_SCALAR 0
#define STEPQ_GATE_CHANNEL 1

/* Bit-width code of an FP16 pivot unit (Sec. 3.2). */
#define STEPQ_PIVOT_BITS 16

typedef struct {
    int dk, dv;              /* must both be 128 */
    int n_layers;            /* recurrent layers held per slot page */
    int n_key_heads;
    int n_value_heads;       /* a multiple of n_key_heads */
    int gate_kind;           /* STEPQ_GATE_SCALAR (head units) or STEPQ_GATE_CHANNEL (row units) */
    int nominal_bits;        /* average code budget b (Eq. allocation): 4, 6 or 8 */
    int n_candidates;        /* 1..4 */
    int candidates[4];       /* distinct widths from {2, 4, 6, 8} (Table `config`) */
    int n_pivots;            /* FP16 pivot units, 0 <= n_pivots <= units */
    int horizon;             /* H of the lifetime weight L_u (Eq. calibration_lifetime) */
    int fit_iters;           /* fixed-code column updates per fit (App. C.1), >= 1 */
} stepq_config;

/* Calibration statistics (App. A.3), host arrays. Units are the allocation
 * units: n_layers*n_value_heads heads (scalar gate) or that times 128 key rows
 * (channel gate), ordered (layer, head[, row]). */
typedef struct {
    const float *omega;          /* [L][Hv][128] row-impact scores E[g_i^2] (Sec. 4.1) */
    const double *mean_log_ret;  /* [units] mean log retention ell_u */
    const double *distortion;    /* [units][n_candidates+1] per-element distortion d_u(b);
                                    last column: the FP16 reconstruction distortion */
    const uint8_t *pivot_mask;   /* [units] 1 = FP16 pivot, or NULL: chosen as in
                                    stepq_select_pivots from `distortion` */
} stepq_calib;

typedef struct stepq_plan stepq_plan;   /* opaque; owned by the library */

typedef struct {                        /* views into plan-owned host memory */
    size_t slot_stride;                 /* bytes per slot page (multiple of 256) */
    size_t n_units;
    const int8_t *unit_bits;            /* [units] 2/4/6/8, or 16 for an FP16 pivot */
    const uint8_t *pivot_mask;          /* [units] */
    const float *w;                     /* [L][Hv][128] row-impact factors w_i */
    const double *lifetime;             /* [units] L_u */
    const uint64_t *head_offset;        /* [L][Hv] byte offset of each head segment in a page */
    const uint32_t *head_bytes;         /* [L][Hv] bytes of each head segment */
} stepq_plan_info;

/* ---------------------------------------------------------------- offline plan
 * All host-side; deterministic for identical inputs. */

/* Number of allocation units of a configuration (0 if it is invalid). */
size_t stepq_num_units(const stepq_config *cfg);

/* Row-impact factors, footnote of Sec. 4.3 / Eq. kda_precond:
 * w_i = omega_i^(gamma/2) / GM_k(omega_k^(gamma/2)), gamma = 0.25, per head;
 * omega is floored at 1e-30. omega, w_out: host [L][Hv][128]. */
stepq_status stepq_row_weights(const stepq_config *cfg, const float *omega, float *w_out);

/* Lifetime weight L_u = sum_{j<H} exp(2 j ell_u) (Eq. calibration_lifetime). */
double stepq_lifetime_weight(double mean_log_ret, int horizon);

/* FP16 pivots (Sec. 3.2, Table `config`, App. C.2). Head units rank by the
 * residual allocation risk L_u d_u(b_u) of the pivot-free allocation; row
 * units by the lifetime-weighted reduction L_u (d_u(nominal) - d_u(FP16)).
 * The n_pivots highest risks win (ties: lower unit index).
 * pivot_mask_out: host [units]. */
stepq_status stepq_select_pivots(const stepq_config *cfg, const double *mean_log_ret,
                                 const double *distortion, uint8_t *pivot_mask_out);

/* Build the frozen plan (Sec. 3.2, Sec. 4.3, App. C.2, App. D): w from omega,
 * L_u, pivots, Lifetime-aware Bit Allocation (Eq. allocation: exact
 * multiple-choice DP for head units, Lagrangian with discrete repair for row
 * units; pivots count as 8-bit replacements), and the packed page layout. It
 * uploads the plan's device tables to the current device (this call
 * allocates and synchronises; it is offline). On a machine without a CUDA
 * device the plan is host-only: stepq_plan_query works, device calls with it
 * return STEPQ_ERR_CUDA. STEPQ_ERR_BUDGET if no assignment fits the budget. */
stepq_status stepq_fit_scales(const stepq_config *cfg, const stepq_calib *calib,
                              stepq_plan **plan_out);
stepq_status stepq_plan_query(const stepq_plan *plan, stepq_plan_info *info);
void stepq_plan_destroy(stepq_plan *plan);

/* ----------------------------------------------------------------- device path
 * Pool: device, pool_slots * slot_stride bytes, 256-byte aligned. Slot page s
 * starts at pool + s * slot_stride and holds every (layer, head) segment:
 *   integer head unit: r[128] fp16 | c[128] fp16 | codes in chunks: the 16
 *                      codes of band g (rows 16g..16g+15) in column j take 2b
 *                      bytes, chunk index ((j / 4) * 8 + g) * 4 + j % 4
 *   FP16 pivot head:   the same chunk order of fp16 values (32 bytes per chunk)
 *   row-unit head:     r[128] fp16 | c[128] fp16 | the rows, 16*b_i bytes each
 *                      (b_i = 16: fp16 row), stored by decreasing width, rows of
 *                      equal width in index order
 * Codes are offset binary u = q + 2^(b-1), packed LSB-first per row; row units
 * reconstruct with z = 2^(8-b_i) q (App. C.1).
 * layer: 0..L-1 for one layer, or -1 for every layer (quantize/dequantize only).
 * slots: device int32 [B]; B = 0 is a no-op. */

/* Fit and pack dense fp32 states into the pool (App. C.3 steps 4-7 without the
 * update; the prefill boundary). states: device [B][Hv][128][128] for one
 * layer, [B][L][Hv][128][128] for layer = -1. */
stepq_status stepq_quantize_pool(const stepq_plan *plan, int layer, const float *states,
                                 const int32_t *slots, int B, void *pool, int pool_slots,
                                 stepq_stream_t stream);

/* Reconstruct dense fp32 states X_hat_ij = r_i c_j z_ij (or the FP16 value),
 * rounded once to fp32. states_out: as for stepq_quantize_pool. */
stepq_status stepq_dequantize_pool(const stepq_plan *plan, int layer, const void *pool,
                                   int pool_slots, const int32_t *slots, int B,
                                   float *states_out, stepq_stream_t stream);

/* One persistent decode step of one layer for B slots (App. C.3 steps 1-7,
 * Eq. compressed_recurrence), fused into one kernel:
 *   X = D S_hat + beta k (v^T - k^T D S_hat),  y = X^T q  (read before requantization),
 *   then Key-Row-Aware Dual-axis Fitting and packed writeback in place.
 * q, k: device fp32 [B][Hk][128]; v: [B][Hv][128]; beta: [B][Hv];
 * gate: [B][Hv] (scalar) or [B][Hv][128] (channel); y: [B][Hv][128] out.
 * All 16-byte aligned. */
stepq_status stepq_decode_step(const stepq_plan *plan, int layer, void *pool, int pool_slots,
                               const int32_t *slots, int B, const float *q, const float *k,
                               const float *v, const float *beta, const float *gate, float *y,
                               stepq_stream_t stream);

/* Prefill of T tokens on FP32 states (the uncompressed side of the prefill
 * boundary, App. F: the chunk computation runs on the uncompressed state, which
 * stepq_quantize_pool then packs once). Evaluates the gated Delta rule
 * (Eq. delta_update) for every slot and value head over T tokens, 32 tokens at
 * a time in its chunkwise (WY) form, and writes every token's readout.
 * states: device fp32 [B][Hv][128][128], read as the state before the first
 *   token and overwritten with the state after the last (zero for a new
 *   sequence; stepq_dequantize_pool unpacks a stored one).
 * q, k: [B][T][Hk][128]; v: [B][T][Hv][128]; beta: [B][T][Hv]; gate:
 *   [B][T][Hv] (scalar) or [B][T][Hv][128] (channel), values in (0, 1]: the
 *   product of one chunk's gates must stay above 1e-30.
 * y: [B][T][Hv][128] out. Only dk, dv, heads and gate_kind of cfg are read;
 * all buffers 16-byte aligned. */
stepq_status stepq_prefill_fp32(const stepq_config *cfg, int B, int T, float *states,
                                const float *q, const float *k, const float *v,
                                const float *beta, const float *gate, float *y,
                                stepq_stream_t stream);

/* The decode step split in two for a side stream (Sec. 4.4, App. F.1: after the
 * readout, scale fitting and packed writeback run on a separate CUDA stream
 * while later layers process the token; writeback completes before the next
 * recurrent step reads the state). Head-unit and row-unit plans.
 *
 * stepq_decode_readout: App. C.3 steps 1-3 of stepq_decode_step: reconstruct,
 *   Delta update, readout. Writes y [B][Hv][128] and delta [B][Hv][128]
 *   (delta_j = v_j - k^T D S_hat, device fp32, 16-byte aligned) and leaves the
 *   pages unchanged. y is bit-identical to stepq_decode_step's.
 * stepq_decode_writeback: steps 4-7 in place: rebuilds the updated tile from
 *   the unchanged page, k, beta, gate and the readout's delta, refits and
 *   packs it. The page is byte-identical to the one stepq_decode_step writes.
 *   Order it after the readout of the same (layer, slots) (an event across
 *   streams) and before the next step that reads those pages.
 * Arguments and errors otherwise as for stepq_decode_step. */
stepq_status stepq_decode_readout(const stepq_plan *plan, int layer, const void *pool,
                                  int pool_slots, const int32_t *slots, int B, const float *q,
                                  const float *k, const float *v, const float *beta,
                                  const float *gate, float *y, float *delta,
                                  stepq_stream_t stream);
stepq_status stepq_decode_writeback(const stepq_plan *plan, int layer, void *pool, int pool_slots,
                                    const int32_t *slots, int B, const float *k,
                                    const float *beta, const float *gate, const float *delta,
                                    stepq_stream_t stream);

/* --------------------------------------------------- comparison kernels (same build)
 * FP32-state decode (the serving default the paper compares against, Sec. 5.1):
 * pool: device fp32 [pool_slots][L][Hv][128][128]; the step updates the layer's
 * states in place and writes y. Only dk, dv, n_layers, heads and gate_kind of
 * cfg are read. */
stepq_status stepq_fp32_decode_step(const stepq_config *cfg, int layer, float *pool,
                                    int pool_slots, const int32_t *slots, int B, const float *q,
                                    const float *k, const float *v, const float *beta,
                                    const float *gate, float *y, stepq_stream_t stream);

/* The exact-read counterpart of stepq_fp32_decode_step used by the feedback
 * experiment of App. B.1 ("exact-read oracle"): the retrieval reads the
 * reference states, u = k^T D S_ref with S_ref from read_pool (same layout as
 * pool, not modified), while the update writes D S + beta k (v - u)^T into
 * pool. A state error E = S - S_ref then evolves as D E, without the Delta
 * rule's own correction (Eq. self_correction). */
stepq_status stepq_fp32_exact_read_step(const stepq_config *cfg, int layer, float *pool,
                                        const float *read_pool, int pool_slots,
                                        const int32_t *slots, int B, const float *q,
                                        const float *k, const float *v, const float *beta,
                                        const float *gate, float *y, stepq_stream_t stream);

/* "Temporal only" ablation state (Sec. 5.4): the plan's calibrated widths
 * and FP16 pivots, with the uniform rowwise quantizer of App. B.5 in place of
 * the dual-axis fit. A key row of width b < 16 stores s_i = fp16(clamp(
 * absmax_i / q_b, 2^-14, 65504)) and nearest codes of X * fp32(1/s_i) in
 * [-q_b, q_b] (offset-binary, LSB-first); a pivot row stores fp16(X) with
 * s_i = 0. Head segment: s[128] fp16 | row i in index order, 16 b_i bytes;
 * segments in (layer, head) order; slot stride = stepq_temporal_slot_bytes()
 * (a multiple of 256; 0 for a null plan). States, slots, layer = -1 and the
 * errors behave as in stepq_quantize_pool / stepq_dequantize_pool. A decode
 * step with this codec is dequantize, stepq_fp32_decode_step, quantize: it
 * serves accuracy ablations and has no fused kernel. */
size_t stepq_temporal_slot_bytes(const stepq_plan *plan);
stepq_status stepq_temporal_quantize_pool(const stepq_plan *plan, int layer, const float *states,
                                          const int32_t *slots, int B, void *pool, int pool_slots,
                                          stepq_stream_t stream);
stepq_status stepq_temporal_dequantize_pool(const stepq_plan *plan, int layer, const void *pool,
                                            int pool_slots, const int32_t *slots, int B,
                                            float *states_out, stepq_stream_t stream);

/* Uniform rowwise-absmax INT-b state (App. B.5): per key row an FP16 scale
 * absmax/q_b clamped to [2^-14, 65504], nearest codes in [-q_b, q_b]. Head
 * segment: s[128] fp16 | 128 rows x 16b bytes; segments in (layer, head)
 * order; slot stride = stepq_intb_slot_bytes(). bits: 4, 6 or 8 (codes
 * offset-binary, LSB-first along the row); other widths give 0 bytes and
 * STEPQ_ERR_UNSUPPORTED. */
size_t stepq_intb_slot_bytes(const stepq_config *cfg, int bits);
stepq_status stepq_intb_quantize_pool(const stepq_config *cfg, int bits, int layer,
                                      const float *states, const int32_t *slots, int B,
                                      void *pool, int pool_slots, stepq_stream_t stream);
stepq_status stepq_intb_dequantize_pool(const stepq_config *cfg, int bits, int layer,
                                        const void *pool, int pool_slots, const int32_t *slots,
                                        int B, float *states_out, stepq_stream_t stream);
stepq_status stepq_intb_decode_step(const stepq_config *cfg, int bits, int layer, void *pool,
                                    int pool_slots, const int32_t *slots, int B, const float *q,
                                    const float *k, const float *v, const float *beta,
                                    const float *gate, float *y, stepq_stream_t stream);

/* ------------------------------------------------------------- calibration (App. A.3)
 * Accumulate sum_t g_{t,i}^2 with g_t = A_t^T q_t (Sec. 4.1, Eq.
 * kda_sensitivity) and sum_t log r_{t,u} for n calibration tokens of one layer.
 * Inputs shaped as for stepq_decode_step with B = n. omega_sum: device fp64
 * [L][Hv][128]; logret_sum: device fp64 [units]. */
stepq_status stepq_calib_observe(const stepq_config *cfg, int layer, const float *q,
                                 const float *k, const float *beta, const float *gate, int n,
                                 double *omega_sum, double *logret_sum, stepq_stream_t stream);

/* Accumulate candidate distortions of n sampled reference states of one layer
 * (Eqs. qwen_calibration_distortion, kda_calibration_distortion): each state
 * head is fitted at every candidate width (uniform over the head) with the
 * dual-axis codec; head units add the w^2-weighted per-element MSE, row units
 * the per-row MSE; the last column adds the FP16 error. pivot_rows (device
 * [units] or NULL, row units only) keeps those rows in FP16 and out of the
 * column fit. w: device fp32 [L][Hv][128]; states: device [n][Hv][128][128];
 * acc: device fp64 [units][n_candidates+1] (sums; divide by the sample count). */
stepq_status stepq_calib_distortion(const stepq_config *cfg, int layer, const float *w,
                                    const uint8_t *pivot_rows, const float *states, int n,
                                    double *acc, stepq_stream_t stream);

/* The whole calibration protocol of App. A.3 on a recorded trace, behind one
 * call (the sequence of stepq_calib_observe, FP32-state replay and
 * stepq_calib_distortion launches, the means and the pivot choice):
 *   pass A  omega_i = mean_t g_{t,i}^2 (Sec. 4.1) and ell_u = mean_t log r_{t,u}
 *           (Eq. calibration_lifetime) over the n * T tokens of every layer;
 *   pass B  per layer, the FP32-state recurrence replayed from a zero state over
 *           the T tokens of each sequence; every `every`-th state is fitted at
 *           each candidate width (Eqs. qwen_calibration_distortion,
 *           kda_calibration_distortion), one sample per sequence, and
 *           d_u(b) is the mean over the samples;
 *   pivots  as stepq_select_pivots from ell and the pass-B distortions; row
 *           units then repeat pass B with the chosen pivot rows kept in FP16 and
 *           out of the column fit (App. C.2), and that second measurement is
 *           the `distortion` the plan takes.
 * Trace, device fp32 (16-byte aligned; beta 4-byte): q, k [L][T][n][Hk][128];
 * v [L][T][n][Hv][128]; beta [L][T][n][Hv]; gate [L][T][n][Hv] (scalar) or
 * [L][T][n][Hv][128] (channel). workspace: device, 256-byte aligned, at least
 * stepq_calib_workspace_bytes(cfg, n) bytes (contents clobbered). The result
 * arrays are host memory the caller owns, written before the call returns.
 * This is an offline call: it synchronises `stream` and allocates nothing. */
typedef struct {
    float *omega;               /* out [L][Hv][128] */
    double *mean_log_ret;       /* out [units] */
    double *distortion;         /* out [units][n_candidates+1], last column FP16 */
    double *distortion_stage1;  /* out [units][n_candidates+1] of the first pass, or NULL */
    uint8_t *pivot_mask;        /* out [units] */
    int n_tokens, n_samples;    /* out: tokens per layer (n T) and samples per layer */
} stepq_calib_result;
size_t stepq_calib_workspace_bytes(const stepq_config *cfg, int n);
stepq_status stepq_calibrate_from_trace(const stepq_config *cfg, int n, int T, int every,
                                        const float *q, const float *k, const float *v,
                                        const float *beta, const float *gate, void *workspace,
                                        size_t workspace_bytes, stepq_calib_result *out,
                                        stepq_stream_t stream);

/* ----------------------------------------------------------------- diagnostics */
/* Check on the device that slots[0..B) are distinct and in [0, pool_slots).
 * scratch: device, >= (pool_slots + 31) / 32 uint32 words (contents clobbered).
 * status_out: device int32, set to STEPQ_OK / STEPQ_ERR_SLOT_RANGE / STEPQ_ERR_DUP_SLOT. */
stepq_status stepq_validate_slots(const int32_t *slots, int B, int pool_slots, uint32_t *scratch,
                                  int32_t *status_out, stepq_stream_t stream);

/* The same check for callers that cannot allocate device memory and have no
 * spare scratch buffer to pass -- for example code running where a host
 * framework owns every device allocation, or on a path where cudaMalloc's
 * implicit synchronisation is not acceptable. The paper has no counterpart;
 * this entry point allocates nothing.
 * The bitmap lives in a file-scope device array sized for pool_slots up to
 * 1,048,576 (128 KiB, kept by every GPU that loads the library until the
 * process exits); larger pools return STEPQ_ERR_UNSUPPORTED before any work.
 * The first call on a device looks up the array's device address (set-up that
 * should happen before any stream capture). Every call shares the array and
 * clears the part it uses first; calls that overlap on the GPU race with each
 * other. status_out: device int32, as for stepq_validate_slots. */
stepq_status stepq_validate_slots_noalloc(const int32_t *slots, int B, int pool_slots,
                                          int32_t *status_out, stepq_stream_t stream);

/* Read and clear the sticky device error of the current device (synchronises
 * `stream`): STEPQ_OK, or the first error a kernel raised. */
stepq_status stepq_device_error(stepq_stream_t stream);
/* The same read-and-clear of the sticky device error under a second name:
 * surfaces what the asynchronous calls queued on `stream` reported.
 * Synchronises `stream`. */
stepq_status stepq_stream_status(stepq_stream_t stream);

/* Test support for the bounded waits (not for production use). Every wait of
 * the pipelined decode kernels (stepq_decode_step, the split halves, the FP32
 * and INT-b decode steps) gives up after `wait_cycles` SM clock cycles
 * (default 2e9, about one second; at least 1000), raises STEPQ_ERR_TIMEOUT and
 * lets its CTA return. withhold_item >= 0 makes every later launch skip the
 * copies of that item (head * B + batch entry), so that its wait runs out and
 * the launch reports STEPQ_ERR_TIMEOUT with its results undefined; -1 restores
 * normal operation. The values are process-wide, read at each launch, and not
 * safe to change while another thread launches. STEPQ_ERR_ARG for values out of
 * range. The paper has no counterpart; this exists to test failure detection. */
stepq_status stepq_debug_stall(long long wait_cycles, int withhold_item);

const char *stepq_status_str(stepq_status s);
const char *stepq_version(void);

#ifdef __cplusplus
}
#endif
#endif /* STEPQ_H */
