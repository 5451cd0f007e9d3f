/*
 * gas_fp8.h — the consumer side of a per-layer FP8 scale on one GB300 (sm_103a).
 *
 * The scale of gas.h is used in Stage 3 of Algorithm 1: the attention logits S of a
 * layer are divided by the layer's scale and cast to FP8 E4M3 (largest finite value
 * R_max = 448, Section 1).  This header covers that cast and the bookkeeping around it:
 *
 *   gas_fp8_quantize        S~ = S / scale, E4M3 codes, and the per-call statistics
 *                           Table 4 reports per layer: the largest scaled logit
 *                           ("Max Scaled") and the number of scaled logits beyond 448
 *                           (a layer overflows when that number is not zero).
 *   gas_fp8_delayed_scales  the delayed-scaling comparator of Eq. 1,
 *                           scale_t = max(history) / (448 eta), from a per-layer
 *                           history of observed maxima (16 steps, initialised to 1.0,
 *                           eta = 0.9 in Appendix G).
 *   gas_fp8_end_step        pushes each layer's observed maximum of the step into the
 *                           history and, during an auto-alpha burn-in, records the
 *                           slack ratio r_t = max|S^(t)| / B_max^(t) of Eq. 16,
 *                           B_max = sigma_l d / sqrt(d_h) (Section 3.5).
 *   gas_fp8_auto_alpha      Algorithm 4: alpha_final = Quantile_q(R) * kappa.
 *
 * E4M3 here is the format with 1 sign, 4 exponent (bias 7) and 3 mantissa bits, no
 * infinities, NaN = S.1111.111 (code 0x7F is the only NaN this library writes).
 * Rounding is to nearest, ties to even.  S / scale is one float32 division (IEEE,
 * round to nearest).  An element "overflows" when its scaled value is NaN or of
 * magnitude above 448; it is then written as +-448 (GAS_FP8_SATURATE) or as NaN.
 * The sign of zero is kept (-0.0 -> 0x80).
 *
 * Conventions: as gas.h (caller-owned buffers, asynchronous stream-ordered calls, host
 * argument checks that enqueue nothing on error, no exceptions).  A handle is not
 * thread-safe: calls on one handle must not overlap on the GPU.
 */
#ifndef GAS_FP8_H_
#define GAS_FP8_H_

#include "gas.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef struct gas_fp8_ctx *gas_fp8_handle;

/* Statistics of one gas_fp8_quantize call (written to device memory). */
typedef struct gas_fp8_stats {
    float amax;                   /* max |S| over the call's elements; NaN if any S is NaN;
                                     0 for an empty call */
    float max_scaled;             /* amax / scale in float32: the largest scaled logit */
    unsigned long long overflow;  /* elements whose S / scale is NaN or beyond +-448 */
    unsigned long long count;     /* elements quantised */
} gas_fp8_stats;

/* GAS_DTYPE_BF16 / GAS_DTYPE_F32 logits (defined in gas.h). */

#define GAS_FP8_SATURATE 0x1      /* overflowing elements become +-448 (else NaN, 0x7F) */

/* Largest slack buffer (burn-in steps x layers) gas_fp8_auto_alpha sorts on chip. */
#define GAS_FP8_MAX_SLACK 16384

/*
 * Create the per-model state: for every layer a ring of `history_len` observed maxima
 * (initialised to 1.0, Appendix G) and the maximum observed in the current step;
 * a slack buffer of `burn_in_steps` x `layers` ratios for auto-alpha (0: none).
 * Allocates device memory on the current device; synchronous.
 * Errors: layers < 1 or > 512, history_len < 1 or > 1024, burn_in_steps < 0,
 * burn_in_steps * layers > GAS_FP8_MAX_SLACK -> GAS_ERR_INVALID_ARG / GAS_ERR_UNSUPPORTED;
 * no device -> GAS_ERR_CUDA; out of memory -> GAS_ERR_ALLOC.  Message: gas_fp8_last_error(NULL).
 */
gas_status gas_fp8_create(int layers, int history_len, int burn_in_steps, gas_fp8_handle *out);
gas_status gas_fp8_destroy(gas_fp8_handle h);

/* Refill every history entry with `history_init` (a fresh buffer after loading a
 * checkpoint, Section 5.2), clear the step maxima and the slack buffer. */
gas_status gas_fp8_reset(gas_fp8_handle h, float history_init, void *stream);

/*
 * Eq. 1 for every layer: scale_out[l] = max_j history[l][j] / float32(448 * eta),
 * a float32 division; NaN in the history gives a NaN scale.
 * scale_out: device [layers], 4-byte aligned.  Errors: eta <= 0 -> GAS_ERR_INVALID_ARG.
 */
gas_status gas_fp8_delayed_scales(gas_fp8_handle h, double eta, float *scale_out, void *stream);

/*
 * Algorithm 1, Stage 3 on one layer's logits.
 *   layer    which layer's step maximum the call's amax is merged into (max over the
 *            calls of a step; gas_fp8_end_step consumes it).
 *   s        device, n elements of `dtype` (GAS_DTYPE_BF16 or GAS_DTYPE_F32), 16-byte
 *            aligned, any logical shape (e.g. [batch][heads][T][T]) flattened.
 *   scale    device pointer to the layer's scale (one float; e.g. &s_out[l] of gas_refresh
 *            or of gas_fp8_delayed_scales), read on the device.
 *   q_out    device, n bytes of E4M3 codes in the same order, 16-byte aligned; NULL =
 *            statistics only.
 *   flags    GAS_FP8_SATURATE or 0.
 *   stats    device, one gas_fp8_stats (8-byte aligned), written when the call completes.
 * n = 0 is allowed (stats {0, 0/scale, 0, 0}).  Concurrent calls for the same layer race.
 * Errors: bad layer, null or misaligned pointers, n < 0, unknown dtype -> GAS_ERR_INVALID_ARG.
 */
gas_status gas_fp8_quantize(gas_fp8_handle h, int layer, const void *s, int dtype, long long n,
                            const float *scale, unsigned char *q_out, int flags, gas_fp8_stats *stats,
                            void *stream);

/*
 * Close a step: history[l] <- the step maximum of layer l (a layer with no quantize
 * call this step pushes 0), then clear the step maxima.  When `sigma` is not NULL and
 * the slack buffer has room, also append r_l = amax_l / (sigma_l * float32(d / sqrt(d_h)))
 * (Eq. 16, float32; sigma_l = max over the layer's n_q heads, NaN-propagating) for every
 * layer.  sigma: device [layers][n_q] (the per-head output of gas_spectral_norms /
 * gas_refresh).  Errors: n_q, d or d_h < 1 -> GAS_ERR_INVALID_ARG.
 */
gas_status gas_fp8_end_step(gas_fp8_handle h, const float *sigma, int n_q, int d, int d_h, void *stream);

/*
 * Algorithm 4: alpha_out[0] = Quantile_q(R) * kappa over the finite slack ratios
 * recorded so far (NaN when there are none); the quantile interpolates linearly between
 * order statistics at position q (m - 1) of the m sorted values, in float64, rounded to
 * float32 at the end.  alpha_out: device, one float.
 * Errors: q outside [0, 1], kappa <= 0 -> GAS_ERR_INVALID_ARG.
 */
gas_status gas_fp8_auto_alpha(gas_fp8_handle h, double q, double kappa, float *alpha_out, void *stream);

/* Number of slack ratios recorded (steps x layers, capped at the buffer size); synchronises. */
gas_status gas_fp8_slack_count(gas_fp8_handle h, int *count);

/* Message for the last error on this handle (or the last gas_fp8_create failure when NULL). */
const char *gas_fp8_last_error(gas_fp8_handle h);

#ifdef __cplusplus
}
#endif

#endif /* GAS_FP8_H_ */
