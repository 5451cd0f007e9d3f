/*
 * gas.h — geometry-aware FP8 attention scales on one GB300 (sm_103a).
 *
 * For every query head h of every layer l this library computes the spectral norm
 *     sigma_{l,h} = || W^Q_h W^K_{g(h)}^T ||_2            (paper, Eq. 4 and Eq. 7)
 * by implicit power iteration (Section 4.1, Algorithm 2): the d x d interaction
 * matrix is never formed, and under grouped-query attention the shared key block
 * W^K_g is read unexpanded (Section 4.2, Algorithm 3, Proposition 4.1).  From the
 * per-head sigmas it evaluates the per-layer geometry-aware scale (Section 3.4, Eq. 15)
 *     scale_l = alpha * max_h sigma_{l,h} * (d / sqrt(d_h)) / (eta_fp8 * R_max),
 * with alpha >= alpha_min from Eq. 13 and the typicality gamma from Eq. 12.
 *
 * Conventions shared by every entry point
 *  - Weights use the nn.Linear layout, bf16, row-major, one pointer per layer:
 *      Wq[l] : [n_q  * d_h, d]   rows h*d_h .. h*d_h+d_h-1 are (W^Q_h)^T
 *      Wk[l] : [n_kv * d_h, d]   rows g*d_h .. are (W^K_g)^T
 *    contiguous by default; gas_set_weight_layout describes padded rows and
 *    per-head-interleaved (fused projection) storage.  Query head h uses KV group
 *    g(h) = h / (n_q / n_kv) (RepeatBlocks order, Appendix F).  Each layer pointer
 *    must be 16-byte aligned.
 *  - Vectors are fp32, [layers][n_q][d] contiguous, 16-byte aligned.
 *  - The caller owns every buffer passed in.  The handle owns only its workspace
 *    (device memory sized at gas_create) and cached TMA descriptors.
 *  - Calls that take a stream are asynchronous and stream-ordered; the host checks
 *    arguments synchronously and enqueues nothing on error.  `stream` is a
 *    cudaStream_t (NULL = legacy default stream).
 *  - CUDA graphs: the first call with a new set of weight pointers (or after
 *    gas_set_weight_layout) builds their TMA descriptors and synchronises the stream
 *    once to upload them; every later call with the same pointers is pure stream work
 *    and can be captured (cudaStreamBeginCapture) and replayed.  Replays read the
 *    weights and v_in afresh; the fused kernel's key-tile flags take a new value on
 *    every replay (advanced on the device), so replays never see stale Gram blocks.
 *  - No exceptions cross this boundary.  A handle is not thread-safe; concurrent
 *    calls on one handle (or overlapping launches of one handle on two streams)
 *    race on its workspace.
 *  - Device-side failures (a bounded wait that ran out, a NaN/Inf sigma) set bits
 *    in a device status word read by gas_get_device_status; kernels never trap
 *    and never wait without a limit.
 */
#ifndef GAS_H_
#define GAS_H_

#include <stddef.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct gas_ctx *gas_handle;

typedef enum {
    GAS_OK = 0,
    GAS_ERR_INVALID_ARG = 1,   /* null/misaligned pointer, bad count, gamma in (0,1] ... */
    GAS_ERR_UNSUPPORTED = 2,   /* shape outside what the kernels implement */
    GAS_ERR_CUDA = 3,          /* a CUDA runtime/driver call failed (see gas_last_error) */
    GAS_ERR_ALLOC = 4,         /* workspace allocation failed */
    GAS_ERR_DEVICE_TIMEOUT = 5 /* a device-side bounded wait ran out (status word) */
} gas_status;

/* Device status word bits (gas_get_device_status). */
#define GAS_DEV_NONFINITE_SIGMA 0x1  /* some sigma came out NaN or Inf */
#define GAS_DEV_WAIT_TIMEOUT    0x2  /* a bounded mbarrier/flag wait gave up */

/* Power-iteration back ends (gas_set_method). */
#define GAS_METHOD_AUTO   0  /* library picks (the fused Gram back end) */
#define GAS_METHOD_STREAM 1  /* per-iteration streaming matvec chain, Algorithm 2 literally */
#define GAS_METHOD_GRAM   2  /* one weight pass to d_h x d_h Gram matrices, iterate in R^{d_h}
                                (separate iteration kernel) */
#define GAS_METHOD_FUSED  3  /* as GRAM, with the iterations run inside the Gram kernel from
                                tensor memory (cooperative launch: needs every SM free) */

/*
 * Create a handle for one model shape (the paper's Section 4 cost model
 * O(n_q * d_h * d) per layer per iteration).
 *   layers >= 1; d >= 8 and d % 8 == 0 (16-byte rows); n_q, n_kv >= 1 with
 *   n_q % n_kv == 0; d_h in {64, 80, 96, 128, 256}; for d_h 64 / 80 / 96 / 128 the
 *   group size n_q/n_kv <= 32 (d_h 64) or 64 (the others).  The tensor-core back ends
 *   (fused, gram) need d_h 64, 80, 96 or 128 (a d_h 80 / 96 head fills the top rows of
 *   a 128-row tile, the rest reads as zero), 16-bit weights, and for the Conv1D layout
 *   d_h 64 or 128; d_h 256 and fp32 weights run on the streaming back end, which
 *   GAS_METHOD_AUTO then selects.
 * Allocates the device workspace on the current device (see gas_workspace_bytes).
 * Errors: GAS_ERR_INVALID_ARG (out == NULL, non-positive sizes), GAS_ERR_UNSUPPORTED
 * (shape limits above), GAS_ERR_ALLOC, GAS_ERR_CUDA.  *out is NULL on error.
 */
gas_status gas_create(int layers, int d, int n_q, int n_kv, int d_h, gas_handle *out);

/* Free the workspace (synchronises the device first).  NULL is a no-op. */
gas_status gas_destroy(gas_handle h);

/* Bytes of device workspace the handle holds. */
size_t gas_workspace_bytes(gas_handle h);

/*
 * Calibration constants used by gas_scales / gas_refresh (Sections 3.2, 3.4):
 *   seq_len L (Eq. 12-13, default 1024), eta_fp8 (Eq. 15, default 0.8),
 *   alpha_override > 0 replaces alpha_min (the paper's rounded 0.08/0.04/0.03/0.02
 *   or an auto-alpha result, Section 3.5); <= 0 restores alpha_min.
 * Errors: GAS_ERR_INVALID_ARG for seq_len < 1 or eta_fp8 outside (0, 1].
 */
gas_status gas_set_calibration(gas_handle h, int seq_len, double eta_fp8, double alpha_override);

/* Select the power-iteration back end (GAS_METHOD_*). */
gas_status gas_set_method(gas_handle h, int method);

/*
 * Per-head spectral norms by `iters` power iterations (Algorithm 2 per head; one
 * iteration = u' = M v, sigma = ||u'||, u = u'/sigma, v' = M^T u, v = v'/||v'||;
 * the reported sigma is the last iteration's ||M v_{k-1}||).
 *   wq, wk : HOST arrays of `layers` DEVICE pointers to the bf16 Wq[l], Wk[l].
 *   iters  : >= 1 (cold start: the paper uses 5; warm refresh: 1-2).
 *   v_in   : device fp32 [layers][n_q][d] start vectors (any scale; a zero vector
 *            gives sigma = 0 and v_out = 0).  Warm start: pass last call's v_out.
 *   v_out  : device fp32, same shape, unit right singular vector estimates; may
 *            alias v_in; NULL skips the write-back.
 *   sigma  : device fp32 [layers][n_q].
 * Errors: GAS_ERR_INVALID_ARG (NULL or misaligned pointers, iters < 1),
 * GAS_ERR_CUDA (launch failure).
 */
gas_status gas_spectral_norms(gas_handle h, const void *const *wq, const void *const *wk,
                              int iters, const float *v_in, float *v_out, float *sigma,
                              void *stream);

/*
 * Per-layer scale (Eq. 15) from per-head sigmas: s[l] = alpha * max_h sigma[l][h] *
 * (d / sqrt(d_h)) / (eta_fp8 * r_max).  N = layers * n_q heads enter Eq. 12-13.
 *   gamma      : > 1 uses it; <= 0 solves Eq. 12 for the minimal gamma; (0, 1] is an error.
 *   delta_star : target overflow probability, > 0 (paper: 1e-6).
 *   r_max      : format maximum, > 0 (448 for E4M3).
 *   sigma, s   : device fp32 [layers][n_q] in, [layers] out.
 * A NaN sigma propagates into its layer's scale.
 */
gas_status gas_scales(gas_handle h, const float *sigma, double gamma, double delta_star,
                      double r_max, float *s, void *stream);

/*
 * gas_spectral_norms followed by gas_scales, with the per-layer max and the
 * scale evaluated inside the last power-iteration kernel (no separate pass).
 * Arguments as above.
 */
gas_status gas_refresh(gas_handle h, const void *const *wq, const void *const *wk, int iters,
                       const float *v_in, float *v_out, float *sigma, double gamma,
                       double delta_star, double r_max, float *s, void *stream);

/*
 * Whole-layer spectral norm (Section 4.2, Appendix E): sigma_l = ||M||_2 for
 * M = W^Q W^K_exp^T with W^Q = all n_q heads ([d x n_q*d_h]) and W^K_exp = W^K with each
 * KV group repeated for its query heads (never formed: the repeat and its transpose, a
 * sum over each group's query blocks, act on the n_kv*d_h-vectors).  Power iteration
 * with one persistent v per layer; sigma_l = ||M v|| of the last iteration.
 *   v_in, v_out : device fp32 [layers][d] (v_out may alias v_in or be NULL).
 *   sigma       : device fp32 [layers].
 *   s           : device fp32 [layers] or NULL; if given, the layer scale of Eq. 15 with
 *                 sigma_l (gamma, delta_star, r_max as for gas_scales).
 * Each iteration streams W^Q and W^K twice (no d_h x d_h reduction exists for the
 * n_q*d_h-dimensional inner space).  Errors as gas_refresh; GAS_ERR_UNSUPPORTED when
 * d or n_q*d_h exceeds what one CTA's shared memory holds (about 57000 floats).
 */
gas_status gas_layer_refresh(gas_handle h, const void *const *wq, const void *const *wk, int iters,
                             const float *v_in, float *v_out, float *sigma, double gamma,
                             double delta_star, double r_max, float *s, void *stream);

/* Host helpers in float64: Eq. 12 (smallest gamma > 1; 1.0 if the bound holds for
 * every gamma; NaN on invalid input) and Eq. 13 (alpha_min for a given gamma). */
double gas_gamma_min(int d_h, long long n_heads_total, int seq_len, double delta_star);
double gas_alpha_min(double gamma, int d, int d_h, long long n_heads_total, int seq_len,
                     double delta_star);

/* Gamma and alpha the handle would use for gas_scales with this gamma / delta*. */
gas_status gas_resolve_calibration(gas_handle h, double gamma, double delta_star,
                                   double *gamma_out, double *alpha_out);

/* Element types (weights: gas_set_weight_dtype; logits: gas_fp8_quantize). */
#define GAS_DTYPE_BF16 0
#define GAS_DTYPE_F32  1
#define GAS_DTYPE_F16  2

/*
 * Weight element type: GAS_DTYPE_BF16 (default), GAS_DTYPE_F16 (IEEE binary16) or
 * GAS_DTYPE_F32.  With binary16 weights the tensor-core operands (weights, and the
 * hi + lo split start and write-back vectors) are binary16 too; sigma and v keep the
 * same fp32 accumulation.  The write-back's y / ||v'|| operand must lie inside binary16's
 * range, which holds unless ||W^K_g||_2 is below about 2^-14.  fp32 weights are read by
 * the streaming back end and the whole-layer path only (d_h <= 128); AUTO selects the
 * streaming back end for them, and the fused / gram back ends return
 * GAS_ERR_UNSUPPORTED.  Host only; applies to later calls.  Unknown values ->
 * GAS_ERR_INVALID_ARG.  gas_spectral_norms_static always reads bf16.
 */
gas_status gas_set_weight_dtype(gas_handle h, int dtype);

/*
 * Weight layout (the paper fixes none; it writes W^Q in R^{d x n_q d_h}).  By default a
 * layer's Wq[l] is the contiguous nn.Linear matrix [n_q * d_h, d].  Weights that are a
 * strided view of a larger allocation are described by two strides per matrix, in
 * elements:
 *     element (row i of head j, column c) of Wq[l] is at Wq[l][j * hs_q + i * ld_q + c]
 * (likewise Wk[l] with ld_k, hs_k and key groups j).  This covers rows padded beyond d
 * (ld > d), and fused projections whose query and key blocks are interleaved per head,
 * e.g. [heads][3][d_h][d] gives ld = d, hs = 3 * d_h * d with Wk[l] = Wq[l] + d_h * d.
 *   layout  GAS_LAYOUT_ROWS as above, or GAS_LAYOUT_COLS, the transposed (GPT-2
 *           Conv1D) storage [d, n * d_h] with the output features contiguous:
 *               element (row r = head * d_h + i, column c) at W[l][c * ld + r],
 *           e.g. GPT-2's c_attn weight [d, 3d] gives Wq = W, Wk = W + d, ld = 3d.
 *   ld_q, ld_k  ROWS: row strides, >= d; 0 = d.  COLS: column strides, >= n * d_h;
 *               0 = n * d_h
 *   hs_q, hs_k  ROWS: head strides, >= d_h * row stride (heads do not overlap);
 *               0 = d_h * ld.  COLS: heads are contiguous, 0 or d_h only
 * All strides must be multiples of 8 elements (16-byte rows and heads, as TMA needs).
 * GAS_LAYOUT_COLS is read by the tensor-core back ends (fused, gram); with it the
 * streaming back end and gas_layer_refresh return GAS_ERR_UNSUPPORTED.
 * Host only; applies to every later call on the handle (gas_spectral_norms_static always
 * uses the contiguous layout).  Errors: GAS_ERR_INVALID_ARG with a message.
 */
#define GAS_LAYOUT_ROWS 0
#define GAS_LAYOUT_COLS 1
gas_status gas_set_weight_layout(gas_handle h, int layout, long long ld_q, long long ld_k, long long hs_q,
                                 long long hs_k);

/* Message for the last error on this handle (or the last gas_create failure when h is NULL). */
const char *gas_last_error(gas_handle h);
const char *gas_status_string(gas_status s);

/* Read (blocking: synchronises the device) and optionally clear the device status
 * word (GAS_DEV_* bits).  Returns GAS_ERR_DEVICE_TIMEOUT when the timeout bit is set. */
gas_status gas_get_device_status(gas_handle h, int *code, int clear);

/*
 * Self-test of the device-side failure detection (library infrastructure; the paper has
 * no counterpart).  Enqueues on `stream` one small
 * kernel whose bounded wait runs out on purpose, the same wait the Gram and write-back
 * kernels use: which = 0 waits for an mbarrier phase that nothing completes, which = 1
 * for a global flag that nothing writes.  After the library's wait limit (2 s) the
 * kernel sets GAS_DEV_WAIT_TIMEOUT in this handle's device status word and returns;
 * it holds no tensor memory and leaves no copy in flight, so the context stays usable.
 * Read the outcome with gas_get_device_status.  Touches no caller buffer.
 * Errors: GAS_ERR_INVALID_ARG (NULL handle, which not 0 or 1), GAS_ERR_CUDA (launch).
 */
gas_status gas_selftest_wait_timeout(gas_handle h, int which, void *stream);

/* Number of kernel launches the last gas_spectral_norms / gas_refresh enqueued. */
int gas_last_launch_count(gas_handle h);

/*
 * Diagnostic timing hook.  When events != NULL, every kernel that a later
 * gas_spectral_norms / gas_refresh / gas_scales enqueues (in order, i = 0, 1, ...)
 * is bracketed by cudaEventRecord(events[2i]) before and events[2i+1] after, on the
 * call's stream, for the first n_events/2 kernels.  The events are caller-owned
 * cudaEvent_t handles (created without cudaEventDisableTiming) and must outlive the
 * calls; pass NULL / 0 to switch recording off.  Names of the kernels in launch order
 * are available from gas_last_launch_name.
 * Errors: GAS_ERR_INVALID_ARG for n_events < 0 or odd.
 */
gas_status gas_set_launch_events(gas_handle h, void *const *events, int n_events);

/* Kernel name of launch i of the last call ("" when out of range). */
const char *gas_last_launch_name(gas_handle h, int i);

/*
 * Allocation-free spectral norms (no counterpart in the paper).
 *
 * For callers that cannot allocate device memory: code running under another
 * framework's memory manager that owns all of HBM, latency-critical paths where the
 * device synchronisation implied by cudaMalloc / cudaFree is not allowed, and plugins
 * with nowhere to keep a handle alive.  Same result as gas_spectral_norms with
 * GAS_METHOD_STREAM (Algorithm 2 per head, streaming matvec chain), but it takes the
 * shape directly, needs no handle, and calls no cudaMalloc, cudaFree or allocating
 * library routine: its scratch is a file-scope device array of
 * GAS_STATIC_SCRATCH_BYTES that every GPU loading the library holds until the
 * process exits.
 *   Arguments: layers, d, n_q, n_kv, d_h as for gas_create, with narrower limits:
 *   d_h 64 or 128, d % 8 == 0, layers <= 512.  Weights are bf16 in the default
 *   contiguous nn.Linear layout ([n_q*d_h, d] and [n_kv*d_h, d] row-major; no row or
 *   head stride, no Conv1D layout, no fp16 / fp32).  wq, wk: host arrays of device
 *   pointers (16-byte aligned); v_in, v_out, sigma: device fp32 as for
 *   gas_spectral_norms (v_out may be NULL or alias v_in).
 *   Scratch needed: gas_static_scratch_bytes(layers, d, n_q, d_h), that is, with
 *   nch = ceil(d / 256) and a(x) = x rounded up to a multiple of 256:
 *     2*a(layers*n_q*nch*d_h*4) + 2*a(layers*n_q*nch*4) + 2*a(layers*n_q*d_h*4)
 *     + 2*a(layers*n_q*4) bytes
 *   (17,965,056 bytes for 32 layers, d 4096, 32 heads, d_h 128).  Shapes that need
 *   more than GAS_STATIC_SCRATCH_BYTES are rejected with GAS_ERR_UNSUPPORTED before
 *   any device work.
 *   Errors: as gas_spectral_norms; gas_last_error(NULL) holds the message.
 * Every call looks up the array's device address in the current context
 * (cudaGetSymbolAddress), so the address stays right after cudaDeviceReset or under
 * another context.  The first call on a device also loads the library's device code:
 * make that first call before any stream capture.  All calls share the array and it
 * keeps the last call's contents; every value a call reads from it was written earlier
 * in the same call, so nothing needs clearing.  Calls whose kernels overlap on the GPU
 * (other streams, other threads) race on the array.
 */
#define GAS_STATIC_SCRATCH_BYTES (32u * 1024u * 1024u)
gas_status gas_spectral_norms_static(int layers, int d, int n_q, int n_kv, int d_h,
                                     const void *const *wq, const void *const *wk, int iters,
                                     const float *v_in, float *v_out, float *sigma, void *stream);

/* Scratch bytes gas_spectral_norms_static needs for a shape (the expression above; 0
 * when a size is not positive).  Host only; no device work. */
size_t gas_static_scratch_bytes(int layers, int d, int n_q, int d_h);

#ifdef __cplusplus
}
#endif

#endif /* GAS_H_ */
