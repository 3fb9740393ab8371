/*
 * gsq.h -- C ABI of libgsq: one optimisation step of the GSQ relaxed scalar
 * quantizer (Gumbel-Softmax Quantization) for a linear layer, on one sm_103a GPU.
 *
 * The method (paper: "GSQ: Highly-Accurate Low-Precision Scalar Quantization for
 * LLMs via Gumbel-Softmax Sampling"):
 *   - every weight w_i of W gets one learnable logit l_{i,k} per level q_k of an
 *     ordered grid (§3.2, "General scalar quantization": l in R^{d x 2^b});
 *   - each step draws Gumbel noise g_{i,k} (Alg. 1), forms the tempered softmax
 *     p_{i,k} = softmax_k((kappa*l_{i,k} + g_{i,k}) / tau) (Alg. 1), the soft value
 *     w~_i = sum_k p_{i,k} q_k and the soft weight W^_i = s_{group(i)} * w~_i with one
 *     learnable scale per group of consecutive inputs (§3.2; §4.1 "Quantization
 *     configuration");
 *   - the loss is the layer-wise reconstruction error of Eq. 1 for a linear layer,
 *     L = sum_t ||(W^ - W) x_t||^2 = tr(D H D^T), D = W^ - W, H = X^T X;
 *   - logits and scales are updated with Lion (§3.3 "Optimizer", App. B);
 *   - after training the logits are hard-projected by argmax (Alg. 2, last lines)
 *     and packed into a symmetric group-wise scalar format (§4.1) or a two-level
 *     K-Quant-like format (§4.4, App. E).
 *
 * Conventions for every entry point:
 *   - All functions return a gsq_status (int32_t).  GSQ_OK = 0.  On failure
 *     gsq_last_error() returns a thread-local, human-readable message.
 *   - No C++ exception crosses this boundary.
 *   - "device" pointers are CUDA device (or managed) memory on the current device;
 *     "host" pointers are ordinary host memory.  Nothing here allocates device
 *     memory: the caller provides a workspace and every output buffer.
 *   - `stream` is a cudaStream_t passed as void* (NULL = the legacy default stream).
 *     Work is enqueued on it; calls return without waiting for the GPU except
 *     where a function says it synchronises.
 *   - The tensor-core and backward kernels of gsq_step and gsq_step_tokens are
 *     launched as programmatic dependents of the kernel before them on the
 *     stream: they may be scheduled while it drains, and wait for it to complete
 *     (griddepcontrol.wait) before their first global memory access, so stream
 *     order holds as for plain launches, also inside a captured CUDA graph.
 *     With the environment variable GSQ_PDL=0 they are launched plainly.
 *   - Argument errors are detected on the host before anything is enqueued.
 *     Launch errors are reported as GSQ_ERR_CUDA.
 *   - Fault injection for host-side tests: with the environment variable
 *     GSQ_FAULT_INJECT=<function name>:<n>, the n-th call (1-based) of that
 *     function returns GSQ_ERR_INJECTED before touching the GPU.
 */
#ifndef GSQ_H_
#define GSQ_H_

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define GSQ_API __attribute__((visibility("default")))
#else
#define GSQ_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes -------------------------------------------------------- */
enum {
  GSQ_OK = 0,
  GSQ_ERR_INVALID_ARG = 1, /* null pointer, bad enum, non-positive tau, ...   */
  GSQ_ERR_SHAPE = 2,       /* shape not supported (divisibility, limits)      */
  GSQ_ERR_WORKSPACE = 3,   /* workspace too small or misaligned               */
  GSQ_ERR_CUDA = 4,        /* a CUDA runtime/driver call or launch failed     */
  GSQ_ERR_NONFINITE = 5,   /* W or the calibration input holds NaN/Inf        */
  GSQ_ERR_STATE = 6,       /* call out of order (e.g. destroyed handle)       */
  GSQ_ERR_TIMEOUT = 7,     /* a bounded device-side wait gave up              */
  GSQ_ERR_INJECTED = 8,    /* GSQ_FAULT_INJECT fired                          */
  GSQ_ERR_UNSUPPORTED = 9  /* device is not sm_103 / feature not available    */
};
typedef int32_t gsq_status;

/* ---- descriptor enums ---------------------------------------------------- */
#define GSQ_MAX_LEVELS 8
enum { GSQ_DTYPE_F32 = 0, GSQ_DTYPE_BF16 = 1 };
enum { GSQ_CALIB_H = 0, GSQ_CALIB_X = 1, GSQ_CALIB_BATCHES = 2 };
enum { GSQ_SCALE_GROUP = 0, GSQ_SCALE_KQUANT2 = 1 };
enum { GSQ_GEMM_BF16 = 0, GSQ_GEMM_F32 = 1 };
enum {
  GSQ_FLAG_NO_NOISE = 1u, /* g = 0: plain tempered softmax, no Gumbel draw             */
                          /* bits 2 and 4 are reserved (rejected)                      */
  GSQ_FLAG_UNSTAGED = 8u  /* gsq_step's backward reads its input streams with direct
                             global loads instead of staging them through shared
                             memory with bulk asynchronous copies; the same kernel
                             body and the same results bit for bit (for comparison) */
};
enum { GSQ_PARAM_FULL = 0, GSQ_PARAM_SHIFT5 = 1, GSQ_PARAM_MASK_SIGN = 2 };

/* Layer problem (Eq. 1 with a linear f; §3.2; §4.1; Table 5 for the defaults).
 *
 * W            device, borrowed during gsq_init_layer only.  Row-major
 *              [num_experts][out_features][in_features], dtype w_dtype.
 * calib        device, borrowed during gsq_init_layer only, fp32.
 *              GSQ_CALIB_H: Gram matrices H_e = X_e^T X_e, [E][C][C] row-major
 *              (symmetrised as (H + H^T)/2 on copy).
 *              GSQ_CALIB_X: tokens X_e, [E][n_tokens][C] row-major; H_e is formed
 *              from them at init (fp32, on the GPU).
 *              GSQ_CALIB_BATCHES: no calibration at init (calib may be NULL);
 *              tokens arrive with every micro-batch through gsq_step_tokens,
 *              n_tokens being the most tokens per micro-batch and expert
 *              (a multiple of 8).
 * grid         the K ordered levels q_0 < ... < q_{K-1} (host values, copied).
 * group_size   scale group along the input dim, power of two in [4, 128],
 *              in_features % group_size == 0.  GSQ_SCALE_KQUANT2 requires 16.
 * scale_mode   GSQ_SCALE_GROUP: one fp32 scale per group, learned (signed).
 *              GSQ_SCALE_KQUANT2: two-level frozen scales: per 16-weight sub-block
 *              s = d * sc with an fp16 d per 256-weight super-block and a 6-bit
 *              signed sc; requires lr_scales == 0 and in_features % 256 == 0.
 * init_bias    logit given to the round-to-nearest level at init (others 0).
 * seed         key of the counter-based Gumbel noise (Philox4x32-10).
 * lr_*, beta*, wd_*  Lion hyper-parameters; lr_scales = wd_scales = 0 freezes
 *              the scales.
 * gemm_precision  GSQ_GEMM_BF16: the loss contraction G = D (H + H^T) runs on the
 *              tensor cores with bf16 D and H and fp32 accumulation;
 *              GSQ_GEMM_F32: fp32 D and H on the CUDA cores (validation).
 * param_mode   GSQ_PARAM_FULL: one logit per grid level (§3.2, l in R^{d x 2^b}).
 *              GSQ_PARAM_SHIFT5: local shift (§3.2 "Higher bit-widths", Fig. 1):
 *              five logits per weight for shifts delta = -2..2 around the initial
 *              (round-to-nearest) index j0; shift delta uses level
 *              grid[clip(j0 + delta, 0, K - 1)].  The projection gives the code
 *              clip(j0 + argmax - 2).  Logit tensors then hold 5 planes.
 *              GSQ_PARAM_MASK_SIGN: ternary mask x sign (§3.1, Alg. 2): the grid
 *              must be {-a, 0, a} (a > 0); two logits per weight, plane 0 the
 *              mask l_m and plane 1 the sign l_b, each relaxed by a binary GS
 *              with tied logits (-l, l); W^ = s a m~ b~.  Init: Eq. 3 applied to
 *              the round-to-nearest code, times init_bias.  Projection:
 *              m = [l_m >= 0], b = 2 [l_b >= 0] - 1; code 0, 1, 2 for -a, 0, a;
 *              margin = 2|l_m|, or min(2|l_m|, 2|l_b|) when m = 1.
 * index_offset flat index, within a larger layer this one is a shard of, of this
 *              layer's first weight: weight (e, r, c) draws its noise with the
 *              counter index index_offset + (e*R + r)*C + c (0 for a whole layer).
 *              Rows and experts are independent in Eq. 1 with a linear f (the
 *              loss is a sum over rows, L = sum_r D_r H D_r^T, and Lion acts
 *              elementwise), so a shard holding rows [r0, r0 + R) of a one-expert
 *              layer with C inputs (index_offset = r0*C), or experts [e0, e0 + E)
 *              of a layer with R rows per expert (index_offset = e0*R*C), steps
 *              its weights exactly as the whole layer would, and the shards'
 *              losses sum to the layer's.  A multiple of 8.
 * Limits: 1 <= E, 1 <= R, 8 <= C, C % 8 == 0, E*R*C < 2^40, 2 <= K <= 8.
 */
typedef struct gsq_layer_desc {
  int32_t num_experts;
  int32_t out_features;
  int32_t in_features;
  int32_t w_dtype;
  const void* W;
  const float* calib;
  int64_t n_tokens;
  int32_t calib_kind;
  int32_t num_levels;
  float grid[GSQ_MAX_LEVELS];
  int32_t group_size;
  int32_t scale_mode;
  float init_bias;
  uint32_t flags;
  uint64_t seed;
  float lr_logits;
  float lr_scales;
  float beta1;
  float beta2;
  float wd_logits;
  float wd_scales;
  int32_t gemm_precision;
  int32_t param_mode;
  uint64_t index_offset;
} gsq_layer_desc;

typedef struct gsq_layer gsq_layer; /* opaque handle, host memory owned by libgsq */

/* Bytes of device workspace gsq_init_layer needs for this descriptor.  Pure
 * host arithmetic; no CUDA call.  The workspace must be 256-byte aligned. */
GSQ_API gsq_status gsq_workspace_size(const gsq_layer_desc* desc, size_t* bytes);

/* Validate `desc`, carve `workspace` (device, caller-owned, must outlive the
 * handle), and initialise the state on `stream`: copy W; form H (from X if
 * GSQ_CALIB_X), symmetrise it and convert it to the GEMM operand precision;
 * initial scales (absmax / max|q|, or the two-level K-Quant scales); RTN codes;
 * logits = init_bias on the RTN level; Lion momenta = 0.  Synchronises `stream`
 * once, to report GSQ_ERR_NONFINITE if W or calib holds NaN/Inf.  On success
 * *out receives a new handle (release with gsq_destroy). */
GSQ_API gsq_status gsq_init_layer(const gsq_layer_desc* desc, void* workspace, size_t bytes,
                          void* stream, gsq_layer** out);

/* Diagnostics of the current logits (no noise), for monitoring a run; the paper
 * has no entry point for them but uses the first as the evidence for the local
 * shift (App. L) and relates the second to vanishing gradients (App. B):
 *   displacement[d]  number of weights whose projected code is d grid steps
 *                    from the initial code (RTN, or the codes of
 *                    gsq_init_logits); d = 7 counts 7 and more;
 *   margin[b]        number of weights whose top-two logit margin (as
 *                    gsq_project reports it) falls in bin b: [0, 1e-6),
 *                    [1e-6, 1e-5), ..., [1, 10), [10, inf);
 *   mean_max_prob    mean over weights of max_k p_k, p = softmax(kappa l / tau)
 *                    (mask x sign: the three-value distribution of the two
 *                    binary instances); near 1 means saturated.
 * Uses the loss-reduction scratch of the workspace, so it must not overlap a
 * step of the same layer.  Synchronises `stream`.  Errors: GSQ_ERR_INVALID_ARG,
 * GSQ_ERR_CUDA. */
#define GSQ_DIAG_SHIFT_BINS 8
#define GSQ_DIAG_MARGIN_BINS 9
typedef struct gsq_diagnostics {
  int64_t displacement[GSQ_DIAG_SHIFT_BINS];
  int64_t margin[GSQ_DIAG_MARGIN_BINS];
  double mean_max_prob;
} gsq_diagnostics;
GSQ_API gsq_status gsq_diagnose(gsq_layer* layer, float tau, float kappa, void* stream,
                        gsq_diagnostics* out);

/* Warm start from a supplied solution (§3.1 "Initialization", Eq. 3-4; App. A),
 * on `stream`, replacing the logits of gsq_init_layer:
 *   l = sigma * (eps + alpha * l_prior), logit momenta = 0, where l_prior is,
 *   for every weight with supplied code c (a grid index):
 *     GSQ_PARAM_FULL       -(q_k - q_c)^2 / 2 minus its mean over k (App. A, b = 2);
 *     GSQ_PARAM_SHIFT5     -d^2 / 2 for d = -2..2 minus its mean (App. A, b > 2),
 *                          and j0 := c (the window is re-centred on the code);
 *     GSQ_PARAM_MASK_SIGN  Eq. 3: l_m = +1 if c != 1 else -1, l_b = +1/-1/0 for
 *                          c = 2/0/1.
 * codes_dev  device uint8 [E][R][C], caller-owned; a code >= K acts as K-1.
 * eps_dev    device fp32 [L][E][R][C] (L logit planes), caller-owned, nullable
 *            (eps = 0): the N(0, I) draw of Eq. 4, made by the caller.
 * alpha, sigma  Eq. 4's warm-start strength and logit scale (finite).
 * Scales and scale momenta are left as they are (set them with gsq_set_tensor
 * to start from the solution's scales).  Never synchronises.
 * Errors: GSQ_ERR_INVALID_ARG (handle, NULL codes_dev, non-finite alpha or
 * sigma), GSQ_ERR_CUDA. */
GSQ_API gsq_status gsq_init_logits(gsq_layer* layer, const uint8_t* codes_dev, const float* eps_dev,
                           float alpha, float sigma, void* stream);

/* One optimisation step t (Alg. 2 loop body generalised to K levels):
 *   forward   noise for step t, p = softmax((kappa l + g)/tau), W^, D = W^ - W
 *             (skipped when the previous call already produced D for
 *             (t, tau, kappa) through its look-ahead);
 *   loss      G = dL/dW^ = D (H + H^T) on the tensor cores (or fp32 cores),
 *             L_t = 1/2 sum D*G = tr(D H D^T);
 *   backward  dL/dl_k = (kappa/tau) G s p_k (q_k - w~),  dL/ds_g = sum_g G w~;
 *   update    Lion on logits and scales, in place;
 *   look-ahead (next_tau > 0): the same kernel then draws the noise of step t+1
 *             and writes D for (t+1, next_tau, next_kappa), so the next call
 *             skips its forward.  Results are identical either way.
 * step         noise counter t, < 2^32.  tau > 0, kappa finite.
 * loss_dev     device fp32 scalar, nullable: receives L_t (the loss of this
 *              step's forward, before the update).
 * grad_logits_dev / grad_scales_dev  device, nullable.  If either is non-null
 *              the step runs in gradient-export mode: it writes the raw
 *              gradients ([L][E][R][C] fp32, L logits per weight, and
 *              [E][R][C/G] fp32), skips the Lion update and ignores next_tau.
 * Kernels: the contraction and the backward (+ update + look-ahead) are two
 * kernels.  Outside export mode the backward
 * brings its input streams into shared memory with bulk asynchronous copies a
 * tile of 1,024 weights ahead (unless GSQ_FLAG_UNSTAGED, or the layer is too
 * small to give each block more than one tile); the results are the same bit
 * for bit, apart from the summation order of the loss.  The D of noise counter t lives in one
 * of two buffers by the parity of t, so a look-ahead never overwrites the D
 * that its own step's contraction reads.
 * Never synchronises; graph-capturable for a fixed argument list. */
GSQ_API gsq_status gsq_step(gsq_layer* layer, uint64_t step, float tau, float kappa, float next_tau,
                    float next_kappa, void* stream, float* loss_dev, float* grad_logits_dev,
                    float* grad_scales_dev);

/* One micro-batch of an optimisation step on per-step calibration tokens, with
 * gradient accumulation over resampled noise (§3.3 "Objective" and "Gradient
 * accumulation"); layers described with GSQ_CALIB_BATCHES only.
 * Step `step` has n_micro micro-batches, issued in order micro = 0..n_micro-1
 * (another order returns GSQ_ERR_STATE).  Micro-batch j of step t:
 *   forward   fresh noise with the counter t*n_micro + j (every forward pass
 *             draws anew), W^_j, D_j = W^_j - W;
 *   loss      G = 2 D_j X^T X (X = X_dev, this micro-batch's tokens), as
 *             Y = D_j X^T, G = 2 Y X, or on the tensor cores, where it costs fewer
 *             flops (C (T + 2R) < 4 R T at the descriptor's n_tokens = T), through
 *             the micro-batch's Gram matrix H = X^T X (bf16, formed from the tiles
 *             of its upper triangle and mirrored), G = 2 D_j H;
 *             GSQ_TOKEN_ROUTE=direct|gram in the environment at gsq_init_layer
 *             (and gsq_workspace_size) forces one, GSQ_TOKEN_SYM=0 forms every tile
 *             of H (the rule then reads C (T + R) < 2 R T);
 *             L_j = 1/2 sum D_j*G = sum over the tokens of ||D_j x||^2;
 *   backward  the gradients of L_j, added into an accumulator;
 *   update    after the last micro-batch only: Lion with the mean gradient
 *             (accumulated sum / n_micro); the state is untouched before that.
 * Each call's kernel also draws the next pass's noise and writes its D: the
 * next micro-batch's (same tau, kappa) or, after the last micro-batch and when
 * next_tau > 0, micro-batch 0 of step+1 with (next_tau, next_kappa).
 * X_dev      device fp32 [E][n_tokens][C], caller-owned, borrowed for the call;
 *            the tensor-core path converts it to bf16.
 * n_tokens   tokens of this micro-batch per expert: a multiple of 8, at most the
 *            descriptor's n_tokens.
 * loss_dev   device fp32 scalar, nullable: receives L_j.
 * Errors: GSQ_ERR_INVALID_ARG (handle, layer not GSQ_CALIB_BATCHES, NULL X,
 * bad n_tokens, micro >= n_micro, tau, counter >= 2^32), GSQ_ERR_STATE,
 * GSQ_ERR_CUDA.  Never synchronises. */
GSQ_API gsq_status gsq_step_tokens(gsq_layer* layer, uint64_t step, uint32_t micro, uint32_t n_micro,
                           float tau, float kappa, float next_tau, float next_kappa,
                           const float* X_dev, int64_t n_tokens, void* stream, float* loss_dev);

/* Forward only (Alg. 1 for every weight): writes D for (step, tau, kappa) into
 * the workspace and, if what_dev (device fp32 [E][R][C]) is non-null, the soft
 * weight W^.  A following gsq_step with the same (step, tau, kappa) reuses D. */
GSQ_API gsq_status gsq_forward(gsq_layer* layer, uint64_t step, float tau, float kappa, void* stream,
                       float* what_dev);

/* Hard projection (Alg. 2, last lines, for K levels): codes_dev (device uint8
 * [E][R][C], nullable) receives argmax_k l_k of the noise-free logits, lowest k on
 * ties; margin_dev (device fp32 [E][R][C], nullable) receives l_(1) - l_(2). */
GSQ_API gsq_status gsq_project(gsq_layer* layer, void* stream, uint8_t* codes_dev, float* margin_dev);

/* Size of the packed output of gsq_pack. */
GSQ_API gsq_status gsq_packed_size(const gsq_layer* layer, size_t* bytes);

/* Project and pack (§4.1; §4.4 and App. E) into out_dev (device, cap bytes):
 *  GSQ_SCALE_GROUP: code stream (2-bit codes for K <= 4, 3-bit for K <= 8; within
 *    each chunk of 32 consecutive weights of the row-major [E][R][C] order, code j
 *    sits at bit b*j of a little-endian b*32-bit word), padded to 16 bytes, then
 *    the fp16 (round-to-nearest-even) group scales [E][R][C/G], little-endian.
 *  GSQ_SCALE_KQUANT2: one 110-byte record per 256 consecutive weights: 96 B of
 *    3-bit codes (same stream), 12 B of sixteen 6-bit sub-scale codes sc+32
 *    (little-endian stream, code j at bit 6j), 2 B fp16 d.
 * *written (host, nullable) receives the byte count. */
GSQ_API gsq_status gsq_pack(gsq_layer* layer, void* stream, void* out_dev, size_t cap, size_t* written);

/* State tensors for inspection, checkpoint and resume. */
enum {
  GSQ_T_LOGITS = 0,     /* fp32 [L][E][R][C], L = K (FULL) or 5 (SHIFT5)       */
  GSQ_T_SCALES = 1,     /* fp32 [E][R][C/G] (effective scale d*sc for KQUANT2)  */
  GSQ_T_MOM_LOGITS = 2, /* fp32 [L][E][R][C]                                   */
  GSQ_T_MOM_SCALES = 3, /* fp32 [E][R][C/G]                                    */
  GSQ_T_D = 4,          /* last forward's D = W^ - W, [E][R][C], bf16 or fp32  */
  GSQ_T_G = 5,          /* last step's dL/dW^, fp32 [E][R][C]                  */
  GSQ_T_W = 6,          /* stored copy of W, [E][R][C], w_dtype                */
  GSQ_T_H = 7,          /* GEMM operand H (symmetrised), [E][C][C], bf16/fp32; *
                         * per-step tokens: the last micro-batch's X^T X (bf16) *
                         * on the Gram route, size 0 otherwise                  */
  GSQ_T_KQ_D = 8,       /* fp16 bits [E*R*C/256] (KQUANT2 only)                */
  GSQ_T_KQ_SC = 9,      /* int8 [E*R*C/16] (KQUANT2 only)                      */
  GSQ_T_J0 = 10         /* uint8 [E][R][C] initial grid index (SHIFT5 only);   *
                         * a value >= K set through gsq_set_tensor acts as K-1  *
                         * (every index is clipped to the grid before use)      */
};

/* Byte size of tensor `which` (0 when the layer has no such tensor). */
GSQ_API gsq_status gsq_tensor_size(const gsq_layer* layer, int32_t which, size_t* bytes);

/* Copy tensor `which` to/from caller device memory (bytes must equal its size).
 * gsq_set_tensor invalidates a pending look-ahead forward.  Saving LOGITS,
 * SCALES, MOM_LOGITS, MOM_SCALES and the step index and restoring them into a
 * layer built from the same descriptor resumes the trajectory bit for bit. */
GSQ_API gsq_status gsq_get_tensor(gsq_layer* layer, int32_t which, void* dst_dev, size_t bytes,
                          void* stream);
GSQ_API gsq_status gsq_set_tensor(gsq_layer* layer, int32_t which, const void* src_dev, size_t bytes,
                          void* stream);

/* Synchronise `stream` and report GSQ_ERR_TIMEOUT if a bounded device-side wait
 * of an earlier launch gave up (the error word is then cleared). */
GSQ_API gsq_status gsq_sync_status(gsq_layer* layer, void* stream);

/* Per-kernel CUDA-event timing.  While enabled, every launch made by libgsq for
 * this layer is bracketed by events recorded on the launch stream.
 * gsq_profile_read synchronises on the last event, returns per-kernel launch
 * counts and total milliseconds (kinds: GSQ_K_*), and clears the record. */
enum {
  GSQ_K_FORWARD = 0,  /* standalone forward (noise + softmax + D)              */
  GSQ_K_GEMM = 1,     /* loss contraction G = D (H + H^T)                     */
  GSQ_K_BACKWARD = 2, /* fused backward + Lion (+ look-ahead forward) + loss   */
  GSQ_K_PROJECT = 3,
  GSQ_K_PACK = 4,
  GSQ_K_INIT = 5,
  GSQ_K_TOKENS = 6,   /* per-step tokens to the tensor-core operands (bf16, X^T) */
  GSQ_K_COUNT = 7
};
typedef struct gsq_profile {
  int32_t launches[GSQ_K_COUNT];
  float total_ms[GSQ_K_COUNT];
} gsq_profile;
GSQ_API gsq_status gsq_profile_enable(gsq_layer* layer, int32_t on);
GSQ_API gsq_status gsq_profile_read(gsq_layer* layer, gsq_profile* out);

/* ---- allocation-free backward update --------------------------------------
 * The paper has no counterpart: this entry point exists for callers that
 * cannot allocate device memory (a host that owns a fixed pool, a plugin whose
 * host forbids allocation, code running where allocation is not allowed).
 * It runs the fused backward + Lion kernel of gsq_step on buffers the caller
 * owns, for a dL/dW^ the caller supplies (from this library's loss GEMM, read
 * with gsq_get_tensor(GSQ_T_G), or from any other objective):
 *   recompute noise and p for (step, tau, kappa); dL/dl and dL/ds from G;
 *   Lion on logits and scales in place; loss_dev (nullable) = 1/2 sum D*G with
 *   D = s w~ - W rounded to d_dtype (as the loss GEMM consumed it).
 * Full parameterisation only (one logit per level).  Layouts are those of
 * gsq_get_tensor: logits and m_logits [K][E][R][C] fp32, scales and m_scales
 * [E][R][C/G] fp32, W [E][R][C] (w_dtype), G [E][R][C] fp32.
 * Its only scratch (a counter and one double per thread block) is a static
 * 131,328-byte device array inside libgsq that every GPU loading the library
 * holds until the process exits; nothing is allocated, so E*R*C is limited to
 * 16,777,216 weights (larger layers return GSQ_ERR_SHAPE).  The first call in a
 * CUDA context looks up that array's device address (cudaGetSymbolAddress) and
 * caches it under the context's ID; a later call in another context (after
 * cudaDeviceReset, or with another context current on the device) looks it up
 * again.  Make the first call in each context before any stream capture.
 * flags accepts GSQ_FLAG_NO_NOISE only; any other bit is GSQ_ERR_INVALID_ARG.  All calls on one GPU
 * share its copy of the array and it keeps the last call's contents (the call
 * clears the counter before launching): calls that overlap on the same GPU (for
 * instance on two streams) race and corrupt each other's loss value; the state
 * update itself does not depend on the array.  Errors: GSQ_ERR_INVALID_ARG,
 * GSQ_ERR_SHAPE, GSQ_ERR_UNSUPPORTED, GSQ_ERR_CUDA, message via gsq_last_error(). */
typedef struct gsq_backward_args {
  int32_t num_experts;
  int32_t out_features;
  int32_t in_features;
  int32_t num_levels;
  float grid[GSQ_MAX_LEVELS];
  int32_t group_size;
  int32_t w_dtype;
  int32_t d_dtype;
  uint32_t flags;      /* GSQ_FLAG_NO_NOISE */
  const void* W;
  const float* G;
  float* logits;
  float* m_logits;
  float* scales;
  float* m_scales;
  float* loss_dev;
  uint64_t seed;
  uint64_t step;
  float tau;
  float kappa;
  float lr_logits;
  float lr_scales;
  float beta1;
  float beta2;
  float wd_logits;
  float wd_scales;
} gsq_backward_args;
GSQ_API gsq_status gsq_backward_update_noalloc(const gsq_backward_args* args, void* stream);

/* Release the handle (host memory only; the workspace stays the caller's).
 * Returns GSQ_ERR_INVALID_ARG for NULL. */
GSQ_API gsq_status gsq_destroy(gsq_layer* layer);

/* Message of the last failure on this thread ("" if none). */
GSQ_API const char* gsq_last_error(void);

/* Library version, "major.minor.patch". */
GSQ_API const char* gsq_version(void);

/* Name of the kernel that gsq_step launches for the part `kind` of a
 * non-exporting step of this layer (GSQ_K_GEMM: "k_tc_gemm_pair",
 * "k_tc_gemm_quad" (clusters of two CTA pairs), "k_tc_gemm" or "k_simt_gemm"; GSQ_K_BACKWARD: "k_backward_staged" or
 * "k_backward"), so timings can be
 * attributed (the paper has no counterpart: a reporting aid).  Static string
 * owned by the library; NULL for an invalid handle or another kind. */
GSQ_API const char* gsq_kernel_name(gsq_layer* layer, int32_t kind);

#ifdef __cplusplus
}
#endif

#endif /* GSQ_H_ */
