/*
 * catq.h — C ABI of the CAT-Q soft-ternary calibration hot path on GB300 (sm_103a).
 *
 * CAT-Q ternarizes a linear layer W [N out, K in] as W ~ alpha * T, T in {-1, 0, +1},
 * per non-overlapping group of g consecutive elements of row-major W (App. B.2).
 * Each group carries frozen statistics (mu0, alpha0, Delta0) and three learnable
 * factors (d_mu, d_alpha, d_delta) (Eq. 3, §2.2):
 *
 *   mu = mu0 + d_mu * alpha0,  alpha = d_alpha * alpha0,  Delta = d_delta * Delta0,
 *   What = (W - mu) / alpha                                  (Eq. 3)
 *   T    = W                       (teacher, t = 0)          (Eq. 6)
 *        = f(What; s, Delta)       (soft stage, 0 < t <= gamma)
 *        = Q(What; Delta)          (hard stage, gamma < t <= 1)
 *   f(x; s, D) = [tanh(s(x-D)) + tanh(s(x+D))] / (2 tanh s)  (Eq. 5)
 *   Q(x; D)    = +1 if x > D, 0 if |x| <= D, -1 if x < -D   (Eq. 2)
 *   Wq   = alpha * T  (no mu in the reconstruction, §2.2 and App. B.2); Wq = W for the teacher.
 *
 * A calibration step for one linear computes Y = X Wq^T, the reconstruction loss
 * against the teacher output (Eq. 7, one linear), and the gradients into X and into the
 * three factors.  The GEMMs never write Wq to HBM: the modulation, the transition
 * function and alpha are applied while the weight tile sits in shared memory.
 *
 * Conventions for every call:
 *   - All tensors are caller-owned.  No call allocates device or host memory.
 *   - Pointers named "device" must be CUDA device pointers of the current device.
 *   - Every call is asynchronous on `stream` (NULL = legacy default stream).
 *   - Argument errors return a non-zero catq_status before anything is launched.
 *   - Conditions detected on the device (a bounded wait that expired) are latched in a
 *     per-device status word; read and clear it with catq_device_status().
 *   - Shapes: g divides K.  bf16 weights need g % 64 == 0 and N % 8 == 0; fp32 weights
 *     need g % 64 == 0 or g in {4, 8, 16, 32}.  The weight and activation dtypes must
 *     match: both CATQ_F32 (CUDA-core path) or both CATQ_BF16 (tensor-core path,
 *     fp32 accumulation).  W, X, Y, dY, dX and Wq buffers must be 16-byte aligned.
 *   - A group whose alpha is exactly 0 (constant weights, or d_alpha == 0) has Wq = 0,
 *     hard code 0 and zero factor gradients.
 */
#ifndef CATQ_H
#define CATQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t; NULL selects the legacy default stream. */
typedef struct CUstream_st* catq_stream;

typedef enum {
  CATQ_OK = 0,
  CATQ_ERR_INVALID_ARG = 1, /* null pointer, bad enum, non-finite or non-positive s */
  CATQ_ERR_SHAPE = 2,       /* g does not divide K, unsupported g, M < 0, N/K < 1 */
  CATQ_ERR_DTYPE = 3,       /* unknown dtype or mixed weight/activation dtypes */
  CATQ_ERR_ALIGN = 4,       /* buffer misaligned: 16 bytes for TMA operands, 256 for workspaces,
                               4 for the fp32 arrays of catq_factor_adamw_step */
  CATQ_ERR_CUDA = 5,        /* a CUDA runtime call failed (launch, attribute, tensor map) */
  CATQ_ERR_TIMEOUT = 6,     /* a bounded device-side wait expired (latched) */
  CATQ_ERR_NONFINITE = 7,   /* reserved: non-finite data detected (latched) */
  CATQ_ERR_UNSUPPORTED = 8, /* valid request this build does not implement (e.g. no sm_100-class GPU) */
  CATQ_ERR_WORKSPACE = 9    /* workspace missing or smaller than the *_workspace_bytes() result */
} catq_status;

typedef enum { CATQ_F32 = 0, CATQ_BF16 = 1 } catq_dtype;

/* Eq. 6: which branch of the softened ternarization produces T. */
typedef enum {
  CATQ_PHASE_TEACHER = 0, /* t = 0: T = W, Wq = W (the full-precision teacher) */
  CATQ_PHASE_SOFT = 1,    /* 0 < t <= gamma: T = f(What; s, Delta) */
  CATQ_PHASE_HARD = 2     /* gamma < t <= 1: T = Q(What; Delta) */
} catq_phase;

/* Base statistics and initial threshold Delta0 (in What units) of each group (§2.2). */
typedef enum {
  CATQ_THR_HALF = 0,  /* Eq. 3's mu0, alpha0 with Delta0 = 0.5, the paper's default (§2.2, App. B.1) */
  CATQ_THR_TWN07 = 1, /* Eq. 3's mu0, alpha0 with Delta0 = 0.7 * mean|W_group| / alpha0: TWN's
                         0.7 mean|W| threshold in What units (alpha*Delta equals it at identity
                         factors) */
  CATQ_THR_ABSMEAN = 2,    /* the absmean static rule §2.2 quotes (BitNet b1.58 and others):
                              mu0 = 0, alpha0 = mean|W|, Delta0 = 0.5 (Delta = alpha / 2) */
  CATQ_THR_TWN_STATIC = 3  /* TWN's static rule (§2.2): mu0 = 0, Delta_W = 0.7 mean|W|,
                              alpha0 = mean |W_i| over |W_i| > Delta_W, Delta0 = Delta_W / alpha0
                              (0.5 when no element is above) */
} catq_thr_init;

typedef enum { CATQ_REDUCE_MEAN = 0, CATQ_REDUCE_SUM = 1 } catq_reduction;

/* Which reconstruction a layer's quantized weight uses. */
typedef enum {
  CATQ_RECON_ALPHA_T = 0,   /* W ~ alpha T (§2.2, App. B.2; the paper's choice): Wq = alpha T */
  CATQ_RECON_ALPHA_T_MU = 1 /* W ~ alpha T + mu (the variant of the tab:mu ablation):
                               Wq = alpha T + mu with mu = mu0 + d_mu alpha0 per group; the
                               factor gradient of d_mu then follows dWq/dmu = 1 - f'(What).
                               A group with alpha == 0 has Wq = mu. */
} catq_recon;

/* Eq. 6 schedule point.  SOFT: s = (t / gamma) * s0 > 0.  HARD: s is the sharpness of the
 * surrogate f used for the backward pass (§2.3: the last soft epoch's sharpness, see
 * catq_schedule_at_epoch).  TEACHER: s is ignored. */
typedef struct {
  int32_t phase; /* catq_phase */
  float s;
} catq_schedule;

/* One linear layer.  All pointers are device pointers owned by the caller.
 * G = N*K/g groups; group j holds elements [j*g, (j+1)*g) of row-major W. */
typedef struct {
  int64_t N;       /* out_features (rows of W) */
  int64_t K;       /* in_features (columns of W) */
  int32_t g;       /* group size; g == K is channel-wise */
  int32_t w_dtype; /* catq_dtype of W */
  const void* W;   /* [N, K] row-major, read-only */
  float* mu0;      /* [G] written by catq_group_stats, read by every other call */
  float* alpha0;   /* [G] */
  float* delta0;   /* [G] */
  const float* d_mu;    /* [G] learnable factor d_mu    (Eq. 3), -1 < d_mu < 1 */
  const float* d_alpha; /* [G] learnable factor d_alpha (Eq. 3), > 0 */
  const float* d_delta; /* [G] learnable factor d_delta (§2.2), > 0 */
  /* [4*G] fp32 ([5*G] when recon is CATQ_RECON_ALPHA_T_MU), 16-byte aligned; required for
   * bf16 layers by the forward and by a backward that computes dX, ignored otherwise.  Each
   * such call first writes here the four per-group constants of its schedule point that
   * turn a weight into its Eq. 6 operand (SOFT: s/alpha, -s mu/alpha, s Delta,
   * alpha/(2 tanh s); HARD: 1/alpha, -mu/alpha, Delta, alpha), as float4 in
   * group-column-major order [K/g][N], then (CATQ_RECON_ALPHA_T_MU only) the G group offsets
   * mu in the same order; the fused GEMMs read one 16-byte vector (and one mu) per group
   * and row.  Contents are overwritten by every call, so two calls on one layer must not
   * overlap on the GPU. */
  float* op_const;
  int32_t recon;    /* catq_recon */
  int32_t reserved; /* must be 0 */
} catq_layer;

/* ABI version of this header; bumped on any incompatible change. */
#define CATQ_ABI_VERSION 3
int32_t catq_abi_version(void);

/* Human-readable name of a status code (static storage, never NULL). */
const char* catq_status_string(int32_t status);

/* Group statistics (Eq. 3; the threshold rules of §2.2, see catq_thr_init):
 *   mu0[j] = mean of group j;  alpha0[j] = mean |W - mu0[j]| over group j;
 *   delta0[j] = 0.5, or 0.7 * mean|W| / alpha0[j] (0.5 if alpha0[j] == 0);
 * or, for the static rules, the values catq_thr_init states.  Sums are compensated fp32
 * (two-sum; about twice fp32's precision) for the signed mean and pairwise fp32 for the
 * all-positive ones; results are stored as fp32.  Reads W once. */
catq_status catq_group_stats(const catq_layer* layer, int32_t thr_init, catq_stream stream);

/* Materialises the Eq. 6 weight for inspection (not used inside the GEMMs, which fuse it).
 *   Wq_out   [N, K], dtype w_dtype, nullable: alpha * T for the schedule's phase (W for
 *            TEACHER), computed exactly as the fused GEMM operand producer computes it.
 *   T_out    [N, K] int8, nullable: hard codes Q(What; Delta) in {-1, 0, 1} (Eq. 4).
 *   alpha_out [G] fp32, nullable: alpha = d_alpha * alpha0.                              */
catq_status catq_modulate_ternarize(const catq_layer* layer, catq_schedule sched, void* Wq_out,
                                    int8_t* T_out, float* alpha_out, catq_stream stream);

/* Forward Y = X Wq^T (Eq. 6 weight, Eq. 7 window output for one linear).
 *   X [M, K] row-major, Y [M, N] row-major, both of dtype x_dtype (== w_dtype); fp32
 *   accumulation.  M == 0 is a no-op.                                                    */
catq_status catq_soft_ternary_linear_fwd(const catq_layer* layer, catq_schedule sched,
                                         const void* X, int64_t M, int32_t x_dtype, void* Y,
                                         catq_stream stream);

/* Forward with the two options the plain forward lacks (Eq. 6 weight; §1 and App. B.2's
 * weight-activation setting):
 *   Y[m, :] = x_row_scale[m] * (X Wq^T)[m, :]   (x_row_scale NULL: scale 1)
 * x_row_scale [M] fp32 (4-byte aligned) is the per-token scale of 8-bit activation codes
 * in X (catq_act_quant_a8): X then holds the integer codes, exact in bf16, and the scale
 * is applied to the fp32 accumulator before the output rounding.  y_dtype is x_dtype or
 * CATQ_F32 (an fp32 output of a bf16 layer, e.g. a full-precision teacher output for
 * catq_soft_ternary_linear_fwd_loss); fp32 layers need CATQ_F32.  Other arguments and
 * errors as catq_soft_ternary_linear_fwd. */
catq_status catq_soft_ternary_linear_fwd_ex(const catq_layer* layer, catq_schedule sched, const void* X,
                                            int64_t M, int32_t x_dtype, const float* x_row_scale, void* Y,
                                            int32_t y_dtype, catq_stream stream);

/* Workspace bytes catq_soft_ternary_linear_fwd_loss needs for this layer and M on the
 * current device (fp64 partial sums of the loss). */
size_t catq_fwd_loss_workspace_bytes(const catq_layer* layer, int64_t M);

/* Forward and reconstruction loss of one linear in one pass (Eq. 6 weight, Eq. 7 loss):
 *   Y = diag(x_row_scale) X Wq^T     (the accumulator, never rounded before the loss)
 *   loss_out[0] = sum (Y - Y_ref)^2 / (M N)  (CATQ_REDUCE_MEAN)  or the plain sum (SUM)
 *   dY          = 2 (Y - Y_ref) / (M N)      (MEAN)              or 2 (Y - Y_ref) (SUM)
 * The bf16 path forms Y - Y_ref in the GEMM's epilogue from the fp32 accumulator, so Y is
 * rounded neither before the difference nor (unless requested) at all; dY is rounded once
 * to bf16.  Y_ref [M, N] has ref_dtype: x_dtype, or CATQ_F32 for a full-precision teacher of
 * a bf16 layer.  dY [M, N] (x_dtype) is required; Y [M, N] (x_dtype) is optional (NULL:
 * not stored).  x_row_scale as in catq_soft_ternary_linear_fwd_ex (NULL: 1).  loss_out:
 * device fp32 scalar.  The loss sums fp32 compensated partials per epilogue warp, then
 * the partials in fp64, in a fixed order (deterministic for a given device and shape).
 * fp32 layers run the CUDA-core forward (into Y, or into dY as scratch) and then the loss
 * kernel.  M >= 1 (else CATQ_ERR_SHAPE); X, Y_ref, dY, Y 16-byte aligned; workspace
 * >= catq_fwd_loss_workspace_bytes(layer, M), 256-byte aligned.
 * Cost: the loss lengthens the GEMM's accumulator drain, which the next tile's MMAs wait
 * for, so on a GB300 this call takes longer than catq_soft_ternary_linear_fwd followed by
 * catq_recon_loss (8B-shaped gate_proj, 8192 tokens: 827 us against 571 + 121 us).  Use it
 * where the unrounded Y - Y_ref matters; the two calls are the faster path. */
catq_status catq_soft_ternary_linear_fwd_loss(const catq_layer* layer, catq_schedule sched, const void* X,
                                              int64_t M, int32_t x_dtype, const float* x_row_scale,
                                              const void* Y_ref, int32_t ref_dtype, int32_t reduction,
                                              float* loss_out, void* dY, void* Y, void* workspace,
                                              size_t ws_bytes, catq_stream stream);

/* Per-token symmetric 8-bit quantization of activations X [M, K] (the weight-activation
 * setting W1.58A8 of §1 and App. B.2, which leaves the activation quantizer unstated; this
 * library reads it as dynamic per-token absmax quantization):
 *   scale[m]    = max_k |X[m, k]| / 127                      (fp32, IEEE division)
 *   codes[m, k] = clamp(rint(X[m, k] / scale[m]), -127, 127)  (fp32 IEEE division, ties to
 *                 even), 0 for a row of zeros (scale 0)
 *   X_deq[m, k] = scale[m] * codes[m, k], computed in fp32 and rounded to x_dtype (nullable)
 * codes and X_deq have x_dtype (integers up to 127 are exact in bf16) and [M, K] layout;
 * scale [M] fp32.  The forward uses codes with x_row_scale = scale
 * (catq_soft_ternary_linear_fwd_ex / _fwd_loss); the backward's dW uses X_deq (the
 * rounding is passed straight through to dX).  K * sizeof(x_dtype) must be a multiple of 16
 * (else CATQ_ERR_SHAPE); X, codes, X_deq 16-byte aligned, scale 4-byte.  M == 0 is a
 * no-op. */
catq_status catq_act_quant_a8(const void* X, int64_t M, int64_t K, int32_t x_dtype, void* codes, float* scale,
                              void* X_deq, catq_stream stream);

/* Workspace bytes catq_soft_ternary_linear_bwd needs for this layer and M (partial
 * per-group sums); 0 is never returned for M > 0. */
size_t catq_bwd_workspace_bytes(const catq_layer* layer, int64_t M);

/* Backward of Y = X Wq^T given dY = dL/dY [M, N] (dtype x_dtype):
 *   dX [M, K] = dY Wq            (nullable: skipped when NULL)
 *   with G = dY^T X [N, K] (never written to memory), per group j:
 *   g_dmu[j]    = -alpha0 * sum_j G * f'(What)
 *   g_dalpha[j] =  alpha0 * sum_j G * (T - What * f'(What))
 *   g_ddelta[j] =  Delta0 * alpha * sum_j G * df/dDelta(What)
 * f' and df/dDelta are the derivatives of Eq. 5 at the schedule's s.  In the HARD phase T
 * is the forward value Q(What; Delta) and the derivatives are those of f at s (the
 * surrogate reading of §2.3's stage-2 rule).  In the TEACHER phase Wq = W does not depend
 * on the factors: the three gradients are written as zeros.  Gradients are overwritten,
 * not accumulated.  g_dmu, g_dalpha, g_ddelta: device fp32 [G], all three or none (NULL
 * skips the factor gradients, e.g. a dX-only backward through frozen layers).
 * workspace: device, >= catq_bwd_workspace_bytes(layer, M) bytes, 256-byte aligned,
 * contents scratch; may be NULL when no factor gradients are computed.                  */
catq_status catq_soft_ternary_linear_bwd(const catq_layer* layer, catq_schedule sched,
                                         const void* X, const void* dY, int64_t M,
                                         int32_t x_dtype, void* dX, float* g_dmu,
                                         float* g_dalpha, float* g_ddelta, void* workspace,
                                         size_t ws_bytes, catq_stream stream);

/* Allocation-free backward (this library's addition; the paper has no counterpart).
 * For callers that cannot allocate device memory themselves, e.g. a host runtime without
 * access to a device allocator, or a service whose device memory is fixed when it starts:
 * identical to catq_soft_ternary_linear_bwd except that the partial group sums live in a
 * scratch array inside the library (catq_bwd_noalloc_max_scratch_bytes() = 16 MiB, held
 * by every GPU that loads the library until the process exits) instead of a workspace.
 *   - Calls needing more scratch than that (catq_bwd_workspace_bytes(layer, M) > 16 MiB)
 *     return CATQ_ERR_WORKSPACE before launching anything.
 *   - The first call on a device looks up the array's device address on that device (make
 *     it before any stream capture); this call allocates nothing, neither does any other.
 *   - All calls share the one array: calls whose kernels overlap on the GPU (e.g. on two
 *     streams) race and give wrong gradients.  Calls in order on one stream are safe; the
 *     array keeps the last call's contents, which every call overwrites before reading. */
catq_status catq_soft_ternary_linear_bwd_noalloc(const catq_layer* layer, catq_schedule sched,
                                                 const void* X, const void* dY, int64_t M,
                                                 int32_t x_dtype, void* dX, float* g_dmu,
                                                 float* g_dalpha, float* g_ddelta,
                                                 catq_stream stream);

/* Size in bytes of the scratch array catq_soft_ternary_linear_bwd_noalloc uses. */
size_t catq_bwd_noalloc_max_scratch_bytes(void);

/* Workspace bytes catq_recon_loss needs for `count` elements (block partial sums). */
size_t catq_recon_loss_workspace_bytes(int64_t count);

/* Reconstruction loss of Eq. 7 for one linear output, and its gradient:
 *   loss_out[0] = sum (Y - Y_ref)^2 / count   (CATQ_REDUCE_MEAN)  or the plain sum (SUM)
 *   dY          = 2 (Y - Y_ref) / count       (MEAN)              or 2 (Y - Y_ref) (SUM)
 * Y, Y_ref, dY: device, `count` elements of `dtype`; dY nullable.  loss_out: device fp32
 * scalar.  The sum runs in fp64 with a fixed reduction order (deterministic).
 * workspace: device, >= catq_recon_loss_workspace_bytes(count) bytes, 256-byte aligned. */
catq_status catq_recon_loss(const void* Y, const void* Y_ref, int64_t count, int32_t dtype,
                            int32_t reduction, float* loss_out, void* dY, void* workspace,
                            size_t ws_bytes, catq_stream stream);

/* Final hard ternarization and 2-bit packing (Eq. 2 / Eq. 4 at the end of calibration,
 * deployment keeps only T and the group scale alpha, App. B.2):
 *   codes [N*K/4] uint8: element e of row-major W stores Q(What_e; Delta) + 1 in bits
 *         [2*(e%4), 2*(e%4)+1] of byte e/4 (values 0, 1, 2; 3 never occurs).
 *   alpha [G] fp32, nullable: d_alpha * alpha0.
 *   mu    [G] fp32, nullable: mu0 + d_mu * alpha0, the group offsets a layer with
 *         CATQ_RECON_ALPHA_T_MU deploys beside alpha.
 * Requires N*K % 4 == 0.  The encoding is this library's; the paper fixes none.          */
catq_status catq_hard_ternarize_pack(const catq_layer* layer, uint8_t* codes, float* alpha, float* mu,
                                     catq_stream stream);

/* ------------------------------------------------------------------ calibration schedule and update
 * App. B.1 calibrates the learnable factors with AdamW for m = 60 epochs at learning rate
 * 1e-3 decayed linearly to zero, gamma = 0.8, s0 = 30; §2.3 maps the normalised epoch t to
 * the branch and sharpness of Eq. 6.  These calls give a calibration loop what it needs
 * beyond the step itself. */

/* Eq. 6's schedule point of calibration epoch e of m (host only, no device work):
 * t = e / m; e == 0 is the teacher branch (t = 0); e <= floor(gamma m + 1e-9) the soft
 * stage with s = (t / gamma) s0; later epochs the hard stage, whose backward sharpness is
 * the last soft epoch's, (floor(gamma m) / m / gamma) s0 (§2.3 keeps the gradients of the
 * first stage's last iteration): s0 when gamma m is an integer, as at the paper's
 * defaults; s0 also when no epoch is soft (gamma m < 1).  Requires 0 <= e <= m, m >= 1,
 * 0 < gamma <= 1, finite s0 > 0 and a non-null `out`; else CATQ_ERR_INVALID_ARG. */
catq_status catq_schedule_at_epoch(int32_t e, int32_t m, double gamma, double s0, catq_schedule* out);

/* Learning rate of update k (0-based) of `total` under App. B.1's linear decay to zero
 * (host only): lr0 (1 - k / total).  Requires 0 <= k < total, finite lr0 >= 0 and a
 * non-null `lr_out`; else CATQ_ERR_INVALID_ARG. */
catq_status catq_linear_decay_lr(double lr0, int64_t k, int64_t total, float* lr_out);

/* AdamW hyperparameters beyond the learning rate (App. B.1 names the optimizer only). */
typedef struct {
  float beta1;        /* first-moment decay, 0 <= beta1 < 1 (the optimizer's usual 0.9) */
  float beta2;        /* second-moment decay, 0 <= beta2 < 1 (0.999) */
  float eps;          /* added to sqrt(v_hat), finite and > 0 (1e-8) */
  float weight_decay; /* decoupled decay, scaled by the learning rate, >= 0 (0: a decay of the
                         factors towards zero would shrink alpha and Delta) */
  float margin;       /* projection margin of §2.2's constraints, 0 <= margin < 0.5 */
} catq_adamw;

/* The update of the learnable factors after a calibration step: for each of d_mu, d_alpha,
 * d_delta (in place, [G] fp32 device) with its gradient ([G] fp32 device, e.g. the output
 * of catq_soft_ternary_linear_bwd), one AdamW step (Loshchilov & Hutter's decoupled weight
 * decay, Adam's bias-corrected moments, update count t >= 1):
 *   p <- p (1 - lr weight_decay)
 *   m <- beta1 m + (1 - beta1) grad,  v <- beta2 v + (1 - beta2) grad^2
 *   p <- p - (lr / (1 - beta1^t)) m / (sqrt(v) / sqrt(1 - beta2^t) + eps)
 * then the projection of §2.2's constraints -1 < d_mu < 1, d_alpha > 0, d_delta > 0 onto
 * [-1 + margin, 1 - margin], [margin, inf), [margin, inf) (NaN passes through unchanged).
 * moments: [6, G] fp32 device, the optimizer state m_mu, m_alpha, m_delta, v_mu, v_alpha,
 * v_delta, zero before the first update and updated in place.  fp32 arithmetic with
 * IEEE division and square root.  For a stacked MoE layer pass G = E * groups per expert.
 * G == 0 is a no-op whatever the pointers.  Pointers 4-byte aligned.  Errors: G < 0 CATQ_ERR_SHAPE; a null
 * pointer, t < 1, a negative or non-finite lr or out-of-range hyperparameters
 * CATQ_ERR_INVALID_ARG. */
catq_status catq_factor_adamw_step(int64_t G, float* d_mu, float* d_alpha, float* d_delta, const float* g_dmu,
                                   const float* g_dalpha, const float* g_ddelta, float* moments,
                                   const catq_adamw* hp, int64_t t, float lr, catq_stream stream);

/* Direct learning (DL) of a group's scale and threshold, the alternative to the modulation
 * that §2.2 compares (Fig. fig:error; the paper gives no formula, so this is the library's
 * reading).  DL learns alpha and the weight-space threshold Delta_W = alpha Delta with mu
 * fixed at mu0 (0 for the static rules it starts from, e.g. CATQ_THR_ABSMEAN), in units of
 * the group's static statistics, so that the paper's learning rate means the same relative
 * step as for the modulation's factors:
 *   a = alpha / alpha0 = d_alpha,   d = Delta_W / (alpha0 Delta0) = d_alpha d_delta.
 * From the factor gradients of catq_soft_ternary_linear_bwd (the same forward, d_mu unused):
 *   dL/da = g_dalpha - g_ddelta d_delta / d_alpha,   dL/dd = g_ddelta / d_alpha,
 * then one AdamW step on a and on d as in catq_factor_adamw_step, the constraints
 * alpha > 0, Delta > 0 as a, d >= hp->margin, and d_alpha = a, d_delta = d / a (in place).
 * moments: [4, G] fp32 device (m_a, m_d, v_a, v_d), zero before the first update.  A group
 * with d_alpha == 0 is left unchanged.  Errors and G == 0 as catq_factor_adamw_step. */
catq_status catq_direct_adamw_step(int64_t G, float* d_alpha, float* d_delta, const float* g_dalpha,
                                   const float* g_ddelta, float* moments, const catq_adamw* hp, int64_t t, float lr,
                                   catq_stream stream);

/* Per-group weight reconstruction error of the hard ternarization (Fig. fig:error):
 *   err[j] = (1/g) sum over group j of (W - Wq)^2,  Wq = alpha Q(What; Delta) (+ mu with
 *   CATQ_RECON_ALPHA_T_MU), with the codes the pack and the HARD forward take.
 * err: [G] fp32 device, 4-byte aligned.  fp32 sums. */
catq_status catq_group_recon_error(const catq_layer* layer, float* err, catq_stream stream);

/* ------------------------------------------------------------------ grouped (MoE) layers
 * A mixture-of-experts layer quantizes every expert's linear like a dense one (App. B.2:
 * experts are quantized, routers are not).  E experts of identical shape are stacked:
 * W [E, N, K] and the per-group arrays [E, G] (expert e's groups follow expert e-1's), so
 * catq_group_stats / catq_modulate_ternarize / catq_hard_ternarize_pack apply unchanged to
 * the stacked layer seen as a dense [E*N, K] layer.  Tokens routed to experts are given
 * expert-sorted: rows row_offsets[e] .. row_offsets[e+1]-1 of X [R, K] / Y [R, N] belong to
 * expert e; row_offsets is a HOST array of E+1 non-decreasing int64 values, row_offsets[0]
 * == 0, row_offsets[E] == R.  Experts with no rows get zero factor gradients. */
typedef struct {
  int32_t E;       /* number of experts */
  int32_t g;       /* group size */
  int64_t N, K;    /* one expert's out_features, in_features */
  int32_t w_dtype; /* catq_dtype */
  int32_t recon;   /* catq_recon, for every expert */
  const void* W;   /* [E, N, K] */
  float* mu0;      /* [E, G] */
  float* alpha0;
  float* delta0;
  const float* d_mu;
  const float* d_alpha;
  const float* d_delta;
  float* op_const; /* [E, 4*G] ([E, 5*G] with CATQ_RECON_ALPHA_T_MU): per expert as
                      catq_layer.op_const */
} catq_grouped_layer;

/* Forward of every expert: Y[rows of e] = X[rows of e] Wq_e^T (Eq. 6 weight per expert).
 * bf16 layers with at most 128 experts and fewer than 2^31 rows run as one persistent
 * launch over every expert's tiles (X, Y 16-byte aligned; op_const as for dense layers);
 * other layers, expert by expert.  Calls on one layer must not overlap on the GPU (they
 * rewrite op_const). */
catq_status catq_grouped_soft_ternary_linear_fwd(const catq_grouped_layer* layer, catq_schedule sched,
                                                 const void* X, const int64_t* row_offsets,
                                                 int32_t x_dtype, void* Y, catq_stream stream);

/* Workspace bytes catq_grouped_soft_ternary_linear_fwd_loss needs on the current device. */
size_t catq_grouped_fwd_loss_workspace_bytes(const catq_grouped_layer* layer, const int64_t* row_offsets);

/* Forward of every expert and the reconstruction loss over all routed rows R in one pass
 * (see catq_soft_ternary_linear_fwd_loss; count = R N): loss_out, dY [R, N] (required) and
 * Y [R, N] (nullable) from X [R, K] and Y_ref [R, N] of x_dtype.  bf16 layers with at most
 * 128 experts run one persistent launch over every expert's tiles with the loss in its
 * epilogue; other layers compute Y expert by expert (into dY when Y is NULL), then the
 * loss.  R >= 1 (else CATQ_ERR_SHAPE). */
catq_status catq_grouped_soft_ternary_linear_fwd_loss(const catq_grouped_layer* layer, catq_schedule sched,
                                                      const void* X, const int64_t* row_offsets, int32_t x_dtype,
                                                      const void* Y_ref, int32_t reduction, float* loss_out,
                                                      void* dY, void* Y, void* workspace, size_t ws_bytes,
                                                      catq_stream stream);

/* Workspace bytes catq_grouped_soft_ternary_linear_bwd needs: for bf16 layers with at most
 * 128 experts, every expert's partial group sums at once (E * 3 * N * K/gcd(g, 128) fp32);
 * otherwise the largest expert's catq_bwd_workspace_bytes. */
size_t catq_grouped_bwd_workspace_bytes(const catq_grouped_layer* layer, const int64_t* row_offsets);

/* Backward of every expert (see catq_soft_ternary_linear_bwd): dX [R, K] (nullable) and the
 * factor gradients [E, G] (all three or none).  For bf16 layers with at most 128 experts,
 * dX runs as one launch over every expert's tiles and the factor gradients as launches of
 * up to 64 experts with rows each (each expert's contraction stops at its last row) plus
 * one reduction; otherwise expert by expert. */
catq_status catq_grouped_soft_ternary_linear_bwd(const catq_grouped_layer* layer, catq_schedule sched,
                                                 const void* X, const void* dY,
                                                 const int64_t* row_offsets, int32_t x_dtype,
                                                 void* dX, float* g_dmu, float* g_dalpha,
                                                 float* g_ddelta, void* workspace, size_t ws_bytes,
                                                 catq_stream stream);

/* Inference with the deployed form of a calibrated layer (App. B.2: only the ternary codes
 * and the group scale are kept, W ~ alpha T, Eq. 4):
 *   Y[b, n] = sum_k X[b, k] * (alpha[n * K/g + k/g] * T[n, k] + mu[n * K/g + k/g])
 * with T[n, k] read from `codes` in catq_hard_ternarize_pack's layout (element e = n*K + k
 * of row-major W stores T + 1 in bits 2(e%4)..2(e%4)+1 of byte e/4), alpha [N*K/g] fp32
 * (that call's alpha output) and mu [N*K/g] fp32 (its mu output, for a layer calibrated with
 * CATQ_RECON_ALPHA_T_MU; NULL for the W ~ alpha T form, mu = 0).  X [B, K] and Y [B, N] are
 * row-major bf16 (x_dtype must be CATQ_BF16), fp32 accumulation, one rounding of Y.  Meant
 * for decode-shaped B (a few token rows); B == 0 is a no-op.  g must be a multiple of 64
 * and divide K.  codes and X 16-byte aligned, alpha and mu 4-byte, Y 2-byte aligned; all
 * device pointers owned by the caller. */
catq_status catq_ternary_infer(const uint8_t* codes, const float* alpha, const float* mu, int64_t N, int64_t K,
                               int32_t g, const void* X, int64_t B, int32_t x_dtype, void* Y,
                               catq_stream stream);

/* One layer of catq_ternary_infer_batched (device pointers owned by the caller, layouts as in
 * catq_ternary_infer). */
typedef struct {
  const uint8_t* codes; /* [N*K/4], 16-byte aligned */
  const float* alpha;   /* [N*K/g] */
  const float* mu;      /* [N*K/g] or NULL; NULL for every layer or for none */
  int64_t N, K;
  const void* X;        /* [B, K] bf16, 16-byte aligned */
  void* Y;              /* [B, N] bf16 */
} catq_infer_layer;

/* Maximum layers of one catq_ternary_infer_batched call. */
int32_t catq_ternary_infer_max_layers(void);

/* catq_ternary_infer for several layers of group size g and B token rows in one persistent
 * launch (this library's addition; the paper's deployment runs layers one by one).  Each
 * layer's Y depends only on its own codes, scales and X, so the layers must be independent of
 * each other within the call (e.g. the q, k and v projections of a block, or gate and up):
 * no layer's X may be another's Y.  The launch walks every layer's 16-row blocks as one
 * stream of code slabs, so the next block's codes load while the current one computes.
 * layers: HOST array of n_layers entries, 1 <= n_layers <= catq_ternary_infer_max_layers().
 * Errors as catq_ternary_infer for each layer; mixing layers with and without mu is
 * CATQ_ERR_INVALID_ARG. */
catq_status catq_ternary_infer_batched(const catq_infer_layer* layers, int32_t n_layers, int32_t g, int64_t B,
                                       int32_t x_dtype, catq_stream stream);

/* Maximum stages of one catq_ternary_infer_staged call, and the bytes of its sync buffer. */
int32_t catq_ternary_infer_max_stages(void);
size_t catq_ternary_infer_sync_bytes(void);

/* The layers of a decode step in dependency order in one launch (this library's addition,
 * like catq_ternary_infer_batched): layer i belongs to stage stage_of_layer[i] (a HOST array;
 * 0 for the first layer, then non-decreasing in steps of 1, at most
 * catq_ternary_infer_max_stages() stages).  Layers of one stage are independent of each
 * other; a layer of stage s + 1 may read, as its X, the Y of a layer of an earlier stage (e.g.
 * q/k/v -> o -> gate/up -> down of consecutive blocks).  Each layer computes exactly what
 * catq_ternary_infer computes.  The launch is cooperative (every CTA resident at once) and
 * the stages meet at device-wide barriers whose waits are bounded: on expiry the call latches
 * CATQ_ERR_TIMEOUT (read with catq_device_status) and its outputs are undefined.  Copies of
 * the next stage's codes start before its barrier, so the weight stream does not stop at a
 * stage boundary.  sync: device memory of catq_ternary_infer_sync_bytes() bytes, 4-byte
 * aligned, zero before the first call (e.g. cudaMemset); every call, completed or timed out,
 * leaves it zero again.  Calls that may run at the same time (other streams) need separate
 * sync buffers.  Errors as catq_ternary_infer_batched; a missing or malformed stage array or
 * a NULL sync: CATQ_ERR_INVALID_ARG. */
catq_status catq_ternary_infer_staged(const catq_infer_layer* layers, int32_t n_layers, const int32_t* stage_of_layer,
                                      int32_t g, int64_t B, int32_t x_dtype, uint32_t* sync, catq_stream stream);

/* ------------------------------------------------------------------ decoder-block layers
 * Eq. 7 reconstructs the output of a sliding window of layers (§2.4); with a window of one
 * decoder block the loss reaches each linear's factors through the layers
 * between the linears.  These calls are those layers for the Llama / Qwen block (pre-norm,
 * causal grouped-query attention with rotary position embedding, SwiGLU MLP), forward and
 * backward, on bf16 activations with fp32 arithmetic and an fp32 residual stream.  Tokens are
 * rows t = b S + s of [T = B S, *]
 * row-major activations; every activation pointer is device memory, 16-byte aligned, owned by
 * the caller; vectors (gamma, r, lse) are fp32.  T == 0 (or n == 0) is a no-op.  Errors:
 * negative sizes or a violated shape rule CATQ_ERR_SHAPE, a required NULL pointer
 * CATQ_ERR_INVALID_ARG, misalignment CATQ_ERR_ALIGN, a failed launch CATQ_ERR_CUDA. */

/* RMSNorm of each row, with the residual add fused in front:
 *   h = X + residual (in fp32, never rounded; h = X when residual is NULL), stored into h_out
 *       when it is given (the block's residual stream, kept in fp32);
 *   r[t] = 1 / sqrt(mean_i h[t,i]^2 + eps),  Z = gamma * h * r  (bf16).
 * X [T, H] has x_dtype (CATQ_BF16 or CATQ_F32), residual [T, H] bf16, h_out [T, H] fp32,
 * Z [T, H] bf16; gamma [H]; r [T] (kept for the backward).  H % 8 == 0, eps >= 0. */
catq_status catq_rmsnorm_fwd(const void* X, int32_t x_dtype, const void* residual, const float* gamma, int64_t T,
                             int64_t H, float eps, float* h_out, void* Z, float* r, catq_stream stream);

/* Backward of catq_rmsnorm_fwd at h (its input, or the stored residual sum; h_dtype
 * CATQ_BF16 or CATQ_F32):
 *   u = gamma * (dZ + dZ2),  dX = r u - h r^3 mean_i(u h) (+ d_residual)
 * dZ2 (a second consumer of Z, e.g. the gate and up projections) and d_residual (the
 * gradient reaching h around the norm) are nullable; dZ, dZ2, d_residual, dX bf16.  dX may
 * alias dZ, dZ2 or d_residual. */
catq_status catq_rmsnorm_bwd(const void* h, int32_t h_dtype, const float* gamma, const float* r, const void* dZ,
                             const void* dZ2, const void* d_residual, int64_t T, int64_t H, void* dX,
                             catq_stream stream);

/* Rotary position embedding in place on X [T, n_heads d]: in every head, elements i and
 * i + d/2 rotate together by the angle s base^(-2i/d), s = t mod S the token's position
 * (inverse != 0: by its negative, which is the backward of the rotation).  d even, 8 <= d,
 * S >= 1, base > 1. */
catq_status catq_rope(void* X, int64_t T, int64_t S, int32_t n_heads, int32_t d, float base, int32_t inverse,
                      catq_stream stream);

/* SwiGLU: M = silu(gate) * up elementwise over n elements. */
catq_status catq_swiglu_fwd(const void* gate, const void* up, int64_t n, void* M, catq_stream stream);

/* Backward of catq_swiglu_fwd: d_gate = dM up sigma(gate) (1 + gate (1 - sigma(gate))),
 * d_up = dM silu(gate). */
catq_status catq_swiglu_bwd(const void* gate, const void* up, const void* dM, int64_t n, void* d_gate, void* d_up,
                            catq_stream stream);

/* The block output and Eq. 7's loss on it, in one pass over count elements:
 *   out = h + branch          (h fp32, the residual stream; branch bf16, e.g. the down
 *                              projection's output); stored into out (fp32) when given;
 *   with out_ref (fp32, the teacher block's output; NULL computes out only):
 *   loss_out[0] = sum (out - out_ref)^2 / count (CATQ_REDUCE_MEAN) or the plain sum (SUM),
 *   d_out = 2 (out - out_ref) / count (MEAN) or 2 (out - out_ref) (SUM), rounded once to
 *   bf16 (nullable).
 * The difference is taken in fp32 before any rounding, so the residual stream's magnitude
 * does not swamp the student-teacher difference.  count % 8 == 0.  With out_ref: loss_out
 * (device fp32 scalar) required, workspace >= catq_recon_loss_workspace_bytes(count),
 * 256-byte aligned (else CATQ_ERR_WORKSPACE).  Summation as in catq_recon_loss
 * (deterministic). */
catq_status catq_block_output_loss(const float* h, const void* branch, int64_t count, const float* out_ref,
                                   int32_t reduction, float* loss_out, void* d_out, float* out, void* workspace,
                                   size_t ws_bytes, catq_stream stream);

/* Causal grouped-query attention of the decoder block that forms the reconstruction window
 * of Eq. 7 (§2.4): query head h uses key/value head h / (n_heads / n_kv_heads),
 *   O = softmax(Q K^T / sqrt(d), keys s' <= s) V   for every sequence b and head h,
 * with Q, O [B S, n_heads d], K, V [B S, n_kv_heads d] (bf16, device, row-major, caller-owned),
 * and lse [B, n_heads, S] (device fp32) the natural log-sum-exp of each row's scaled scores
 * (kept for the backward).  Scores, the softmax and the accumulation run in fp32; the
 * probabilities enter P V in bf16.  d is 64 or 128; S % 64 == 0; 0 <= B <= 65535;
 * n_heads % n_kv_heads == 0 (else CATQ_ERR_SHAPE).  Null pointers: CATQ_ERR_INVALID_ARG;
 * Q, K, V, O not 16-byte or lse not 4-byte aligned: CATQ_ERR_ALIGN.  d = 128 with
 * S % 128 == 0 runs on the tcgen05 tensor cores, other shapes on the mma.sync path; the two
 * agree up to rounding. */
catq_status catq_attention_fwd(const void* Q, const void* K, const void* V, int32_t B, int32_t S, int32_t n_heads,
                               int32_t n_kv_heads, int32_t d, void* O, float* lse, catq_stream stream);

/* Backward of catq_attention_fwd from dO [B S, n_heads d] and the forward's O and lse:
 *   dS = P (dO V^T - rowsum(dO O)),  dQ = dS K / sqrt(d),
 *   dK = sum over the heads sharing it of dS^T Q / sqrt(d),  dV = the same sum of P^T dO.
 * delta: device fp32 scratch [B, n_heads, S].  dQ like Q, dK and dV like K; all three are
 * overwritten (no atomics: the result does not depend on scheduling).  Shapes, errors and
 * the choice of kernels as for catq_attention_fwd. */
catq_status catq_attention_bwd(const void* Q, const void* K, const void* V, const void* O, const void* dO,
                               const float* lse, int32_t B, int32_t S, int32_t n_heads, int32_t n_kv_heads,
                               int32_t d, float* delta, void* dQ, void* dK, void* dV, catq_stream stream);

/* Self-test of the device-side failure detection (no counterpart in the paper): launches
 * one thread that waits, through the library's bounded mbarrier wait, on a barrier nothing
 * arrives on.  After timeout_ns (1 us .. 1 s) the wait gives up, latches CATQ_ERR_TIMEOUT
 * in the status word and the kernel returns; nothing faults and the context stays usable.
 * Read the result with catq_device_status.  Out-of-range timeouts: CATQ_ERR_INVALID_ARG. */
catq_status catq_selftest_wait_timeout(uint64_t timeout_ns, catq_stream stream);

/* Synchronises `stream`, then returns in *out the status latched on the current device
 * since the last call (CATQ_OK if none) and clears it.  The return value reports whether
 * the query itself succeeded. */
catq_status catq_device_status(catq_stream stream, int32_t* out);

#ifdef __cplusplus
}
#endif

#endif /* CATQ_H */
