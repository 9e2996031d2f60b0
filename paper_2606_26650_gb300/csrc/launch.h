// launch.h — host-side launchers shared between the C-ABI layer (api.cu) and the kernel
// translation units.  Arguments are validated by api.cu before any of these is called.
#pragma once
#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>

#include "catq_math.cuh"

namespace catq {

struct StepScalars {
  int32_t phase;
  float s;
  float inv_2tanh_s;  // 1 / (2 tanh s); 0 when unused
};

// elementwise.cu
cudaError_t launch_group_stats(const LayerDev& L, int32_t w_dtype, int32_t thr_init, float* mu0, float* alpha0,
                               float* delta0, cudaStream_t st);
cudaError_t launch_modulate_ternarize(const LayerDev& L, int32_t w_dtype, StepScalars sc, void* Wq, int8_t* T,
                                      float* alpha, cudaStream_t st);
int recon_loss_blocks(int64_t count);
// loss[0] = out_scale * (sum of n fp64 partials), in a fixed order.
cudaError_t launch_loss_final(const double* partials, int n, double out_scale, float* loss, cudaStream_t st);
cudaError_t launch_recon_loss(const void* Y, const void* Yr, int64_t count, int32_t dtype, int32_t reduction,
                              float* loss_out, void* dY, double* partials, cudaStream_t st);
cudaError_t launch_hard_pack(const LayerDev& L, int32_t w_dtype, uint8_t* codes, float* alpha, float* mu,
                             cudaStream_t st);
// Per-token symmetric 8-bit quantization of X [M, K] (dtype 1 bf16, 0 fp32): scale[m] =
// max|X[m, :]| / 127, codes q = rint(X / scale) in [-127, 127] written as exact values of
// the same dtype, and (nullable) the dequantized scale q rounded once to that dtype.
cudaError_t launch_act_quant_a8(const void* X, int64_t M, int64_t K, int32_t dtype, void* codes, float* scale,
                                void* deq, cudaStream_t st);
// Sums the partial group sums of the dW epilogue ([splits][3][N][K/P]) into the factor
// gradients and applies the per-group scales.
cudaError_t launch_grad_reduce(const LayerDev& L, StepScalars sc, const float* partials, int32_t splits, int32_t P,
                               float* g_dmu, float* g_dalpha, float* g_ddelta, cudaStream_t st);

// simt_f32.cu (fp32 CUDA-core path)
// row_scale (nullable): Y row m is multiplied by row_scale[m].
cudaError_t launch_simt_fwd(const LayerDev& L, StepScalars sc, const float* X, int64_t M, float* Y, cudaStream_t st,
                            const float* row_scale = nullptr);
cudaError_t launch_simt_dx(const LayerDev& L, StepScalars sc, const float* dY, int64_t M, float* dX, cudaStream_t st);
cudaError_t launch_simt_dw(const LayerDev& L, StepScalars sc, const float* X, const float* dY, int64_t M,
                           float* partials, cudaStream_t st);
constexpr int32_t kSimtTile = 64;

// tc_gemm.cu (bf16 tensor-core path)
struct TcPlan {
  int32_t dw_cg;      // CTA group of the dW kernel (1 or 2)
  int32_t dw_splits;  // contraction splits of the dW kernel
  int32_t dw_P;       // partial-sum chunk width (columns)
};
TcPlan tc_plan_bwd(const LayerDev& L, int64_t M, int sm_count);
// Epilogue options of the bf16 forward (defaults: Y stored in bf16).
struct EpiOpts {
  bool y_f32 = false;               // store Y in fp32
  const float* row_scale = nullptr; // [M] per-row scale of the accumulator (8-bit activation codes)
  const void* yref = nullptr;       // fused Eq. 7 loss against this teacher output [M, N]
  bool yref_f32 = false;
  float dscale = 0.0f;              // dY = dscale (Y - Y_ref)
  void* dY = nullptr;               // bf16 [M, N]
  double* loss_part = nullptr;      // partial sums of (Y - Y_ref)^2
  int* n_parts = nullptr;           // out: partials written
};
// Y [B, N] = X [B, K] (alpha T + mu)^T from 2-bit codes, group scales and (nullable) group
// offsets (bf16 X and Y).
cudaError_t launch_ternary_infer(const uint8_t* codes, const float* alpha, const float* mu, int64_t N, int64_t K,
                                 int32_t g, const void* X, int64_t B, void* Y, cudaStream_t st);
// Several layers of one group size in one persistent launch (at most ternary_infer_max_layers()).
struct InferDesc {
  const uint8_t* codes;
  const float* alpha;
  const float* mu;
  int64_t N, K;
  const void* X;
  int64_t B;
  void* Y;
};
int ternary_infer_max_layers();
cudaError_t launch_ternary_infer_batched(const InferDesc* layers, int n, int32_t g, cudaStream_t st);
// A chain of layer sets in one cooperative launch: layer i belongs to stage stage_of[i]
// (0, then non-decreasing in steps of 1); stage s + 1 may read what stage s wrote.  sync:
// ternary_infer_sync_bytes() of device memory, zero on entry, zero again on exit.
int ternary_infer_max_stages();
size_t ternary_infer_sync_bytes();
cudaError_t launch_ternary_infer_staged(const InferDesc* layers, int n, const int32_t* stage_of, int32_t g,
                                        uint32_t* sync, cudaStream_t st);

// Wait control (abort word, status word, epoch, time limit) for one launch of a kernel with
// bounded waits; false when the device's status words are unavailable.
struct WaitCtl;
bool launch_wait_ctl(WaitCtl* out);

// One-thread kernel whose bounded wait runs out after timeout_ns (self-test).
cudaError_t launch_wait_probe(uint64_t timeout_ns, cudaStream_t st);

// One AdamW step on the three factor arrays p[q] with gradients g[q] and moments m[q], v[q]
// (q = mu, alpha, delta; each [G] fp32), then the projection onto [lo[q], hi[q]].  The
// scalars that depend only on the update count are folded on the host.
struct AdamwArgs {
  float* p[3];
  const float* g[3];
  float* m[3];
  float* v[3];
  float decay;        // 1 - lr weight_decay
  float beta1, one_minus_beta1, beta2, one_minus_beta2;
  float step;         // lr / (1 - beta1^t)
  float inv_sqrt_bc2; // 1 / sqrt(1 - beta2^t)
  float eps;
  float lo[3], hi[3];
};
cudaError_t launch_factor_adamw(int64_t G, const AdamwArgs& a, cudaStream_t st);

// Direct learning's update of (d_alpha, d_delta) (see catq_direct_adamw_step): moments m[2G]
// (a, then d) and v[2G]; the scalars as in AdamwArgs; the projection floor `margin`.
struct DirectArgs {
  float* d_alpha;
  float* d_delta;
  const float* g_dalpha;
  const float* g_ddelta;
  float* m;
  float* v;
  float decay, beta1, one_minus_beta1, beta2, one_minus_beta2, step, inv_sqrt_bc2, eps, margin;
};
cudaError_t launch_direct_adamw(int64_t G, const DirectArgs& a, cudaStream_t st);

// err[j] = mean over group j of (W - alpha Q(What; Delta) [- mu])^2.
cudaError_t launch_group_recon_error(const LayerDev& L, int32_t w_dtype, float* err, cudaStream_t st);

// Writes L.op_const (operand_const_vec of every group, [K/g][N]) for schedule point sc.
cudaError_t launch_operand_consts(const LayerDev& L, StepScalars sc, cudaStream_t st);

// Grouped (MoE) launches: E experts of identical shape, L0 is expert 0's layer with the
// stacked weights [E N, K] from L0.W on; per-group arrays of expert e start e G after
// expert 0's, its operand constants const_stride floats after; rows of A and C are
// expert-sorted with host offsets off[0..E].
constexpr int32_t kGroupedMaxExperts = 128;
struct GroupSpec {
  int32_t E;
  const int64_t* off;
  int64_t const_stride;
};
cudaError_t launch_operand_consts_grouped(const LayerDev& L0, StepScalars sc, int32_t E, int64_t const_stride,
                                          cudaStream_t st);
cudaError_t launch_tc_fwd_grouped(const LayerDev& L0, StepScalars sc, const void* X, const GroupSpec& grp, void* Y,
                                  cudaStream_t st, const EpiOpts* opts = nullptr);
cudaError_t launch_tc_dx_grouped(const LayerDev& L0, StepScalars sc, const void* dY, const GroupSpec& grp, void* dX,
                                 cudaStream_t st);
// Partial group sums of every expert with rows, [E][3][N][K/P] (P = gcd(g, 128)).
cudaError_t launch_tc_dw_grouped(const LayerDev& L0, StepScalars sc, const void* X, const void* dY,
                                 const GroupSpec& grp, int32_t P, float* partials, cudaStream_t st);
// Factor gradients [E G] from those partials; zeros for experts without rows.
cudaError_t launch_grad_reduce_grouped(const LayerDev& L0, StepScalars sc, const float* partials, int32_t P,
                                       const GroupSpec& grp, float* g_dmu, float* g_dalpha, float* g_ddelta,
                                       cudaStream_t st);

// Upper bound of EpiOpts::n_parts for any launch on a device with `sm_count` SMs.
int fused_loss_max_parts(int sm_count);
cudaError_t launch_tc_fwd(const LayerDev& L, StepScalars sc, const void* X, int64_t M, void* Y, cudaStream_t st,
                         const EpiOpts* opts = nullptr);
cudaError_t launch_tc_dx(const LayerDev& L, StepScalars sc, const void* dY, int64_t M, void* dX, cudaStream_t st);
cudaError_t launch_tc_dw(const LayerDev& L, StepScalars sc, const void* X, const void* dY, int64_t M,
                         const TcPlan& plan, float* partials, cudaStream_t st);
// block.cu (the layers between the linears of a decoder block; bf16 activations)
// x (fp32 or bf16) + res (bf16, nullable) -> h_out (fp32, nullable), z (bf16), r.
cudaError_t launch_rmsnorm_fwd(const void* x, bool x_f32, const void* res, const float* gamma, int64_t T, int64_t H,
                               float eps, float* h_out, void* z, float* r, cudaStream_t st);
cudaError_t launch_rmsnorm_bwd(const void* x, bool x_f32, const float* gamma, const float* r, const void* dy,
                               const void* dy2, const void* dres, int64_t T, int64_t H, void* dx, cudaStream_t st);
cudaError_t launch_rope(void* x, int64_t T, int64_t S, int32_t nheads, int32_t d, float base, int32_t inverse,
                        cudaStream_t st);
// dm == nullptr: out = silu(gt) u; else dgt, du = the backward from dm.
cudaError_t launch_swiglu(const void* gt, const void* u, const void* dm, int64_t n, void* out, void* dgt, void* du,
                          cudaStream_t st);
// out = h + branch (fp32; nullable); with ref: loss_out = Eq. 7 loss, d_out (bf16, nullable);
// partials: recon_loss_blocks(count) doubles.  count % 8 == 0.
cudaError_t launch_block_output_loss(const float* h, const void* branch, const float* ref, int64_t count,
                                     int32_t reduction, float* out, void* d_out, float* loss_out, double* partials,
                                     cudaStream_t st);
struct AttnIo {
  const void *q, *k, *v;
  const void *o, *dO;  // backward only
  void* out;           // forward only
  void *dq, *dk, *dv;  // backward only
  float* lse;
  float* delta;        // backward scratch
};
cudaError_t launch_attention(const AttnIo& io, int32_t B, int32_t S, int32_t nh, int32_t nkv, int32_t d, bool backward,
                             cudaStream_t st);
// The forward on the tcgen05 tensor cores (attn_tc.cu): head dimension 128, S a multiple of 128.
bool attention_fwd_tc_supported(int32_t S, int32_t d);
cudaError_t launch_attention_fwd_tc(const void* q, const void* k, const void* v, void* out, float* lse, int32_t B,
                                    int32_t S, int32_t nh, int32_t nkv, cudaStream_t st);
// dQ, dK, dV on tcgen05 from the forward's log-sum-exp and delta = rowsum(dO * O).
cudaError_t launch_attention_bwd_tc(const void* q, const void* k, const void* v, const void* dO, const float* lse,
                                    const float* delta, void* dq, void* dk, void* dv, int32_t B, int32_t S, int32_t nh,
                                    int32_t nkv, cudaStream_t st);
// Status word latched by device-side bounded waits (0 = none); read-and-clear.
cudaError_t read_and_clear_device_status(int32_t* out);
bool tensor_map_encoder_available();

}  // namespace catq
