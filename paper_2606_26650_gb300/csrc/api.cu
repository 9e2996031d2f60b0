// api.cu — the extern "C" boundary (include/catq.h): argument validation, dtype routing
// (bf16 -> tensor-core kernels, fp32 -> CUDA-core kernels) and workspace sizing.  Nothing
// here allocates memory; every launch goes to the caller's stream.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdint>
#include <mutex>
#include <numeric>

#include "catq.h"
#include "launch.h"

using namespace catq;

namespace {

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
bool aligned256(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 255u) == 0; }

size_t round256(size_t b) { return (b + 255) & ~static_cast<size_t>(255); }

catq_status cuda_status(cudaError_t e) { return e == cudaSuccess ? CATQ_OK : CATQ_ERR_CUDA; }

// Shape / dtype / pointer checks common to every layer call.  `need_factors` also requires
// the statistics and learnable-factor arrays.
catq_status check_layer(const catq_layer* L, bool need_factors) {
  if (!L || !L->W) return CATQ_ERR_INVALID_ARG;
  if (L->w_dtype != CATQ_F32 && L->w_dtype != CATQ_BF16) return CATQ_ERR_DTYPE;
  if (L->N < 1 || L->K < 1 || L->g < 1) return CATQ_ERR_SHAPE;
  if (L->K % L->g != 0) return CATQ_ERR_SHAPE;
  if (L->N * L->K / L->g >= (int64_t(1) << 31) || L->N >= (int64_t(1) << 31) || L->K >= (int64_t(1) << 31))
    return CATQ_ERR_SHAPE;  // group and row indices are 32-bit inside the kernels
  if (L->w_dtype == CATQ_BF16) {
    if (L->g % 64 != 0 || L->N % 8 != 0) return CATQ_ERR_SHAPE;
  } else {
    if (!(L->g % 64 == 0 || L->g == 4 || L->g == 8 || L->g == 16 || L->g == 32)) return CATQ_ERR_SHAPE;
  }
  if (!aligned16(L->W)) return CATQ_ERR_ALIGN;
  if (L->recon != CATQ_RECON_ALPHA_T && L->recon != CATQ_RECON_ALPHA_T_MU) return CATQ_ERR_INVALID_ARG;
  if (L->reserved != 0) return CATQ_ERR_INVALID_ARG;
  if (!L->mu0 || !L->alpha0 || !L->delta0) return CATQ_ERR_INVALID_ARG;
  if (need_factors && (!L->d_mu || !L->d_alpha || !L->d_delta)) return CATQ_ERR_INVALID_ARG;
  return CATQ_OK;
}

// The fused bf16 GEMMs of a SOFT or HARD step read their operand constants from op_const.
catq_status check_op_const(const catq_layer* L, catq_schedule sc) {
  if (L->w_dtype != CATQ_BF16 || sc.phase == CATQ_PHASE_TEACHER) return CATQ_OK;
  if (!L->op_const) return CATQ_ERR_INVALID_ARG;
  return aligned16(L->op_const) ? CATQ_OK : CATQ_ERR_ALIGN;
}

catq_status check_schedule(catq_schedule sc, bool need_s) {
  if (sc.phase != CATQ_PHASE_TEACHER && sc.phase != CATQ_PHASE_SOFT && sc.phase != CATQ_PHASE_HARD)
    return CATQ_ERR_INVALID_ARG;
  if (need_s && !(std::isfinite(sc.s) && sc.s > 0.0f)) return CATQ_ERR_INVALID_ARG;
  return CATQ_OK;
}

LayerDev to_dev(const catq_layer* L) {
  LayerDev d;
  d.W = L->W;
  d.N = L->N;
  d.K = L->K;
  d.g = L->g;
  d.groups_per_row = static_cast<int32_t>(L->K / L->g);
  d.mu0 = L->mu0;
  d.alpha0 = L->alpha0;
  d.delta0 = L->delta0;
  d.d_mu = L->d_mu;
  d.d_alpha = L->d_alpha;
  d.d_delta = L->d_delta;
  d.op_const = reinterpret_cast<float4*>(L->op_const);
  d.recon = L->recon;
  d.op_mu = (L->recon && L->op_const) ? L->op_const + 4 * (L->N * L->K / L->g) : nullptr;
  return d;
}

StepScalars scalars(catq_schedule sc) {
  StepScalars s;
  s.phase = sc.phase;
  s.s = sc.s;
  const double t = (sc.s > 0.0f && std::isfinite(sc.s)) ? std::tanh(static_cast<double>(sc.s)) : 0.0;
  s.inv_2tanh_s = t > 0.0 ? static_cast<float>(1.0 / (2.0 * t)) : 0.0f;
  return s;
}

// The bf16 path needs an sm_100-class GPU (tcgen05, TMA) and the driver's tensor-map encoder.
catq_status check_tensor_core_device() {
  int dev = 0, major = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return CATQ_ERR_CUDA;
  if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess) return CATQ_ERR_CUDA;
  if (major != 10) return CATQ_ERR_UNSUPPORTED;
  if (!tensor_map_encoder_available()) return CATQ_ERR_UNSUPPORTED;
  return CATQ_OK;
}

int current_sm_count() {
  int dev = 0, n = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
  return n > 0 ? n : 1;
}

size_t bwd_partials_bytes(const catq_layer* L, int64_t M, TcPlan* plan_out, int32_t* P_out, int32_t* splits_out) {
  if (L->w_dtype == CATQ_BF16) {
    const TcPlan p = tc_plan_bwd(to_dev(L), M, current_sm_count());
    if (plan_out) *plan_out = p;
    if (P_out) *P_out = p.dw_P;
    if (splits_out) *splits_out = p.dw_splits;
    return static_cast<size_t>(p.dw_splits) * 3 * static_cast<size_t>(L->N) * static_cast<size_t>(L->K / p.dw_P) *
           sizeof(float);
  }
  const int32_t P = L->g < kSimtTile ? L->g : kSimtTile;
  if (P_out) *P_out = P;
  if (splits_out) *splits_out = 1;
  return 3 * static_cast<size_t>(L->N) * static_cast<size_t>(L->K / P) * sizeof(float);
}

// Fused-loss workspace: the fp64 loss partials (one per epilogue warp of the bf16 GEMM, or
// the loss kernel's block partials on the fp32 path).
size_t fwd_loss_ws_bytes(int64_t count) {
  const int parts = std::max(fused_loss_max_parts(current_sm_count()), recon_loss_blocks(count < 1 ? 1 : count));
  return round256(static_cast<size_t>(parts) * sizeof(double));
}

// Scratch of catq_soft_ternary_linear_bwd_noalloc: the dW epilogue's partial group sums.
// Every GPU that loads the library holds this array until the process exits.
constexpr size_t kNoAllocScratchBytes = size_t(16) << 20;
static __device__ __align__(256) unsigned char g_bwd_scratch[kNoAllocScratchBytes];

// Device address of g_bwd_scratch on the current device, looked up once per device with
// that device current (host code cannot use the array's name as a device address).
catq_status noalloc_scratch(void** out) {
  static std::mutex mu;
  static void* addr[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return CATQ_ERR_CUDA;
  std::lock_guard<std::mutex> lock(mu);
  if (!addr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_bwd_scratch) != cudaSuccess || !p) return CATQ_ERR_CUDA;
    addr[dev] = p;
  }
  *out = addr[dev];
  return CATQ_OK;
}

}  // namespace

extern "C" {

int32_t catq_abi_version(void) { return CATQ_ABI_VERSION; }

const char* catq_status_string(int32_t s) {
  switch (s) {
    case CATQ_OK: return "CATQ_OK";
    case CATQ_ERR_INVALID_ARG: return "CATQ_ERR_INVALID_ARG";
    case CATQ_ERR_SHAPE: return "CATQ_ERR_SHAPE";
    case CATQ_ERR_DTYPE: return "CATQ_ERR_DTYPE";
    case CATQ_ERR_ALIGN: return "CATQ_ERR_ALIGN";
    case CATQ_ERR_CUDA: return "CATQ_ERR_CUDA";
    case CATQ_ERR_TIMEOUT: return "CATQ_ERR_TIMEOUT";
    case CATQ_ERR_NONFINITE: return "CATQ_ERR_NONFINITE";
    case CATQ_ERR_UNSUPPORTED: return "CATQ_ERR_UNSUPPORTED";
    case CATQ_ERR_WORKSPACE: return "CATQ_ERR_WORKSPACE";
    default: return "CATQ_ERR_UNKNOWN";
  }
}

catq_status catq_group_stats(const catq_layer* layer, int32_t thr_init, catq_stream stream) {
  catq_status st = check_layer(layer, false);
  if (st != CATQ_OK) return st;
  if (thr_init != CATQ_THR_HALF && thr_init != CATQ_THR_TWN07 && thr_init != CATQ_THR_ABSMEAN &&
      thr_init != CATQ_THR_TWN_STATIC)
    return CATQ_ERR_INVALID_ARG;
  const LayerDev L = to_dev(layer);
  return cuda_status(launch_group_stats(L, layer->w_dtype, thr_init, layer->mu0, layer->alpha0, layer->delta0,
                                        reinterpret_cast<cudaStream_t>(stream)));
}

catq_status catq_modulate_ternarize(const catq_layer* layer, catq_schedule sched, void* Wq_out, int8_t* T_out,
                                    float* alpha_out, catq_stream stream) {
  catq_status st = check_layer(layer, true);
  if (st != CATQ_OK) return st;
  if ((st = check_schedule(sched, sched.phase == CATQ_PHASE_SOFT)) != CATQ_OK) return st;
  if (Wq_out && !aligned16(Wq_out)) return CATQ_ERR_ALIGN;
  if (T_out && !aligned16(T_out)) return CATQ_ERR_ALIGN;
  if (!Wq_out && !T_out && !alpha_out) return CATQ_OK;
  return cuda_status(launch_modulate_ternarize(to_dev(layer), layer->w_dtype, scalars(sched), Wq_out, T_out,
                                               alpha_out, reinterpret_cast<cudaStream_t>(stream)));
}

catq_status catq_soft_ternary_linear_fwd(const catq_layer* layer, catq_schedule sched, const void* X, int64_t M,
                                         int32_t x_dtype, void* Y, catq_stream stream) {
  catq_status st = check_layer(layer, sched.phase != CATQ_PHASE_TEACHER);
  if (st != CATQ_OK) return st;
  if ((st = check_schedule(sched, sched.phase == CATQ_PHASE_SOFT)) != CATQ_OK) return st;
  if (x_dtype != layer->w_dtype) return CATQ_ERR_DTYPE;
  if (M < 0) return CATQ_ERR_SHAPE;
  if (M == 0) return CATQ_OK;
  if (!X || !Y) return CATQ_ERR_INVALID_ARG;
  if (!aligned16(X) || !aligned16(Y)) return CATQ_ERR_ALIGN;
  if ((st = check_op_const(layer, sched)) != CATQ_OK) return st;
  const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const LayerDev L = to_dev(layer);
  if (layer->w_dtype == CATQ_F32)
    return cuda_status(launch_simt_fwd(L, scalars(sched), static_cast<const float*>(X), M, static_cast<float*>(Y), s));
  if ((st = check_tensor_core_device()) != CATQ_OK) return st;
  return cuda_status(launch_tc_fwd(L, scalars(sched), X, M, Y, s));
}

catq_status catq_soft_ternary_linear_fwd_ex(const catq_layer* layer, catq_schedule sched, const void* X, int64_t M,
                                            int32_t x_dtype, const float* x_row_scale, void* Y, int32_t y_dtype,
                                            catq_stream stream) {
  catq_status st = check_layer(layer, sched.phase != CATQ_PHASE_TEACHER);
  if (st != CATQ_OK) return st;
  if ((st = check_schedule(sched, sched.phase == CATQ_PHASE_SOFT)) != CATQ_OK) return st;
  if (x_dtype != layer->w_dtype) return CATQ_ERR_DTYPE;
  if (y_dtype != x_dtype && y_dtype != CATQ_F32) return CATQ_ERR_DTYPE;
  if (M < 0) return CATQ_ERR_SHAPE;
  if (M == 0) return CATQ_OK;
  if (!X || !Y) return CATQ_ERR_INVALID_ARG;
  if (!aligned16(X) || !aligned16(Y) || (reinterpret_cast<uintptr_t>(x_row_scale) & 3u)) return CATQ_ERR_ALIGN;
  if ((st = check_op_const(layer, sched)) != CATQ_OK) return st;
  const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const LayerDev L = to_dev(layer);
  if (layer->w_dtype == CATQ_F32)
    return cuda_status(
        launch_simt_fwd(L, scalars(sched), static_cast<const float*>(X), M, static_cast<float*>(Y), s, x_row_scale));
  if ((st = check_tensor_core_device()) != CATQ_OK) return st;
  EpiOpts o;
  o.y_f32 = y_dtype == CATQ_F32;
  o.row_scale = x_row_scale;
  return cuda_status(launch_tc_fwd(L, scalars(sched), X, M, Y, s, &o));
}

size_t catq_fwd_loss_workspace_bytes(const catq_layer* layer, int64_t M) {
  if (!layer || layer->N < 1) return 0;
  if (M < 1) M = 1;
  return fwd_loss_ws_bytes(M * layer->N);
}

catq_status catq_soft_ternary_linear_fwd_loss(const catq_layer* layer, catq_schedule sched, const void* X, int64_t M,
                                              int32_t x_dtype, const float* x_row_scale, const void* Y_ref,
                                              int32_t ref_dtype, int32_t reduction, float* loss_out, void* dY,
                                              void* Y, void* workspace, size_t ws_bytes, catq_stream stream) {
  catq_status st = check_layer(layer, sched.phase != CATQ_PHASE_TEACHER);
  if (st != CATQ_OK) return st;
  if ((st = check_schedule(sched, sched.phase == CATQ_PHASE_SOFT)) != CATQ_OK) return st;
  if (x_dtype != layer->w_dtype) return CATQ_ERR_DTYPE;
  if (ref_dtype != x_dtype && ref_dtype != CATQ_F32) return CATQ_ERR_DTYPE;
  if (reduction != CATQ_REDUCE_MEAN && reduction != CATQ_REDUCE_SUM) return CATQ_ERR_INVALID_ARG;
  if (M < 1) return CATQ_ERR_SHAPE;
  if (!X || !Y_ref || !loss_out || !dY) return CATQ_ERR_INVALID_ARG;
  if (!aligned16(X) || !aligned16(Y_ref) || !aligned16(dY) || (Y && !aligned16(Y)) ||
      (reinterpret_cast<uintptr_t>(x_row_scale) & 3u))
    return CATQ_ERR_ALIGN;
  if (!workspace || ws_bytes < catq_fwd_loss_workspace_bytes(layer, M)) return CATQ_ERR_WORKSPACE;
  if (!aligned256(workspace)) return CATQ_ERR_ALIGN;
  if ((st = check_op_const(layer, sched)) != CATQ_OK) return st;
  const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const LayerDev L = to_dev(layer);
  const int64_t count = M * layer->N;
  const double inv = reduction == CATQ_REDUCE_MEAN ? 1.0 / static_cast<double>(count) : 1.0;
  double* part = static_cast<double*>(workspace);
  if (layer->w_dtype == CATQ_F32) {
    // fp32 layers: the CUDA-core forward (into Y, or into dY as scratch), then the loss kernel
    // in place (each element of dY is read before it is written by the same thread)
    float* Yw = static_cast<float*>(Y ? Y : dY);
    if (launch_simt_fwd(L, scalars(sched), static_cast<const float*>(X), M, Yw, s, x_row_scale) != cudaSuccess)
      return CATQ_ERR_CUDA;
    return cuda_status(launch_recon_loss(Yw, Y_ref, count, CATQ_F32, reduction, loss_out, dY, part, s));
  }
  if ((st = check_tensor_core_device()) != CATQ_OK) return st;
  EpiOpts o;
  o.row_scale = x_row_scale;
  o.yref = Y_ref;
  o.yref_f32 = ref_dtype == CATQ_F32;
  o.dscale = static_cast<float>(2.0 * inv);
  o.dY = dY;
  o.loss_part = part;
  int nparts = 0;
  o.n_parts = &nparts;
  if (launch_tc_fwd(L, scalars(sched), X, M, Y, s, &o) != cudaSuccess) return CATQ_ERR_CUDA;
  return cuda_status(launch_loss_final(part, nparts, inv, loss_out, s));
}

catq_status catq_act_quant_a8(const void* X, int64_t M, int64_t K, int32_t x_dtype, void* codes, float* scale,
                              void* X_deq, catq_stream stream) {
  if (x_dtype != CATQ_F32 && x_dtype != CATQ_BF16) return CATQ_ERR_DTYPE;
  if (M < 0 || K < 1) return CATQ_ERR_SHAPE;
  if (K % (x_dtype == CATQ_BF16 ? 8 : 4) != 0) return CATQ_ERR_SHAPE;  // 16-byte rows
  if (M == 0) return CATQ_OK;
  if (!X || !codes || !scale) return CATQ_ERR_INVALID_ARG;
  if (!aligned16(X) || !aligned16(codes) || (X_deq && !aligned16(X_deq)) ||
      (reinterpret_cast<uintptr_t>(scale) & 3u))
    return CATQ_ERR_ALIGN;
  return cuda_status(
      launch_act_quant_a8(X, M, K, x_dtype, codes, scale, X_deq, reinterpret_cast<cudaStream_t>(stream)));
}

size_t catq_bwd_workspace_bytes(const catq_layer* layer, int64_t M) {
  if (!layer || layer->g < 1 || layer->K % layer->g != 0 || layer->N < 1) return 0;
  if (M < 1) M = 1;
  return round256(bwd_partials_bytes(layer, M, nullptr, nullptr, nullptr));
}

catq_status catq_soft_ternary_linear_bwd(const catq_layer* layer, catq_schedule sched, const void* X, const void* dY,
                                         int64_t M, int32_t x_dtype, void* dX, float* g_dmu, float* g_dalpha,
                                         float* g_ddelta, void* workspace, size_t ws_bytes, catq_stream stream) {
  catq_status st = check_layer(layer, sched.phase != CATQ_PHASE_TEACHER);
  if (st != CATQ_OK) return st;
  if ((st = check_schedule(sched, sched.phase != CATQ_PHASE_TEACHER)) != CATQ_OK) return st;
  if (x_dtype != layer->w_dtype) return CATQ_ERR_DTYPE;
  if (M < 0) return CATQ_ERR_SHAPE;
  const bool want_grads = g_dmu || g_dalpha || g_ddelta;
  if (want_grads && !(g_dmu && g_dalpha && g_ddelta)) return CATQ_ERR_INVALID_ARG;
  const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const LayerDev L = to_dev(layer);
  const int64_t G = layer->N * layer->K / layer->g;
  const bool need_dw = want_grads && sched.phase != CATQ_PHASE_TEACHER && M > 0;
  if (M > 0) {
    if (!X || !dY) return CATQ_ERR_INVALID_ARG;
    if (!aligned16(X) || !aligned16(dY) || (dX && !aligned16(dX))) return CATQ_ERR_ALIGN;
    if (dX && (st = check_op_const(layer, sched)) != CATQ_OK) return st;
  }
  TcPlan plan{};
  int32_t P = 0, splits = 0;
  if (need_dw) {
    const size_t need = bwd_partials_bytes(layer, M, &plan, &P, &splits);
    if (!workspace || ws_bytes < need) return CATQ_ERR_WORKSPACE;
    if (!aligned256(workspace)) return CATQ_ERR_ALIGN;
  }
  if (layer->w_dtype == CATQ_BF16 && M > 0 && (st = check_tensor_core_device()) != CATQ_OK) return st;
  const StepScalars sc = scalars(sched);
  cudaError_t e = cudaSuccess;
  if (dX && M > 0) {
    e = layer->w_dtype == CATQ_F32
            ? launch_simt_dx(L, sc, static_cast<const float*>(dY), M, static_cast<float*>(dX), s)
            : launch_tc_dx(L, sc, dY, M, dX, s);
    if (e != cudaSuccess) return CATQ_ERR_CUDA;
  }
  if (!want_grads) return CATQ_OK;
  if (!need_dw) {
    const size_t b = static_cast<size_t>(G) * sizeof(float);
    if (cudaMemsetAsync(g_dmu, 0, b, s) != cudaSuccess || cudaMemsetAsync(g_dalpha, 0, b, s) != cudaSuccess ||
        cudaMemsetAsync(g_ddelta, 0, b, s) != cudaSuccess)
      return CATQ_ERR_CUDA;
    return CATQ_OK;
  }
  float* part = static_cast<float*>(workspace);
  e = layer->w_dtype == CATQ_F32
          ? launch_simt_dw(L, sc, static_cast<const float*>(X), static_cast<const float*>(dY), M, part, s)
          : launch_tc_dw(L, sc, X, dY, M, plan, part, s);
  if (e != cudaSuccess) return CATQ_ERR_CUDA;
  return cuda_status(launch_grad_reduce(L, sc, part, splits, P, g_dmu, g_dalpha, g_ddelta, s));
}

catq_status catq_soft_ternary_linear_bwd_noalloc(const catq_layer* layer, catq_schedule sched, const void* X,
                                                 const void* dY, int64_t M, int32_t x_dtype, void* dX,
                                                 float* g_dmu, float* g_dalpha, float* g_ddelta,
                                                 catq_stream stream) {
  // Same validation and kernels as catq_soft_ternary_linear_bwd; only the scratch differs.
  catq_status st = check_layer(layer, sched.phase != CATQ_PHASE_TEACHER);
  if (st != CATQ_OK) return st;
  const bool want_grads = g_dmu || g_dalpha || g_ddelta;
  if (!want_grads || sched.phase == CATQ_PHASE_TEACHER || M <= 0)
    return catq_soft_ternary_linear_bwd(layer, sched, X, dY, M, x_dtype, dX, g_dmu, g_dalpha, g_ddelta, nullptr,
                                        0, stream);
  if (bwd_partials_bytes(layer, M, nullptr, nullptr, nullptr) > kNoAllocScratchBytes) return CATQ_ERR_WORKSPACE;
  void* scratch = nullptr;
  if ((st = noalloc_scratch(&scratch)) != CATQ_OK) return st;
  return catq_soft_ternary_linear_bwd(layer, sched, X, dY, M, x_dtype, dX, g_dmu, g_dalpha, g_ddelta, scratch,
                                      kNoAllocScratchBytes, stream);
}

size_t catq_bwd_noalloc_max_scratch_bytes(void) { return kNoAllocScratchBytes; }

size_t catq_recon_loss_workspace_bytes(int64_t count) {
  return round256(static_cast<size_t>(recon_loss_blocks(count < 1 ? 1 : count)) * sizeof(double));
}

catq_status catq_recon_loss(const void* Y, const void* Y_ref, int64_t count, int32_t dtype, int32_t reduction,
                            float* loss_out, void* dY, void* workspace, size_t ws_bytes, catq_stream stream) {
  if (dtype != CATQ_F32 && dtype != CATQ_BF16) return CATQ_ERR_DTYPE;
  if (reduction != CATQ_REDUCE_MEAN && reduction != CATQ_REDUCE_SUM) return CATQ_ERR_INVALID_ARG;
  if (count < 1) return CATQ_ERR_SHAPE;
  if (!Y || !Y_ref || !loss_out) return CATQ_ERR_INVALID_ARG;
  if (!aligned16(Y) || !aligned16(Y_ref) || (dY && !aligned16(dY))) return CATQ_ERR_ALIGN;
  if (!workspace || ws_bytes < catq_recon_loss_workspace_bytes(count)) return CATQ_ERR_WORKSPACE;
  if (!aligned256(workspace)) return CATQ_ERR_ALIGN;
  return cuda_status(launch_recon_loss(Y, Y_ref, count, dtype, reduction, loss_out, dY,
                                       static_cast<double*>(workspace), reinterpret_cast<cudaStream_t>(stream)));
}

catq_status catq_hard_ternarize_pack(const catq_layer* layer, uint8_t* codes, float* alpha, float* mu,
                                     catq_stream stream) {
  catq_status st = check_layer(layer, true);
  if (st != CATQ_OK) return st;
  if (!codes) return CATQ_ERR_INVALID_ARG;
  if ((layer->N * layer->K) % 4 != 0) return CATQ_ERR_SHAPE;
  if (layer->g % 16 == 0 && !aligned16(codes)) return CATQ_ERR_ALIGN;
  return cuda_status(launch_hard_pack(to_dev(layer), layer->w_dtype, codes, alpha, mu,
                                      reinterpret_cast<cudaStream_t>(stream)));
}

// ------------------------------------------------------------------ grouped (MoE) layers

namespace {

// Expert e of a stacked layer as a dense layer (pointer offsets only).
catq_layer expert_layer(const catq_grouped_layer* G, int32_t e) {
  const int64_t groups = G->N * G->K / G->g;
  const size_t esize = G->w_dtype == CATQ_BF16 ? 2 : 4;
  catq_layer L;
  L.N = G->N;
  L.K = G->K;
  L.g = G->g;
  L.w_dtype = G->w_dtype;
  L.W = static_cast<const char*>(G->W) + static_cast<size_t>(e) * G->N * G->K * esize;
  L.mu0 = G->mu0 ? G->mu0 + e * groups : nullptr;
  L.alpha0 = G->alpha0 ? G->alpha0 + e * groups : nullptr;
  L.delta0 = G->delta0 ? G->delta0 + e * groups : nullptr;
  L.d_mu = G->d_mu ? G->d_mu + e * groups : nullptr;
  L.d_alpha = G->d_alpha ? G->d_alpha + e * groups : nullptr;
  L.d_delta = G->d_delta ? G->d_delta + e * groups : nullptr;
  L.op_const = G->op_const ? G->op_const + (G->recon ? 5 : 4) * e * groups : nullptr;
  L.recon = G->recon;
  L.reserved = 0;
  return L;
}

catq_status check_grouped(const catq_grouped_layer* G, const int64_t* off) {
  if (!G || !off || G->E < 1) return CATQ_ERR_INVALID_ARG;
  if (off[0] != 0) return CATQ_ERR_SHAPE;
  for (int32_t e = 0; e < G->E; ++e)
    if (off[e + 1] < off[e]) return CATQ_ERR_SHAPE;
  return CATQ_OK;
}

}  // namespace

// Whether the factor gradients of a grouped layer run as grouped launches (bf16, at most
// kGroupedMaxExperts experts, fewer than 2^31 rows); otherwise expert by expert.
bool grouped_dw_ok(const catq_grouped_layer* G, const int64_t* off) {
  return G->w_dtype == CATQ_BF16 && G->E <= kGroupedMaxExperts && off[G->E] < (int64_t(1) << 31) && G->g > 0 &&
         G->K % G->g == 0;
}

int32_t grouped_dw_P(const catq_grouped_layer* G) { return std::gcd(G->g, 128); }

// Partial group sums of every expert: [E][3][N][K/P] fp32.
size_t grouped_partials_bytes(const catq_grouped_layer* G) {
  return static_cast<size_t>(G->E) * 3 * static_cast<size_t>(G->N) * static_cast<size_t>(G->K / grouped_dw_P(G)) *
         sizeof(float);
}

// The bf16 forward or dX of every expert as one grouped tensor-core launch: every expert's
// tiles in one persistent sweep.  *used is false when the layer does not qualify (fp32,
// more experts than one launch takes, 2^31 rows or more), and the caller loops instead.
catq_status grouped_tc(const catq_grouped_layer* G, catq_schedule sched, const void* A, const int64_t* off,
                       int32_t x_dtype, void* C, bool dx, catq_stream stream, bool* used,
                       const EpiOpts* opts = nullptr) {
  *used = false;
  if (G->w_dtype != CATQ_BF16 || x_dtype != CATQ_BF16 || G->E > kGroupedMaxExperts) return CATQ_OK;
  const int64_t R = off[G->E];
  if (R >= (int64_t(1) << 31)) return CATQ_OK;
  const catq_layer L = expert_layer(G, 0);
  catq_status st = check_layer(&L, sched.phase != CATQ_PHASE_TEACHER);
  if (st != CATQ_OK) return st;
  if ((st = check_schedule(sched, sched.phase == CATQ_PHASE_SOFT)) != CATQ_OK) return st;
  if ((st = check_op_const(&L, sched)) != CATQ_OK) return st;
  const int64_t groups = G->N * G->K / G->g;
  const int64_t const_stride = (G->recon ? 5 : 4) * groups;
  if (const_stride % 4 != 0) return CATQ_OK;
  *used = true;
  if (R == 0) return CATQ_OK;
  if (!A || (!C && !opts)) return CATQ_ERR_INVALID_ARG;
  if (!aligned16(A) || (C && !aligned16(C))) return CATQ_ERR_ALIGN;
  if ((st = check_tensor_core_device()) != CATQ_OK) return st;
  const GroupSpec grp{G->E, off, const_stride};
  const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  return cuda_status(dx ? launch_tc_dx_grouped(to_dev(&L), scalars(sched), A, grp, C, s)
                        : launch_tc_fwd_grouped(to_dev(&L), scalars(sched), A, grp, C, s, opts));
}

catq_status catq_grouped_soft_ternary_linear_fwd(const catq_grouped_layer* G, catq_schedule sched, const void* X,
                                                 const int64_t* off, int32_t x_dtype, void* Y, catq_stream stream) {
  catq_status st = check_grouped(G, off);
  if (st != CATQ_OK) return st;
  bool used = false;
  if ((st = grouped_tc(G, sched, X, off, x_dtype, Y, false, stream, &used)) != CATQ_OK || used) return st;
  const size_t esize = x_dtype == CATQ_BF16 ? 2 : 4;
  for (int32_t e = 0; e < G->E; ++e) {
    const catq_layer L = expert_layer(G, e);
    const int64_t m = off[e + 1] - off[e];
    st = catq_soft_ternary_linear_fwd(&L, sched, static_cast<const char*>(X) + off[e] * G->K * esize, m, x_dtype,
                                      static_cast<char*>(Y) + off[e] * G->N * esize, stream);
    if (st != CATQ_OK) return st;
  }
  return CATQ_OK;
}

size_t catq_grouped_fwd_loss_workspace_bytes(const catq_grouped_layer* G, const int64_t* off) {
  if (check_grouped(G, off) != CATQ_OK || G->N < 1) return 0;
  return fwd_loss_ws_bytes(std::max<int64_t>(1, off[G->E] * G->N));
}

catq_status catq_grouped_soft_ternary_linear_fwd_loss(const catq_grouped_layer* G, catq_schedule sched,
                                                      const void* X, const int64_t* off, int32_t x_dtype,
                                                      const void* Y_ref, int32_t reduction, float* loss_out,
                                                      void* dY, void* Y, void* workspace, size_t ws_bytes,
                                                      catq_stream stream) {
  catq_status st = check_grouped(G, off);
  if (st != CATQ_OK) return st;
  if (x_dtype != G->w_dtype) return CATQ_ERR_DTYPE;
  if (reduction != CATQ_REDUCE_MEAN && reduction != CATQ_REDUCE_SUM) return CATQ_ERR_INVALID_ARG;
  const int64_t R = off[G->E];
  if (R < 1 || G->N < 1) return CATQ_ERR_SHAPE;
  if (!X || !Y_ref || !loss_out || !dY) return CATQ_ERR_INVALID_ARG;
  if (!aligned16(X) || !aligned16(Y_ref) || !aligned16(dY) || (Y && !aligned16(Y))) return CATQ_ERR_ALIGN;
  if (!workspace || ws_bytes < catq_grouped_fwd_loss_workspace_bytes(G, off)) return CATQ_ERR_WORKSPACE;
  if (!aligned256(workspace)) return CATQ_ERR_ALIGN;
  const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int64_t count = R * G->N;
  const double inv = reduction == CATQ_REDUCE_MEAN ? 1.0 / static_cast<double>(count) : 1.0;
  double* part = static_cast<double*>(workspace);
  EpiOpts o;
  o.yref = Y_ref;
  o.dscale = static_cast<float>(2.0 * inv);
  o.dY = dY;
  o.loss_part = part;
  int nparts = 0;
  o.n_parts = &nparts;
  bool used = false;
  if ((st = grouped_tc(G, sched, X, off, x_dtype, Y, false, stream, &used, &o)) != CATQ_OK) return st;
  if (used) return cuda_status(launch_loss_final(part, nparts, inv, loss_out, s));
  // expert by expert into Y (or into dY as scratch), then the loss over every routed row
  void* Yw = Y ? Y : dY;
  if ((st = catq_grouped_soft_ternary_linear_fwd(G, sched, X, off, x_dtype, Yw, stream)) != CATQ_OK) return st;
  return cuda_status(launch_recon_loss(Yw, Y_ref, count, x_dtype, reduction, loss_out, dY, part, s));
}

size_t catq_grouped_bwd_workspace_bytes(const catq_grouped_layer* G, const int64_t* off) {
  if (check_grouped(G, off) != CATQ_OK) return 0;
  if (grouped_dw_ok(G, off)) return round256(grouped_partials_bytes(G));
  size_t best = 0;
  for (int32_t e = 0; e < G->E; ++e) {
    const catq_layer L = expert_layer(G, e);
    const size_t b = catq_bwd_workspace_bytes(&L, off[e + 1] - off[e]);
    if (b > best) best = b;
  }
  return best;
}

catq_status catq_grouped_soft_ternary_linear_bwd(const catq_grouped_layer* G, catq_schedule sched, const void* X,
                                                 const void* dY, const int64_t* off, int32_t x_dtype, void* dX,
                                                 float* g_dmu, float* g_dalpha, float* g_ddelta, void* workspace,
                                                 size_t ws_bytes, catq_stream stream) {
  catq_status st = check_grouped(G, off);
  if (st != CATQ_OK) return st;
  const size_t esize = x_dtype == CATQ_BF16 ? 2 : 4;
  const int64_t groups = G->N * G->K / G->g;
  // dX of every expert in one grouped launch where the layer qualifies; the factor
  // gradients (and dX otherwise) expert by expert
  bool dx_done = false;
  if (dX && (st = grouped_tc(G, sched, dY, off, x_dtype, dX, true, stream, &dx_done)) != CATQ_OK) return st;
  const bool want_grads = g_dmu || g_dalpha || g_ddelta;
  bool dw_done = !want_grads;
  if (want_grads && x_dtype == CATQ_BF16 && grouped_dw_ok(G, off)) {
    if (!(g_dmu && g_dalpha && g_ddelta)) return CATQ_ERR_INVALID_ARG;
    const catq_layer L = expert_layer(G, 0);
    if ((st = check_layer(&L, sched.phase != CATQ_PHASE_TEACHER)) != CATQ_OK) return st;
    if ((st = check_schedule(sched, sched.phase != CATQ_PHASE_TEACHER)) != CATQ_OK) return st;
    const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    const int64_t R = off[G->E];
    if (sched.phase == CATQ_PHASE_TEACHER || R == 0) {
      const size_t b = static_cast<size_t>(G->E) * groups * sizeof(float);
      if (cudaMemsetAsync(g_dmu, 0, b, s) != cudaSuccess || cudaMemsetAsync(g_dalpha, 0, b, s) != cudaSuccess ||
          cudaMemsetAsync(g_ddelta, 0, b, s) != cudaSuccess)
        return CATQ_ERR_CUDA;
    } else {
      if (!X || !dY) return CATQ_ERR_INVALID_ARG;
      if (!aligned16(X) || !aligned16(dY)) return CATQ_ERR_ALIGN;
      if (!workspace || ws_bytes < grouped_partials_bytes(G)) return CATQ_ERR_WORKSPACE;
      if (!aligned256(workspace)) return CATQ_ERR_ALIGN;
      if ((st = check_tensor_core_device()) != CATQ_OK) return st;
      const GroupSpec grp{G->E, off, 0};
      const LayerDev L0 = to_dev(&L);
      const StepScalars sc = scalars(sched);
      float* part = static_cast<float*>(workspace);
      const int32_t P = grouped_dw_P(G);
      if (launch_tc_dw_grouped(L0, sc, X, dY, grp, P, part, s) != cudaSuccess) return CATQ_ERR_CUDA;
      if ((st = cuda_status(launch_grad_reduce_grouped(L0, sc, part, P, grp, g_dmu, g_dalpha, g_ddelta, s))) !=
          CATQ_OK)
        return st;
    }
    dw_done = true;
  }
  if (dw_done && (dx_done || !dX)) return CATQ_OK;
  for (int32_t e = 0; e < G->E; ++e) {
    const catq_layer L = expert_layer(G, e);
    const int64_t m = off[e + 1] - off[e];
    st = catq_soft_ternary_linear_bwd(
        &L, sched, static_cast<const char*>(X) + off[e] * G->K * esize,
        static_cast<const char*>(dY) + off[e] * G->N * esize, m, x_dtype,
        dX && !dx_done ? static_cast<char*>(dX) + off[e] * G->K * esize : nullptr,
        g_dmu && !dw_done ? g_dmu + e * groups : nullptr,
        g_dalpha && !dw_done ? g_dalpha + e * groups : nullptr,
        g_ddelta && !dw_done ? g_ddelta + e * groups : nullptr, workspace, ws_bytes, stream);
    if (st != CATQ_OK) return st;
  }
  return CATQ_OK;
}

catq_status catq_ternary_infer(const uint8_t* codes, const float* alpha, const float* mu, int64_t N, int64_t K,
                              int32_t g, const void* X, int64_t B, int32_t x_dtype, void* Y, catq_stream stream) {
  if (!codes || !alpha) return CATQ_ERR_INVALID_ARG;
  if (x_dtype != CATQ_BF16) return CATQ_ERR_DTYPE;
  if (N < 1 || K < 1 || g < 64 || g % 64 != 0 || K % g != 0 || B < 0) return CATQ_ERR_SHAPE;
  if (N * K / g >= (int64_t(1) << 31) || N >= (int64_t(1) << 31) || K >= (int64_t(1) << 31)) return CATQ_ERR_SHAPE;
  if (B == 0) return CATQ_OK;
  if (!X || !Y) return CATQ_ERR_INVALID_ARG;
  if (!aligned16(codes) || !aligned16(X) || (reinterpret_cast<uintptr_t>(alpha) & 3u) != 0 ||
      (reinterpret_cast<uintptr_t>(mu) & 3u) != 0 || (reinterpret_cast<uintptr_t>(Y) & 1u) != 0)
    return CATQ_ERR_ALIGN;
  return cuda_status(
      launch_ternary_infer(codes, alpha, mu, N, K, g, X, B, Y, reinterpret_cast<cudaStream_t>(stream)));
}

int32_t catq_ternary_infer_max_layers(void) { return ternary_infer_max_layers(); }

namespace {
catq_status infer_descs(const catq_infer_layer* layers, int32_t n_layers, int32_t g, int64_t B, int32_t x_dtype,
                        InferDesc* d) {
  if (!layers || n_layers < 1 || n_layers > ternary_infer_max_layers()) return CATQ_ERR_INVALID_ARG;
  if (x_dtype != CATQ_BF16) return CATQ_ERR_DTYPE;
  if (g < 64 || g % 64 != 0 || B < 0) return CATQ_ERR_SHAPE;
  const bool with_mu = layers[0].mu != nullptr;
  for (int32_t i = 0; i < n_layers; ++i) {
    const catq_infer_layer& L = layers[i];
    if (!L.codes || !L.alpha) return CATQ_ERR_INVALID_ARG;
    if ((L.mu != nullptr) != with_mu) return CATQ_ERR_INVALID_ARG;
    if (L.N < 1 || L.K < 1 || L.K % g != 0) return CATQ_ERR_SHAPE;
    if (L.N * L.K / g >= (int64_t(1) << 31) || L.N >= (int64_t(1) << 31) || L.K >= (int64_t(1) << 31))
      return CATQ_ERR_SHAPE;
    if (B > 0 && (!L.X || !L.Y)) return CATQ_ERR_INVALID_ARG;
    if (!aligned16(L.codes) || (B > 0 && !aligned16(L.X)) || (reinterpret_cast<uintptr_t>(L.alpha) & 3u) != 0 ||
        (reinterpret_cast<uintptr_t>(L.mu) & 3u) != 0 || (reinterpret_cast<uintptr_t>(L.Y) & 1u) != 0)
      return CATQ_ERR_ALIGN;
    d[i] = InferDesc{L.codes, L.alpha, L.mu, L.N, L.K, L.X, B, L.Y};
  }
  return CATQ_OK;
}
}  // namespace

catq_status catq_ternary_infer_batched(const catq_infer_layer* layers, int32_t n_layers, int32_t g, int64_t B,
                                       int32_t x_dtype, catq_stream stream) {
  InferDesc d[64];
  const catq_status st = infer_descs(layers, n_layers, g, B, x_dtype, d);
  if (st != CATQ_OK || B == 0) return st;
  return cuda_status(launch_ternary_infer_batched(d, n_layers, g, reinterpret_cast<cudaStream_t>(stream)));
}

int32_t catq_ternary_infer_max_stages(void) { return ternary_infer_max_stages(); }

size_t catq_ternary_infer_sync_bytes(void) { return ternary_infer_sync_bytes(); }

catq_status catq_ternary_infer_staged(const catq_infer_layer* layers, int32_t n_layers, const int32_t* stage_of_layer,
                                      int32_t g, int64_t B, int32_t x_dtype, uint32_t* sync, catq_stream stream) {
  InferDesc d[64];
  catq_status st = infer_descs(layers, n_layers, g, B, x_dtype, d);
  if (st != CATQ_OK) return st;
  if (!stage_of_layer || !sync) return CATQ_ERR_INVALID_ARG;
  if (stage_of_layer[0] != 0) return CATQ_ERR_INVALID_ARG;
  for (int32_t i = 1; i < n_layers; ++i)
    if (stage_of_layer[i] != stage_of_layer[i - 1] && stage_of_layer[i] != stage_of_layer[i - 1] + 1)
      return CATQ_ERR_INVALID_ARG;
  if (stage_of_layer[n_layers - 1] + 1 > ternary_infer_max_stages()) return CATQ_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(sync) & 3u) != 0) return CATQ_ERR_ALIGN;
  if (B == 0) return CATQ_OK;
  return cuda_status(
      launch_ternary_infer_staged(d, n_layers, stage_of_layer, g, sync, reinterpret_cast<cudaStream_t>(stream)));
}

catq_status catq_schedule_at_epoch(int32_t e, int32_t m, double gamma, double s0, catq_schedule* out) {
  if (!out || m < 1 || e < 0 || e > m) return CATQ_ERR_INVALID_ARG;
  if (!(gamma > 0.0 && gamma <= 1.0) || !(s0 > 0.0) || !std::isfinite(s0)) return CATQ_ERR_INVALID_ARG;
  const int64_t soft_epochs = static_cast<int64_t>(std::floor(gamma * m + 1e-9));
  if (e == 0) {
    *out = catq_schedule{CATQ_PHASE_TEACHER, 0.0f};
  } else if (e <= soft_epochs) {
    const double t = static_cast<double>(e) / m;
    *out = catq_schedule{CATQ_PHASE_SOFT, static_cast<float>(t / gamma * s0)};
  } else if (soft_epochs == 0) {
    *out = catq_schedule{CATQ_PHASE_HARD, static_cast<float>(s0)};  // no soft epoch to inherit from
  } else {
    // the last soft epoch's sharpness (§2.3): s0 when gamma m is an integer
    const double t_last = static_cast<double>(soft_epochs) / m;
    *out = catq_schedule{CATQ_PHASE_HARD, static_cast<float>(t_last / gamma * s0)};
  }
  return CATQ_OK;
}

catq_status catq_linear_decay_lr(double lr0, int64_t k, int64_t total, float* lr_out) {
  if (!lr_out || k < 0 || k >= total || !(lr0 >= 0.0) || !std::isfinite(lr0)) return CATQ_ERR_INVALID_ARG;
  *lr_out = static_cast<float>(lr0 * (1.0 - static_cast<double>(k) / static_cast<double>(total)));
  return CATQ_OK;
}

catq_status catq_factor_adamw_step(int64_t G, float* d_mu, float* d_alpha, float* d_delta, const float* g_dmu,
                                   const float* g_dalpha, const float* g_ddelta, float* moments,
                                   const catq_adamw* hp, int64_t t, float lr, catq_stream stream) {
  if (G < 0) return CATQ_ERR_SHAPE;
  if (G == 0) return CATQ_OK;
  if (!d_mu || !d_alpha || !d_delta || !g_dmu || !g_dalpha || !g_ddelta || !moments || !hp)
    return CATQ_ERR_INVALID_ARG;
  if (t < 1 || !(lr >= 0.0f) || !std::isfinite(lr)) return CATQ_ERR_INVALID_ARG;
  if (!(hp->beta1 >= 0.0f && hp->beta1 < 1.0f) || !(hp->beta2 >= 0.0f && hp->beta2 < 1.0f) ||
      !(hp->eps > 0.0f) || !std::isfinite(hp->eps) || !(hp->weight_decay >= 0.0f) ||
      !std::isfinite(hp->weight_decay) || !(hp->margin >= 0.0f && hp->margin < 0.5f))
    return CATQ_ERR_INVALID_ARG;
  const void* ptrs[7] = {d_mu, d_alpha, d_delta, g_dmu, g_dalpha, g_ddelta, moments};
  for (const void* p : ptrs)
    if (reinterpret_cast<uintptr_t>(p) & 3u) return CATQ_ERR_ALIGN;
  AdamwArgs a{};
  float* const p[3] = {d_mu, d_alpha, d_delta};
  const float* const g[3] = {g_dmu, g_dalpha, g_ddelta};
  for (int q = 0; q < 3; ++q) {
    a.p[q] = p[q];
    a.g[q] = g[q];
    a.m[q] = moments + q * G;
    a.v[q] = moments + (3 + q) * G;
  }
  const double b1 = hp->beta1, b2 = hp->beta2;
  a.decay = static_cast<float>(1.0 - static_cast<double>(lr) * hp->weight_decay);
  a.beta1 = hp->beta1;
  a.one_minus_beta1 = static_cast<float>(1.0 - b1);
  a.beta2 = hp->beta2;
  a.one_minus_beta2 = static_cast<float>(1.0 - b2);
  a.step = static_cast<float>(lr / (1.0 - std::pow(b1, static_cast<double>(t))));
  a.inv_sqrt_bc2 = static_cast<float>(1.0 / std::sqrt(1.0 - std::pow(b2, static_cast<double>(t))));
  a.eps = hp->eps;
  a.lo[0] = -1.0f + hp->margin;
  a.hi[0] = 1.0f - hp->margin;
  a.lo[1] = a.lo[2] = hp->margin;
  a.hi[1] = a.hi[2] = INFINITY;
  return cuda_status(launch_factor_adamw(G, a, reinterpret_cast<cudaStream_t>(stream)));
}

catq_status catq_direct_adamw_step(int64_t G, float* d_alpha, float* d_delta, const float* g_dalpha,
                                   const float* g_ddelta, float* moments, const catq_adamw* hp, int64_t t, float lr,
                                   catq_stream stream) {
  if (G < 0) return CATQ_ERR_SHAPE;
  if (G == 0) return CATQ_OK;
  if (!d_alpha || !d_delta || !g_dalpha || !g_ddelta || !moments || !hp) return CATQ_ERR_INVALID_ARG;
  if (t < 1 || !(lr >= 0.0f) || !std::isfinite(lr)) return CATQ_ERR_INVALID_ARG;
  if (!(hp->beta1 >= 0.0f && hp->beta1 < 1.0f) || !(hp->beta2 >= 0.0f && hp->beta2 < 1.0f) ||
      !(hp->eps > 0.0f) || !std::isfinite(hp->eps) || !(hp->weight_decay >= 0.0f) ||
      !std::isfinite(hp->weight_decay) || !(hp->margin >= 0.0f && hp->margin < 0.5f))
    return CATQ_ERR_INVALID_ARG;
  const void* ptrs[5] = {d_alpha, d_delta, g_dalpha, g_ddelta, moments};
  for (const void* p : ptrs)
    if (reinterpret_cast<uintptr_t>(p) & 3u) return CATQ_ERR_ALIGN;
  DirectArgs a{};
  a.d_alpha = d_alpha;
  a.d_delta = d_delta;
  a.g_dalpha = g_dalpha;
  a.g_ddelta = g_ddelta;
  a.m = moments;
  a.v = moments + 2 * G;
  const double b1 = hp->beta1, b2 = hp->beta2;
  a.decay = static_cast<float>(1.0 - static_cast<double>(lr) * hp->weight_decay);
  a.beta1 = hp->beta1;
  a.one_minus_beta1 = static_cast<float>(1.0 - b1);
  a.beta2 = hp->beta2;
  a.one_minus_beta2 = static_cast<float>(1.0 - b2);
  a.step = static_cast<float>(lr / (1.0 - std::pow(b1, static_cast<double>(t))));
  a.inv_sqrt_bc2 = static_cast<float>(1.0 / std::sqrt(1.0 - std::pow(b2, static_cast<double>(t))));
  a.eps = hp->eps;
  a.margin = hp->margin;
  return cuda_status(launch_direct_adamw(G, a, reinterpret_cast<cudaStream_t>(stream)));
}

catq_status catq_group_recon_error(const catq_layer* layer, float* err, catq_stream stream) {
  catq_status st = check_layer(layer, true);
  if (st != CATQ_OK) return st;
  if (!err) return CATQ_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(err) & 3u) return CATQ_ERR_ALIGN;
  return cuda_status(launch_group_recon_error(to_dev(layer), layer->w_dtype, err, reinterpret_cast<cudaStream_t>(stream)));
}

catq_status catq_selftest_wait_timeout(uint64_t timeout_ns, catq_stream stream) {
  if (timeout_ns < 1000 || timeout_ns > 1000000000ull) return CATQ_ERR_INVALID_ARG;
  return cuda_status(launch_wait_probe(timeout_ns, reinterpret_cast<cudaStream_t>(stream)));
}

catq_status catq_device_status(catq_stream stream, int32_t* out) {
  if (!out) return CATQ_ERR_INVALID_ARG;
  if (cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess) return CATQ_ERR_CUDA;
  return cuda_status(read_and_clear_device_status(out));
}

// ------------------------------------------------------------------ decoder-block layers

namespace {
bool aligned4(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 3u) == 0; }
cudaStream_t as_stream(catq_stream s) { return reinterpret_cast<cudaStream_t>(s); }
}  // namespace

catq_status catq_rmsnorm_fwd(const void* X, int32_t x_dtype, const void* residual, const float* gamma, int64_t T,
                             int64_t H, float eps, float* h_out, void* Z, float* r, catq_stream stream) {
  if (x_dtype != CATQ_BF16 && x_dtype != CATQ_F32) return CATQ_ERR_DTYPE;
  if (T < 0 || H < 1 || H % 8 != 0 || T > 0x7fffffff) return CATQ_ERR_SHAPE;
  if (!(eps >= 0.0f) || !std::isfinite(eps)) return CATQ_ERR_INVALID_ARG;
  if (T == 0) return CATQ_OK;
  if (!X || !gamma || !Z || !r) return CATQ_ERR_INVALID_ARG;
  if (!aligned16(X) || !aligned16(Z) || (residual && !aligned16(residual)) || (h_out && !aligned16(h_out)) ||
      !aligned4(gamma) || !aligned4(r))
    return CATQ_ERR_ALIGN;
  return cuda_status(launch_rmsnorm_fwd(X, x_dtype == CATQ_F32, residual, gamma, T, H, eps, h_out, Z, r,
                                        as_stream(stream)));
}

catq_status catq_rmsnorm_bwd(const void* h, int32_t h_dtype, const float* gamma, const float* r, const void* dZ,
                             const void* dZ2, const void* d_residual, int64_t T, int64_t H, void* dX,
                             catq_stream stream) {
  if (h_dtype != CATQ_BF16 && h_dtype != CATQ_F32) return CATQ_ERR_DTYPE;
  if (T < 0 || H < 1 || H % 8 != 0 || T > 0x7fffffff) return CATQ_ERR_SHAPE;
  if (T == 0) return CATQ_OK;
  if (!h || !gamma || !r || !dZ || !dX) return CATQ_ERR_INVALID_ARG;
  if (!aligned16(h) || !aligned16(dZ) || !aligned16(dX) || (dZ2 && !aligned16(dZ2)) ||
      (d_residual && !aligned16(d_residual)) || !aligned4(gamma) || !aligned4(r))
    return CATQ_ERR_ALIGN;
  return cuda_status(launch_rmsnorm_bwd(h, h_dtype == CATQ_F32, gamma, r, dZ, dZ2, d_residual, T, H, dX,
                                        as_stream(stream)));
}

catq_status catq_rope(void* X, int64_t T, int64_t S, int32_t n_heads, int32_t d, float base, int32_t inverse,
                      catq_stream stream) {
  if (T < 0 || S < 1 || n_heads < 1 || d < 8 || d % 2 != 0) return CATQ_ERR_SHAPE;
  if (!(base > 1.0f) || !std::isfinite(base)) return CATQ_ERR_INVALID_ARG;
  if (T == 0) return CATQ_OK;
  if (!X) return CATQ_ERR_INVALID_ARG;
  if (!aligned16(X)) return CATQ_ERR_ALIGN;
  return cuda_status(launch_rope(X, T, S, n_heads, d, base, inverse, as_stream(stream)));
}

catq_status catq_swiglu_fwd(const void* gate, const void* up, int64_t n, void* M, catq_stream stream) {
  if (n < 0) return CATQ_ERR_SHAPE;
  if (n == 0) return CATQ_OK;
  if (!gate || !up || !M) return CATQ_ERR_INVALID_ARG;
  if (!aligned16(gate) || !aligned16(up) || !aligned16(M)) return CATQ_ERR_ALIGN;
  return cuda_status(launch_swiglu(gate, up, nullptr, n, M, nullptr, nullptr, as_stream(stream)));
}

catq_status catq_swiglu_bwd(const void* gate, const void* up, const void* dM, int64_t n, void* d_gate, void* d_up,
                            catq_stream stream) {
  if (n < 0) return CATQ_ERR_SHAPE;
  if (n == 0) return CATQ_OK;
  if (!gate || !up || !dM || !d_gate || !d_up) return CATQ_ERR_INVALID_ARG;
  if (!aligned16(gate) || !aligned16(up) || !aligned16(dM) || !aligned16(d_gate) || !aligned16(d_up))
    return CATQ_ERR_ALIGN;
  return cuda_status(launch_swiglu(gate, up, dM, n, nullptr, d_gate, d_up, as_stream(stream)));
}

catq_status catq_block_output_loss(const float* h, const void* branch, int64_t count, const float* out_ref,
                                   int32_t reduction, float* loss_out, void* d_out, float* out, void* workspace,
                                   size_t ws_bytes, catq_stream stream) {
  if (count < 0 || count % 8 != 0) return CATQ_ERR_SHAPE;
  if (reduction != CATQ_REDUCE_MEAN && reduction != CATQ_REDUCE_SUM) return CATQ_ERR_INVALID_ARG;
  if (count == 0) return CATQ_OK;
  if (!h || !branch || (out_ref && !loss_out)) return CATQ_ERR_INVALID_ARG;
  if (!aligned16(h) || !aligned16(branch) || (out_ref && !aligned16(out_ref)) || (out && !aligned16(out)) ||
      (d_out && !aligned16(d_out)) || (loss_out && !aligned4(loss_out)))
    return CATQ_ERR_ALIGN;
  if (out_ref) {
    if (!workspace || ws_bytes < catq_recon_loss_workspace_bytes(count)) return CATQ_ERR_WORKSPACE;
    if (!aligned256(workspace)) return CATQ_ERR_ALIGN;
  }
  return cuda_status(launch_block_output_loss(h, branch, out_ref, count, reduction, out, d_out, loss_out,
                                              static_cast<double*>(workspace), as_stream(stream)));
}

namespace {
catq_status check_attention(int32_t B, int32_t S, int32_t nh, int32_t nkv, int32_t d) {
  if (B < 0 || B > 65535 || S < 64 || S % 64 != 0 || nh < 1 || nh > 65535 || nkv < 1 || nh % nkv != 0 ||
      (d != 64 && d != 128))
    return CATQ_ERR_SHAPE;
  return CATQ_OK;
}
}  // namespace

catq_status catq_attention_fwd(const void* Q, const void* K, const void* V, int32_t B, int32_t S, int32_t n_heads,
                               int32_t n_kv_heads, int32_t d, void* O, float* lse, catq_stream stream) {
  catq_status st = check_attention(B, S, n_heads, n_kv_heads, d);
  if (st != CATQ_OK) return st;
  if (B == 0) return CATQ_OK;
  if (!Q || !K || !V || !O || !lse) return CATQ_ERR_INVALID_ARG;
  if (!aligned16(Q) || !aligned16(K) || !aligned16(V) || !aligned16(O) || !aligned4(lse)) return CATQ_ERR_ALIGN;
  AttnIo io{};
  io.q = Q;
  io.k = K;
  io.v = V;
  io.out = O;
  io.lse = lse;
  return cuda_status(launch_attention(io, B, S, n_heads, n_kv_heads, d, false, as_stream(stream)));
}

catq_status catq_attention_bwd(const void* Q, const void* K, const void* V, const void* O, const void* dO,
                               const float* lse, int32_t B, int32_t S, int32_t n_heads, int32_t n_kv_heads,
                               int32_t d, float* delta, void* dQ, void* dK, void* dV, catq_stream stream) {
  catq_status st = check_attention(B, S, n_heads, n_kv_heads, d);
  if (st != CATQ_OK) return st;
  if (B == 0) return CATQ_OK;
  if (!Q || !K || !V || !O || !dO || !lse || !delta || !dQ || !dK || !dV) return CATQ_ERR_INVALID_ARG;
  if (!aligned16(Q) || !aligned16(K) || !aligned16(V) || !aligned16(O) || !aligned16(dO) || !aligned16(dQ) ||
      !aligned16(dK) || !aligned16(dV) || !aligned4(lse) || !aligned4(delta))
    return CATQ_ERR_ALIGN;
  AttnIo io{};
  io.q = Q;
  io.k = K;
  io.v = V;
  io.o = O;
  io.dO = dO;
  io.dq = dQ;
  io.dk = dK;
  io.dv = dV;
  io.lse = const_cast<float*>(lse);
  io.delta = delta;
  return cuda_status(launch_attention(io, B, S, n_heads, n_kv_heads, d, true, as_stream(stream)));
}

}  // extern "C"
