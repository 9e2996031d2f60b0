// elementwise.cu — the HBM-bound kernels of the path: group statistics (Eq. 3), the
// materialised Eq. 6 weight (inspection only), the reconstruction loss of Eq. 7 with its
// gradient, the final hard ternarization + 2-bit pack, and the reduction of the dW
// epilogue's partial sums into the three factor gradients, and the optimizer's update of
// the factors after a step.
#include <cuda_bf16.h>

#include "launch.h"

namespace catq {
namespace {

constexpr int kThreads = 256;

__device__ __forceinline__ double warp_sum(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}


template <typename T>
struct Vec16;  // 16-byte vector of T, unpacked to floats
template <>
struct Vec16<float> {
  static constexpr int n = 4;
  __device__ static void load(const float* p, float (&v)[4]) {
    const float4 q = __ldg(reinterpret_cast<const float4*>(p));
    v[0] = q.x; v[1] = q.y; v[2] = q.z; v[3] = q.w;
  }
};
template <>
struct Vec16<__nv_bfloat16> {
  static constexpr int n = 8;
  __device__ static void load(const __nv_bfloat16* p, float (&v)[8]) {
    const uint4 q = __ldg(reinterpret_cast<const uint4*>(p));
    const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      v[2 * i] = bf16lo_to_f32(w[i]);
      v[2 * i + 1] = bf16hi_to_f32(w[i]);
    }
  }
};

// Rounded once to fp32 (all a stored fp32 statistic needs; avoids fp64 arithmetic).
__device__ __forceinline__ float sum2_float(Sum2 v) { return v.hi + v.lo; }

// mu0, alpha0, Delta0 of one group from its compensated sums (Eq. 3; TWN rule of §2.2).
__device__ __forceinline__ void store_group_stats(int64_t j, int32_t g, int32_t thr_init, float mu, Sum2 dev,
                                                  Sum2 mag, float* mu0, float* alpha0, float* delta0) {
  const float inv_g = 1.0f / static_cast<float>(g);
  const float a0 = sum2_float(dev) * inv_g;
  mu0[j] = mu;
  alpha0[j] = a0;
  delta0[j] = (thr_init == 1 && a0 > 0.0f) ? 0.7f * (sum2_float(mag) * inv_g) / a0 : 0.5f;
}

// ---------------------------------------------------------------- Eq. 3 statistics
// Register variant: a team of `team` lanes owns one group and each lane keeps kStatsVPL
// 16-byte vectors of it in registers, so the mean and the deviations need one read of W.
// Lane `sub` of a team takes vectors sub, sub + team, ..., so each load instruction of a
// team reads team x 16 contiguous bytes.  A vector is summed pairwise in fp32 and added to a
// compensated (two-sum) accumulator, the team merges the compensated sums, and the
// all-positive deviation and magnitude sums are plain pairwise fp32 sums (relative error a
// few ulp).  The magnitude sum is only formed for the TWN threshold rule.
constexpr int kStatsVPL = 4;

template <int V>
__device__ __forceinline__ float pairwise_sum(const float (&x)[V]) {
  float t[V];
#pragma unroll
  for (int q = 0; q < V; ++q) t[q] = x[q];
#pragma unroll
  for (int w = 1; w < V; w <<= 1)
#pragma unroll
    for (int q = 0; q + w < V; q += 2 * w) t[q] += t[q + w];
  return t[0];
}

template <int V>
__device__ __forceinline__ float pairwise_abs_sum(const float (&x)[V], float shift) {
  float t[V];
#pragma unroll
  for (int q = 0; q < V; ++q) t[q] = fabsf(x[q] - shift);
#pragma unroll
  for (int w = 1; w < V; w <<= 1)
#pragma unroll
    for (int q = 0; q + w < V; q += 2 * w) t[q] += t[q + w];
  return t[0];
}

__device__ __forceinline__ float team_sum(float v, int team) {
  for (int o = team >> 1; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

template <typename T, bool TWN>
__global__ void __launch_bounds__(kThreads) group_stats_team_kernel(const T* __restrict__ W, int64_t G, int32_t g,
                                                                    int32_t team, float* __restrict__ mu0,
                                                                    float* __restrict__ alpha0,
                                                                    float* __restrict__ delta0) {
  constexpr int V = Vec16<T>::n;
  constexpr int VPL = kStatsVPL;
  const int lane = threadIdx.x & 31;
  const int sub = lane & (team - 1);
  const int per_warp = 32 / team;
  const int64_t warp = (static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x) >> 5;
  const int64_t nwarps = static_cast<int64_t>(gridDim.x) * (kThreads / 32);
  const float inv_g = 1.0f / static_cast<float>(g);
  for (int64_t wbase = warp * per_warp; wbase < G; wbase += nwarps * per_warp) {
    const int64_t j = wbase + lane / team;
    const bool live = j < G;
    float v[VPL][V];
#pragma unroll
    for (int r = 0; r < VPL; ++r) {
      if (live) {
        Vec16<T>::load(W + j * g + static_cast<int64_t>(r * team + sub) * V, v[r]);
      } else {
#pragma unroll
        for (int q = 0; q < V; ++q) v[r][q] = 0.f;
      }
    }
    Sum2 sum{0.f, 0.f};
#pragma unroll
    for (int r = 0; r < VPL; ++r) sum2_add(sum, pairwise_sum<V>(v[r]));
    sum = sum2_team(sum, team);
    const float mu = sum2_float(sum) * inv_g;
    float dev = 0.f, mag = 0.f;
#pragma unroll
    for (int r = 0; r < VPL; ++r) {
      dev += pairwise_abs_sum<V>(v[r], mu);
      if constexpr (TWN) mag += pairwise_abs_sum<V>(v[r], 0.0f);
    }
    dev = team_sum(dev, team);
    if constexpr (TWN) mag = team_sum(mag, team);
    if (live && sub == 0) {
      const float a0 = dev * inv_g;
      mu0[j] = mu;
      alpha0[j] = a0;
      delta0[j] = (TWN && a0 > 0.0f) ? 0.7f * (mag * inv_g) / a0 : 0.5f;
    }
  }
}

// §2.2's static rules as base statistics for the modulation (mu0 = 0, What = W / alpha):
//   absmean: alpha0 = mean|W|, Delta0 = 0.5 (Delta = alpha / 2);
//   TWN:     Delta_W = 0.7 mean|W|, alpha0 = mean of |W_i| over |W_i| > Delta_W,
//            Delta0 = Delta_W / alpha0 (0.5 when no element is above the threshold).
constexpr int32_t kThrAbsmean = 2, kThrTwnStatic = 3;

__device__ __forceinline__ void store_static_stats(int64_t j, int32_t rule, float mean_abs, float above_sum,
                                                   float above_cnt, float* mu0, float* alpha0, float* delta0) {
  mu0[j] = 0.0f;
  if (rule == kThrAbsmean) {
    alpha0[j] = mean_abs;
    delta0[j] = 0.5f;
    return;
  }
  const float a0 = above_cnt > 0.0f ? above_sum / above_cnt : 0.0f;
  alpha0[j] = a0;
  delta0[j] = a0 > 0.0f ? 0.7f * mean_abs / a0 : 0.5f;
}

// Register variant of the static rules (layout of group_stats_team_kernel): mean|W| from the
// registers, then (TWN) a second pass over the same registers for the elements above
// 0.7 mean|W|.
template <typename T, int RULE>
__global__ void __launch_bounds__(kThreads) group_stats_static_kernel(const T* __restrict__ W, int64_t G, int32_t g,
                                                                      int32_t team, float* __restrict__ mu0,
                                                                      float* __restrict__ alpha0,
                                                                      float* __restrict__ delta0) {
  constexpr int V = Vec16<T>::n;
  constexpr int VPL = kStatsVPL;
  const int lane = threadIdx.x & 31;
  const int sub = lane & (team - 1);
  const int per_warp = 32 / team;
  const int64_t warp = (static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x) >> 5;
  const int64_t nwarps = static_cast<int64_t>(gridDim.x) * (kThreads / 32);
  const float inv_g = 1.0f / static_cast<float>(g);
  for (int64_t wbase = warp * per_warp; wbase < G; wbase += nwarps * per_warp) {
    const int64_t j = wbase + lane / team;
    const bool live = j < G;
    float v[VPL][V];
#pragma unroll
    for (int r = 0; r < VPL; ++r) {
      if (live) {
        Vec16<T>::load(W + j * g + static_cast<int64_t>(r * team + sub) * V, v[r]);
      } else {
#pragma unroll
        for (int q = 0; q < V; ++q) v[r][q] = 0.f;
      }
    }
    float mag = 0.f;
#pragma unroll
    for (int r = 0; r < VPL; ++r) mag += pairwise_abs_sum<V>(v[r], 0.0f);
    const float mean_abs = team_sum(mag, team) * inv_g;
    float s = 0.f, cnt = 0.f;
    if constexpr (RULE == kThrTwnStatic) {
      const float dW = 0.7f * mean_abs;
#pragma unroll
      for (int r = 0; r < VPL; ++r)
#pragma unroll
        for (int q = 0; q < V; ++q) {
          const float a = fabsf(v[r][q]);
          if (a > dW) {
            s += a;
            cnt += 1.0f;
          }
        }
      s = team_sum(s, team);
      cnt = team_sum(cnt, team);
    }
    if (live && sub == 0) store_static_stats(j, RULE, mean_abs, s, cnt, mu0, alpha0, delta0);
  }
}

// Streaming variant for any g (one warp per group, second pass re-reads the group).
template <typename T>
__global__ void __launch_bounds__(kThreads) group_stats_stream_kernel(const T* __restrict__ W, int64_t G, int32_t g,
                                                                      int32_t thr_init, float* __restrict__ mu0,
                                                                      float* __restrict__ alpha0,
                                                                      float* __restrict__ delta0) {
  constexpr int V = Vec16<T>::n;
  const int lane = threadIdx.x & 31;
  const int64_t warp = (static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x) >> 5;
  const int64_t nwarps = static_cast<int64_t>(gridDim.x) * (kThreads / 32);
  for (int64_t j = warp; j < G; j += nwarps) {
    const T* base = W + j * g;
    Sum2 sum{0.f, 0.f};
    for (int i = lane * V; i < g; i += 32 * V) {
      float v[V];
      Vec16<T>::load(base + i, v);
#pragma unroll
      for (int q = 0; q < V; ++q) sum2_add(sum, v[q]);
    }
    sum = sum2_team(sum, 32);
    const float mu = sum2_float(sum) / static_cast<float>(g);
    Sum2 dev{0.f, 0.f}, mag{0.f, 0.f};
    for (int i = lane * V; i < g; i += 32 * V) {
      float v[V];
      Vec16<T>::load(base + i, v);
#pragma unroll
      for (int q = 0; q < V; ++q) {
        sum2_add(dev, fabsf(v[q] - mu));
        sum2_add(mag, fabsf(v[q]));
      }
    }
    dev = sum2_team(dev, 32);
    mag = sum2_team(mag, 32);
    if (thr_init == kThrAbsmean || thr_init == kThrTwnStatic) {
      const float mean_abs = sum2_float(mag) / static_cast<float>(g);
      float s = 0.f, cnt = 0.f;
      if (thr_init == kThrTwnStatic) {
        const float dW = 0.7f * mean_abs;
        for (int i = lane * V; i < g; i += 32 * V) {
          float v[V];
          Vec16<T>::load(base + i, v);
#pragma unroll
          for (int q = 0; q < V; ++q) {
            const float a = fabsf(v[q]);
            if (a > dW) {
              s += a;
              cnt += 1.0f;
            }
          }
        }
        s = team_sum(s, 32);
        cnt = team_sum(cnt, 32);
      }
      if (lane == 0) store_static_stats(j, thr_init, mean_abs, s, cnt, mu0, alpha0, delta0);
      continue;
    }
    if (lane == 0) store_group_stats(j, g, thr_init, mu, dev, mag, mu0, alpha0, delta0);
  }
}

// ---------------------------------------------------------------- materialised Eq. 6 weight
// One thread per 8 consecutive elements (g % 8 == 0 on the bf16 path keeps them in one
// group and one row); the bf16 arithmetic is the fused producer's.
__global__ void __launch_bounds__(kThreads) modulate_bf16_kernel(LayerDev L, StepScalars sc, uint16_t* __restrict__ Wq,
                                                                 int8_t* __restrict__ Tout, float* __restrict__ alpha) {
  const int64_t nchunks = L.N * L.K / 8;
  const int64_t G = L.N * L.K / L.g;
  const uint16_t* W = static_cast<const uint16_t*>(L.W);
  for (int64_t c = blockIdx.x * (int64_t)kThreads + threadIdx.x; c < nchunks; c += (int64_t)gridDim.x * kThreads) {
    const int64_t e = c * 8;
    const int64_t j = e / L.g;
    const GroupConst gc = group_const(L, j);
    const uint4 v = __ldg(reinterpret_cast<const uint4*>(W + e));
    if (Wq) {
      const ProducerConst pc = producer_const(gc, sc.s, sc.inv_2tanh_s, sc.phase);
      *reinterpret_cast<uint4*>(Wq + e) = transform_chunk_bf16(v, pc, sc.phase, L.recon);
    }
    if (Tout) {
      const uint32_t w[4] = {v.x, v.y, v.z, v.w};
      uint32_t packed[2] = {0u, 0u};
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const float x = (i & 1) ? bf16hi_to_f32(w[i >> 1]) : bf16lo_to_f32(w[i >> 1]);
        const int t = (gc.alpha != 0.0f) ? static_cast<int>(hard_q(what(x, gc), gc.delta)) : 0;
        packed[i >> 2] |= (static_cast<uint32_t>(static_cast<uint8_t>(static_cast<int8_t>(t)))) << (8 * (i & 3));
      }
      *reinterpret_cast<uint2*>(Tout + e) = make_uint2(packed[0], packed[1]);
    }
  }
  if (alpha)
    for (int64_t j = blockIdx.x * (int64_t)kThreads + threadIdx.x; j < G; j += (int64_t)gridDim.x * kThreads)
      alpha[j] = __ldg(L.d_alpha + j) * __ldg(L.alpha0 + j);
}

__global__ void __launch_bounds__(kThreads) modulate_f32_kernel(LayerDev L, StepScalars sc, float* __restrict__ Wq,
                                                                int8_t* __restrict__ Tout, float* __restrict__ alpha) {
  const int64_t n = L.N * L.K;
  const int64_t G = n / L.g;
  const float* W = static_cast<const float*>(L.W);
  for (int64_t e = blockIdx.x * (int64_t)kThreads + threadIdx.x; e < n; e += (int64_t)gridDim.x * kThreads) {
    const GroupConst gc = group_const(L, e / L.g);
    const float w = W[e];
    if (Wq) Wq[e] = ternary_weight_f32(w, gc, sc.s, sc.inv_2tanh_s, sc.phase, L.recon);
    if (Tout) Tout[e] = (gc.alpha != 0.0f) ? static_cast<int8_t>(hard_q(what(w, gc), gc.delta)) : int8_t(0);
  }
  if (alpha)
    for (int64_t j = blockIdx.x * (int64_t)kThreads + threadIdx.x; j < G; j += (int64_t)gridDim.x * kThreads)
      alpha[j] = __ldg(L.d_alpha + j) * __ldg(L.alpha0 + j);
}

// ---------------------------------------------------------------- hard ternarize + pack
// EPT consecutive elements per thread (EPT divides g, so one group), EPT/4 output bytes.
template <typename T, int EPT>
__global__ void __launch_bounds__(kThreads) hard_pack_kernel(LayerDev L, uint8_t* __restrict__ codes,
                                                             float* __restrict__ alpha, float* __restrict__ mu) {
  const int64_t n = L.N * L.K;
  const int64_t G = n / L.g;
  const T* W = static_cast<const T*>(L.W);
  for (int64_t t = blockIdx.x * (int64_t)kThreads + threadIdx.x; t * EPT < n; t += (int64_t)gridDim.x * kThreads) {
    const int64_t e0 = t * EPT;
    const GroupConst gc = group_const(L, e0 / L.g);
    float v[EPT];
    constexpr int V = Vec16<T>::n;
    if constexpr (EPT % V == 0) {
#pragma unroll
      for (int i = 0; i < EPT; i += V) {
        float q[V];
        Vec16<T>::load(W + e0 + i, q);
#pragma unroll
        for (int k = 0; k < V; ++k) v[i + k] = q[k];
      }
    } else {
#pragma unroll
      for (int i = 0; i < EPT; ++i) {
        if constexpr (sizeof(T) == 4)
          v[i] = W[e0 + i];
        else
          v[i] = bf16lo_to_f32(static_cast<uint32_t>(reinterpret_cast<const uint16_t*>(W)[e0 + i]));
      }
    }
    uint32_t words[(EPT + 15) / 16] = {};
#pragma unroll
    for (int i = 0; i < EPT; ++i) {
      const int q = (gc.alpha != 0.0f) ? static_cast<int>(hard_q(what(v[i], gc), gc.delta)) : 0;
      words[i / 16] |= static_cast<uint32_t>(q + 1) << (2 * (i & 15));
    }
    if constexpr (EPT == 64)
      *reinterpret_cast<uint4*>(codes + e0 / 4) = make_uint4(words[0], words[1], words[2], words[3]);
    else if constexpr (EPT == 16)
      reinterpret_cast<uint32_t*>(codes)[e0 / 16] = words[0];
    else
      codes[e0 / 4] = static_cast<uint8_t>(words[0]);
  }
  if (alpha || mu)
    for (int64_t j = blockIdx.x * (int64_t)kThreads + threadIdx.x; j < G; j += (int64_t)gridDim.x * kThreads) {
      const GroupConst gc = group_const(L, j);
      if (alpha) alpha[j] = gc.alpha;
      if (mu) mu[j] = gc.mu;
    }
}

// Warp-cooperative pack for power-of-two g >= 8 V: a warp takes batches of 32 x 8 16-byte
// chunks; load c of lane l reads chunk 32 c + l, so each load instruction covers 512
// contiguous bytes.  The at most 32 groups a batch touches get their constants from one
// lane each (alpha = 0 groups get a threshold no value exceeds, so their codes are 0) and
// reach the lanes that need them by shuffles.  A chunk's V elements lie in one group and give
// 2 V code bits.
template <typename T>
__global__ void __launch_bounds__(kThreads) hard_pack_warp_kernel(LayerDev L, int32_t log2g,
                                                                  uint8_t* __restrict__ codes,
                                                                  float* __restrict__ alpha,
                                                                  float* __restrict__ mu) {
  constexpr int V = Vec16<T>::n;
  constexpr int kLoads = 8;
  constexpr int64_t kBatch = 32 * kLoads * V;  // elements per warp batch
  const int64_t n = L.N * L.K;
  const int64_t G = n >> log2g;
  const T* W = static_cast<const T*>(L.W);
  const int lane = threadIdx.x & 31;
  const int64_t warp = (static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x) >> 5;
  const int64_t nwarps = static_cast<int64_t>(gridDim.x) * (kThreads / 32);
  for (int64_t b0 = warp * kBatch; b0 < n; b0 += nwarps * kBatch) {
    const int64_t j0 = b0 >> log2g;
    const int64_t jl = j0 + lane;
    float r = 0.0f, b = 0.0f, delta = __int_as_float(0x7f800000);  // +inf
    if (jl < G && (jl << log2g) < b0 + kBatch) {
      const GroupConst gc = group_const(L, jl);
      if (gc.alpha != 0.0f) {
        r = gc.r;
        b = gc.b;
        delta = gc.delta;
      }
      if ((jl << log2g) >= b0) {  // the batch holding the group's start
        if (alpha) alpha[jl] = gc.alpha;
        if (mu) mu[jl] = gc.mu;
      }
    }
    const int first = static_cast<int>(b0 - (j0 << log2g));  // offset of b0 inside group j0
#pragma unroll
    for (int c = 0; c < kLoads; ++c) {
      const int off = (c * 32 + lane) * V;  // element offset inside the batch
      const int src = (first + off) >> log2g;
      const float rr = __shfl_sync(0xffffffffu, r, src);
      const float bb = __shfl_sync(0xffffffffu, b, src);
      const float dd = __shfl_sync(0xffffffffu, delta, src);
      const int64_t e = b0 + off;
      if (e < n) {
        float v[V];
        Vec16<T>::load(W + e, v);
        uint32_t bits = 0;
#pragma unroll
        for (int k = 0; k < V; ++k) {
          const float x = fmaf(v[k], rr, bb);
          const int q = x > dd ? 1 : (x < -dd ? -1 : 0);
          bits |= static_cast<uint32_t>(q + 1) << (2 * k);
        }
        if constexpr (V == 8)
          reinterpret_cast<uint16_t*>(codes)[e / 8] = static_cast<uint16_t>(bits);
        else
          codes[e / 4] = static_cast<uint8_t>(bits);
      }
    }
  }
}

// ---------------------------------------------------------------- fused-GEMM operand constants
// operand_const_vec of every group for one schedule point, stored [K/g][N] so that a fused
// GEMM producer warp (consecutive W rows, one group column) reads contiguous 16-byte
// vectors; with mu in the reconstruction the group offsets go to op_mu in the same order.
// A 32 x 32 (row x group column) tile goes through shared memory so both the row-major
// [N][K/g] group arrays and the output are accessed coalesced.
constexpr int kConstTile = 32;

// blockIdx.z: expert of a stacked (grouped) layer, whose per-group arrays start z G after
// expert 0's and whose constants start z const_stride floats after (0 for a dense layer).
__global__ void __launch_bounds__(kConstTile * kConstTile) operand_consts_kernel(LayerDev L, StepScalars sc,
                                                                                 int64_t const_stride) {
  if (blockIdx.z > 0) {
    const int64_t G = L.N * L.groups_per_row, e = blockIdx.z;
    L.mu0 += e * G;
    L.alpha0 += e * G;
    L.delta0 += e * G;
    L.d_mu += e * G;
    L.d_alpha += e * G;
    L.d_delta += e * G;
    L.op_const = reinterpret_cast<float4*>(reinterpret_cast<float*>(L.op_const) + e * const_stride);
    if (L.op_mu) L.op_mu += e * const_stride;
  }
  __shared__ float4 tile[kConstTile][kConstTile + 1];
  __shared__ float tile_mu[kConstTile][kConstTile + 1];
  const int64_t gpr = L.groups_per_row;
  const int64_t c0 = static_cast<int64_t>(blockIdx.x) * kConstTile;
  for (int64_t n0 = static_cast<int64_t>(blockIdx.y) * kConstTile; n0 < L.N;
       n0 += static_cast<int64_t>(gridDim.y) * kConstTile) {
    {
      const int64_t n = n0 + threadIdx.y, c = c0 + threadIdx.x;
      if (n < L.N && c < gpr) {
        const GroupConst gc = group_const(L, n * gpr + c);
        tile[threadIdx.y][threadIdx.x] = operand_const_vec(gc, sc.s, sc.inv_2tanh_s, sc.phase);
        tile_mu[threadIdx.y][threadIdx.x] = gc.mu;
      }
    }
    __syncthreads();
    const int64_t n = n0 + threadIdx.x, c = c0 + threadIdx.y;
    if (n < L.N && c < gpr) {
      L.op_const[c * L.N + n] = tile[threadIdx.x][threadIdx.y];
      if (L.recon) L.op_mu[c * L.N + n] = tile_mu[threadIdx.x][threadIdx.y];
    }
    __syncthreads();
  }
}

// ---------------------------------------------------------------- Eq. 7 loss and dY
constexpr int kLossMaxBlocks = 1216;

template <typename T>
__device__ __forceinline__ void store_scaled(T* p, const float (&d)[Vec16<T>::n], float scale);
template <>
__device__ __forceinline__ void store_scaled<float>(float* p, const float (&d)[4], float scale) {
  *reinterpret_cast<float4*>(p) = make_float4(d[0] * scale, d[1] * scale, d[2] * scale, d[3] * scale);
}
template <>
__device__ __forceinline__ void store_scaled<__nv_bfloat16>(__nv_bfloat16* p, const float (&d)[8], float scale) {
  uint4 q;
  q.x = pack_bf16x2(d[0] * scale, d[1] * scale);
  q.y = pack_bf16x2(d[2] * scale, d[3] * scale);
  q.z = pack_bf16x2(d[4] * scale, d[5] * scale);
  q.w = pack_bf16x2(d[6] * scale, d[7] * scale);
  *reinterpret_cast<uint4*>(p) = q;
}

__device__ __forceinline__ float load_scalar(const float* p) { return *p; }
__device__ __forceinline__ float load_scalar(const __nv_bfloat16* p) { return __bfloat162float(*p); }
__device__ __forceinline__ void store_scalar(float* p, float v) { *p = v; }
__device__ __forceinline__ void store_scalar(__nv_bfloat16* p, float v) { *p = __float2bfloat16_rn(v); }

template <typename T>
__global__ void __launch_bounds__(kThreads) recon_loss_partial_kernel(const T* __restrict__ Y, const T* __restrict__ Yr,
                                                                      int64_t count, float scale, T* __restrict__ dY,
                                                                      double* __restrict__ partials) {
  constexpr int V = Vec16<T>::n;
  const int64_t nvec = count / V;
  Sum2 acc{0.f, 0.f};
  for (int64_t i = blockIdx.x * (int64_t)kThreads + threadIdx.x; i < nvec; i += (int64_t)gridDim.x * kThreads) {
    float a[V], b[V], d[V];
    Vec16<T>::load(Y + i * V, a);
    Vec16<T>::load(Yr + i * V, b);
    Sum2 local{0.f, 0.f};
#pragma unroll
    for (int q = 0; q < V; ++q) {
      d[q] = a[q] - b[q];
      sum2_add(local, d[q] * d[q]);
    }
    acc = sum2_merge(acc, local);
    if (dY) store_scaled<T>(dY + i * V, d, scale);
  }
  if (blockIdx.x == 0)
    for (int64_t i = nvec * V + threadIdx.x; i < count; i += kThreads) {
      const float d = load_scalar(Y + i) - load_scalar(Yr + i);
      sum2_add(acc, d * d);
      if (dY) store_scalar(dY + i, d * scale);
    }
  __shared__ Sum2 red[kThreads / 32];
  acc = sum2_team(acc, 32);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x < 32) {
    Sum2 v = threadIdx.x < kThreads / 32 ? red[threadIdx.x] : Sum2{0.f, 0.f};
    v = sum2_team(v, 32);
    if (threadIdx.x == 0) partials[blockIdx.x] = sum2_value(v);
  }
}

__global__ void __launch_bounds__(kThreads) recon_loss_final_kernel(const double* __restrict__ partials, int nblocks,
                                                                    double out_scale, float* __restrict__ loss) {
  double acc = 0.0;
  for (int i = threadIdx.x; i < nblocks; i += kThreads) acc += partials[i];
  __shared__ double red[kThreads / 32];
  acc = warp_sum(acc);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x < 32) {
    double v = threadIdx.x < kThreads / 32 ? red[threadIdx.x] : 0.0;
    v = warp_sum(v);
    if (threadIdx.x == 0) loss[0] = static_cast<float>(v * out_scale);
  }
}

// ---------------------------------------------------------------- 8-bit activations
// Per-token symmetric absmax quantization of one row per warp (the W1.58A8 setting): the
// warp's max |x| gives scale = max / 127 (IEEE division); each element's code is
// rint(x / scale) (IEEE division, ties to even), clamped to [-127, 127]; a zero row has
// scale 0 and codes 0.  Codes are written as exact values of the input dtype (|q| <= 127
// is exact in bf16), and `deq` (nullable) gets scale * q rounded once to that dtype.
template <typename T>
__device__ __forceinline__ void store_vec(T* p, const float (&v)[Vec16<T>::n]);
template <>
__device__ __forceinline__ void store_vec<float>(float* p, const float (&v)[4]) {
  *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
}
template <>
__device__ __forceinline__ void store_vec<__nv_bfloat16>(__nv_bfloat16* p, const float (&v)[8]) {
  uint4 q;
  q.x = pack_bf16x2(v[0], v[1]);
  q.y = pack_bf16x2(v[2], v[3]);
  q.z = pack_bf16x2(v[4], v[5]);
  q.w = pack_bf16x2(v[6], v[7]);
  *reinterpret_cast<uint4*>(p) = q;
}

template <typename T>
__global__ void __launch_bounds__(kThreads) act_quant_a8_kernel(const T* __restrict__ X, int64_t M, int64_t K,
                                                                 T* __restrict__ codes, float* __restrict__ scale,
                                                                 T* __restrict__ deq) {
  constexpr int V = Vec16<T>::n;
  const int lane = threadIdx.x & 31;
  const int64_t nvec = K / V;  // K is a multiple of V (16-byte rows)
  for (int64_t m = (blockIdx.x * (int64_t)kThreads + threadIdx.x) >> 5; m < M;
       m += ((int64_t)gridDim.x * kThreads) >> 5) {
    const T* row = X + m * K;
    float amax = 0.0f;
    for (int64_t v = lane; v < nvec; v += 32) {
      float x[V];
      Vec16<T>::load(row + v * V, x);
#pragma unroll
      for (int q = 0; q < V; ++q) amax = fmaxf(amax, fabsf(x[q]));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
    const float s = __fdiv_rn(amax, 127.0f);
    if (lane == 0) scale[m] = s;
    for (int64_t v = lane; v < nvec; v += 32) {
      float x[V], q[V], d[V];
      Vec16<T>::load(row + v * V, x);
#pragma unroll
      for (int i = 0; i < V; ++i) {
        q[i] = s > 0.0f ? fminf(fmaxf(rintf(__fdiv_rn(x[i], s)), -127.0f), 127.0f) : 0.0f;
        d[i] = q[i] * s;
      }
      store_vec<T>(codes + m * K + v * V, q);
      if (deq) store_vec<T>(deq + m * K + v * V, d);
    }
  }
}

// ---------------------------------------------------------------- factor-gradient reduction
// One thread per group: sums the dW epilogue's partial sums over contraction splits and
// over the g/P column chunks of the group in a fixed order, then applies
//   d_mu = -alpha0 k S_mu,  d_alpha = alpha0 S_alpha,  d_delta = Delta0 alpha k S_delta,
// k = s / (2 tanh s).
__global__ void __launch_bounds__(kThreads) grad_reduce_kernel(LayerDev L, StepScalars sc,
                                                               const float* __restrict__ part, int32_t splits,
                                                               int32_t P, float* __restrict__ g_dmu,
                                                               float* __restrict__ g_dalpha,
                                                               float* __restrict__ g_ddelta) {
  const int64_t G = L.N * L.K / L.g;
  const int64_t cpr = L.K / P;  // partial chunks per row
  const int32_t cpg = L.g / P;  // partial chunks per group
  const int64_t plane = L.N * cpr;
  for (int64_t j = blockIdx.x * (int64_t)kThreads + threadIdx.x; j < G; j += (int64_t)gridDim.x * kThreads) {
    const int64_t n = j / L.groups_per_row;
    const int64_t c0 = (j % L.groups_per_row) * cpg;
    float s3[3] = {0.f, 0.f, 0.f};
    for (int32_t sp = 0; sp < splits; ++sp)
#pragma unroll
      for (int q = 0; q < 3; ++q) {
        const float* p = part + (static_cast<int64_t>(sp) * 3 + q) * plane + n * cpr + c0;
        for (int32_t c = 0; c < cpg; ++c) s3[q] += p[c];
      }
    const GroupConst gc = group_const(L, j);
    const float k = sc.s * sc.inv_2tanh_s;
    const bool live = gc.alpha != 0.0f;
    g_dmu[j] = live ? -gc.alpha0 * k * s3[0] : 0.0f;
    g_dalpha[j] = live ? gc.alpha0 * s3[1] : 0.0f;
    g_ddelta[j] = live ? gc.delta0 * gc.alpha * k * s3[2] : 0.0f;
  }
}

// Grouped: groups of all experts of a stacked layer; expert e's partials [3][N][K/P] start
// e 3 N K/P floats in, its group arrays e G in; experts without rows get zeros.
struct ExpertRows {
  int32_t rows[kGroupedMaxExperts];
};

__global__ void __launch_bounds__(kThreads) grad_reduce_grouped_kernel(LayerDev L, StepScalars sc,
                                                                       const float* __restrict__ part, int32_t P,
                                                                       int32_t E, const ExpertRows er,
                                                                       float* __restrict__ g_dmu,
                                                                       float* __restrict__ g_dalpha,
                                                                       float* __restrict__ g_ddelta) {
  const int64_t G = L.N * L.K / L.g;
  const int64_t cpr = L.K / P;
  const int32_t cpg = L.g / P;
  const int64_t plane = L.N * cpr;
  const float k = sc.s * sc.inv_2tanh_s;
  for (int64_t ej = blockIdx.x * (int64_t)kThreads + threadIdx.x; ej < E * G; ej += (int64_t)gridDim.x * kThreads) {
    const int64_t e = ej / G, j = ej - e * G;
    float s3[3] = {0.f, 0.f, 0.f};
    bool live = false;
    GroupConst gc{};
    if (er.rows[e] > 0) {
      const int64_t n = j / L.groups_per_row;
      const int64_t c0 = (j % L.groups_per_row) * cpg;
#pragma unroll
      for (int q = 0; q < 3; ++q) {
        const float* p = part + (e * 3 + q) * plane + n * cpr + c0;
        for (int32_t c = 0; c < cpg; ++c) s3[q] += p[c];
      }
      gc = group_const(L, ej);
      live = gc.alpha != 0.0f;
    }
    g_dmu[ej] = live ? -gc.alpha0 * k * s3[0] : 0.0f;
    g_dalpha[ej] = live ? gc.alpha0 * s3[1] : 0.0f;
    g_ddelta[ej] = live ? gc.delta0 * gc.alpha * k * s3[2] : 0.0f;
  }
}

// ---------------------------------------------------------------- factor update (AdamW)
// One thread per group and factor array (blockIdx.y = the factor): decoupled decay, the two
// moment updates, the bias-corrected step and the projection of the factor's constraint.
// Comparisons keep NaN as NaN (a NaN factor is not hidden at a bound).  Reads 16 B and
// writes 12 B per element.
template <int Q>
__device__ __forceinline__ void factor_adamw_array(int64_t G, const AdamwArgs& a) {
  float* const P = a.p[Q];
  const float* const Gr = a.g[Q];
  float* const Mo = a.m[Q];
  float* const Vo = a.v[Q];
  const float lo = a.lo[Q], hi = a.hi[Q];
  for (int64_t i = blockIdx.x * (int64_t)kThreads + threadIdx.x; i < G; i += (int64_t)gridDim.x * kThreads) {
    const float grad = Gr[i];
    float p = P[i] * a.decay;
    const float m = fmaf(a.beta1, Mo[i], a.one_minus_beta1 * grad);
    const float v = fmaf(a.beta2, Vo[i], a.one_minus_beta2 * (grad * grad));
    const float denom = fmaf(sqrtf(v), a.inv_sqrt_bc2, a.eps);
    p -= a.step * (m / denom);
    p = p < lo ? lo : (p > hi ? hi : p);
    P[i] = p;
    Mo[i] = m;
    Vo[i] = v;
  }
}

__global__ void __launch_bounds__(kThreads) factor_adamw_kernel(int64_t G, const AdamwArgs a) {
  // blockIdx.y is uniform per block: each block walks one factor array, no per-element
  // division or pointer select
  if (blockIdx.y == 0) factor_adamw_array<0>(G, a);
  else if (blockIdx.y == 1) factor_adamw_array<1>(G, a);
  else factor_adamw_array<2>(G, a);
}

// ---------------------------------------------------------------- direct learning (DL)
// One thread per group: DL's parameters a = d_alpha and d = d_alpha d_delta (the scale and
// the weight-space threshold in units of the group's static statistics), their gradients
// from the factor gradients by the chain rule, one AdamW step on each, the constraints
// a, d >= margin, and the return to d_alpha = a, d_delta = d / a.  A group with d_alpha == 0
// (only reachable with margin 0) is left unchanged.
__global__ void __launch_bounds__(kThreads) direct_adamw_kernel(int64_t G, const DirectArgs a) {
  for (int64_t i = blockIdx.x * (int64_t)kThreads + threadIdx.x; i < G; i += (int64_t)gridDim.x * kThreads) {
    const float dal = a.d_alpha[i], ddl = a.d_delta[i];
    if (dal == 0.0f) continue;
    const float gal = a.g_dalpha[i], gdl = a.g_ddelta[i];
    const float ga = gal - gdl * ddl / dal;
    const float gd = gdl / dal;
    float p[2] = {dal, dal * ddl};
    const float g2[2] = {ga, gd};
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      float* const Mo = a.m + q * G;
      float* const Vo = a.v + q * G;
      const float m = fmaf(a.beta1, Mo[i], a.one_minus_beta1 * g2[q]);
      const float v = fmaf(a.beta2, Vo[i], a.one_minus_beta2 * (g2[q] * g2[q]));
      const float denom = fmaf(sqrtf(v), a.inv_sqrt_bc2, a.eps);
      float x = p[q] * a.decay;
      x -= a.step * (m / denom);
      p[q] = x < a.margin ? a.margin : x;
      Mo[i] = m;
      Vo[i] = v;
    }
    a.d_alpha[i] = p[0];
    a.d_delta[i] = p[1] / p[0];
  }
}

// ---------------------------------------------------------------- weight reconstruction error
// One warp per group: mean over the group of (W - Wq)^2 with Wq the hard reconstruction
// alpha Q(What; Delta) (+ mu for W ~ alpha T + mu), as the pack and the HARD forward decide
// the codes.  fp32 sums, reduced across the warp in a fixed order.
template <typename T>
__global__ void __launch_bounds__(kThreads) group_recon_error_kernel(LayerDev L, float* __restrict__ err) {
  const int lane = threadIdx.x & 31;
  const int64_t G = L.N * L.K / L.g;
  const T* W = static_cast<const T*>(L.W);
  for (int64_t j = (blockIdx.x * (int64_t)kThreads + threadIdx.x) >> 5; j < G; j += ((int64_t)gridDim.x * kThreads) >> 5) {
    const GroupConst c = group_const(L, j);
    const float m = L.recon ? c.mu : 0.0f;
    float acc = 0.0f;
    for (int32_t e = lane; e < L.g; e += 32) {
      const float w = load_scalar(W + j * L.g + e);
      const float q = c.alpha != 0.0f ? c.alpha * hard_q(what(w, c), c.delta) : 0.0f;
      const float d = w - (q + m);
      acc = fmaf(d, d, acc);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (lane == 0) err[j] = acc / static_cast<float>(L.g);
  }
}

int grid_for(int64_t work, int64_t per_block) {
  int64_t b = (work + per_block - 1) / per_block;
  if (b < 1) b = 1;
  if (b > 152 * 16) b = 152 * 16;
  return static_cast<int>(b);
}

}  // namespace

cudaError_t launch_group_stats(const LayerDev& L, int32_t w_dtype, int32_t thr_init, float* mu0, float* alpha0,
                               float* delta0, cudaStream_t st) {
  const int64_t G = L.N * L.K / L.g;
  const int V = w_dtype == 1 ? 8 : 4;  // elements per 16-byte vector
  const int nvec = L.g / V;            // vectors per group
  const int team = nvec / kStatsVPL;
  if (L.g % V == 0 && nvec % kStatsVPL == 0 && team <= 32 && (team & (team - 1)) == 0) {
    const int per_warp = 32 / team;
    const int grid = grid_for((G + per_warp - 1) / per_warp, kThreads / 32);
    if (thr_init == kThrAbsmean || thr_init == kThrTwnStatic) {
#define CATQ_STATS_STATIC(TT, RULE)                                                                          \
  group_stats_static_kernel<TT, RULE><<<grid, kThreads, 0, st>>>(static_cast<const TT*>(L.W), G, L.g, team, \
                                                                 mu0, alpha0, delta0)
      if (w_dtype == 1) {
        if (thr_init == kThrAbsmean) CATQ_STATS_STATIC(__nv_bfloat16, kThrAbsmean);
        else CATQ_STATS_STATIC(__nv_bfloat16, kThrTwnStatic);
      } else {
        if (thr_init == kThrAbsmean) CATQ_STATS_STATIC(float, kThrAbsmean);
        else CATQ_STATS_STATIC(float, kThrTwnStatic);
      }
#undef CATQ_STATS_STATIC
      return cudaGetLastError();
    }
    const bool twn = thr_init == 1;
#define CATQ_STATS_TEAM(TT, TWN)                                                                                  \
  group_stats_team_kernel<TT, TWN><<<grid, kThreads, 0, st>>>(static_cast<const TT*>(L.W), G, L.g, team, mu0, \
                                                              alpha0, delta0)
    if (w_dtype == 1) {
      if (twn) CATQ_STATS_TEAM(__nv_bfloat16, true);
      else CATQ_STATS_TEAM(__nv_bfloat16, false);
    } else {
      if (twn) CATQ_STATS_TEAM(float, true);
      else CATQ_STATS_TEAM(float, false);
    }
#undef CATQ_STATS_TEAM
    return cudaGetLastError();
  }
  const int grid = grid_for(G, kThreads / 32);
  if (w_dtype == 1)
    group_stats_stream_kernel<__nv_bfloat16><<<grid, kThreads, 0, st>>>(static_cast<const __nv_bfloat16*>(L.W), G,
                                                                          L.g, thr_init, mu0, alpha0, delta0);
  else
    group_stats_stream_kernel<float><<<grid, kThreads, 0, st>>>(static_cast<const float*>(L.W), G, L.g, thr_init,
                                                                mu0, alpha0, delta0);
  return cudaGetLastError();
}

cudaError_t launch_modulate_ternarize(const LayerDev& L, int32_t w_dtype, StepScalars sc, void* Wq, int8_t* T,
                                      float* alpha, cudaStream_t st) {
  if (w_dtype == 1) {
    const int grid = grid_for(L.N * L.K / 8, kThreads);
    modulate_bf16_kernel<<<grid, kThreads, 0, st>>>(L, sc, static_cast<uint16_t*>(Wq), T, alpha);
  } else {
    const int grid = grid_for(L.N * L.K, kThreads);
    modulate_f32_kernel<<<grid, kThreads, 0, st>>>(L, sc, static_cast<float*>(Wq), T, alpha);
  }
  return cudaGetLastError();
}

int recon_loss_blocks(int64_t count) {
  int64_t b = (count + 8LL * kThreads * 4 - 1) / (8LL * kThreads * 4);
  if (b < 1) b = 1;
  if (b > kLossMaxBlocks) b = kLossMaxBlocks;
  return static_cast<int>(b);
}

cudaError_t launch_recon_loss(const void* Y, const void* Yr, int64_t count, int32_t dtype, int32_t reduction,
                              float* loss_out, void* dY, double* partials, cudaStream_t st) {
  const int nb = recon_loss_blocks(count);
  const double inv = reduction == 0 ? 1.0 / static_cast<double>(count) : 1.0;
  const float scale = static_cast<float>(2.0 * inv);
  if (dtype == 1)
    recon_loss_partial_kernel<__nv_bfloat16><<<nb, kThreads, 0, st>>>(
        static_cast<const __nv_bfloat16*>(Y), static_cast<const __nv_bfloat16*>(Yr), count, scale,
        static_cast<__nv_bfloat16*>(dY), partials);
  else
    recon_loss_partial_kernel<float><<<nb, kThreads, 0, st>>>(static_cast<const float*>(Y),
                                                              static_cast<const float*>(Yr), count, scale,
                                                              static_cast<float*>(dY), partials);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  recon_loss_final_kernel<<<1, kThreads, 0, st>>>(partials, nb, inv, loss_out);
  return cudaGetLastError();
}

cudaError_t launch_loss_final(const double* partials, int n, double out_scale, float* loss, cudaStream_t st) {
  recon_loss_final_kernel<<<1, kThreads, 0, st>>>(partials, n, out_scale, loss);
  return cudaGetLastError();
}

cudaError_t launch_act_quant_a8(const void* X, int64_t M, int64_t K, int32_t dtype, void* codes, float* scale,
                                void* deq, cudaStream_t st) {
  const int grid = grid_for((M + kThreads / 32 - 1) / (kThreads / 32), 1);
  if (dtype == 1)
    act_quant_a8_kernel<__nv_bfloat16><<<grid, kThreads, 0, st>>>(static_cast<const __nv_bfloat16*>(X), M, K,
                                                                   static_cast<__nv_bfloat16*>(codes), scale,
                                                                   static_cast<__nv_bfloat16*>(deq));
  else
    act_quant_a8_kernel<float><<<grid, kThreads, 0, st>>>(static_cast<const float*>(X), M, K,
                                                           static_cast<float*>(codes), scale,
                                                           static_cast<float*>(deq));
  return cudaGetLastError();
}

cudaError_t launch_hard_pack(const LayerDev& L, int32_t w_dtype, uint8_t* codes, float* alpha, float* mu,
                             cudaStream_t st) {
  const int64_t n = L.N * L.K;
  const int V = w_dtype == 1 ? 8 : 4;
  if (L.g % 64 == 0 && (L.g & (L.g - 1)) == 0 && L.g >= 8 * V) {
    int log2g = 0;
    while ((1 << log2g) < L.g) ++log2g;
    const int64_t batches = (n + 256LL * V - 1) / (256LL * V);
    const int grid = grid_for(batches, kThreads / 32);
    if (w_dtype == 1)
      hard_pack_warp_kernel<__nv_bfloat16><<<grid, kThreads, 0, st>>>(L, log2g, codes, alpha, mu);
    else
      hard_pack_warp_kernel<float><<<grid, kThreads, 0, st>>>(L, log2g, codes, alpha, mu);
  } else if (L.g % 64 == 0) {
    const int grid = grid_for(n / 64, kThreads);
    if (w_dtype == 1)
      hard_pack_kernel<__nv_bfloat16, 64><<<grid, kThreads, 0, st>>>(L, codes, alpha, mu);
    else
      hard_pack_kernel<float, 64><<<grid, kThreads, 0, st>>>(L, codes, alpha, mu);
  } else if (L.g % 16 == 0) {
    const int grid = grid_for(n / 16, kThreads);
    if (w_dtype == 1)
      hard_pack_kernel<__nv_bfloat16, 16><<<grid, kThreads, 0, st>>>(L, codes, alpha, mu);
    else
      hard_pack_kernel<float, 16><<<grid, kThreads, 0, st>>>(L, codes, alpha, mu);
  } else {
    const int grid = grid_for(n / 4, kThreads);
    if (w_dtype == 1)
      hard_pack_kernel<__nv_bfloat16, 4><<<grid, kThreads, 0, st>>>(L, codes, alpha, mu);
    else
      hard_pack_kernel<float, 4><<<grid, kThreads, 0, st>>>(L, codes, alpha, mu);
  }
  return cudaGetLastError();
}

cudaError_t launch_operand_consts(const LayerDev& L, StepScalars sc, cudaStream_t st) {
  const int64_t row_tiles = (L.N + kConstTile - 1) / kConstTile;
  const dim3 grid(static_cast<unsigned>((L.groups_per_row + kConstTile - 1) / kConstTile),
                  static_cast<unsigned>(row_tiles < 65535 ? row_tiles : 65535));
  operand_consts_kernel<<<grid, dim3(kConstTile, kConstTile), 0, st>>>(L, sc, 0);
  return cudaGetLastError();
}

cudaError_t launch_operand_consts_grouped(const LayerDev& L0, StepScalars sc, int32_t E, int64_t const_stride,
                                          cudaStream_t st) {
  const int64_t row_tiles = (L0.N + kConstTile - 1) / kConstTile;
  const dim3 grid(static_cast<unsigned>((L0.groups_per_row + kConstTile - 1) / kConstTile),
                  static_cast<unsigned>(row_tiles < 65535 ? row_tiles : 65535), static_cast<unsigned>(E));
  operand_consts_kernel<<<grid, dim3(kConstTile, kConstTile), 0, st>>>(L0, sc, const_stride);
  return cudaGetLastError();
}

cudaError_t launch_grad_reduce_grouped(const LayerDev& L0, StepScalars sc, const float* partials, int32_t P,
                                       const GroupSpec& grp, float* g_dmu, float* g_dalpha, float* g_ddelta,
                                       cudaStream_t st) {
  ExpertRows er{};
  for (int32_t e = 0; e < grp.E; ++e) er.rows[e] = static_cast<int32_t>(grp.off[e + 1] - grp.off[e] > 0 ? 1 : 0);
  const int64_t G = L0.N * L0.K / L0.g;
  grad_reduce_grouped_kernel<<<grid_for(grp.E * G, kThreads), kThreads, 0, st>>>(L0, sc, partials, P, grp.E, er, g_dmu,
                                                                                 g_dalpha, g_ddelta);
  return cudaGetLastError();
}

cudaError_t launch_grad_reduce(const LayerDev& L, StepScalars sc, const float* partials, int32_t splits, int32_t P,
                               float* g_dmu, float* g_dalpha, float* g_ddelta, cudaStream_t st) {
  const int64_t G = L.N * L.K / L.g;
  grad_reduce_kernel<<<grid_for(G, kThreads), kThreads, 0, st>>>(L, sc, partials, splits, P, g_dmu, g_dalpha,
                                                                 g_ddelta);
  return cudaGetLastError();
}

cudaError_t launch_direct_adamw(int64_t G, const DirectArgs& a, cudaStream_t st) {
  if (G == 0) return cudaSuccess;
  direct_adamw_kernel<<<grid_for(G, kThreads), kThreads, 0, st>>>(G, a);
  return cudaGetLastError();
}

cudaError_t launch_group_recon_error(const LayerDev& L, int32_t w_dtype, float* err, cudaStream_t st) {
  const int64_t G = L.N * L.K / L.g;
  const int grid = grid_for((G + kThreads / 32 - 1) / (kThreads / 32), 1);
  if (w_dtype == 1) group_recon_error_kernel<__nv_bfloat16><<<grid, kThreads, 0, st>>>(L, err);
  else group_recon_error_kernel<float><<<grid, kThreads, 0, st>>>(L, err);
  return cudaGetLastError();
}

cudaError_t launch_factor_adamw(int64_t G, const AdamwArgs& a, cudaStream_t st) {
  if (G == 0) return cudaSuccess;
  factor_adamw_kernel<<<dim3(grid_for(G, kThreads), 3), kThreads, 0, st>>>(G, a);
  return cudaGetLastError();
}

}  // namespace catq
