// catq_math.cuh — per-group constants and per-element arithmetic of LM + ST, shared by
// every kernel of the library so the fused GEMM operand producer, the materialising
// kernel and the pack kernel take identical decisions.
#pragma once
#include <cstdint>

namespace catq {

enum : int32_t { PHASE_TEACHER = 0, PHASE_SOFT = 1, PHASE_HARD = 2 };

// Device view of one layer (catq_layer plus derived sizes).
struct LayerDev {
  const void* W;
  int64_t N, K;
  int32_t g;
  int32_t groups_per_row;  // K / g
  const float* mu0;
  const float* alpha0;
  const float* delta0;
  const float* d_mu;
  const float* d_alpha;
  const float* d_delta;
};

// Eq. 3 and §2.2 for group j:
//   mu = mu0 + d_mu alpha0, alpha = d_alpha alpha0, Delta = d_delta Delta0,
//   What = (W - mu) / alpha evaluated as fma(W, r, b) with r = 1/alpha, b = -mu r.
// alpha == 0 (degenerate group) gives r = b = 0, so What = 0 and alpha * T = 0.
struct GroupConst {
  float r, b, alpha, delta, alpha0, delta0;
};

__device__ __forceinline__ GroupConst group_const(const LayerDev& L, int64_t j) {
  const float a0 = __ldg(L.alpha0 + j);
  const float m0 = __ldg(L.mu0 + j);
  const float D0 = __ldg(L.delta0 + j);
  const float mu = fmaf(__ldg(L.d_mu + j), a0, m0);
  const float alpha = __ldg(L.d_alpha + j) * a0;
  const float delta = __ldg(L.d_delta + j) * D0;
  const float r = (alpha != 0.0f) ? 1.0f / alpha : 0.0f;
  GroupConst c;
  c.r = r;
  c.b = -mu * r;
  c.alpha = alpha;
  c.delta = delta;
  c.alpha0 = a0;
  c.delta0 = D0;
  return c;
}

__device__ __forceinline__ float what(float w, const GroupConst& c) { return fmaf(w, c.r, c.b); }

// Eq. 2 on What.
__device__ __forceinline__ float hard_q(float x, float delta) {
  return x > delta ? 1.0f : (x < -delta ? -1.0f : 0.0f);
}

// ---------------------------------------------------------------- bf16 helpers

__device__ __forceinline__ float bf16lo_to_f32(uint32_t w2) { return __uint_as_float(w2 << 16); }
__device__ __forceinline__ float bf16hi_to_f32(uint32_t w2) { return __uint_as_float(w2 & 0xFFFF0000u); }

// (lo, hi) -> packed bf16x2, round to nearest even.
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  uint32_t d;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
  return d;
}

__device__ __forceinline__ uint32_t tanh_bf16x2(uint32_t x) {
  uint32_t d;
  asm("tanh.approx.bf16x2 %0, %1;" : "=r"(d) : "r"(x));
  return d;
}

__device__ __forceinline__ uint32_t add_bf16x2(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("add.rn.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}

__device__ __forceinline__ uint32_t mul_bf16x2(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("mul.rn.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}

// Per-row constants of the bf16 operand producer for one group (see soft_pair_bf16).
struct ProducerConst {
  float A, B, D;   // SOFT: u = s * What = fma(w, A, B); D = s * Delta
  uint32_t C2;     // SOFT: alpha / (2 tanh s) as bf16x2; HARD: alpha as bf16x2
  float r, b, delta;  // HARD: What = fma(w, r, b), threshold Delta
};

__device__ __forceinline__ ProducerConst producer_const(const GroupConst& c, float s, float inv_2tanh_s,
                                                        int32_t phase) {
  ProducerConst p;
  p.A = s * c.r;
  p.B = s * c.b;
  p.D = s * c.delta;
  const float C = (phase == PHASE_SOFT) ? c.alpha * inv_2tanh_s : c.alpha;
  p.C2 = pack_bf16x2(C, C);
  p.r = c.r;
  p.b = c.b;
  p.delta = c.delta;
  return p;
}

// Eq. 5/6 SOFT weight for two bf16 weights: alpha f(What; s, Delta) =
//   [alpha / (2 tanh s)] * [tanh(u - s Delta) + tanh(u + s Delta)],  u = s What,
// with u computed in fp32, both tanh arguments rounded to bf16 and evaluated together by
// one packed tanh, and the sum and scale in bf16 (the operand's precision).
__device__ __forceinline__ uint32_t soft_pair_bf16(uint32_t w2, const ProducerConst& p) {
  const float u0 = fmaf(bf16lo_to_f32(w2), p.A, p.B);
  const float u1 = fmaf(bf16hi_to_f32(w2), p.A, p.B);
  const uint32_t tm = tanh_bf16x2(pack_bf16x2(u0 - p.D, u1 - p.D));
  const uint32_t tp = tanh_bf16x2(pack_bf16x2(u0 + p.D, u1 + p.D));
  return mul_bf16x2(add_bf16x2(tm, tp), p.C2);
}

// Eq. 2/6 HARD weight for two bf16 weights: alpha Q(What; Delta).
__device__ __forceinline__ uint32_t hard_pair_bf16(uint32_t w2, const ProducerConst& p) {
  const float x0 = fmaf(bf16lo_to_f32(w2), p.r, p.b);
  const float x1 = fmaf(bf16hi_to_f32(w2), p.r, p.b);
  const uint32_t a = p.C2 & 0xFFFFu;
  const uint32_t lo = x0 > p.delta ? a : (x0 < -p.delta ? (a | 0x8000u) : 0u);
  const uint32_t hi = x1 > p.delta ? a : (x1 < -p.delta ? (a | 0x8000u) : 0u);
  return lo | (hi << 16);
}

__device__ __forceinline__ uint4 transform_chunk_bf16(uint4 v, const ProducerConst& p, int32_t phase) {
  if (phase == PHASE_SOFT) {
    v.x = soft_pair_bf16(v.x, p);
    v.y = soft_pair_bf16(v.y, p);
    v.z = soft_pair_bf16(v.z, p);
    v.w = soft_pair_bf16(v.w, p);
  } else if (phase == PHASE_HARD) {
    v.x = hard_pair_bf16(v.x, p);
    v.y = hard_pair_bf16(v.y, p);
    v.z = hard_pair_bf16(v.z, p);
    v.w = hard_pair_bf16(v.w, p);
  }
  return v;
}

// ---------------------------------------------------------------- fp32 path

// Eq. 5/6 in fp32 with accurate tanh (CUDA-core path).
__device__ __forceinline__ float ternary_weight_f32(float w, const GroupConst& c, float s, float inv_2tanh_s,
                                                    int32_t phase) {
  if (phase == PHASE_TEACHER) return w;
  const float x = what(w, c);
  if (phase == PHASE_HARD) return c.alpha * hard_q(x, c.delta);
  return c.alpha * inv_2tanh_s * (tanhf(s * (x - c.delta)) + tanhf(s * (x + c.delta)));
}

// ---------------------------------------------------------------- factor-gradient element

// tanh(y) and 1 - tanh(y)^2 with good relative accuracy in the tails:
// e = exp(-2|y|), tanh|y| = (1 - e)/(1 + e), sech^2 y = 4 e / (1 + e)^2.
__device__ __forceinline__ void tanh_sech2(float y, float& t, float& s2) {
  const float e = expf(-2.0f * fabsf(y));
  const float rcp = 1.0f / (1.0f + e);
  t = copysignf((1.0f - e) * rcp, y);
  s2 = 4.0f * e * rcp * rcp;
}

// Running per-group sums of the chain rule (Eq. 3, 5, 6):
//   smu = sum G f'(What) / k,  salpha = sum G (T - What f'(What)),  sdelta = sum G df/dDelta / k
// with f' = k (sech^2 a + sech^2 b), df/dDelta = k (sech^2 b - sech^2 a), k = s / (2 tanh s).
struct GradSums {
  float smu, salpha, sdelta;
};

__device__ __forceinline__ void grad_element(float G, float w, const GroupConst& c, float s, float inv_2tanh_s,
                                             int32_t phase, GradSums& acc) {
  const float x = what(w, c);
  float ta, sa, tb, sb;
  tanh_sech2(s * (x - c.delta), ta, sa);
  tanh_sech2(s * (x + c.delta), tb, sb);
  const float k = s * inv_2tanh_s;
  const float fp_over_k = sa + sb;
  const float T = (phase == PHASE_SOFT) ? inv_2tanh_s * (ta + tb) : hard_q(x, c.delta);
  acc.smu = fmaf(G, fp_over_k, acc.smu);
  acc.salpha = fmaf(G, T - x * k * fp_over_k, acc.salpha);
  acc.sdelta = fmaf(G, sb - sa, acc.sdelta);
}

}  // namespace catq
