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
  float4* op_const;  // [K/g][N] operand constants (operand_const_vec), written per call
  float* op_mu;      // [K/g][N] group offsets mu after op_const when recon, else nullptr
  int32_t recon;     // 0: W ~ alpha T (§2.2);  1: W ~ alpha T + mu (the tab:mu variant)
};

// Eq. 3 and §2.2 for group j:
//   mu = mu0 + d_mu alpha0, alpha = d_alpha alpha0, Delta = d_delta Delta0,
//   What = (W - mu) / alpha evaluated as fma(W, r, b) with r = 1/alpha, b = -mu r.
// alpha == 0 (degenerate group) gives r = b = 0, so What = 0 and alpha * T = 0.
struct GroupConst {
  float r, b, alpha, delta, alpha0, delta0, mu;
};

// The six per-group inputs, loaded separately from the arithmetic so callers can issue the
// loads a pipeline stage before they need the constants.
struct GroupRaw {
  float a0, m0, D0, dmu, dal, ddl;
};

__device__ __forceinline__ GroupRaw group_raw(const LayerDev& L, int64_t j) {
  GroupRaw g;
  g.a0 = __ldg(L.alpha0 + j);
  g.m0 = __ldg(L.mu0 + j);
  g.D0 = __ldg(L.delta0 + j);
  g.dmu = __ldg(L.d_mu + j);
  g.dal = __ldg(L.d_alpha + j);
  g.ddl = __ldg(L.d_delta + j);
  return g;
}

__device__ __forceinline__ GroupConst group_const(const GroupRaw& g) {
  const float mu = fmaf(g.dmu, g.a0, g.m0);
  const float alpha = g.dal * g.a0;
  const float delta = g.ddl * g.D0;
  const float r = (alpha != 0.0f) ? __frcp_rn(alpha) : 0.0f;  // correctly rounded 1 / alpha
  GroupConst c;
  c.r = r;
  c.b = -mu * r;
  c.alpha = alpha;
  c.delta = delta;
  c.alpha0 = g.a0;
  c.delta0 = g.D0;
  c.mu = mu;
  return c;
}

__device__ __forceinline__ GroupConst group_const(const LayerDev& L, int64_t j) { return group_const(group_raw(L, j)); }

__device__ __forceinline__ float what(float w, const GroupConst& c) { return fmaf(w, c.r, c.b); }

// Eq. 2 on What.
__device__ __forceinline__ float hard_q(float x, float delta) {
  return x > delta ? 1.0f : (x < -delta ? -1.0f : 0.0f);
}

// ---------------------------------------------------------------- compensated fp32 sums
// (used by the statistics, the loss and the fused forward + loss epilogue)
// fp64 arithmetic is slow on this GPU, so sums use an fp32 value plus an fp32 error term
// (Knuth's two-sum), which carries about twice fp32's precision.
struct Sum2 {
  float hi, lo;
};

__device__ __forceinline__ void sum2_add(Sum2& a, float x) {
  const float s = a.hi + x;
  const float bp = s - a.hi;
  const float err = (a.hi - (s - bp)) + (x - bp);
  a.hi = s;
  a.lo += err;
}

__device__ __forceinline__ Sum2 sum2_merge(Sum2 a, Sum2 b) {
  const float s = a.hi + b.hi;
  const float bp = s - a.hi;
  const float err = (a.hi - (s - bp)) + (b.hi - bp);
  return Sum2{s, a.lo + b.lo + err};
}

// Butterfly reduction over aligned teams of `team` lanes (team a power of two <= 32).
__device__ __forceinline__ Sum2 sum2_team(Sum2 v, int team) {
  for (int o = team >> 1; o > 0; o >>= 1) {
    Sum2 w;
    w.hi = __shfl_xor_sync(0xffffffffu, v.hi, o);
    w.lo = __shfl_xor_sync(0xffffffffu, v.lo, o);
    v = sum2_merge(v, w);
  }
  return v;
}

__device__ __forceinline__ double sum2_value(Sum2 v) { return static_cast<double>(v.hi) + static_cast<double>(v.lo); }

// ---------------------------------------------------------------- bf16 helpers

__device__ __forceinline__ float bf16lo_to_f32(uint32_t w2) { return __uint_as_float(w2 << 16); }
__device__ __forceinline__ float bf16hi_to_f32(uint32_t w2) { return __uint_as_float(w2 & 0xFFFF0000u); }

// (lo, hi) -> packed bf16x2, round to nearest even.
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  uint32_t d;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
  return d;
}

// Per-row constants of the bf16 operand producer for one group.
//   SOFT: u = s What = fma(w, A, B), D = s Delta, C = alpha / (2 tanh s);
//         `one_tanh` when D >= 6: for u >= 0 the term tanh(u + D) >= tanh 6 = 1 - 1.2e-5 is
//         1 to well below bf16 resolution (and symmetrically for u < 0), so
//         alpha f = sign(u) C (1 + tanh(|u| - D)) needs one tanh instead of two.
//   HARD: What = fma(w, r, b), threshold Delta, C = alpha.
//   M: the group offset mu added to alpha T in the W ~ alpha T + mu reconstruction (read only
//   by the transforms of that reconstruction).
struct ProducerConst {
  float A, B, D, C;
  float r, b, delta;
  float M;
  bool one_tanh;
};

__device__ __forceinline__ ProducerConst producer_const(const GroupConst& c, float s, float inv_2tanh_s,
                                                        int32_t phase) {
  ProducerConst p;
  p.M = c.mu;
  p.A = s * c.r;
  p.B = s * c.b;
  p.D = s * c.delta;
  p.C = (phase == PHASE_SOFT) ? c.alpha * inv_2tanh_s : c.alpha;
  p.r = c.r;
  p.b = c.b;
  p.delta = c.delta;
  p.one_tanh = p.D >= 6.0f;
  return p;
}

__device__ __forceinline__ float tanh_fast(float x) {
  float y;
  asm("tanh.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Eq. 5/6 SOFT weight alpha f(What; s, Delta) for two bf16 weights, fp32 arithmetic with
// the hardware tanh, rounded once to bf16.  ONE_TANH selects the one-tanh form (valid when
// p.one_tanh); the choice is made once per row, outside the element loop.
// MU adds the group offset (alpha f + mu, one rounding).
template <bool ONE_TANH, bool MU = false>
__device__ __forceinline__ uint32_t soft_pair_bf16(uint32_t w2, const ProducerConst& p) {
  const float u0 = fmaf(bf16lo_to_f32(w2), p.A, p.B);
  const float u1 = fmaf(bf16hi_to_f32(w2), p.A, p.B);
  float y0, y1;
  if constexpr (ONE_TANH) {
    const float c0 = copysignf(p.C, u0), c1 = copysignf(p.C, u1);
    y0 = fmaf(tanh_fast(fabsf(u0) - p.D), c0, MU ? c0 + p.M : c0);
    y1 = fmaf(tanh_fast(fabsf(u1) - p.D), c1, MU ? c1 + p.M : c1);
  } else if constexpr (MU) {
    y0 = fmaf(p.C, tanh_fast(u0 - p.D) + tanh_fast(u0 + p.D), p.M);
    y1 = fmaf(p.C, tanh_fast(u1 - p.D) + tanh_fast(u1 + p.D), p.M);
  } else {
    y0 = p.C * (tanh_fast(u0 - p.D) + tanh_fast(u0 + p.D));
    y1 = p.C * (tanh_fast(u1 - p.D) + tanh_fast(u1 + p.D));
  }
  return pack_bf16x2(y0, y1);
}

// Eq. 2/6 HARD weight alpha Q(What; Delta) (+ mu when MU) for two bf16 weights.
template <bool MU = false>
__device__ __forceinline__ uint32_t hard_pair_bf16(uint32_t w2, const ProducerConst& p) {
  const float x0 = fmaf(bf16lo_to_f32(w2), p.r, p.b);
  const float x1 = fmaf(bf16hi_to_f32(w2), p.r, p.b);
  float y0 = fabsf(x0) > p.delta ? copysignf(p.C, x0) : 0.0f;  // Q(x) = sign(x) [|x| > Delta]
  float y1 = fabsf(x1) > p.delta ? copysignf(p.C, x1) : 0.0f;
  if constexpr (MU) {
    y0 += p.M;
    y1 += p.M;
  }
  return pack_bf16x2(y0, y1);
}

// The four per-group values a producer row needs, packed for one 16-byte load:
//   SOFT {A, B, D, C} = {s r, s b, s Delta, alpha / (2 tanh s)}, HARD {r, b, Delta, alpha}.
__device__ __forceinline__ float4 operand_const_vec(const GroupConst& c, float s, float inv_2tanh_s, int32_t phase) {
  const ProducerConst p = producer_const(c, s, inv_2tanh_s, phase);
  return phase == PHASE_HARD ? make_float4(p.r, p.b, p.delta, p.C) : make_float4(p.A, p.B, p.D, p.C);
}

// Inverse of operand_const_vec for the transform of `phase`; m is the group offset mu (0
// when the reconstruction has none).
__device__ __forceinline__ ProducerConst producer_const_from(float4 v, float m) {
  ProducerConst p;
  p.M = m;
  p.A = p.r = v.x;
  p.B = p.b = v.y;
  p.D = p.delta = v.z;
  p.C = v.w;
  p.one_tanh = v.z >= 6.0f;
  return p;
}

// Element transforms; XF_MU marks the W ~ alpha T + mu forms of SOFT1, SOFT2 and HARD.
enum : int32_t { XF_COPY = 0, XF_SOFT1 = 1, XF_SOFT2 = 2, XF_HARD = 3, XF_MU = 4 };

// Which element transform a row uses in `phase` (`recon` as LayerDev::recon).
__device__ __forceinline__ int32_t transform_kind(const ProducerConst& p, int32_t phase, int32_t recon) {
  const int32_t mu = recon ? XF_MU : 0;
  if (phase == PHASE_SOFT) return (p.one_tanh ? XF_SOFT1 : XF_SOFT2) | mu;
  return phase == PHASE_HARD ? (XF_HARD | mu) : XF_COPY;
}

template <int KIND>
__device__ __forceinline__ uint4 transform_chunk(uint4 v, const ProducerConst& p) {
  constexpr bool MU = (KIND & XF_MU) != 0;
  constexpr int BASE = KIND & ~XF_MU;
  if constexpr (BASE == XF_SOFT1) {
    v.x = soft_pair_bf16<true, MU>(v.x, p);
    v.y = soft_pair_bf16<true, MU>(v.y, p);
    v.z = soft_pair_bf16<true, MU>(v.z, p);
    v.w = soft_pair_bf16<true, MU>(v.w, p);
  } else if constexpr (BASE == XF_SOFT2) {
    v.x = soft_pair_bf16<false, MU>(v.x, p);
    v.y = soft_pair_bf16<false, MU>(v.y, p);
    v.z = soft_pair_bf16<false, MU>(v.z, p);
    v.w = soft_pair_bf16<false, MU>(v.w, p);
  } else if constexpr (BASE == XF_HARD) {
    v.x = hard_pair_bf16<MU>(v.x, p);
    v.y = hard_pair_bf16<MU>(v.y, p);
    v.z = hard_pair_bf16<MU>(v.z, p);
    v.w = hard_pair_bf16<MU>(v.w, p);
  }
  return v;
}

// The Eq. 6 operand for one 16-byte chunk of a row (8 bf16 weights of one group).
__device__ __forceinline__ uint4 transform_chunk_bf16(uint4 v, const ProducerConst& p, int32_t phase, int32_t recon) {
  switch (transform_kind(p, phase, recon)) {
    case XF_SOFT1: return transform_chunk<XF_SOFT1>(v, p);
    case XF_SOFT2: return transform_chunk<XF_SOFT2>(v, p);
    case XF_HARD: return transform_chunk<XF_HARD>(v, p);
    case XF_SOFT1 | XF_MU: return transform_chunk<XF_SOFT1 | XF_MU>(v, p);
    case XF_SOFT2 | XF_MU: return transform_chunk<XF_SOFT2 | XF_MU>(v, p);
    case XF_HARD | XF_MU: return transform_chunk<XF_HARD | XF_MU>(v, p);
    default: return v;
  }
}

// ---------------------------------------------------------------- fp32 path

// Eq. 5/6 in fp32 with accurate tanh (CUDA-core path); recon adds mu.
__device__ __forceinline__ float ternary_weight_f32(float w, const GroupConst& c, float s, float inv_2tanh_s,
                                                    int32_t phase, int32_t recon) {
  if (phase == PHASE_TEACHER) return w;
  const float x = what(w, c);
  const float m = recon ? c.mu : 0.0f;
  if (phase == PHASE_HARD) return fmaf(c.alpha, hard_q(x, c.delta), m);
  return fmaf(c.alpha * inv_2tanh_s, tanhf(s * (x - c.delta)) + tanhf(s * (x + c.delta)), m);
}

// ---------------------------------------------------------------- factor-gradient element

// tanh(y) and 1 - tanh(y)^2 with good relative accuracy in the tails:
// e = exp(-2|y|), tanh|y| = (1 - e)/(1 + e), sech^2 y = 4 e / (1 + e)^2.
// FAST uses the hardware exp2 and reciprocal (__expf, __fdividef; relative error near
// 1e-6, also in the tails) for the bf16 path; otherwise the correctly rounded library calls.
template <bool FAST = false>
__device__ __forceinline__ void tanh_sech2(float y, float& t, float& s2) {
  const float e = FAST ? __expf(-2.0f * fabsf(y)) : expf(-2.0f * fabsf(y));
  const float rcp = FAST ? __fdividef(1.0f, 1.0f + e) : 1.0f / (1.0f + e);
  t = copysignf((1.0f - e) * rcp, y);
  s2 = 4.0f * e * rcp * rcp;
}

// Running per-group sums of the chain rule (Eq. 3, 5, 6):
//   smu = sum G f'(What) / k,  salpha = sum G (T - What f'(What)),  sdelta = sum G df/dDelta / k
// with f' = k (sech^2 a + sech^2 b), df/dDelta = k (sech^2 b - sech^2 a), k = s / (2 tanh s).
// With mu in the reconstruction (W ~ alpha T + mu) dWq/dmu is 1 - f' instead of -f', and
// MU accumulates smu = sum G (f' - 1) / k instead (inv_k = 1/k), so that the factor
// gradient is -alpha0 k smu in both cases.
struct GradSums {
  float smu, salpha, sdelta;
};

template <bool FAST = false, bool MU = false>
__device__ __forceinline__ void grad_element(float G, float w, const GroupConst& c, float s, float inv_2tanh_s,
                                             int32_t phase, GradSums& acc, float inv_k = 0.0f) {
  const float x = what(w, c);
  float ta, sa, tb, sb;
  tanh_sech2<FAST>(s * (x - c.delta), ta, sa);
  tanh_sech2<FAST>(s * (x + c.delta), tb, sb);
  const float k = s * inv_2tanh_s;
  const float fp_over_k = sa + sb;
  const float T = (phase == PHASE_SOFT) ? inv_2tanh_s * (ta + tb) : hard_q(x, c.delta);
  acc.smu = fmaf(G, MU ? fp_over_k - inv_k : fp_over_k, acc.smu);
  acc.salpha = fmaf(G, T - x * k * fp_over_k, acc.salpha);
  acc.sdelta = fmaf(G, sb - sa, acc.sdelta);
}

// One-exponential form of grad_element for a group whose threshold in sharpness units is
// D = s Delta >= kOneExpD.  For x >= 0 the term tanh(s(x + Delta)) is then within
// 2 exp(-2 D) <= 3e-8 of 1 and its sech^2 below 4 exp(-2 D) <= 6e-8, both under fp32
// resolution of the O(1) terms they join (symmetrically for x < 0), so with the near term
// y = s|x| - D alone:
//   f'/k = sech^2 y,   (df/dDelta)/k = -sign(x) sech^2 y,
//   SOFT T = f = sign(x) (1 + tanh y) / (2 tanh s)     (the producer's one-tanh form).
constexpr float kOneExpD = 9.0f;

// That near-term form through the logistic function, for the dW epilogue, which runs it on
// every weight: with y = s|x| - D,
//   exp(-2y) = 2^(|x| c1 + c2),   c1 = -2 s log2(e),  c2 = 2 D log2(e),
//   p = 1 + tanh y = 2 / (1 + exp(-2y)),   sech^2 y = (1 - tanh y)(1 + tanh y) = p^2 exp(-2y),
//   SOFT T = sign(x) p / (2 tanh s),
// one exp2, one reciprocal and a handful of multiply-adds per element (the phase is a template
// argument, decided once per chunk).  Where a group's exponent can pass 126 it is capped there,
// which happens only far inside the threshold where sech^2 y is below fp32 resolution anyway,
// so exp(-2y) stays finite.
struct OneExp {
  float c1, c2;
};

__device__ __forceinline__ OneExp one_exp_consts(float s, float D) {
  constexpr float kLog2e = 1.4426950408889634f;
  return OneExp{-2.0f * kLog2e * s, 2.0f * kLog2e * D};
}

__device__ __forceinline__ float ex2_approx(float a) {
  float r;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(a));
  return r;
}

__device__ __forceinline__ float rcp_approx(float a) {
  float r;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(a));
  return r;
}

// Running sums of the logistic form, with the per-element work cut to what varies per weight:
//   smu   = sum G s2   (MU: sum G (s2 - 1/k)),
//   st    = sum G sign(x) p   (SOFT; HARD: sum G Q(x)),
//   sxs   = sum G x s2,
//   sdelta = -sum G sign(x) s2,
// from which salpha = (1/(2 tanh s)) st - k sxs (SOFT; HARD: st - k sxs) once per partial.
struct LogiSums {
  float smu, st, sxs, sdelta;
};

__device__ __forceinline__ GradSums grad_sums(const LogiSums& l, bool soft, float inv_2tanh_s, float k) {
  return GradSums{l.smu, fmaf(-k, l.sxs, soft ? inv_2tanh_s * l.st : l.st), l.sdelta};
}

// grad_element's two-exponential form into the same sums (T without its 1/(2 tanh s) factor
// in the SOFT phase), for groups whose threshold in sharpness units is below kOneExpD.
template <bool MU>
__device__ __forceinline__ void grad_element_sums(float G, float w, const GroupConst& c, float s, int32_t phase,
                                                  LogiSums& acc, float inv_k) {
  const float x = what(w, c);
  float ta, sa, tb, sb;
  tanh_sech2<true>(s * (x - c.delta), ta, sa);
  tanh_sech2<true>(s * (x + c.delta), tb, sb);
  const float a = G * (sa + sb);
  acc.smu += MU ? fmaf(-G, inv_k, a) : a;
  acc.sxs = fmaf(x, a, acc.sxs);
  acc.st = fmaf(G, phase == PHASE_SOFT ? ta + tb : hard_q(x, c.delta), acc.st);
  acc.sdelta = fmaf(G, sb - sa, acc.sdelta);
}

// a times the sign of -x: a's sign bit flipped unless x's is set (one logic operation; x = +0
// counts as positive, as copysign(1, -x) does).
__device__ __forceinline__ float times_sign_of_neg(float a, float x) {
  return __int_as_float(__float_as_int(a) ^ (~__float_as_int(x) & 0x80000000));
}

// CLAMP caps the exponent at 126; a group needs it only when its largest exponent, c2 (at
// x = 0), is above that.
template <bool MU, bool SOFT, bool CLAMP>
__device__ __forceinline__ void grad_element_logistic(float G, float w, const GroupConst& c, const OneExp& oe,
                                                      LogiSums& acc, float inv_k) {
  const float x = what(w, c);
  float y = fmaf(fabsf(x), oe.c1, oe.c2);
  if constexpr (CLAMP) y = fminf(y, 126.0f);
  const float e = ex2_approx(y);
  const float p = rcp_approx(fmaf(e, 0.5f, 0.5f));
  const float a = G * (p * p * e);
  acc.smu += MU ? fmaf(-G, inv_k, a) : a;
  acc.sxs = fmaf(x, a, acc.sxs);
  acc.st = fmaf(G, SOFT ? copysignf(p, x) : hard_q(x, c.delta), acc.st);
  acc.sdelta += times_sign_of_neg(a, x);
}

// 32 consecutive elements of one row: fp32 accumulator values g[0..31] and the bf16 weights
// packed two per word in w[0..3].
template <bool MU, bool SOFT, bool CLAMP>
__device__ __forceinline__ void grad_chunk_logistic(const uint32_t (&g)[32], const uint4 (&w)[4], const GroupConst& c,
                                                    const OneExp& oe, LogiSums& acc, float inv_k) {
#pragma unroll
  for (int v = 0; v < 4; ++v) {
    const uint32_t w4[4] = {w[v].x, w[v].y, w[v].z, w[v].w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      grad_element_logistic<MU, SOFT, CLAMP>(__uint_as_float(g[8 * v + 2 * e]), bf16lo_to_f32(w4[e]), c, oe, acc,
                                             inv_k);
      grad_element_logistic<MU, SOFT, CLAMP>(__uint_as_float(g[8 * v + 2 * e + 1]), bf16hi_to_f32(w4[e]), c, oe,
                                             acc, inv_k);
    }
  }
}

}  // namespace catq
