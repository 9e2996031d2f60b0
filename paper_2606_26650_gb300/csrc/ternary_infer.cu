// ternary_infer.cu — inference with the deployed form of a calibrated layer (App. B.2: only
// the ternary codes T and the group scale alpha are kept, W ~ alpha T):
//   Y[b, n] = sum_k X[b, k] * alpha[n, k / g] * T[n, k]
// reading T from the 2-bit codes catq_hard_ternarize_pack writes.  Decode-shaped (a few
// token rows), so the bound is HBM: every weight costs 0.25 byte of codes plus its share of
// a 4-byte group scale.
//
// A warp computes R output rows at once (R = 4, 2 or 1 by the layer's height, so the GPU
// still gets enough warps).  A lane takes 64 consecutive columns (one 16-byte code load per
// row) at a time: it reads those 64 activations of a token row once and uses them for all R
// rows, which keeps the activation reads through L1 at 1/R per weight (they, not the codes,
// bound a one-row-per-warp kernel).  The 64 codes of a row lie in one group (g is a multiple
// of 64), so each row's chunk sum is scaled by alpha once.  Lane sums are added by a fixed
// shuffle tree, so results are deterministic.
//
// Decoding without conversions or per-element shifts: code i of a word (bits 2i, 2i+1, i < 8;
// the upper 8 codes come from word >> 16) masked in place and OR-ed into the bit pattern of
// 2^23 is the float 2^23 + c 4^i exactly; subtracting 2^23 + 4^i leaves (c - 1) 4^i = T 4^i,
// and multiplying by x 4^-i (the activation pre-scaled once per chunk by a power of two,
// exact for activations above ~1e-30) gives T x exactly.  Pairs of elements go through the
// packed fp32x2 add and fma.
//
// With the group offsets of the W ~ alpha T + mu reconstruction (MU), a row's chunk also adds
// mu times the chunk's activation sum, which is formed once per chunk for all R rows.
#include <cstdint>

#include "launch.h"

namespace catq {
namespace {

constexpr int kInferThreads = 256;

using f32x2 = unsigned long long;  // two fp32 lanes in one 64-bit register pair

__device__ __forceinline__ f32x2 pack2(uint32_t lo_bits, uint32_t hi_bits) {
  f32x2 r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "r"(lo_bits), "r"(hi_bits));
  return r;
}

__device__ __forceinline__ void unpack2(f32x2 v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}

__device__ __forceinline__ f32x2 add2(f32x2 a, f32x2 b) {
  f32x2 d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}

__device__ __forceinline__ f32x2 fma2(f32x2 a, f32x2 b, f32x2 c) {
  f32x2 d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}

// -(2^23 + 4^i) for codes i and i + 1 of a pair (i even, 0 <= i < 8)
__device__ __forceinline__ f32x2 neg_magic(int i) {
  return pack2(__float_as_uint(-(8388608.0f + static_cast<float>(1 << (2 * i)))),
               __float_as_uint(-(8388608.0f + static_cast<float>(1 << (2 * (i + 1))))));
}

// T 4^i for codes i and i + 1 of word w (i even, i < 8): exact small integers times 4^i.
__device__ __forceinline__ f32x2 codes_scaled(uint32_t w, int i) {
  return add2(pack2((w & (3u << (2 * i))) | 0x4B000000u, (w & (3u << (2 * (i + 1)))) | 0x4B000000u), neg_magic(i));
}

template <int R, bool MU>
__global__ void __launch_bounds__(kInferThreads) ternary_gemv_kernel(const uint8_t* __restrict__ codes,
                                                                     const float* __restrict__ alpha,
                                                                     const float* __restrict__ mu, int64_t N,
                                                                     int64_t K, int32_t g,
                                                                     const uint16_t* __restrict__ X, int64_t B,
                                                                     uint16_t* __restrict__ Y) {
  const int lane = threadIdx.x & 31;
  const int64_t warp = (static_cast<int64_t>(blockIdx.x) * kInferThreads + threadIdx.x) >> 5;
  const int64_t nwarps = static_cast<int64_t>(gridDim.x) * (kInferThreads / 32);
  const int64_t chunks = K / 64;
  const int64_t gpr = K / g;
  for (int64_t n0 = warp * R; n0 < N; n0 += nwarps * R) {
    // token rows one after the other: a warp re-reads its R rows' codes (a few KB, from
    // L1 / L2) per token row instead of holding every token row's sums in registers
    for (int64_t b = 0; b < B; ++b) {
      float acc[R];
#pragma unroll
      for (int r = 0; r < R; ++r) acc[r] = 0.0f;
      for (int64_t c = lane; c < chunks; c += 32) {
        uint4 w[R];
        float a[R], m[R];
#pragma unroll
        for (int r = 0; r < R; ++r) {
          const int64_t n = n0 + r < N ? n0 + r : N - 1;  // rows past N repeat the last (not stored)
          w[r] = __ldg(reinterpret_cast<const uint4*>(codes + n * (K / 4)) + c);
          a[r] = __ldg(alpha + n * gpr + (c * 64) / g);
          if constexpr (MU) m[r] = __ldg(mu + n * gpr + (c * 64) / g);
        }
        f32x2 p[R];
#pragma unroll
        for (int r = 0; r < R; ++r) p[r] = 0ull;
        f32x2 xsum = 0ull;  // activation sum of the chunk (MU only)
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const uint4* xp = reinterpret_cast<const uint4*>(X + b * K + c * 64 + q * 16);
          const uint4 h0 = __ldg(xp), h1 = __ldg(xp + 1);
          const uint32_t xw[8] = {h0.x, h0.y, h0.z, h0.w, h1.x, h1.y, h1.z, h1.w};
          // activation pairs (e, e + 1) of this word, pre-scaled by 4^-(e mod 8)
          f32x2 xs[8];
#pragma unroll
          for (int e2 = 0; e2 < 8; ++e2) {
            const int i = (2 * e2) & 7;
            const float s0 = __uint_as_float(static_cast<uint32_t>(127 - 2 * i) << 23);
            const float s1 = __uint_as_float(static_cast<uint32_t>(127 - 2 * (i + 1)) << 23);
            xs[e2] = pack2(__float_as_uint(bf16lo_to_f32(xw[e2]) * s0), __float_as_uint(bf16hi_to_f32(xw[e2]) * s1));
            if constexpr (MU)
              xsum = add2(xsum, pack2(__float_as_uint(bf16lo_to_f32(xw[e2])), __float_as_uint(bf16hi_to_f32(xw[e2]))));
          }
#pragma unroll
          for (int r = 0; r < R; ++r) {
            const uint32_t word = q == 0 ? w[r].x : q == 1 ? w[r].y : q == 2 ? w[r].z : w[r].w;
            const uint32_t hi = word >> 16;
#pragma unroll
            for (int e2 = 0; e2 < 8; ++e2) {
              const int i = (2 * e2) & 7;
              p[r] = fma2(codes_scaled(e2 < 4 ? word : hi, i), xs[e2], p[r]);
            }
          }
        }
        float xs_lo = 0.0f, xs_hi = 0.0f;
        if constexpr (MU) unpack2(xsum, xs_lo, xs_hi);
#pragma unroll
        for (int r = 0; r < R; ++r) {
          float lo, hi;
          unpack2(p[r], lo, hi);
          acc[r] = fmaf(a[r], lo + hi, acc[r]);
          if constexpr (MU) acc[r] = fmaf(m[r], xs_lo + xs_hi, acc[r]);
        }

      }
#pragma unroll
      for (int r = 0; r < R; ++r)
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) acc[r] += __shfl_xor_sync(0xffffffffu, acc[r], o);
      if (lane < R && n0 + lane < N) {
        float v = acc[0];
#pragma unroll
        for (int r = 1; r < R; ++r)
          if (lane == r) v = acc[r];
        Y[b * N + n0 + lane] = static_cast<uint16_t>(pack_bf16x2(v, 0.0f) & 0xFFFFu);
      }
    }
  }
}

template <int R>
cudaError_t launch_gemv(const uint8_t* codes, const float* alpha, const float* mu, int64_t N, int64_t K, int32_t g,
                        const uint16_t* X, int64_t B, uint16_t* Y, cudaStream_t st) {
  const int64_t warps = (N + R - 1) / R;
  int64_t blocks = (warps + kInferThreads / 32 - 1) / (kInferThreads / 32);
  if (blocks > 152 * 16) blocks = 152 * 16;
  if (mu)
    ternary_gemv_kernel<R, true><<<static_cast<int>(blocks), kInferThreads, 0, st>>>(codes, alpha, mu, N, K, g, X,
                                                                                    B, Y);
  else
    ternary_gemv_kernel<R, false><<<static_cast<int>(blocks), kInferThreads, 0, st>>>(codes, alpha, nullptr, N, K, g,
                                                                                     X, B, Y);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_ternary_infer(const uint8_t* codes, const float* alpha, const float* mu, int64_t N, int64_t K,
                                 int32_t g, const void* X, int64_t B, void* Y, cudaStream_t st) {
  const uint16_t* x = static_cast<const uint16_t*>(X);
  uint16_t* y = static_cast<uint16_t*>(Y);
  // Rows per warp by the layer's height: enough warps to fill the GPU, as few activation
  // reads per weight as that allows.
  if (N >= 8192) return launch_gemv<4>(codes, alpha, mu, N, K, g, x, B, y, st);
  if (N >= 2048) return launch_gemv<2>(codes, alpha, mu, N, K, g, x, B, y, st);
  return launch_gemv<1>(codes, alpha, mu, N, K, g, x, B, y, st);
}

}  // namespace catq
