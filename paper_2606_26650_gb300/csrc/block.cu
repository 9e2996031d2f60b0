// block.cu — the layers around the seven soft-ternary linears of one decoder block, for the
// block-output reconstruction step (§2.4, Eq. 7 over a window of one block): RMSNorm (with the
// residual add fused into the forward, and the residual and second upstream gradient fused
// into the backward; one CTA per long row, one warp per short row such as an attention head),
// rotary position embedding, SwiGLU, the fp32 block output with the loss on it, and causal
// grouped-query attention (forward, and a deterministic backward in two kernels).
//
// Attention with 128-wide heads over whole 128-token tiles runs on tcgen05 (attn_tc.cu); the
// kernels here serve the other shapes (d = 64, or S a multiple of 64 only) on the tensor pipe
// with mma.sync m16n8k16 (bf16 in, fp32 accumulate): blocks of 64 queries (four warps of 16) against blocks of 64 keys, which stream through two
// shared-memory buffers by cp.async; an online softmax in fp32 with the probabilities fed back
// as the A operand of P V straight from the score accumulators, and operand fragments read
// from shared memory with ldmatrix (transposed where the contraction runs along rows).  The
// backward recomputes the probabilities from the forward's log-sum-exp: one kernel per query
// block accumulates dQ; one per key block accumulates dK and dV (32 queries per step) over
// every query head that shares the key/value head, so no atomics are needed and the result is
// deterministic.
#include <cuda_bf16.h>

#include <algorithm>

#include "launch.h"
#include "ptx_sm100.cuh"

namespace catq {
namespace {

constexpr int kRowThreads = 256;

__device__ __forceinline__ float bf16_at(const uint16_t* p, int64_t i) { return __uint_as_float(uint32_t(p[i]) << 16); }
__device__ __forceinline__ uint16_t to_bf16(float v) { return static_cast<uint16_t>(pack_bf16x2(v, 0.0f) & 0xFFFFu); }

__device__ __forceinline__ float block_sum(float v, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) red[w] = v;
  __syncthreads();
  float t = 0.0f;
#pragma unroll
  for (int i = 0; i < kRowThreads / 32; ++i) t += red[i];
  return t;
}

// ---------------------------------------------------------------- RMSNorm
__device__ __forceinline__ float load_act(const uint16_t* p, int64_t i) { return bf16_at(p, i); }
__device__ __forceinline__ float load_act(const float* p, int64_t i) { return p[i]; }

// One CTA per token row: h = x (+ residual, in fp32, stored unrounded when h_out is given),
// r = 1 / sqrt(mean(h^2) + eps), z = gamma * h * r.
template <typename TX>
__global__ void __launch_bounds__(kRowThreads) rmsnorm_fwd_kernel(const TX* __restrict__ x,
                                                                   const uint16_t* __restrict__ res,
                                                                   const float* __restrict__ gamma, int64_t H,
                                                                   float eps, float* __restrict__ h_out,
                                                                   uint16_t* __restrict__ z, float* __restrict__ r) {
  __shared__ float red[kRowThreads / 32];
  const int64_t t = blockIdx.x;
  float ss = 0.0f;
  for (int64_t i = threadIdx.x; i < H; i += kRowThreads) {
    float h = load_act(x, t * H + i);
    if (res) h += bf16_at(res, t * H + i);
    if (h_out) h_out[t * H + i] = h;
    ss = fmaf(h, h, ss);
  }
  const float rr = rsqrtf(block_sum(ss, red) / static_cast<float>(H) + eps);
  if (threadIdx.x == 0) r[t] = rr;
  for (int64_t i = threadIdx.x; i < H; i += kRowThreads) {
    float h = load_act(x, t * H + i);
    if (res) h += bf16_at(res, t * H + i);
    z[t * H + i] = to_bf16(gamma[i] * h * rr);
  }
}

// dx = r u - h r^3 mean(u h) (+ dres), u = gamma (dy + dy2).
template <typename TH>
__global__ void __launch_bounds__(kRowThreads) rmsnorm_bwd_kernel(const TH* __restrict__ x,
                                                                   const float* __restrict__ gamma,
                                                                   const float* __restrict__ r, const uint16_t* dy,
                                                                   const uint16_t* dy2, const uint16_t* dres,
                                                                   int64_t H, uint16_t* dx) {  // dx may alias
  __shared__ float red[kRowThreads / 32];
  const int64_t t = blockIdx.x;
  const float rr = r[t];
  float sux = 0.0f;
  for (int64_t i = threadIdx.x; i < H; i += kRowThreads) {
    const float g = bf16_at(dy, t * H + i) + (dy2 ? bf16_at(dy2, t * H + i) : 0.0f);
    sux = fmaf(gamma[i] * g, load_act(x, t * H + i), sux);
  }
  const float c = block_sum(sux, red) / static_cast<float>(H) * rr * rr * rr;
  for (int64_t i = threadIdx.x; i < H; i += kRowThreads) {
    const float g = bf16_at(dy, t * H + i) + (dy2 ? bf16_at(dy2, t * H + i) : 0.0f);
    float v = rr * gamma[i] * g - load_act(x, t * H + i) * c;
    if (dres) v += bf16_at(dres, t * H + i);
    dx[t * H + i] = to_bf16(v);
  }
}

// Rows of at most 1024 elements (e.g. one attention head, the Qwen3 query/key norm): one warp
// per row, the same arithmetic as the kernels above.
constexpr int kRowWarps = kRowThreads / 32;

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

template <typename TX>
__global__ void __launch_bounds__(kRowThreads) rmsnorm_fwd_warp_kernel(const TX* __restrict__ x,
                                                                        const uint16_t* __restrict__ res,
                                                                        const float* __restrict__ gamma, int64_t T,
                                                                        int64_t H, float eps,
                                                                        float* __restrict__ h_out,
                                                                        uint16_t* __restrict__ z,
                                                                        float* __restrict__ r) {
  const int lane = threadIdx.x & 31;
  for (int64_t t = (blockIdx.x * (int64_t)kRowWarps) + (threadIdx.x >> 5); t < T; t += (int64_t)gridDim.x * kRowWarps) {
    float ss = 0.0f;
    for (int64_t i = lane; i < H; i += 32) {
      float h = load_act(x, t * H + i);
      if (res) h += bf16_at(res, t * H + i);
      if (h_out) h_out[t * H + i] = h;
      ss = fmaf(h, h, ss);
    }
    const float rr = rsqrtf(warp_sum(ss) / static_cast<float>(H) + eps);
    if (lane == 0) r[t] = rr;
    for (int64_t i = lane; i < H; i += 32) {
      float h = load_act(x, t * H + i);
      if (res) h += bf16_at(res, t * H + i);
      z[t * H + i] = to_bf16(gamma[i] * h * rr);
    }
  }
}

template <typename TH>
__global__ void __launch_bounds__(kRowThreads) rmsnorm_bwd_warp_kernel(const TH* __restrict__ x,
                                                                        const float* __restrict__ gamma,
                                                                        const float* __restrict__ r,
                                                                        const uint16_t* dy, const uint16_t* dy2,
                                                                        const uint16_t* dres, int64_t T, int64_t H,
                                                                        uint16_t* dx) {  // dx may alias
  const int lane = threadIdx.x & 31;
  for (int64_t t = (blockIdx.x * (int64_t)kRowWarps) + (threadIdx.x >> 5); t < T; t += (int64_t)gridDim.x * kRowWarps) {
    const float rr = r[t];
    float sux = 0.0f;
    for (int64_t i = lane; i < H; i += 32) {
      const float g = bf16_at(dy, t * H + i) + (dy2 ? bf16_at(dy2, t * H + i) : 0.0f);
      sux = fmaf(gamma[i] * g, load_act(x, t * H + i), sux);
    }
    const float c = warp_sum(sux) / static_cast<float>(H) * rr * rr * rr;
    for (int64_t i = lane; i < H; i += 32) {
      const float g = bf16_at(dy, t * H + i) + (dy2 ? bf16_at(dy2, t * H + i) : 0.0f);
      float v = rr * gamma[i] * g - load_act(x, t * H + i) * c;
      if (dres) v += bf16_at(dres, t * H + i);
      dx[t * H + i] = to_bf16(v);
    }
  }
}

// ---------------------------------------------------------------- rotary embedding
// Element pair (i, i + d/2) of every head of token t (position s = t mod S) rotated by the
// angle s base^(-2i/d) (its negative for the inverse), in place.
__global__ void __launch_bounds__(kRowThreads) rope_kernel(uint16_t* __restrict__ x, int64_t T, int64_t S,
                                                            int32_t nheads, int32_t d, float log2_base,
                                                            int32_t inverse) {
  const int32_t half = d / 2;
  const int64_t pairs = T * nheads * half;
  for (int64_t e = blockIdx.x * (int64_t)kRowThreads + threadIdx.x; e < pairs; e += (int64_t)gridDim.x * kRowThreads) {
    const int32_t i = static_cast<int32_t>(e % half);
    const int64_t th = e / half;  // token * nheads + head
    const int64_t t = th / nheads;
    const float inv_freq = exp2f(-log2_base * (2.0f * i) / static_cast<float>(d));
    float sn, cs;
    sincosf(static_cast<float>(t % S) * inv_freq, &sn, &cs);
    if (inverse) sn = -sn;
    uint16_t* p = x + th * d;
    const float a = bf16_at(p, i), b = bf16_at(p, i + half);
    p[i] = to_bf16(a * cs - b * sn);
    p[i + half] = to_bf16(a * sn + b * cs);
  }
}

// Rows of 8 consecutive elements of d = 16 k (half = 8 k) heads: one thread per (token, 8
// consecutive i), its 8 angles computed once and applied to every head of the token with
// 16-byte loads and stores.
__global__ void __launch_bounds__(kRowThreads) rope_vec_kernel(uint16_t* __restrict__ x, int64_t T, int64_t S,
                                                                int32_t nheads, int32_t d, float log2_base,
                                                                int32_t inverse) {
  const int32_t half = d / 2, groups = half / 8;
  const int64_t items = T * groups;
  for (int64_t e = blockIdx.x * (int64_t)kRowThreads + threadIdx.x; e < items; e += (int64_t)gridDim.x * kRowThreads) {
    const int32_t i0 = static_cast<int32_t>(e % groups) * 8;
    const int64_t t = e / groups;
    const float pos = static_cast<float>(t % S);
    float cs[8], sn[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const float inv_freq = exp2f(-log2_base * (2.0f * (i0 + j)) / static_cast<float>(d));
      sincosf(pos * inv_freq, &sn[j], &cs[j]);
      if (inverse) sn[j] = -sn[j];
    }
    for (int32_t h = 0; h < nheads; ++h) {
      uint16_t* p = x + (t * nheads + h) * d;
      const uint4 av = *reinterpret_cast<const uint4*>(p + i0), bv = *reinterpret_cast<const uint4*>(p + i0 + half);
      const uint32_t aw[4] = {av.x, av.y, av.z, av.w}, bw[4] = {bv.x, bv.y, bv.z, bv.w};
      uint32_t ow[4], qw[4];
#pragma unroll
      for (int w = 0; w < 4; ++w) {
        const float a0 = bf16lo_to_f32(aw[w]), a1 = bf16hi_to_f32(aw[w]);
        const float b0 = bf16lo_to_f32(bw[w]), b1 = bf16hi_to_f32(bw[w]);
        const int j = 2 * w;
        ow[w] = pack_bf16x2(a0 * cs[j] - b0 * sn[j], a1 * cs[j + 1] - b1 * sn[j + 1]);
        qw[w] = pack_bf16x2(a0 * sn[j] + b0 * cs[j], a1 * sn[j + 1] + b1 * cs[j + 1]);
      }
      *reinterpret_cast<uint4*>(p + i0) = make_uint4(ow[0], ow[1], ow[2], ow[3]);
      *reinterpret_cast<uint4*>(p + i0 + half) = make_uint4(qw[0], qw[1], qw[2], qw[3]);
    }
  }
}

// ---------------------------------------------------------------- SwiGLU
// Eight elements per thread and iteration (16-byte loads and stores); block 0 takes the tail.
__device__ __forceinline__ float sigmoidf(float a) { return 1.0f / (1.0f + expf(-a)); }

__device__ __forceinline__ void unpack8(const uint4& v, float (&f)[8]) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    f[2 * i] = bf16lo_to_f32(w[i]);
    f[2 * i + 1] = bf16hi_to_f32(w[i]);
  }
}

__device__ __forceinline__ uint4 pack8(const float (&f)[8]) {
  return make_uint4(pack_bf16x2(f[0], f[1]), pack_bf16x2(f[2], f[3]), pack_bf16x2(f[4], f[5]),
                    pack_bf16x2(f[6], f[7]));
}

__global__ void __launch_bounds__(kRowThreads) swiglu_fwd_kernel(const uint16_t* __restrict__ gt,
                                                                  const uint16_t* __restrict__ u, int64_t n,
                                                                  uint16_t* __restrict__ m) {
  const int64_t nvec = n / 8;
  for (int64_t e = blockIdx.x * (int64_t)kRowThreads + threadIdx.x; e < nvec; e += (int64_t)gridDim.x * kRowThreads) {
    float a[8], b[8], o[8];
    unpack8(reinterpret_cast<const uint4*>(gt)[e], a);
    unpack8(reinterpret_cast<const uint4*>(u)[e], b);
#pragma unroll
    for (int i = 0; i < 8; ++i) o[i] = a[i] * sigmoidf(a[i]) * b[i];
    reinterpret_cast<uint4*>(m)[e] = pack8(o);
  }
  if (blockIdx.x == 0)
    for (int64_t e = nvec * 8 + threadIdx.x; e < n; e += kRowThreads) {
      const float a = bf16_at(gt, e);
      m[e] = to_bf16(a * sigmoidf(a) * bf16_at(u, e));
    }
}

// d_gate = dm u sigma(a) (1 + a (1 - sigma(a))), d_up = dm a sigma(a).
__device__ __forceinline__ void swiglu_grad(float a, float b, float g, float& dg, float& du) {
  const float s = sigmoidf(a);
  dg = g * b * s * (1.0f + a * (1.0f - s));
  du = g * a * s;
}

__global__ void __launch_bounds__(kRowThreads) swiglu_bwd_kernel(const uint16_t* __restrict__ gt,
                                                                  const uint16_t* __restrict__ u,
                                                                  const uint16_t* __restrict__ dm, int64_t n,
                                                                  uint16_t* __restrict__ dgt,
                                                                  uint16_t* __restrict__ du) {
  const int64_t nvec = n / 8;
  for (int64_t e = blockIdx.x * (int64_t)kRowThreads + threadIdx.x; e < nvec; e += (int64_t)gridDim.x * kRowThreads) {
    float a[8], b[8], g[8], dg[8], dd[8];
    unpack8(reinterpret_cast<const uint4*>(gt)[e], a);
    unpack8(reinterpret_cast<const uint4*>(u)[e], b);
    unpack8(reinterpret_cast<const uint4*>(dm)[e], g);
#pragma unroll
    for (int i = 0; i < 8; ++i) swiglu_grad(a[i], b[i], g[i], dg[i], dd[i]);
    reinterpret_cast<uint4*>(dgt)[e] = pack8(dg);
    reinterpret_cast<uint4*>(du)[e] = pack8(dd);
  }
  if (blockIdx.x == 0)
    for (int64_t e = nvec * 8 + threadIdx.x; e < n; e += kRowThreads) {
      float dg, dd;
      swiglu_grad(bf16_at(gt, e), bf16_at(u, e), bf16_at(dm, e), dg, dd);
      dgt[e] = to_bf16(dg);
      du[e] = to_bf16(dd);
    }
}

// Block output in fp32, out = h + branch, and (with a teacher output) Eq. 7's loss: partial
// sums of (out - ref)^2 per CTA (compensated fp32, then fp64) and d_out = scale (out - ref)
// rounded once to bf16.  Eight elements per thread and iteration (count % 8 == 0).
__global__ void __launch_bounds__(kRowThreads) block_output_loss_kernel(const float* __restrict__ h,
                                                                         const uint16_t* __restrict__ branch,
                                                                         const float* __restrict__ ref, int64_t count,
                                                                         float scale, float* __restrict__ out,
                                                                         uint16_t* __restrict__ d_out,
                                                                         double* __restrict__ partials) {
  Sum2 acc{0.f, 0.f};
  const int64_t nvec = count / 8;
  for (int64_t i = blockIdx.x * (int64_t)kRowThreads + threadIdx.x; i < nvec; i += (int64_t)gridDim.x * kRowThreads) {
    const float4 h0 = reinterpret_cast<const float4*>(h)[2 * i], h1 = reinterpret_cast<const float4*>(h)[2 * i + 1];
    const uint4 bw = reinterpret_cast<const uint4*>(branch)[i];
    float o[8] = {h0.x + bf16lo_to_f32(bw.x), h0.y + bf16hi_to_f32(bw.x), h0.z + bf16lo_to_f32(bw.y),
                  h0.w + bf16hi_to_f32(bw.y), h1.x + bf16lo_to_f32(bw.z), h1.y + bf16hi_to_f32(bw.z),
                  h1.z + bf16lo_to_f32(bw.w), h1.w + bf16hi_to_f32(bw.w)};
    if (out) {
      reinterpret_cast<float4*>(out)[2 * i] = make_float4(o[0], o[1], o[2], o[3]);
      reinterpret_cast<float4*>(out)[2 * i + 1] = make_float4(o[4], o[5], o[6], o[7]);
    }
    if (ref) {
      const float4 r0 = reinterpret_cast<const float4*>(ref)[2 * i], r1 = reinterpret_cast<const float4*>(ref)[2 * i + 1];
      const float rv[8] = {r0.x, r0.y, r0.z, r0.w, r1.x, r1.y, r1.z, r1.w};
      Sum2 local{0.f, 0.f};
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        o[q] -= rv[q];
        sum2_add(local, o[q] * o[q]);
      }
      acc = sum2_merge(acc, local);
      if (d_out) {
        uint4 w;
        w.x = pack_bf16x2(o[0] * scale, o[1] * scale);
        w.y = pack_bf16x2(o[2] * scale, o[3] * scale);
        w.z = pack_bf16x2(o[4] * scale, o[5] * scale);
        w.w = pack_bf16x2(o[6] * scale, o[7] * scale);
        reinterpret_cast<uint4*>(d_out)[i] = w;
      }
    }
  }
  if (!ref) return;
  __shared__ Sum2 red[kRowThreads / 32];
  acc = sum2_team(acc, 32);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x < 32) {
    Sum2 v = threadIdx.x < kRowThreads / 32 ? red[threadIdx.x] : Sum2{0.f, 0.f};
    v = sum2_team(v, 32);
    if (threadIdx.x == 0) partials[blockIdx.x] = sum2_value(v);
  }
}

// ---------------------------------------------------------------- attention
constexpr int kBlk = 64;          // queries / keys per block
constexpr int kAttnThreads = 128; // four warps of 16 rows

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                               uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// A shared-memory tile of 64 rows x HD bf16, rows padded by 16 bytes (conflict-free ldmatrix).
template <int HD>
struct Tile {
  static constexpr int kStride = HD + 8;  // elements per row
  static constexpr int kBytes = kBlk * kStride * 2;
};

// Rows row0.. row0 + 63 of a [rows, ld] bf16 matrix, columns col0 .. col0 + HD - 1, into a tile.
template <int HD>
__device__ __forceinline__ void load_tile(uint16_t* tile, const uint16_t* src, int64_t row0, int64_t ld,
                                          int64_t col0) {
  constexpr int kChunks = kBlk * HD / 8;  // 16-byte chunks
  for (int c = threadIdx.x; c < kChunks; c += kAttnThreads) {
    const int r = c / (HD / 8), k = (c % (HD / 8)) * 8;
    *reinterpret_cast<uint4*>(tile + r * Tile<HD>::kStride + k) =
        *reinterpret_cast<const uint4*>(src + (row0 + r) * ld + col0 + k);
  }
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async4(uint32_t dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// load_tile through cp.async (16-byte copies that complete with the thread's next wait).
template <int HD>
__device__ __forceinline__ void load_tile_async(uint32_t tile, const uint16_t* src, int64_t row0, int64_t ld,
                                                int64_t col0) {
  constexpr int kChunks = kBlk * HD / 8;
  for (int c = threadIdx.x; c < kChunks; c += kAttnThreads) {
    const int r = c / (HD / 8), k = (c % (HD / 8)) * 8;
    cp_async16(tile + static_cast<uint32_t>((r * Tile<HD>::kStride + k) * 2), src + (row0 + r) * ld + col0 + k);
  }
}

// Address of the row that this lane supplies to an ldmatrix.x4 of a 16 x 16 fragment at
// (row0, col0) of a tile: matrix m = lane / 8 covers rows + (m & 1) 8 when `row_from_bit0`
// (A operands and transposed B operands), else + (m >> 1) 8 (B operands stored n-major), and
// columns + the other bit times 8.
template <int HD>
__device__ __forceinline__ uint32_t frag_addr(uint32_t tile, int row0, int col0, bool row_from_bit0) {
  const int lane = threadIdx.x & 31, m = lane >> 3, r = lane & 7;
  const int dr = row_from_bit0 ? (m & 1) * 8 : (m >> 1) * 8;
  const int dc = row_from_bit0 ? (m >> 1) * 8 : (m & 1) * 8;
  return tile + static_cast<uint32_t>(((row0 + dr + r) * Tile<HD>::kStride + col0 + dc) * 2);
}

// Scores of this warp's 16 rows of A (tile rows a_row0..) against the 64 rows of B (an
// n-major tile of keys), over HD columns: acc[n-tile 0..7][4].
template <int HD>
__device__ __forceinline__ void scores_16x64(float (&acc)[8][4], uint32_t a_tile, int a_row0, uint32_t b_tile) {
#pragma unroll
  for (int nt = 0; nt < 8; ++nt)
#pragma unroll
    for (int e = 0; e < 4; ++e) acc[nt][e] = 0.0f;
#pragma unroll
  for (int kk = 0; kk < HD / 16; ++kk) {
    uint32_t a0, a1, a2, a3;
    ldsm_x4(frag_addr<HD>(a_tile, a_row0, kk * 16, true), a0, a1, a2, a3);
#pragma unroll
    for (int p = 0; p < 4; ++p) {
      uint32_t b0, b1, b2, b3;
      ldsm_x4(frag_addr<HD>(b_tile, p * 16, kk * 16, false), b0, b1, b2, b3);
      mma_bf16_16816(acc[2 * p], a0, a1, a2, a3, b0, b1);
      mma_bf16_16816(acc[2 * p + 1], a0, a1, a2, a3, b2, b3);
    }
  }
}

// acc[d-tile 0 .. HD/8)[4] += P (16 x 64, as bf16 A fragments from fp32 values p[n-tile][4])
// times the 64 x HD tile (rows = the contraction), read transposed.
template <int HD>
__device__ __forceinline__ void accum_pv(float (&acc)[HD / 8][4], const float (&p)[8][4], uint32_t v_tile) {
#pragma unroll
  for (int ks = 0; ks < 4; ++ks) {
    const uint32_t a0 = pack_bf16x2(p[2 * ks][0], p[2 * ks][1]);
    const uint32_t a1 = pack_bf16x2(p[2 * ks][2], p[2 * ks][3]);
    const uint32_t a2 = pack_bf16x2(p[2 * ks + 1][0], p[2 * ks + 1][1]);
    const uint32_t a3 = pack_bf16x2(p[2 * ks + 1][2], p[2 * ks + 1][3]);
#pragma unroll
    for (int dp = 0; dp < HD / 16; ++dp) {
      uint32_t b0, b1, b2, b3;
      ldsm_x4_t(frag_addr<HD>(v_tile, ks * 16, dp * 16, true), b0, b1, b2, b3);
      mma_bf16_16816(acc[2 * dp], a0, a1, a2, a3, b0, b1);
      mma_bf16_16816(acc[2 * dp + 1], a0, a1, a2, a3, b2, b3);
    }
  }
}

struct AttnArgs {
  const uint16_t *q, *k, *v, *o, *dO;
  uint16_t *out, *dq, *dk, *dv;
  float *lse, *delta;
  int32_t B, S, nh, nkv;
  float scale_log2;  // log2(e) / sqrt(d)
  float scale;       // 1 / sqrt(d)
};

// Forward: one CTA per (query block, head, sequence).  Rows g and g + 8 of the warp's 16 are
// the thread's (lane / 4); its columns within each 8-wide n-tile are 2 (lane % 4) + {0, 1}.
// Key/value blocks stream through two shared-memory buffers: block kb + 1's copies are in
// flight while block kb is computed.
template <int HD>
__global__ void __launch_bounds__(kAttnThreads) attn_fwd_kernel(const AttnArgs a) {
  extern __shared__ __align__(16) uint8_t smem[];
  uint16_t* Qs = reinterpret_cast<uint16_t*>(smem);
  const uint32_t qa = smem_u32(Qs);
  const uint32_t kv0 = qa + Tile<HD>::kBytes;  // buffer b: K at kv0 + 2 b tile, V after it
  const int nqb = a.S / kBlk;
  const int qb = nqb - 1 - static_cast<int>(blockIdx.x);  // the longest rows first
  const int h = blockIdx.y, b = blockIdx.z, hk = h / (a.nh / a.nkv);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, t4 = lane & 3;
  const int64_t tok0 = static_cast<int64_t>(b) * a.S;
  const int64_t ldq = static_cast<int64_t>(a.nh) * HD, ldk = static_cast<int64_t>(a.nkv) * HD;
  auto load_kv = [&](int kb) {
    const uint32_t kt = kv0 + static_cast<uint32_t>((kb & 1) * 2 * Tile<HD>::kBytes);
    load_tile_async<HD>(kt, a.k, tok0 + kb * kBlk, ldk, static_cast<int64_t>(hk) * HD);
    load_tile_async<HD>(kt + Tile<HD>::kBytes, a.v, tok0 + kb * kBlk, ldk, static_cast<int64_t>(hk) * HD);
  };
  load_tile_async<HD>(qa, a.q, tok0 + qb * kBlk, ldq, static_cast<int64_t>(h) * HD);
  load_kv(0);
  cp_async_commit();
  float o[HD / 8][4];
#pragma unroll
  for (int i = 0; i < HD / 8; ++i)
#pragma unroll
    for (int e = 0; e < 4; ++e) o[i][e] = 0.0f;
  float mrow[2] = {-INFINITY, -INFINITY}, lrow[2] = {0.0f, 0.0f};
  for (int kb = 0; kb <= qb; ++kb) {
    if (kb < qb) {
      load_kv(kb + 1);
      cp_async_commit();
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    const uint32_t ka = kv0 + static_cast<uint32_t>((kb & 1) * 2 * Tile<HD>::kBytes), va = ka + Tile<HD>::kBytes;
    float s[8][4];
    scores_16x64<HD>(s, qa, warp * 16, ka);
    float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
    for (int nt = 0; nt < 8; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        float v = s[nt][e] * a.scale_log2;
        if (kb == qb) {
          const int key = nt * 8 + 2 * t4 + (e & 1), qry = warp * 16 + g + (e >> 1) * 8;
          if (key > qry) v = -INFINITY;
        }
        s[nt][e] = v;
        mx[e >> 1] = fmaxf(mx[e >> 1], v);
      }
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      mx[i] = fmaxf(mx[i], __shfl_xor_sync(0xffffffffu, mx[i], 1));
      mx[i] = fmaxf(mx[i], __shfl_xor_sync(0xffffffffu, mx[i], 2));
    }
    float corr[2], ls[2] = {0.0f, 0.0f};
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const float mn = fmaxf(mrow[i], mx[i]);
      corr[i] = mrow[i] == -INFINITY ? 0.0f : exp2f(mrow[i] - mn);
      mrow[i] = mn;
    }
#pragma unroll
    for (int nt = 0; nt < 8; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float p = exp2f(s[nt][e] - mrow[e >> 1]);
        s[nt][e] = p;
        ls[e >> 1] += p;
      }
#pragma unroll
    for (int i = 0; i < 2; ++i) lrow[i] = lrow[i] * corr[i] + ls[i];
#pragma unroll
    for (int dn = 0; dn < HD / 8; ++dn) {
      o[dn][0] *= corr[0];
      o[dn][1] *= corr[0];
      o[dn][2] *= corr[1];
      o[dn][3] *= corr[1];
    }
    accum_pv<HD>(o, s, va);
    __syncthreads();  // buffer kb & 1 is refilled with block kb + 2 next
  }
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    lrow[i] += __shfl_xor_sync(0xffffffffu, lrow[i], 1);
    lrow[i] += __shfl_xor_sync(0xffffffffu, lrow[i], 2);
  }
  const float inv[2] = {1.0f / lrow[0], 1.0f / lrow[1]};
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int64_t tok = tok0 + qb * kBlk + warp * 16 + g + 8 * i;
    uint16_t* orow = a.out + tok * ldq + static_cast<int64_t>(h) * HD;
#pragma unroll
    for (int dn = 0; dn < HD / 8; ++dn)
      *reinterpret_cast<uint32_t*>(orow + dn * 8 + 2 * t4) = pack_bf16x2(o[dn][2 * i] * inv[i], o[dn][2 * i + 1] * inv[i]);
    if (t4 == 0)  // natural log-sum-exp of the scaled scores
      a.lse[(static_cast<int64_t>(b) * a.nh + h) * a.S + qb * kBlk + warp * 16 + g + 8 * i] =
          (mrow[i] + log2f(lrow[i])) * 0.69314718055994531f;
  }
}

// delta[b, h, s] = sum over the head's columns of dO * O (one warp per token and head).
template <int HD>
__global__ void __launch_bounds__(kRowThreads) attn_delta_kernel(const AttnArgs a) {
  const int64_t rows = static_cast<int64_t>(a.B) * a.S * a.nh;
  const int lane = threadIdx.x & 31;
  for (int64_t w = (blockIdx.x * (int64_t)kRowThreads + threadIdx.x) >> 5; w < rows;
       w += ((int64_t)gridDim.x * kRowThreads) >> 5) {
    const int64_t tok = w / a.nh;
    const int h = static_cast<int>(w % a.nh);
    const uint16_t* o = a.o + tok * a.nh * HD + static_cast<int64_t>(h) * HD;
    const uint16_t* d = a.dO + tok * a.nh * HD + static_cast<int64_t>(h) * HD;
    float s = 0.0f;
    for (int i = lane; i < HD; i += 32) s = fmaf(bf16_at(o, i), bf16_at(d, i), s);
#pragma unroll
    for (int o2 = 16; o2 > 0; o2 >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o2);
    if (lane == 0) {
      const int64_t b = tok / a.S, sidx = tok % a.S;
      a.delta[(b * a.nh + h) * a.S + sidx] = s;
    }
  }
}

// dQ: one CTA per (query block, head, sequence), over the key blocks up to the diagonal,
// which stream through two buffers as in the forward.
template <int HD>
__global__ void __launch_bounds__(kAttnThreads) attn_bwd_dq_kernel(const AttnArgs a) {
  extern __shared__ __align__(16) uint8_t smem[];
  const uint32_t qa = smem_u32(smem), da = qa + Tile<HD>::kBytes;  // Q, dO
  const uint32_t kv0 = da + Tile<HD>::kBytes;                       // buffer b: K, V at kv0 + 2 b tile
  const int nqb = a.S / kBlk;
  const int qb = nqb - 1 - static_cast<int>(blockIdx.x);
  const int h = blockIdx.y, b = blockIdx.z, hk = h / (a.nh / a.nkv);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, t4 = lane & 3;
  const int64_t tok0 = static_cast<int64_t>(b) * a.S;
  const int64_t ldq = static_cast<int64_t>(a.nh) * HD, ldk = static_cast<int64_t>(a.nkv) * HD;
  auto load_kv = [&](int kb) {
    const uint32_t kt = kv0 + static_cast<uint32_t>((kb & 1) * 2 * Tile<HD>::kBytes);
    load_tile_async<HD>(kt, a.k, tok0 + kb * kBlk, ldk, static_cast<int64_t>(hk) * HD);
    load_tile_async<HD>(kt + Tile<HD>::kBytes, a.v, tok0 + kb * kBlk, ldk, static_cast<int64_t>(hk) * HD);
  };
  load_tile_async<HD>(qa, a.q, tok0 + qb * kBlk, ldq, static_cast<int64_t>(h) * HD);
  load_tile_async<HD>(da, a.dO, tok0 + qb * kBlk, ldq, static_cast<int64_t>(h) * HD);
  load_kv(0);
  cp_async_commit();
  float lse2[2], dl[2];  // this thread's two rows: log-sum-exp in log2 units, and delta
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int64_t idx = (static_cast<int64_t>(b) * a.nh + h) * a.S + qb * kBlk + warp * 16 + g + 8 * i;
    lse2[i] = a.lse[idx] * 1.4426950408889634f;
    dl[i] = a.delta[idx];
  }
  float dq[HD / 8][4];
#pragma unroll
  for (int i = 0; i < HD / 8; ++i)
#pragma unroll
    for (int e = 0; e < 4; ++e) dq[i][e] = 0.0f;
  for (int kb = 0; kb <= qb; ++kb) {
    if (kb < qb) {
      load_kv(kb + 1);
      cp_async_commit();
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    const uint32_t ka = kv0 + static_cast<uint32_t>((kb & 1) * 2 * Tile<HD>::kBytes), va = ka + Tile<HD>::kBytes;
    float s[8][4], dp[8][4];
    scores_16x64<HD>(s, qa, warp * 16, ka);   // Q K^T
    scores_16x64<HD>(dp, da, warp * 16, va);  // dO V^T
#pragma unroll
    for (int nt = 0; nt < 8; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        float p = exp2f(s[nt][e] * a.scale_log2 - lse2[e >> 1]);
        if (kb == qb) {
          const int key = nt * 8 + 2 * t4 + (e & 1), qry = warp * 16 + g + (e >> 1) * 8;
          if (key > qry) p = 0.0f;
        }
        s[nt][e] = p * (dp[nt][e] - dl[e >> 1]);  // dS
      }
    accum_pv<HD>(dq, s, ka);  // dS K
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int64_t tok = tok0 + qb * kBlk + warp * 16 + g + 8 * i;
    uint16_t* row = a.dq + tok * ldq + static_cast<int64_t>(h) * HD;
#pragma unroll
    for (int dn = 0; dn < HD / 8; ++dn)
      *reinterpret_cast<uint32_t*>(row + dn * 8 + 2 * t4) = pack_bf16x2(dq[dn][2 * i] * a.scale, dq[dn][2 * i + 1] * a.scale);
  }
}

// dK, dV: one CTA per (key block, key/value head, sequence), over every query head of the
// group and the query blocks from the diagonal on (one stream of (head, query block) pairs
// through two buffers of Q, dO and their rows' log-sum-exp and delta), 32 queries at a time.
// Scores are formed transposed (keys as rows) so that P^T and dS^T feed the A operand from
// registers.
template <int HD>
__global__ void __launch_bounds__(kAttnThreads) attn_bwd_dkdv_kernel(const AttnArgs a) {
  extern __shared__ __align__(16) uint8_t smem[];
  const uint32_t ka = smem_u32(smem), va = ka + Tile<HD>::kBytes;
  const uint32_t qd0 = va + Tile<HD>::kBytes;  // buffer b: Q at qd0 + 2 b tile, dO after it
  float* const lsd0 = reinterpret_cast<float*>(smem + 6 * Tile<HD>::kBytes);  // buffer b: lse [64], delta [64]
  const int nqb = a.S / kBlk;
  const int kb = static_cast<int>(blockIdx.x);  // the most query blocks first
  const int hk = blockIdx.y, b = blockIdx.z, rep = a.nh / a.nkv;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, t4 = lane & 3;
  const int64_t tok0 = static_cast<int64_t>(b) * a.S;
  const int64_t ldq = static_cast<int64_t>(a.nh) * HD, ldk = static_cast<int64_t>(a.nkv) * HD;
  const int per_head = nqb - kb, n_it = rep * per_head;  // (head, query block) pairs
  auto load_q = [&](int it) {
    const int h = hk * rep + it / per_head, qb = kb + it % per_head;
    const uint32_t qt = qd0 + static_cast<uint32_t>((it & 1) * 2 * Tile<HD>::kBytes);
    load_tile_async<HD>(qt, a.q, tok0 + qb * kBlk, ldq, static_cast<int64_t>(h) * HD);
    load_tile_async<HD>(qt + Tile<HD>::kBytes, a.dO, tok0 + qb * kBlk, ldq, static_cast<int64_t>(h) * HD);
    if (threadIdx.x < kBlk) {
      const int64_t idx = (static_cast<int64_t>(b) * a.nh + h) * a.S + qb * kBlk + threadIdx.x;
      float* l = lsd0 + (it & 1) * 2 * kBlk;
      cp_async4(smem_u32(l + threadIdx.x), a.lse + idx);
      cp_async4(smem_u32(l + kBlk + threadIdx.x), a.delta + idx);
    }
  };
  load_tile_async<HD>(ka, a.k, tok0 + kb * kBlk, ldk, static_cast<int64_t>(hk) * HD);
  load_tile_async<HD>(va, a.v, tok0 + kb * kBlk, ldk, static_cast<int64_t>(hk) * HD);
  load_q(0);
  cp_async_commit();
  float dk[HD / 8][4], dv[HD / 8][4];
#pragma unroll
  for (int i = 0; i < HD / 8; ++i)
#pragma unroll
    for (int e = 0; e < 4; ++e) dk[i][e] = dv[i][e] = 0.0f;
  for (int it = 0; it < n_it; ++it) {
    if (it + 1 < n_it) {
      load_q(it + 1);
      cp_async_commit();
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    const int qb = kb + it % per_head;
    const uint32_t qa = qd0 + static_cast<uint32_t>((it & 1) * 2 * Tile<HD>::kBytes), da = qa + Tile<HD>::kBytes;
    const float* lse_s = lsd0 + (it & 1) * 2 * kBlk;
    const float* dl_s = lse_s + kBlk;
#pragma unroll 1
    for (int qs = 0; qs < kBlk / 32; ++qs) {
      // S^T and dP^T of the warp's 16 keys against 32 queries: four n-tiles each
      float st[4][4], dpt[4][4];
#pragma unroll
      for (int nt = 0; nt < 4; ++nt)
#pragma unroll
        for (int e = 0; e < 4; ++e) st[nt][e] = dpt[nt][e] = 0.0f;
#pragma unroll
      for (int kk = 0; kk < HD / 16; ++kk) {
        uint32_t a0, a1, a2, a3, b0, b1, b2, b3;
        ldsm_x4(frag_addr<HD>(ka, warp * 16, kk * 16, true), a0, a1, a2, a3);
#pragma unroll
        for (int hq = 0; hq < 2; ++hq) {
          ldsm_x4(frag_addr<HD>(qa, qs * 32 + hq * 16, kk * 16, false), b0, b1, b2, b3);
          mma_bf16_16816(st[2 * hq], a0, a1, a2, a3, b0, b1);
          mma_bf16_16816(st[2 * hq + 1], a0, a1, a2, a3, b2, b3);
        }
        ldsm_x4(frag_addr<HD>(va, warp * 16, kk * 16, true), a0, a1, a2, a3);
#pragma unroll
        for (int hq = 0; hq < 2; ++hq) {
          ldsm_x4(frag_addr<HD>(da, qs * 32 + hq * 16, kk * 16, false), b0, b1, b2, b3);
          mma_bf16_16816(dpt[2 * hq], a0, a1, a2, a3, b0, b1);
          mma_bf16_16816(dpt[2 * hq + 1], a0, a1, a2, a3, b2, b3);
        }
      }
      uint32_t pk[2][4], sk[2][4];  // P^T and dS^T as bf16 A fragments, one per 16 queries
#pragma unroll
      for (int hq = 0; hq < 2; ++hq) {
        float pt[2][4], dst[2][4];
#pragma unroll
        for (int j = 0; j < 2; ++j)
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const int nt = 2 * hq + j;
            const int qry = qs * 32 + nt * 8 + 2 * t4 + (e & 1);  // within the query block
            const int key = warp * 16 + g + (e >> 1) * 8;          // within the key block
            float p = exp2f((st[nt][e] * a.scale - lse_s[qry]) * 1.4426950408889634f);
            if (qb == kb && key > qry) p = 0.0f;
            pt[j][e] = p;
            dst[j][e] = p * (dpt[nt][e] - dl_s[qry]);
          }
        pk[hq][0] = pack_bf16x2(pt[0][0], pt[0][1]);
        pk[hq][1] = pack_bf16x2(pt[0][2], pt[0][3]);
        pk[hq][2] = pack_bf16x2(pt[1][0], pt[1][1]);
        pk[hq][3] = pack_bf16x2(pt[1][2], pt[1][3]);
        sk[hq][0] = pack_bf16x2(dst[0][0], dst[0][1]);
        sk[hq][1] = pack_bf16x2(dst[0][2], dst[0][3]);
        sk[hq][2] = pack_bf16x2(dst[1][0], dst[1][1]);
        sk[hq][3] = pack_bf16x2(dst[1][2], dst[1][3]);
      }
      // dV += P^T dO and dK += dS^T Q over these 32 queries (two k-steps)
#pragma unroll
      for (int hq = 0; hq < 2; ++hq)
#pragma unroll
        for (int dp = 0; dp < HD / 16; ++dp) {
          uint32_t b0, b1, b2, b3;
          ldsm_x4_t(frag_addr<HD>(da, qs * 32 + hq * 16, dp * 16, true), b0, b1, b2, b3);
          mma_bf16_16816(dv[2 * dp], pk[hq][0], pk[hq][1], pk[hq][2], pk[hq][3], b0, b1);
          mma_bf16_16816(dv[2 * dp + 1], pk[hq][0], pk[hq][1], pk[hq][2], pk[hq][3], b2, b3);
          ldsm_x4_t(frag_addr<HD>(qa, qs * 32 + hq * 16, dp * 16, true), b0, b1, b2, b3);
          mma_bf16_16816(dk[2 * dp], sk[hq][0], sk[hq][1], sk[hq][2], sk[hq][3], b0, b1);
          mma_bf16_16816(dk[2 * dp + 1], sk[hq][0], sk[hq][1], sk[hq][2], sk[hq][3], b2, b3);
        }
    }
    __syncthreads();  // buffer it & 1 is refilled with pair it + 2 next
  }
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int64_t tok = tok0 + kb * kBlk + warp * 16 + g + 8 * i;
    uint16_t* krow = a.dk + tok * ldk + static_cast<int64_t>(hk) * HD;
    uint16_t* vrow = a.dv + tok * ldk + static_cast<int64_t>(hk) * HD;
#pragma unroll
    for (int dn = 0; dn < HD / 8; ++dn) {
      *reinterpret_cast<uint32_t*>(krow + dn * 8 + 2 * t4) = pack_bf16x2(dk[dn][2 * i] * a.scale, dk[dn][2 * i + 1] * a.scale);
      *reinterpret_cast<uint32_t*>(vrow + dn * 8 + 2 * t4) = pack_bf16x2(dv[dn][2 * i], dv[dn][2 * i + 1]);
    }
  }
}

int elem_grid(int64_t n) {
  int64_t b = (n + kRowThreads - 1) / kRowThreads;
  if (b < 1) b = 1;
  if (b > 152 * 16) b = 152 * 16;
  return static_cast<int>(b);
}

template <int HD>
cudaError_t attn_launch(const AttnArgs& a, bool backward, cudaStream_t st) {
  const dim3 grid(static_cast<unsigned>(a.S / kBlk), static_cast<unsigned>(a.nh), static_cast<unsigned>(a.B));
  if (!backward) {
    const int smem = 5 * Tile<HD>::kBytes;
    cudaError_t e = cudaFuncSetAttribute(attn_fwd_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    attn_fwd_kernel<HD><<<grid, kAttnThreads, smem, st>>>(a);
    return cudaGetLastError();
  }
  const int64_t rows = static_cast<int64_t>(a.B) * a.S * a.nh;
  attn_delta_kernel<HD><<<elem_grid(rows * 32), kRowThreads, 0, st>>>(a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  // 128-wide heads over whole 128-token tiles: dQ and dK/dV on tcgen05 (attn_tc.cu)
  if (attention_fwd_tc_supported(a.S, HD))
    return launch_attention_bwd_tc(a.q, a.k, a.v, a.dO, a.lse, a.delta, a.dq, a.dk, a.dv, a.B, a.S, a.nh, a.nkv, st);
  const int smem_q = 6 * Tile<HD>::kBytes;
  e = cudaFuncSetAttribute(attn_bwd_dq_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_q);
  if (e != cudaSuccess) return e;
  attn_bwd_dq_kernel<HD><<<grid, kAttnThreads, smem_q, st>>>(a);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  const int smem_k = 6 * Tile<HD>::kBytes + 4 * kBlk * static_cast<int>(sizeof(float));
  e = cudaFuncSetAttribute(attn_bwd_dkdv_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_k);
  if (e != cudaSuccess) return e;
  const dim3 gk(static_cast<unsigned>(a.S / kBlk), static_cast<unsigned>(a.nkv), static_cast<unsigned>(a.B));
  attn_bwd_dkdv_kernel<HD><<<gk, kAttnThreads, smem_k, st>>>(a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_rmsnorm_fwd(const void* x, bool x_f32, const void* res, const float* gamma, int64_t T, int64_t H,
                               float eps, float* h_out, void* z, float* r, cudaStream_t st) {
  const auto* rp = static_cast<const uint16_t*>(res);
  auto* zp = static_cast<uint16_t*>(z);
  if (H <= 1024) {
    const unsigned grid = static_cast<unsigned>(std::min<int64_t>((T + kRowWarps - 1) / kRowWarps, 152 * 16));
    if (x_f32)
      rmsnorm_fwd_warp_kernel<float><<<grid, kRowThreads, 0, st>>>(static_cast<const float*>(x), rp, gamma, T, H, eps,
                                                                   h_out, zp, r);
    else
      rmsnorm_fwd_warp_kernel<uint16_t><<<grid, kRowThreads, 0, st>>>(static_cast<const uint16_t*>(x), rp, gamma, T, H,
                                                                      eps, h_out, zp, r);
    return cudaGetLastError();
  }
  if (x_f32)
    rmsnorm_fwd_kernel<float><<<static_cast<unsigned>(T), kRowThreads, 0, st>>>(static_cast<const float*>(x), rp, gamma,
                                                                                H, eps, h_out, zp, r);
  else
    rmsnorm_fwd_kernel<uint16_t><<<static_cast<unsigned>(T), kRowThreads, 0, st>>>(static_cast<const uint16_t*>(x), rp,
                                                                                   gamma, H, eps, h_out, zp, r);
  return cudaGetLastError();
}

cudaError_t launch_rmsnorm_bwd(const void* x, bool x_f32, const float* gamma, const float* r, const void* dy,
                               const void* dy2, const void* dres, int64_t T, int64_t H, void* dx, cudaStream_t st) {
  const auto* dyp = static_cast<const uint16_t*>(dy);
  const auto* dy2p = static_cast<const uint16_t*>(dy2);
  const auto* drp = static_cast<const uint16_t*>(dres);
  auto* dxp = static_cast<uint16_t*>(dx);
  if (H <= 1024) {
    const unsigned grid = static_cast<unsigned>(std::min<int64_t>((T + kRowWarps - 1) / kRowWarps, 152 * 16));
    if (x_f32)
      rmsnorm_bwd_warp_kernel<float><<<grid, kRowThreads, 0, st>>>(static_cast<const float*>(x), gamma, r, dyp, dy2p,
                                                                   drp, T, H, dxp);
    else
      rmsnorm_bwd_warp_kernel<uint16_t><<<grid, kRowThreads, 0, st>>>(static_cast<const uint16_t*>(x), gamma, r, dyp,
                                                                      dy2p, drp, T, H, dxp);
    return cudaGetLastError();
  }
  if (x_f32)
    rmsnorm_bwd_kernel<float><<<static_cast<unsigned>(T), kRowThreads, 0, st>>>(static_cast<const float*>(x), gamma, r,
                                                                                dyp, dy2p, drp, H, dxp);
  else
    rmsnorm_bwd_kernel<uint16_t><<<static_cast<unsigned>(T), kRowThreads, 0, st>>>(static_cast<const uint16_t*>(x),
                                                                                   gamma, r, dyp, dy2p, drp, H, dxp);
  return cudaGetLastError();
}

cudaError_t launch_rope(void* x, int64_t T, int64_t S, int32_t nheads, int32_t d, float base, int32_t inverse,
                        cudaStream_t st) {
  if (d % 16 == 0)
    rope_vec_kernel<<<elem_grid(T * (d / 16)), kRowThreads, 0, st>>>(static_cast<uint16_t*>(x), T, S, nheads, d,
                                                                      log2f(base), inverse);
  else
    rope_kernel<<<elem_grid(T * nheads * (d / 2)), kRowThreads, 0, st>>>(static_cast<uint16_t*>(x), T, S, nheads, d,
                                                                          log2f(base), inverse);
  return cudaGetLastError();
}

cudaError_t launch_swiglu(const void* gt, const void* u, const void* dm, int64_t n, void* out, void* dgt, void* du,
                          cudaStream_t st) {
  if (!dm)
    swiglu_fwd_kernel<<<elem_grid((n + 7) / 8), kRowThreads, 0, st>>>(static_cast<const uint16_t*>(gt),
                                                             static_cast<const uint16_t*>(u), n,
                                                             static_cast<uint16_t*>(out));
  else
    swiglu_bwd_kernel<<<elem_grid((n + 7) / 8), kRowThreads, 0, st>>>(
        static_cast<const uint16_t*>(gt), static_cast<const uint16_t*>(u), static_cast<const uint16_t*>(dm), n,
        static_cast<uint16_t*>(dgt), static_cast<uint16_t*>(du));
  return cudaGetLastError();
}

cudaError_t launch_block_output_loss(const float* h, const void* branch, const float* ref, int64_t count,
                                     int32_t reduction, float* out, void* d_out, float* loss_out, double* partials,
                                     cudaStream_t st) {
  const int nb = ref ? recon_loss_blocks(count) : elem_grid(count / 8);
  const double inv = reduction == 0 ? 1.0 / static_cast<double>(count) : 1.0;
  block_output_loss_kernel<<<nb, kRowThreads, 0, st>>>(h, static_cast<const uint16_t*>(branch), ref, count,
                                                        static_cast<float>(2.0 * inv), out,
                                                        static_cast<uint16_t*>(d_out), partials);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess || !ref) return e;
  return launch_loss_final(partials, nb, inv, loss_out, st);
}

cudaError_t launch_attention(const AttnIo& io, int32_t B, int32_t S, int32_t nh, int32_t nkv, int32_t d, bool backward,
                             cudaStream_t st) {
  AttnArgs a{};
  a.q = static_cast<const uint16_t*>(io.q);
  a.k = static_cast<const uint16_t*>(io.k);
  a.v = static_cast<const uint16_t*>(io.v);
  a.o = static_cast<const uint16_t*>(io.o);
  a.dO = static_cast<const uint16_t*>(io.dO);
  a.out = static_cast<uint16_t*>(io.out);
  a.dq = static_cast<uint16_t*>(io.dq);
  a.dk = static_cast<uint16_t*>(io.dk);
  a.dv = static_cast<uint16_t*>(io.dv);
  a.lse = io.lse;
  a.delta = io.delta;
  a.B = B;
  a.S = S;
  a.nh = nh;
  a.nkv = nkv;
  a.scale = 1.0f / sqrtf(static_cast<float>(d));
  a.scale_log2 = a.scale * 1.4426950408889634f;
  // the forward of 128-wide heads over whole 128-token tiles runs on tcgen05 (attn_tc.cu)
  if (!backward && attention_fwd_tc_supported(S, d))
    return launch_attention_fwd_tc(io.q, io.k, io.v, io.out, io.lse, B, S, nh, nkv, st);
  return d == 128 ? attn_launch<128>(a, backward, st) : attn_launch<64>(a, backward, st);
}

}  // namespace catq
