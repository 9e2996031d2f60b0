// attn_tc.cu — causal grouped-query attention on the tcgen05 tensor cores (head dimension 128,
// sequences in whole 128-token tiles), for the block window's attention: the forward
// (softmax(Q K^T / sqrt(d)) V per head over the keys up to the query's position, and the row's
// natural log-sum-exp for the backward), and the backward in two kernels (dQ per query tile,
// persistent over the forward's work items; dK and dV per key tile over the query heads
// sharing it), without atomics.
//
// Forward: a persistent CTA per SM takes every gridDim-th (128-query tile, head, sequence) work
// item, longest rows first; the output accumulator has two TMEM buffers, so one item's
// epilogue overlaps the next item's first products.  Warp roles:
//   warps 0-3  softmax and epilogue: thread = query row = TMEM lane (warp w owns lanes 32w..);
//   warp 4     TMA: each item's Q tile, then its key/value tiles of 128 through two stages;
//   warp 5     tcgen05: S_j = Q K_j^T into one of two TMEM score buffers, then
//              O += P_j V_j with P_j read from TMEM (the softmax stores it, bf16, over S_j).
// S_{j+1} is issued before the MMA warp waits for P_j, so the next tile's scores are computed
// while the softmax works on this one.  The running maximum is raised lazily: only when a
// tile's maximum exceeds it by more than 8 (log2 units) is O rescaled (the thread's own TMEM
// row, after the previous P V has completed), so P stays below 2^8 and most tiles leave O alone;
// O / l and the log-sum-exp are exact for whichever maximum was used.  Every wait is bounded.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <cmath>
#include <cstdint>
#include <mutex>

#include "launch.h"
#include "ptx_sm100.cuh"

namespace catq {
namespace {

constexpr int kTq = 128;             // query rows per tile (MMA M, TMEM lanes)
constexpr int kTk = 128;             // keys per tile (MMA N of Q K^T, K of P V)
constexpr int kHd = 128;             // head dimension
constexpr int kThreadsTc = 6 * 32;   // 4 softmax warps, TMA warp, MMA warp
constexpr int kTmaWarp = 4, kMmaWarp = 5;
constexpr uint32_t kBox = 128 * 128;                 // one 64-column box of 128 rows, bytes
constexpr uint32_t kTile = 2 * kBox;                 // 128 rows x 128 columns, bytes
constexpr uint32_t kOffQ = 0, kOffK = kTile, kOffV = 3 * kTile, kOffBar = 5 * kTile;
constexpr uint32_t kSmem = kOffBar + 128 + 1024;     // + barriers, 1 KB alignment slack
constexpr uint32_t kColS0 = 0, kColO = 256, kTmemCols = 512;  // S0, S1; O0, O1 (one per item parity)
constexpr float kLazy = 8.0f;                        // rescale only past this rise (log2 units)

struct TcAttnArgs {
  uint16_t* out;
  float* lse;
  int32_t B, S, nh, nkv;
  float scale_log2;
  WaitCtl wc;
};

__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
      "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]),
      "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]),
      "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]),
      "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}
__device__ __forceinline__ void tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// D[tmem] (+)= A[tmem] * B[smem] (A: M x K bf16 in TMEM, one row per lane, column j holding
// elements 2j and 2j + 1 of the row).
__device__ __forceinline__ void umma_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc, uint32_t idesc,
                                        uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ float fast_exp2(float x) {
  float r;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}

__device__ __forceinline__ uint32_t pack2(float lo, float hi) {
  uint32_t r;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

// Bounded wait for copies or MMAs still in flight when a launch gives up.
__device__ __forceinline__ void drain(uint32_t bar, uint32_t parity) {
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity))
    if (globaltimer_ns() - t0 > 200000000ull) return;
}

__global__ void __launch_bounds__(kThreadsTc, 1)
    attn_tc_fwd_kernel(const __grid_constant__ CUtensorMap tmq, const __grid_constant__ CUtensorMap tmk,
                       const __grid_constant__ CUtensorMap tmv, const TcAttnArgs a) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem_raw + (base - raw) + kOffBar + 120);
  const uint32_t bar = base + kOffBar;
  // per item: q_full, q_empty; per tile: kv_full[2], kv_empty[2], s_full[2], p_full, o_bar;
  // per item and output buffer: item_done[2], o_free[2]; final_bar once
  const uint32_t q_full = bar, q_empty = bar + 8, kv_full0 = bar + 16, kv_empty0 = bar + 32, s_full0 = bar + 48,
                 p_full = bar + 64, o_bar = bar + 72, item_done0 = bar + 80, o_free0 = bar + 96,
                 final_bar = bar + 112;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nqt = a.S / kTq;
  const int n_items = nqt * a.nh * a.B;
  // item -> (query tile, head, sequence), the longest rows first
  auto item_of = [&](int it, int& qt, int& h, int& b) {
    qt = nqt - 1 - it / (a.nh * a.B);
    const int rem = it % (a.nh * a.B);
    h = rem % a.nh;
    b = rem / a.nh;
  };

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    mbar_init(q_empty, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(kv_full0 + 8u * i, 1);
      mbar_init(kv_empty0 + 8u * i, 1);
      mbar_init(s_full0 + 8u * i, 1);
      mbar_init(item_done0 + 8u * i, 1);
      mbar_init(o_free0 + 8u * i, kTq);
    }
    mbar_init(p_full, kTq);
    mbar_init(o_bar, 1);
    mbar_init(final_bar, 1);
    fence_mbar_init_cluster();
  }
  if (warp == kMmaWarp) tmem_alloc<1>(smem_u32(tmem_slot), kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  bool ok = true;

  if (warp == kTmaWarp) {
    if (lane == 0) {
      prefetch_tmap(&tmq);
      prefetch_tmap(&tmk);
      prefetch_tmap(&tmv);
      int g = 0, li = 0, q_loads = 0;
      for (int it = blockIdx.x; ok && it < n_items; it += gridDim.x, ++li) {
        int qt, h, b;
        item_of(it, qt, h, b);
        const int hk = h / (a.nh / a.nkv);
        const int32_t row0 = b * a.S;
        // the Q buffer is free once every score product of the previous item has completed
        if (li > 0 && !mbar_wait(q_empty, (li - 1) & 1, a.wc)) { ok = false; break; }
        ++q_loads;
        mbar_arrive_expect_tx(q_full, kTile);
        for (int hf = 0; hf < 2; ++hf)
          tma_load_2d(base + kOffQ + hf * kBox, &tmq, q_full, h * kHd + 64 * hf, row0 + qt * kTq);
        for (int j = 0; j <= qt; ++j, ++g) {
          const int st = g & 1;
          if (g >= 2 && !mbar_wait(kv_empty0 + 8u * st, ((g >> 1) & 1) ^ 1, a.wc)) { ok = false; break; }
          mbar_arrive_expect_tx(kv_full0 + 8u * st, 2 * kTile);
          for (int hf = 0; hf < 2; ++hf) {
            tma_load_2d(base + kOffK + st * kTile + hf * kBox, &tmk, kv_full0 + 8u * st, hk * kHd + 64 * hf,
                        row0 + j * kTk);
            tma_load_2d(base + kOffV + st * kTile + hf * kBox, &tmv, kv_full0 + 8u * st, hk * kHd + 64 * hf,
                        row0 + j * kTk);
          }
        }
      }
      // copies still in flight (the last item's Q, the last two tiles) land before the CTA exits
      if (q_loads > 0) drain(q_full, (q_loads - 1) & 1);
      for (int t = g - 2 < 0 ? 0 : g - 2; t < g; ++t) drain(kv_full0 + 8u * (t & 1), (t >> 1) & 1);
    }
  } else if (warp == kMmaWarp) {
    if (lane == 0) {
      constexpr uint32_t idesc_s = idesc_bf16_f32(kTq, kTk, false, false);  // Q, K both K-major
      constexpr uint32_t idesc_o = idesc_bf16_f32(kTq, kHd, false, true);   // V MN-major
      // S_t = Q K^T of global tile t into score buffer t & 1; after an item's last one, the Q
      // buffer is released
      auto issue_s = [&](int t, bool last) -> bool {
        if (!mbar_wait(kv_full0 + 8u * (t & 1), (t >> 1) & 1, a.wc)) return false;
        tc_fence_after();
        const uint32_t kt = base + kOffK + (t & 1) * kTile;
#pragma unroll
        for (int kk = 0; kk < kHd / 16; ++kk) {
          const uint32_t off = (kk >> 2) * kBox + (kk & 3) * 32;
          umma_bf16<1>(tmem + kColS0 + 128u * (t & 1), smem_desc_sw128(base + kOffQ + off, 16, 1024),
                       smem_desc_sw128(kt + off, 16, 1024), idesc_s, kk > 0 ? 1u : 0u);
        }
        umma_commit<1>(s_full0 + 8u * (t & 1));
        if (last) umma_commit<1>(q_empty);
        return true;
      };
      int g = 0, li = 0;
      for (int it = blockIdx.x; ok && it < n_items; it += gridDim.x, ++li) {
        int qt, h, b;
        item_of(it, qt, h, b);
        const int n = qt + 1;
        const uint32_t ocol = tmem + kColO + 128u * (li & 1);
        if (!mbar_wait(q_full, li & 1, a.wc) || !issue_s(g, n == 1)) { ok = false; break; }
        for (int j = 0; ok && j < n; ++j) {
          const int t = g + j;
          if (j + 1 < n && !issue_s(t + 1, j + 2 == n)) { ok = false; break; }
          if (!mbar_wait(p_full, t & 1, a.wc)) { ok = false; break; }
          // the item's output buffer is free once the epilogue two items back has read it
          if (j == 0 && li >= 2 && !mbar_wait(o_free0 + 8u * (li & 1), ((li >> 1) & 1) ^ 1, a.wc)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t vt = base + kOffV + (t & 1) * kTile;
          const uint32_t pcol = tmem + kColS0 + 128u * (t & 1);
#pragma unroll
          for (int kk = 0; kk < kTk / 16; ++kk)
            umma_ts(ocol, pcol + 8u * kk, smem_desc_sw128(vt + kk * 2048, kBox, 1024), idesc_o,
                    (j > 0 || kk > 0) ? 1u : 0u);
          umma_commit<1>(o_bar);
          umma_commit<1>(kv_empty0 + 8u * (t & 1));
        }
        if (!ok) break;
        umma_commit<1>(item_done0 + 8u * (li & 1));
        g += n;
      }
      // every MMA has completed before TMEM is released
      umma_commit<1>(final_bar);
      drain(final_bar, 0);
    }
  } else {
    // softmax and epilogue: this thread's query row r of each item's tile (TMEM lane r)
    const int r = warp * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(warp * 32) << 16;
    int g = 0, li = 0;
    for (int it = blockIdx.x; ok && it < n_items; it += gridDim.x, ++li) {
      int qt, h, b;
      item_of(it, qt, h, b);
      const int n = qt + 1;
      const uint32_t orow = tmem + lane_off + kColO + 128u * (li & 1);
      float m = -INFINITY, l = 0.0f;
      for (int j = 0; ok && j < n; ++j) {
        const int t = g + j;
        const uint32_t sbuf = tmem + lane_off + kColS0 + 128u * (t & 1);
        if (!mbar_wait(s_full0 + 8u * (t & 1), (t >> 1) & 1, a.wc)) { ok = false; break; }
        tc_fence_after();
        uint32_t sr[4][32];
#pragma unroll
        for (int c = 0; c < 4; ++c) tmem_ld32(sbuf + 32u * c, sr[c]);
        tmem_ld_wait();
        if (j == qt) {  // the diagonal tile: keys after the row's query do not count
#pragma unroll
          for (int c = 0; c < 4; ++c)
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if (32 * c + i > r) sr[c][i] = __float_as_uint(-INFINITY);
        }
        // the row maximum of the raw scores (scale > 0), in eight independent chains
        float mv[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) mv[i] = -INFINITY;
#pragma unroll
        for (int c = 0; c < 4; ++c)
#pragma unroll
          for (int i = 0; i < 32; ++i) mv[i & 7] = fmaxf(mv[i & 7], __uint_as_float(sr[c][i]));
#pragma unroll
        for (int w = 4; w > 0; w >>= 1)
#pragma unroll
          for (int i = 0; i < w; ++i) mv[i] = fmaxf(mv[i], mv[i + w]);
        const float mx = mv[0] * a.scale_log2;
        if (mx > m + kLazy) {
          if (m != -INFINITY) {
            // raise the maximum: O's row (after the previous P V) and l scale by 2^(m - mx)
            const float f = fast_exp2(m - mx);
            l *= f;
            if (!mbar_wait(o_bar, (t - 1) & 1, a.wc)) { ok = false; break; }
            tc_fence_after();
#pragma unroll
            for (int c = 0; c < 4; ++c) {
              uint32_t o[32];
              tmem_ld32(orow + 32u * c, o);
              tmem_ld_wait();
#pragma unroll
              for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * f);
              tmem_st32(orow + 32u * c, o);
            }
          }
          m = mx;
        }
        uint32_t pk[2][32];
        float ls[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) ls[i] = 0.0f;
#pragma unroll
        for (int c = 0; c < 4; ++c)
#pragma unroll
          for (int i = 0; i < 32; i += 2) {
            const float p0 = fast_exp2(fmaf(__uint_as_float(sr[c][i]), a.scale_log2, -m));
            const float p1 = fast_exp2(fmaf(__uint_as_float(sr[c][i + 1]), a.scale_log2, -m));
            ls[(i >> 1) & 7] += p0 + p1;
            pk[c >> 1][(c & 1) * 16 + i / 2] = pack2(p0, p1);
          }
#pragma unroll
        for (int w = 4; w > 0; w >>= 1)
#pragma unroll
          for (int i = 0; i < w; ++i) ls[i] += ls[i + w];
        l += ls[0];
        // P_t (bf16, keys 2u and 2u + 1 in column u) over the first 64 columns of S_t
        tmem_st32(sbuf, pk[0]);
        tmem_st32(sbuf + 32u, pk[1]);
        tmem_st_wait();
        tc_fence_before();
        mbar_arrive_local(p_full);
      }
      if (!ok) break;
      // the item's output: every P V of the item has completed (item_done, one phase per use
      // of the buffer); then the buffer goes back to the MMA warp for the item after next
      if (!mbar_wait(item_done0 + 8u * (li & 1), (li >> 1) & 1, a.wc)) { ok = false; break; }
      tc_fence_after();
      const float inv = 1.0f / l;
      const int64_t tok = static_cast<int64_t>(b) * a.S + qt * kTq + r;
      uint16_t* dst = a.out + tok * (static_cast<int64_t>(a.nh) * kHd) + static_cast<int64_t>(h) * kHd;
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        uint32_t o[32];
        tmem_ld32(orow + 32u * c, o);
        tmem_ld_wait();
#pragma unroll
        for (int v = 0; v < 4; ++v) {
          uint4 w;
          w.x = pack2(__uint_as_float(o[8 * v + 0]) * inv, __uint_as_float(o[8 * v + 1]) * inv);
          w.y = pack2(__uint_as_float(o[8 * v + 2]) * inv, __uint_as_float(o[8 * v + 3]) * inv);
          w.z = pack2(__uint_as_float(o[8 * v + 4]) * inv, __uint_as_float(o[8 * v + 5]) * inv);
          w.w = pack2(__uint_as_float(o[8 * v + 6]) * inv, __uint_as_float(o[8 * v + 7]) * inv);
          *reinterpret_cast<uint4*>(dst + 32 * c + 8 * v) = w;
        }
      }
      a.lse[(static_cast<int64_t>(b) * a.nh + h) * a.S + qt * kTq + r] = (m + log2f(l)) * 0.69314718055994531f;
      tc_fence_before();
      mbar_arrive_local(o_free0 + 8u * (li & 1));
      g += n;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc<1>(tmem, kTmemCols);
  }
}

// ---------------------------------------------------------------- backward
// With P = exp(scale S - lse) recomputed from the forward's log-sum-exp, dP = dO V^T and
// dS = P * (dP - delta) (delta = rowsum(dO * O), from attn_delta_kernel):
//   dQ = scale dS K,  dK = scale dS^T Q,  dV = P^T dO,
// in two kernels, so that every accumulator has one owner and no atomics are needed.

struct TcBwdArgs {
  uint16_t *dq, *dk, *dv;
  const float* lse;    // natural log-sum-exp per (sequence, head, row)
  const float* delta;  // rowsum(dO * O) per (sequence, head, row)
  int32_t B, S, nh, nkv;
  float scale_log2;
  float scale;
  WaitCtl wc;
};

constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(
          taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]),
      "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}

// K-major SS products of the backward: D (+)= A B^T over d = 128 (A, B: 128 rows x 128
// columns, two 64-column boxes each).
__device__ __forceinline__ void mma_kmajor(uint32_t d_tmem, uint32_t a_smem, uint32_t b_smem, uint32_t idesc) {
#pragma unroll
  for (int kk = 0; kk < kHd / 16; ++kk) {
    const uint32_t off = (kk >> 2) * kBox + (kk & 3) * 32;
    umma_bf16<1>(d_tmem, smem_desc_sw128(a_smem + off, 16, 1024), smem_desc_sw128(b_smem + off, 16, 1024), idesc,
                 kk > 0 ? 1u : 0u);
  }
}

// TS products: D (+)= A[tmem] B[smem] over 128 (A: 128 x 128 bf16 in TMEM, B: the 128-row
// tile read as K x N with N contiguous).
__device__ __forceinline__ void mma_ts_tile(uint32_t d_tmem, uint32_t a_tmem, uint32_t b_smem, uint32_t idesc,
                                            bool accumulate) {
#pragma unroll
  for (int kk = 0; kk < 8; ++kk)
    umma_ts(d_tmem, a_tmem + 8u * kk, smem_desc_sw128(b_smem + kk * 2048, kBox, 1024), idesc,
            (accumulate || kk > 0) ? 1u : 0u);
}

// dQ: persistent CTAs over (128-query tile, head, sequence) items (the forward's order), each
// over the key tiles up to the diagonal.  TMEM: S [0, 128), dP [128, 256), dQ in two buffers
// [256, 512) (one per item parity, so an item's epilogue overlaps the next item's products);
// dS (bf16) goes over S's first 64 columns.
constexpr uint32_t kDqOffQ = 0, kDqOffDo = kTile, kDqOffK = 2 * kTile, kDqOffV = 4 * kTile, kDqOffBar = 6 * kTile;
constexpr uint32_t kDqSmem = kDqOffBar + 128 + 1024;

__global__ void __launch_bounds__(kThreadsTc, 1)
    attn_tc_dq_kernel(const __grid_constant__ CUtensorMap tmq, const __grid_constant__ CUtensorMap tmdo,
                      const __grid_constant__ CUtensorMap tmk, const __grid_constant__ CUtensorMap tmv,
                      const TcBwdArgs a) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem_raw + (base - raw) + kDqOffBar + 120);
  const uint32_t bar = base + kDqOffBar;
  const uint32_t qd_full = bar, qd_empty = bar + 8, kv_full0 = bar + 16, kv_empty0 = bar + 32, s_full = bar + 48,
                 ds_full = bar + 56, item_done0 = bar + 64, dq_free0 = bar + 80, final_bar = bar + 96;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nqt = a.S / kTq;
  const int n_items = nqt * a.nh * a.B;
  auto item_of = [&](int it, int& qt, int& h, int& b) {
    qt = nqt - 1 - it / (a.nh * a.B);
    const int rem = it % (a.nh * a.B);
    h = rem % a.nh;
    b = rem / a.nh;
  };
  constexpr uint32_t kColS = 0, kColP = 128, kColQ = 256;

  if (threadIdx.x == 0) {
    mbar_init(qd_full, 1);
    mbar_init(qd_empty, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(kv_full0 + 8u * i, 1);
      mbar_init(kv_empty0 + 8u * i, 1);
      mbar_init(item_done0 + 8u * i, 1);
      mbar_init(dq_free0 + 8u * i, kTq);
    }
    mbar_init(s_full, 1);
    mbar_init(ds_full, kTq);
    mbar_init(final_bar, 1);
    fence_mbar_init_cluster();
  }
  if (warp == kMmaWarp) tmem_alloc<1>(smem_u32(tmem_slot), kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  bool ok = true;

  if (warp == kTmaWarp) {
    if (lane == 0) {
      int g = 0, li = 0, qd_loads = 0;
      for (int it = blockIdx.x; ok && it < n_items; it += gridDim.x, ++li) {
        int qt, h, b;
        item_of(it, qt, h, b);
        const int hk = h / (a.nh / a.nkv);
        const int32_t row0 = b * a.S;
        // Q and dO are free once the previous item's S and dP products have completed
        if (li > 0 && !mbar_wait(qd_empty, (li - 1) & 1, a.wc)) { ok = false; break; }
        ++qd_loads;
        mbar_arrive_expect_tx(qd_full, 2 * kTile);
        for (int hf = 0; hf < 2; ++hf) {
          tma_load_2d(base + kDqOffQ + hf * kBox, &tmq, qd_full, h * kHd + 64 * hf, row0 + qt * kTq);
          tma_load_2d(base + kDqOffDo + hf * kBox, &tmdo, qd_full, h * kHd + 64 * hf, row0 + qt * kTq);
        }
        for (int j = 0; j <= qt; ++j, ++g) {
          const int st = g & 1;
          if (g >= 2 && !mbar_wait(kv_empty0 + 8u * st, ((g >> 1) & 1) ^ 1, a.wc)) { ok = false; break; }
          mbar_arrive_expect_tx(kv_full0 + 8u * st, 2 * kTile);
          for (int hf = 0; hf < 2; ++hf) {
            tma_load_2d(base + kDqOffK + st * kTile + hf * kBox, &tmk, kv_full0 + 8u * st, hk * kHd + 64 * hf,
                        row0 + j * kTk);
            tma_load_2d(base + kDqOffV + st * kTile + hf * kBox, &tmv, kv_full0 + 8u * st, hk * kHd + 64 * hf,
                        row0 + j * kTk);
          }
        }
      }
      if (qd_loads > 0) drain(qd_full, (qd_loads - 1) & 1);
      for (int t = g - 2 < 0 ? 0 : g - 2; t < g; ++t) drain(kv_full0 + 8u * (t & 1), (t >> 1) & 1);
    }
  } else if (warp == kMmaWarp) {
    if (lane == 0) {
      constexpr uint32_t idesc_s = idesc_bf16_f32(kTq, kTk, false, false);
      constexpr uint32_t idesc_q = idesc_bf16_f32(kTq, kHd, false, true);
      int g = 0, li = 0;
      for (int it = blockIdx.x; ok && it < n_items; it += gridDim.x, ++li) {
        int qt, h, b;
        item_of(it, qt, h, b);
        const int n = qt + 1;
        const uint32_t qcol = tmem + kColQ + 128u * (li & 1);
        if (!mbar_wait(qd_full, li & 1, a.wc)) { ok = false; break; }
        for (int j = 0; ok && j < n; ++j) {
          const int t = g + j;
          const uint32_t kt = base + kDqOffK + (t & 1) * kTile, vt = base + kDqOffV + (t & 1) * kTile;
          if (!mbar_wait(kv_full0 + 8u * (t & 1), (t >> 1) & 1, a.wc)) { ok = false; break; }
          tc_fence_after();
          mma_kmajor(tmem + kColS, base + kDqOffQ, kt, idesc_s);   // S = Q K^T
          mma_kmajor(tmem + kColP, base + kDqOffDo, vt, idesc_s);  // dP = dO V^T
          umma_commit<1>(s_full);
          if (j + 1 == n) umma_commit<1>(qd_empty);
          if (!mbar_wait(ds_full, t & 1, a.wc)) { ok = false; break; }
          // the item's dQ buffer is free once the epilogue two items back has read it
          if (j == 0 && li >= 2 && !mbar_wait(dq_free0 + 8u * (li & 1), ((li >> 1) & 1) ^ 1, a.wc)) {
            ok = false;
            break;
          }
          tc_fence_after();
          mma_ts_tile(qcol, tmem + kColS, kt, idesc_q, j > 0);  // dQ += dS K
          umma_commit<1>(kv_empty0 + 8u * (t & 1));
        }
        if (!ok) break;
        umma_commit<1>(item_done0 + 8u * (li & 1));
        g += n;
      }
      umma_commit<1>(final_bar);
      drain(final_bar, 0);
    }
  } else {
    const int r = warp * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(warp * 32) << 16;
    int g = 0, li = 0;
    for (int it = blockIdx.x; ok && it < n_items; it += gridDim.x, ++li) {
      int qt, h, b;
      item_of(it, qt, h, b);
      const int n = qt + 1;
      const int64_t ridx = (static_cast<int64_t>(b) * a.nh + h) * a.S + qt * kTq + r;
      const float lse2 = a.lse[ridx] * kLog2e, dl = a.delta[ridx];
      for (int j = 0; ok && j < n; ++j) {
        const int t = g + j;
        if (!mbar_wait(s_full, t & 1, a.wc)) { ok = false; break; }
        tc_fence_after();
        const bool diag = j == qt;
#pragma unroll
        for (int c2 = 0; c2 < 4; c2 += 2) {  // two 32-column chunks per TMEM wait
          uint32_t sv[2][32], pv[2][32];
#pragma unroll
          for (int u = 0; u < 2; ++u) {
            tmem_ld32(tmem + lane_off + kColS + 32u * (c2 + u), sv[u]);
            tmem_ld32(tmem + lane_off + kColP + 32u * (c2 + u), pv[u]);
          }
          tmem_ld_wait();
#pragma unroll
          for (int u = 0; u < 2; ++u) {
            const int c = c2 + u;
            uint32_t ds[16];
#pragma unroll
            for (int i = 0; i < 32; i += 2) {
              float p0 = fast_exp2(fmaf(__uint_as_float(sv[u][i]), a.scale_log2, -lse2));
              float p1 = fast_exp2(fmaf(__uint_as_float(sv[u][i + 1]), a.scale_log2, -lse2));
              if (diag && 32 * c + i > r) p0 = 0.0f;
              if (diag && 32 * c + i + 1 > r) p1 = 0.0f;
              ds[i / 2] = pack2(p0 * (__uint_as_float(pv[u][i]) - dl), p1 * (__uint_as_float(pv[u][i + 1]) - dl));
            }
            tmem_st16(tmem + lane_off + kColS + 16u * c, ds);
          }
        }
        tmem_st_wait();
        tc_fence_before();
        mbar_arrive_local(ds_full);
      }
      if (!ok) break;
      // every dQ product of the item has completed (item_done, one phase per use of the buffer)
      if (!mbar_wait(item_done0 + 8u * (li & 1), (li >> 1) & 1, a.wc)) { ok = false; break; }
      tc_fence_after();
      const int64_t tok = static_cast<int64_t>(b) * a.S + qt * kTq + r;
      uint16_t* drow = a.dq + tok * (static_cast<int64_t>(a.nh) * kHd) + static_cast<int64_t>(h) * kHd;
      const uint32_t qrow = tmem + lane_off + kColQ + 128u * (li & 1);
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        uint32_t o[32];
        tmem_ld32(qrow + 32u * c, o);
        tmem_ld_wait();
#pragma unroll
        for (int v = 0; v < 4; ++v) {
          uint4 w;
          w.x = pack2(__uint_as_float(o[8 * v + 0]) * a.scale, __uint_as_float(o[8 * v + 1]) * a.scale);
          w.y = pack2(__uint_as_float(o[8 * v + 2]) * a.scale, __uint_as_float(o[8 * v + 3]) * a.scale);
          w.z = pack2(__uint_as_float(o[8 * v + 4]) * a.scale, __uint_as_float(o[8 * v + 5]) * a.scale);
          w.w = pack2(__uint_as_float(o[8 * v + 6]) * a.scale, __uint_as_float(o[8 * v + 7]) * a.scale);
          *reinterpret_cast<uint4*>(drow + 32 * c + 8 * v) = w;
        }
      }
      tc_fence_before();
      mbar_arrive_local(dq_free0 + 8u * (li & 1));
      g += n;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc<1>(tmem, kTmemCols);
  }
}

// dK, dV: one CTA per (128-key tile, key/value head, sequence), over every query head of the
// group and the query tiles from the diagonal on, with the scores formed transposed (keys as
// TMEM lanes), so P^T and dS^T are the A operands of dV and dK straight from TMEM.
// TMEM: S^T [0, 128), dP^T [128, 256), dV [256, 384), dK [384, 512); P^T and dS^T (bf16)
// over the first 64 columns of S^T and dP^T.  A stage holds the query tile, its dO tile
// and their rows' log-sum-exp and delta.
constexpr uint32_t kKvOffK = 0, kKvOffV = kTile, kKvOffStage = 2 * kTile;
constexpr uint32_t kStageLse = 2 * kTile, kStageDelta = 2 * kTile + 512, kStageBytes = 2 * kTile + 1024;
constexpr uint32_t kKvOffBar = kKvOffStage + 2 * kStageBytes;
constexpr uint32_t kKvSmem = kKvOffBar + 128 + 1024;

__global__ void __launch_bounds__(kThreadsTc, 1)
    attn_tc_dkdv_kernel(const __grid_constant__ CUtensorMap tmq, const __grid_constant__ CUtensorMap tmdo,
                        const __grid_constant__ CUtensorMap tmk, const __grid_constant__ CUtensorMap tmv,
                        const TcBwdArgs a) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(gbase + kKvOffBar + 96);
  const uint32_t bar = base + kKvOffBar;
  const uint32_t kv_full = bar, st_full0 = bar + 8, st_empty0 = bar + 24, s_full = bar + 40, pd_full = bar + 48,
                 final_bar = bar + 64;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nqt = a.S / kTq;
  const int kt = static_cast<int>(blockIdx.x);  // key tile; the first ones have the most query tiles
  const int hk = blockIdx.y, b = blockIdx.z;
  const int rep = a.nh / a.nkv;
  const int per_head = nqt - kt;  // query tiles kt..nqt-1
  const int nsteps = rep * per_head;
  const int32_t row0 = b * a.S;
  constexpr uint32_t kColS = 0, kColP = 128, kColV = 256, kColK = 384;

  if (threadIdx.x == 0) {
    mbar_init(kv_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(st_full0 + 8u * i, 1);
      mbar_init(st_empty0 + 8u * i, 1);
    }
    mbar_init(s_full, 1);
    mbar_init(pd_full, kTq);
    mbar_init(final_bar, 1);
    fence_mbar_init_cluster();
  }
  if (warp == kMmaWarp) tmem_alloc<1>(smem_u32(tmem_slot), kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  bool ok = true;
  auto step_head = [&](int t) { return hk * rep + t / per_head; };
  auto step_tile = [&](int t) { return kt + t % per_head; };

  if (warp == kTmaWarp) {
    if (lane == 0) {
      mbar_arrive_expect_tx(kv_full, 2 * kTile);
      for (int hf = 0; hf < 2; ++hf) {
        tma_load_2d(base + kKvOffK + hf * kBox, &tmk, kv_full, hk * kHd + 64 * hf, row0 + kt * kTk);
        tma_load_2d(base + kKvOffV + hf * kBox, &tmv, kv_full, hk * kHd + 64 * hf, row0 + kt * kTk);
      }
      int issued = 0;
      for (int t = 0; t < nsteps; ++t) {
        const int st = t & 1, h = step_head(t), i = step_tile(t);
        if (t >= 2 && !mbar_wait(st_empty0 + 8u * st, ((t >> 1) & 1) ^ 1, a.wc)) { ok = false; break; }
        const uint32_t sb = base + kKvOffStage + st * kStageBytes;
        mbar_arrive_expect_tx(st_full0 + 8u * st, kStageBytes);
        for (int hf = 0; hf < 2; ++hf) {
          tma_load_2d(sb + hf * kBox, &tmq, st_full0 + 8u * st, h * kHd + 64 * hf, row0 + i * kTq);
          tma_load_2d(sb + kTile + hf * kBox, &tmdo, st_full0 + 8u * st, h * kHd + 64 * hf, row0 + i * kTq);
        }
        const int64_t ridx = (static_cast<int64_t>(b) * a.nh + h) * a.S + i * kTq;
        bulk_load_g2s(sb + kStageLse, a.lse + ridx, kTq * 4, st_full0 + 8u * st);
        bulk_load_g2s(sb + kStageDelta, a.delta + ridx, kTq * 4, st_full0 + 8u * st);
        issued = t + 1;
      }
      drain(kv_full, 0);
      for (int t = issued - 2 < 0 ? 0 : issued - 2; t < issued; ++t) drain(st_full0 + 8u * (t & 1), (t >> 1) & 1);
    }
  } else if (warp == kMmaWarp) {
    if (lane == 0) {
      constexpr uint32_t idesc_s = idesc_bf16_f32(kTk, kTq, false, false);
      constexpr uint32_t idesc_g = idesc_bf16_f32(kTk, kHd, false, true);
      if (!mbar_wait(kv_full, 0, a.wc)) ok = false;
      for (int t = 0; ok && t < nsteps; ++t) {
        const uint32_t sb = base + kKvOffStage + (t & 1) * kStageBytes;
        if (!mbar_wait(st_full0 + 8u * (t & 1), (t >> 1) & 1, a.wc)) { ok = false; break; }
        tc_fence_after();
        mma_kmajor(tmem + kColS, base + kKvOffK, sb, idesc_s);          // S^T = K Q^T
        mma_kmajor(tmem + kColP, base + kKvOffV, sb + kTile, idesc_s);  // dP^T = V dO^T
        umma_commit<1>(s_full);
        if (!mbar_wait(pd_full, t & 1, a.wc)) { ok = false; break; }
        tc_fence_after();
        mma_ts_tile(tmem + kColV, tmem + kColS, sb + kTile, idesc_g, t > 0);  // dV += P^T dO
        mma_ts_tile(tmem + kColK, tmem + kColP, sb, idesc_g, t > 0);          // dK += dS^T Q
        umma_commit<1>(st_empty0 + 8u * (t & 1));
      }
      umma_commit<1>(final_bar);
      drain(final_bar, 0);
    }
  } else {
    const int rk = warp * 32 + lane;  // key row of the tile (TMEM lane)
    const uint32_t lane_off = static_cast<uint32_t>(warp * 32) << 16;
    for (int t = 0; ok && t < nsteps; ++t) {
      if (!mbar_wait(s_full, t & 1, a.wc)) { ok = false; break; }
      tc_fence_after();
      const float* lse = reinterpret_cast<const float*>(gbase + kKvOffStage + (t & 1) * kStageBytes + kStageLse);
      const float* dlt = reinterpret_cast<const float*>(gbase + kKvOffStage + (t & 1) * kStageBytes + kStageDelta);
      const bool diag = step_tile(t) == kt;
#pragma unroll
      for (int c2 = 0; c2 < 4; c2 += 2) {  // two 32-column chunks per TMEM wait
        uint32_t sv[2][32], pv[2][32];
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          tmem_ld32(tmem + lane_off + kColS + 32u * (c2 + u), sv[u]);
          tmem_ld32(tmem + lane_off + kColP + 32u * (c2 + u), pv[u]);
        }
        tmem_ld_wait();
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          const int c = c2 + u;
          uint32_t pp[16], ds[16];
#pragma unroll
          for (int i = 0; i < 32; i += 2) {
            const int q = 32 * c + i;
            float p0 = fast_exp2(fmaf(__uint_as_float(sv[u][i]), a.scale_log2, -lse[q] * kLog2e));
            float p1 = fast_exp2(fmaf(__uint_as_float(sv[u][i + 1]), a.scale_log2, -lse[q + 1] * kLog2e));
            if (diag && q < rk) p0 = 0.0f;
            if (diag && q + 1 < rk) p1 = 0.0f;
            pp[i / 2] = pack2(p0, p1);
            ds[i / 2] =
                pack2(p0 * (__uint_as_float(pv[u][i]) - dlt[q]), p1 * (__uint_as_float(pv[u][i + 1]) - dlt[q + 1]));
          }
          tmem_st16(tmem + lane_off + kColS + 16u * c, pp);
          tmem_st16(tmem + lane_off + kColP + 16u * c, ds);
        }
      }
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive_local(pd_full);
    }
    if (ok && mbar_wait(final_bar, 0, a.wc)) {  // every MMA has completed (one phase)
      tc_fence_after();
      const int64_t tok = static_cast<int64_t>(row0) + kt * kTk + rk;
      const int64_t off = tok * (static_cast<int64_t>(a.nkv) * kHd) + static_cast<int64_t>(hk) * kHd;
#pragma unroll
      for (int g2 = 0; g2 < 2; ++g2) {
        uint16_t* drow = (g2 == 0 ? a.dk : a.dv) + off;
        const uint32_t col = g2 == 0 ? kColK : kColV;
        const float f = g2 == 0 ? a.scale : 1.0f;
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          uint32_t o[32];
          tmem_ld32(tmem + lane_off + col + 32u * c, o);
          tmem_ld_wait();
#pragma unroll
          for (int v = 0; v < 4; ++v) {
            uint4 w;
            w.x = pack2(__uint_as_float(o[8 * v + 0]) * f, __uint_as_float(o[8 * v + 1]) * f);
            w.y = pack2(__uint_as_float(o[8 * v + 2]) * f, __uint_as_float(o[8 * v + 3]) * f);
            w.z = pack2(__uint_as_float(o[8 * v + 4]) * f, __uint_as_float(o[8 * v + 5]) * f);
            w.w = pack2(__uint_as_float(o[8 * v + 6]) * f, __uint_as_float(o[8 * v + 7]) * f);
            *reinterpret_cast<uint4*>(drow + 32 * c + 8 * v) = w;
          }
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc<1>(tmem, kTmemCols);
  }
}

PFN_cuTensorMapEncodeTiled_v12000 g_enc = nullptr;
std::once_flag g_enc_once;

// bf16 row-major [outer, inner] tensor with rows `row_elems` apart, 128-byte swizzled boxes of
// 64 x 128.
bool tmap_rows(CUtensorMap* m, const void* ptr, uint64_t inner, uint64_t outer) {
  std::call_once(g_enc_once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_enc = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  });
  if (!g_enc) return false;
  const cuuint64_t dims[2] = {inner, outer};
  const cuuint64_t strides[1] = {inner * 2};
  const cuuint32_t box[2] = {64, 128};
  const cuuint32_t estr[2] = {1, 1};
  return g_enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

bool attention_fwd_tc_supported(int32_t S, int32_t d) { return d == kHd && S % kTq == 0 && S > 0; }

cudaError_t launch_attention_fwd_tc(const void* q, const void* k, const void* v, void* out, float* lse, int32_t B,
                                    int32_t S, int32_t nh, int32_t nkv, cudaStream_t st) {
  if (!attention_fwd_tc_supported(S, kHd) || B < 1 || nh < 1 || nkv < 1 || nh % nkv != 0)
    return cudaErrorInvalidValue;
  CUtensorMap tq, tk, tv;
  const uint64_t rows = static_cast<uint64_t>(B) * S;
  if (!tmap_rows(&tq, q, static_cast<uint64_t>(nh) * kHd, rows) ||
      !tmap_rows(&tk, k, static_cast<uint64_t>(nkv) * kHd, rows) ||
      !tmap_rows(&tv, v, static_cast<uint64_t>(nkv) * kHd, rows))
    return cudaErrorInvalidValue;
  TcAttnArgs a{};
  a.out = static_cast<uint16_t*>(out);
  a.lse = lse;
  a.B = B;
  a.S = S;
  a.nh = nh;
  a.nkv = nkv;
  a.scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(kHd));
  if (!launch_wait_ctl(&a.wc)) return cudaErrorInvalidDevice;
  cudaError_t e = cudaFuncSetAttribute(attn_tc_fwd_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem);
  if (e != cudaSuccess) return e;
  int sm = 152, dev = 0;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sm, cudaDevAttrMultiProcessorCount, dev);
  const int64_t items = static_cast<int64_t>(S / kTq) * nh * B;
  // persistent: one CTA per SM (shared memory and the 512 TMEM columns allow no second), each
  // taking every gridDim-th work item
  attn_tc_fwd_kernel<<<static_cast<unsigned>(std::min<int64_t>(items, sm)), kThreadsTc, kSmem, st>>>(tq, tk, tv, a);
  return cudaGetLastError();
}


cudaError_t launch_attention_bwd_tc(const void* q, const void* k, const void* v, const void* dO, const float* lse,
                                    const float* delta, void* dq, void* dk, void* dv, int32_t B, int32_t S, int32_t nh,
                                    int32_t nkv, cudaStream_t st) {
  if (!attention_fwd_tc_supported(S, kHd) || B < 1 || nh < 1 || nkv < 1 || nh % nkv != 0)
    return cudaErrorInvalidValue;
  CUtensorMap tq, tdo, tk, tv;
  const uint64_t rows = static_cast<uint64_t>(B) * S;
  if (!tmap_rows(&tq, q, static_cast<uint64_t>(nh) * kHd, rows) ||
      !tmap_rows(&tdo, dO, static_cast<uint64_t>(nh) * kHd, rows) ||
      !tmap_rows(&tk, k, static_cast<uint64_t>(nkv) * kHd, rows) ||
      !tmap_rows(&tv, v, static_cast<uint64_t>(nkv) * kHd, rows))
    return cudaErrorInvalidValue;
  TcBwdArgs a{};
  a.dq = static_cast<uint16_t*>(dq);
  a.dk = static_cast<uint16_t*>(dk);
  a.dv = static_cast<uint16_t*>(dv);
  a.lse = lse;
  a.delta = delta;
  a.B = B;
  a.S = S;
  a.nh = nh;
  a.nkv = nkv;
  a.scale = 1.0f / sqrtf(static_cast<float>(kHd));
  a.scale_log2 = a.scale * kLog2e;
  if (!launch_wait_ctl(&a.wc)) return cudaErrorInvalidDevice;
  cudaError_t e = cudaFuncSetAttribute(attn_tc_dq_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kDqSmem);
  if (e != cudaSuccess) return e;
  int sm = 152, dev = 0;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sm, cudaDevAttrMultiProcessorCount, dev);
  const int64_t items = static_cast<int64_t>(S / kTq) * nh * B;
  attn_tc_dq_kernel<<<static_cast<unsigned>(std::min<int64_t>(items, sm)), kThreadsTc, kDqSmem, st>>>(tq, tdo, tk, tv,
                                                                                                        a);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  e = cudaFuncSetAttribute(attn_tc_dkdv_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kKvSmem);
  if (e != cudaSuccess) return e;
  attn_tc_dkdv_kernel<<<dim3(S / kTk, nkv, B), kThreadsTc, kKvSmem, st>>>(tq, tdo, tk, tv, a);
  return cudaGetLastError();
}

}  // namespace catq
