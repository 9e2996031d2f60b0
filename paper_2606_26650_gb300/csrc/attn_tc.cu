// attn_tc.cu — causal grouped-query attention forward on the tcgen05 tensor cores (head
// dimension 128), for the block window's attention (softmax(Q K^T / sqrt(d)) V per head over the
// keys up to the query's position; the row's natural log-sum-exp is kept for the backward).
//
// One CTA per (128-query tile, head, sequence), longest rows first.  Warp roles:
//   warps 0-3  softmax and epilogue: thread = query row = TMEM lane (warp w owns lanes 32w..);
//   warp 4     TMA: the Q tile once, then key/value tiles of 128 through two stages;
//   warp 5     tcgen05: S_j = Q K_j^T into one of two TMEM score buffers, then
//              O += P_j V_j with P_j read from TMEM (the softmax stores it, bf16, over S_j).
// S_{j+1} is issued before the MMA warp waits for P_j, so the next tile's scores are computed
// while the softmax works on this one.  The running maximum is raised lazily: only when a
// tile's maximum exceeds it by more than 8 (log2 units) is O rescaled (the thread's own TMEM
// row, after the previous P V has completed), so P stays below 2^8 and most tiles leave O alone;
// O / l and the log-sum-exp are exact for whichever maximum was used.  Every wait is bounded.
#include <cuda.h>
#include <cudaTypedefs.h>

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
constexpr uint32_t kColS0 = 0, kColO = 256, kTmemCols = 512;
constexpr float kLazy = 8.0f;                        // rescale only past this rise (log2 units)

struct TcAttnArgs {
  uint16_t* out;
  float* lse;
  int32_t S, nh, nkv;
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
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem_raw + (base - raw) + kOffBar + 96);
  const uint32_t bar = base + kOffBar;
  const uint32_t q_full = bar, kv_full0 = bar + 8, kv_empty0 = bar + 24, s_full0 = bar + 40, p_full = bar + 56,
                 o_bar = bar + 64, final_bar = bar + 72;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nqt = a.S / kTq;
  const int qt = nqt - 1 - static_cast<int>(blockIdx.x);  // the longest rows first
  const int h = blockIdx.y, b = blockIdx.z, hk = h / (a.nh / a.nkv);
  const int ntiles = qt + 1;  // key tiles 0..qt (the last one on the diagonal)
  const int32_t row0 = b * a.S;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(kv_full0 + 8u * i, 1);
      mbar_init(kv_empty0 + 8u * i, 1);
      mbar_init(s_full0 + 8u * i, 1);
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
      mbar_arrive_expect_tx(q_full, kTile);
      for (int hf = 0; hf < 2; ++hf)
        tma_load_2d(base + kOffQ + hf * kBox, &tmq, q_full, h * kHd + 64 * hf, row0 + qt * kTq);
      int issued = 0;
      for (int j = 0; j < ntiles; ++j) {
        const int st = j & 1;
        if (j >= 2 && !mbar_wait(kv_empty0 + 8u * st, ((j >> 1) & 1) ^ 1, a.wc)) { ok = false; break; }
        mbar_arrive_expect_tx(kv_full0 + 8u * st, 2 * kTile);
        for (int hf = 0; hf < 2; ++hf) {
          tma_load_2d(base + kOffK + st * kTile + hf * kBox, &tmk, kv_full0 + 8u * st, hk * kHd + 64 * hf,
                      row0 + j * kTk);
          tma_load_2d(base + kOffV + st * kTile + hf * kBox, &tmv, kv_full0 + 8u * st, hk * kHd + 64 * hf,
                      row0 + j * kTk);
        }
        issued = j + 1;
      }
      // copies still in flight (the last two tiles' and Q's) must land before the CTA exits
      drain(q_full, 0);
      for (int j = issued - 2 < 0 ? 0 : issued - 2; j < issued; ++j) drain(kv_full0 + 8u * (j & 1), (j >> 1) & 1);
    }
  } else if (warp == kMmaWarp) {
    if (lane == 0) {
      constexpr uint32_t idesc_s = idesc_bf16_f32(kTq, kTk, false, false);  // Q, K both K-major
      constexpr uint32_t idesc_o = idesc_bf16_f32(kTq, kHd, false, true);   // V MN-major
      auto issue_s = [&](int j) {  // S_j = Q K_j^T into score buffer j & 1
        const uint32_t kt = base + kOffK + (j & 1) * kTile;
#pragma unroll
        for (int kk = 0; kk < kHd / 16; ++kk) {
          const uint32_t off = (kk >> 2) * kBox + (kk & 3) * 32;
          umma_bf16<1>(tmem + kColS0 + 128u * (j & 1), smem_desc_sw128(base + kOffQ + off, 16, 1024),
                       smem_desc_sw128(kt + off, 16, 1024), idesc_s, kk > 0 ? 1u : 0u);
        }
        umma_commit<1>(s_full0 + 8u * (j & 1));
      };
      if (!mbar_wait(q_full, 0, a.wc)) ok = false;
      if (ok && !mbar_wait(kv_full0, 0, a.wc)) ok = false;
      if (ok) {
        tc_fence_after();
        issue_s(0);
      }
      for (int j = 0; ok && j < ntiles; ++j) {
        if (j + 1 < ntiles) {
          if (!mbar_wait(kv_full0 + 8u * ((j + 1) & 1), ((j + 1) >> 1) & 1, a.wc)) { ok = false; break; }
          tc_fence_after();
          issue_s(j + 1);
        }
        if (!mbar_wait(p_full, j & 1, a.wc)) { ok = false; break; }
        tc_fence_after();
        const uint32_t vt = base + kOffV + (j & 1) * kTile;
        const uint32_t pcol = tmem + kColS0 + 128u * (j & 1);
#pragma unroll
        for (int kk = 0; kk < kTk / 16; ++kk)
          umma_ts(tmem + kColO, pcol + 8u * kk, smem_desc_sw128(vt + kk * 2048, kBox, 1024), idesc_o,
                  (j > 0 || kk > 0) ? 1u : 0u);
        umma_commit<1>(o_bar);
        umma_commit<1>(kv_empty0 + 8u * (j & 1));
      }
      // every MMA has completed before TMEM is released
      umma_commit<1>(final_bar);
      drain(final_bar, 0);
    }
  } else {
    // softmax: this thread's query row r of the tile (TMEM lane r)
    const int r = warp * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(warp * 32) << 16;
    float m = -INFINITY, l = 0.0f;
    for (int j = 0; ok && j < ntiles; ++j) {
      const uint32_t sbuf = tmem + lane_off + kColS0 + 128u * (j & 1);
      if (!mbar_wait(s_full0 + 8u * (j & 1), (j >> 1) & 1, a.wc)) { ok = false; break; }
      tc_fence_after();
      uint32_t sr[4][32];
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld32(sbuf + 32u * c, sr[c]);
      tmem_ld_wait();
      float mx = -INFINITY;
      const bool diag = j == qt;
#pragma unroll
      for (int c = 0; c < 4; ++c)
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          float x = __uint_as_float(sr[c][i]) * a.scale_log2;
          if (diag && 32 * c + i > r) x = -INFINITY;
          sr[c][i] = __float_as_uint(x);
          mx = fmaxf(mx, x);
        }
      if (mx > m + kLazy) {
        if (m != -INFINITY) {
          // raise the maximum: O's row (after the previous P V) and l scale by 2^(m - mx)
          const float f = fast_exp2(m - mx);
          l *= f;
          if (!mbar_wait(o_bar, (j - 1) & 1, a.wc)) { ok = false; break; }
          tc_fence_after();
          const uint32_t orow = tmem + lane_off + kColO;
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
#pragma unroll
      for (int c = 0; c < 4; ++c)
#pragma unroll
        for (int i = 0; i < 32; i += 2) {
          const float p0 = fast_exp2(__uint_as_float(sr[c][i]) - m);
          const float p1 = fast_exp2(__uint_as_float(sr[c][i + 1]) - m);
          l += p0 + p1;
          pk[c >> 1][(c & 1) * 16 + i / 2] = pack2(p0, p1);
        }
      // P_j (bf16, keys 2t and 2t + 1 in column t) over the first 64 columns of S_j
      tmem_st32(sbuf, pk[0]);
      tmem_st32(sbuf + 32u, pk[1]);
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive_local(p_full);
    }
    if (ok && mbar_wait(o_bar, (ntiles - 1) & 1, a.wc)) {
      tc_fence_after();
      const float inv = 1.0f / l;
      const int64_t tok = static_cast<int64_t>(row0) + qt * kTq + r;
      uint16_t* orow = a.out + tok * (static_cast<int64_t>(a.nh) * kHd) + static_cast<int64_t>(h) * kHd;
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        uint32_t o[32];
        tmem_ld32(tmem + lane_off + kColO + 32u * c, o);
        tmem_ld_wait();
#pragma unroll
        for (int v = 0; v < 4; ++v) {
          uint4 w;
          w.x = pack2(__uint_as_float(o[8 * v + 0]) * inv, __uint_as_float(o[8 * v + 1]) * inv);
          w.y = pack2(__uint_as_float(o[8 * v + 2]) * inv, __uint_as_float(o[8 * v + 3]) * inv);
          w.z = pack2(__uint_as_float(o[8 * v + 4]) * inv, __uint_as_float(o[8 * v + 5]) * inv);
          w.w = pack2(__uint_as_float(o[8 * v + 6]) * inv, __uint_as_float(o[8 * v + 7]) * inv);
          *reinterpret_cast<uint4*>(orow + 32 * c + 8 * v) = w;
        }
      }
      a.lse[(static_cast<int64_t>(b) * a.nh + h) * a.S + qt * kTq + r] = (m + log2f(l)) * 0.69314718055994531f;
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
  a.S = S;
  a.nh = nh;
  a.nkv = nkv;
  a.scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(kHd));
  if (!launch_wait_ctl(&a.wc)) return cudaErrorInvalidDevice;
  cudaError_t e = cudaFuncSetAttribute(attn_tc_fwd_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem);
  if (e != cudaSuccess) return e;
  attn_tc_fwd_kernel<<<dim3(S / kTq, nh, B), kThreadsTc, kSmem, st>>>(tq, tk, tv, a);
  return cudaGetLastError();
}

}  // namespace catq
