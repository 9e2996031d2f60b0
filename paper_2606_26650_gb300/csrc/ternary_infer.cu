// ternary_infer.cu — inference with the deployed form of a calibrated layer (App. B.2: only
// the ternary codes T and the group scale alpha are kept, W ~ alpha T, or W ~ alpha T + mu for
// the variant of the tab:mu ablation):
//   Y[b, n] = sum_k X[b, k] * (alpha[n, k / g] * T[n, k] + mu[n, k / g])
// reading T from the 2-bit codes catq_hard_ternarize_pack writes.  Decode-shaped (a few token
// rows), so the bound is HBM: every weight costs 0.25 byte of codes plus its share of a 4-byte
// group scale.
//
// Decoding 2-bit codes and multiplying them on the CUDA cores costs several instructions per
// weight, which binds long before HBM does.  Here the multiply-adds go to the tensor pipe
// (mma.sync m16n8k16, bf16 in, fp32 accumulate; a GEMV has too little work per weight for a
// tcgen05 tile to pay off), and decoding costs 10 integer instructions per 16 codes:
//
// * Code c (T = c - 1) sitting at bits 2i, 2i+1 of a 16-bit half, i < 3, is masked in place
//   and OR-ed into the bit pattern of bf16 128 (0x4300), whose mantissa unit is 1: the half
//   is the bf16 value 128 + c 4^i exactly.  One LOP3 makes two such values (the same position
//   in both halves of a 32-bit code word); positions 3..7 take the word shifted by 6 or 12.
// * The activation of that position enters the B operand pre-scaled by 4^-i (a power of two,
//   exact), so the product sums to  sum (128 4^-i + c) x  over the group's columns.
// * A second MMA per k step with constant A rows gives the same sum for c = 1 (T = 0),
//   sum (128 4^-i + 1) x, and the plain activation sum sum x; the first minus the second is
//   sum T x.  Per group: y += alpha (D - D_corr) + mu sum x.
//
// The k order inside an MMA is free as long as A and B agree: a thread's A columns
// {2q, 2q+1, 2q+8, 2q+9} are two positions of its own code word (lower and upper half), and
// its B rows are the activations of exactly those columns.
//
// A CTA of 8 warps owns 16 R rows.  Its codes come in by bulk copies into shared memory, all
// at once when they fit (so the whole layer is in flight from the first cycles), else in K
// slabs through two buffers.  The warps split K into contiguous ranges, and their partial
// sums meet in shared memory in a fixed order (deterministic).  Token rows are taken 8 at a
// time (the MMA's N); all arithmetic after the MMAs is fp32, with one rounding of Y.
#include <cstdint>
#include <type_traits>

#include "launch.h"
#include "ptx_sm100.cuh"

namespace catq {
namespace {

constexpr int kMmaWarps = 8;
constexpr uint32_t kMagic = 0x43004300u;  // bf16 128.0 in both halves

// D += A B for one m16n8k16 tile (A row-major 16 x 16, B column-major 16 x 8, bf16).
__device__ __forceinline__ void mma_16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                          uint32_t b0, uint32_t b1) {
  asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t mul_bf16x2(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("mul.rn.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}

// Position p (0..7) of a code word's halves: which shifted copy of the word holds it at bits
// 2i..2i+1 (i < 3), the mask selecting it there, and its scale 4^i.
__host__ __device__ constexpr int pos_shift(int p) { return p < 3 ? 0 : (p < 6 ? 1 : 2); }
__host__ __device__ constexpr int pos_i(int p) { return p - 3 * pos_shift(p); }
__host__ __device__ constexpr uint32_t pos_mask(int p) { return 0x00030003u << (2 * pos_i(p)); }
// bf16 pairs: (128 + 4^i) for the correction row, 4^i for the activation-sum row, 4^-i for
// the activations.
__host__ __device__ constexpr uint32_t pos_corr(int p) { return kMagic | (0x00010001u << (2 * pos_i(p))); }
__host__ __device__ constexpr uint32_t pos_unit(int p) {
  return pos_i(p) == 0 ? 0x3F803F80u : (pos_i(p) == 1 ? 0x40804080u : 0x41804180u);
}
__host__ __device__ constexpr uint32_t pos_inv(int p) {
  return pos_i(p) == 0 ? 0x3F803F80u : (pos_i(p) == 1 ? 0x3E803E80u : 0x3D803D80u);
}

// The three shifted copies of a code word, and the magic constant held in a register, so
// that mask-and-insert is one three-input logic operation (a & mask | magic).
struct Shifted {
  uint32_t t[3];
  uint32_t magic;
};
__device__ __forceinline__ Shifted shifted(uint32_t w, uint32_t magic) {
  return Shifted{{w, w >> 6, w >> 12}, magic};
}

template <int P>
__device__ __forceinline__ uint32_t code_pair(const Shifted& s) {
  uint32_t d;
  asm("lop3.b32 %0, %1, %2, %3, 0xEA;" : "=r"(d) : "r"(s.t[pos_shift(P)]), "n"(pos_mask(P)), "r"(s.magic));
  return d;
}

// An opaque copy of the magic constant (kept in a register instead of being folded into
// each logic operation as a second immediate).
__device__ __forceinline__ uint32_t magic_reg() {
  uint32_t m;
  asm volatile("mov.b32 %0, %1;" : "=r"(m) : "n"(kMagic));
  return m;
}

// Activation pair (x[p], x[p + 8]) of 16 consecutive bf16 (h0 = elements 0..7, h1 = 8..15),
// scaled by 4^-i of position p.
template <int P>
__device__ __forceinline__ uint32_t act_pair(const uint4& h0, const uint4& h1) {
  const uint32_t lo = (P / 2) == 0 ? h0.x : (P / 2) == 1 ? h0.y : (P / 2) == 2 ? h0.z : h0.w;
  const uint32_t hi = (P / 2) == 0 ? h1.x : (P / 2) == 1 ? h1.y : (P / 2) == 2 ? h1.z : h1.w;
  const uint32_t v = __byte_perm(lo, hi, (P & 1) ? 0x7632 : 0x5410);
  return pos_i(P) == 0 ? v : mul_bf16x2(v, pos_inv(P));
}

// VW consecutive code words of shared memory (one 4- or 8-byte load).
template <int VW>
__device__ __forceinline__ void ld_shared_words(uint32_t addr, uint32_t (&w)[VW]) {
  if constexpr (VW == 2)
    asm volatile("ld.shared.v2.u32 {%0, %1}, [%2];" : "=r"(w[0]), "=r"(w[1]) : "r"(addr));
  else
    asm volatile("ld.shared.u32 %0, [%1];" : "=r"(w[0]) : "r"(addr));
}

// MMA j of one code word of each of the thread's two rows: positions 2j and 2j + 1.
template <int J>
__device__ __forceinline__ void word_mma(float (&d)[4], const Shifted& r0, const Shifted& r1,
                                         const uint32_t (&xb)[8]) {
  mma_16816(d, code_pair<2 * J>(r0), code_pair<2 * J>(r1), code_pair<2 * J + 1>(r0), code_pair<2 * J + 1>(r1),
            xb[2 * J], xb[2 * J + 1]);
}

// Bounded wait for copies already issued, used when a launch gives up.
__device__ __forceinline__ void drain_wait(uint32_t bar, uint32_t parity) {
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity))
    if (globaltimer_ns() - t0 > 200000000ull) return;
}

// R: 16-row tiles per CTA.  VW: code words per thread per super-chunk (a super-chunk is
// 64 VW columns and lies in one group).  MU: add mu times each group's activation sum.
// The CTA's codes arrive by bulk copies (one per row and K slab of KS columns) into a ring
// of one or two slab buffers; each row's copy lands at a stride padded by 16 VW bytes, so
// the fragment reads (four lanes per row, eight rows per instruction) are free of bank
// conflicts.
template <int R, int VW, bool MU>
__global__ void __launch_bounds__(kMmaWarps * 32, 2) ternary_mma_kernel(const uint8_t* __restrict__ codes,
                                                                     const float* __restrict__ alpha,
                                                                     const float* __restrict__ mu, int64_t N,
                                                                     int64_t K, int32_t g, int64_t KS,
                                                                     const uint16_t* __restrict__ X, int64_t B,
                                                                     uint16_t* __restrict__ Y, const WaitCtl wc) {
  constexpr int ROWS = 16 * R;
  extern __shared__ __align__(128) uint8_t ring[];
  __shared__ float red[kMmaWarps][8][ROWS];
  __shared__ __align__(8) uint64_t full_bar[2];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int gid = lane >> 2, q = lane & 3;
  const uint32_t row_bytes = static_cast<uint32_t>(KS / 4 + 16 * VW);
  const uint32_t ring_base = smem_u32(ring);
  const uint32_t bar0 = smem_u32(&full_bar[0]);
  // column and group counts fit 32 bits (K < 2^31, N K / g < 2^31)
  const int32_t nslabs = static_cast<int32_t>((K + KS - 1) / KS);
  const int32_t sc_per_slab = static_cast<int32_t>(KS / (64 * VW));
  const int32_t sc_per_group = g / (64 * VW);
  const int32_t gpr = static_cast<int32_t>(K / g);
  const int64_t nblocks = (N + ROWS - 1) / ROWS;
  if (threadIdx.x == 0) {
    mbar_init(bar0, 1);
    mbar_init(bar0 + 8, 1);
    fence_mbar_init_cluster();
  }
  __syncthreads();
  uint32_t uses = 0;  // completed phases of both barriers, bit b for barrier b (CTA-uniform)
  const uint32_t magic = magic_reg();

  // Warp 0 issues the bulk copies of slab `slab` of rows n0.. into buffer `buf`.
  auto issue = [&](int64_t n0, int64_t slab, int buf) {
    const int64_t k0 = slab * KS;
    const uint32_t bytes = static_cast<uint32_t>((K - k0 < KS ? K - k0 : KS) / 4);
    const int nvalid = static_cast<int>(N - n0 < ROWS ? N - n0 : ROWS);
    const uint32_t bar = bar0 + 8u * buf;
    if (lane == 0) mbar_arrive_expect_tx(bar, bytes * nvalid);
    __syncwarp();
    for (int r = lane; r < nvalid; r += 32)
      bulk_load_g2s(ring_base + (buf * ROWS + r) * row_bytes, codes + (n0 + r) * (K / 4) + k0 / 4, bytes, bar);
  };

  bool ok = true;
  for (int64_t rb = blockIdx.x; ok && rb < nblocks; rb += gridDim.x) {
    const int64_t n0 = rb * ROWS;
    int32_t goff[R][2];  // group-array offsets of this thread's two rows of each tile (rows
                         // past N take row N - 1's, and are not stored)
#pragma unroll
    for (int r = 0; r < R; ++r)
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int64_t n = n0 + 16 * r + gid + 8 * h;
        goff[r][h] = static_cast<int32_t>((n < N ? n : N - 1) * gpr);
      }
    for (int64_t b0 = 0; ok && b0 < B; b0 += 8) {
      if (warp == 0) {
        issue(n0, 0, 0);
        if (nslabs > 1) issue(n0, 1, 1);
      }
      // Token columns past B read token b0's activations instead: their sums are computed
      // and never stored, so no load needs a predicate.
      const uint16_t* xrow = X + (b0 + gid < B ? b0 + gid : b0) * K;
      float acc[R][4], d[R][4], da[4];
#pragma unroll
      for (int r = 0; r < R; ++r)
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[r][e] = d[r][e] = 0.0f;
#pragma unroll
      for (int e = 0; e < 4; ++e) da[e] = 0.0f;

      for (int32_t slab = 0; slab < nslabs; ++slab) {
        const int buf = slab & 1;
        const bool landed = mbar_wait(bar0 + 8u * buf, (uses >> buf) & 1u, wc);
        if (!__syncthreads_and(landed)) {
          // copies into this buffer, and the next slab's into the other, may still be in flight
          if (threadIdx.x == 0) {
            drain_wait(bar0 + 8u * buf, (uses >> buf) & 1u);
            if (slab + 1 < nslabs) drain_wait(bar0 + 8u * (buf ^ 1), (uses >> (buf ^ 1)) & 1u);
          }
          __syncthreads();
          ok = false;
          break;
        }
        uses ^= 1u << buf;
        // this warp's contiguous range of the slab's super-chunks, and the group it starts in
        const int32_t k0 = slab * static_cast<int32_t>(KS);
        const int32_t n_sc = static_cast<int32_t>(((K - k0 < KS) ? K - k0 : KS) / (64 * VW));
        const int32_t lo = n_sc * warp / kMmaWarps, hi = n_sc * (warp + 1) / kMmaWarps;
        int32_t grp = (slab * sc_per_slab + lo) / sc_per_group;
        int32_t left = (grp + 1) * sc_per_group - (slab * sc_per_slab + lo);  // super-chunks to its end
        const uint32_t tile = ring_base + buf * ROWS * row_bytes;
        // per-thread bases, advanced by the super-chunk index inside the loop
        uint32_t rowa[R][2];  // shared-memory address of the thread's words in each of its rows
#pragma unroll
        for (int r = 0; r < R; ++r)
#pragma unroll
          for (int h = 0; h < 2; ++h) rowa[r][h] = tile + (16 * r + gid + 8 * h) * row_bytes + VW * q * 4;
        const uint4* xbase = reinterpret_cast<const uint4*>(xrow + k0 + 16 * VW * q);
        const bool every_sc = sc_per_group == 1;  // each super-chunk is a whole group
        auto load_x = [&](int32_t sc, uint4 (&xv)[2 * VW]) {
          const uint4* xp = xbase + sc * (8 * VW);
#pragma unroll
          for (int i = 0; i < 2 * VW; ++i) xv[i] = __ldg(xp + i);
        };
        // one super-chunk: this thread's code words from shared memory, its activations xv
        auto step = [&](int32_t sc, const uint4 (&xv)[2 * VW]) {
          const uint32_t woff = static_cast<uint32_t>(sc * 16 * VW);
          uint32_t cw[R][2][VW];  // the thread's code words of rows gid and gid + 8 of each tile
#pragma unroll
          for (int r = 0; r < R; ++r) {
            ld_shared_words<VW>(rowa[r][0] + woff, cw[r][0]);
            ld_shared_words<VW>(rowa[r][1] + woff, cw[r][1]);
          }
#pragma unroll
          for (int v = 0; v < VW; ++v) {
            uint32_t xb[8];
            const uint4 h0 = xv[2 * v], h1 = xv[2 * v + 1];
            xb[0] = act_pair<0>(h0, h1);
            xb[1] = act_pair<1>(h0, h1);
            xb[2] = act_pair<2>(h0, h1);
            xb[3] = act_pair<3>(h0, h1);
            xb[4] = act_pair<4>(h0, h1);
            xb[5] = act_pair<5>(h0, h1);
            xb[6] = act_pair<6>(h0, h1);
            xb[7] = act_pair<7>(h0, h1);
            // rows 0..7 of the constant tile: the correction sums; rows 8..15: activation sums
            mma_16816(da, pos_corr(0), pos_unit(0), pos_corr(1), pos_unit(1), xb[0], xb[1]);
            mma_16816(da, pos_corr(2), pos_unit(2), pos_corr(3), pos_unit(3), xb[2], xb[3]);
            mma_16816(da, pos_corr(4), pos_unit(4), pos_corr(5), pos_unit(5), xb[4], xb[5]);
            mma_16816(da, pos_corr(6), pos_unit(6), pos_corr(7), pos_unit(7), xb[6], xb[7]);
#pragma unroll
            for (int r = 0; r < R; ++r) {
              const Shifted s0 = shifted(cw[r][0][v], magic), s1 = shifted(cw[r][1][v], magic);
              word_mma<0>(d[r], s0, s1, xb);
              word_mma<1>(d[r], s0, s1, xb);
              word_mma<2>(d[r], s0, s1, xb);
              word_mma<3>(d[r], s0, s1, xb);
            }
          }
          if (every_sc || --left == 0 || sc + 1 == hi) {  // the group, or this warp's range, ends
#pragma unroll
            for (int r = 0; r < R; ++r) {
              const float a0 = __ldg(alpha + goff[r][0] + grp), a1 = __ldg(alpha + goff[r][1] + grp);
              acc[r][0] = fmaf(a0, d[r][0] - da[0], acc[r][0]);
              acc[r][1] = fmaf(a0, d[r][1] - da[1], acc[r][1]);
              acc[r][2] = fmaf(a1, d[r][2] - da[0], acc[r][2]);
              acc[r][3] = fmaf(a1, d[r][3] - da[1], acc[r][3]);
              if constexpr (MU) {
                const float m0 = __ldg(mu + goff[r][0] + grp), m1 = __ldg(mu + goff[r][1] + grp);
                acc[r][0] = fmaf(m0, da[2], acc[r][0]);
                acc[r][1] = fmaf(m0, da[3], acc[r][1]);
                acc[r][2] = fmaf(m1, da[2], acc[r][2]);
                acc[r][3] = fmaf(m1, da[3], acc[r][3]);
              }
#pragma unroll
              for (int e = 0; e < 4; ++e) d[r][e] = 0.0f;
            }
#pragma unroll
            for (int e = 0; e < 4; ++e) da[e] = 0.0f;
            if (every_sc) {
              ++grp;
            } else if (left == 0) {
              ++grp;
              left = sc_per_group;
            }
          }
        };
        // activations one super-chunk ahead, in two alternating register sets
        uint4 xa[2 * VW], xc[2 * VW];
        if (lo < hi) load_x(lo, xa);
        for (int32_t sc = lo; sc < hi; sc += 2) {
          if (sc + 1 < hi) load_x(sc + 1, xc);
          step(sc, xa);
          if (sc + 1 >= hi) break;
          if (sc + 2 < hi) load_x(sc + 2, xa);
          step(sc + 1, xc);
        }
        __syncthreads();  // every warp is done with this buffer
        if (warp == 0 && slab + 2 < nslabs) issue(n0, slab + 2, buf);
      }
      if (!ok) break;

      // D fragment: (row gid, tokens 2q, 2q + 1) and (row gid + 8, the same tokens)
#pragma unroll
      for (int r = 0; r < R; ++r) {
        red[warp][2 * q][16 * r + gid] = acc[r][0];
        red[warp][2 * q + 1][16 * r + gid] = acc[r][1];
        red[warp][2 * q][16 * r + gid + 8] = acc[r][2];
        red[warp][2 * q + 1][16 * r + gid + 8] = acc[r][3];
      }
      __syncthreads();
      for (int e = threadIdx.x; e < 8 * ROWS; e += kMmaWarps * 32) {
        const int tok = e / ROWS, row = e % ROWS;
        float s = 0.0f;
#pragma unroll
        for (int w = 0; w < kMmaWarps; ++w) s += red[w][tok][row];
        if (b0 + tok < B && n0 + row < N)
          Y[(b0 + tok) * N + n0 + row] = static_cast<uint16_t>(pack_bf16x2(s, 0.0f) & 0xFFFFu);
      }
      __syncthreads();
    }
  }
}

constexpr int64_t kRingBytes = 72 * 1024;  // code bytes of one slab buffer

template <int R, int VW>
cudaError_t launch_mma(const uint8_t* codes, const float* alpha, const float* mu, int64_t N, int64_t K, int32_t g,
                       const uint16_t* X, int64_t B, uint16_t* Y, cudaStream_t st) {
  WaitCtl wc;
  if (!launch_wait_ctl(&wc)) return cudaErrorInvalidDevice;
  const int64_t rows = 16 * R;
  // K slab: all of K when the CTA's rows fit one buffer, else the largest multiple of
  // 64 VW columns that does (two buffers then alternate).
  int64_t KS = K;
  if (rows * (K / 4 + 16 * VW) > kRingBytes) KS = ((kRingBytes / rows - 16 * VW) * 4) / (64 * VW) * (64 * VW);
  const int64_t nslabs = (K + KS - 1) / KS;
  const int smem = static_cast<int>((nslabs > 1 ? 2 : 1) * rows * (KS / 4 + 16 * VW));
  int64_t blocks = (N + rows - 1) / rows;
  if (blocks > 152 * 16) blocks = 152 * 16;
  auto kern = mu ? ternary_mma_kernel<R, VW, true> : ternary_mma_kernel<R, VW, false>;
  const cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  kern<<<static_cast<int>(blocks), kMmaWarps * 32, smem, st>>>(codes, alpha, mu, N, K, g, KS, X, B, Y, wc);
  return cudaGetLastError();
}

template <int R>
cudaError_t launch_rows(const uint8_t* codes, const float* alpha, const float* mu, int64_t N, int64_t K, int32_t g,
                        const uint16_t* X, int64_t B, uint16_t* Y, cudaStream_t st) {
  if (g % 128 == 0) return launch_mma<R, 2>(codes, alpha, mu, N, K, g, X, B, Y, st);
  return launch_mma<R, 1>(codes, alpha, mu, N, K, g, X, B, Y, st);
}

}  // namespace

cudaError_t launch_ternary_infer(const uint8_t* codes, const float* alpha, const float* mu, int64_t N, int64_t K,
                                 int32_t g, const void* X, int64_t B, void* Y, cudaStream_t st) {
  const uint16_t* x = static_cast<const uint16_t*>(X);
  uint16_t* y = static_cast<uint16_t*>(Y);
  // 16-row tiles per CTA: the fewest rows on the busiest SM (CTAs spread evenly over the
  // SMs), then the most tiles per CTA (the correction MMAs and the activation preparation
  // serve more rows), with the CTA's codes within one ring buffer.
  int sm = 152;
  {
    int dev = 0;
    if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sm, cudaDevAttrMultiProcessorCount, dev);
  }
  int best = 1;
  int64_t best_rows = -1;
  for (int r = 1; r <= 4; ++r) {
    if (r > 1 && 16 * r * (K / 4 + 32) > kRingBytes) break;
    const int64_t ctas = (N + 16 * r - 1) / (16 * r);
    const int64_t busiest = (ctas + sm - 1) / sm * 16 * r;
    if (best_rows < 0 || busiest <= best_rows) {
      best = r;
      best_rows = busiest;
    }
  }
  switch (best) {
    case 4: return launch_rows<4>(codes, alpha, mu, N, K, g, x, B, y, st);
    case 3: return launch_rows<3>(codes, alpha, mu, N, K, g, x, B, y, st);
    case 2: return launch_rows<2>(codes, alpha, mu, N, K, g, x, B, y, st);
    default: return launch_rows<1>(codes, alpha, mu, N, K, g, x, B, y, st);
  }
}

}  // namespace catq
