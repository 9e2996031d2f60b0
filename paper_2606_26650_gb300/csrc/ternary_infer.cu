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
// A launch covers one or several layers (independent of each other).  Its work items are
// blocks of 16 R rows of a layer; a persistent CTA of 8 warps takes every gridDim-th item and
// streams their codes, in K slabs, through two shared-memory buffers by bulk copies, the next
// slab (of this item or the next) on its way while the current one is computed.  The warps
// split each slab into contiguous K ranges, and their partial sums meet in shared memory in a
// fixed order (deterministic).  Token rows are taken 8 at a time (the MMA's N); all
// arithmetic after the MMAs is fp32, with one rounding of Y.
//
// A staged launch runs a chain of such layer sets in one cooperative launch (the layers of a
// decode step in dependency order: stage s + 1 may read what stage s wrote).  The work items
// of all stages form one stream; before its first item of a stage, a CTA arrives at the
// barriers of the stages it is done with and waits (bounded) until every CTA has arrived at
// the previous stage's.  The code slabs of the next items do not depend on earlier stages,
// so their copies are issued before the wait and the HBM stream does not drain at a stage
// boundary.  Activations of a staged launch are read through L2 (ld.global.cg), since a
// previous stage of the same launch may have written them.
#include <algorithm>
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

// One layer of a launch: its buffers, shape and code slabs (KS columns per slab, nslabs per
// token block), its group count per row, and its first work item.
struct InferLayer {
  const uint8_t* codes;
  const float* alpha;
  const float* mu;
  const uint16_t* X;
  uint16_t* Y;
  int64_t N, K, B;
  int32_t gpr;     // groups per row, K / g
  int32_t KS;      // code columns per slab (a multiple of 64 VW)
  int32_t nslabs;  // slabs per token block
  int32_t item0;   // first work item of this layer
};

constexpr int kMaxInferLayers = 32;
constexpr int kMaxInferStages = 32;

struct InferArgs {
  int32_t n_layers;
  int32_t total_items;  // work items (16 R-row blocks) over all layers
  int32_t g;
  int32_t n_stages;     // staged launches: stages; 1 otherwise
  uint32_t* sync;       // staged launches: [kMaxInferStages] barrier counters, then the exit counter
  int32_t stage_end[kMaxInferStages];  // first item after each stage
  InferLayer L[kMaxInferLayers];
};

// Staged launches: arrive at a stage barrier (after every thread's stores, by one thread).
__device__ __forceinline__ void counter_arrive(uint32_t* ctr) {
  asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(ctr) : "memory");
}

__device__ __forceinline__ uint32_t counter_load(const uint32_t* ctr) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(ctr) : "memory");
  return v;
}

// Bounded wait until *ctr >= target: false on timeout (latched) or when another wait of the
// launch has given up.
__device__ __forceinline__ bool counter_wait(const uint32_t* ctr, uint32_t target, const WaitCtl& w) {
  if (counter_load(ctr) >= target) return true;
  const uint64_t t0 = globaltimer_ns();
  for (;;) {
    __nanosleep(128);
    if (counter_load(ctr) >= target) return true;
    if (aborted(w)) return false;
    if (globaltimer_ns() - t0 > w.timeout_ns) {
      signal_timeout(w);
      return false;
    }
  }
}

// A position in a CTA's stream of code slabs: work item t (a block of 16 R rows of layer l),
// token block b0 and slab.  Work items run t = blockIdx.x, blockIdx.x + gridDim.x, ...
struct Cursor {
  int32_t t, l, slab;
  int64_t b0;
};

__device__ __forceinline__ void cursor_at(Cursor& c, int32_t t, const InferArgs& a) {
  c.t = t;
  c.slab = 0;
  c.b0 = 0;
  c.l = 0;
  if (t >= a.total_items) return;
  int lo = 0, hi = a.n_layers;  // last layer whose first item is <= t
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (a.L[mid].item0 <= t) lo = mid;
    else hi = mid;
  }
  c.l = lo;
}

__device__ __forceinline__ void cursor_next(Cursor& c, const InferArgs& a) {
  const InferLayer& L = a.L[c.l];
  if (++c.slab < L.nslabs) return;
  c.slab = 0;
  c.b0 += 8;
  if (c.b0 < L.B) return;
  cursor_at(c, c.t + static_cast<int32_t>(gridDim.x), a);
}

// R: 16-row tiles per work item.  VW: code words per thread per super-chunk (a super-chunk is
// 64 VW columns and lies in one group).  MU: add mu times each group's activation sum.
// A persistent CTA walks its work items (over every layer of the launch) as one stream of
// code slabs through two shared-memory buffers: once every warp has passed slab c + 1's
// barrier (so slab c is consumed), warp 0 issues the bulk copies of slab c + 2 into slab c's
// buffer, whichever item and layer it belongs to, so the next item's codes are on their way
// while this one finishes its slabs and its reduction.  Each row's copy lands at a stride
// padded by 16 VW bytes, so the fragment reads (four lanes per row, eight rows per
// instruction) are free of bank conflicts.  Two CTA barriers per slab or item: the slab's
// landing (which also frees the slab before it) and the partial sums' hand-over.
template <int R, int VW, bool MU, bool STAGED>
__global__ void __launch_bounds__(kMmaWarps * 32, 2) ternary_mma_kernel(const __grid_constant__ InferArgs a,
                                                                     int32_t buf_bytes, const WaitCtl wc) {
  constexpr int ROWS = 16 * R;
  extern __shared__ __align__(128) uint8_t ring[];
  __shared__ float red[kMmaWarps][8][ROWS];
  __shared__ __align__(8) uint64_t full_bar[2];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int gid = lane >> 2, q = lane & 3;
  const uint32_t ring_base = smem_u32(ring);
  const uint32_t bar0 = smem_u32(&full_bar[0]);
  const int32_t sc_per_group = a.g / (64 * VW);
  if (threadIdx.x == 0) {
    mbar_init(bar0, 1);
    mbar_init(bar0 + 8, 1);
    fence_mbar_init_cluster();
  }
  __syncthreads();
  const uint32_t magic = magic_reg();

  // Warp 0 issues the bulk copies of the slab at cursor c into buffer `buf`.
  auto issue = [&](const Cursor& c, int buf) {
    const InferLayer& L = a.L[c.l];
    const int64_t n0 = static_cast<int64_t>(c.t - L.item0) * ROWS;
    const int64_t k0 = static_cast<int64_t>(c.slab) * L.KS;
    const uint32_t bytes = static_cast<uint32_t>((L.K - k0 < L.KS ? L.K - k0 : L.KS) / 4);
    const uint32_t row_bytes = static_cast<uint32_t>(L.KS / 4 + 16 * VW);
    const int nvalid = static_cast<int>(L.N - n0 < ROWS ? L.N - n0 : ROWS);
    const uint32_t bar = bar0 + 8u * buf;
    if (lane == 0) mbar_arrive_expect_tx(bar, bytes * nvalid);
    __syncwarp();
    for (int r = lane; r < nvalid; r += 32)
      bulk_load_g2s(ring_base + buf * buf_bytes + r * row_bytes, L.codes + (n0 + r) * (L.K / 4) + k0 / 4, bytes,
                    bar);
  };

  // The next kernel of the stream may launch now (it waits for this one before it touches
  // anything this one writes).  The codes, scales and offsets are weights that inference
  // never writes, so the first slabs' copies go out before waiting for the previous kernel,
  // whose output may be this launch's X (or whose input may alias this launch's Y).
  grid_launch_dependents();
  Cursor iss, con;
  cursor_at(iss, blockIdx.x, a);
  cursor_at(con, blockIdx.x, a);
  uint32_t issued = 0;  // slabs issued (tracked by warp 0, which issues them)
  if (warp == 0) {
    for (int b = 0; b < 2 && iss.t < a.total_items; ++b) {
      issue(iss, b);
      cursor_next(iss, a);
      ++issued;
    }
  }
  grid_dependency_wait();
  uint32_t qn = 0;  // slabs consumed
  bool ok = true;
  int32_t goff[R][2];
  const uint16_t* xrow = nullptr;
  float acc[R][4], d[R][4], da[4];
  int32_t stage = 0, arrived = 0;  // staged: stage of the current item, barriers arrived at

  while (ok && con.t < a.total_items) {
    if constexpr (STAGED) {
      if (con.slab == 0 && con.b0 == 0) {
        int32_t st = stage;
        while (con.t >= a.stage_end[st]) ++st;
        if (st > stage) {
          // This CTA has no items left in stages before st (items run in order): its outputs
          // there are stored.  Arrive at those stages' barriers, then wait until every CTA has
          // arrived at stage st - 1's.
          __syncthreads();
          bool good = true;
          if (threadIdx.x == 0) {
            __threadfence();
            for (int32_t b = arrived; b < st; ++b) counter_arrive(a.sync + b);
            good = counter_wait(a.sync + (st - 1), gridDim.x, wc);
          }
          arrived = st;
          stage = st;
          if (!__syncthreads_and(good)) {
            if (threadIdx.x == 0) {
              // copies of this CTA's next slabs may be in flight
              if (issued > qn) drain_wait(bar0 + 8u * (qn & 1u), (qn >> 1) & 1u);
              if (issued > qn + 1) drain_wait(bar0 + 8u * ((qn + 1) & 1u), ((qn + 1) >> 1) & 1u);
            }
            __syncthreads();
            ok = false;
            break;
          }
        }
      }
    }
    const InferLayer& L = a.L[con.l];
    const int64_t n0 = static_cast<int64_t>(con.t - L.item0) * ROWS;
    if (con.slab == 0) {
      // a new token block of this item: group offsets of the thread's rows (rows past N take
      // row N - 1's and are not stored), accumulators, and the activation row (token columns
      // past B read token b0's activations: their sums are computed and never stored)
#pragma unroll
      for (int r = 0; r < R; ++r)
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int64_t n = n0 + 16 * r + gid + 8 * h;
          goff[r][h] = static_cast<int32_t>((n < L.N ? n : L.N - 1) * L.gpr);
        }
      xrow = L.X + (con.b0 + gid < L.B ? con.b0 + gid : con.b0) * L.K;
#pragma unroll
      for (int r = 0; r < R; ++r)
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[r][e] = d[r][e] = 0.0f;
#pragma unroll
      for (int e = 0; e < 4; ++e) da[e] = 0.0f;
    }
    const int buf = qn & 1;
    const bool landed = mbar_wait(bar0 + 8u * buf, (qn >> 1) & 1u, wc);
    if (!__syncthreads_and(landed)) {
      // copies into this buffer, and the next slab's into the other, may still be in flight
      if (threadIdx.x == 0) {
        drain_wait(bar0 + 8u * buf, (qn >> 1) & 1u);
        if (issued > qn + 1) drain_wait(bar0 + 8u * (buf ^ 1), ((qn + 1) >> 1) & 1u);
      }
      __syncthreads();
      ok = false;
      break;
    }
    // Every warp is past this slab's barrier, so it is done with the slab before: that buffer
    // takes the slab after this one (the first two went out at the start).
    if (warp == 0 && issued < qn + 2 && iss.t < a.total_items) {
      issue(iss, buf ^ 1);
      cursor_next(iss, a);
      ++issued;
    }
    {
      // this warp's contiguous range of the slab's super-chunks, and the group it starts in
      const int32_t sc_per_slab = L.KS / (64 * VW);
      const int32_t k0 = con.slab * L.KS;
      const int32_t n_sc = static_cast<int32_t>(((L.K - k0 < L.KS) ? L.K - k0 : L.KS) / (64 * VW));
      const int32_t lo = n_sc * warp / kMmaWarps, hi = n_sc * (warp + 1) / kMmaWarps;
      int32_t grp = (con.slab * sc_per_slab + lo) / sc_per_group;
      int32_t left = (grp + 1) * sc_per_group - (con.slab * sc_per_slab + lo);  // super-chunks to its end
      const uint32_t row_bytes = static_cast<uint32_t>(L.KS / 4 + 16 * VW);
      const uint32_t tile = ring_base + buf * buf_bytes;
      uint32_t rowa[R][2];  // shared-memory address of the thread's words in each of its rows
#pragma unroll
      for (int r = 0; r < R; ++r)
#pragma unroll
        for (int h = 0; h < 2; ++h) rowa[r][h] = tile + (16 * r + gid + 8 * h) * row_bytes + VW * q * 4;
      const uint4* xbase = reinterpret_cast<const uint4*>(xrow + k0 + 16 * VW * q);
      const bool every_sc = sc_per_group == 1;  // each super-chunk is a whole group
      const float* alpha = L.alpha;
      const float* mu = L.mu;
      auto load_x = [&](int32_t sc, uint4 (&xv)[2 * VW]) {
        const uint4* xp = xbase + sc * (8 * VW);
#pragma unroll
        for (int i = 0; i < 2 * VW; ++i) xv[i] = STAGED ? __ldcg(xp + i) : __ldg(xp + i);
      };
      // one super-chunk: this thread's code words from shared memory, its activations xv
      auto step = [&](int32_t sc, const uint4 (&xv)[2 * VW]) {
        const uint32_t woff = static_cast<uint32_t>(sc * 16 * VW);
        // The group (or this warp's range) ends with this super-chunk: its scales (and offsets)
        // are requested before the MMAs, which then cover their latency.
        const bool ends = every_sc || left == 1 || sc + 1 == hi;
        float av[R][2], mv[R][2];
        if (ends) {
#pragma unroll
          for (int r = 0; r < R; ++r) {
            av[r][0] = __ldg(alpha + goff[r][0] + grp);
            av[r][1] = __ldg(alpha + goff[r][1] + grp);
            if constexpr (MU) {
              mv[r][0] = __ldg(mu + goff[r][0] + grp);
              mv[r][1] = __ldg(mu + goff[r][1] + grp);
            }
          }
        }
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
        if (ends) {
#pragma unroll
          for (int r = 0; r < R; ++r) {
            acc[r][0] = fmaf(av[r][0], d[r][0] - da[0], acc[r][0]);
            acc[r][1] = fmaf(av[r][0], d[r][1] - da[1], acc[r][1]);
            acc[r][2] = fmaf(av[r][1], d[r][2] - da[0], acc[r][2]);
            acc[r][3] = fmaf(av[r][1], d[r][3] - da[1], acc[r][3]);
            if constexpr (MU) {
              acc[r][0] = fmaf(mv[r][0], da[2], acc[r][0]);
              acc[r][1] = fmaf(mv[r][0], da[3], acc[r][1]);
              acc[r][2] = fmaf(mv[r][1], da[2], acc[r][2]);
              acc[r][3] = fmaf(mv[r][1], da[3], acc[r][3]);
            }
#pragma unroll
            for (int e = 0; e < 4; ++e) d[r][e] = 0.0f;
          }
#pragma unroll
          for (int e = 0; e < 4; ++e) da[e] = 0.0f;
        }
        if (every_sc) {
          ++grp;
        } else if (--left == 0) {
          ++grp;
          left = sc_per_group;
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
    }
    ++qn;
    if (con.slab + 1 == L.nslabs) {
      // the token block's last slab: its partial sums meet in shared memory, in a fixed order
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
        if (con.b0 + tok < L.B && n0 + row < L.N)
          L.Y[(con.b0 + tok) * L.N + n0 + row] = static_cast<uint16_t>(pack_bf16x2(s, 0.0f) & 0xFFFFu);
      }
      // red is written again only after the next slab's barrier, which every thread reaches
      // after this loop
    }
    cursor_next(con, a);
  }
  if constexpr (STAGED) {
    // Arrive at the barriers still owed, then leave; the last CTA to leave (every other one has
    // passed all its waits by then) zeroes the counters for the next launch.
    __syncthreads();
    if (threadIdx.x == 0) {
      __threadfence();
      for (int32_t b = arrived; b < a.n_stages - 1; ++b) counter_arrive(a.sync + b);
      const uint32_t prev = atomicAdd(a.sync + kMaxInferStages, 1u);
      if (prev == gridDim.x - 1) {
        for (int32_t b = 0; b < a.n_stages - 1; ++b) a.sync[b] = 0u;
        a.sync[kMaxInferStages] = 0u;
        __threadfence();
      }
    }
  }
}

// One slab buffer: two per CTA plus the reduction array fit twice in an SM's shared memory.
constexpr int64_t kBufBytes = 46 * 1024;

// Bytes of one slab buffer for KS columns: 16 R rows of codes, each padded by 16 VW bytes.
int64_t slab_bytes(int64_t KS, int R, int VW) { return 16 * R * (KS / 4 + 16 * VW); }

// Code columns per slab for K: all of K when it fits one buffer, else the fewest equal slabs
// (multiples of 64 VW columns) that do.
int64_t slab_cols(int64_t K, int R, int VW) {
  const int64_t unit = 64 * VW;
  if (slab_bytes(K, R, VW) <= kBufBytes) return K;
  const int64_t cap = ((kBufBytes / (16 * R) - 16 * VW) * 4) / unit * unit;
  const int64_t nslabs = (K + cap - 1) / cap;
  return ((K + nslabs - 1) / nslabs + unit - 1) / unit * unit;
}

// stage_of (nullable): the stage of each layer (non-decreasing from 0 in steps of 1); sync: the
// staged launch's counters (zero on entry and on exit).
template <int R, int VW>
cudaError_t launch_mma(const InferDesc* ls, int n, int32_t g, bool with_mu, const int32_t* stage_of, uint32_t* sync,
                       cudaStream_t st) {
  WaitCtl wc;
  if (!launch_wait_ctl(&wc)) return cudaErrorInvalidDevice;
  InferArgs a{};
  a.n_layers = n;
  a.g = g;
  a.n_stages = stage_of ? stage_of[n - 1] + 1 : 1;
  a.sync = sync;
  int64_t items = 0, max_buf = 0;
  for (int i = 0; i < n; ++i) {
    InferLayer& L = a.L[i];
    L.codes = ls[i].codes;
    L.alpha = ls[i].alpha;
    L.mu = ls[i].mu;
    L.X = static_cast<const uint16_t*>(ls[i].X);
    L.Y = static_cast<uint16_t*>(ls[i].Y);
    L.N = ls[i].N;
    L.K = ls[i].K;
    L.B = ls[i].B;
    L.gpr = static_cast<int32_t>(ls[i].K / g);
    const int64_t KS = slab_cols(L.K, R, VW);
    L.KS = static_cast<int32_t>(KS);
    L.nslabs = static_cast<int32_t>((L.K + KS - 1) / KS);
    L.item0 = static_cast<int32_t>(items);
    items += (L.N + 16 * R - 1) / (16 * R);
    max_buf = std::max<int64_t>(max_buf, slab_bytes(KS, R, VW));
    if (stage_of) a.stage_end[stage_of[i]] = static_cast<int32_t>(std::min<int64_t>(items, INT32_MAX));
  }
  if (items >= (int64_t(1) << 31)) return cudaErrorInvalidValue;
  if (items == 0) return cudaSuccess;
  a.total_items = static_cast<int32_t>(items);
  if (!stage_of) a.stage_end[0] = a.total_items;
  int64_t widest = 0;  // most items of one stage
  for (int32_t s = 0, prev = 0; s < a.n_stages; prev = a.stage_end[s], ++s)
    widest = std::max<int64_t>(widest, a.stage_end[s] - prev);
  const int buf_bytes = static_cast<int>((max_buf + 127) / 128 * 128);
  const int smem = 2 * buf_bytes;
  int sm = 152;
  int dev = 0;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sm, cudaDevAttrMultiProcessorCount, dev);
  const bool staged = a.n_stages > 1;
  auto kern = staged ? (with_mu ? ternary_mma_kernel<R, VW, true, true> : ternary_mma_kernel<R, VW, false, true>)
                     : (with_mu ? ternary_mma_kernel<R, VW, true, false> : ternary_mma_kernel<R, VW, false, false>);
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  int64_t blocks = std::min<int64_t>(items, 2 * static_cast<int64_t>(sm));
  cudaLaunchConfig_t cfg{};
  cudaLaunchAttribute attr[1];
  if (staged) {
    // every CTA must be resident at once (they wait on each other): a cooperative launch of
    // at most the co-resident CTAs, and no more than the widest stage has items
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kMmaWarps * 32, static_cast<size_t>(smem));
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    blocks = std::min<int64_t>(widest, static_cast<int64_t>(per_sm) * sm);
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
  } else {
    // programmatic dependent launch: this kernel may start while the previous one in the
    // stream finishes (see grid_dependency_wait in the kernel)
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
  }
  cfg.gridDim = dim3(static_cast<unsigned>(blocks));
  cfg.blockDim = dim3(kMmaWarps * 32);
  cfg.dynamicSmemBytes = static_cast<size_t>(smem);
  cfg.stream = st;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, a, buf_bytes, wc);
}

template <int R>
cudaError_t launch_rows(const InferDesc* ls, int n, int32_t g, bool with_mu, const int32_t* stage_of, uint32_t* sync,
                        cudaStream_t st) {
  if (g % 128 == 0) return launch_mma<R, 2>(ls, n, g, with_mu, stage_of, sync, st);
  return launch_mma<R, 1>(ls, n, g, with_mu, stage_of, sync, st);
}

// 16-row tiles per work item (1 or 2: more hold more registers than two CTAs per SM allow
// without spills): the fewest rows on the busiest SM summed over the stages (two persistent
// CTAs per SM), then the most tiles per item (the correction MMAs and the activation
// preparation serve more rows).
int pick_rows(const InferDesc* ls, int n, const int32_t* stage_of) {
  int sm = 152;
  {
    int dev = 0;
    if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sm, cudaDevAttrMultiProcessorCount, dev);
  }
  int best = 1;
  int64_t best_rows = -1;
  for (int r = 1; r <= 2; ++r) {
    int64_t busiest = 0, items = 0;
    for (int i = 0; i < n; ++i) {
      items += (ls[i].N + 16 * r - 1) / (16 * r);
      if (i + 1 == n || (stage_of && stage_of[i + 1] != stage_of[i])) {
        busiest += (items + 2 * sm - 1) / (2 * sm) * 16 * r;
        items = 0;
      }
    }
    if (best_rows < 0 || busiest <= best_rows) {
      best = r;
      best_rows = busiest;
    }
  }
  return best;
}

cudaError_t launch_infer(const InferDesc* ls, int n, int32_t g, const int32_t* stage_of, uint32_t* sync,
                         cudaStream_t st) {
  if (n < 1 || n > kMaxInferLayers) return cudaErrorInvalidValue;
  const bool with_mu = ls[0].mu != nullptr;
  for (int i = 1; i < n; ++i)
    if ((ls[i].mu != nullptr) != with_mu) return cudaErrorInvalidValue;
  if (stage_of) {
    if (stage_of[0] != 0 || !sync) return cudaErrorInvalidValue;
    for (int i = 1; i < n; ++i)
      if (stage_of[i] != stage_of[i - 1] && stage_of[i] != stage_of[i - 1] + 1) return cudaErrorInvalidValue;
    if (stage_of[n - 1] + 1 > kMaxInferStages) return cudaErrorInvalidValue;
  }
  if (pick_rows(ls, n, stage_of) == 2) return launch_rows<2>(ls, n, g, with_mu, stage_of, sync, st);
  return launch_rows<1>(ls, n, g, with_mu, stage_of, sync, st);
}

}  // namespace

int ternary_infer_max_layers() { return kMaxInferLayers; }

cudaError_t launch_ternary_infer_batched(const InferDesc* ls, int n, int32_t g, cudaStream_t st) {
  return launch_infer(ls, n, g, nullptr, nullptr, st);
}

int ternary_infer_max_stages() { return kMaxInferStages; }
size_t ternary_infer_sync_bytes() { return (kMaxInferStages + 1) * sizeof(uint32_t); }

cudaError_t launch_ternary_infer_staged(const InferDesc* ls, int n, const int32_t* stage_of, int32_t g, uint32_t* sync,
                                        cudaStream_t st) {
  if (!stage_of) return cudaErrorInvalidValue;
  return launch_infer(ls, n, g, stage_of, sync, st);
}

cudaError_t launch_ternary_infer(const uint8_t* codes, const float* alpha, const float* mu, int64_t N, int64_t K,
                                 int32_t g, const void* X, int64_t B, void* Y, cudaStream_t st) {
  const InferDesc d{codes, alpha, mu, N, K, X, B, Y};
  return launch_ternary_infer_batched(&d, 1, g, st);
}

}  // namespace catq
