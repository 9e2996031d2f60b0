// tc_gemm.cu — bf16 tensor-core contractions of the soft-ternary linear on sm_100-class
// GPUs (tcgen05 MMA with TMEM accumulators, TMA-fed, warp-specialised, persistent).
//
// fused_gemm_kernel  C[M, ncols] = A[M, depth] * Wq-operand, with the Eq. 3/5/6 weight
//                    (modulation, transition function, scale alpha) computed by producer
//                    warps on raw W tiles that TMA lands in their own ring, in place, in
//                    the 128-byte-swizzled layout the MMA reads.  Wq never reaches HBM.
//                    A tiles flow TMA -> MMA in a separate ring, off the producers' path.
//                      forward:  A = X  [M, K],  operand = Wq   (K-major), C = Y  [M, N]
//                      dX:       A = dY [M, N],  operand = Wq   (MN-major), C = dX [M, K]
//                    Two M-tiles share each produced operand tile (two accumulators).
// dw_kernel          G = dY^T X accumulated in TMEM (both operands MN-major, straight from
//                    TMA); the epilogue applies the chain rule of Eq. 3/5/6 per element
//                    and reduces each row's columns into per-group partial sums.  G is never
//                    written to memory.
//
// CG = 1: one CTA per tile (MMA M = 128).  CG = 2: a CTA pair (cluster of 2) computes one
// tile with tcgen05 cta_group::2 (MMA M = 256), each CTA holding half of the operand
// columns; only the even CTA issues MMAs.
//
// Every mbarrier wait is bounded (ptx_sm100.cuh); on expiry the launch latches
// CATQ_ERR_TIMEOUT, every role leaves its loop, in-flight copies and MMAs are drained
// with bounded waits, and TMEM is freed before the kernel returns.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <atomic>
#include <map>
#include <mutex>
#include <numeric>
#include <type_traits>

#include "launch.h"
#include "ptx_sm100.cuh"

namespace catq {

__device__ uint32_t g_abort_word;
__device__ int32_t g_status_word;

namespace {

constexpr int BK = 64;    // contraction elements per pipeline stage (one 128-byte row)
constexpr int BN = 256;   // MMA N
constexpr int NACC = 2;   // accumulators sharing one produced operand tile (fused kernel)
constexpr uint32_t kTmemCols = 512;
constexpr uint64_t kWaitTimeoutNs = 4000000000ull;
constexpr uint64_t kDrainTimeoutNs = 200000000ull;

constexpr int gcd_c(int a, int b) { return b == 0 ? a : gcd_c(b, a % b); }

// PAIRS == 2 runs clusters of four CTAs: two CTA pairs compute adjacent 512-row M tiles
// against the same produced operand tiles; each pair produces every other stage and sends
// its transformed half-tiles to the other pair's CTAs through distributed shared memory,
// which halves the per-SM transform work.
template <int CG, int PAIRS = 1>
struct FusedCfg {
  static_assert(PAIRS == 1 || CG == 2, "pairs of pairs need CTA pairs");
  static constexpr int kClusterCtas = CG * PAIRS;
  static constexpr int kRowsPerAcc = 128 * CG;          // MMA M
  static constexpr int kTileRows = kRowsPerAcc * NACC;  // rows of C per pair per tile
  static constexpr int kBRows = BN / CG;                // 128-byte operand rows per CTA per stage
  static constexpr int kABytes = NACC * 128 * BK * 2;   // this CTA's A rows per stage
  static constexpr int kWBytes = kBRows * BK * 2;       // this CTA's operand rows per stage
  static constexpr int kStagesA = CG == 1 ? 3 : 4;      // A ring: TMA -> MMA
  // W ring: TMA -> producers (in place) -> MMA.  Even with two pairs, so every slot is always
  // produced by the same pair (and received by the other).
  static constexpr int kStagesW = PAIRS == 2 ? 6 : (CG == 1 ? 3 : 5);
  static constexpr int kEpiWarps = 4;
  // Two groups of 8 producer warps take alternate stages (of the ones this CTA produces), so
  // each group has two stage periods per operand tile and the groups' MUFU work interleaves.
  static constexpr int kProdGroups = 2;
  static constexpr int kGroupWarps = 8;
  static constexpr int kProdWarps = kProdGroups * kGroupWarps;
  static constexpr int kGroupThreads = 32 * kGroupWarps;
  static constexpr int kThreadsPerRow = kGroupThreads / kBRows;  // 1 (CG 1) or 2 (CG 2)
  static constexpr int kChunksPerThread = 8 / kThreadsPerRow;    // 16-byte chunks of a 128-byte row
  static constexpr int kThreads = 32 * (kEpiWarps + 2 + kProdWarps);
  // Stage q lands on the raw-W barrier of its producer group and slot; that barrier sees one
  // stage in every kRawPeriod, so each group waits on its own barriers strictly in phase
  // order (one barrier per slot shared by the groups would let a group running a full phase
  // ahead read the parity of the other group's pending phase as complete).
  static constexpr int kStep = kProdGroups * PAIRS;  // stages between two of a group's stages
  static constexpr int kRawPeriod = kStagesW / gcd_c(kStagesW, kStep) * kStep;
  static constexpr int kRawBars = kProdGroups * kStagesW;
  static_assert(kRawBars <= 32, "issued-barrier masks are 32 bits");
  static constexpr int kRowsPerWarp = 32 / kThreadsPerRow;     // operand rows one producer warp owns
  static constexpr int kBarBytes = 8 * (2 * kStagesA + kRawBars + 3 * kStagesW + 2 * NACC + 1) + 16;
  static constexpr int kSmemBytes = kStagesA * kABytes + kStagesW * kWBytes + 1024 + kBarBytes;
  // Stages the MMA issuer holds at a tile's edges (see the issuer), bounded by both rings.
  static constexpr int kHold = (kStagesA < kStagesW ? kStagesA : kStagesW) - 1;
};

template <int CG>
struct DwCfg {
  static constexpr int kRowsPerCta = 128;    // G rows (n) per CTA
  static constexpr int kTileRows = 128 * CG; // MMA M
  static constexpr int kBCols = BN / CG;     // G columns (k) whose X slice this CTA loads
  static constexpr int kABytes = 128 * BK * 2;
  static constexpr int kBBytes = kBCols * BK * 2;
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kStages = CG == 1 ? 4 : 6;
  static constexpr int kEpiWarps = 8;        // two warps per TMEM lane quarter (column halves)
  static constexpr int kThreads = 32 * (kEpiWarps + 2);
  static constexpr int kBarBytes = 8 * (2 * kStages + 5) + 16;
  static constexpr int kSmemBytes = kStages * kStageBytes + 1024 + kBarBytes;
};

// Experts of one grouped launch (stacked expert weights, expert-sorted rows).
constexpr int kMaxGroupExperts = kGroupedMaxExperts;

struct FusedArgs {
  LayerDev L;
  StepScalars sc;
  void* C;          // [M, ncols], bf16 (fp32 when c_f32); nullable in the fused-loss epilogue
  int32_t c_f32;
  // Per-row scale of the accumulator (nullable): C row m = row_scale[m] * (A Wq^T)[m], the
  // per-token scale of 8-bit activation codes in A.
  const float* row_scale;
  // Fused reconstruction loss (Eq. 7) when yref is set: the epilogue forms d = Y - Y_ref from
  // the fp32 accumulator, writes dY = dscale d (bf16) and sums d^2 into one partial per
  // epilogue warp, loss_part[blockIdx.x * kEpiWarps + warp].
  const void* yref;  // [M, ncols] bf16, or fp32 when yref_f32
  int32_t yref_f32;
  float dscale;
  uint16_t* dY;      // bf16 [M, ncols]
  double* loss_part;
  int64_t M;        // rows of A and C
  int64_t ncols;    // columns of C
  int32_t num_m_tiles, num_n_tiles, num_k_blocks;
  int32_t group_m;  // M blocks per raster group
  int32_t a_keep;   // a raster group's A rows fit L2 comfortably: keep them (evict_last), stream W
  WaitCtl wc;
  // Grouped launches (E > 0): expert e owns rows [row0[e], row0[e+1]) of A and C, W rows
  // [e N, (e+1) N) of the stacked weights, operand constants from float e * const_stride
  // on, and tiles [tile0[e], tile0[e+1]) (its M blocks, then N blocks).
  int32_t E;
  int64_t const_stride;
  int32_t tile0[kMaxGroupExperts + 1];
  int32_t row0[kMaxGroupExperts + 1];
};

// Tile t of a persistent sequence: its M and N block, expert, first row and row limit.
struct TileInfo {
  int m_blk, n_blk, e;
  int64_t row0, row_end;
};

// Dense: tiles run in groups of group_m M blocks (inside a group the M block varies fastest,
// then the N block).  Grouped: the expert is found by binary search over its first tiles;
// inside an expert the M block varies fastest.
__device__ __forceinline__ TileInfo tile_info(const FusedArgs& a, int t, int rows_per_tile) {
  TileInfo ti;
  if (a.E == 0) {
    const int per_group = a.group_m * a.num_n_tiles;
    const int grp = t / per_group, r = t - grp * per_group;
    const int gm = min(a.group_m, a.num_m_tiles - grp * a.group_m);
    ti.m_blk = grp * a.group_m + r % gm;
    ti.n_blk = r / gm;
    ti.e = 0;
    ti.row0 = (int64_t)ti.m_blk * rows_per_tile;
    ti.row_end = a.M;
    return ti;
  }
  int lo = 0, hi = a.E;  // last e with tile0[e] <= t
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (a.tile0[mid] <= t) lo = mid;
    else hi = mid;
  }
  const int r0 = a.row0[lo], r1 = a.row0[lo + 1];
  const int mt = (r1 - r0 + rows_per_tile - 1) / rows_per_tile;
  const int local = t - a.tile0[lo];
  ti.e = lo;
  ti.m_blk = local % mt;
  ti.n_blk = local / mt;
  ti.row0 = r0 + (int64_t)ti.m_blk * rows_per_tile;
  ti.row_end = r1;
  return ti;
}

struct DwArgs {
  LayerDev L;
  StepScalars sc;
  float* part;      // [splits][3][N][K/P]; grouped: [E][3][N][K/P]
  int64_t M;
  int32_t splits, P, kb_per_split, kb_total;
  int32_t num_n_tiles, num_k_tiles;
  WaitCtl wc;
  int32_t n_experts;  // grouped: experts of this launch (0: dense)
  int32_t x_keep;     // X (the contraction's K side) fits L2 comfortably: keep it (evict_last)
  int32_t k_group;    // raster: k blocks per group (see dw_tile)
};

// Tile r of a split (or expert) of the dW launch: its n block and k block.  Tiles run in groups
// of k_group k blocks; inside a group the k block varies fastest, then the n block.  A wave of
// C clusters then covers about C / k_group n blocks x k_group k blocks, so it reads
// (C / k_group + k_group) column slices of dY and X (M x 256 each) instead of all of X's, which
// k-fastest order over the whole K reads every wave.
__device__ __forceinline__ void dw_tile(const DwArgs& a, int r, int& n_blk, int& k_blk) {
  const int per_group = a.k_group * a.num_n_tiles;
  const int gi = r / per_group, rr = r - gi * per_group;
  const int kw = min(a.k_group, a.num_k_tiles - gi * a.k_group);
  n_blk = rr / kw;
  k_blk = gi * a.k_group + rr % kw;
}

// Grouped dW launch: up to kDwGroupExperts experts with rows, each with tensor maps over its
// own rows of dY and X (so the contraction stops at the expert's last row: rows past it
// read as zeros), its index in the stacked layer and its row count.
constexpr int kDwGroupExperts = 64;
template <int NE>
struct DwMaps {
  CUtensorMap dy[NE];
  CUtensorMap x[NE];
  int32_t expert[NE];
  int32_t rows[NE];
};

// Wait that ignores the abort flag (used to drain work already issued).
__device__ __forceinline__ bool mbar_wait_drain(uint32_t bar, uint32_t parity) {
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity))
    if (globaltimer_ns() - t0 > kDrainTimeoutNs) return false;
  return true;
}

// 32 fp32 accumulator columns of one row per lane (32 rows per warp, 32 consecutive columns
// from `col`) stored as bf16.  A 4 x 4 transpose of 16-byte chunks inside each group of four
// lanes (two xor-shuffle rounds) turns the lane-per-row layout into stores where four lanes
// cover 64 contiguous bytes of one row, so each store instruction writes 8 row segments
// instead of touching 32 rows.  ncols is a multiple of 8, so a chunk is wholly in or out.
__device__ __forceinline__ void store_rows_bf16x32(uint16_t* C, int64_t M, int64_t ncols, int64_t row0, int64_t col,
                                                   const uint32_t (&r)[32], int lane) {
  uint4 v[4];
#pragma unroll
  for (int p = 0; p < 4; ++p) {
    v[p].x = pack_bf16x2(__uint_as_float(r[8 * p + 0]), __uint_as_float(r[8 * p + 1]));
    v[p].y = pack_bf16x2(__uint_as_float(r[8 * p + 2]), __uint_as_float(r[8 * p + 3]));
    v[p].z = pack_bf16x2(__uint_as_float(r[8 * p + 4]), __uint_as_float(r[8 * p + 5]));
    v[p].w = pack_bf16x2(__uint_as_float(r[8 * p + 6]), __uint_as_float(r[8 * p + 7]));
  }
  // Round k exchanges chunk pairs (p, p | k) with lane ^ k; afterwards lane 4a + i holds
  // chunk i of rows 4a .. 4a + 3 in v[0 .. 3].
#pragma unroll
  for (int k = 1; k <= 2; k <<= 1) {
    const bool upper = (lane & k) != 0;
#pragma unroll
    for (int p = 0; p < 4; ++p) {
      if (p & k) continue;
      const uint4 send = upper ? v[p] : v[p | k];
      uint4 got;
      got.x = __shfl_xor_sync(0xffffffffu, send.x, k);
      got.y = __shfl_xor_sync(0xffffffffu, send.y, k);
      got.z = __shfl_xor_sync(0xffffffffu, send.z, k);
      got.w = __shfl_xor_sync(0xffffffffu, send.w, k);
      if (upper) v[p] = got;
      else v[p | k] = got;
    }
  }
  const int64_t c = col + 8 * (lane & 3);
  if (c >= ncols) return;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const int64_t row = row0 + (lane & ~3) + j;
    if (row < M) *reinterpret_cast<uint4*>(C + row * ncols + c) = v[j];
  }
}

// 16 bf16 values of one row per lane (32 rows per warp, columns from `col`, as two 16-byte
// vectors) stored through a 2 x 2 transpose of the vectors between lane pairs (one
// xor-shuffle round), so that two lanes store 32 contiguous bytes of one row.
__device__ __forceinline__ void store_rows_packed16(uint16_t* C, int64_t M, int64_t ncols, int64_t row0, int64_t col,
                                                    uint4 (&v)[2], int lane) {
  // lane 2a + i ends with chunk i of rows 2a, 2a + 1 in v[0], v[1]
  const bool upper = (lane & 1) != 0;
  const uint4 send = upper ? v[0] : v[1];
  uint4 got;
  got.x = __shfl_xor_sync(0xffffffffu, send.x, 1);
  got.y = __shfl_xor_sync(0xffffffffu, send.y, 1);
  got.z = __shfl_xor_sync(0xffffffffu, send.z, 1);
  got.w = __shfl_xor_sync(0xffffffffu, send.w, 1);
  if (upper) v[0] = got;
  else v[1] = got;
  const int64_t c = col + 8 * (lane & 1);
  if (c >= ncols) return;
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    const int64_t row = row0 + (lane & ~1) + j;
    if (row < M) *reinterpret_cast<uint4*>(C + row * ncols + c) = v[j];
  }
}

// 16 fp32 accumulator columns of one row per lane stored as bf16 (store_rows_packed16).
__device__ __forceinline__ void store_rows_bf16x16(uint16_t* C, int64_t M, int64_t ncols, int64_t row0, int64_t col,
                                                   const uint32_t (&r)[16], int lane) {
  uint4 v[2];
#pragma unroll
  for (int p = 0; p < 2; ++p) {
    v[p].x = pack_bf16x2(__uint_as_float(r[8 * p + 0]), __uint_as_float(r[8 * p + 1]));
    v[p].y = pack_bf16x2(__uint_as_float(r[8 * p + 2]), __uint_as_float(r[8 * p + 3]));
    v[p].z = pack_bf16x2(__uint_as_float(r[8 * p + 4]), __uint_as_float(r[8 * p + 5]));
    v[p].w = pack_bf16x2(__uint_as_float(r[8 * p + 6]), __uint_as_float(r[8 * p + 7]));
  }
  store_rows_packed16(C, M, ncols, row0, col, v, lane);
}

// 16 fp32 values of one row per lane (row < M, columns from `col`) stored as fp32: four
// 16-byte stores per lane (used for a full-precision teacher output, off the hot path).
__device__ __forceinline__ void store_row_f32x16(float* C, int64_t M, int64_t ncols, int64_t row, int64_t col,
                                                 const uint32_t (&r)[16]) {
  if (row >= M) return;
#pragma unroll
  for (int p = 0; p < 4; ++p)
    if (col + 4 * p < ncols)
      *reinterpret_cast<float4*>(C + row * ncols + col + 4 * p) =
          make_float4(__uint_as_float(r[4 * p]), __uint_as_float(r[4 * p + 1]), __uint_as_float(r[4 * p + 2]),
                      __uint_as_float(r[4 * p + 3]));
}

// The teacher output of one row's 16 columns from `col` (bf16), as two 16-byte vectors;
// chunks outside the row's columns, and rows past the end, read as 0.
__device__ __forceinline__ void load_yref_bf16x16(const uint16_t* Yr, int64_t ncols, int64_t row, bool row_ok,
                                                  int64_t col, uint4 (&v)[2]) {
#pragma unroll
  for (int p = 0; p < 2; ++p) {
    v[p] = make_uint4(0u, 0u, 0u, 0u);
    if (row_ok && col + 8 * p < ncols) v[p] = __ldg(reinterpret_cast<const uint4*>(Yr + row * ncols + col + 8 * p));
  }
}

// ============================================================================ fused kernel

// Walks the pipeline stages one producer thread handles (every kProdGroups-th stage of its
// CTA's tile sequence) and tracks which W row, K chunk and group its 128-byte operand row
// holds, the group as its index into the [K/g][N] operand-constant array.  Divisions happen
// once per tile; each stage step is a few integer adds.
template <int CG, bool B_MN, int PAIRS>
struct OperandRowIter {
  using Cfg = FusedCfg<CG, PAIRS>;
  int t, kb;      // tile index, k block
  int64_t n, kc;  // W row (within its expert), first K column of the 64-element chunk
  int64_t ci;     // operand-constant index of (n, kc): (kc / g) * N + n, in float4 units from
                  // the launch's first expert's constants
  int64_t mi;     // the same entry's index into the mu plane (floats)
  int kin;        // forward: k blocks into the current group (kc / 64 mod g / 64)
  bool tile_ok;   // forward: n < N; dX: kc < K

  __device__ __forceinline__ void init(const FusedArgs& a, uint32_t cta, int row, int t_, int kb_) {
    t = t_;
    kb = kb_;
    const TileInfo ti = tile_info(a, t, Cfg::kTileRows * PAIRS);
    const int gk = a.L.g / BK;  // k blocks per group
    int64_t local;
    if constexpr (!B_MN) {
      n = (int64_t)ti.n_blk * BN + cta * Cfg::kBRows + row;
      kc = (int64_t)kb * BK;
      tile_ok = n < a.L.N;
      local = (int64_t)(kb / gk) * a.L.N + n;
      kin = kb % gk;
    } else {
      n = (int64_t)kb * BK + (row & 63);
      kc = (int64_t)ti.n_blk * BN + cta * Cfg::kBRows + 64 * (row >> 6);
      tile_ok = kc < a.L.K;
      local = (kc / a.L.g) * a.L.N + n;
      kin = 0;
    }
    ci = (ti.e * a.const_stride) / 4 + local;
    mi = ti.e * a.const_stride + local;
  }

  __device__ __forceinline__ bool live(const FusedArgs& a, int num_tiles) const { return t < num_tiles; }
  __device__ __forceinline__ bool valid(const FusedArgs& a) const {
    if constexpr (!B_MN) return tile_ok;
    else return tile_ok && n < a.L.N;
  }

  __device__ __forceinline__ void step(const FusedArgs& a, uint32_t cta, int row, uint32_t nclusters, int steps) {
    kb += steps;
    if (kb >= a.num_k_blocks) {
      int t2 = t, kb2 = kb;
      while (kb2 >= a.num_k_blocks) {
        kb2 -= a.num_k_blocks;
        t2 += nclusters;
      }
      init(a, cta, row, t2, kb2);
      return;
    }
    if constexpr (!B_MN) {
      kc += (int64_t)steps * BK;
      kin += steps;
      const int gk = a.L.g / BK;
      while (kin >= gk) {
        kin -= gk;
        ci += a.L.N;
        mi += a.L.N;
      }
    } else {
      n += (int64_t)steps * BK;
      ci += (int64_t)steps * BK;
      mi += (int64_t)steps * BK;
    }
  }
};

// MU: the layer reconstructs W ~ alpha T + mu (a separate instantiation, so the W ~ alpha T
// kernel carries none of its work).  EPI: 0 stores C in bf16; 1 is the general epilogue
// (row scale, fp32 C, fused loss), a separate instantiation so the plain forward and dX
// keep their register allocation.
template <int CG, bool B_MN, int PAIRS, bool MU, int EPI = 0>
__global__ void __launch_bounds__(FusedCfg<CG, PAIRS>::kThreads, 1)
    fused_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmW,
                      const FusedArgs args) {
  using Cfg = FusedCfg<CG, PAIRS>;
  constexpr int SA = Cfg::kStagesA, SW = Cfg::kStagesW;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_addr = smem_u32(smem_raw);
  const uint32_t base = (raw_addr + 1023u) & ~1023u;
  uint8_t* base_ptr = smem_raw + (base - raw_addr);
  const uint32_t a_base = base;                                // [SA][kABytes]
  const uint32_t w_base = base + SA * Cfg::kABytes;            // [SW][kWBytes]
  const uint32_t bars = w_base + SW * Cfg::kWBytes;
  auto full_a = [&](int s) { return bars + 8u * s; };                   // A landed (pair: even CTA)
  auto empty_a = [&](int s) { return bars + 8u * (SA + s); };           // A consumed by the MMA
  constexpr int RB = Cfg::kRawBars;
  auto raw_w = [&](int b) { return bars + 8u * (2 * SA + b); };          // raw W landed [group][slot] (local)
  auto full_w = [&](int s) { return bars + 8u * (2 * SA + RB + s); };   // operand ready (pair: even CTA)
  auto empty_w = [&](int s) { return bars + 8u * (2 * SA + RB + SW + s); };
  auto recv_w = [&](int s) { return bars + 8u * (2 * SA + RB + 2 * SW + s); };  // PAIRS 2: received half landed
  // one full/empty pair per accumulator: a tile's accumulators drain and refill separately
  const uint32_t tmem_full0 = bars + 8u * (2 * SA + RB + 3 * SW);     // [NACC]
  const uint32_t tmem_empty0 = tmem_full0 + 8u * NACC;                // [NACC]
  const uint32_t final_bar = tmem_empty0 + 8u * NACC;
  uint32_t* tmem_slot =
      reinterpret_cast<uint32_t*>(base_ptr + (bars - base) + 8 * (2 * SA + RB + 3 * SW + 2 * NACC + 1));

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = CG == 2 ? cluster_ctarank() : 0u;
  const uint32_t cta = rank & 1u;                // half of the pair
  const uint32_t pair = rank >> 1;               // pair within the cluster (PAIRS 2)
  const uint32_t leader = rank & ~1u;            // the pair's MMA-issuing CTA
  const uint32_t cluster = CG == 2 ? cluster_id_x() : blockIdx.x;
  const uint32_t nclusters = CG == 2 ? num_clusters_x() : gridDim.x;
  const WaitCtl& wc = args.wc;
  const int num_tiles = args.num_m_tiles * args.num_n_tiles;
  constexpr int kTmaWarp = Cfg::kEpiWarps, kMmaWarp = Cfg::kEpiWarps + 1;
  // does this CTA produce stage q (PAIRS 1: always)
  auto produces = [&](uint32_t q) { return PAIRS == 1 || (q & 1u) == pair; };

  if (threadIdx.x == 0) {
    for (int s = 0; s < SA; ++s) {
      mbar_init(full_a(s), 1);
      mbar_init(empty_a(s), 1);
    }
    for (int b = 0; b < RB; ++b) mbar_init(raw_w(b), 1);
    for (int s = 0; s < SW; ++s) {
      // With two pairs, slot s is always produced by pair s & 1 (the ring depth is even).
      const bool received = PAIRS == 2 && (static_cast<uint32_t>(s) & 1u) != pair;
      // Produced slots: one arrival per producer warp of the pair.  Received slots: the even
      // CTA's half lands on full_w itself (the copies complete their bytes there), which the
      // MMA thread arms, plus one arrival from the odd CTA once its half has landed.
      mbar_init(full_w(s), received ? 2 : Cfg::kGroupWarps * CG);
      mbar_init(empty_w(s), PAIRS);  // every pair's MMA frees the slot in all CTAs
      mbar_init(recv_w(s), 1);       // odd CTA: its received half landed
      // Barriers that count received bytes are armed for a slot's next use as soon as its
      // current use has landed; this arms the first use.
      if (received) mbar_arrive_expect_tx(cta == 0 ? full_w(s) : recv_w(s), Cfg::kWBytes);
    }
    for (int a = 0; a < NACC; ++a) {
      mbar_init(tmem_full0 + 8u * a, 1);
      mbar_init(tmem_empty0 + 8u * a, Cfg::kEpiWarps * CG);
    }
    mbar_init(final_bar, 1);
    fence_mbar_init_cluster();
  }
  if (warp == kMmaWarp) tmem_alloc<CG>(smem_u32(tmem_slot), kTmemCols);
  if (warp == kTmaWarp && lane == 0) {
    prefetch_tmap(&tmA);
    prefetch_tmap(&tmW);
  }
  tc_fence_before();
  if constexpr (CG == 2) cluster_sync_all(); else __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  // Barriers a whole pair signals live in the pair's even CTA.
  const uint32_t leader_full_a0 = CG == 2 ? mapa_shared(full_a(0), leader) : full_a(0);
  const uint32_t leader_full_w0 = CG == 2 ? mapa_shared(full_w(0), leader) : full_w(0);
  const uint32_t leader_tmem_empty0 = CG == 2 ? mapa_shared(tmem_empty0, leader) : tmem_empty0;
  const uint16_t pair_mask = static_cast<uint16_t>(3u << (2 * pair));
  const uint16_t all_mask = static_cast<uint16_t>((1u << Cfg::kClusterCtas) - 1u);

  if (warp == kTmaWarp) {
    if (lane == 0) {
      // ---------------------------------------------------------- TMA: A tiles (to the MMA)
      // A raster group's A rows are read by every tile wave of the group: kept in L2 ahead of
      // the streamed W tiles when they fit comfortably (args.a_keep).
      const uint64_t pol_a = args.a_keep ? l2_policy_evict_last() : l2_policy_evict_normal();
      uint32_t q = 0, issued_mask = 0, issued_phase = 0;
      bool ok = true;
      for (int t = cluster; ok && t < num_tiles; t += nclusters) {
        const TileInfo ti = tile_info(args, t, Cfg::kTileRows * PAIRS);
        const int32_t m0 = static_cast<int32_t>(ti.row0) + pair * Cfg::kTileRows;
        for (int kb = 0; kb < args.num_k_blocks; ++kb, ++q) {
          const uint32_t s = q % SA, ph = (q / SA) & 1u;
          if (!mbar_wait(empty_a(s), ph ^ 1u, wc)) { ok = false; break; }
          if (cta == 0) mbar_arrive_expect_tx(full_a(s), Cfg::kABytes * CG);
          const uint32_t dst = a_base + s * Cfg::kABytes, fb = leader_full_a0 + 8u * s;
#pragma unroll
          for (int acc = 0; acc < NACC; ++acc) {
            const int32_t row = m0 + acc * Cfg::kRowsPerAcc + cta * 128;
            if constexpr (CG == 1) tma_load_2d_hint(dst + acc * (128 * BK * 2), &tmA, fb, kb * BK, row, pol_a);
            else tma_load_2d_pair_hint(dst + acc * (128 * BK * 2), &tmA, fb, kb * BK, row, pol_a);
          }
          issued_mask |= 1u << s;
          issued_phase = (issued_phase & ~(1u << s)) | (ph << s);
        }
      }
      if (cta == 0)
        for (int s = 0; s < SA; ++s)
          if (issued_mask & (1u << s)) mbar_wait_drain(full_a(s), (issued_phase >> s) & 1u);
    } else if (lane == 1) {
      // ---------------------------------------------------------- TMA: raw W tiles this CTA produces
      // (a W tile serves the raster group's M blocks at about the same time, then is done)
      const uint64_t pol_w = args.a_keep ? l2_policy_evict_first() : l2_policy_evict_normal();
      uint32_t q = 0, issued_mask = 0, issued_phase = 0;
      bool ok = true;
      for (int t = cluster; ok && t < num_tiles; t += nclusters) {
        const TileInfo ti = tile_info(args, t, Cfg::kTileRows * PAIRS);
        const int32_t n0 = ti.n_blk * BN + cta * Cfg::kBRows;
        const int32_t wrow = static_cast<int32_t>(ti.e * args.L.N);  // the expert's first W row
        for (int kb = 0; kb < args.num_k_blocks; ++kb, ++q) {
          if (!produces(q)) continue;
          const uint32_t s = q % SW, ph = (q / SW) & 1u;
          const uint32_t rb = ((q / PAIRS) % Cfg::kProdGroups) * SW + s;  // the producing group's barrier
          const uint32_t rph = (q / Cfg::kRawPeriod) & 1u;
          if (!mbar_wait(empty_w(s), ph ^ 1u, wc)) { ok = false; break; }
          mbar_arrive_expect_tx(raw_w(rb), Cfg::kWBytes);
          const uint32_t dst = w_base + s * Cfg::kWBytes;
          if constexpr (!B_MN) {
            tma_load_2d_hint(dst, &tmW, raw_w(rb), kb * BK, wrow + n0, pol_w);
          } else {
#pragma unroll
            for (int b = 0; b < Cfg::kBRows / 64; ++b)
              tma_load_2d_hint(dst + b * 8192, &tmW, raw_w(rb), n0 + 64 * b, wrow + kb * BK, pol_w);
          }
          issued_mask |= 1u << rb;
          issued_phase = (issued_phase & ~(1u << rb)) | (rph << rb);
        }
      }
      for (int b = 0; b < RB; ++b)
        if (issued_mask & (1u << b)) mbar_wait_drain(raw_w(b), (issued_phase >> b) & 1u);
    }
  } else if (warp == kMmaWarp) {
    // ------------------------------------------------------------ MMA issuer (even CTA of each pair)
    if (cta == 0 && lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(Cfg::kRowsPerAcc, BN, false, B_MN);
      const int T = args.num_k_blocks;
      // Accumulators drain and refill separately, so the epilogue overlaps the MMAs: a tile's
      // last J stages run accumulator 0 first (the epilogue drains it while accumulator 1
      // finishes), and the next tile's first J stages start accumulator 0 as soon as it is
      // drained (accumulator 1 follows once it is).  Those stages stay held in between.
      const int J = min(Cfg::kHold, T / 2);
      uint32_t q = 0, it = 0;
      bool ok = true;
      auto stage_in = [&](uint32_t qq) -> bool {  // wait for stage qq; arm a received slot's next use
        const uint32_t sa = qq % SA, pa = (qq / SA) & 1u, sw = qq % SW, pw = (qq / SW) & 1u;
        if (!mbar_wait(full_a(sa), pa, wc) || !mbar_wait(full_w(sw), pw, wc)) return false;
        if (PAIRS == 2 && (qq & 1u) != pair) mbar_arrive_expect_tx(full_w(sw), Cfg::kWBytes);
        tc_fence_after();
        return true;
      };
      // An accumulator whose rows all lie past the tile's last row (an expert's short last M
      // block, or a ragged M) gets no MMAs; the epilogue stores nothing from it.
      bool live[NACC] = {};
      auto issue = [&](uint32_t qq, int acc, bool first) {  // one accumulator's MMAs of stage qq
        if (!live[acc]) return;
        const uint32_t aa = a_base + (qq % SA) * Cfg::kABytes, ww = w_base + (qq % SW) * Cfg::kWBytes;
#pragma unroll
        for (int kk = 0; kk < BK / 16; ++kk) {
          const uint64_t bdesc = B_MN ? smem_desc_sw128(ww + kk * 2048, 8192, 1024)
                                      : smem_desc_sw128(ww + kk * 32, 16, 1024);
          const uint64_t adesc = smem_desc_sw128(aa + acc * (128 * BK * 2) + kk * 32, 16, 1024);
          umma_bf16<CG>(tmem_base + acc * BN, adesc, bdesc, idesc, (first && kk == 0) ? 0u : 1u);
        }
      };
      auto release = [&](uint32_t qq) {  // both accumulators are done with stage qq
        if constexpr (PAIRS == 1) {
          umma_commit<CG>(empty_a(qq % SA));
          umma_commit<CG>(empty_w(qq % SW));
        } else {
          umma_commit_pair_mask(empty_a(qq % SA), pair_mask);
          umma_commit_pair_mask(empty_w(qq % SW), all_mask);
        }
      };
      auto full = [&](int acc) {
        if constexpr (PAIRS == 1) umma_commit<CG>(tmem_full0 + 8u * acc);
        else umma_commit_pair_mask(tmem_full0 + 8u * acc, pair_mask);
      };
      for (int t = cluster; ok && t < num_tiles; t += nclusters, ++it) {
        {
          const TileInfo ti = tile_info(args, t, Cfg::kTileRows * PAIRS);
          const int64_t prow = ti.row0 + pair * Cfg::kTileRows;
#pragma unroll
          for (int acc = 0; acc < NACC; ++acc) live[acc] = prow + acc * Cfg::kRowsPerAcc < ti.row_end;
        }
        const uint32_t ep = (it & 1u) ^ 1u;  // the epilogue has drained the previous tile's accumulator
        // head: accumulator 0 over stages 0 .. J-1
        if (!mbar_wait(tmem_empty0, ep, wc)) break;
        tc_fence_after();
        for (int h = 0; ok && h < J; ++h) {
          if (!stage_in(q + h)) { ok = false; break; }
          issue(q + h, 0, h == 0);
        }
        if (!ok || !mbar_wait(tmem_empty0 + 8u * (NACC - 1), ep, wc)) break;
        tc_fence_after();
        for (int h = 0; h < J; ++h) {
          issue(q + h, 1, h == 0);
          release(q + h);
        }
        q += J;
        // body: both accumulators per stage
        for (int kb = J; kb < T - J; ++kb, ++q) {
          if (!stage_in(q)) { ok = false; break; }
          issue(q, 0, kb == 0);
          issue(q, 1, kb == 0);
          release(q);
        }
        if (!ok) break;
        // tail: accumulator 0 over the last J stages, which the epilogue then drains while
        // accumulator 1 finishes them
        for (int h = 0; ok && h < J; ++h) {
          if (!stage_in(q + h)) { ok = false; break; }
          issue(q + h, 0, false);
        }
        if (!ok) break;
        full(0);
        for (int h = 0; h < J; ++h) {
          issue(q + h, 1, false);
          release(q + h);
        }
        q += J;
        full(1);
      }
      if constexpr (PAIRS == 1) umma_commit<CG>(final_bar);
      else umma_commit_pair_mask(final_bar, pair_mask);
      mbar_wait_drain(final_bar, 0);
    } else if (PAIRS == 2 && cta == 1 && lane == 0) {
      // ---------------------------------------------------------- odd CTA: received stages
      // Once this CTA's half of a received stage has landed, arm the slot's next use and
      // report the half to the pair's MMA.
      uint32_t q = 0;
      bool ok = true;
      for (int t = cluster; ok && t < num_tiles; t += nclusters) {
        for (int kb = 0; kb < args.num_k_blocks; ++kb, ++q) {
          if ((q & 1u) == pair) continue;
          const uint32_t s = q % SW, ph = (q / SW) & 1u;
          if (!mbar_wait(recv_w(s), ph, wc)) { ok = false; break; }
          mbar_arrive_expect_tx(recv_w(s), Cfg::kWBytes);
          mbar_arrive_cluster(leader_full_w0 + 8u * s);
        }
      }
    }
  } else if (warp < Cfg::kEpiWarps) {
    // ------------------------------------------------------------ epilogue
    // Lane l of warp qd owns accumulator row qd * 32 + l.
    //   EPI 0:  Y in bf16, transposed through lane quads for contiguous stores.
    //   EPI 1:  16 columns per TMEM load: the accumulator times the row's scale (when given),
    //           stored as bf16 or fp32 when C is given, and, with a teacher output, the fused
    //           loss: d = Y - Y_ref from the unrounded accumulator, dY = dscale d in bf16 and a
    //           compensated sum of d^2 over every element the warp owns.  The teacher rows
    //           of both accumulators are sent to L2 when the tile begins, and each lane keeps
    //           two 16-column chunks of its row in flight ahead of the arithmetic.
    const int qd = warp;  // TMEM lane quarter
    const bool fused_loss = EPI == 1 && args.yref != nullptr;
    const uint16_t* yref16 = static_cast<const uint16_t*>(args.yref);
    const float* yref32 = static_cast<const float*>(args.yref);
    Sum2 lacc{0.f, 0.f};
    uint32_t it = 0;
    bool ok = true;
    for (int t = cluster; ok && t < num_tiles; t += nclusters, ++it) {
      const TileInfo ti = tile_info(args, t, Cfg::kTileRows * PAIRS);
      const int64_t col0 = (int64_t)ti.n_blk * BN;
      if (fused_loss) {
        const int64_t ncols_here = args.ncols - col0 < BN ? args.ncols - col0 : (int64_t)BN;
        const int64_t esz = args.yref_f32 ? 4 : 2;
#pragma unroll
        for (int acc = 0; acc < NACC; ++acc) {
          const int64_t row = ti.row0 + pair * Cfg::kTileRows + acc * Cfg::kRowsPerAcc + cta * 128 + qd * 32 + lane;
          if (row < ti.row_end && ncols_here > 0)
            prefetch_l2_bulk(static_cast<const char*>(args.yref) + (row * args.ncols + col0) * esz,
                             static_cast<uint32_t>(ncols_here * esz));
        }
      }
#pragma unroll 1
      for (int acc = 0; acc < NACC; ++acc) {
        const int64_t row0 = ti.row0 + pair * Cfg::kTileRows + acc * Cfg::kRowsPerAcc + cta * 128 +
                             qd * 32;  // this warp's first row
        if constexpr (EPI == 0) {
          if (!mbar_wait(tmem_full0 + 8u * acc, it & 1u, wc)) { ok = false; break; }
          tc_fence_after();
#pragma unroll 1
          for (int c = 0; c < BN / 32; ++c) {
            const int64_t col = col0 + c * 32;
            if (col >= args.ncols || row0 >= ti.row_end) break;  // warp-uniform
            uint32_t r[32];
            tmem_ld32(tmem_base + (static_cast<uint32_t>(qd * 32) << 16) + acc * BN + c * 32, r);
            tmem_ld_wait();
            store_rows_bf16x32(static_cast<uint16_t*>(args.C), ti.row_end, args.ncols, row0, col, r, lane);
          }
        } else {
          const int64_t row = row0 + lane;
          const bool row_ok = row < ti.row_end;
          const float rs = args.row_scale ? (row_ok ? __ldg(args.row_scale + row) : 0.0f) : 1.0f;
          const bool ref16 = fused_loss && !args.yref_f32;
          uint4 y0[2], y1[2];
          if (ref16) {
            load_yref_bf16x16(yref16, args.ncols, row, row_ok, col0, y0);
            load_yref_bf16x16(yref16, args.ncols, row, row_ok, col0 + 16, y1);
          }
          if (!mbar_wait(tmem_full0 + 8u * acc, it & 1u, wc)) { ok = false; break; }
          tc_fence_after();
#pragma unroll 1
          for (int c = 0; c < BN / 16; ++c) {
            const int64_t col = col0 + c * 16;
            if (col >= args.ncols || row0 >= ti.row_end) break;  // warp-uniform
            uint32_t r[16];
            tmem_ld16(tmem_base + (static_cast<uint32_t>(qd * 32) << 16) + acc * BN + c * 16, r);
            uint4 y2[2];
            if (ref16) load_yref_bf16x16(yref16, args.ncols, row, row_ok, col + 32, y2);
            tmem_ld_wait();
            if (args.row_scale) {
#pragma unroll
              for (int i = 0; i < 16; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * rs);
            }
            if (args.C) {
              if (args.c_f32) store_row_f32x16(static_cast<float*>(args.C), ti.row_end, args.ncols, row, col, r);
              else store_rows_bf16x16(static_cast<uint16_t*>(args.C), ti.row_end, args.ncols, row0, col, r, lane);
            }
            if (fused_loss) {
              uint4 pk[2];        // dY, packed as it is formed
              float csum = 0.0f;  // this chunk's sum of d^2 (16 terms), then one compensated add
#pragma unroll
              for (int q = 0; q < 2; ++q) {  // 8 columns at a time
                const bool live = row_ok && col + 8 * q < args.ncols;  // ncols is a multiple of 8
                float4 ra = make_float4(0.f, 0.f, 0.f, 0.f), rb = ra;  // fp32 teacher
                if (!ref16 && live) {
                  const float4* qv = reinterpret_cast<const float4*>(yref32 + row * args.ncols + col + 8 * q);
                  ra = __ldg(qv);
                  rb = __ldg(qv + 1);
                }
                uint32_t* out = reinterpret_cast<uint32_t*>(&pk[q]);
#pragma unroll
                for (int e = 0; e < 4; ++e) {  // columns 2e, 2e + 1 of the eight
                  const uint32_t w = ref16 ? (e == 0 ? y0[q].x : e == 1 ? y0[q].y : e == 2 ? y0[q].z : y0[q].w) : 0u;
                  const float4 rr = (e >> 1) ? rb : ra;
                  const float t0 = ref16 ? bf16lo_to_f32(w) : ((e & 1) ? rr.z : rr.x);
                  const float t1 = ref16 ? bf16hi_to_f32(w) : ((e & 1) ? rr.w : rr.y);
                  const float d0 = live ? __uint_as_float(r[8 * q + 2 * e]) - t0 : 0.0f;
                  const float d1 = live ? __uint_as_float(r[8 * q + 2 * e + 1]) - t1 : 0.0f;
                  csum = fmaf(d0, d0, csum);
                  csum = fmaf(d1, d1, csum);
                  out[e] = pack_bf16x2(d0 * args.dscale, d1 * args.dscale);
                }
              }
              sum2_add(lacc, csum);
              if (args.dY) store_rows_packed16(args.dY, ti.row_end, args.ncols, row0, col, pk, lane);
              if (ref16) {
                y0[0] = y1[0];
                y0[1] = y1[1];
                y1[0] = y2[0];
                y1[1] = y2[1];
              }
            }
          }
        }
        // this accumulator is drained: the MMA may refill it
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_cluster(leader_tmem_empty0 + 8u * acc);
      }
    }
    if (fused_loss) {
      lacc = sum2_team(lacc, 32);
      if (lane == 0) args.loss_part[blockIdx.x * Cfg::kEpiWarps + qd] = sum2_value(lacc);
    }
  } else {
    // ------------------------------------------------------------ operand producers
    // Within its group, each thread owns one row (CG 1) or half a row (CG 2) of the stage's
    // raw W tile and rewrites it in place as the Eq. 6 weight.  A row holds 64 consecutive K
    // elements of one W row, so it lies in one group (g is a multiple of 64).  Rows outside
    // W were zero-filled by the copy and stay 0.  The CTA's produced stages are
    // pair, pair + PAIRS, ...; group g takes every second of them.
    constexpr int CPT = Cfg::kChunksPerThread;
    constexpr int STEP = Cfg::kStep;
    const int pw = warp - (Cfg::kEpiWarps + 2);  // producer warp index
    const int grp = pw / Cfg::kGroupWarps;
    // PAIRS 2: this warp's rows of a produced half-tile go to the same slot of the CTA with
    // the same half in the other pair.
    const uint32_t my_rows = static_cast<uint32_t>(pw % Cfg::kGroupWarps) * Cfg::kRowsPerWarp * 128u;
    const uint32_t peer = rank ^ 2u;
    const uint32_t peer_w = PAIRS == 2 ? mapa_shared(w_base + my_rows, peer) : 0u;
    // the peer's barrier that counts the bytes: full_w in an even CTA, recv_w in an odd one
    const uint32_t peer_recv0 = PAIRS == 2 ? mapa_shared(cta == 0 ? full_w(0) : recv_w(0), peer) : 0u;
    const int tt = threadIdx.x - 32 * (Cfg::kEpiWarps + 2) - grp * Cfg::kGroupThreads;
    const int row = tt / Cfg::kThreadsPerRow;
    const int c_begin = (tt % Cfg::kThreadsPerRow) * CPT;
    const LayerDev& L = args.L;
    const int32_t phase_t = args.sc.phase;
    const bool transform = phase_t != PHASE_TEACHER;
    const uint32_t q0 = (PAIRS == 2 ? pair : 0u) + PAIRS * grp;
    // `cur` is the stage being produced; `ahead` runs two of this thread's stages ahead and
    // requests that stage's operand constants (one 16-byte vector, precomputed per call), so
    // an L2 round trip is hidden behind two stages.
    OperandRowIter<CG, B_MN, PAIRS> cur, ahead;
    cur.init(args, cta, row, cluster, 0);
    cur.step(args, cta, row, nclusters, q0);
    ahead = cur;
    // With mu in the reconstruction the group offset comes from its own [K/g][N] plane.
    float4 raw0{}, raw1{};
    float m0 = 0.0f, m1 = 0.0f;
    int64_t j0 = -1, j1 = -1;
    constexpr bool with_mu = MU;
    auto request = [&](const OperandRowIter<CG, B_MN, PAIRS>& it, float4& dst, float& dm, int64_t& jd,
                       const float4& other, float om, int64_t jo) {
      if (transform && it.live(args, num_tiles) && it.valid(args)) {
        if (jo == it.ci) {
          dst = other;
          dm = om;
        } else {
          dst = __ldg(L.op_const + it.ci);
          if (with_mu) dm = __ldg(L.op_mu + it.mi);
        }
        jd = it.ci;
      }
    };
    request(ahead, raw0, m0, j0, raw1, m1, j1);
    ahead.step(args, cta, row, nclusters, STEP);
    request(ahead, raw1, m1, j1, raw0, m0, j0);
    ahead.step(args, cta, row, nclusters, STEP);
    int64_t j_have = -1;
    ProducerConst pc{};
    uint32_t q = q0;
    bool ok = true;
    // One stage: consume `mine` (requested two stages ago), then refill it two stages ahead.
    auto produce = [&](float4& mine, float& mm, int64_t& jm, const float4& other, float om, int64_t jo) {
      const uint32_t s = q % SW;
      const bool live = transform && cur.valid(args);
      if (live && cur.ci != j_have) {
        pc = producer_const_from(mine, mm);
        j_have = cur.ci;
      }
      if (!mbar_wait(raw_w(grp * SW + s), (q / Cfg::kRawPeriod) & 1u, wc)) {
        ok = false;
        return;
      }
      if (live) {
        uint8_t* rowp = base_ptr + (w_base - base) + s * Cfg::kWBytes + row * 128;
        // One straight-line transform per row: the kind is uniform over the row's chunks.
        auto run = [&](auto kind_tag) {
          constexpr int KIND = decltype(kind_tag)::value;
          uint4 v[CPT];
#pragma unroll
          for (int i = 0; i < CPT; ++i) v[i] = *reinterpret_cast<const uint4*>(rowp + (((c_begin + i) ^ (row & 7)) * 16));
#pragma unroll
          for (int i = 0; i < CPT; ++i)
            *reinterpret_cast<uint4*>(rowp + (((c_begin + i) ^ (row & 7)) * 16)) = transform_chunk<KIND>(v[i], pc);
        };
        constexpr int kMu = MU ? XF_MU : 0;
        switch (transform_kind(pc, phase_t, MU ? 1 : 0)) {
          case XF_SOFT1 | kMu: run(std::integral_constant<int, XF_SOFT1 | kMu>{}); break;
          case XF_SOFT2 | kMu: run(std::integral_constant<int, XF_SOFT2 | kMu>{}); break;
          case XF_HARD | kMu: run(std::integral_constant<int, XF_HARD | kMu>{}); break;
          default: break;
        }
        fence_proxy_async_smem();
      }
      __syncwarp();
      if (lane == 0) {
        if constexpr (PAIRS == 2)
          bulk_copy_to_peer(peer_w + s * Cfg::kWBytes, w_base + my_rows + s * Cfg::kWBytes, Cfg::kRowsPerWarp * 128u,
                            peer_recv0 + 8u * s);
        mbar_arrive_cluster(leader_full_w0 + 8u * s);
      }
      // Issued after the proxy fence, which would otherwise wait for these loads.
      request(ahead, mine, mm, jm, other, om, jo);
      ahead.step(args, cta, row, nclusters, STEP);
      q += STEP;
      cur.step(args, cta, row, nclusters, STEP);
    };
    while (ok && cur.live(args, num_tiles)) {
      produce(raw0, m0, j0, raw1, m1, j1);
      if (!ok || !cur.live(args, num_tiles)) break;
      produce(raw1, m1, j1, raw0, m0, j0);
    }
  }

  tc_fence_before();
  if constexpr (CG == 2) cluster_sync_all(); else __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc<CG>(tmem_base, kTmemCols);
  }
}

// ============================================================================ wait probe

// Self-test of the bounded waits: one thread waits on a shared-memory barrier nothing
// arrives on, with the caller's limit, through the same mbar_wait the GEMMs use.  When the
// limit passes the wait latches CATQ_ERR_TIMEOUT and returns; nothing faults or hangs.
__global__ void wait_probe_kernel(const WaitCtl wc) {
  __shared__ __align__(8) uint64_t bar;
  const uint32_t b = smem_u32(&bar);
  mbar_init(b, 1);
  fence_mbar_init_cluster();
  mbar_wait(b, 0, wc);
}

// ============================================================================ dW kernel

// NE > 1: a grouped launch over gm's experts (tmDY, tmX unused).
template <int CG, bool MU, int NE>
__global__ void __launch_bounds__(DwCfg<CG>::kThreads, 1)
    dw_kernel(const __grid_constant__ CUtensorMap tmDY, const __grid_constant__ CUtensorMap tmX, const DwArgs args,
              const __grid_constant__ DwMaps<NE> gm) {
  using Cfg = DwCfg<CG>;
  constexpr int S = Cfg::kStages;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_addr = smem_u32(smem_raw);
  const uint32_t base = (raw_addr + 1023u) & ~1023u;
  uint8_t* base_ptr = smem_raw + (base - raw_addr);
  const uint32_t bars = base + S * Cfg::kStageBytes;
  auto full = [&](int s) { return bars + 8u * s; };
  auto empty = [&](int s) { return bars + 8u * (S + s); };
  const uint32_t tmem_full0 = bars + 8u * (2 * S);      // [2]
  const uint32_t tmem_empty0 = tmem_full0 + 16;         // [2]
  const uint32_t final_bar = tmem_full0 + 32;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(base_ptr + (bars - base) + 8 * (2 * S + 5));

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t cta = CG == 2 ? cluster_ctarank() : 0u;
  const uint32_t cluster = CG == 2 ? cluster_id_x() : blockIdx.x;
  const uint32_t nclusters = CG == 2 ? num_clusters_x() : gridDim.x;
  const WaitCtl& wc = args.wc;
  const int tiles_per_split = args.num_n_tiles * args.num_k_tiles;
  // grouped: expert slot i owns tiles [i tiles_per_split, (i + 1) tiles_per_split)
  const int num_tiles = tiles_per_split * (NE > 1 ? args.n_experts : args.splits);
  // The contraction range of tile t: its split's k blocks (dense) or its expert's rows.
  auto kb_range = [&](int t, int& kb0, int& kb1) {
    if constexpr (NE > 1) {
      kb0 = 0;
      kb1 = (gm.rows[t / tiles_per_split] + BK - 1) / BK;
    } else {
      const int split = t / tiles_per_split;
      kb0 = split * args.kb_per_split;
      kb1 = min(kb0 + args.kb_per_split, args.kb_total);
    }
  };
  constexpr int kTma = Cfg::kEpiWarps, kMma = Cfg::kEpiWarps + 1;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(full(s), 1);
      mbar_init(empty(s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(tmem_full0 + 8u * b, 1);
      mbar_init(tmem_empty0 + 8u * b, Cfg::kEpiWarps * CG);
    }
    mbar_init(final_bar, 1);
    fence_mbar_init_cluster();
  }
  if (warp == kMma) tmem_alloc<CG>(smem_u32(tmem_slot), kTmemCols);
  if (NE == 1 && warp == kTma && lane == 0) {
    prefetch_tmap(&tmDY);
    prefetch_tmap(&tmX);
  }
  tc_fence_before();
  if constexpr (CG == 2) cluster_sync_all(); else __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const uint32_t leader_full0 = CG == 2 ? mapa_shared(full(0), 0) : full(0);
  const uint32_t leader_tmem_empty0 = CG == 2 ? mapa_shared(tmem_empty0, 0) : tmem_empty0;

  if (warp == kTma) {
    if (lane == 0) {
      uint32_t stage = 0, phase = 0, issued_mask = 0, issued_phase = 0, it_tma = 0;
      const uint64_t pol_keep = args.x_keep ? l2_policy_evict_last() : l2_policy_evict_normal();
      bool ok = true;
      for (int t = cluster; ok && t < num_tiles; t += nclusters) {
        const int r = t % tiles_per_split;
        int k_blk, n_blk;
        dw_tile(args, r, n_blk, k_blk);
        int kb0, kb1;
        kb_range(t, kb0, kb1);
        const void* mdy = &tmDY;
        const void* mx = &tmX;
        if constexpr (NE > 1) {
          mdy = &gm.dy[t / tiles_per_split];
          mx = &gm.x[t / tiles_per_split];
        }
        // Serpentine contraction: tiles of odd iterations (every other tile wave) run their M
        // blocks backwards, so a wave starts where the previous one ended, with that part of
        // X still in L2.  The MMA loop walks the same order.
        const bool rev = (it_tma & 1u) != 0;
        ++it_tma;
        for (int j = 0; j < kb1 - kb0; ++j) {
          const int kb = rev ? kb1 - 1 - j : kb0 + j;
          if (!mbar_wait(empty(stage), phase ^ 1u, wc)) { ok = false; break; }
          const uint32_t sa = base + stage * Cfg::kStageBytes, sb = sa + Cfg::kABytes;
          const int32_t m = kb * BK;
          if (cta == 0) mbar_arrive_expect_tx(full(stage), Cfg::kStageBytes * CG);
          const uint32_t fb = leader_full0 + 8u * stage;
          // X is read by every tile wave, so it is kept in L2 ahead of the W the epilogue
          // streams when it fits (args.x_keep); dY keeps the normal policy: its column blocks
          // serve every k block of their n rows within one wave.
#pragma unroll
          for (int b = 0; b < 2; ++b) {
            const int32_t n = n_blk * Cfg::kTileRows + cta * 128 + 64 * b;
            if constexpr (CG == 1) tma_load_2d(sa + b * 8192, mdy, fb, n, m);
            else tma_load_2d_pair(sa + b * 8192, mdy, fb, n, m);
          }
#pragma unroll
          for (int b = 0; b < Cfg::kBCols / 64; ++b) {
            const int32_t k = k_blk * BN + cta * Cfg::kBCols + 64 * b;
            if constexpr (CG == 1) tma_load_2d_hint(sb + b * 8192, mx, fb, k, m, pol_keep);
            else tma_load_2d_pair_hint(sb + b * 8192, mx, fb, k, m, pol_keep);
          }
          issued_mask |= 1u << stage;
          issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
          if (++stage == S) { stage = 0; phase ^= 1u; }
        }
      }
      // Drain (the even CTA's barriers observe both CTAs' copies).
      if (cta == 0)
        for (int s = 0; s < S; ++s)
          if (issued_mask & (1u << s)) mbar_wait_drain(full(s), (issued_phase >> s) & 1u);
    }
  } else if (warp == kMma) {
    if (cta == 0 && lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(Cfg::kTileRows, BN, true, true);
      uint32_t stage = 0, phase = 0, it = 0;
      bool ok = true;
      for (int t = cluster; ok && t < num_tiles; t += nclusters, ++it) {
        int kb0, kb1;
        kb_range(t, kb0, kb1);
        const uint32_t buf = it & 1u;
        if (!mbar_wait(tmem_empty0 + 8u * buf, ((it >> 1) & 1u) ^ 1u, wc)) break;
        tc_fence_after();
        // Stages arrive in the TMA's order (forwards or, on odd iterations, backwards over M);
        // the sum does not depend on it, and the tile's first stage clears the accumulator.
        for (int j = 0; j < kb1 - kb0; ++j) {
          if (!mbar_wait(full(stage), phase, wc)) { ok = false; break; }
          tc_fence_after();
          const uint32_t sa = base + stage * Cfg::kStageBytes, sb = sa + Cfg::kABytes;
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk) {
            const uint64_t adesc = smem_desc_sw128(sa + kk * 2048, 8192, 1024);
            const uint64_t bdesc = smem_desc_sw128(sb + kk * 2048, 8192, 1024);
            umma_bf16<CG>(tmem_base + buf * BN, adesc, bdesc, idesc, (j > 0 || kk > 0) ? 1u : 0u);
          }
          umma_commit<CG>(empty(stage));
          if (++stage == S) { stage = 0; phase ^= 1u; }
        }
        if (ok) umma_commit<CG>(tmem_full0 + 8u * buf);
      }
      umma_commit<CG>(final_bar);
      mbar_wait_drain(final_bar, 0);
    }
  } else {
    // ------------------------------------------------------------ factor-gradient epilogue
    const int q = warp & 3;        // TMEM lane quarter
    const int half = warp >> 2;    // column half of the tile
    const int64_t cpr = args.L.K / args.P;
    const int64_t plane = args.L.N * cpr;
    const float k_sc = args.sc.s * args.sc.inv_2tanh_s;
    const float inv_k = (MU && k_sc > 0.0f) ? 1.0f / k_sc : 0.0f;
    const uint64_t pol_w = l2_policy_evict_first();
    uint32_t it = 0;
    for (int t = cluster; t < num_tiles; t += nclusters, ++it) {
      const int split = t / tiles_per_split, r = t % tiles_per_split;
      int k_blk, n_blk;
      dw_tile(args, r, n_blk, k_blk);
      // the tile's layer: the dense one, or (grouped) its expert's slice of the stacked layer
      // (grouped: the expert's weights and per-group arrays start e N K elements and e G
      // groups after expert 0's; its group j is group jbase + j of the stacked arrays)
      const LayerDev& L = args.L;
      int64_t slab = split;  // which [3][N][K/P] partial block the tile writes
      const uint16_t* W = static_cast<const uint16_t*>(L.W);
      int64_t jbase = 0;
      if constexpr (NE > 1) {
        const int64_t e = gm.expert[split];
        W += e * L.N * L.K;
        jbase = e * L.N * L.groups_per_row;
        slab = e;
      }
      const uint32_t buf = it & 1u;
      const int64_t n = (int64_t)n_blk * Cfg::kTileRows + cta * 128 + q * 32 + lane;
      const bool row_ok = n < L.N;
      float* out = args.part + slab * 3 * plane;
      LogiSums lacc{0.f, 0.f, 0.f, 0.f};
      const bool soft = args.sc.phase == PHASE_SOFT;
      constexpr int kChunks = (BN / 2) / 32;
      const int64_t k0 = (int64_t)k_blk * BN + half * (BN / 2);
      auto load_w = [&](int c, uint4 (&dst)[4]) {  // W is read once per launch: streamed through L2
        const int64_t k = k0 + c * 32;
        if (row_ok && k < L.K) {
          const uint4* wp = reinterpret_cast<const uint4*>(W + n * L.K + k);
#pragma unroll
          for (int v = 0; v < 4; ++v) dst[v] = ldg_hint(wp + v, pol_w);
        }
      };
      // The first two chunks' weights and the group constants the tile starts in are requested
      // before the wait for the accumulator, so their latency overlaps the tile's MMAs; later
      // chunks' weights are loaded two chunks ahead of the arithmetic.
      uint4 wcur[4], wnext[4], wnext2[4];
      load_w(0, wcur);
      if (kChunks > 1) load_w(1, wnext);
      int64_t cur_j = -1;
      GroupRaw graw{};
      if (row_ok && k0 < L.K) {
        cur_j = n * L.groups_per_row + k0 / L.g;
        graw = group_raw(L, jbase + cur_j);
      }
      if (!mbar_wait(tmem_full0 + 8u * buf, (it >> 1) & 1u, wc)) break;
      tc_fence_after();
      GroupConst gc = group_const(graw);
#pragma unroll 1
      for (int c = 0; c < kChunks; ++c) {
        const int col = half * (BN / 2) + c * 32;
        uint32_t rg[32];
        tmem_ld32(tmem_base + (static_cast<uint32_t>(q * 32) << 16) + buf * BN + col, rg);
        if (c + 2 < kChunks) load_w(c + 2, wnext2);
        tmem_ld_wait();
        const int64_t k = k0 + c * 32;
        if (row_ok && k < L.K) {
          const int64_t j = n * L.groups_per_row + k / L.g;
          if (j != cur_j) {
            gc = group_const(L, jbase + j);
            cur_j = j;
          }
          const float D = args.sc.s * gc.delta;
          if (gc.alpha != 0.0f && D >= kOneExpD) {
            // one exponential per weight (the far tanh term is 1 to fp32 resolution)
            const OneExp oe = one_exp_consts(args.sc.s, D);
            if (oe.c2 <= 126.0f) {
              if (soft) grad_chunk_logistic<MU, true, false>(rg, wcur, gc, oe, lacc, inv_k);
              else grad_chunk_logistic<MU, false, false>(rg, wcur, gc, oe, lacc, inv_k);
            } else {
              if (soft) grad_chunk_logistic<MU, true, true>(rg, wcur, gc, oe, lacc, inv_k);
              else grad_chunk_logistic<MU, false, true>(rg, wcur, gc, oe, lacc, inv_k);
            }
          } else if (gc.alpha != 0.0f) {
#pragma unroll
            for (int v = 0; v < 4; ++v) {
              const uint32_t w4[4] = {wcur[v].x, wcur[v].y, wcur[v].z, wcur[v].w};
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                grad_element_sums<MU>(__uint_as_float(rg[8 * v + 2 * e]), bf16lo_to_f32(w4[e]), gc, args.sc.s,
                                      args.sc.phase, lacc, inv_k);
                grad_element_sums<MU>(__uint_as_float(rg[8 * v + 2 * e + 1]), bf16hi_to_f32(w4[e]), gc, args.sc.s,
                                      args.sc.phase, lacc, inv_k);
              }
            }
          }
          if (((k + 32) % args.P) == 0 || k + 32 >= L.K) {
            const GradSums acc = grad_sums(lacc, soft, args.sc.inv_2tanh_s, k_sc);
            const int64_t idx = n * cpr + k / args.P;
            out[idx] = acc.smu;
            out[plane + idx] = acc.salpha;
            out[2 * plane + idx] = acc.sdelta;
            lacc = LogiSums{0.f, 0.f, 0.f, 0.f};
          }
        }
#pragma unroll
        for (int v = 0; v < 4; ++v) {
          wcur[v] = wnext[v];
          wnext[v] = wnext2[v];
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(leader_tmem_empty0 + 8u * buf);
    }
  }

  tc_fence_before();
  if constexpr (CG == 2) cluster_sync_all(); else __syncthreads();
  if (warp == kMma) {
    tc_fence_after();
    tmem_dealloc<CG>(tmem_base, kTmemCols);
  }
}

// ============================================================================ host side

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;
std::atomic<uint32_t> g_epoch{1};

void init_encoder() {
  std::call_once(g_encode_once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  });
}

// bf16 row-major [outer, inner] tensor, 128-byte swizzled boxes of box_inner x box_outer.
bool make_tmap(CUtensorMap* m, const void* ptr, uint64_t inner, uint64_t outer, uint32_t box_inner,
               uint32_t box_outer) {
  init_encoder();
  if (!g_encode) return false;
  const cuuint64_t dims[2] = {inner, outer};
  const cuuint64_t strides[1] = {inner * 2};
  const cuuint32_t box[2] = {box_inner, box_outer};
  const cuuint32_t estr[2] = {1, 1};
  return g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

struct DeviceInfo {
  int sm_count = 0;
  uint32_t* abort_word = nullptr;
  int32_t* status_word = nullptr;
  bool ok = false;
};

DeviceInfo& device_info() {
  static std::mutex mu;
  static DeviceInfo infos[64];
  int dev = 0;
  cudaGetDevice(&dev);
  std::lock_guard<std::mutex> lock(mu);
  DeviceInfo& d = infos[dev & 63];
  if (!d.ok) {
    cudaDeviceGetAttribute(&d.sm_count, cudaDevAttrMultiProcessorCount, dev);
    void* a = nullptr;
    void* s = nullptr;
    if (cudaGetSymbolAddress(&a, g_abort_word) == cudaSuccess &&
        cudaGetSymbolAddress(&s, g_status_word) == cudaSuccess) {
      d.abort_word = static_cast<uint32_t*>(a);
      d.status_word = static_cast<int32_t*>(s);
      d.ok = true;
    }
  }
  return d;
}

WaitCtl make_wait_ctl(const DeviceInfo& d) {
  WaitCtl w;
  w.abort_word = d.abort_word;
  w.status_word = d.status_word;
  uint32_t e = g_epoch.fetch_add(1);
  if (e == 0) e = g_epoch.fetch_add(1);
  w.epoch = e;
  w.timeout_ns = kWaitTimeoutNs;
  return w;
}

template <typename Kern>
cudaError_t launch_persistent(Kern kern, int cg, int grid_ctas, int threads, int smem, cudaStream_t st,
                              void** params) {
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(grid_ctas);
  cfg.blockDim = dim3(threads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cg;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelExC(&cfg, reinterpret_cast<const void*>(kern), params);
}

// Largest number of co-resident clusters of `cluster_ctas` CTAs for a kernel, cached per
// (device, kernel); a persistent grid larger than this would run a second, partial wave.
// (The kernel variants share one function type, so the cache is keyed by the kernel's
// address, not by the template instance.)
template <typename Kern>
int max_active_clusters(Kern kern, int cluster_ctas, int threads, int smem, int fallback) {
  static std::mutex mu;
  static std::map<std::pair<int, const void*>, int> cache;
  int dev = 0;
  cudaGetDevice(&dev);
  const std::pair<int, const void*> key{dev, reinterpret_cast<const void*>(kern)};
  std::lock_guard<std::mutex> lock(mu);
  const auto hit = cache.find(key);
  if (hit != cache.end()) return hit->second;
  cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(cluster_ctas * 64);
  cfg.blockDim = dim3(threads);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cluster_ctas;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, reinterpret_cast<const void*>(kern), &cfg) != cudaSuccess || n <= 0)
    n = fallback;
  cache[key] = n;
  return n;
}

// Tile shape by M: pairs of pairs (1024 rows per cluster tile) once M fills both pairs,
// CTA pairs (512 rows) from 512 rows, single CTAs below.
int fused_variant_for(int64_t M) { return M >= 1024 ? 4 : (M >= 512 ? 2 : 1); }

// grp (nullable): a grouped launch over grp->E experts whose weights are stacked from L.W on
// and whose rows of A and C are expert-sorted (host offsets grp->off).
template <int CG, bool B_MN, int PAIRS, bool MU, int EPI = 0>
cudaError_t run_fused(const LayerDev& L, StepScalars sc, const void* A, int64_t M, int64_t depth, void* C,
                      int64_t ncols, cudaStream_t st, const GroupSpec* grp = nullptr, const EpiOpts* opts = nullptr) {
  using Cfg = FusedCfg<CG, PAIRS>;
  DeviceInfo& d = device_info();
  if (!d.ok) return cudaErrorInvalidDevice;
  const int64_t wrows = grp ? grp->E * L.N : L.N;
  CUtensorMap ta, tw;
  if (!make_tmap(&ta, A, depth, M, BK, 128)) return cudaErrorInvalidValue;
  if constexpr (!B_MN) {
    if (!make_tmap(&tw, L.W, L.K, wrows, BK, Cfg::kBRows)) return cudaErrorInvalidValue;
  } else {
    if (!make_tmap(&tw, L.W, L.K, wrows, 64, BK)) return cudaErrorInvalidValue;
  }
  FusedArgs args;
  args.L = L;
  args.sc = sc;
  args.C = C;
  args.c_f32 = opts && opts->y_f32 ? 1 : 0;
  args.row_scale = opts ? opts->row_scale : nullptr;
  args.yref = opts ? opts->yref : nullptr;
  args.yref_f32 = opts && opts->yref_f32 ? 1 : 0;
  args.dscale = opts ? opts->dscale : 0.0f;
  args.dY = opts ? static_cast<uint16_t*>(opts->dY) : nullptr;
  args.loss_part = opts ? opts->loss_part : nullptr;
  if (opts && opts->n_parts) *opts->n_parts = 0;
  args.M = M;
  args.ncols = ncols;
  args.num_m_tiles = static_cast<int32_t>((M + Cfg::kTileRows * PAIRS - 1) / (Cfg::kTileRows * PAIRS));
  args.num_n_tiles = static_cast<int32_t>((ncols + BN - 1) / BN);
  args.num_k_blocks = static_cast<int32_t>((depth + BK - 1) / BK);
  args.group_m = std::min(4, args.num_m_tiles);
  {
    // A rows of one raster group: kept in L2 when they take at most a third of it (dense
    // launches; grouped ones stream every expert's W once and reuse little A)
    const int64_t group_rows = static_cast<int64_t>(args.group_m) * Cfg::kTileRows * PAIRS;
    args.a_keep = (!grp && std::min<int64_t>(group_rows, M) * depth * 2 <= (int64_t(40) << 20)) ? 1 : 0;
  }
  args.wc = make_wait_ctl(d);
  args.E = 0;
  args.const_stride = 0;
  int tiles = args.num_m_tiles * args.num_n_tiles;
  if (grp) {
    if (grp->E < 1 || grp->E > kMaxGroupExperts) return cudaErrorInvalidValue;
    args.E = grp->E;
    args.const_stride = grp->const_stride;
    const int64_t rows_per_tile = Cfg::kTileRows * PAIRS;
    int64_t t = 0;
    for (int e = 0; e <= grp->E; ++e) {
      args.tile0[e] = static_cast<int32_t>(t);
      args.row0[e] = static_cast<int32_t>(grp->off[e]);
      if (e < grp->E) t += (grp->off[e + 1] - grp->off[e] + rows_per_tile - 1) / rows_per_tile * args.num_n_tiles;
    }
    tiles = static_cast<int>(t);
    args.num_m_tiles = static_cast<int32_t>(t / args.num_n_tiles);  // the kernel's tile count is M x N blocks
    if (tiles == 0) return cudaSuccess;
  }
  auto kern = fused_gemm_kernel<CG, B_MN, PAIRS, MU, EPI>;
  const int fit = max_active_clusters(kern, Cfg::kClusterCtas, Cfg::kThreads, Cfg::kSmemBytes,
                                      d.sm_count / Cfg::kClusterCtas);
  const int clusters = std::min(tiles, fit);
  if (opts && opts->n_parts) *opts->n_parts = clusters * Cfg::kClusterCtas * Cfg::kEpiWarps;
  void* params[3] = {&ta, &tw, &args};
  return launch_persistent(kern, Cfg::kClusterCtas, clusters * Cfg::kClusterCtas, Cfg::kThreads, Cfg::kSmemBytes,
                           st, params);
}

// k blocks per raster group of the dW launch: about the square root of the clusters, so that
// a wave's tiles span as many n blocks as k blocks.
int dw_k_group(int num_k_tiles, int clusters) {
  int kg = 1;
  while ((kg + 1) * (kg + 1) <= clusters) ++kg;
  return std::max(1, std::min(kg, num_k_tiles));
}

template <int CG, bool MU>
cudaError_t run_dw(const LayerDev& L, StepScalars sc, const void* X, const void* dY, int64_t M, const TcPlan& plan,
                   float* part, cudaStream_t st) {
  static DwMaps<1> unused_maps;  // the dense kernel's (unread) grouped-map parameter
  using Cfg = DwCfg<CG>;
  DeviceInfo& d = device_info();
  if (!d.ok) return cudaErrorInvalidDevice;
  CUtensorMap tdy, tx;
  if (!make_tmap(&tdy, dY, L.N, M, 64, BK)) return cudaErrorInvalidValue;
  if (!make_tmap(&tx, X, L.K, M, 64, BK)) return cudaErrorInvalidValue;
  DwArgs args;
  args.L = L;
  args.sc = sc;
  args.part = part;
  args.M = M;
  args.splits = plan.dw_splits;
  args.P = plan.dw_P;
  args.kb_total = static_cast<int32_t>((M + BK - 1) / BK);
  args.kb_per_split = (args.kb_total + plan.dw_splits - 1) / plan.dw_splits;
  args.num_n_tiles = static_cast<int32_t>((L.N + Cfg::kTileRows - 1) / Cfg::kTileRows);
  args.num_k_tiles = static_cast<int32_t>((L.K + BN - 1) / BN);
  args.wc = make_wait_ctl(d);
  args.n_experts = 0;
  // every tile wave reads all of X: kept in L2 when it takes at most about 60 % of it (a
  // larger X under evict_last thrashes the cache it cannot fit)
  args.x_keep = M * L.K * 2 <= (int64_t(80) << 20) ? 1 : 0;
  // X kept in L2: every wave may read all of it (k fastest over the whole K, each dY slice
  // then read by one wave); otherwise waves about as wide in n as in k
  args.k_group = args.x_keep ? args.num_k_tiles : dw_k_group(args.num_k_tiles, d.sm_count / CG);
  const int tiles = args.num_n_tiles * args.num_k_tiles * args.splits;
  const int clusters = std::min(tiles, d.sm_count / CG);
  void* params[4] = {&tdy, &tx, &args, &unused_maps};
  return launch_persistent(dw_kernel<CG, MU, 1>, CG, clusters * CG, Cfg::kThreads, Cfg::kSmemBytes, st, params);
}

// Grouped dW: every expert with rows, kDwGroupExperts per launch; partials [E][3][N][K/P].
template <int CG, bool MU>
cudaError_t run_dw_grouped(const LayerDev& L0, StepScalars sc, const void* X, const void* dY, const GroupSpec& grp,
                           int32_t P, float* part, cudaStream_t st) {
  using Cfg = DwCfg<CG>;
  DeviceInfo& d = device_info();
  if (!d.ok) return cudaErrorInvalidDevice;
  static std::mutex mu;  // the parameter block below is reused per call
  std::lock_guard<std::mutex> lock(mu);
  static DwMaps<kDwGroupExperts> gm;
  CUtensorMap unused{};
  DwArgs args;
  args.L = L0;
  args.sc = sc;
  args.part = part;
  args.M = 0;
  args.splits = 1;
  args.P = P;
  args.kb_total = 0;
  args.kb_per_split = 0;
  args.num_n_tiles = static_cast<int32_t>((L0.N + Cfg::kTileRows - 1) / Cfg::kTileRows);
  args.num_k_tiles = static_cast<int32_t>((L0.K + BN - 1) / BN);
  args.x_keep = 0;  // an expert's rows are few: its X is read by few waves
  args.k_group = dw_k_group(args.num_k_tiles, d.sm_count / CG);
  const uint16_t* x = static_cast<const uint16_t*>(X);
  const uint16_t* dy = static_cast<const uint16_t*>(dY);
  int32_t e = 0;
  while (e < grp.E) {
    int n = 0;
    for (; e < grp.E && n < kDwGroupExperts; ++e) {
      const int64_t rows = grp.off[e + 1] - grp.off[e];
      if (rows == 0) continue;
      if (!make_tmap(&gm.dy[n], dy + grp.off[e] * L0.N, L0.N, rows, 64, BK) ||
          !make_tmap(&gm.x[n], x + grp.off[e] * L0.K, L0.K, rows, 64, BK))
        return cudaErrorInvalidValue;
      gm.expert[n] = e;
      gm.rows[n] = static_cast<int32_t>(rows);
      ++n;
    }
    if (n == 0) break;
    args.n_experts = n;
    args.wc = make_wait_ctl(d);
    const int tiles = args.num_n_tiles * args.num_k_tiles * n;
    const int clusters = std::min(tiles, d.sm_count / CG);
    void* params[4] = {&unused, &unused, &args, &gm};
    const cudaError_t err = launch_persistent(dw_kernel<CG, MU, kDwGroupExperts>, CG, clusters * CG, Cfg::kThreads,
                                              Cfg::kSmemBytes, st, params);
    if (err != cudaSuccess) return err;
  }
  return cudaSuccess;
}

// Tile shape by M, and the W ~ alpha T + mu instantiation for such layers outside TEACHER.
// Tile shape by rows (M, or a grouped launch's mean rows per expert) and the W ~ alpha T + mu
// instantiation for such layers outside TEACHER; the general epilogue (EPI 1) for a forward
// with epilogue options.
template <bool B_MN, int EPI>
cudaError_t dispatch_fused_epi(const LayerDev& L, StepScalars sc, const void* A, int64_t M, int64_t tile_rows,
                               int64_t depth, void* C, int64_t ncols, cudaStream_t st, const GroupSpec* grp,
                               const EpiOpts* opts) {
  const bool mu = L.recon != 0 && sc.phase != PHASE_TEACHER;
  switch (fused_variant_for(tile_rows) * 2 + (mu ? 1 : 0)) {
    case 8: return run_fused<2, B_MN, 2, false, EPI>(L, sc, A, M, depth, C, ncols, st, grp, opts);
    case 9: return run_fused<2, B_MN, 2, true, EPI>(L, sc, A, M, depth, C, ncols, st, grp, opts);
    case 4: return run_fused<2, B_MN, 1, false, EPI>(L, sc, A, M, depth, C, ncols, st, grp, opts);
    case 5: return run_fused<2, B_MN, 1, true, EPI>(L, sc, A, M, depth, C, ncols, st, grp, opts);
    case 3: return run_fused<1, B_MN, 1, true, EPI>(L, sc, A, M, depth, C, ncols, st, grp, opts);
    default: return run_fused<1, B_MN, 1, false, EPI>(L, sc, A, M, depth, C, ncols, st, grp, opts);
  }
}

template <bool B_MN>
cudaError_t dispatch_fused(const LayerDev& L, StepScalars sc, const void* A, int64_t M, int64_t depth, void* C,
                           int64_t ncols, cudaStream_t st, const EpiOpts* opts = nullptr) {
  if constexpr (!B_MN)
    if (opts) return dispatch_fused_epi<false, 1>(L, sc, A, M, M, depth, C, ncols, st, nullptr, opts);
  return dispatch_fused_epi<B_MN, 0>(L, sc, A, M, M, depth, C, ncols, st, nullptr, nullptr);
}

// Grouped: the tile shape by the mean rows per expert.
template <bool B_MN>
cudaError_t dispatch_fused_grouped(const LayerDev& L, StepScalars sc, const void* A, int64_t depth, void* C,
                                   int64_t ncols, const GroupSpec& grp, cudaStream_t st,
                                   const EpiOpts* opts = nullptr) {
  const int64_t R = grp.off[grp.E];
  if constexpr (!B_MN)
    if (opts) return dispatch_fused_epi<false, 1>(L, sc, A, R, R / grp.E, depth, C, ncols, st, &grp, opts);
  return dispatch_fused_epi<B_MN, 0>(L, sc, A, R, R / grp.E, depth, C, ncols, st, &grp, nullptr);
}

}  // namespace

cudaError_t launch_tc_fwd_grouped(const LayerDev& L0, StepScalars sc, const void* X, const GroupSpec& grp, void* Y,
                                  cudaStream_t st, const EpiOpts* opts) {
  if (sc.phase != PHASE_TEACHER) {
    const cudaError_t e = launch_operand_consts_grouped(L0, sc, grp.E, grp.const_stride, st);
    if (e != cudaSuccess) return e;
  }
  return dispatch_fused_grouped<false>(L0, sc, X, L0.K, Y, L0.N, grp, st, opts);
}

int fused_loss_max_parts(int sm_count) { return (sm_count > 0 ? sm_count : 1) * FusedCfg<1>::kEpiWarps; }

cudaError_t launch_tc_dx_grouped(const LayerDev& L0, StepScalars sc, const void* dY, const GroupSpec& grp, void* dX,
                                 cudaStream_t st) {
  if (sc.phase != PHASE_TEACHER) {
    const cudaError_t e = launch_operand_consts_grouped(L0, sc, grp.E, grp.const_stride, st);
    if (e != cudaSuccess) return e;
  }
  return dispatch_fused_grouped<true>(L0, sc, dY, L0.N, dX, L0.K, grp, st);
}

bool tensor_map_encoder_available() {
  init_encoder();
  return g_encode != nullptr;
}

TcPlan tc_plan_bwd(const LayerDev& L, int64_t M, int sm_count) {
  TcPlan p;
  p.dw_cg = L.N >= 256 ? 2 : 1;
  const int64_t rows = 128 * p.dw_cg;
  const int64_t tiles = ((L.N + rows - 1) / rows) * ((L.K + BN - 1) / BN);
  const int64_t clusters = std::max(1, sm_count / p.dw_cg);
  const int64_t kb_total = std::max<int64_t>(1, (M + BK - 1) / BK);
  // Split the contraction (M) only when the tiles leave clusters idle: every split re-runs
  // the per-element factor-gradient epilogue on its tile, which costs about as much as the
  // tile's MMA work, so splitting a full wave buys nothing.
  int64_t splits = 1;
  if (tiles < clusters) splits = std::min<int64_t>(clusters / tiles, std::max<int64_t>(1, kb_total / 8));
  const int64_t per = (kb_total + splits - 1) / splits;
  splits = (kb_total + per - 1) / per;
  p.dw_splits = static_cast<int32_t>(std::max<int64_t>(1, splits));
  p.dw_P = std::gcd(L.g, 128);
  return p;
}

cudaError_t launch_tc_fwd(const LayerDev& L, StepScalars sc, const void* X, int64_t M, void* Y, cudaStream_t st,
                         const EpiOpts* opts) {
  if (sc.phase != PHASE_TEACHER) {
    const cudaError_t e = launch_operand_consts(L, sc, st);
    if (e != cudaSuccess) return e;
  }
  return dispatch_fused<false>(L, sc, X, M, L.K, Y, L.N, st, opts);
}

cudaError_t launch_tc_dx(const LayerDev& L, StepScalars sc, const void* dY, int64_t M, void* dX, cudaStream_t st) {
  if (sc.phase != PHASE_TEACHER) {
    const cudaError_t e = launch_operand_consts(L, sc, st);
    if (e != cudaSuccess) return e;
  }
  return dispatch_fused<true>(L, sc, dY, M, L.N, dX, L.K, st);
}

bool launch_wait_ctl(WaitCtl* out) {
  DeviceInfo& d = device_info();
  if (!d.ok) return false;
  *out = make_wait_ctl(d);
  return true;
}

cudaError_t launch_wait_probe(uint64_t timeout_ns, cudaStream_t st) {
  DeviceInfo& d = device_info();
  if (!d.ok) return cudaErrorInvalidDevice;
  WaitCtl w = make_wait_ctl(d);
  w.timeout_ns = timeout_ns;
  wait_probe_kernel<<<1, 1, 0, st>>>(w);
  return cudaGetLastError();
}

cudaError_t launch_tc_dw(const LayerDev& L, StepScalars sc, const void* X, const void* dY, int64_t M,
                         const TcPlan& plan, float* partials, cudaStream_t st) {
  if (L.recon) {
    if (plan.dw_cg == 2) return run_dw<2, true>(L, sc, X, dY, M, plan, partials, st);
    return run_dw<1, true>(L, sc, X, dY, M, plan, partials, st);
  }
  if (plan.dw_cg == 2) return run_dw<2, false>(L, sc, X, dY, M, plan, partials, st);
  return run_dw<1, false>(L, sc, X, dY, M, plan, partials, st);
}

cudaError_t launch_tc_dw_grouped(const LayerDev& L0, StepScalars sc, const void* X, const void* dY,
                                 const GroupSpec& grp, int32_t P, float* partials, cudaStream_t st) {
  const bool cg2 = L0.N >= 256;
  if (L0.recon) return cg2 ? run_dw_grouped<2, true>(L0, sc, X, dY, grp, P, partials, st)
                           : run_dw_grouped<1, true>(L0, sc, X, dY, grp, P, partials, st);
  return cg2 ? run_dw_grouped<2, false>(L0, sc, X, dY, grp, P, partials, st)
             : run_dw_grouped<1, false>(L0, sc, X, dY, grp, P, partials, st);
}

cudaError_t read_and_clear_device_status(int32_t* out) {
  int32_t v = 0;
  cudaError_t e = cudaMemcpyFromSymbol(&v, g_status_word, sizeof(v));
  if (e != cudaSuccess) return e;
  const int32_t zero = 0;
  e = cudaMemcpyToSymbol(g_status_word, &zero, sizeof(zero));
  *out = v;
  return e;
}

}  // namespace catq
