// simt_f32.cu — fp32 CUDA-core path of the three contractions, used when W and X are fp32
// (a tensor-core path cannot meet an fp32 tolerance).  Tiled FFMA GEMMs, 64 x 64 output
// tiles, 16-deep k-slices, 4 x 4 outputs per thread, fp32 accumulation, accurate tanhf.
// The Eq. 6 weight is computed while its tile is staged into shared memory, and the dW
// contraction reduces straight into per-group partial sums (G = dY^T X is never stored).
#include "launch.h"

namespace catq {
namespace {

constexpr int TM = kSimtTile;  // output tile rows
constexpr int TN = kSimtTile;  // output tile cols
constexpr int TK = 16;         // contraction slice
constexpr int kThr = 256;

enum : int { MODE_FWD = 0, MODE_DX = 1, MODE_DW = 2 };

struct SimtArgs {
  LayerDev L;
  StepScalars sc;
  const float* A;  // FWD: X [M,K]; DX: dY [M,N]; DW: dY [M,N]
  const float* B;  // DW: X [M,K]; otherwise unused (W comes from L)
  float* C;        // FWD: Y [M,N]; DX: dX [M,K]; DW: partials [3][N][K/P]
  int64_t M;
  int32_t P;       // DW partial chunk width
  const float* row_scale;  // FWD, nullable: Y row m times row_scale[m]
};

__device__ __forceinline__ float w_elem(const SimtArgs& a, int64_t n, int64_t k) {
  const float w = static_cast<const float*>(a.L.W)[n * a.L.K + k];
  if (a.sc.phase == PHASE_TEACHER) return w;
  const GroupConst gc = group_const(a.L, n * a.L.groups_per_row + k / a.L.g);
  return ternary_weight_f32(w, gc, a.sc.s, a.sc.inv_2tanh_s, a.sc.phase, a.L.recon);
}

// C[i][j] = sum_c A(i, c) B(j, c) with
//   FWD: i = m, j = n, c = k:  A = X[m][k],  B = Wq[n][k]
//   DX : i = m, j = k, c = n:  A = dY[m][n], B = Wq[n][k]
//   DW : i = n, j = k, c = m:  A = dY[m][n], B = X[m][k]
template <int MODE>
__global__ void __launch_bounds__(kThr) simt_gemm_kernel(SimtArgs a) {
  __shared__ float As[TK][TM + 4];
  __shared__ float Bs[TK][TN + 4];
  const LayerDev& L = a.L;
  const int64_t rowsI = MODE == MODE_DW ? L.N : a.M;
  const int64_t colsJ = MODE == MODE_FWD ? L.N : L.K;
  const int64_t depth = MODE == MODE_FWD ? L.K : (MODE == MODE_DX ? L.N : a.M);
  const int64_t i0 = static_cast<int64_t>(blockIdx.y) * TM;
  const int64_t j0 = static_cast<int64_t>(blockIdx.x) * TN;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  float acc[4][4] = {};

  for (int64_t c0 = 0; c0 < depth; c0 += TK) {
    // Stage A and B slices: element e of the 1024-element slice is (row e/16, col e%16)
    // for "i/j-major" sources and (row e/64, col e%64) for "c-major" sources.
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int e = threadIdx.x + q * kThr;
      if (MODE == MODE_FWD || MODE == MODE_DX) {
        // A(i, c): X[m][k] or dY[m][n] — contiguous along c.
        const int r = e >> 4, cc = e & 15;
        const int64_t i = i0 + r, c = c0 + cc;
        const int64_t ld = MODE == MODE_FWD ? L.K : L.N;
        As[cc][r] = (i < rowsI && c < depth) ? a.A[i * ld + c] : 0.0f;
      } else {
        // DW: A(i = n, c = m) = dY[m][n] — contiguous along i.
        const int cc = e >> 6, r = e & 63;
        const int64_t i = i0 + r, c = c0 + cc;
        As[cc][r] = (i < rowsI && c < depth) ? a.A[c * L.N + i] : 0.0f;
      }
      if (MODE == MODE_FWD) {
        // B(j = n, c = k) = Wq[n][k] — contiguous along c.
        const int r = e >> 4, cc = e & 15;
        const int64_t j = j0 + r, c = c0 + cc;
        Bs[cc][r] = (j < colsJ && c < depth) ? w_elem(a, j, c) : 0.0f;
      } else if (MODE == MODE_DX) {
        // B(j = k, c = n) = Wq[n][k] — contiguous along j.
        const int cc = e >> 6, r = e & 63;
        const int64_t j = j0 + r, c = c0 + cc;
        Bs[cc][r] = (j < colsJ && c < depth) ? w_elem(a, c, j) : 0.0f;
      } else {
        // DW: B(j = k, c = m) = X[m][k] — contiguous along j.
        const int cc = e >> 6, r = e & 63;
        const int64_t j = j0 + r, c = c0 + cc;
        Bs[cc][r] = (j < colsJ && c < depth) ? a.B[c * L.K + j] : 0.0f;
      }
    }
    __syncthreads();
#pragma unroll
    for (int cc = 0; cc < TK; ++cc) {
      float av[4], bv[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        av[u] = As[cc][ty + 16 * u];
        bv[u] = Bs[cc][tx + 16 * u];
      }
#pragma unroll
      for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int v = 0; v < 4; ++v) acc[u][v] = fmaf(av[u], bv[v], acc[u][v]);
    }
    __syncthreads();
  }

  if (MODE != MODE_DW) {
    const int64_t ldc = colsJ;
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
      for (int v = 0; v < 4; ++v) {
        const int64_t i = i0 + ty + 16 * u, j = j0 + tx + 16 * v;
        if (i < rowsI && j < colsJ) a.C[i * ldc + j] = a.row_scale ? acc[u][v] * a.row_scale[i] : acc[u][v];
      }
    return;
  }

  // DW epilogue: per (row n, chunk of P columns) partial sums of the chain rule.
  // Column tx + 16 v of the tile lies in chunk (tx + 16 v) / P; lanes sharing a chunk
  // are the aligned groups of min(P, 16) consecutive tx.
  const int32_t P = a.P;
  const int lanes = P < 16 ? P : 16;
  const int64_t cpr = L.K / P;
  const int64_t plane = L.N * cpr;
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const int64_t n = i0 + ty + 16 * u;
    const bool row_ok = n < L.N;
    // v runs over the thread's 4 columns; consecutive v with the same chunk are summed.
    GradSums run{0.f, 0.f, 0.f};
    int cur_chunk = -1;
#pragma unroll
    for (int v = 0; v < 4; ++v) {
      const int col = tx + 16 * v;
      const int chunk = col / P;
      const int64_t k = j0 + col;
      GradSums e{0.f, 0.f, 0.f};
      if (row_ok && k < L.K) {
        const GroupConst gc = group_const(L, n * L.groups_per_row + k / L.g);
        if (gc.alpha != 0.0f) {
          const float w = static_cast<const float*>(L.W)[n * L.K + k];
          if (L.recon)
            grad_element<false, true>(acc[u][v], w, gc, a.sc.s, a.sc.inv_2tanh_s, a.sc.phase, e,
                                      1.0f / (a.sc.s * a.sc.inv_2tanh_s));
          else
            grad_element(acc[u][v], w, gc, a.sc.s, a.sc.inv_2tanh_s, a.sc.phase, e);
        }
      }
      if (P >= 16) {  // all 16 tx share the chunk of this v; accumulate over v in the chunk
        run.smu += e.smu;
        run.salpha += e.salpha;
        run.sdelta += e.sdelta;
        cur_chunk = chunk;
        const bool last_in_chunk = (v == 3) || ((tx + 16 * (v + 1)) / P != chunk);
        if (!last_in_chunk) continue;
        e = run;
        run = GradSums{0.f, 0.f, 0.f};
      }
      // Reduce over the lanes sharing this chunk (fixed xor order: deterministic).
      for (int o = 1; o < lanes; o <<= 1) {
        e.smu += __shfl_xor_sync(0xffffffffu, e.smu, o);
        e.salpha += __shfl_xor_sync(0xffffffffu, e.salpha, o);
        e.sdelta += __shfl_xor_sync(0xffffffffu, e.sdelta, o);
      }
      const int64_t kc = j0 + static_cast<int64_t>(chunk) * P;
      if (row_ok && (tx % lanes) == 0 && kc < L.K) {
        const int64_t idx = n * cpr + kc / P;
        a.C[idx] = e.smu;
        a.C[plane + idx] = e.salpha;
        a.C[2 * plane + idx] = e.sdelta;
      }
      (void)cur_chunk;
    }
  }
}

}  // namespace

static dim3 grid2(int64_t rows, int64_t cols) {
  return dim3(static_cast<unsigned>((cols + TN - 1) / TN), static_cast<unsigned>((rows + TM - 1) / TM));
}

cudaError_t launch_simt_fwd(const LayerDev& L, StepScalars sc, const float* X, int64_t M, float* Y, cudaStream_t st,
                            const float* row_scale) {
  SimtArgs a{L, sc, X, nullptr, Y, M, 0, row_scale};
  simt_gemm_kernel<MODE_FWD><<<grid2(M, L.N), kThr, 0, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_simt_dx(const LayerDev& L, StepScalars sc, const float* dY, int64_t M, float* dX, cudaStream_t st) {
  SimtArgs a{L, sc, dY, nullptr, dX, M, 0, nullptr};
  simt_gemm_kernel<MODE_DX><<<grid2(M, L.K), kThr, 0, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_simt_dw(const LayerDev& L, StepScalars sc, const float* X, const float* dY, int64_t M,
                           float* partials, cudaStream_t st) {
  const int32_t P = L.g < TN ? L.g : TN;
  SimtArgs a{L, sc, dY, X, partials, M, P, nullptr};
  simt_gemm_kernel<MODE_DW><<<grid2(L.N, L.K), kThr, 0, st>>>(a);
  return cudaGetLastError();
}

}  // namespace catq
