// CUDA-core GEMM for the decode projections: C[j][n] = sum_k X[j][k] W[n][k]
// (X compact active rows, W in nn.Linear layout), fp32 accumulation.
// Used for fp32 models (tensor cores would round operands) and for shapes the
// tcgen05 path does not cover.  One warp per output unit (a weight row, or the
// gate/up row pair of the SwiGLU epilogue), rows processed 4 at a time.
#include <cuda_runtime.h>

#include "common.cuh"
#include "internal.h"

namespace buddy {

constexpr int kSimtRows = 4;

template <typename T, int EPI>
__global__ void __launch_bounds__(256) gemm_simt_kernel(const T* __restrict__ W,
                                                        const T* __restrict__ X, const T* __restrict__ X_lo,
                                                        int N, int K,
                                                        const int32_t* rows, const int32_t* count,
                                                        int n, float* __restrict__ out_f32,
                                                        T* __restrict__ out_act, T* __restrict__ out_act_lo,
                                                        const float* resid_src, float* resid_dst,
                                                        const int32_t* status) {
  pdl_wait();
  pdl_trigger();
  if (call_aborted(status)) return;
  const int m = count ? *count : n;
  const int unit = blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (unit >= N) return;
  constexpr int NR = (EPI == EPI_SWIGLU) ? 2 : 1;
  const T* w[NR];
  w[0] = W + (size_t)unit * K;
  if (NR == 2) w[NR - 1] = W + (size_t)(N + unit) * K;
  for (int j0 = 0; j0 < m; j0 += kSimtRows) {
    float acc[NR][kSimtRows];
#pragma unroll
    for (int a = 0; a < NR; ++a)
#pragma unroll
      for (int r = 0; r < kSimtRows; ++r) acc[a][r] = 0.f;
    for (int k = lane * 8; k < K; k += 256) {
      float wv[NR][8];
#pragma unroll
      for (int a = 0; a < NR; ++a) load8(w[a] + k, wv[a]);
#pragma unroll
      for (int r = 0; r < kSimtRows; ++r) {
        if (j0 + r < m) {
          float xv[8];
          load8(X + (size_t)(j0 + r) * K + k, xv);
          if (X_lo) {
            float xl[8];
            load8(X_lo + (size_t)(j0 + r) * K + k, xl);
#pragma unroll
            for (int u = 0; u < 8; ++u) xv[u] += xl[u];
          }
#pragma unroll
          for (int a = 0; a < NR; ++a)
#pragma unroll
            for (int u = 0; u < 8; ++u) acc[a][r] += wv[a][u] * xv[u];
        }
      }
    }
#pragma unroll
    for (int a = 0; a < NR; ++a)
#pragma unroll
      for (int r = 0; r < kSimtRows; ++r) acc[a][r] = warp_sum(acc[a][r]);
    if (lane < kSimtRows && j0 + lane < m) {
      const int j = j0 + lane;
      float v0 = 0.f, v1 = 0.f;
#pragma unroll
      for (int r = 0; r < kSimtRows; ++r)
        if (r == lane) {
          v0 = acc[0][r];
          v1 = acc[NR - 1][r];
        }
      if (EPI == EPI_STORE_F32) {
        out_f32[(size_t)j * N + unit] = v0;
      } else if (EPI == EPI_RESID) {
        const int i = rows ? rows[j] : j;
        resid_dst[(size_t)i * N + unit] = resid_src[(size_t)i * N + unit] + v0;
      } else {
        const float a = silu_f(v0) * v1;
        const T hi = from_f<T>(a);
        out_act[(size_t)j * N + unit] = hi;
        if (out_act_lo) out_act_lo[(size_t)j * N + unit] = from_f<T>(a - to_f(hi));
      }
    }
  }
}

template <typename T>
static void simt_dispatch(int epi, const GemmArgs& a, cudaStream_t s, bool pdl) {
  const unsigned grid = (unsigned)((a.N + 7) / 8);
  const T* W = (const T*)a.W;
  const T* X = (const T*)a.X;
  const T* Xl = a.split ? (const T*)a.X_lo : nullptr;
  switch (epi) {
    case EPI_STORE_F32:
      launch_k(gemm_simt_kernel<T, EPI_STORE_F32>, grid, 256, 0, s, pdl, W, X, Xl, a.N, a.K, a.sel.rows,
               a.sel.count, a.sel.n, a.out_f32, (T*)nullptr, (T*)nullptr, (const float*)nullptr, (float*)nullptr,
               a.status);
      break;
    case EPI_RESID:
      launch_k(gemm_simt_kernel<T, EPI_RESID>, grid, 256, 0, s, pdl, W, X, Xl, a.N, a.K, a.sel.rows,
               a.sel.count, a.sel.n, (float*)nullptr, (T*)nullptr, (T*)nullptr, a.resid_src, a.resid_dst,
               a.status);
      break;
    default:
      launch_k(gemm_simt_kernel<T, EPI_SWIGLU>, grid, 256, 0, s, pdl, W, X, Xl, a.N, a.K, a.sel.rows,
               a.sel.count, a.sel.n, (float*)nullptr, (T*)a.out_act, (T*)a.out_act_lo, (const float*)nullptr,
               (float*)nullptr, a.status);
  }
}

void launch_gemm_simt(const Ctx& c, int epi, const GemmArgs& a, cudaStream_t s) {
  if (c.dtype == BUDDY_DTYPE_BF16) simt_dispatch<bf16>(epi, a, s, c.pdl);
  else simt_dispatch<float>(epi, a, s, c.pdl);
}

}  // namespace buddy
