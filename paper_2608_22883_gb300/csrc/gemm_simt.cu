// SIMT GEMM C = A . B^T (fp32 FMA) for the fp32 path: the projections of the
// memory, the query, the scores and the two fusion layers when the workload
// stores fp32 (tensor cores would round fp32 operands).
#include "gemm_epilogue.cuh"

namespace fovea {

constexpr int kSimtTile = 64, kSimtK = 16, kSimtThreads = 256;

template <class T>
__device__ __forceinline__ float load_a(const GemmArgs& a, const GemmGroup& g, int m, int k) {
  if (m < a.a_split)
    return to_f32(static_cast<const T*>(a.A0)[(long long)(g.a_row0 + m) * a.lda0 + k]);
  return to_f32(static_cast<const T*>(a.A1)[(long long)(m - a.a_split) * a.lda1 + k]);
}
template <class T>
__device__ __forceinline__ float load_b(const GemmArgs& a, const GemmGroup& g, int n, int k) {
  const long long row = (long long)g.b_row0 + n;
  if (k < a.b_split) return to_f32(static_cast<const T*>(a.B0)[row * a.ldb0 + k]);
  return to_f32(static_cast<const T*>(a.B1)[row * a.ldb1 + (k - a.b_split)]);
}

template <class T, int EPI>
__global__ void __launch_bounds__(kSimtThreads) simt_gemm_kernel(const __grid_constant__ GemmArgs a) {
  const GemmGroup& g = a.groups[blockIdx.z];
  const int m0 = blockIdx.x * kSimtTile, n0 = blockIdx.y * kSimtTile;
  if (m0 >= g.m || n0 >= g.n) return;
  __shared__ float As[kSimtK][kSimtTile + 1];
  __shared__ float Bs[kSimtK][kSimtTile + 1];
  const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;   // 4x4 outputs each
  float acc[4][4] = {};
  for (int k0 = 0; k0 < a.k_total; k0 += kSimtK) {
    for (int i = threadIdx.x; i < kSimtTile * kSimtK; i += kSimtThreads) {
      const int r = i / kSimtK, kk = i % kSimtK;
      const int m = m0 + r, n = n0 + r;
      As[kk][r] = m < g.m ? load_a<T>(a, g, m, k0 + kk) : 0.0f;
      Bs[kk][r] = n < g.n ? load_b<T>(a, g, n, k0 + kk) : 0.0f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < kSimtK; ++kk) {
      float av[4], bv[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        av[i] = As[kk][tx + 16 * i];
        bv[i] = Bs[kk][ty + 16 * i];
      }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int m = m0 + tx + 16 * i, n = n0 + ty + 16 * j;
      if (m < g.m && n < g.n) gemm_epilogue<T, EPI>(a, g, m, n, acc[i][j]);
    }
}

template <class T>
static cudaError_t dispatch_simt(int epi, const GemmArgs& a, dim3 grid, cudaStream_t s) {
  switch (epi) {
    case kEpiStore: simt_gemm_kernel<T, kEpiStore><<<grid, kSimtThreads, 0, s>>>(a); break;
    case kEpiScores: simt_gemm_kernel<T, kEpiScores><<<grid, kSimtThreads, 0, s>>>(a); break;
    case kEpiBiasSilu: simt_gemm_kernel<T, kEpiBiasSilu><<<grid, kSimtThreads, 0, s>>>(a); break;
    case kEpiStoreHiLo: simt_gemm_kernel<T, kEpiStoreHiLo><<<grid, kSimtThreads, 0, s>>>(a); break;
    default: simt_gemm_kernel<T, kEpiBiasF32><<<grid, kSimtThreads, 0, s>>>(a); break;
  }
  return cudaGetLastError();
}

cudaError_t launch_gemm_simt(int dtype, int epi, const GemmArgs& a, int max_m, int max_n,
                             cudaStream_t s) {
  if (max_m <= 0 || max_n <= 0 || a.ngroups <= 0) return cudaSuccess;
  dim3 grid((max_m + kSimtTile - 1) / kSimtTile, (max_n + kSimtTile - 1) / kSimtTile, a.ngroups);
  cudaError_t e = dtype == FOVEA_BF16 ? dispatch_simt<__nv_bfloat16>(epi, a, grid, s)
                                      : dispatch_simt<float>(epi, a, grid, s);
  return e;
}

}  // namespace fovea
