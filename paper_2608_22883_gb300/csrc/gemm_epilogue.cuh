// Epilogues of C = A . B^T shared by the SIMT and tcgen05 GEMM kernels.
// (m, n) are group-local: m an A row (output column), n a B row (output row).
#pragma once
#include "common.cuh"

namespace fovea {

template <class T, int EPI>
__device__ __forceinline__ void gemm_epilogue(const GemmArgs& a, const GemmGroup& g, int m, int n,
                                              float acc) {
  if constexpr (EPI == kEpiStore) {
    const long long row = (long long)g.b_row0 + n;
    if (m < a.epi_split)
      static_cast<T*>(a.out0)[row * a.ldc + m] = from_f32<T>(acc);
    else
      static_cast<T*>(a.out1)[row * a.ldc + (m - a.epi_split)] = from_f32<T>(acc);
  } else if constexpr (EPI == kEpiScores) {
    const float rs = a.row_scale ? a.row_scale[g.b_row0 + n] : 1.0f;
    static_cast<float*>(a.out0)[g.c_off + (long long)n * g.m + m] = acc * a.scale * rs;
  } else if constexpr (EPI == kEpiBiasSilu) {
    const long long row = (long long)g.b_row0 + n;
    const float bias = m < a.epi_split ? to_f32(static_cast<const T*>(a.bias0)[m])
                                       : to_f32(static_cast<const T*>(a.bias1)[m - a.epi_split]);
    const float z = acc + bias;
    static_cast<T*>(a.out0)[row * a.ldc + m] = from_f32<T>(z * sigmoidf_(z));
  } else if constexpr (EPI == kEpiStoreHiLo) {
    const long long row = (long long)g.b_row0 + n;
    const T hi = from_f32<T>(acc);
    static_cast<T*>(a.out0)[row * a.ldc + m] = hi;
    static_cast<T*>(a.out1)[row * a.ldc + m] = from_f32<T>(acc - to_f32(hi));
  } else {  // kEpiBiasF32
    const long long row = (long long)g.b_row0 + n;
    static_cast<float*>(a.out0)[row * a.ldc + m] = acc + to_f32(static_cast<const T*>(a.bias0)[m]);
  }
}

}  // namespace fovea
