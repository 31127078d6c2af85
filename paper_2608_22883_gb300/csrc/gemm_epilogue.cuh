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
  } else if constexpr (EPI == kEpiScores || EPI == kEpiScoresFolded) {
    if (EPI == kEpiScoresFolded && m >= a.epi_split) {
      static_cast<float*>(a.out2)[((long long)g.b_row0 + n) * a.ldc2 + (m - a.epi_split)] = acc;
      return;
    }
    const int stride = EPI == kEpiScoresFolded ? min(g.m, a.epi_split) : g.m;
    const float rs = a.row_scale ? a.row_scale[g.b_row0 + n] : 1.0f;
    static_cast<float*>(a.out0)[g.c_off + (long long)n * stride + m] = acc * a.scale * rs;
  } else if constexpr (EPI == kEpiBiasSilu || EPI == kEpiAct) {
    const long long row = (long long)g.b_row0 + n;
    const float bias = m < a.epi_split ? to_f32(static_cast<const T*>(a.bias0)[m])
                                       : to_f32(static_cast<const T*>(a.bias1)[m - a.epi_split]);
    float z = acc + bias;
    if constexpr (EPI == kEpiAct) z += a.add_in[row * a.ldc2 + m];
    static_cast<T*>(a.out0)[row * a.ldc + m] = from_f32<T>(z * sigmoidf_(z));
  } else if constexpr (EPI == kEpiStoreHiLo || EPI == kEpiQueryH) {
    const long long row = (long long)g.b_row0 + n;
    if (EPI == kEpiQueryH && m >= a.epi_split) {
      static_cast<float*>(a.out2)[row * a.ldc2 + (m - a.epi_split)] = acc;
      return;
    }
    const T hi = from_f32<T>(acc);
    static_cast<T*>(a.out0)[row * a.ldc + m] = hi;
    static_cast<T*>(a.out1)[row * a.ldc + m] = from_f32<T>(acc - to_f32(hi));
  } else {  // kEpiBiasF32
    const long long row = (long long)g.b_row0 + n;
    static_cast<float*>(a.out0)[row * a.ldc + m] = acc + to_f32(static_cast<const T*>(a.bias0)[m]);
  }
}

// Epilogue of four consecutive columns m .. m+3 (nv <= 4 of them in range) of
// output row n: one 8-byte (bf16) or 16-byte (fp32) store per output array
// where the four are contiguous and aligned, else per element.  bias4 holds
// the four columns' biases (bias epilogues, vector case).
template <int EPI>
__device__ __forceinline__ void gemm_epilogue4(const GemmArgs& a, const GemmGroup& g, int m, int n,
                                               const float (&v)[4], int nv, const float* bias4) {
  typedef __nv_bfloat16 T;
  const long long row = (long long)g.b_row0 + n;
  bool vec = nv == 4;
  if constexpr (EPI == kEpiStore || EPI == kEpiBiasSilu || EPI == kEpiAct)
    vec = vec && (m + 3 < a.epi_split || m >= a.epi_split);
  if constexpr (EPI == kEpiScores || EPI == kEpiScoresFolded) {
    if (EPI == kEpiScoresFolded && m >= a.epi_split) {
      const long long o2 = row * a.ldc2 + (m - a.epi_split);
      if (vec && (o2 & 3) == 0) {
        *reinterpret_cast<float4*>(static_cast<float*>(a.out2) + o2) = make_float4(v[0], v[1], v[2], v[3]);
        return;
      }
    }
    const int stride = EPI == kEpiScoresFolded ? min(g.m, a.epi_split) : g.m;
    const long long o = g.c_off + (long long)n * stride + m;
    if (vec && (o & 3) == 0 && (EPI != kEpiScoresFolded || m + 3 < a.epi_split)) {
      const float rs = a.row_scale ? a.row_scale[g.b_row0 + n] : 1.0f;
      *reinterpret_cast<float4*>(static_cast<float*>(a.out0) + o) =
          make_float4(v[0] * a.scale * rs, v[1] * a.scale * rs, v[2] * a.scale * rs,
                      v[3] * a.scale * rs);
      return;
    }
  } else if constexpr (EPI == kEpiBiasF32) {
    const long long o = row * a.ldc + m;
    if (vec && (o & 3) == 0) {
      *reinterpret_cast<float4*>(static_cast<float*>(a.out0) + o) =
          make_float4(v[0] + bias4[0], v[1] + bias4[1], v[2] + bias4[2], v[3] + bias4[3]);
      return;
    }
  } else if constexpr (EPI == kEpiStoreHiLo || EPI == kEpiQueryH) {
    if (EPI == kEpiQueryH && m >= a.epi_split) {
      const long long o = row * a.ldc2 + (m - a.epi_split);
      if (vec && (o & 3) == 0) {
        *reinterpret_cast<float4*>(static_cast<float*>(a.out2) + o) = make_float4(v[0], v[1], v[2], v[3]);
        return;
      }
    }
    const long long o = row * a.ldc + m;
    if (vec && (o & 3) == 0 && (EPI != kEpiQueryH || m + 3 < a.epi_split)) {
      T hi[4], lo[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        hi[j] = from_f32<T>(v[j]);
        lo[j] = from_f32<T>(v[j] - to_f32(hi[j]));
      }
      *reinterpret_cast<uint2*>(static_cast<T*>(a.out0) + o) = *reinterpret_cast<const uint2*>(hi);
      *reinterpret_cast<uint2*>(static_cast<T*>(a.out1) + o) = *reinterpret_cast<const uint2*>(lo);
      return;
    }
  } else if constexpr (EPI == kEpiBiasSilu || EPI == kEpiAct) {
    const long long o = row * a.ldc + m;
    if (vec && (o & 3) == 0) {
      float add[4] = {0.0f, 0.0f, 0.0f, 0.0f};
      if constexpr (EPI == kEpiAct) {
        const float4 a4 = *reinterpret_cast<const float4*>(a.add_in + row * a.ldc2 + m);
        add[0] = a4.x; add[1] = a4.y; add[2] = a4.z; add[3] = a4.w;
      }
      T r[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const float z = v[j] + bias4[j] + add[j];
        r[j] = from_f32<T>(z * sigmoidf_(z));
      }
      *reinterpret_cast<uint2*>(static_cast<T*>(a.out0) + o) = *reinterpret_cast<const uint2*>(r);
      return;
    }
  } else if constexpr (EPI == kEpiStore) {
    const long long o = m < a.epi_split ? row * a.ldc + m : row * a.ldc + (m - a.epi_split);
    if (vec && (o & 3) == 0) {
      T r[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) r[j] = from_f32<T>(v[j]);
      T* out = m < a.epi_split ? static_cast<T*>(a.out0) : static_cast<T*>(a.out1);
      *reinterpret_cast<uint2*>(out + o) = *reinterpret_cast<const uint2*>(r);
      return;
    }
  }
#pragma unroll
  for (int j = 0; j < 4; ++j)
    if (j < nv) gemm_epilogue<T, EPI>(a, g, m + j, n, v[j]);
}

}  // namespace fovea
