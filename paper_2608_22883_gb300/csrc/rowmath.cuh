// Row helpers shared by the row kernels (LN, readout, finalize):
// 16-byte vector loads of a row segment, the double-float warp sum, and the
// single rounding of a double-float value to the stored type.
#pragma once
#include "common.cuh"
#include "dfloat.cuh"

namespace fovea {

template <class T> struct VecOf;      // elements in one 16-byte vector
template <> struct VecOf<__nv_bfloat16> { static constexpr int N = 8; };
template <> struct VecOf<float> { static constexpr int N = 4; };

template <class T>
__device__ __forceinline__ void ln_load(const T* p, float (&v)[VecOf<T>::N]);
template <>
__device__ __forceinline__ void ln_load<__nv_bfloat16>(const __nv_bfloat16* p, float (&v)[8]) {
  const uint4 raw = *reinterpret_cast<const uint4*>(p);
  const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&raw);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 f = __bfloat1622float2(h2[i]);
    v[2 * i] = f.x;
    v[2 * i + 1] = f.y;
  }
}
template <>
__device__ __forceinline__ void ln_load<float>(const float* p, float (&v)[4]) {
  const float4 raw = *reinterpret_cast<const float4*>(p);
  v[0] = raw.x; v[1] = raw.y; v[2] = raw.z; v[3] = raw.w;
}

// The 16-byte vector `raw` (as loaded) widened to fp32.
template <class T>
__device__ __forceinline__ void ln_unpack(const uint4& raw, float (&v)[VecOf<T>::N]);
template <>
__device__ __forceinline__ void ln_unpack<__nv_bfloat16>(const uint4& raw, float (&v)[8]) {
  const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&raw);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 f = __bfloat1622float2(h2[i]);
    v[2 * i] = f.x;
    v[2 * i + 1] = f.y;
  }
}
template <>
__device__ __forceinline__ void ln_unpack<float>(const uint4& raw, float (&v)[4]) {
  v[0] = __uint_as_float(raw.x); v[1] = __uint_as_float(raw.y);
  v[2] = __uint_as_float(raw.z); v[3] = __uint_as_float(raw.w);
}

template <class T> __device__ __forceinline__ T df_store(dfloat y);
template <> __device__ __forceinline__ float df_store<float>(dfloat y) { return y.hi; }
template <> __device__ __forceinline__ __nv_bfloat16 df_store<__nv_bfloat16>(dfloat y) {
  return df_to_bf16(y);
}

__device__ __forceinline__ dfloat warp_sum_df(dfloat v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const dfloat t = {__shfl_xor_sync(0xffffffffu, v.hi, o), __shfl_xor_sync(0xffffffffu, v.lo, o)};
    v = df_add(v, t);
  }
  return v;
}

}  // namespace fovea
