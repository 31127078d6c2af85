// Double-float arithmetic (a value carried as an unevaluated sum hi + lo of
// two fp32 numbers, about 48 significant bits) built from the error-free
// transformations of Knuth (TwoSum), Dekker (Fast2Sum) and the FMA product
// error.  Used where a value is rounded to bf16 right after it is computed, so
// that the rounding decision is taken on an (almost) exact value instead of
// an fp32 approximation: GB300's native fp64 rate is too low for the per-step
// path.  Nothing here may be reassociated; nvcc does not reassociate fp32
// additions without fast-math flags.
#pragma once
#include <cuda_bf16.h>
#include <stdint.h>

namespace fovea {

struct dfloat {
  float hi, lo;
};

__device__ __forceinline__ dfloat df_two_sum(float a, float b) {        // Knuth
  const float s = __fadd_rn(a, b);
  const float bb = __fsub_rn(s, a);
  const float e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
  return {s, e};
}
__device__ __forceinline__ dfloat df_fast_two_sum(float a, float b) {   // Dekker, |a| >= |b|
  const float s = __fadd_rn(a, b);
  return {s, __fsub_rn(b, __fsub_rn(s, a))};
}
__device__ __forceinline__ dfloat df_two_prod(float a, float b) {
  const float p = __fmul_rn(a, b);
  return {p, __fmaf_rn(a, b, -p)};
}
__device__ __forceinline__ dfloat df_add(dfloat a, dfloat b) {
  dfloat s = df_two_sum(a.hi, b.hi);
  const dfloat t = df_two_sum(a.lo, b.lo);
  s.lo = __fadd_rn(s.lo, t.hi);
  s = df_fast_two_sum(s.hi, s.lo);
  s.lo = __fadd_rn(s.lo, t.lo);
  return df_fast_two_sum(s.hi, s.lo);
}
__device__ __forceinline__ dfloat df_add_f(dfloat a, float b) {
  dfloat s = df_two_sum(a.hi, b);
  s.lo = __fadd_rn(s.lo, a.lo);
  return df_fast_two_sum(s.hi, s.lo);
}
__device__ __forceinline__ dfloat df_mul(dfloat a, dfloat b) {
  dfloat p = df_two_prod(a.hi, b.hi);
  p.lo = __fmaf_rn(a.hi, b.lo, __fmaf_rn(a.lo, b.hi, p.lo));
  return df_fast_two_sum(p.hi, p.lo);
}
__device__ __forceinline__ dfloat df_mul_f(dfloat a, float b) {
  dfloat p = df_two_prod(a.hi, b);
  p.lo = __fmaf_rn(a.lo, b, p.lo);
  return df_fast_two_sum(p.hi, p.lo);
}
// a / b for a float divisor: one correction step of the quotient.
__device__ __forceinline__ dfloat df_div_f(dfloat a, float b) {
  const float q1 = __fdiv_rn(a.hi, b);
  const dfloat p = df_two_prod(q1, b);
  const dfloat r = df_add(a, dfloat{-p.hi, -p.lo});
  const float q2 = __fdiv_rn(r.hi, b);
  return df_fast_two_sum(q1, q2);
}
// 1 / sqrt(a) for a > 0: an fp32 seed and two Newton steps in double-float,
// r <- r + r (1 - a r^2) / 2.
__device__ __forceinline__ dfloat df_rsqrt(dfloat a) {
  dfloat r = {__fdiv_rn(1.0f, __fsqrt_rn(a.hi)), 0.0f};
#pragma unroll
  for (int it = 0; it < 2; ++it) {
    const dfloat r2 = df_mul(r, r);
    const dfloat ar2 = df_mul(a, r2);
    const dfloat e = df_add_f(dfloat{-ar2.hi, -ar2.lo}, 1.0f);
    r = df_add(r, df_mul_f(df_mul(r, e), 0.5f));
  }
  return r;
}

// Round hi + lo to the nearest bf16 (ties to even).  bf16 rounding of hi alone
// is exact unless hi sits exactly on a bf16 midpoint, where lo decides.
__device__ __forceinline__ __nv_bfloat16 df_to_bf16(dfloat a) {
  const uint32_t u = __float_as_uint(a.hi);
  if ((u & 0xFFFFu) == 0x8000u && a.lo != 0.0f && (u & 0x7F800000u) != 0x7F800000u) {
    // exactly halfway between two bf16 values: move toward the sign of lo
    const bool away = (a.lo > 0.0f) == (a.hi > 0.0f);
    const uint32_t t = away ? (u + 0x8000u) : (u - 0x8000u);
    return __ushort_as_bfloat16((unsigned short)(t >> 16));
  }
  return __float2bfloat16_rn(a.hi);
}

}  // namespace fovea
