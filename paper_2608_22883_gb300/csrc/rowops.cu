// Row-wise kernels of the FOVEA path: LayerNorm (+ depth embedding), mask
// compaction, the gather-and-weighted-sum readout, and the gate + gated
// residual + RMSNorm finalisation.
#include "common.cuh"
#include "dfloat.cuh"

namespace fovea {

// ---------------------------------------------------------------------------
// LN over rows of d elements (memory equation: LN(v_i); query equation:
// LN(h_n) + E_dep[l_n]).  One CTA per row; the row stays in registers.
// Mean, variance, 1/sqrt and the affine map are evaluated in double-float so
// the single rounding to the stored type is taken on an almost exact value
// (the same value a float64 evaluation rounds).  Optional gather of source
// rows, optional depth embedding (depth checked against [0, D]; an invalid
// depth sets kErrDepth and uses depth 0).
// ---------------------------------------------------------------------------
constexpr int kLnThreads = 256;
constexpr int kLnMaxPerThread = FOVEA_MAX_D / kLnThreads;

__device__ __forceinline__ dfloat block_sum_df(dfloat v, dfloat* scratch) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const dfloat t = {__shfl_xor_sync(0xffffffffu, v.hi, o), __shfl_xor_sync(0xffffffffu, v.lo, o)};
    v = df_add(v, t);
  }
  __syncthreads();
  if (lane == 0) scratch[warp] = v;
  __syncthreads();
  dfloat t = lane < nw ? scratch[lane] : dfloat{0.0f, 0.0f};
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const dfloat u = {__shfl_xor_sync(0xffffffffu, t.hi, o), __shfl_xor_sync(0xffffffffu, t.lo, o)};
    t = df_add(t, u);
  }
  return t;
}

template <class T> __device__ __forceinline__ T df_store(dfloat y);
template <> __device__ __forceinline__ float df_store<float>(dfloat y) { return y.hi; }
template <> __device__ __forceinline__ __nv_bfloat16 df_store<__nv_bfloat16>(dfloat y) {
  return df_to_bf16(y);
}

template <class T>
__global__ void __launch_bounds__(kLnThreads) ln_rows_kernel(
    const T* __restrict__ x, const int32_t* __restrict__ src_row, int d,
    const T* __restrict__ gamma, const T* __restrict__ beta, float eps,
    const T* __restrict__ E, const int32_t* __restrict__ depth, int max_depth, int* err,
    T* __restrict__ out) {
  __shared__ dfloat scratch[32];
  const int row = blockIdx.x;
  const long long src = src_row ? (long long)src_row[row] : (long long)row;
  const T* xr = x + src * d;
  float vals[kLnMaxPerThread];
  dfloat s = {0.0f, 0.0f};
#pragma unroll
  for (int j = 0; j < kLnMaxPerThread; ++j) {
    const int i = threadIdx.x + j * kLnThreads;
    vals[j] = i < d ? to_f32(xr[i]) : 0.0f;
    s = df_add_f(s, vals[j]);
  }
  const dfloat mean = df_div_f(block_sum_df(s, scratch), (float)d);
  const dfloat neg_mean = {-mean.hi, -mean.lo};
  dfloat ss = {0.0f, 0.0f};
#pragma unroll
  for (int j = 0; j < kLnMaxPerThread; ++j) {
    const int i = threadIdx.x + j * kLnThreads;
    if (i < d) {
      const dfloat c = df_add_f(neg_mean, vals[j]);
      ss = df_add(ss, df_mul(c, c));
    }
  }
  const dfloat var = df_div_f(block_sum_df(ss, scratch), (float)d);
  const dfloat rstd = df_rsqrt(df_add_f(var, eps));
  int dep = 0;
  if (E != nullptr) {
    dep = depth[row];
    if (dep < 0 || dep > max_depth) {
      if (threadIdx.x == 0) atomicOr(err, kErrDepth);
      dep = 0;
    }
  }
  T* o = out + (long long)row * d;
#pragma unroll
  for (int j = 0; j < kLnMaxPerThread; ++j) {
    const int i = threadIdx.x + j * kLnThreads;
    if (i < d) {
      dfloat y = df_mul(df_add_f(neg_mean, vals[j]), rstd);
      y = df_add_f(df_mul_f(y, to_f32(gamma[i])), to_f32(beta[i]));
      if (E != nullptr) y = df_add_f(y, to_f32(E[(long long)dep * d + i]));
      o[i] = df_store<T>(y);
    }
  }
}

cudaError_t launch_ln_rows(int dtype, const void* x, const int32_t* src_row, int rows, int d,
                           const void* gamma, const void* beta, float eps, const void* E,
                           const int32_t* depth, int max_depth, int* err, void* out,
                           cudaStream_t s) {
  if (rows == 0) return cudaSuccess;
  if (dtype == FOVEA_BF16) {
    using T = __nv_bfloat16;
    ln_rows_kernel<T><<<rows, kLnThreads, 0, s>>>((const T*)x, src_row, d, (const T*)gamma,
                                                  (const T*)beta, eps, (const T*)E, depth,
                                                  max_depth, err, (T*)out);
  } else {
    ln_rows_kernel<float><<<rows, kLnThreads, 0, s>>>((const float*)x, src_row, d,
                                                      (const float*)gamma, (const float*)beta,
                                                      eps, (const float*)E, depth, max_depth,
                                                      err, (float*)out);
  }
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Mask compaction (memory validity m_i and the valid set V): per-image valid
// counts, then an ordered compaction of valid positions.
// ---------------------------------------------------------------------------
constexpr int kScanThreads = 256;

__global__ void __launch_bounds__(kScanThreads) count_valid_kernel(const uint8_t* __restrict__ mask,
                                                                  int M_max,
                                                                  int32_t* __restrict__ counts) {
  __shared__ float scratch[32];
  const int b = blockIdx.x;
  int c = 0;
  for (int i = threadIdx.x; i < M_max; i += kScanThreads)
    c += mask[(long long)b * M_max + i] != 0;
  const float tot = block_sum((float)c, scratch);   // exact: counts < 2^24
  if (threadIdx.x == 0) counts[b] = (int32_t)tot;
}

__global__ void __launch_bounds__(kScanThreads) compact_kernel(const uint8_t* __restrict__ mask,
                                                              int M_max,
                                                              const int32_t* __restrict__ key_off,
                                                              int32_t* __restrict__ orig_index,
                                                              int32_t* __restrict__ src_row) {
  __shared__ int warp_tot[kScanThreads / 32];
  const int b = blockIdx.x;
  const int chunk = (M_max + kScanThreads - 1) / kScanThreads;
  const int beg = min(M_max, threadIdx.x * chunk), end = min(M_max, beg + chunk);
  const uint8_t* mb = mask ? mask + (long long)b * M_max : nullptr;
  int c = 0;
  for (int i = beg; i < end; ++i) c += mb ? (mb[i] != 0) : 1;
  // exclusive scan of c over the block (thread order = position order)
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int incl = c;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int t = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += t;
  }
  if (lane == 31) warp_tot[warp] = incl;
  __syncthreads();
  int base = 0;
  for (int w = 0; w < warp; ++w) base += warp_tot[w];
  int rank = base + incl - c;
  const int off = key_off[b];
  for (int i = beg; i < end; ++i) {
    if (mb == nullptr || mb[i] != 0) {
      orig_index[off + rank] = i;
      src_row[off + rank] = b * M_max + i;
      ++rank;
    }
  }
}

cudaError_t launch_count_valid(const uint8_t* mask, int B, int M_max, int32_t* counts,
                               cudaStream_t s) {
  count_valid_kernel<<<B, kScanThreads, 0, s>>>(mask, M_max, counts);
  return cudaGetLastError();
}

cudaError_t launch_compact(const uint8_t* mask, int B, int M_max, const int32_t* key_off,
                           int32_t* orig_index, int32_t* src_row, cudaStream_t s) {
  compact_kernel<<<B, kScanThreads, 0, s>>>(mask, M_max, key_off, orig_index, src_row);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Readout r_n = sum_{t < K} alpha_t u_{pi(t)} (the alpha / r_n equation).
// Grid (N, column chunks); each thread owns one 16-byte vector of columns
// and walks the selected entries in pi order (fp32 accumulation, fixed
// order).  The weights were renormalised over I_n by the select kernel.
// ---------------------------------------------------------------------------
constexpr int kReadoutThreads = 128;

template <class T>
struct Vec16;
template <> struct Vec16<__nv_bfloat16> { static constexpr int N = 8; };
template <> struct Vec16<float> { static constexpr int N = 4; };

template <class T>
__device__ __forceinline__ void load_vec(const T* p, float (&v)[Vec16<T>::N]);
template <>
__device__ __forceinline__ void load_vec<__nv_bfloat16>(const __nv_bfloat16* p, float (&v)[8]) {
  const uint4 raw = __ldg(reinterpret_cast<const uint4*>(p));
  const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&raw);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 f = __bfloat1622float2(h2[i]);
    v[2 * i] = f.x;
    v[2 * i + 1] = f.y;
  }
}
template <>
__device__ __forceinline__ void load_vec<float>(const float* p, float (&v)[4]) {
  const float4 raw = __ldg(reinterpret_cast<const float4*>(p));
  v[0] = raw.x; v[1] = raw.y; v[2] = raw.z; v[3] = raw.w;
}

template <class T>
__global__ void __launch_bounds__(kReadoutThreads) readout_kernel(
    const T* __restrict__ U, const int32_t* __restrict__ sel_cnt,
    const int32_t* __restrict__ sel_pos, const float* __restrict__ sel_w, int k_max, int d,
    float* __restrict__ r_out, T* __restrict__ r_lo) {
  constexpr int V = Vec16<T>::N;
  const int n = blockIdx.x;
  const int col = (blockIdx.y * kReadoutThreads + threadIdx.x) * V;
  if (col >= d) return;
  const int K = sel_cnt[n];
  const int32_t* pos = sel_pos + (long long)n * k_max;
  const float* w = sel_w + (long long)n * k_max;
  float acc[V];
#pragma unroll
  for (int i = 0; i < V; ++i) acc[i] = 0.0f;
  int t = 0;
  for (; t + 4 <= K; t += 4) {
    float u0[V], u1[V], u2[V], u3[V];
    load_vec<T>(U + (long long)pos[t] * d + col, u0);
    load_vec<T>(U + (long long)pos[t + 1] * d + col, u1);
    load_vec<T>(U + (long long)pos[t + 2] * d + col, u2);
    load_vec<T>(U + (long long)pos[t + 3] * d + col, u3);
    const float w0 = w[t], w1 = w[t + 1], w2 = w[t + 2], w3 = w[t + 3];
#pragma unroll
    for (int i = 0; i < V; ++i) {
      acc[i] = fmaf(w0, u0[i], acc[i]);
      acc[i] = fmaf(w1, u1[i], acc[i]);
      acc[i] = fmaf(w2, u2[i], acc[i]);
      acc[i] = fmaf(w3, u3[i], acc[i]);
    }
  }
  for (; t < K; ++t) {
    float u0[V];
    load_vec<T>(U + (long long)pos[t] * d + col, u0);
    const float w0 = w[t];
#pragma unroll
    for (int i = 0; i < V; ++i) acc[i] = fmaf(w0, u0[i], acc[i]);
  }
  if (r_out != nullptr) {
#pragma unroll
    for (int i = 0; i < V; ++i) r_out[(long long)n * d + col + i] = acc[i];
  }
#pragma unroll
  for (int i = 0; i < V; ++i) r_lo[(long long)n * d + col + i] = from_f32<T>(acc[i]);
}

cudaError_t launch_readout(int dtype, const void* U, const int32_t* sel_cnt, const int32_t* sel_pos,
                           const float* sel_w, int N, int k_max, int d, float* r_out, void* r_lo,
                           cudaStream_t s) {
  if (N == 0) return cudaSuccess;
  if (dtype == FOVEA_BF16) {
    using T = __nv_bfloat16;
    dim3 grid(N, (d / 8 + kReadoutThreads - 1) / kReadoutThreads);
    readout_kernel<T><<<grid, kReadoutThreads, 0, s>>>((const T*)U, sel_cnt, sel_pos, sel_w, k_max,
                                                       d, r_out, (T*)r_lo);
  } else {
    dim3 grid(N, (d / 4 + kReadoutThreads - 1) / kReadoutThreads);
    readout_kernel<float><<<grid, kReadoutThreads, 0, s>>>((const float*)U, sel_cnt, sel_pos,
                                                           sel_w, k_max, d, r_out, (float*)r_lo);
  }
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Exact rounding of listed key elements (memory equation k_i = W_K LN(v_i)):
// one warp per element; products of two bf16 values are exact in fp32 and are
// summed in double-float, then rounded once.
// ---------------------------------------------------------------------------
constexpr int kRefineThreads = 256;

__global__ void __launch_bounds__(kRefineThreads) refine_keys_kernel(
    const __nv_bfloat16* __restrict__ xv, const __nv_bfloat16* __restrict__ W, int d,
    const KeyFix* __restrict__ list, const int* __restrict__ count, int cap, long long total,
    __nv_bfloat16* __restrict__ K) {
  const int lane = threadIdx.x & 31;
  const long long warps = (long long)gridDim.x * (kRefineThreads / 32);
  const long long n_items = list ? (long long)min(*count, cap) : total;
  for (long long it = blockIdx.x * (kRefineThreads / 32) + (threadIdx.x >> 5); it < n_items;
       it += warps) {
    long long row;
    int col;
    if (list) {
      row = list[it].row;
      col = list[it].col;
    } else {
      row = it / d;
      col = (int)(it % d);
    }
    const __nv_bfloat16* x = xv + row * d;
    const __nv_bfloat16* w = W + (long long)col * d;
    dfloat acc = {0.0f, 0.0f};
    for (int l = lane; l < d; l += 32) {
      const float p = __bfloat162float(x[l]) * __bfloat162float(w[l]);   // exact
      acc = df_add_f(acc, p);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const dfloat t = {__shfl_xor_sync(0xffffffffu, acc.hi, o), __shfl_xor_sync(0xffffffffu, acc.lo, o)};
      acc = df_add(acc, t);
    }
    if (lane == 0) K[row * d + col] = df_to_bf16(acc);
  }
}

cudaError_t launch_refine_keys(const void* xv, const void* W, int d, const KeyFix* list,
                               const int* count, int cap, int rows, void* K, cudaStream_t s) {
  const long long total = (long long)rows * d;
  if (total == 0) return cudaSuccess;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  refine_keys_kernel<<<sms * 8, kRefineThreads, 0, s>>>(
      (const __nv_bfloat16*)xv, (const __nv_bfloat16*)W, d, list, count, cap, total,
      (__nv_bfloat16*)K);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Gate, gated residual and RMSNorm (Eq. hidden_correction):
// g = sigma(a_g . w_g2 + b_g2), y = h + g c, h_hat = y / sqrt(mean(y^2) + eps) * gamma.
// One CTA per row; `act` is [N, 2H] with a_f in columns 0..H-1 and a_g in H..2H-1.
// ---------------------------------------------------------------------------
constexpr int kFinThreads = 256;

template <class T>
__global__ void __launch_bounds__(kFinThreads) finalize_kernel(
    const T* __restrict__ h, const float* __restrict__ c, const T* __restrict__ act, int H, int d,
    const T* __restrict__ w_g2, const T* __restrict__ b_g2, const T* __restrict__ rms_gamma,
    float eps, T* __restrict__ h_out, float* __restrict__ gate_out) {
  __shared__ float scratch[32];
  const int n = blockIdx.x;
  const T* a_g = act + (long long)n * 2 * H + H;
  float part = 0.0f;
  for (int j = threadIdx.x; j < H; j += kFinThreads) part = fmaf(to_f32(a_g[j]), to_f32(w_g2[j]), part);
  const float z = block_sum(part, scratch) + to_f32(b_g2[0]);
  const float g = sigmoidf_(z);
  float y[kLnMaxPerThread];
  float ss = 0.0f;
#pragma unroll
  for (int j = 0; j < kLnMaxPerThread; ++j) {
    const int i = threadIdx.x + j * kFinThreads;
    y[j] = 0.0f;
    if (i < d) {
      y[j] = fmaf(g, c[(long long)n * d + i], to_f32(h[(long long)n * d + i]));
      ss = fmaf(y[j], y[j], ss);
    }
  }
  const float tot = block_sum(ss, scratch);
  const float inv = 1.0f / sqrtf(tot / (float)d + eps);
#pragma unroll
  for (int j = 0; j < kLnMaxPerThread; ++j) {
    const int i = threadIdx.x + j * kFinThreads;
    if (i < d) h_out[(long long)n * d + i] = from_f32<T>(y[j] * inv * to_f32(rms_gamma[i]));
  }
  if (gate_out != nullptr && threadIdx.x == 0) gate_out[n] = g;
}

cudaError_t launch_finalize(int dtype, const void* h, const float* c, const void* act, int H, int d,
                            const void* w_g2, const void* b_g2, const void* rms_gamma, float eps,
                            int N, void* h_out, float* gate_out, cudaStream_t s) {
  if (N == 0) return cudaSuccess;
  if (dtype == FOVEA_BF16) {
    using T = __nv_bfloat16;
    finalize_kernel<T><<<N, kFinThreads, 0, s>>>((const T*)h, c, (const T*)act, H, d,
                                                 (const T*)w_g2, (const T*)b_g2,
                                                 (const T*)rms_gamma, eps, (T*)h_out, gate_out);
  } else {
    finalize_kernel<float><<<N, kFinThreads, 0, s>>>((const float*)h, c, (const float*)act, H, d,
                                                     (const float*)w_g2, (const float*)b_g2,
                                                     (const float*)rms_gamma, eps, (float*)h_out,
                                                     gate_out);
  }
  return cudaGetLastError();
}

}  // namespace fovea
