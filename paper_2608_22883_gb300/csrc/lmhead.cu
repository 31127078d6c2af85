// Draft logits and tree-expansion candidates: z_n = W_LM h_hat_n (Eq.
// hidden_correction) and, per row, the K_c largest logits in descending
// order, ties broken by the smaller token index (the candidate width K_c of
// the experimental setup).  The logits come from the tensor-core GEMM
// (gemm_tc.cu) streaming W_LM; this file holds the per-row candidate
// selection.
#include "common.cuh"

namespace fovea {

namespace {

constexpr int kTopKThreads = 256;    // registers: up to FOVEA_MAX_KC 64-bit keys per thread
constexpr int kBatch = 16;           // logits loaded together per thread

// Order-preserving map of a float to an unsigned key (larger float, larger key).
__device__ __forceinline__ uint32_t logit_key(float f) {
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// One CTA per row.  Each thread keeps the k largest of its strided logits as
// 64-bit keys (logit key << 32 | ~index: distinct, and on equal logits the
// smaller index is larger) in KC register slots (KC >= k, a compile-time
// size so the slots stay in registers), unsorted, with the position of the
// smallest: a larger key replaces the smallest.  Then k rounds of a
// block-wide maximum over the threads' largest keys, the owner clearing the
// winner.  A zero key is below every real one (the key of -inf is
// 0x007FFFFF in the upper half); slots k .. KC-1 stay zero.
template <int KC>
__global__ void __launch_bounds__(kTopKThreads) topk_rows_kernel(const float* __restrict__ logits,
                                                                long long V, int k,
                                                                int32_t* __restrict__ top_idx,
                                                                float* __restrict__ top_val) {
  __shared__ unsigned long long red[kTopKThreads / 32];
  __shared__ unsigned long long best;
  const int n = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const float* z = logits + (long long)n * V;
  pdl_wait();
  pdl_trigger();
  unsigned long long loc[KC];
#pragma unroll
  for (int i = 0; i < KC; ++i) loc[i] = 0ull;
  unsigned long long lowest = 0ull;           // the smallest of slots 0 .. k-1
  int low_pos = 0;
  // the thread's logits in batches of kBatch, every load of a batch in
  // flight before the first comparison
  for (long long j0 = tid; j0 < V; j0 += (long long)kBatch * kTopKThreads) {
    float v[kBatch];
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
      const long long j = j0 + (long long)u * kTopKThreads;
      v[u] = j < V ? z[j] : 0.0f;
    }
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
      const long long j = j0 + (long long)u * kTopKThreads;
      if (j >= V) continue;
      const unsigned long long key =
          ((unsigned long long)logit_key(v[u]) << 32) | (0xFFFFFFFFu - (uint32_t)j);
      if (key <= lowest) continue;
#pragma unroll
      for (int i = 0; i < KC; ++i)
        if (i == low_pos) loc[i] = key;
      lowest = loc[0];
      low_pos = 0;
#pragma unroll
      for (int i = 1; i < KC; ++i)
        if (i < k && loc[i] < lowest) {
          lowest = loc[i];
          low_pos = i;
        }
    }
  }
  for (int r = 0; r < k; ++r) {
    unsigned long long mine = loc[0];
    int mine_pos = 0;
#pragma unroll
    for (int i = 1; i < KC; ++i)
      if (loc[i] > mine) {
        mine = loc[i];
        mine_pos = i;
      }
    unsigned long long m = mine;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const unsigned long long t = __shfl_xor_sync(0xffffffffu, m, o);
      m = t > m ? t : m;
    }
    if (lane == 0) red[warp] = m;
    __syncthreads();
    if (warp == 0) {
      m = lane < kTopKThreads / 32 ? red[lane] : 0ull;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const unsigned long long t = __shfl_xor_sync(0xffffffffu, m, o);
        m = t > m ? t : m;
      }
      if (lane == 0) best = m;
    }
    __syncthreads();
    const unsigned long long b = best;
    if (mine == b && b != 0ull) {             // the owner clears the winner
#pragma unroll
      for (int i = 0; i < KC; ++i)
        if (i == mine_pos) loc[i] = 0ull;
    }
    if (tid == 0) {
      const uint32_t j = 0xFFFFFFFFu - (uint32_t)(b & 0xFFFFFFFFull);
      top_idx[(long long)n * k + r] = (int32_t)j;
      if (top_val != nullptr) top_val[(long long)n * k + r] = z[j];
    }
  }
}

}  // namespace

cudaError_t launch_topk_rows(const float* logits, int N, long long V, int k, int32_t* top_idx,
                             float* top_val, cudaStream_t s) {
  if (N == 0) return cudaSuccess;
  if (k < 1 || k > FOVEA_MAX_KC || V < k) return cudaErrorInvalidValue;
  if (k <= 8)
    return launch_pdl(topk_rows_kernel<8>, dim3(N), dim3(kTopKThreads), 0, s, logits, V, k,
                      top_idx, top_val);
  return launch_pdl(topk_rows_kernel<FOVEA_MAX_KC>, dim3(N), dim3(kTopKThreads), 0, s, logits, V,
                    k, top_idx, top_val);
}

}  // namespace fovea
