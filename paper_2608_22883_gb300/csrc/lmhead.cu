// Draft logits and tree-expansion candidates: z_n = W_LM h_hat_n (Eq.
// hidden_correction) and, per row, the K_c largest logits in descending
// order, ties broken by the smaller token index (the candidate width K_c of
// the experimental setup).  The logits come from the tensor-core GEMM
// (gemm_tc.cu) streaming W_LM, whose epilogue also keeps, per row and tile,
// the K_c largest of the tile's logits; this file merges those candidates.
#include "common.cuh"

namespace fovea {

namespace {

constexpr int kMergeThreads = 256;   // registers: up to FOVEA_MAX_KC 64-bit keys per thread

// One CTA per row over the row's candidate keys (each the cand_k largest of
// one GEMM tile's columns, as logit order key << 32 | ~token: distinct, and
// on equal logits the smaller token is larger).  Each thread keeps the k
// largest of its strided keys in KC register slots (KC >= k, a compile-time
// size so the slots stay in registers), unsorted, with the position of the
// smallest; then k rounds of a block-wide maximum, the owner clearing the
// winner.  A zero key (a tile with fewer columns than k) is below every real
// one.  The logit is recovered from the key (the order map is a bijection).
template <int KC>
__global__ void __launch_bounds__(kMergeThreads) merge_candidates_kernel(
    const unsigned long long* __restrict__ cand, int total, int k, int32_t* __restrict__ top_idx,
    float* __restrict__ top_val) {
  __shared__ unsigned long long red[kMergeThreads / 32];
  __shared__ unsigned long long best;
  const int n = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const unsigned long long* c = cand + (long long)n * total;
  pdl_wait();
  pdl_trigger();
  unsigned long long loc[KC];
#pragma unroll
  for (int i = 0; i < KC; ++i) loc[i] = 0ull;
  unsigned long long lowest = 0ull;           // the smallest of slots 0 .. k-1
  int low_pos = 0;
  constexpr int kBatch = 4;
  for (int j0 = tid; j0 < total; j0 += kBatch * kMergeThreads) {
    unsigned long long v[kBatch];
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
      const int j = j0 + u * kMergeThreads;
      v[u] = j < total ? c[j] : 0ull;
    }
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
      const unsigned long long key = v[u];
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
      m = lane < kMergeThreads / 32 ? red[lane] : 0ull;
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
      const uint32_t key = (uint32_t)(b >> 32);
      const uint32_t bits = (key & 0x80000000u) ? (key & 0x7FFFFFFFu) : ~key;
      top_idx[(long long)n * k + r] = (int32_t)(0xFFFFFFFFu - (uint32_t)(b & 0xFFFFFFFFull));
      if (top_val != nullptr) top_val[(long long)n * k + r] = __uint_as_float(bits);
    }
  }
}

}  // namespace

cudaError_t launch_merge_candidates(const unsigned long long* cand, int N, int slots, int k,
                                    int32_t* top_idx, float* top_val, cudaStream_t s) {
  if (N == 0) return cudaSuccess;
  if (k < 1 || k > FOVEA_MAX_KC || slots < 1) return cudaErrorInvalidValue;
  const int total = slots * k;
  if (k <= 8)
    return launch_pdl(merge_candidates_kernel<8>, dim3(N), dim3(kMergeThreads), 0, s, cand, total,
                      k, top_idx, top_val);
  return launch_pdl(merge_candidates_kernel<FOVEA_MAX_KC>, dim3(N), dim3(kMergeThreads), 0, s, cand,
                    total, k, top_idx, top_val);
}

}  // namespace fovea
