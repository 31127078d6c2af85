// Cumulative-mass selection kernel: one CTA of 256 threads per draft state
// (the algorithm is in select_core.cuh).  The row's scores are staged in
// shared memory first.
#include "select_core.cuh"

namespace fovea {

struct BlockSync {
  __device__ __forceinline__ void operator()() const { __syncthreads(); }
};

__global__ void __launch_bounds__(kSelThreads) select_kernel(const __grid_constant__ SelectArgs a,
                                                             const __grid_constant__ SeqTable tab) {
  extern __shared__ float s_sc[];                            // [M] scores of this row
  __shared__ SelectSmem sm;
  const int n = blockIdx.x;
  const int tid = threadIdx.x;
  pdl_wait();
  pdl_trigger();
  const int b = seq_of_row(tab, n);
  const int M = tab.m[b];
  if (M == 0) {                           // empty valid set: K = 0, nothing selected
    select_empty(a, n, tid);
    return;
  }
  const float* src = a.scores + tab.score_off[b] + (long long)(n - tab.row_start[b]) * M;
  for (int i = tid; i < M; i += kSelThreads) {
    float v = src[i];
    if (v == 0.0f) v = 0.0f;              // -0 -> +0 so equal scores get equal keys
    s_sc[i] = v;
  }
  __syncthreads();
  select_row(a, n, M, tab.key_off[b], s_sc, sm, tid, BlockSync{});
}

cudaError_t launch_select(const float* scores, const SeqTable& tab, int N, const int32_t* orig_index,
                          float rho, int k_min, int k_max, int max_m, int32_t* counts,
                          int32_t* indices, int32_t* sel_pos, float* sel_w, int32_t* sel_cnt,
                          cudaStream_t s) {
  if (N == 0) return cudaSuccess;
  const size_t smem = (size_t)max(max_m, 1) * sizeof(float);
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         FOVEA_MAX_ENTRIES * (int)sizeof(float));
    if (e != cudaSuccess) return e;
    configured = true;
  }
  SelectArgs a{scores, orig_index, rho, k_min, k_max, counts, indices, sel_pos, sel_w, sel_cnt};
  return launch_pdl(select_kernel, dim3(N), dim3(kSelThreads), smem, s, a, tab);
}

}  // namespace fovea
