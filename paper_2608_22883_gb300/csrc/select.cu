// Cumulative-mass selection kernels (the algorithm is in select_core.cuh):
// the selection alone (one CTA of 256 threads per draft state), and the
// selection fused with the readout r_n = sum_{t < K} alpha_t u_{pi(t)} (the
// alpha / r_n equation of the retrieval section).  The row's scores are
// staged in shared memory first.
#include <algorithm>

#include "select_core.cuh"
#include "tc_ptx.cuh"

namespace fovea {

// The CTA barrier; kLarge: the caller may pass caps above kRankMax (the
// large-cap ordering is compiled in only then, so the kernel for small caps
// keeps its short code).
template <bool kLargeCaps>
struct BlockSyncT {
  static constexpr bool kLarge = kLargeCaps;
  __device__ __forceinline__ void operator()() const { __syncthreads(); }
};
using BlockSync = BlockSyncT<false>;

template <bool kLargeCaps>
__global__ void __launch_bounds__(kSelThreads) select_kernel(const __grid_constant__ SelectArgs a,
                                                             const __grid_constant__ SeqTable tab) {
  extern __shared__ float s_sc[];                            // [M] scores of this row
  __shared__ SelectSmem sm;
  const int n = blockIdx.x;
  const int tid = threadIdx.x;
  pdl_wait();
  pdl_trigger();
  clear_alpha(a, n, tid, kSelThreads);    // ordered before the weights by the group barriers
  const int b = seq_of_row(tab, n);
  const int M = tab.m[b];
  if (M == 0 || row_gated(a.gate, n)) {   // empty valid set or past the depth gate: K = 0
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
  select_row(a, n, M, tab.key_off[b], s_sc, sm, tid, BlockSyncT<kLargeCaps>{});
}

cudaError_t launch_select(const float* scores, const SeqTable& tab, int N, const int32_t* orig_index,
                          float rho, int k_min, int k_max, int max_m, const DepthGate& gate,
                          int32_t* counts, int32_t* indices, int32_t* sel_pos, float* sel_w,
                          int32_t* sel_cnt, cudaStream_t s, void* alpha_hi, void* alpha_lo,
                          int alpha_ld) {
  if (N == 0) return cudaSuccess;
  const size_t smem = (size_t)max(max_m, 1) * sizeof(float);
  static bool configured = false;
  if (!configured) {
    for (auto k : {(const void*)select_kernel<false>, (const void*)select_kernel<true>}) {
      cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           FOVEA_MAX_ENTRIES * (int)sizeof(float));
      if (e != cudaSuccess) return e;
    }
    configured = true;
  }
  SelectArgs a{scores, orig_index, rho, k_min, k_max, counts, indices, sel_pos, sel_w, sel_cnt,
               nullptr, nullptr, nullptr, gate,
               static_cast<__nv_bfloat16*>(alpha_hi), static_cast<__nv_bfloat16*>(alpha_lo),
               alpha_ld};
  if (k_max > kRankMax)
    return launch_pdl(select_kernel<true>, dim3(N), dim3(kSelThreads), smem, s, a, tab);
  return launch_pdl(select_kernel<false>, dim3(N), dim3(kSelThreads), smem, s, a, tab);
}

// Selection and the gathers that consume it, in one kernel: one
// thread-block cluster of C CTAs per draft state n.  CTA rank 0 runs the
// selection of n into its shared memory; after a cluster barrier the other
// CTAs copy the selected rows and weights through distributed shared memory,
// so the selection is computed once and never travels through global memory.
// CTA y then gathers its column chunks of
//   the readout     r_n = sum_{t < K} alpha_t u_{pi(t)}          (U, d columns)
//   the projected readout  sum_t alpha_t p_{pi(t)}, p_i = W_r u_i  (P, 2H columns)
// whichever the call needs.  The first fusion layer is linear in r_n, so
// [W_f1 ; W_g1] [h_n ; r_n] = G_h[n] + sum_t alpha_t p_{pi(t)} with
// G_h = [W_f1 ; W_g1]_h h_n computed beside the query projection; the
// projected chunk is finished here: act = SiLU(G_h + sum + [b_f1 ; b_g1]).
// Gathers: the threads own 16-byte column vectors; for a chunk of fewer than
// 256 vectors, G = 256 / vectors groups of threads split the selected entries
// (group g takes t = g, g + G, ...), eight gathers in flight per thread, and
// their partial sums are combined in group order (fixed order, fp32).  CTA
// rank 0 writes counts and indices.
constexpr int kRoUnroll = 8;
constexpr int kStageRows = 64;                 // staged gather: rows per round
constexpr int kGatherSmemMax = 200 * 1024;     // dynamic shared memory of the gather kernel
static inline size_t align_up_sz(size_t x, size_t a) { return (x + a - 1) / a * a; }
using tc::cluster_sync;
using tc::ld_dsmem_f4;
using tc::map_dsmem;
using tc::smem_u32;

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cluster_arrive() {
  asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() {
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ int ld_dsmem_s32(uint32_t caddr) {
  int v;
  asm volatile("ld.shared::cluster.s32 %0, [%1];" : "=r"(v) : "r"(caddr) : "memory");
  return v;
}

struct GatherArgs {
  // readout: U [rows, d] -> r_out [N, d] fp32 and / or r_lo [N, d] (either may be null)
  const void* U;
  int d, chunk_u;
  float* r_out;
  void* r_lo;
  // projected readout: P [rows, HP] -> act [N, HP] = SiLU(Gh + sum + bias) (P null: none)
  const void* P;
  int HP, H, chunk_p;
  const float* Gh;                  // [N, HP] fp32
  const void* b_f1;                 // [H]: bias of columns < H
  const void* b_g1;                 // [H]: bias of columns >= H
  void* act;                        // [N, HP]
  long long p_prefetch;             // bytes of P prefetched into L2 before the wait
  int red_floats;                   // dynamic shared memory: the row's scores
  // > 0: the selected rows of P are staged in shared memory by bulk copies,
  // this many per round, at dyn + stage_off, with the group sums at dyn + red_off
  int stage_rows, stage_off, red_off;
  int self_select;                  // the CTAs of a row each select (no cluster)
  int* err;
};

// Weighted gather-sum over the selected rows of X [*, ld], columns
// [c0, c0 + w) (w a multiple of V): out(vector index, element, sum) once per
// column.  A warp covers VPW column vectors with 32 / VPW groups of lanes;
// group g sums the entries t = g, g + 32 / VPW, ... (eight gathers in flight
// per lane) and the groups' sums are combined by a fixed xor-shuffle tree
// (every lane of a vector ends with the full sums), so no shared memory or
// barrier is involved and the order is deterministic; group g then emits
// elements g, g + 32 / VPW, ... of its vector, so the epilogue work is spread
// over all lanes.
template <class T, int NT, class Out>
__device__ __forceinline__ void gather_chunk(const T* X, long long ld, int c0, int w, int K,
                                             const int32_t* pos, const float* wt, int tid, Out out) {
  constexpr int V = 16 / (int)sizeof(T);
  constexpr int kWarps = NT / 32;
  const int nvec = w / V;
  if (nvec <= 0) return;
  int vpw = 1;                            // vectors per warp: a power of two <= 32
  while (vpw < 32 && vpw * 2 * kWarps <= nvec) vpw *= 2;
  const int gpw = 32 / vpw;               // lane groups per warp
  const int lane = tid & 31, warp = tid >> 5;
  const int g = lane / vpw, v = lane - g * vpw;
  for (int vbase = 0; vbase < nvec; vbase += kWarps * vpw) {
    const int vc = vbase + warp * vpw + v;
    float acc[V];
#pragma unroll
    for (int i = 0; i < V; ++i) acc[i] = 0.0f;
    if (vc < nvec) {
      const T* col = X + c0 + (long long)vc * V;
      int t = g;
      for (; t + (kRoUnroll - 1) * gpw < K; t += kRoUnroll * gpw) {
        uint4 raw[kRoUnroll];
#pragma unroll
        for (int j = 0; j < kRoUnroll; ++j)
          raw[j] = __ldg(reinterpret_cast<const uint4*>(col + (long long)pos[t + j * gpw] * ld));
#pragma unroll
        for (int j = 0; j < kRoUnroll; ++j) {
          const float wj = wt[t + j * gpw];
          const T* e = reinterpret_cast<const T*>(&raw[j]);
#pragma unroll
          for (int i = 0; i < V; ++i) acc[i] = fmaf(wj, to_f32(e[i]), acc[i]);
        }
      }
      for (; t < K; t += gpw) {
        const uint4 raw = __ldg(reinterpret_cast<const uint4*>(col + (long long)pos[t] * ld));
        const float wj = wt[t];
        const T* e = reinterpret_cast<const T*>(&raw);
#pragma unroll
        for (int i = 0; i < V; ++i) acc[i] = fmaf(wj, to_f32(e[i]), acc[i]);
      }
    }
    // combine the groups: lanes v, v + vpw, v + 2 vpw, ... (every lane takes part)
    for (int o = 16; o >= vpw; o >>= 1)
#pragma unroll
      for (int i = 0; i < V; ++i) acc[i] += __shfl_xor_sync(0xffffffffu, acc[i], o);
    if (vc < nvec) {
#pragma unroll
      for (int i = 0; i < V; ++i)
        if (i % gpw == g) out(vc, i, acc[i]);
    }
  }
}

// Weighted sum over the selected rows of X [*, ld], columns [c0, c0 + w),
// staged in shared memory: each selected row's w elements arrive by one bulk
// copy (cp.async.bulk into buf, completing on the mbarrier `bar`), up to
// buf_rows rows per round.  Thread tid owns column vector tid % nvec of entry
// group tid / nvec (a warp reads 512 contiguous bytes of one staged row, free
// of bank conflicts); the groups' sums meet in `red` [G][w] fp32 and are
// added in group order (deterministic).  out(column, sum) once per column.
// A wait that gives up sets kErrTimeout; the copies already issued are waited
// for before the function returns.
template <class T, int NT, class Out>
__device__ __forceinline__ void gather_rows_smem(const T* X, long long ld, int c0, int w, int K,
                                                 const int32_t* pos, const float* wt, int tid,
                                                 T* buf, int buf_rows, float* red, uint64_t* bar,
                                                 int* err, Out out) {
  constexpr int V = 16 / (int)sizeof(T);
  const int nvec = w / V;
  const int G = NT / nvec;                       // entry groups (NT % nvec == 0)
  const int vec = tid % nvec, grp = tid / nvec;
  const uint32_t row_bytes = (uint32_t)(w * sizeof(T));
  float acc[V];
#pragma unroll
  for (int i = 0; i < V; ++i) acc[i] = 0.0f;
  uint32_t parity = 0;
  for (int t0 = 0; t0 < K; t0 += buf_rows) {
    const int cnt = min(buf_rows, K - t0);
    if (tid == 0) tc::mbar_expect_tx(bar, (uint32_t)cnt * row_bytes);
    __syncthreads();                             // bytes posted; buf free for this round
    if (tid < cnt)
      tc::bulk_load(buf + (size_t)tid * w, X + (long long)pos[t0 + tid] * ld + c0, row_bytes, bar);
    bool landed = tc::mbar_wait(bar, parity, nullptr);
    if (!landed) {
      if (tid == 0) atomicOr(err, kErrTimeout);
      tc::mbar_wait(bar, parity, nullptr);      // the copies in flight land first
    }
    parity ^= 1u;
    if (!__syncthreads_and(landed)) break;
    for (int t = grp; t < cnt; t += G) {
      const uint4 raw = *reinterpret_cast<const uint4*>(buf + (size_t)t * w + vec * V);
      const float wj = wt[t0 + t];
      const T* e = reinterpret_cast<const T*>(&raw);
#pragma unroll
      for (int i = 0; i < V; ++i) acc[i] = fmaf(wj, to_f32(e[i]), acc[i]);
    }
  }
  float* mine = red + (size_t)grp * w + vec * V;
#pragma unroll
  for (int i = 0; i < V; i += 4)
    *reinterpret_cast<float4*>(mine + i) = make_float4(acc[i], acc[i + 1], acc[i + 2], acc[i + 3]);
  __syncthreads();
  for (int c = tid; c < w; c += NT) {
    float sum = 0.0f;
    for (int g = 0; g < G; ++g) sum += red[(size_t)g * w + c];
    out(c, sum);
  }
}

// The selection group: the first kSelThreads threads of the CTA, synchronised
// with a named barrier when the CTA is larger.
struct SelGroupSync {
  static constexpr bool kLarge = false;   // the gather kernel takes caps <= kRankMax
  __device__ __forceinline__ void operator()() const {
    asm volatile("bar.sync 1, %0;" ::"n"(kSelThreads) : "memory");
  }
};

// NT threads per CTA: 256 (chunks of a row over a cluster) or 1024 (one CTA
// per row: the selection on the first 256 threads, the gathers on all).
template <class T, int NT>
__global__ void __launch_bounds__(NT) select_gather_kernel(
    const __grid_constant__ SelectArgs args, const __grid_constant__ SeqTable tab,
    const __grid_constant__ GatherArgs ga) {
  constexpr int V = 16 / (int)sizeof(T);                     // elements per 16-byte vector
  // dynamic: [red_floats] scores | [chunk_p] G_h | [chunk_p] bias | [red_floats] original
  // positions of the row's sequence (int32)
  extern __shared__ __align__(16) float dyn[];
  __shared__ SelectSmem sm;
  __shared__ __align__(16) int32_t loc_pos[kRankMax];
  __shared__ __align__(16) float loc_w[kRankMax];
  __shared__ int loc_cnt;
  __shared__ __align__(8) uint64_t stage_bar;      // staged gather rounds
  const int n = blockIdx.x;
  const int tid = threadIdx.x;
  const uint32_t rank = cluster_rank();
  if (tid == 0 && ga.stage_rows > 0) {
    tc::mbar_init(&stage_bar, 1);
    tc::fence_mbar_init();
  }
  float* s_sc = dyn;
  float* gh_s = dyn + ga.red_floats;
  T* bias_s = reinterpret_cast<T*>(gh_s + ga.chunk_p);
  if (ga.p_prefetch > 0 && tid == 0) {
    // the projected values (memory: not written by the previous kernel),
    // this CTA's share, into L2 while the scores are computed
    const int ncta = (int)(gridDim.x * gridDim.y);
    const int cid = (int)(blockIdx.x + gridDim.x * blockIdx.y);
    const long long bytes = ga.p_prefetch & ~15ll;
    const long long share = ((bytes + ncta - 1) / ncta + 15) & ~15ll;
    const long long beg = (long long)cid * share;
    const long long len = min(share, bytes - beg);
    const uint8_t* base = static_cast<const uint8_t*>(ga.P) + beg;
    for (long long off = 0; off < len; off += 32768)
      tc::prefetch_l2_bulk(base + off, (uint32_t)min(32768ll, len - off));
  }
  pdl_wait();
  pdl_trigger();
  // G_h and the biases of this CTA's projected chunk, and (rank 0) the
  // original positions of the sequence's entries: requested now, used last
  int32_t* orig_s = reinterpret_cast<int32_t*>(reinterpret_cast<uint8_t*>(bias_s) +
                                               ((ga.chunk_p * (int)sizeof(T) + 15) & ~15));
  // self_select: every CTA of the row selects for itself (the selection is
  // deterministic, so all reach the same result) and CTA y = 0 writes the
  // row's counts and indices; otherwise CTA rank 0 of the row's cluster
  // selects and the others copy its result through distributed shared memory
  const bool selector = ga.self_select || rank == 0;
  const bool writer = ga.self_select ? blockIdx.y == 0 : rank == 0;
  if (writer && args.indices != nullptr) {
    const int b = seq_of_row(tab, n);
    const int M = tab.m[b];
    const int32_t* src = args.orig_index + tab.key_off[b];
    if ((tab.key_off[b] & 3) == 0) {
      for (int q = tid; q < M / 4; q += NT) cp_async16(orig_s + 4 * q, src + 4 * q);
      for (int i = (M / 4) * 4 + tid; i < M; i += NT) orig_s[i] = src[i];
    } else {
      for (int i = tid; i < M; i += NT) orig_s[i] = src[i];
    }
  }
  const int cp0 = blockIdx.y * ga.chunk_p;
  const int wp = ga.P != nullptr ? max(0, min(ga.chunk_p, ga.HP - cp0)) : 0;
  for (int q = tid; q < wp / 4; q += NT)
    cp_async16(gh_s + 4 * q, ga.Gh + (long long)n * ga.HP + cp0 + 4 * q);
  for (int q = tid; q < wp / V; q += NT) {
    const int c = cp0 + q * V;
    const T* src = c < ga.H ? static_cast<const T*>(ga.b_f1) + c
                            : static_cast<const T*>(ga.b_g1) + (c - ga.H);
    cp_async16(bias_s + q * V, src);
  }
  if (selector && tid < kSelThreads) {
    SelectArgs a = args;
    a.counts = nullptr;                   // written after the cluster barrier (below), so
    a.indices = nullptr;                  // the barrier's release has no global writes to wait for
    a.loc_pos = loc_pos;
    a.loc_w = loc_w;
    a.loc_cnt = &loc_cnt;
    const int b = seq_of_row(tab, n);
    const int M = tab.m[b];
    if (M == 0 || row_gated(a.gate, n)) {   // empty valid set or past the depth gate:
      select_empty(a, n, tid);              // K = 0, r_n = 0
    } else {
      const float* src = a.scores + tab.score_off[b] + (long long)(n - tab.row_start[b]) * M;
      if (M <= kFastMaxM) {
        // every load of the thread in flight at once (8 per thread at most)
        constexpr int PT = kFastMaxM / kSelThreads;
        float v[PT];
#pragma unroll
        for (int j = 0; j < PT; ++j) {
          const int i = tid + j * kSelThreads;
          v[j] = i < M ? src[i] : 0.0f;
        }
#pragma unroll
        for (int j = 0; j < PT; ++j) {
          const int i = tid + j * kSelThreads;
          if (i < M) s_sc[i] = v[j] == 0.0f ? 0.0f : v[j];   // -0 -> +0: equal keys
        }
      } else {
        for (int i = tid; i < M; i += kSelThreads) {
          float v = src[i];
          if (v == 0.0f) v = 0.0f;        // -0 -> +0 so equal scores get equal keys
          s_sc[i] = v;
        }
      }
      if constexpr (NT == kSelThreads) {
        __syncthreads();
        select_row(a, n, M, tab.key_off[b], s_sc, sm, tid, BlockSync{});
      } else {
        SelGroupSync{}();
        select_row(a, n, M, tab.key_off[b], s_sc, sm, tid, SelGroupSync{});
      }
    }
  }
  // rank 0's selection visible to the cluster (one CTA: a CTA barrier, which
  // does not wait for the selection's global writes to complete)
  const bool clustered = !ga.self_select && gridDim.y > 1;
  if (clustered) cluster_sync(); else __syncthreads();
  if (!selector) {
    const int K = ld_dsmem_s32(map_dsmem(smem_u32(&loc_cnt), 0));
    for (int q = tid; q < (K + 3) / 4; q += NT) {
      const float4 p4 = ld_dsmem_f4(map_dsmem(smem_u32(&loc_pos[4 * q]), 0));
      const float4 w4 = ld_dsmem_f4(map_dsmem(smem_u32(&loc_w[4 * q]), 0));
      *reinterpret_cast<float4*>(&loc_pos[4 * q]) = p4;
      *reinterpret_cast<float4*>(&loc_w[4 * q]) = w4;
    }
    if (tid == 0) loc_cnt = K;
  }
  if (clustered) cluster_arrive();        // done reading rank 0 (waited for before exit)
  cp_async_wait_all();
  __syncthreads();
  const int K = loc_cnt;
  if (writer) {                           // counts and indices of row n
    const long long out_row = (long long)n * args.k_max;
    if (args.indices != nullptr) {
      const int key_off = tab.key_off[seq_of_row(tab, n)];
      for (int t = tid; t < args.k_max; t += NT)
        args.indices[out_row + t] = t < K ? orig_s[loc_pos[t] - key_off] : -1;
    }
    if (args.counts != nullptr && tid == 0) args.counts[n] = K;
  }
  // projected readout -> act = SiLU(G_h + sum + bias)
  if (wp > 0) {
    T* act = static_cast<T*>(ga.act) + (long long)n * ga.HP + cp0;
    auto fin = [&](int vc, int i, float sum) {
      const int c = vc * V + i;
      const float z = sum + gh_s[c] + to_f32(bias_s[c]);
      act[c] = from_f32<T>(z * sigmoidf_(z));
    };
    if (ga.stage_rows > 0) {
      T* buf = reinterpret_cast<T*>(reinterpret_cast<uint8_t*>(dyn) + ga.stage_off);
      float* red = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(dyn) + ga.red_off);
      auto fin_c = [&](int c, float sum) { fin(c / V, c % V, sum); };
      gather_rows_smem<T, NT>(static_cast<const T*>(ga.P), ga.HP, cp0, wp, K, loc_pos, loc_w, tid,
                              buf, ga.stage_rows, red, &stage_bar, ga.err, fin_c);
    } else {
      gather_chunk<T, NT>(static_cast<const T*>(ga.P), ga.HP, cp0, wp, K, loc_pos, loc_w, tid, fin);
    }
  }
  // readout r_n
  const int cu0 = blockIdx.y * ga.chunk_u;
  const int wu = (ga.r_out != nullptr || ga.r_lo != nullptr) ? max(0, min(ga.chunk_u, ga.d - cu0)) : 0;
  if (wu > 0) {
    const long long o = (long long)n * ga.d + cu0;
    auto fin = [&](int vc, int i, float sum) {
      if (ga.r_out != nullptr) ga.r_out[o + vc * V + i] = sum;
      if (ga.r_lo != nullptr) static_cast<T*>(ga.r_lo)[o + vc * V + i] = from_f32<T>(sum);
    };
    gather_chunk<T, NT>(static_cast<const T*>(ga.U), ga.d, cu0, wu, K, loc_pos, loc_w, tid, fin);
  }
  if (clustered) cluster_wait();          // rank 0 stays until every CTA has copied
}

bool select_readout_fits(int max_m, int k_max) { return max_m <= kFastMaxM && k_max <= kRankMax; }

cudaError_t launch_select_gather(int dtype, const float* scores, const SeqTable& tab, int N,
                                 const int32_t* orig_index, float rho, int k_min, int k_max,
                                 int max_m, const DepthGate& gate, int32_t* counts,
                                 int32_t* indices, const void* U, int d,
                                 float* r_out, void* r_lo, const void* P, int H, const float* Gh,
                                 const void* b_f1, const void* b_g1, void* act, int* err,
                                 cudaStream_t s, long long p_prefetch_bytes) {
  if (N == 0) return cudaSuccess;
  if (!select_readout_fits(max_m, k_max) || d % 64 != 0 || (P != nullptr && H % 64 != 0))
    return cudaErrorInvalidValue;
  // CTAs per row (one cluster): about two per SM in one wave, each chunk a
  // multiple of 64 columns
  int sms = 0;
  cudaError_t e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, 0);
  if (e != cudaSuccess) return e;
  const int HP = 2 * H;
  // projected readout: CTAs of 1024 threads (the selection on 256 of them),
  // one per row, or two per row that each select for themselves when the
  // batch leaves most SMs idle; the readout alone: a cluster of CTAs of 256
  // threads per row, about two CTAs per SM in one wave, each chunk a multiple
  // of 64 columns
  const bool wide = P != nullptr;
  int nchunk = 1;
  while (!wide && nchunk < 8 && (long long)N * nchunk * 2 <= 2LL * sms &&
         d % (nchunk * 2 * 64) == 0)
    nchunk *= 2;
  // projected readout: a batch that leaves most SMs idle gives each row two
  // CTAs, each selecting for itself and gathering half of the 2H columns (the
  // gather of a row's selected projected rows is bound by what one SM takes
  // in from L2)
  if (wide && (long long)N * 2 <= sms && HP % 128 == 0) nchunk = 2;
  GatherArgs ga{};
  ga.U = U;
  ga.d = d;
  ga.chunk_u = d / nchunk;
  ga.r_out = r_out;
  ga.r_lo = r_lo;
  ga.P = P;
  ga.HP = P != nullptr ? HP : 0;
  ga.H = H;
  ga.chunk_p = P != nullptr ? HP / nchunk : 0;
  ga.Gh = Gh;
  ga.b_f1 = b_f1;
  ga.b_g1 = b_g1;
  ga.act = act;
  ga.p_prefetch = P != nullptr ? p_prefetch_bytes : 0;
  ga.red_floats = (int)align_up_sz((size_t)std::max(max_m, 1), 4);
  const size_t es = dtype == FOVEA_BF16 ? 2 : 4;
  // dynamic: scores | G_h | biases | original positions
  size_t smem = (size_t)ga.red_floats * 4 + (size_t)ga.chunk_p * 4 +
                align_up_sz((size_t)ga.chunk_p * es, 16) + (size_t)ga.red_floats * 4;
  if (smem > 64 * 1024) return cudaErrorInvalidValue;
  ga.err = err;
  if (wide && dtype == FOVEA_BF16 && ga.chunk_p % 8 == 0 && 1024 % (ga.chunk_p / 8) == 0) {
    // stage the selected projected rows in shared memory: up to 64 rows per
    // round (128 KB at 2H = 1024), the group sums after them
    const int rows = std::min(k_max, kStageRows);
    ga.stage_off = (int)align_up_sz(smem, 128);
    const size_t stage_bytes = (size_t)rows * ga.chunk_p * es;
    ga.red_off = (int)align_up_sz(ga.stage_off + stage_bytes, 128);
    const size_t red_bytes = (size_t)(1024 / (ga.chunk_p / 8)) * ga.chunk_p * 4;
    if (ga.red_off + red_bytes <= (size_t)kGatherSmemMax) {
      ga.stage_rows = rows;
      smem = ga.red_off + red_bytes;
    }
  }
  static bool configured = false;
  if (!configured) {
    for (auto k : {(const void*)select_gather_kernel<__nv_bfloat16, 1024>,
                   (const void*)select_gather_kernel<__nv_bfloat16, kSelThreads>,
                   (const void*)select_gather_kernel<float, 1024>,
                   (const void*)select_gather_kernel<float, kSelThreads>}) {
      e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, kGatherSmemMax);
      if (e != cudaSuccess) return e;
    }
    configured = true;
  }
  SelectArgs a{scores, orig_index, rho, k_min, k_max, counts, indices,
               nullptr, nullptr, nullptr, nullptr, nullptr, nullptr, gate};
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(N, nchunk);
  cfg.blockDim = dim3(wide ? 1024 : kSelThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;   // the chunks of one row form a cluster
  attr[1].val.clusterDim.x = 1;
  attr[1].val.clusterDim.y = nchunk;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = wide ? 1 : 2;              // projected rows: self-selecting CTAs, no cluster
  ga.self_select = wide ? 1 : 0;
  if (dtype == FOVEA_BF16)
    return wide ? cudaLaunchKernelEx(&cfg, select_gather_kernel<__nv_bfloat16, 1024>, a, tab, ga)
                : cudaLaunchKernelEx(&cfg, select_gather_kernel<__nv_bfloat16, kSelThreads>, a, tab, ga);
  return wide ? cudaLaunchKernelEx(&cfg, select_gather_kernel<float, 1024>, a, tab, ga)
              : cudaLaunchKernelEx(&cfg, select_gather_kernel<float, kSelThreads>, a, tab, ga);
}

}  // namespace fovea
