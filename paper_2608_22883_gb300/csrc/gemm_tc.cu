// tcgen05 GEMM C = A . B^T for the bf16 path (sm_103a): the memory
// projections k = W_K LN(v), u = W_U LN(v), the folded keys W_Q^T k, the
// query projection W_Q, the scores per sequence, and the two fusion layers.
// Neither score form rounds the query map to bf16: the unfolded scores carry
// q = W_Q x as a bf16 hi/lo pair (q ~= q_hi + q_lo, about 16 significant
// bits) and each key tile meets both parts; the folded scores carry the
// folded keys kappa = W_Q^T k as a hi/lo pair and each x tile meets both.
//
// Operand roles.  In the GemmArgs vocabulary A holds the output columns
// (weights, keys: the "feature" operand) and B the output rows (draft states,
// tokens: the "row" operand).  On the tensor core the row operand is the MMA
// A operand (M = 128 rows; a 64-row batch is zero-filled by TMA) and the
// feature operand is the MMA B operand (N = BN <= 256 features).  A tcgen05
// MMA costs about the same time for any N up to 256, so a wide feature tile
// consumes twice the weight bytes per MMA of a 128-feature tile: the
// weight-streaming GEMMs are limited by that consumption rate per SM.
// Both operands are K-major bf16, staged by TMA into 128-byte-swizzled
// shared-memory tiles of 64 contraction elements; fp32 accumulators live in
// tensor memory (lane = row, column = feature) and are read back with
// tcgen05.ld: each epilogue thread owns one row and its BN features.
//
// Roles (256 threads): lanes of warp 0 issue the TMA loads into a ring of
// shared-memory stages (lane 0 the feature tiles, lane 1 the row tiles, lane
// 2 the lo row tiles of the scores: the copies one thread issues complete one
// after another, so each operand gets its own issuing lane), warp 1 owns the
// tensor-memory allocation and its lane 0 issues the MMAs (one elected
// thread), and all eight warps run the epilogue: warp w reads accumulator
// lanes (rows) 32 (w % 4) .. +31.  Every mbarrier wait is bounded (~2 s, or
// the limit fovea_debug_wait_limit sets); a wait that gives up sets
// kErrTimeout in the error word and the CTA unwinds: the producer waits for
// the copies it issued, the MMA issuer commits what it issued, and the
// epilogue waits for those MMAs before the tensor memory is freed.
//
// Split K: when the output tiles cannot fill the GPU (a 64-row batch against
// a weight matrix), S <= 8 CTAs share one output tile, each contracting a
// slice of K.  The S CTAs of a tile form a thread-block cluster: each stages
// its fp32 partial tile in its own shared memory (over the idle stage ring),
// the cluster synchronises, and CTA r sums the S partials of column quads
// [r Q/S, (r+1) Q/S) (Q = BN/4) in rank order through distributed shared
// memory (so the result does not depend on timing) and runs the epilogue for
// them; a second cluster barrier keeps every partial alive until it is read.
// (Pushing the partials into the owners' shared memory with remote stores and
// an mbarrier handshake measured slower: remote stores issue one at a time.)
//
// Launch overlap: kernels are launched with programmatic dependent launch.
// The producer issues the feature-operand (weight / key) loads of the first
// stages before griddepcontrol.wait; those operands never depend on the
// previous kernel, so the weight stream starts while the predecessor drains.
#include <atomic>
#include <cstring>
#include <cstdio>
#include <string>
#include <unordered_map>

#include "gemm_epilogue.cuh"
#include "tc_ptx.cuh"

namespace fovea {
namespace tc {

constexpr int BM = 128;          // UMMA M: rows per tile
constexpr int BK = 64;           // contraction elements per stage (128 bytes bf16)
constexpr int UMMA_K = 16;       // contraction elements per tcgen05.mma (kind::f16)
constexpr int kThreads = 256;
constexpr int kSmemBudget = 200 * 1024;   // shared-memory stages, one CTA per SM
constexpr int kSmemBudgetPair = 100 * 1024;  // two CTAs per SM
constexpr int kSmemExtra = 1024 /*alignment*/ + 256 /*barriers*/ + 1024 /*tile biases*/;
constexpr int kMaxStages = 8;
constexpr int kRasterRows = 16;          // row tiles per band of the tile order

// BN features per tile; DUAL: the row stage holds two tiles (hi and lo parts
// of the row operand), and each feature tile is multiplied by both into the
// same accumulator.
//
// A ring stage holds KPS consecutive k-blocks of 64, loaded with one 3-D TMA
// box per operand (k within the block, row, k-block), because a copy costs
// its issuing thread about the same time for any box up to 64 KB: few large
// copies keep the ring fed.  Stage layout: row tiles [KPS][rbox][128 B]
// (twice for DUAL: hi, then lo), then feature tiles [KPS][BN][128 B].  The MMA
// reads 128 rows from each row tile's start; rows past rbox (>= 64, so the
// read stays inside the stage) only feed accumulator rows that are never
// stored.
// DF (dual feature, the folded scores): the feature stage holds two tiles (hi
// and lo parts of the folded keys), each multiplied by the same row tile into
// the same accumulator.
template <int BN, bool DUAL = false>
struct Cfg {
  static constexpr uint32_t TMEM_COLS = BN < 32 ? 32 : BN;
  __host__ __device__ static constexpr int stage_bytes(int kps, int rbox, bool df = false) {
    return kps * (rbox * (DUAL ? 2 : 1) + BN * (df ? 2 : 1)) * 128;
  }
  // Instruction descriptor, kind::f16: D fp32 (bits 4-5 = 1), A bf16 (bits 7-9
  // = 1), B bf16 (bits 10-12 = 1), both K-major (bits 15, 16 = 0), N >> 3 at
  // bits 17-22, M >> 4 at bits 24-28.
  static constexpr uint32_t IDESC = (1u << 4) | (1u << 7) | (1u << 10) |
                                    ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);
};

// Key epilogue: a key element is listed for exact recomputation when its
// fp32 accumulator lies within w * max(|acc|, scale) of a bf16 rounding
// midpoint, scale being the RMS of the token's values in this tile (the
// magnitude of the partial sums) and w = 2^-15 * max(1, K / 4096) for a
// contraction of length K.  The largest distance of a mis-rounded element
// from its midpoint, measured over 4.1e7 keys at K = 3584 .. 5120, was
// 2^-16.2 of that magnitude, so the window keeps a margin above 2x and an
// element outside it rounds as the exact value would.
__device__ __forceinline__ bool near_midpoint(float acc, __nv_bfloat16 r, float scale, int k_total) {
  const unsigned short bits = __bfloat16_as_ushort(r);
  const float rf = __bfloat162float(r);
  const float up = __bfloat162float(__ushort_as_bfloat16((unsigned short)(bits + 1)));
  const float dn = __bfloat162float(__ushort_as_bfloat16((unsigned short)(bits - 1)));
  const float dist = fminf(fabsf(acc - 0.5f * (rf + up)), fabsf(acc - 0.5f * (rf + dn)));
  const float window =
      ldexpf(fmaxf(fabsf(acc), scale), -15) * fmaxf(1.0f, (float)k_total * (1.0f / 4096.0f));
  return !(dist > window);
}

// kEpiAct: the fp32 term added before the activation (G_h), for the column
// quads [qlo, qlo + qn) of the tile's rows, staged in shared memory as
// addt[rows_real][qn * 4] with every thread's loads in flight together
// (read row by row inside the epilogue they would serialise its rounds).
__device__ __forceinline__ void stage_add_tile(const GemmArgs& a, const GemmGroup& g, int m0,
                                               int n0, int rows_real, int n_cols, int qlo, int qn,
                                               float* addt) {
  constexpr int kBatch = 8;
  const int total = rows_real * qn;
  for (int it0 = threadIdx.x; it0 < total; it0 += kThreads * kBatch) {
    float4 v[kBatch];
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      const int it = it0 + j * kThreads;
      v[j] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
      if (it < total) {
        const int rr = it / qn, col = (qlo + it - rr * qn) * 4;
        if (col < n_cols)
          v[j] = __ldg(reinterpret_cast<const float4*>(
              a.add_in + ((long long)g.b_row0 + n0 + rr) * a.ldc2 + m0 + col));
      }
    }
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      const int it = it0 + j * kThreads;
      if (it < total) *reinterpret_cast<float4*>(addt + 4 * (long long)it) = v[j];
    }
  }
}

// Order-preserving map of a float to an unsigned key (larger float, larger key).
__device__ __forceinline__ uint32_t logit_order_key(float f) {
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Compare-exchange: a keeps the larger key, b the smaller.
__device__ __forceinline__ void cx_desc(uint32_t& a, uint32_t& b) {
  const uint32_t hi = max(a, b);
  b = min(a, b);
  a = hi;
}

// Sorts 8 keys into descending order (odd-even merge network, 19
// compare-exchanges).
__device__ __forceinline__ void sort8_desc(uint32_t& x0, uint32_t& x1, uint32_t& x2, uint32_t& x3,
                                           uint32_t& x4, uint32_t& x5, uint32_t& x6, uint32_t& x7) {
  cx_desc(x0, x1); cx_desc(x2, x3); cx_desc(x4, x5); cx_desc(x6, x7);
  cx_desc(x0, x2); cx_desc(x1, x3); cx_desc(x4, x6); cx_desc(x5, x7);
  cx_desc(x1, x2); cx_desc(x5, x6);
  cx_desc(x0, x4); cx_desc(x1, x5); cx_desc(x2, x6); cx_desc(x3, x7);
  cx_desc(x2, x4); cx_desc(x3, x5);
  cx_desc(x1, x2); cx_desc(x3, x4); cx_desc(x5, x6);
}

constexpr int kTopkPer = 16;                 // candidates listed per thread by the threshold pass
constexpr int kTopkLd = 4 * kTopkPer + 1;    // a row's lists (rows of a warp on distinct banks)

// kEpiLogits for cand_k <= 8, the threshold form.  Four threads per row,
// thread q taking columns q, q + 4, ... (consecutive lanes on consecutive
// banks).  Pass 1: each thread's two largest order keys; the k-th largest of
// the row's eight is a lower bound T on the row's k-th largest key (they are
// eight of the row's keys).  Pass 2: each thread lists its keys >= T, as
// 64-bit candidate keys, in its own part of the row's list in shared memory
// (a handful per row; eight loads in flight before any store).  Pass 3: each
// listed key's rank is its count of larger listed keys (the keys are
// distinct), and ranks below k are the row's candidates, in order; slots past
// the row's columns hold 0.  Integer work per element: three min / max, one
// compare.  Returns false, having written nothing that the caller's fallback
// does not overwrite, when a thread lists more than kTopkPer keys (many equal
// logits) or the scratch is too small.
template <int BN>
__device__ __forceinline__ bool tile_topk_threshold(const GemmArgs& a, long long row0,
                                                    int rows_real, const float* vals, int ld,
                                                    int col0, int ncols, int slot,
                                                    uint8_t* scratch, int scratch_bytes) {
  constexpr int kRows = kThreads / 4;              // rows per pass
  constexpr int kB = 8;                            // columns per thread and batch
  const int k = a.cand_k;
  if (scratch_bytes < kRows * kTopkLd * 8 + 16) return false;
  unsigned long long* list = reinterpret_cast<unsigned long long*>(scratch);
  int* overflow = reinterpret_cast<int*>(scratch + kRows * kTopkLd * 8);
  const int q = threadIdx.x & 3;
  const int lr = (int)(threadIdx.x >> 2);          // the row within a pass
  if (threadIdx.x == 0) *overflow = 0;
  __syncthreads();
  const uint32_t list_s = smem_u32(list);
  for (int rbase = 0; rbase < rows_real; rbase += kRows) {
    const int rr = rbase + lr;
    const bool real = rr < rows_real;
    const uint32_t row_s = smem_u32(vals) + (uint32_t)(rr * ld) * 4u;
    // pass 1: this thread's two largest keys
    uint32_t m1 = 0u, m2 = 0u;
    if (real) {
      for (int c0 = q; c0 < ncols; c0 += 4 * kB) {
        uint32_t x[kB];
#pragma unroll
        for (int u = 0; u < kB; ++u) {
          const int c = c0 + 4 * u;
          x[u] = c < ncols ? logit_order_key(lds_f32(row_s + 4u * (uint32_t)c)) : 0u;
        }
#pragma unroll
        for (int u = 0; u < kB; ++u) {
          m2 = max(m2, min(m1, x[u]));
          m1 = max(m1, x[u]);
        }
      }
    }
    uint32_t v0 = m1, v1 = m2;
    uint32_t v2 = __shfl_xor_sync(0xffffffffu, m1, 1);
    uint32_t v3 = __shfl_xor_sync(0xffffffffu, m2, 1);
    uint32_t v4 = __shfl_xor_sync(0xffffffffu, v0, 2);
    uint32_t v5 = __shfl_xor_sync(0xffffffffu, v1, 2);
    uint32_t v6 = __shfl_xor_sync(0xffffffffu, v2, 2);
    uint32_t v7 = __shfl_xor_sync(0xffffffffu, v3, 2);
    sort8_desc(v0, v1, v2, v3, v4, v5, v6, v7);
    uint32_t T = k <= 1 ? v0 : k == 2 ? v1 : k == 3 ? v2 : k == 4 ? v3 :
                 k == 5 ? v4 : k == 6 ? v5 : k == 7 ? v6 : v7;
    T = max(T, 1u);                                // a zero key is never a candidate
    // pass 2: this thread's keys >= T, in a short list of its own
    const uint32_t lst_s = list_s + (uint32_t)(lr * kTopkLd) * 8u;
    const uint32_t own_s = lst_s + (uint32_t)(q * kTopkPer) * 8u;
    int mine = 0;
    if (real) {
      for (int c0 = q; c0 < ncols; c0 += 4 * kB) {
        uint32_t x[kB];
#pragma unroll
        for (int u = 0; u < kB; ++u) {
          const int c = c0 + 4 * u;
          x[u] = c < ncols ? logit_order_key(lds_f32(row_s + 4u * (uint32_t)c)) : 0u;
        }
#pragma unroll
        for (int u = 0; u < kB; ++u) {           // branch-free: a predicated store
          const uint32_t hit = x[u] >= T ? 1u : 0u;
          sts_u64_if(own_s + 8u * (uint32_t)min(mine, kTopkPer - 1),
                     ((unsigned long long)x[u] << 32) |
                         (0xFFFFFFFFu - (uint32_t)col0 - (uint32_t)(c0 + 4 * u)),
                     hit & (mine < kTopkPer ? 1u : 0u));
          mine += (int)hit;
        }
      }
    }
    // the row's lists packed in thread order at the front of its list area
    // (read into registers first: a list may move onto another's place)
    int incl = mine;                               // prefix over the row's four threads
    int up = __shfl_up_sync(0xffffffffu, incl, 1);
    incl += q >= 1 ? up : 0;
    up = __shfl_up_sync(0xffffffffu, incl, 2);
    incl += q >= 2 ? up : 0;
    const int before = incl - mine;
    int total = __shfl_xor_sync(0xffffffffu, mine, 1) + mine;
    total += __shfl_xor_sync(0xffffffffu, total, 2);
    const int over = __shfl_xor_sync(0xffffffffu, mine > kTopkPer ? 1 : 0, 1) | (mine > kTopkPer);
    const bool overflowed = (over | __shfl_xor_sync(0xffffffffu, over, 2)) != 0;
    unsigned long long held[kTopkPer];
#pragma unroll
    for (int j = 0; j < kTopkPer; ++j)
      held[j] = j < mine && !overflowed ? lds_u64(own_s + 8u * (uint32_t)j) : 0ull;
    __syncwarp();
    if (!overflowed) {
#pragma unroll
      for (int j = 0; j < kTopkPer; ++j)
        if (j < mine) sts_u64(lst_s + 8u * (uint32_t)(before + j), held[j]);
    }
    __syncwarp();
    // pass 3: ranks within the row's list
    if (real) {
      if (overflowed) {
        *overflow = 1;
      } else {
        unsigned long long* dst = a.cand + (row0 + rr) * a.cand_ld + (long long)slot * k;
        for (int j = q; j < total; j += 4) {
          const unsigned long long key = lds_u64(lst_s + 8u * (uint32_t)j);
          int rank = 0;
          for (int i = 0; i < total; ++i) rank += lds_u64(lst_s + 8u * (uint32_t)i) > key ? 1 : 0;
          if (rank < k) dst[rank] = key;
        }
        for (int j = total + q; j < k; j += 4) dst[j] = 0ull;
      }
    }
    __syncwarp();
  }
  __syncthreads();
  return *overflow == 0;
}

// kEpiLogits: per row of the tile, the cand_k largest of `ncols` logits
// (vals [rows_real][ld] in shared memory, column c is token col0 + c) into
// the row's candidate slot as 64-bit keys, logit order key << 32 | ~token
// (on equal logits the smaller token is larger).  Up to 8 candidates the
// threshold form above; otherwise (or when it gives up) one warp per row, each lane
// holding the order keys of columns lane, lane + 32, ...; each of the k rounds
// takes the lane maxima (the smallest column on equal keys), a warp maximum,
// the smallest column holding it (warp minimum), and clears that key: short,
// independent steps.  A zero key (fewer columns than cand_k) sorts below every
// real one.
template <int BN>
__device__ __forceinline__ void tile_topk(const GemmArgs& a, long long row0, int rows_real,
                                          const float* vals, int ld, int col0, int ncols,
                                          int slot, uint8_t* scratch, int scratch_bytes) {
  if (a.cand_k <= 8 && tile_topk_threshold<BN>(a, row0, rows_real, vals, ld, col0, ncols, slot,
                                               scratch, scratch_bytes))
    return;
  constexpr int J = (BN + 31) / 32;
  constexpr int R = 4;                       // rows a warp works on together (independent chains)
  constexpr int kWarps = kThreads / 32;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int k = a.cand_k;
  for (int base = warp; base < rows_real; base += kWarps * R) {
    uint32_t key[R][J];
#pragma unroll
    for (int u = 0; u < R; ++u) {
      const int rr = base + u * kWarps;
#pragma unroll
      for (int j = 0; j < J; ++j) {
        const int c = lane + 32 * j;
        key[u][j] = (rr < rows_real && c < ncols) ? logit_order_key(vals[rr * ld + c]) : 0u;
      }
    }
    for (int r = 0; r < k; ++r) {
      uint32_t w[R], cmin[R];
#pragma unroll
      for (int u = 0; u < R; ++u) {
        uint32_t m = key[u][0];
        int jm = 0;
#pragma unroll
        for (int j = 1; j < J; ++j)
          if (key[u][j] > m) {
            m = key[u][j];
            jm = j;
          }
        w[u] = __reduce_max_sync(0xffffffffu, m);
        const uint32_t col = m == w[u] ? (uint32_t)(lane + 32 * jm) : 0xFFFFFFFFu;
        cmin[u] = __reduce_min_sync(0xffffffffu, col);
        if (col == cmin[u]) {
#pragma unroll
          for (int j = 0; j < J; ++j)
            if (j == jm) key[u][j] = 0u;
        }
      }
      if (lane < R) {
        const int rr = base + lane * kWarps;
        uint32_t wl = 0u, cl = 0u;
#pragma unroll
        for (int u = 0; u < R; ++u)
          if (u == lane) {
            wl = w[u];
            cl = cmin[u];
          }
        if (rr < rows_real)
          a.cand[(row0 + rr) * a.cand_ld + (long long)slot * k + r] =
              wl == 0u ? 0ull : ((unsigned long long)wl << 32) | (0xFFFFFFFFu - (uint32_t)col0 - cl);
      }
    }
  }
}

// kEpiAct: four consecutive activations of output row n (group-local),
// columns m .. m + nv - 1: SiLU(acc + added term + bias), stored as bf16 (one
// 8-byte store for a full, aligned quad).
__device__ __forceinline__ void act_store4(const GemmArgs& a, const GemmGroup& g, int m, int n,
                                           const float (&v)[4], const float* add4,
                                           const float* bias4, int nv) {
  __nv_bfloat16* out = static_cast<__nv_bfloat16*>(a.out0) + ((long long)g.b_row0 + n) * a.ldc + m;
  float y[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const float z = v[j] + add4[j] + bias4[j];
    y[j] = z * sigmoidf_(z);
  }
  if (nv == 4 && (reinterpret_cast<uintptr_t>(out) & 7) == 0) {
    const __nv_bfloat162 lo = __floats2bfloat162_rn(y[0], y[1]);
    const __nv_bfloat162 hi = __floats2bfloat162_rn(y[2], y[3]);
    uint2 u;
    u.x = *reinterpret_cast<const uint32_t*>(&lo);
    u.y = *reinterpret_cast<const uint32_t*>(&hi);
    *reinterpret_cast<uint2*>(out) = u;
  } else {
    for (int j = 0; j < nv; ++j) out[j] = __float2bfloat16_rn(y[j]);
  }
}

template <int BN, int EPI>
__global__ void __launch_bounds__(kThreads, 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap tmF0, const __grid_constant__ CUtensorMap tmF1,
                   const __grid_constant__ CUtensorMap tmF2, const __grid_constant__ CUtensorMap tmR0,
                   const __grid_constant__ CUtensorMap tmR1, const __grid_constant__ GemmArgs args) {
  constexpr bool DUAL = EPI == kEpiScores || EPI == kEpiAct;
  using C = Cfg<BN, DUAL>;
  const int S = args.splits;
  const uint32_t rank = (uint32_t)((int)blockIdx.x % S);
  const GemmGroup& g = args.groups[blockIdx.z];
  // Output columns (features) [0, a_split) come from F0, [a_split, a_split2)
  // from F1 and [a_split2, m) from F2; each part is tiled on its own so no
  // tile straddles two operands.  A group smaller than the grid leaves its
  // extra tiles idle.  The S CTAs of a tile share these decisions, so a
  // tile's CTAs exit together.
  const int s1 = min(args.a_split, g.m);
  const int s2 = max(s1, min(args.a_split2, g.m));
  const int t0 = (s1 + BN - 1) / BN, t1 = (s2 - s1 + BN - 1) / BN, t2 = (g.m - s2 + BN - 1) / BN;
  // Tile order: with one group and no split, consecutive CTAs walk
  // kRasterRows row tiles per feature tile, so that a wave of resident CTAs
  // shares both operands through L2 (in feature-fastest order every wave
  // re-reads all feature tiles from HBM).
  int bx = (int)blockIdx.x, by = (int)blockIdx.y;
  if (S == 1 && gridDim.z == 1 && (int)gridDim.y > kRasterRows) {
    const int FX = (int)gridDim.x;
    const int L = bx + FX * by;
    const int sr = L / (kRasterRows * FX);
    const int rows_here = min(kRasterRows, (int)gridDim.y - sr * kRasterRows);
    const int local = L - sr * kRasterRows * FX;
    by = sr * kRasterRows + local % rows_here;
    bx = local / rows_here;
  }
  const int tx = bx / S;
  if (tx >= t0 + t1 + t2) return;
  const int part = tx < t0 ? 0 : (tx < t0 + t1 ? 1 : 2);
  const int pbeg = part == 0 ? 0 : (part == 1 ? s1 : s2);
  const int m0 = pbeg + (tx - (part == 0 ? 0 : (part == 1 ? t0 : t0 + t1))) * BN;
  const int m_end = part == 0 ? s1 : (part == 1 ? s2 : g.m);
  const int n0 = by * BM;
  if (m0 >= m_end || n0 >= g.n) return;

  // folded scores: the folded keys (part 0) are a hi / lo pair of bf16 values,
  // the lo part f_lo_kb k-blocks after the hi part in the same rows
  const bool dual_f = EPI == kEpiScoresFolded && args.f_lo_kb > 0 && part == 0;
  const int kProducers = (DUAL || dual_f) ? 3 : 2;   // TMA-issuing lanes of warp 0
  const int KPS = args.kps, rbox = args.rbox;
  const int r_tile = rbox * 128;                       // one k-block of the row operand
  const int r_bytes = KPS * r_tile * (DUAL ? 2 : 1);
  const int f_tile = BN * 128;                         // one k-block of the feature operand
  const int stage_bytes = C::stage_bytes(KPS, rbox, dual_f);
  const int stages = dual_f ? max(1, min(args.stages, args.region / stage_bytes)) : args.stages;
  extern __shared__ uint8_t smem_raw[];
  // the 1024-byte aligned base, derived from smem_raw by pointer arithmetic
  // so that the compiler keeps every access through it in the shared space
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  // stage st: row tiles at smem + st * stage_bytes, feature tiles r_bytes later
  // barriers after the ring, or after the partial-tile staging area when that
  // is larger (split K)
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + args.region);
  uint64_t* empty = full + stages;
  uint64_t* accum = empty + stages;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(accum + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  float* bias_s = reinterpret_cast<float*>(smem + args.region + 256);   // [BN] tile biases

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int st = 0; st < stages; ++st) {
      mbar_init(&full[st], kProducers);
      mbar_init(&empty[st], 1);
    }
    mbar_init(accum, 1);
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(part == 0 ? &tmF0 : (part == 1 ? &tmF1 : &tmF2));
    prefetch_tmap(&tmR0);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, C::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int kb_total = args.k_total / BK;
  const int r_split_kb = args.b_split / BK;
  const int su_total = kb_total / KPS;                 // stage units (KPS k-blocks each)
  const int su_lo = (int)((long long)rank * su_total / S);
  const int su_hi = (int)((long long)(rank + 1) * su_total / S);
  const int nkb = su_hi - su_lo;                       // stages of this CTA

  if (warp == 0 && lane < kProducers) {
    // ---- TMA producers: lane 0 loads the feature tiles, lane 1 the row tiles
    // (lane 2 the lo row tiles of DUAL, or the lo feature tiles of the folded
    // keys).  Each lane posts its own bytes on the stage's full barrier
    // (initialised with one arrival per producer lane).
    const uint32_t f_bytes = (uint32_t)(KPS * f_tile);
    const uint32_t r_lane_bytes = (uint32_t)(KPS * r_tile);
    const CUtensorMap* mapF = part == 0 ? &tmF0 : (part == 1 ? &tmF1 : &tmF2);
    const int fy = part == 0 ? g.a_row0 + m0 : m0 - pbeg;
    const int ry = g.b_row0 + n0;
    const bool f_lane = lane == 0 || (dual_f && lane == 2);   // loads feature tiles
    const int f_off = lane == 0 ? 0 : KPS * f_tile;            // hi, or lo after it
    const int f_kb = lane == 0 ? 0 : args.f_lo_kb;
    // weights / keys of the first stages: independent of the previous kernel
    const int pre = f_lane ? (nkb < stages ? nkb : stages) : 0;
    for (int i = 0; i < pre; ++i) {
      mbar_expect_tx(&full[i], f_bytes);
      tma_load_3d(smem + i * stage_bytes + r_bytes + f_off, mapF, &full[i], 0, fy,
                  (su_lo + i) * KPS + f_kb);
    }
    if (lane == 0) {
      // L2 prefetch of data later kernels of the step read (memory entries,
      // weights: none of it is written by the previous kernel), this CTA's
      // share of each range, in copies of up to 32 KB
      const int ncta = (int)(gridDim.x * gridDim.y * gridDim.z);
      const int cid = (int)(blockIdx.x + gridDim.x * (blockIdx.y + gridDim.y * blockIdx.z));
      for (int r = 0; r < args.n_prefetch; ++r) {
        const long long bytes = args.pf_bytes[r] & ~15ll;
        const long long share = ((bytes + ncta - 1) / ncta + 15) & ~15ll;
        const long long beg = (long long)cid * share;
        const long long len = min(share, bytes - beg);
        const uint8_t* base = static_cast<const uint8_t*>(args.pf_ptr[r]) + beg;
        for (long long off = 0; off < len; off += 32768)
          prefetch_l2_bulk(base + off, (uint32_t)min(32768ll, len - off));
      }
    }
    pdl_wait();
    pdl_trigger();
    int issued = 0;
    for (int i = 0; i < nkb; ++i) {
      const int kb = (su_lo + i) * KPS;
      const int st = i % stages;
      const uint32_t ph = (uint32_t)(i / stages) & 1u;
      uint8_t* stg = smem + st * stage_bytes;
      if (i >= pre) {
        if (!mbar_wait(&empty[st], ph ^ 1u, abort_flag, args.wait_ns)) {
          *abort_flag = 1;
          break;
        }
        if (f_lane) {
          mbar_expect_tx(&full[st], f_bytes);
          tma_load_3d(stg + r_bytes + f_off, mapF, &full[st], 0, fy, kb + f_kb);
        } else {
          mbar_expect_tx(&full[st], r_lane_bytes);
          if constexpr (DUAL) {
            if (lane == 1)
              tma_load_3d(stg, &tmR0, &full[st], 0, ry, kb);
            else
              tma_load_3d(stg + KPS * r_tile, &tmR1, &full[st], 0, ry, kb);
          } else {
            // the row operand: by contraction index (B1 from b_split on),
            // or by feature part (B1 for the columns of F1 and F2)
            const bool r_second = args.r_by_part ? part != 0 : kb >= r_split_kb;
            tma_load_3d(stg, r_second ? &tmR1 : &tmR0, &full[st], 0, ry,
                        (r_second && !args.r_by_part) ? kb - r_split_kb : kb);
          }
        }
      }
      ++issued;
    }
    // every copy in flight has landed before the ring is reused or the CTA
    // leaves (in the normal case these stages completed long ago)
    for (int i = issued > stages ? issued - stages : 0; i < issued; ++i)
      mbar_wait(&full[i % stages], (uint32_t)(i / stages) & 1u, nullptr, 20000000ull);
  } else if (warp == 1 && lane == 0 && nkb > 0) {
    // ---- MMA issuer (single elected thread) ----
    for (int i = 0; i < nkb; ++i) {
      const int st = i % stages;
      const uint32_t ph = (uint32_t)(i / stages) & 1u;
      if (!mbar_wait(&full[st], ph, abort_flag, args.wait_ns)) {
        *abort_flag = 1;
        break;
      }
      // no tcgen05 fence here: the stage was written by TMA and published by
      // the mbarrier
      const uint32_t stg = smem_u32(smem + st * stage_bytes);
      for (int j = 0; j < KPS; ++j) {
        const uint64_t adesc = sw128_desc(stg + (uint32_t)(j * r_tile));
        const uint64_t bdesc = sw128_desc(stg + (uint32_t)(r_bytes + j * f_tile));
#pragma unroll
        for (int k = 0; k < BK / UMMA_K; ++k) {
          // advance the start address by k * 32 bytes inside the swizzle atom
          umma_bf16(tmem_base, adesc + (uint64_t)(2 * k), bdesc + (uint64_t)(2 * k), C::IDESC,
                    (i > 0 || j > 0 || k > 0) ? 1u : 0u);
          if constexpr (DUAL) {
            const uint64_t adesc_lo = sw128_desc(stg + (uint32_t)((KPS + j) * r_tile));
            umma_bf16(tmem_base, adesc_lo + (uint64_t)(2 * k), bdesc + (uint64_t)(2 * k), C::IDESC,
                      1u);
          }
          if (dual_f) {
            const uint64_t bdesc_lo = sw128_desc(stg + (uint32_t)(r_bytes + (KPS + j) * f_tile));
            umma_bf16(tmem_base, adesc + (uint64_t)(2 * k), bdesc_lo + (uint64_t)(2 * k), C::IDESC,
                      1u);
          }
        }
      }
      umma_commit(&empty[st]);      // frees this stage once its MMAs have read it
    }
    umma_commit(accum);             // all issued MMAs complete -> accumulator ready
  }

  // ---- epilogue: all eight warps.  Warp w reads accumulator lanes (rows)
  // 32 (w % 4) .. +31; warps w and w + 4 take the two halves of the columns.
  if constexpr (EPI == kEpiBiasSilu || EPI == kEpiBiasF32 || EPI == kEpiAct) {
    // the tile's biases (weights: independent of the predecessor), fetched by
    // warps 2-7 while the accumulator is produced
    typedef __nv_bfloat16 Tb;
    for (int c = (int)threadIdx.x - 64; c < BN; c += kThreads - 64) {
      if (c < 0) continue;
      const int m = m0 + c;
      float b = 0.0f;
      if (m < m_end) {
        if ((EPI == kEpiBiasSilu || EPI == kEpiAct) && m >= args.epi_split)
          b = to_f32(static_cast<const Tb*>(args.bias1)[m - args.epi_split]);
        else
          b = to_f32(static_cast<const Tb*>(args.bias0)[m]);
      }
      bias_s[c] = b;
    }
  }
  pdl_wait();
  __syncwarp();
  bool ok = true;
  if (nkb > 0) {
    const bool waited = mbar_wait(accum, 0, abort_flag, args.wait_ns);
    // after a wait that gave up, the MMAs already issued (the issuer commits
    // them to `accum` however its loop ended) complete before the tensor
    // memory they write is freed
    if (!waited) mbar_wait(accum, 0, nullptr, kDefaultWaitLimitNs);
    // warp-uniform decision: tcgen05.ld below is a .sync.aligned instruction
    ok = __all_sync(0xffffffffu, waited && *abort_flag == 0);
  }
  if (!ok && lane == 0) atomicOr(args.err, kErrTimeout);
  tc_fence_after();
  const int quarter = warp & 3, half = warp >> 2;
  const int row_in_tile = quarter * 32 + lane;
  const int n = n0 + row_in_tile;
  const bool row_ok = n < g.n;
  const uint32_t taddr = tmem_base + ((uint32_t)(quarter * 32) << 16);
  const int n_cols = min(BN, m_end - m0);

  if constexpr (EPI == kEpiStoreKeys) {
    // keys and values (never split).  Each thread owns one token's row: warps
    // 0-3 the first half of the tile's columns, warps 4-7 the second (both
    // take the row's scale over all columns).  The bf16 values go row-major
    // into shared memory over the idle stage ring (pitch BN + 8 elements: a
    // quarter warp's 16-byte stores hit distinct banks), the listed key
    // elements into the fix list with one atomic per warp, and the CTA then
    // writes the tile with 16-byte stores along the rows.
    constexpr int kPitch = BN * 2 + 16;
    constexpr int kChunks = BN / 64;                 // 32-column chunks per half
    const int rows_real = min(BM, g.n - n0);
    if (ok) {
      float ss = 0.0f;
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 32) {
        float v[32];
        tmem_ld32(taddr + (uint32_t)c0, v);
#pragma unroll
        for (int j = 0; j < 32; ++j)
          if (c0 + j < n_cols) ss = fmaf(v[j], v[j], ss);
      }
      const float key_scale = sqrtf(ss / (float)max(n_cols, 1));
      uint32_t need[kChunks];
      int cnt = 0;
#pragma unroll
      for (int ci = 0; ci < kChunks; ++ci) {
        need[ci] = 0u;
        const int c0 = half * (BN / 2) + ci * 32;
        if (c0 >= n_cols) continue;                  // uniform across the warp
        float v[32];
        tmem_ld32(taddr + (uint32_t)c0, v);
        uint32_t pk[16];
#pragma unroll
        for (int j = 0; j < 32; j += 2) {
          const __nv_bfloat16 r0 = __float2bfloat16_rn(v[j]), r1 = __float2bfloat16_rn(v[j + 1]);
          pk[j / 2] = (uint32_t)__bfloat16_as_ushort(r0) | ((uint32_t)__bfloat16_as_ushort(r1) << 16);
          const int m = m0 + c0 + j;
          if (row_ok && m < args.epi_split && c0 + j < n_cols &&
              near_midpoint(v[j], r0, key_scale, args.k_total))
            need[ci] |= 1u << j;
          if (row_ok && m + 1 < args.epi_split && c0 + j + 1 < n_cols &&
              near_midpoint(v[j + 1], r1, key_scale, args.k_total))
            need[ci] |= 2u << j;
        }
        uint4* dst = reinterpret_cast<uint4*>(smem + row_in_tile * kPitch + c0 * 2);
#pragma unroll
        for (int q = 0; q < 4; ++q)
          dst[q] = make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
        cnt += __popc(need[ci]);
      }
      // the warp's listed elements take consecutive slots of the fix list
      int incl = cnt;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int t = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += t;
      }
      const int wtotal = __shfl_sync(0xffffffffu, incl, 31);
      int base = 0;
      if (lane == 31 && wtotal > 0) base = atomicAdd(args.fix_count, wtotal);
      int slot = __shfl_sync(0xffffffffu, base, 31) + incl - cnt;
      const long long row = (long long)g.b_row0 + n;
#pragma unroll
      for (int ci = 0; ci < kChunks; ++ci) {
        uint32_t bits = need[ci];
        while (bits != 0u) {
          const int j = __ffs(bits) - 1;
          bits &= bits - 1u;
          if (slot < args.fix_cap)
            args.fix_list[slot] = KeyFix{(int)row, m0 + half * (BN / 2) + ci * 32 + j};
          ++slot;
        }
      }
    }
    __syncthreads();
    typedef __nv_bfloat16 Tb;
    constexpr int kRowChunks = BN / 8;                // 16-byte chunks of a row
    for (int it = threadIdx.x; it < rows_real * kRowChunks; it += kThreads) {
      const int r = it / kRowChunks, c8 = (it % kRowChunks) * 8;
      if (c8 >= n_cols) continue;
      const int m = m0 + c8;                         // epi_split % 8 == 0
      const long long row = (long long)g.b_row0 + n0 + r;
      Tb* dst = m < args.epi_split
                    ? static_cast<Tb*>(args.out0) + row * args.ldc + m
                    : static_cast<Tb*>(args.out1) + row * args.ldc + (m - args.epi_split);
      *reinterpret_cast<uint4*>(dst) = *reinterpret_cast<const uint4*>(smem + r * kPitch + c8 * 2);
    }
  } else {
    // The accumulator tile goes row-major [rows_real][BN + 4] fp32 into shared
    // memory over the stage ring (idle: every MMA has completed, every copy
    // has landed); the pitch of BN + 4 floats spreads a warp's 16-byte stores
    // over all banks.  Without split K the CTA then writes it out with
    // consecutive threads on consecutive columns; with split K the S CTAs of
    // the tile's cluster meet, and CTA `rank` sums columns [rank cpo,
    // (rank+1) cpo) of the S partial tiles in rank order through distributed
    // shared memory before writing them.
    const int rows_real = min(BM, g.n - n0);
    const bool have_acc = ok && nkb > 0;          // warp-uniform
    if (S == 1) {
      float* part = reinterpret_cast<float*>(smem);
      const int ldp = BN + 4;
      if (quarter * 32 < rows_real) {             // warp-uniform
#pragma unroll 1
        for (int c0 = half * (BN / 2); c0 < (half + 1) * (BN / 2); c0 += 32) {
          float v[32];
          if (have_acc) {
            tmem_ld32(taddr + (uint32_t)c0, v);   // the whole warp, converged
          } else {
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] = 0.0f;
          }
          if (row_in_tile < rows_real) {
#pragma unroll
            for (int q = 0; q < 8; ++q)
              *reinterpret_cast<float4*>(part + row_in_tile * ldp + c0 + 4 * q) =
                  make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
          }
        }
      }
      __syncthreads();
      const int q4 = BN / 4;
      const int items = rows_real * q4;
      float* addt = part + rows_real * ldp;        // kEpiAct: the added term, [rows][BN]
      if constexpr (EPI == kEpiAct) {
        stage_add_tile(args, g, m0, n0, rows_real, n_cols, 0, q4, addt);
        __syncthreads();
      }
      for (int it = threadIdx.x; it < items; it += kThreads) {
        const int rr = it / q4, cc = (it - rr * q4) * 4;
        const float4 a4 = *reinterpret_cast<const float4*>(part + rr * ldp + cc);
        if (ok && cc < n_cols) {
          float vals[4] = {a4.x, a4.y, a4.z, a4.w};
          if constexpr (EPI == kEpiAct) {
            act_store4(args, g, m0 + cc, n0 + rr, vals, addt + 4 * it, bias_s + cc,
                       min(4, n_cols - cc));
          } else if constexpr (EPI == kEpiLogits) {
            if (args.out2 != nullptr)               // the logits, when asked for
              gemm_epilogue4<kEpiQueryH>(args, g, m0 + cc, n0 + rr, vals, min(4, n_cols - cc),
                                         bias_s + cc);
          } else {
            gemm_epilogue4<EPI>(args, g, m0 + cc, n0 + rr, vals, min(4, n_cols - cc), bias_s + cc);
          }
        }
      }
      if constexpr (EPI == kEpiLogits)
        tile_topk<BN>(args, (long long)g.b_row0 + n0, rows_real, part, ldp, m0, n_cols, tx,
                      reinterpret_cast<uint8_t*>(part + rows_real * ldp),
                      args.region - rows_real * ldp * 4);
    } else {
      // Split K: each CTA stages its fp32 partial tile row-major [rows][BN + 4]
      // over its idle ring (the pitch spreads a warp's 16-byte stores over all
      // banks); the cluster meets, and CTA `rank` sums the column quads
      // [qlo, qhi) of the S partial tiles in rank order through distributed
      // shared memory; a second cluster barrier keeps every partial alive
      // until it has been read.
      float* part = reinterpret_cast<float*>(smem);
      const int ldp = BN + 4;
      if (quarter * 32 < rows_real) {             // warp-uniform
#pragma unroll 1
        for (int c0 = half * (BN / 2); c0 < (half + 1) * (BN / 2); c0 += 32) {
          float v[32];
          if (have_acc) {
            tmem_ld32(taddr + (uint32_t)c0, v);   // the whole warp, converged
          } else {
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] = 0.0f;
          }
          if (row_in_tile < rows_real) {
#pragma unroll
            for (int q = 0; q < 8; ++q)
              *reinterpret_cast<float4*>(part + row_in_tile * ldp + c0 + 4 * q) =
                  make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
          }
        }
      }
      __syncwarp();
      cluster_sync();
      const int qlo = (int)rank * (BN / 4) / S, qhi = ((int)rank + 1) * (BN / 4) / S;
      const int q4 = qhi - qlo;
      const int items = rows_real * q4;
      float* addt = part + rows_real * ldp;        // kEpiAct: the added term, [rows][q4 * 4]
      float* sums = part + rows_real * ldp;        // kEpiLogits: the reduced logits, [rows][q4 * 4]
      if constexpr (EPI == kEpiAct) {
        stage_add_tile(args, g, m0, n0, rows_real, n_cols, qlo, q4, addt);
        __syncthreads();
      }
      // two items per thread and round, all their remote loads in flight
      // together.  The closing cluster barrier is split: each thread arrives
      // once its last round's remote loads have been summed, before that
      // round's global stores, so the arrival's release orders no global
      // write; it waits after the stores.
      const int rounds = (items + 2 * kThreads - 1) / (2 * kThreads);   // uniform in the CTA
      for (int rd = 0; rd < rounds; ++rd) {
        const int it0 = threadIdx.x + rd * 2 * kThreads;
        float4 t[2][8];
        int rr[2], cc[2];
#pragma unroll
        for (int k = 0; k < 2; ++k) {
          const int it = it0 + k * kThreads;
          rr[k] = -1;
          if (it < items) {
            rr[k] = it / q4;
            cc[k] = (qlo + (it - rr[k] * q4)) * 4;
            const uint32_t laddr = smem_u32(part + rr[k] * ldp + cc[k]);
#pragma unroll
            for (int sidx = 0; sidx < 8; ++sidx)
              if (sidx < S) t[k][sidx] = ld_dsmem_f4(map_dsmem(laddr, (uint32_t)sidx));
          }
        }
        float4 acc[2];
#pragma unroll
        for (int k = 0; k < 2; ++k) {
          if (rr[k] < 0) continue;
          acc[k] = t[k][0];
#pragma unroll
          for (int sidx = 1; sidx < 8; ++sidx)
            if (sidx < S) {
              acc[k].x += t[k][sidx].x;
              acc[k].y += t[k][sidx].y;
              acc[k].z += t[k][sidx].z;
              acc[k].w += t[k][sidx].w;
            }
        }
        if (rd == rounds - 1) {
          __syncwarp();
          cluster_arrive();   // this CTA's remote reads are done
        }
#pragma unroll
        for (int k = 0; k < 2; ++k) {
          if (rr[k] < 0) continue;
          if (ok && cc[k] < n_cols) {
            float vals[4] = {acc[k].x, acc[k].y, acc[k].z, acc[k].w};
            if constexpr (EPI == kEpiAct) {
              const int it = it0 + k * kThreads;
              act_store4(args, g, m0 + cc[k], n0 + rr[k], vals, addt + 4 * it, bias_s + cc[k],
                         min(4, n_cols - cc[k]));
            } else if constexpr (EPI == kEpiLogits) {
              const int it = it0 + k * kThreads;
              *reinterpret_cast<float4*>(sums + 4 * it) = acc[k];
              if (args.out2 != nullptr)
                gemm_epilogue4<kEpiQueryH>(args, g, m0 + cc[k], n0 + rr[k], vals,
                                           min(4, n_cols - cc[k]), bias_s + cc[k]);
            } else {
              gemm_epilogue4<EPI>(args, g, m0 + cc[k], n0 + rr[k], vals, min(4, n_cols - cc[k]),
                                  bias_s + cc[k]);
            }
          }
        }
      }
      if (rounds == 0) {
        __syncwarp();
        cluster_arrive();
      }
      if constexpr (EPI == kEpiLogits) {
        __syncthreads();
        tile_topk<BN>(args, (long long)g.b_row0 + n0, rows_real, sums, q4 * 4, m0 + qlo * 4,
                      max(0, min(q4 * 4, n_cols - qlo * 4)), tx * S + (int)rank,
                      reinterpret_cast<uint8_t*>(sums + rows_real * q4 * 4),
                      args.region - (rows_real * ldp + rows_real * q4 * 4) * 4);
      }
      cluster_wait();   // no CTA leaves while another still reads its partial tile
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, C::TMEM_COLS);
  }
}

}  // namespace tc

// ---------------------------------------------------------------------------
// Host side: tensor maps and dispatch
// ---------------------------------------------------------------------------
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encoder() {
  static EncodeTiledFn fn = nullptr;
  if (fn == nullptr) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

// [rows, cols] bf16, row stride ld elements; box = 64 columns x box_rows rows.
static bool make_map(CUtensorMap* m, const TmaOperand& op, int box_rows) {
  EncodeTiledFn enc = encoder();
  if (enc == nullptr || op.base == nullptr || op.rows <= 0 || op.cols <= 0) return false;
  cuuint64_t dims[2] = {(cuuint64_t)op.cols, (cuuint64_t)op.rows};
  cuuint64_t strides[1] = {(cuuint64_t)op.ld * 2};
  cuuint32_t box[2] = {(cuuint32_t)tc::BK, (cuuint32_t)box_rows};
  cuuint32_t es[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(op.base), dims, strides, box,
             es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// [rows, cols] bf16 (row stride ld elements, cols a multiple of 64) viewed as
// (64 k, rows, cols / 64 k-blocks); box = 64 x box_rows x kps: kps
// consecutive k-blocks of box_rows rows per copy, one 128-byte-swizzled
// [box_rows][128 B] tile per k-block in shared memory.
static bool make_map3(CUtensorMap* m, const TmaOperand& op, int box_rows, int kps) {
  EncodeTiledFn enc = encoder();
  if (enc == nullptr || op.base == nullptr || op.rows <= 0 || op.cols <= 0 || op.cols % 64 != 0)
    return false;
  cuuint64_t dims[3] = {64, (cuuint64_t)op.rows, (cuuint64_t)(op.cols / 64)};
  cuuint64_t strides[2] = {(cuuint64_t)op.ld * 2, 128};
  cuuint32_t box[3] = {64, (cuuint32_t)box_rows, (cuuint32_t)kps};
  cuuint32_t es[3] = {1, 1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(op.base), dims, strides, box,
             es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Encoded maps of this thread, by their parameters: a tensor map is a pure
// function of (base, shape, row stride, box), so a draft step that runs with
// the same buffers reuses its maps instead of encoding ~10 per call.
struct MapKey {
  const void* base;
  long long rows, cols, ld;
  int box_rows, kps;
  bool operator==(const MapKey& o) const {
    return base == o.base && rows == o.rows && cols == o.cols && ld == o.ld &&
           box_rows == o.box_rows && kps == o.kps;
  }
};
struct MapKeyHash {
  size_t operator()(const MapKey& k) const {
    size_t h = std::hash<const void*>()(k.base);
    for (long long v : {k.rows, k.cols, k.ld, (long long)k.box_rows, (long long)k.kps})
      h = h * 1000003u ^ std::hash<long long>()(v);
    return h;
  }
};
static bool cached_map3(CUtensorMap* m, const TmaOperand& op, int box_rows, int kps) {
  static thread_local std::unordered_map<MapKey, CUtensorMap, MapKeyHash> cache;
  const MapKey key{op.base, op.rows, op.cols, op.ld, box_rows, kps};
  auto it = cache.find(key);
  if (it != cache.end()) {
    *m = it->second;
    return true;
  }
  if (!make_map3(m, op, box_rows, kps)) return false;
  if (cache.size() >= 512) cache.clear();          // bounded: many distinct buffers
  cache.emplace(key, *m);
  return true;
}

bool encode_bf16_map(CUtensorMap* m, const void* base, long long rows, long long cols,
                     long long ld, int box_rows) {
  return make_map(m, TmaOperand{base, rows, cols, ld}, box_rows);
}

static std::atomic<unsigned long long> g_wait_limit_ns{kDefaultWaitLimitNs};
void set_wait_limit_ns(unsigned long long ns) { g_wait_limit_ns.store(ns); }
unsigned long long wait_limit_ns() { return g_wait_limit_ns.load(); }

static int num_sms() {
  static int sms = 0;
  if (sms == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (sms <= 0) sms = 148;
  }
  return sms;
}

template <int BN, int EPI>
static auto tc_kernel() {
  auto kern = tc::tc_gemm_kernel<BN, EPI>;
  static bool configured = false;
  if (!configured) {
    cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         tc::kSmemBudget + tc::kSmemExtra);
    configured = true;
  }
  return kern;
}

static int stages_for(int nkb, int budget, int stage_bytes) {
  int st = budget / stage_bytes;
  st = st > tc::kMaxStages ? tc::kMaxStages : st;
  st = st > nkb ? nkb : st;
  return st < 1 ? 1 : st;
}

// CTAs of this kernel resident on the GPU at once.
template <int BN, int EPI>
static int resident_ctas(int smem) {
  static int cache[64];      // by smem / 4 KB
  const int mi = (smem >> 12) & 63;
  if (cache[mi] != 0) return cache[mi];
  auto kern = tc_kernel<BN, EPI>();
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, tc::kThreads, smem) !=
          cudaSuccess || per_sm <= 0) {
    cudaGetLastError();
    per_sm = 1;
  }
  cache[mi] = per_sm * num_sms();
  return cache[mi];
}

// Clusters of S CTAs of this kernel resident on the GPU at once.
template <int BN, int EPI>
static int resident_clusters(int smem, int S) {
  static int cache[64][9];   // by smem / 4 KB, S
  const int mi = (smem >> 12) & 63, si = S & 7 ? S : 8;
  if (cache[mi][si] != 0) return cache[mi][si];
  auto kern = tc_kernel<BN, EPI>();
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(S, 1, 1);
  cfg.blockDim = dim3(tc::kThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = S;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess || n <= 0) {
    cudaGetLastError();
    n = -1;                  // cannot be launched with this configuration
  }
  cache[mi][si] = n;
  return n;
}

template <int BN, int EPI>
static cudaError_t launch_tc_inst(GemmArgs& a, const CUtensorMap* maps, int tiles_x, int max_n,
                                  const GemmPlan& p, cudaStream_t s) {
  constexpr bool DUAL = EPI == kEpiScores || EPI == kEpiAct;
  auto kern = tc_kernel<BN, EPI>();
  a.splits = p.splits;
  a.stages = p.stages;
  a.region = p.region;
  a.kps = p.kps;
  a.rbox = p.rbox;
  a.tx_bytes = tc::Cfg<BN, DUAL>::stage_bytes(p.kps, p.rbox,
                                              EPI == kEpiScoresFolded && a.f_lo_kb > 0);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(tiles_x * p.splits, (max_n + tc::BM - 1) / tc::BM, a.ngroups);
  cfg.blockDim = dim3(tc::kThreads, 1, 1);
  cfg.dynamicSmemBytes = p.region + tc::kSmemExtra;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (p.splits > 1) {
    // the S CTAs of an output tile form one cluster
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = p.splits;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.numAttrs = 2;
  }
  return cudaLaunchKernelEx(&cfg, kern, maps[0], maps[1], maps[2], maps[3], maps[4], a);
}

template <int EPI>
static cudaError_t launch_tc_epi(GemmArgs& a, const CUtensorMap* maps, const GemmPlan& p,
                                 int tiles_x, int max_n, cudaStream_t s) {
  switch (p.bn) {
    case 64: return launch_tc_inst<64, EPI>(a, maps, tiles_x, max_n, p, s);
    case 128: return launch_tc_inst<128, EPI>(a, maps, tiles_x, max_n, p, s);
    default: return launch_tc_inst<256, EPI>(a, maps, tiles_x, max_n, p, s);
  }
}

// Feature tiles of the widest group: each operand part is tiled on its own.
static int feature_tiles(const GemmArgs& a, int max_m, int bn) {
  const int s1 = std::min(a.a_split, max_m);
  const int s2 = std::max(s1, std::min(a.a_split2, max_m));
  return (s1 + bn - 1) / bn + (s2 - s1 + bn - 1) / bn + (max_m - s2 + bn - 1) / bn;
}

// Issue time of one tcgen05.mma (M = 128, K = 16) by feature-tile width, in
// cycles, measured on GB300 with back-to-back instructions.
static int mma_cycles(int bn) { return bn <= 64 ? 50 : bn <= 128 ? 66 : bn <= 192 ? 98 : 129; }

// Estimated time (us) of a plan, fitted to stage timings measured on GB300
// (per-CTA globaltimer stamps over the draft-step GEMMs, cold L2):
//   first   the first stage lands: ~0.8 us plus the first stages of all CTAs
//           at the HBM rate (~7 TB/s);
//   stage   when the feature operand streams from HBM (one row tile per
//           group: every feature byte is read once), a ring stage costs
//           ~0.45 us plus ~7.5 ns per KB (a producer lane lands about one
//           copy at a time from HBM); when row tiles share the feature
//           operand through L2, ~0.31 us plus the stage at ~200 KB/us.  At
//           least the MMAs it feeds and the feature bytes of all CTAs'
//           stages at the HBM rate; with a one-stage ring the copies and the
//           MMAs do not overlap;
//   tail    epilogue: ~2 us, plus the cluster reduction for split K
//           (~2.4 us + 0.25 us per CTA of the cluster);
// per wave of resident CTAs.
static double plan_cost_us(bool streaming, double stage_kb, double stage_f_bytes, double mma_us,
                           int stages, int nst, long long ctas_resident, int per_sm, long long waves,
                           int S) {
  const double hbm = 7.0e6;                        // bytes per us
  const double all_f = (double)ctas_resident * stage_f_bytes / hbm;
  const double t_copy = streaming ? 0.45 + 0.0075 * stage_kb : 0.31 + stage_kb / 200.0;
  double t_stage = std::max(t_copy, mma_us) * per_sm;
  if (stages == 1) t_stage += mma_us;
  t_stage = std::max(t_stage, all_f);
  const double t_first = 0.8 + all_f;
  const double t_tail = S == 1 ? 2.0 : 2.4 + 0.25 * S;
  return waves * (t_first + nst * t_stage) + t_tail;
}

template <int BN, int EPI>
static void plan_for(const GemmArgs& a, int max_m, int max_n, long long row_tiles,
                     GemmPlan& best, double& best_t) {
  constexpr bool DUAL = EPI == kEpiScores || EPI == kEpiAct;
  using C = tc::Cfg<BN, DUAL>;
  // folded scores with hi / lo folded keys: the key part's stages hold two
  // feature tiles and issue two MMAs per k-step (the plan is sized for them)
  const bool DF = EPI == kEpiScoresFolded && a.f_lo_kb > 0;
  const int kb_total = a.k_total / tc::BK;
  const int r_split_kb = a.b_split / tc::BK;
  const long long ftiles = feature_tiles(a, max_m, BN);
  const long long tiles = ftiles * row_tiles;          // the grid (every group sized to the largest)
  // tiles with work: groups of ragged sizes leave the rest of their grid
  // slots empty (those CTAs exit at once), so the cost counts these
  long long active = 0;
  for (int gi = 0; gi < a.ngroups; ++gi)
    active += (long long)feature_tiles(a, a.groups[gi].m, BN) *
              ((a.groups[gi].n + tc::BM - 1) / tc::BM);
  if (active <= 0 || active > tiles) active = tiles;
  // the same at the narrowest feature tile: the parallelism the GEMM has
  long long active64 = 0;
  for (int gi = 0; gi < a.ngroups; ++gi)
    active64 += (long long)feature_tiles(a, a.groups[gi].m, 64) *
                ((a.groups[gi].n + tc::BM - 1) / tc::BM);
  const int rows = max_n < tc::BM ? max_n : tc::BM;
  // rows of a row tile: >= 64 so that the MMA's 128-row read stays inside its stage
  const int rbox = std::max(64, std::min(tc::BM, (max_n + 7) / 8 * 8));
  const int sms = num_sms();
  const bool streaming = max_n <= tc::BM;             // one row tile per group
  for (int kps = 4; kps >= 1; kps >>= 1) {
    if (kb_total % kps != 0 || r_split_kb % kps != 0) continue;
    const int su_total = kb_total / kps;
    const double stage_f = (double)kps * BN * 128 * (DF ? 2 : 1);
    const double stage_mma_us =
        (double)kps * 4.0 * mma_cycles(BN) * ((DUAL || DF) ? 2 : 1) / 2070.0;
    const int sb = C::stage_bytes(kps, rbox, DF);
    for (int S = 1; S <= 8; ++S) {
      if (S > 1 && (EPI == kEpiStoreKeys || S > su_total)) break;
      // the weighted-sum GEMM over <= 1024 entries: when its narrowest tiles
      // already fill half the GPU, the split-K reduction and activation
      // epilogue (measured ~4 us per round) outweigh the shorter main loop,
      // so it runs unsplit
      if (S > 1 && EPI == kEpiAct && kb_total <= 16 && 2 * active64 >= sms) break;
      const int nst = (su_total + S - 1) / S;
      const long long ctas = active * S;
      // the accumulator tile [rows][BN + 4] fp32 (and after it, for kEpiAct
      // the added term, for split kEpiLogits the reduced logits, [rows][BN])
      const int staging = EPI == kEpiStoreKeys ? rows * (BN * 2 + 16)
                          : rows * (BN + 4 + ((EPI == kEpiAct || (EPI == kEpiLogits && S > 1)) ? BN : 0)) * 4;
      for (int budget : {tc::kSmemBudget, tc::kSmemBudgetPair}) {
        if (sb > budget) continue;
        const int stages = stages_for(nst, budget, sb);
        const int region = std::max(stages * sb, staging);
        const int smem = region + tc::kSmemExtra;
        if (region > tc::kSmemBudget) continue;
        long long cap = resident_ctas<BN, EPI>(smem);
        if (S > 1) {
          const int nc = resident_clusters<BN, EPI>(smem, S);
          if (nc <= 0) continue;
          cap = std::min<long long>(cap, (long long)nc * S);
        }
        if (cap <= 0) continue;
        const long long waves = (ctas + cap - 1) / cap;
        const long long per_sm = std::max<long long>(1, (std::min(ctas, cap) + sms - 1) / sms);
        const double t = plan_cost_us(streaming, sb / 1024.0, stage_f,
                                      stage_mma_us, stages, nst, std::min(ctas, cap), (int)per_sm,
                                      waves, S);
        if (t < best_t - 1e-6 || (t < best_t + 1e-6 && tiles * S < best.tiles * best.splits)) {
          best_t = t;
          best = GemmPlan{BN, S, stages, 0, tiles, rbox, region, kps};
        }
      }
    }
  }
}

template <int EPI>
static GemmPlan plan_epi(const GemmArgs& a, int max_m, int max_n) {
  const long long row_tiles = (long long)(max_n + tc::BM - 1) / tc::BM * a.ngroups;
  GemmPlan best{256, 1, 2, 0, 1 << 30, 128, 0, 1};
  double best_t = 1e30;
  plan_for<256, EPI>(a, max_m, max_n, row_tiles, best, best_t);
  plan_for<128, EPI>(a, max_m, max_n, row_tiles, best, best_t);
  plan_for<64, EPI>(a, max_m, max_n, row_tiles, best, best_t);
  return best;
}

static GemmPlan plan_gemm_tc_uncached(int epi, const GemmArgs& a, int max_m, int max_n) {
  switch (epi) {
    case kEpiStore: return plan_epi<kEpiStore>(a, max_m, max_n);
    case kEpiScores: return plan_epi<kEpiScores>(a, max_m, max_n);
    case kEpiBiasSilu: return plan_epi<kEpiBiasSilu>(a, max_m, max_n);
    case kEpiStoreHiLo: return plan_epi<kEpiStoreHiLo>(a, max_m, max_n);
    case kEpiStoreKeys: return plan_epi<kEpiStoreKeys>(a, max_m, max_n);
    case kEpiQueryH: return plan_epi<kEpiQueryH>(a, max_m, max_n);
    case kEpiScoresFolded: return plan_epi<kEpiScoresFolded>(a, max_m, max_n);
    case kEpiAct: return plan_epi<kEpiAct>(a, max_m, max_n);
    case kEpiLogits: return plan_epi<kEpiLogits>(a, max_m, max_n);
    default: return plan_epi<kEpiBiasF32>(a, max_m, max_n);
  }
}

// Plans of this thread, by the arguments the planner reads (a draft step
// plans the same few GEMMs on every call).
GemmPlan plan_gemm_tc(int epi, const GemmArgs& a, int max_m, int max_n) {
  static thread_local std::unordered_map<std::string, GemmPlan> cache;
  std::string key;
  key.reserve(64 + 16 * a.ngroups);
  char buf[160];
  snprintf(buf, sizeof buf, "%d|%d|%d|%d|%d|%d|%d|%d|%d|", epi, max_m, max_n, a.k_total, a.b_split,
           a.a_split, a.a_split2, a.f_lo_kb, a.ngroups);
  key += buf;
  for (int g = 0; g < a.ngroups; ++g) {
    snprintf(buf, sizeof buf, "%d,%d;", a.groups[g].m, a.groups[g].n);
    key += buf;
  }
  auto it = cache.find(key);
  if (it != cache.end()) return it->second;
  const GemmPlan p = plan_gemm_tc_uncached(epi, a, max_m, max_n);
  if (cache.size() >= 256) cache.clear();
  cache.emplace(key, p);
  return p;
}

int lm_head_slots(int vocab, int d_model, int N) {
  static thread_local GemmArgs a;
  memset(&a, 0, sizeof(a));
  a.k_total = d_model;
  a.b_split = d_model;
  a.a_split = 0x7fffffff;
  a.a_split2 = 0x7fffffff;
  a.epi_split = 0;
  a.ngroups = 1;
  a.groups[0] = GemmGroup{0, vocab, 0, N, 0};
  const GemmPlan p = plan_gemm_tc(kEpiLogits, a, vocab, N);
  return feature_tiles(a, vocab, p.bn) * p.splits;
}

cudaError_t launch_gemm_tc(int epi, const GemmArgs& args, const TmaOperand& A0, const TmaOperand& A1,
                           const TmaOperand& B0, const TmaOperand& B1, int max_m, int max_n,
                           cudaStream_t s, const TmaOperand& A2) {
  if (max_m <= 0 || max_n <= 0 || args.ngroups <= 0) return cudaSuccess;
  static thread_local GemmArgs a;
  a = args;
  a.wait_ns = wait_limit_ns();
  // L2 prefetch for later kernels: at most half of the 129 MB L2 in all (a
  // larger range evicts its own first lines before they are read, and its
  // HBM reads compete with this GEMM's), taken from the front of each range
  // in order
  long long pf_left = 64ll << 20;
  for (int r = 0; r < a.n_prefetch; ++r) {
    a.pf_bytes[r] = std::min(a.pf_bytes[r], pf_left);
    pf_left -= a.pf_bytes[r];
  }
  const GemmPlan plan = plan_gemm_tc(epi, a, max_m, max_n);
  if (plan.region <= 0) return cudaErrorInvalidConfiguration;
  CUtensorMap maps[5];            // F0, F1, F2, R0, R1
  const TmaOperand& a1 = A1.base ? A1 : A0;
  const TmaOperand& a2 = A2.base ? A2 : a1;
  const TmaOperand& b1 = B1.base ? B1 : B0;
  if (!cached_map3(&maps[0], A0, plan.bn, plan.kps) || !cached_map3(&maps[1], a1, plan.bn, plan.kps) ||
      !cached_map3(&maps[2], a2, plan.bn, plan.kps) || !cached_map3(&maps[3], B0, plan.rbox, plan.kps) ||
      !cached_map3(&maps[4], b1, plan.rbox, plan.kps))
    return cudaErrorInvalidValue;
  const int tiles_x = feature_tiles(a, max_m, plan.bn);
  switch (epi) {
    case kEpiStore: return launch_tc_epi<kEpiStore>(a, maps, plan, tiles_x, max_n, s);
    case kEpiScores: return launch_tc_epi<kEpiScores>(a, maps, plan, tiles_x, max_n, s);
    case kEpiBiasSilu: return launch_tc_epi<kEpiBiasSilu>(a, maps, plan, tiles_x, max_n, s);
    case kEpiStoreHiLo: return launch_tc_epi<kEpiStoreHiLo>(a, maps, plan, tiles_x, max_n, s);
    case kEpiStoreKeys: return launch_tc_epi<kEpiStoreKeys>(a, maps, plan, tiles_x, max_n, s);
    case kEpiQueryH: return launch_tc_epi<kEpiQueryH>(a, maps, plan, tiles_x, max_n, s);
    case kEpiScoresFolded: return launch_tc_epi<kEpiScoresFolded>(a, maps, plan, tiles_x, max_n, s);
    case kEpiAct: return launch_tc_epi<kEpiAct>(a, maps, plan, tiles_x, max_n, s);
    case kEpiLogits: return launch_tc_epi<kEpiLogits>(a, maps, plan, tiles_x, max_n, s);
    default: return launch_tc_epi<kEpiBiasF32>(a, maps, plan, tiles_x, max_n, s);
  }
}

}  // namespace fovea
