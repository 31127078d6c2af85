// Cumulative-mass selection of one draft state by a group of 256 threads
// (retrieval section of the paper: the global softmax alpha-tilde over the
// valid entries, the descending order pi_n, the cardinality
// K_raw = min{k : sum_{t<=k} alpha-tilde_{pi(t)} >= rho}, its clamp
// K = min(|V|, K_max, max(K_min, K_raw)), and the renormalised weights over
// I_n = pi_n(1..K)).
//
// The caller stages the row's scores in shared memory (-0 mapped to +0) and
// calls select_row.  A histogram of the distance to the maximum finds the
// bin holding the K_eff-th largest score (K_eff = min(K_max, |V|)) without
// sorting the row: in registers for rows of up to 2048 entries (select_fast),
// in strided passes over shared memory above that (select_wide).  The entries
// of the bins up to it are the candidates; only they are put in order, by
// (score desc, position asc): each candidate's rank is its count of larger
// candidates for up to 256 candidates, a bucket order above that.  An fp32
// inclusive scan of exp(s - s_max) over the first K_eff gives the cumulative
// mass, and the first prefix reaching rho sets K.  More than 1024 candidates
// (many equal scores) take a 4-pass 8-bit radix select of the K_eff-th key
// instead (select_finish).
//
// Used by the standalone select kernel (a CTA of 256 threads, __syncthreads)
// and by the selection + gather kernel (its first 256 threads, a named
// barrier): `sync` is the group barrier, `tid` the thread's index in the
// group, and the group's warps are whole hardware warps.
#pragma once
#include "common.cuh"

namespace fovea {

constexpr int kSelThreads = 256;
constexpr int kSelWarps = kSelThreads / 32;
constexpr int kRankMax = 256;          // direct ranking up to this many candidates

// Monotone map of a float to uint32 (larger float -> larger key); -0 is
// mapped like +0 by the caller.
__device__ __forceinline__ uint32_t ord_key(float f) {
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

struct SelectArgs {
  const float* scores;
  const int32_t* orig_index;
  float rho;
  int k_min, k_max;
  int32_t* counts;     // [N] or null
  int32_t* indices;    // [N, k_max] or null
  int32_t* sel_pos;    // [N, k_max] compacted memory row of each selected entry, or null
  float* sel_w;        // [N, k_max] renormalised weight alpha, or null
  int32_t* sel_cnt;    // [N] or null
  // the same selection for the calling group alone (shared memory, entry t at
  // [t]; K <= kRankMax when used), or null
  int32_t* loc_pos;
  float* loc_w;
  int* loc_cnt;
  DepthGate gate;      // rows past the depth gate select nothing (K = 0)
  // the renormalised weights as dense rows over the sequence's entries, a
  // bf16 hi / lo pair [N, alpha_ld] (zero where not selected), or null
  __nv_bfloat16* alpha_hi;
  __nv_bfloat16* alpha_lo;
  int alpha_ld;
};

// Weight alpha of the entry at position pos (within its sequence) of row n
// into the dense rows (the caller zero-filled them first).
__device__ __forceinline__ void put_alpha(const SelectArgs& a, int n, int pos, float w) {
  if (a.alpha_hi == nullptr) return;
  const __nv_bfloat16 hi = __float2bfloat16_rn(w);
  const long long o = (long long)n * a.alpha_ld + pos;
  a.alpha_hi[o] = hi;
  a.alpha_lo[o] = __float2bfloat16_rn(w - __bfloat162float(hi));
}

// Zero-fills row n of the dense weights (group of `nthreads`, index tid).
__device__ __forceinline__ void clear_alpha(const SelectArgs& a, int n, int tid, int nthreads) {
  if (a.alpha_hi == nullptr) return;
  const long long o = (long long)n * a.alpha_ld;
  const __nv_bfloat16 z = __float2bfloat16_rn(0.0f);
  for (int j = tid; j < a.alpha_ld; j += nthreads) {
    a.alpha_hi[o + j] = z;
    a.alpha_lo[o + j] = z;
  }
}

struct SelectSmem {
  unsigned long long cand[FOVEA_MAX_K];      // (key << 32) | ~position
  unsigned long long sorted[FOVEA_MAX_K];     // ordered keys; scratch of bucket_order
  float cum[FOVEA_MAX_K];                    // inclusive scan of exp(s - s_max)
  unsigned int hist[256];
  float red_m[kSelWarps], red_s[kSelWarps], red_lo[kSelWarps];
  float warp_tot_f[kSelWarps];
  int warp_tot[kSelWarps];
  int warp_first[kSelWarps];
  unsigned int red_u[kSelWarps];
  unsigned int sh_digit, sh_above;
  int sh_cnt_gt, sh_first;
  float sh_max, sh_sum;
};

// (max, sum of exp(x - max)) pairs combine as a softmax denominator.
__device__ __forceinline__ void combine_ms(float& m, float& s, float m2, float s2) {
  if (m2 > m) {
    s = s * expf(m - m2) + s2;
    m = m2;
  } else if (m2 != -INFINITY) {
    s = s + s2 * expf(m2 - m);
  }
}

// Group-wide combination of the threads' (max, sum) pairs: warps first, then
// warp 0's lane 0 folds the warps in order.  Every thread returns the result.
template <class Sync>
__device__ __forceinline__ void select_stats(float lmax, float lsum, SelectSmem& sm, int tid,
                                             Sync sync, float& smax, float& sumexp) {
  const int lane = tid & 31, warp = tid >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, lmax, o);
    const float s2 = __shfl_xor_sync(0xffffffffu, lsum, o);
    combine_ms(lmax, lsum, m2, s2);
  }
  if (lane == 0) {
    sm.red_m[warp] = lmax;
    sm.red_s[warp] = lsum;
  }
  sync();
  if (tid == 0) {
    float m = sm.red_m[0], s = sm.red_s[0];
    for (int w = 1; w < kSelWarps; ++w) combine_ms(m, s, sm.red_m[w], sm.red_s[w]);
    sm.sh_max = m;
    sm.sh_sum = s;
  }
  sync();
  smax = sm.sh_max;
  sumexp = sm.sh_sum;
}

// The score a key was made from (ord_key inverted).
__device__ __forceinline__ float key_score(unsigned long long key) {
  const uint32_t k = (uint32_t)(key >> 32);
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k);
}

// Orders the C (<= FOVEA_MAX_K) distinct keys of sm.cand descending, in
// place: a histogram of the candidates' scores over kOrderBins bins of equal
// width between their maximum and minimum (the bin is monotone in the score),
// an exclusive scan of the bins, a scatter of the keys into bin order
// (sm.sorted), and each key's rank among the keys of its own bin.  The
// histogram lives in sm.cum (dead until the mass scan).
constexpr int kOrderBins = 1024;
static_assert(kOrderBins <= FOVEA_MAX_K && kOrderBins == 4 * kSelThreads, "bins in SelectSmem::cum");

template <class Sync>
__device__ void bucket_order(SelectSmem& sm, int C, int tid, Sync sync) {
  const int lane = tid & 31, warp = tid >> 5;
  unsigned int* hist = reinterpret_cast<unsigned int*>(sm.cum);
  float smax = -INFINITY, smin = INFINITY;
  for (int c = tid; c < C; c += kSelThreads) {
    const float v = key_score(sm.cand[c]);
    smax = fmaxf(smax, v);
    smin = fminf(smin, v);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    smax = fmaxf(smax, __shfl_xor_sync(0xffffffffu, smax, o));
    smin = fminf(smin, __shfl_xor_sync(0xffffffffu, smin, o));
  }
  for (int i = tid; i < kOrderBins; i += kSelThreads) hist[i] = 0u;
  if (lane == 0) {
    sm.red_m[warp] = smax;
    sm.red_lo[warp] = smin;
  }
  sync();
#pragma unroll
  for (int w = 0; w < kSelWarps; ++w) {
    smax = fmaxf(smax, sm.red_m[w]);
    smin = fminf(smin, sm.red_lo[w]);
  }
  const float range = smax - smin;
  const float inv_w = range > 0.0f ? (float)(kOrderBins - 1) / range : 0.0f;
  auto bin_of = [&](unsigned long long key) {
    const int b = (int)((smax - key_score(key)) * inv_w);
    return b < 0 ? 0 : (b > kOrderBins - 1 ? kOrderBins - 1 : b);
  };
  for (int c = tid; c < C; c += kSelThreads) atomicAdd(&hist[bin_of(sm.cand[c])], 1u);
  sync();
  // exclusive scan of the bins: thread tid owns bins 4 tid .. 4 tid + 3
  unsigned int cnt[4], tot = 0u;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    cnt[j] = hist[4 * tid + j];
    tot += cnt[j];
  }
  unsigned int incl = tot;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned int t = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += t;
  }
  if (lane == 31) sm.red_u[warp] = incl;
  sync();
  unsigned int run = incl - tot;
  for (int w = 0; w < warp; ++w) run += sm.red_u[w];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    hist[4 * tid + j] = run;                       // start of the bin
    run += cnt[j];
  }
  sync();
  for (int c = tid; c < C; c += kSelThreads) {
    const unsigned long long key = sm.cand[c];
    sm.sorted[atomicAdd(&hist[bin_of(key)], 1u)] = key;
  }
  sync();
  // hist[b] is now the end of bin b, and the start of bin b + 1
  for (int i = tid; i < C; i += kSelThreads) {
    const unsigned long long me = sm.sorted[i];
    const int b = bin_of(me);
    const int beg = b ? (int)hist[b - 1] : 0, end = (int)hist[b];
    int r = beg;
    for (int j = beg; j < end; ++j) r += sm.sorted[j] > me;
    sm.cand[r] = me;
  }
  sync();
}

template <class Sync>
__device__ __forceinline__ void select_tail(const SelectArgs& a, int n, int key_off,
                                            const float* s_sc, int K_eff, int C, float smax,
                                            float sumexp, SelectSmem& sm, int tid, Sync sync);

// Radix select, candidate ordering, mass scan and the outputs of draft state
// n, whose M (>= 1) scores are staged in s_sc.  key_off is the compacted row
// of the sequence's first memory entry.
template <class Sync>
__device__ void select_finish(const SelectArgs& a, int n, int M, int key_off, const float* s_sc,
                              float smax, float sumexp, SelectSmem& sm, int tid, Sync sync) {
  const int lane = tid & 31, warp = tid >> 5;
  const int K_eff = min(a.k_max, M);

  // ---- radix select of the K_eff-th largest key ----------------------------
  // (every entry selected, the dense setting: no threshold to find; every
  // key is above 0, so T = 0 takes them all)
  uint32_t prefix = 0, pmask = 0;
  int krem = K_eff;                       // entries still to take at the current prefix
  if (K_eff == M) krem = 0;
  for (int shift = 24; shift >= 0 && K_eff < M; shift -= 8) {
    for (int i = tid; i < 256; i += kSelThreads) sm.hist[i] = 0;
    sync();
    // warp-aggregated histogram: lanes with the same digit add once
    for (int base = 0; base < M; base += kSelThreads) {
      const int i = base + tid;
      uint32_t bin = 0xFFFFFFFFu;
      if (i < M) {
        const uint32_t k = ord_key(s_sc[i]);
        if ((k & pmask) == prefix) bin = (k >> shift) & 255u;
      }
      const unsigned int peers = __match_any_sync(0xffffffffu, bin);
      if (bin != 0xFFFFFFFFu && lane == __ffs(peers) - 1)
        atomicAdd(&sm.hist[bin], (unsigned)__popc(peers));
    }
    sync();
    if (warp == 0) {
      // lane l owns bins 255-8l .. 248-8l (lane 0 the largest digits)
      unsigned int cnt[8], lsum_bins = 0;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        cnt[j] = sm.hist[255 - 8 * lane - j];
        lsum_bins += cnt[j];
      }
      unsigned int incl = lsum_bins;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const unsigned int t = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += t;
      }
      const unsigned int ballot = __ballot_sync(0xffffffffu, incl >= (unsigned)krem);
      const int L = __ffs(ballot) - 1;    // exists: the prefix class holds >= krem entries
      if (lane == L) {
        unsigned int running = incl - lsum_bins;
        unsigned int digit = 0, above = running;
        for (int j = 0; j < 8; ++j) {
          if (running + cnt[j] >= (unsigned)krem) {
            digit = 255 - 8 * lane - j;
            above = running;
            break;
          }
          running += cnt[j];
        }
        sm.sh_digit = digit;
        sm.sh_above = above;
      }
    }
    sync();
    prefix |= sm.sh_digit << shift;
    pmask |= 255u << shift;
    krem -= (int)sm.sh_above;
  }
  const uint32_t T = prefix;              // K_eff-th largest key; take krem entries equal to T

  // ---- collect the K_eff candidates ----------------------------------------
  if (tid == 0) sm.sh_cnt_gt = 0;
  sync();
  for (int base = 0; base < M; base += kSelThreads) {
    const int i = base + tid;
    uint32_t k = 0;
    const bool take = i < M && (k = ord_key(s_sc[i])) > T;
    const unsigned int bal = __ballot_sync(0xffffffffu, take);
    int slot0 = 0;
    if (lane == 0 && bal) slot0 = atomicAdd(&sm.sh_cnt_gt, __popc(bal));
    slot0 = __shfl_sync(0xffffffffu, slot0, 0);
    if (take) {
      const int slot = slot0 + __popc(bal & ((1u << lane) - 1u));
      sm.cand[slot] = ((unsigned long long)k << 32) | (0xFFFFFFFFu - (uint32_t)i);
    }
  }
  const int c_gt = K_eff - krem;
  {
    // entries equal to T: the krem with the smallest positions (ordered scan)
    const int chunk = (M + kSelThreads - 1) / kSelThreads;
    const int beg = min(M, tid * chunk), end = min(M, beg + chunk);
    int c = 0;
    for (int i = beg; i < end; ++i) c += ord_key(s_sc[i]) == T;
    int incl = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int t = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += t;
    }
    if (lane == 31) sm.warp_tot[warp] = incl;
    sync();
    int rank = incl - c;
    for (int w = 0; w < warp; ++w) rank += sm.warp_tot[w];
    for (int i = beg; i < end && rank < krem; ++i) {
      if (ord_key(s_sc[i]) == T) {
        sm.cand[c_gt + rank] = ((unsigned long long)T << 32) | (0xFFFFFFFFu - (uint32_t)i);
        ++rank;
      }
    }
  }
  sync();

  select_tail(a, n, key_off, s_sc, K_eff, K_eff, smax, sumexp, sm, tid, sync);
}

// select_tail for K_eff > kRankMax: the C (K_eff <= C <= FOVEA_MAX_K)
// candidates bucket-ordered, the cumulative mass over the first K_eff four
// contiguous entries per thread, and the outputs, the original indices of a
// thread's outputs requested together before any is written.
template <class Sync>
__device__ __forceinline__ void select_tail_large(const SelectArgs& a, int n, int key_off,
                                                   const float* s_sc, int K_eff, int C, float smax,
                                                   float sumexp, SelectSmem& sm, int tid, Sync sync) {
  static_assert(FOVEA_MAX_K <= 4 * kSelThreads, "four ordered entries per thread");
  const int lane = tid & 31, warp = tid >> 5;
  const int k_max = a.k_max;
  bucket_order(sm, C, tid, sync);           // ends with a barrier
  const unsigned long long* ordered = sm.cand;
  // ---- cumulative mass: thread tid holds ordered entries 4 tid .. 4 tid + 3
  constexpr int per = 4;
  float e[4];
  float run = 0.0f;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int t = per * tid + q;
    e[q] = q < per && t < K_eff
               ? expf(s_sc[0xFFFFFFFFu - (uint32_t)(ordered[t] & 0xFFFFFFFFull)] - smax)
               : 0.0f;
    run += e[q];
  }
  float incl = run;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const float u = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += u;
  }
  if (lane == 31) sm.warp_tot_f[warp] = incl;
  sync();
  float before = incl - run;
  for (int w = 0; w < warp; ++w) before += sm.warp_tot_f[w];
  int my_first = K_eff;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int t = per * tid + q;
    before += e[q];
    if (q < per && t < K_eff) {
      sm.cum[t] = before;
      if (my_first == K_eff && before / sumexp >= a.rho) my_first = t;
    }
  }
  my_first = __reduce_min_sync(0xffffffffu, my_first);
  if (lane == 0) sm.warp_first[warp] = my_first;
  sync();
  int first = K_eff;
  for (int w = 0; w < kSelWarps; ++w) first = min(first, sm.warp_first[w]);
  const int K = first < K_eff ? min(K_eff, max(a.k_min, first + 1)) : K_eff;
  const float denom = sm.cum[K - 1];                          // sum over I_n of exp(s - s_max)
  const long long out_row = (long long)n * k_max;
  int pu[4], oi[4];
  float wu[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const int u = tid + j * kSelThreads;
    pu[j] = 0;
    oi[j] = -1;
    wu[j] = 0.0f;
    if (u < K) {
      pu[j] = (int)(0xFFFFFFFFu - (uint32_t)(ordered[u] & 0xFFFFFFFFull));
      wu[j] = expf(s_sc[pu[j]] - smax) / denom;
      if (a.indices) oi[j] = a.orig_index[key_off + pu[j]];
    }
  }
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const int u = tid + j * kSelThreads;
    if (u < K) {
      const int row = key_off + pu[j];
      if (a.sel_pos) a.sel_pos[out_row + u] = row;
      if (a.sel_w) a.sel_w[out_row + u] = wu[j];
      put_alpha(a, n, pu[j], wu[j]);
      if (a.loc_pos) {
        a.loc_pos[u] = row;
        a.loc_w[u] = wu[j];
      }
      if (a.indices) a.indices[out_row + u] = oi[j];
    } else if (u < k_max && a.indices) {
      a.indices[out_row + u] = -1;
    }
  }
  if (tid == 0) {
    if (a.sel_cnt) a.sel_cnt[n] = K;
    if (a.loc_cnt) *a.loc_cnt = K;
    if (a.counts) a.counts[n] = K;
  }
}

// K_eff <= kRankMax: ranking of the C (>= K_eff) candidates in sm.cand by (score desc,
// position asc), which puts the top K_eff in order in sm.sorted; then the
// cumulative mass, one ordered entry per thread (K_eff <= kRankMax), the
// count K and the outputs of draft state n.
template <class Sync>
__device__ __forceinline__ void select_tail(const SelectArgs& a, int n, int key_off,
                                            const float* s_sc, int K_eff, int C, float smax,
                                            float sumexp, SelectSmem& sm, int tid, Sync sync) {
  if constexpr (Sync::kLarge) {               // otherwise the launcher keeps K_max <= kRankMax
    if (K_eff > kRankMax) {
      select_tail_large(a, n, key_off, s_sc, K_eff, C, smax, sumexp, sm, tid, sync);
      return;
    }
  }
  const int lane = tid & 31, warp = tid >> 5;
  const int k_max = a.k_max;
  // ---- rank the candidates: rank = #larger (keys are distinct) -------------
  for (int c = tid; c < C; c += kSelThreads) {
    const unsigned long long me = sm.cand[c];
    int r0 = 0, r1 = 0, r2 = 0, r3 = 0;
    int j = 0;
    for (; j + 3 < C; j += 4) {
      r0 += sm.cand[j] > me;
      r1 += sm.cand[j + 1] > me;
      r2 += sm.cand[j + 2] > me;
      r3 += sm.cand[j + 3] > me;
    }
    for (; j < C; ++j) r0 += sm.cand[j] > me;
    const int r = (r0 + r1) + (r2 + r3);
    if (r < K_eff) sm.sorted[r] = me;
  }
  sync();                                                     // (4)
  // ---- cumulative mass, one ordered entry per thread -----------------------
  const int t = tid;
  float e = 0.0f;
  int pos = 0;
  if (t < K_eff) {
    pos = (int)(0xFFFFFFFFu - (uint32_t)(sm.sorted[t] & 0xFFFFFFFFull));
    e = expf(s_sc[pos] - smax);
  }
  float incl = e;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const float u = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += u;
  }
  if (lane == 31) sm.warp_tot_f[warp] = incl;
  sync();                                                     // (5)
  float before = 0.0f;
  for (int w = 0; w < warp; ++w) before += sm.warp_tot_f[w];
  const float cum = before + incl;
  if (t < K_eff) sm.cum[t] = cum;
  {
    const unsigned int bal = __ballot_sync(0xffffffffu, t < K_eff && cum / sumexp >= a.rho);
    if (lane == 0) sm.warp_first[warp] = bal ? warp * 32 + __ffs(bal) - 1 : K_eff;
  }
  sync();                                                     // (6)
  int first = K_eff;
  for (int w = 0; w < kSelWarps; ++w) first = min(first, sm.warp_first[w]);
  const int K = first < K_eff ? min(K_eff, max(a.k_min, first + 1)) : K_eff;
  const float denom = sm.cum[K - 1];                          // sum over I_n of exp(s - s_max)
  const long long out_row = (long long)n * k_max;
  for (int u = tid; u < k_max; u += kSelThreads) {
    if (u < K) {
      const int pu = u == t ? pos : (int)(0xFFFFFFFFu - (uint32_t)(sm.sorted[u] & 0xFFFFFFFFull));
      const float eu = u == t ? e : expf(s_sc[pu] - smax);
      const int row = key_off + pu;
      if (a.sel_pos) a.sel_pos[out_row + u] = row;
      if (a.sel_w) a.sel_w[out_row + u] = eu / denom;
      put_alpha(a, n, pu, eu / denom);
      if (a.loc_pos) {
        a.loc_pos[u] = row;
        a.loc_w[u] = eu / denom;
      }
      if (a.indices) a.indices[out_row + u] = a.orig_index[row];
    } else if (a.indices) {
      a.indices[out_row + u] = -1;
    }
  }
  if (tid == 0) {
    if (a.sel_cnt) a.sel_cnt[n] = K;
    if (a.loc_cnt) *a.loc_cnt = K;
    if (a.counts) a.counts[n] = K;
  }
}

// Fast path for rows of at most kFastMaxM entries (any K_eff <= FOVEA_MAX_K),
// with six group barriers and short dependency chains between them: the
// threads keep their scores in registers; (1) the maximum and the minimum
// score; (2) the softmax denominator (independent exponentials, summed in a
// fixed tree) and a 256-bin histogram of s_max - s over [0, s_max - s_min],
// which gives the bin b* holding the K_eff-th largest score (the bin index is
// monotone in the score, so the top K_eff entries all lie in bins <= b*);
// (3) the entries of bins <= b* are gathered (one shared-memory atomic per
// warp) and ordered among themselves by (score desc, position asc), which
// puts the top K_eff in order; the mass scan follows (select_tail).  Returns false, having written nothing, when the candidates
// exceed kFastMaxCand; the caller then runs the radix path.
constexpr int kFastMaxM = 2048;                   // 8 scores per thread
constexpr int kFastMaxCand = FOVEA_MAX_K;         // candidates ranked directly

template <class Sync>
__device__ bool select_fast(const SelectArgs& a, int n, int M, int key_off, const float* s_sc,
                            SelectSmem& sm, int tid, Sync sync) {
  constexpr int PT = kFastMaxM / kSelThreads;
  static_assert(PT == 8, "the denominator tree below sums eight terms per thread");
  const int lane = tid & 31, warp = tid >> 5;
  const int k_max = a.k_max;
  const int K_eff = min(k_max, M);
  float v[PT];
  float lmax = -INFINITY, lmin = INFINITY;
#pragma unroll
  for (int j = 0; j < PT; ++j) {
    const int i = tid + j * kSelThreads;
    v[j] = i < M ? s_sc[i] : -INFINITY;
    if (i < M) {
      lmax = fmaxf(lmax, v[j]);
      lmin = fminf(lmin, v[j]);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    lmax = fmaxf(lmax, __shfl_xor_sync(0xffffffffu, lmax, o));
    lmin = fminf(lmin, __shfl_xor_sync(0xffffffffu, lmin, o));
  }
  for (int i = tid; i < 256; i += kSelThreads) sm.hist[i] = 0;
  if (lane == 0) {
    sm.red_m[warp] = lmax;
    sm.red_lo[warp] = lmin;
  }
  if (tid == 0) sm.sh_cnt_gt = 0;
  sync();                                                     // (1)
  float smax = sm.red_m[0], smin = sm.red_lo[0];
#pragma unroll
  for (int w = 1; w < kSelWarps; ++w) {
    smax = fmaxf(smax, sm.red_m[w]);
    smin = fminf(smin, sm.red_lo[w]);
  }
  // ---- softmax denominator and histogram of the distance to the maximum ----
  const float range = smax - smin;
  const float inv_w = range > 0.0f ? 255.0f / range : 0.0f;
  float ex[PT];
  int bin[PT];
#pragma unroll
  for (int j = 0; j < PT; ++j) {
    const int i = tid + j * kSelThreads;
    ex[j] = i < M ? expf(v[j] - smax) : 0.0f;
    bin[j] = 256;
    if (i < M) {
      const int b = (int)((smax - v[j]) * inv_w);
      bin[j] = b < 0 ? 0 : (b > 255 ? 255 : b);
      atomicAdd(&sm.hist[bin[j]], 1u);
    }
  }
  float lsum = ((ex[0] + ex[1]) + (ex[2] + ex[3])) + ((ex[4] + ex[5]) + (ex[6] + ex[7]));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) lsum += __shfl_xor_sync(0xffffffffu, lsum, o);
  if (lane == 0) sm.red_s[warp] = lsum;
  sync();                                                     // (2)
  float sumexp = sm.red_s[0];
#pragma unroll
  for (int w = 1; w < kSelWarps; ++w) sumexp += sm.red_s[w];
  // every warp finds b* itself: lane l owns bins 8l .. 8l + 7
  int bstar;
  {
    unsigned int cnt[8], tot = 0;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      cnt[j] = sm.hist[8 * lane + j];
      tot += cnt[j];
    }
    unsigned int incl = tot;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const unsigned int t = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += t;
    }
    const unsigned int ballot = __ballot_sync(0xffffffffu, incl >= (unsigned)K_eff);
    const int L = __ffs(ballot) - 1;      // exists: the bins hold M >= K_eff entries
    int bl = 0;
    if (lane == L) {
      unsigned int run = incl - tot;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        if (bl == 0 && run + cnt[j] >= (unsigned)K_eff) bl = 8 * lane + j + 1;
        run += cnt[j];
      }
    }
    bstar = __shfl_sync(0xffffffffu, bl, L) - 1;
  }
  // ---- candidates: the entries of bins <= b*, one atomic per warp ----------
  {
    unsigned int bal[PT];
    int wtot = 0;
#pragma unroll
    for (int j = 0; j < PT; ++j) {
      bal[j] = __ballot_sync(0xffffffffu, bin[j] <= bstar);
      wtot += __popc(bal[j]);
    }
    int slot = 0;
    if (lane == 0 && wtot > 0) slot = atomicAdd(&sm.sh_cnt_gt, wtot);
    slot = __shfl_sync(0xffffffffu, slot, 0);
    const unsigned int below = (1u << lane) - 1u;
#pragma unroll
    for (int j = 0; j < PT; ++j) {
      if (bin[j] <= bstar) {
        const int sj = slot + __popc(bal[j] & below);
        if (sj < kFastMaxCand)
          sm.cand[sj] = ((unsigned long long)ord_key(v[j]) << 32) |
                        (0xFFFFFFFFu - (uint32_t)(tid + j * kSelThreads));
      }
      slot += __popc(bal[j]);
    }
  }
  sync();                                                     // (3)
  const int C = sm.sh_cnt_gt;
  if (C > kFastMaxCand) return false;                         // uniform
  select_tail(a, n, key_off, s_sc, K_eff, C, smax, sumexp, sm, tid, sync);
  return true;
}

// Wide path: the fast path's steps for rows of more than kFastMaxM entries, the scores read from shared memory in strided passes
// instead of registers and the distance to the maximum binned into kWideBins
// bins (the histogram occupies sm.cum, which the mass scan only writes after
// it is dead): (1) maximum and minimum; (2) softmax denominator (each
// thread's terms in index order, then a fixed tree) and histogram; (3, 4) the
// bin b* holding the K_eff-th largest score by a block scan of the bins;
// (5) the entries of bins <= b* gathered as candidates.  Returns false,
// having written nothing, when they exceed kFastMaxCand.
constexpr int kWideBins = 1024;
static_assert(kWideBins <= FOVEA_MAX_K, "the histogram lives in SelectSmem::cum");
static_assert(kWideBins == 4 * kSelThreads, "four bins per thread in the scan");

template <class Sync>
__device__ bool select_wide(const SelectArgs& a, int n, int M, int key_off, const float* s_sc,
                            SelectSmem& sm, int tid, Sync sync) {
  const int lane = tid & 31, warp = tid >> 5;
  const int K_eff = min(a.k_max, M);
  unsigned int* hist = reinterpret_cast<unsigned int*>(sm.cum);
  float lmax = -INFINITY, lmin = INFINITY;
  for (int i = tid; i < M; i += kSelThreads) {
    const float v = s_sc[i];
    lmax = fmaxf(lmax, v);
    lmin = fminf(lmin, v);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    lmax = fmaxf(lmax, __shfl_xor_sync(0xffffffffu, lmax, o));
    lmin = fminf(lmin, __shfl_xor_sync(0xffffffffu, lmin, o));
  }
  for (int i = tid; i < kWideBins; i += kSelThreads) hist[i] = 0u;
  if (lane == 0) {
    sm.red_m[warp] = lmax;
    sm.red_lo[warp] = lmin;
  }
  if (tid == 0) sm.sh_cnt_gt = 0;
  sync();                                                     // (1)
  float smax = sm.red_m[0], smin = sm.red_lo[0];
#pragma unroll
  for (int w = 1; w < kSelWarps; ++w) {
    smax = fmaxf(smax, sm.red_m[w]);
    smin = fminf(smin, sm.red_lo[w]);
  }
  const float range = smax - smin;
  const float inv_w = range > 0.0f ? (float)(kWideBins - 1) / range : 0.0f;
  auto bin_of = [&](float v) {
    const int b = (int)((smax - v) * inv_w);
    return b < 0 ? 0 : (b > kWideBins - 1 ? kWideBins - 1 : b);
  };
  float lsum = 0.0f;
  for (int i = tid; i < M; i += kSelThreads) {
    const float v = s_sc[i];
    lsum += expf(v - smax);
    atomicAdd(&hist[bin_of(v)], 1u);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) lsum += __shfl_xor_sync(0xffffffffu, lsum, o);
  if (lane == 0) sm.red_s[warp] = lsum;
  sync();                                                     // (2)
  float sumexp = sm.red_s[0];
#pragma unroll
  for (int w = 1; w < kSelWarps; ++w) sumexp += sm.red_s[w];
  // thread tid owns bins 4 tid .. 4 tid + 3 (ascending distance)
  unsigned int cnt[4], tot = 0;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    cnt[j] = hist[4 * tid + j];
    tot += cnt[j];
  }
  unsigned int incl = tot;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned int t = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += t;
  }
  if (lane == 31) sm.warp_tot[warp] = (int)incl;
  sync();                                                     // (3)
  unsigned int run = incl - tot;
  for (int w = 0; w < warp; ++w) run += (unsigned int)sm.warp_tot[w];
  if (run < (unsigned)K_eff && run + tot >= (unsigned)K_eff) {   // exactly one thread
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      if (run < (unsigned)K_eff && run + cnt[j] >= (unsigned)K_eff) sm.sh_digit = 4 * tid + j;
      run += cnt[j];
    }
  }
  sync();                                                     // (4)
  const int bstar = (int)sm.sh_digit;
  for (int base = 0; base < M; base += kSelThreads) {
    const int i = base + tid;
    float v = 0.0f;
    const bool take = i < M && bin_of(v = s_sc[i]) <= bstar;
    const unsigned int bal = __ballot_sync(0xffffffffu, take);
    int slot = 0;
    if (lane == 0 && bal) slot = atomicAdd(&sm.sh_cnt_gt, __popc(bal));
    slot = __shfl_sync(0xffffffffu, slot, 0) + __popc(bal & ((1u << lane) - 1u));
    if (take && slot < kFastMaxCand)
      sm.cand[slot] = ((unsigned long long)ord_key(v) << 32) | (0xFFFFFFFFu - (uint32_t)i);
  }
  sync();                                                     // (5)
  const int C = sm.sh_cnt_gt;
  if (C > kFastMaxCand) return false;                         // uniform
  select_tail(a, n, key_off, s_sc, K_eff, C, smax, sumexp, sm, tid, sync);
  return true;
}

// Selection of draft state n from its staged scores (s_sc, M >= 1 entries,
// staged and visible to the group): the fast or wide path where it applies,
// else the radix path.
template <class Sync>
__device__ __forceinline__ void select_row(const SelectArgs& a, int n, int M, int key_off,
                                           const float* s_sc, SelectSmem& sm, int tid, Sync sync) {
  if (M <= kFastMaxM ? select_fast(a, n, M, key_off, s_sc, sm, tid, sync)
                     : select_wide(a, n, M, key_off, s_sc, sm, tid, sync))
    return;
  float lmax = -INFINITY, lsum = 0.0f;
  for (int i = tid; i < M; i += kSelThreads) combine_ms(lmax, lsum, s_sc[i], 1.0f);
  float smax, sumexp;
  select_stats(lmax, lsum, sm, tid, sync, smax, sumexp);
  select_finish(a, n, M, key_off, s_sc, smax, sumexp, sm, tid, sync);
}

// Outputs of a draft state whose sequence has no valid entry: K = 0.
__device__ __forceinline__ void select_empty(const SelectArgs& a, int n, int tid) {
  const long long out_row = (long long)n * a.k_max;
  for (int t = tid; t < a.k_max; t += kSelThreads)
    if (a.indices) a.indices[out_row + t] = -1;
  if (tid == 0) {
    if (a.sel_cnt) a.sel_cnt[n] = 0;
    if (a.loc_cnt) *a.loc_cnt = 0;
    if (a.counts) a.counts[n] = 0;
  }
}

}  // namespace fovea
