// Plan, parameters and launcher of the persistent step kernel (step_fused.cu).
#pragma once
#include <algorithm>
#include <cstring>
#include <cmath>

#include "common.cuh"

namespace fovea {
namespace fused {

constexpr int kPhases = 4;
enum : int { kPhaseQuery = 0, kPhaseScore = 1, kPhaseFuse1 = 2, kPhaseFuse2 = 3 };
constexpr int kMaxSeq = 64;          // sequences (images) of one call on this path
constexpr int kNumMaps = 11;

// One GEMM phase C = R . F^T cut into units (group, row tile of 128, feature
// tile of bn, K split).  Units are numbered group by group, row tile, then
// feature tile, split fastest.
struct PhaseGemm {
  int bn;            // feature tile width (64 | 128 | 256; <= 128 for the scores)
  int splits;        // K splits per output tile
  int kb_total;      // contraction length in blocks of 64
  int r_split_kb;    // k-blocks >= r_split_kb read the row operand from rmap1
  int f_split;       // features >= f_split come from fmap1 (a multiple of bn)
  int dual;          // scores: the row stage holds q_hi and q_lo tiles (rmap0, rmap1)
  int rbox;          // rows per row-operand load (<= 128; the MMA's rows beyond it are unused)
  int fmap0, fmap1, rmap0, rmap1;   // tensor-map indices
  int wait_r0, wait_r1;             // grid barrier the row loads from rmap0 / rmap1 wait for
  int ngroups, units;
  int unit0[kMaxSeq + 1];           // first unit of each group
  int a_row0[kMaxSeq];              // first feature-operand row of each group
  int m[kMaxSeq];                   // features (output columns) per group
  int b_row0[kMaxSeq];              // first draft row of each group
  int n[kMaxSeq];                   // draft rows per group
  int ftiles[kMaxSeq];              // feature tiles per group
};

struct FusedMaps {
  CUtensorMap m[kNumMaps];
};

struct FusedArgs {
  PhaseGemm g[kPhases];
  int N, d, H, B, k_max, k_min, max_depth;
  float rho, scale, ln_eps, rms_eps;
  // inputs
  const __nv_bfloat16* h;
  const int32_t* depth;
  const float* row_scale;
  const __nv_bfloat16 *ln_gamma, *ln_beta, *E;
  const __nv_bfloat16* U;
  const int32_t* orig_index;
  const __nv_bfloat16 *b_f1, *b_g1, *b_f2, *w_g2, *b_g2, *rms_gamma;
  // per sequence
  int row_start[kMaxSeq + 1];
  int key_off[kMaxSeq];
  int mseq[kMaxSeq];
  int seq_group[kMaxSeq];           // group of the score phase, -1 when no rows or no keys
  // workspace
  __nv_bfloat16 *x, *q_hi, *q_lo, *r, *act;
  float* partials;
  int32_t* sel_pos;
  float* sel_w;
  int32_t* sel_cnt;
  int* err;
  int* sync;                        // [1..9] grid-barrier arrivals, [10] exit count, [11] abort
  // outputs
  __nv_bfloat16* h_out;
  int32_t* counts;
  int32_t* indices;
  float* readout;
  float* gate;
  // readout items: (sequence ro_seq[i], column slice of ro_w features)
  int ro_w, ro_rows, ro_items;
  int ro_seq[kMaxSeq];
  // L2 prefetch ranges
  int n_prefetch;
  const void* pf_ptr[6];
  long long pf_bytes[6];
};

}  // namespace fused

// Shape of one call, for planning.
struct FusedShape {
  bool bf16;
  int N, d, H, B, k_max;
  const int32_t* row_offsets;   // [B + 1] host
  const int32_t* m;             // [B] valid entries per sequence
};

struct FusedPlan {
  int G;                        // CTAs (one per SM)
  fused::PhaseGemm g[fused::kPhases];
  int seq_group[fused::kMaxSeq];
  int n_score_groups;
  int ro_w, ro_rows, ro_nseq;
  int ro_seq[fused::kMaxSeq];
  long long partial_floats;     // fp32 scratch of the partial tiles
};

// Everything one launch needs (device pointers unless noted).
struct FusedLaunch {
  int N, d, H, B, k_max, k_min, max_depth;
  float rho, ln_eps, rms_eps;
  const int32_t* row_offsets;   // host
  const int32_t* key_off;       // host, compacted row of each sequence's first entry
  const int32_t* m;             // host
  long long total_keys;
  bool prefetch_values;
  const void *h, *ln_gamma, *ln_beta, *E, *W_Q, *keys, *values, *W_f1, *W_g1, *W_f2;
  const void *b_f1, *b_g1, *b_f2, *w_g2, *b_g2, *rms_gamma;
  const int32_t* depth;
  const float* row_scale;
  const int32_t* orig_index;
  void *x, *q_hi, *q_lo, *r, *act;
  float* partials;
  int32_t* sel_pos;
  float* sel_w;
  int32_t* sel_cnt;
  int* err;
  int* sync;
  void* h_out;
  int32_t* counts;
  int32_t* indices;
  float* readout;
  float* gate;
};

// False when the call's shape is outside what the persistent kernel handles.
bool fused_plan(const FusedShape& sh, FusedPlan* out);
cudaError_t launch_fused_step(const FusedPlan& plan, const FusedLaunch& L, cudaStream_t s);

}  // namespace fovea
