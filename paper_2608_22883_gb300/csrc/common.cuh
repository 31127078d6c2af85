// Shared device helpers and internal launch interfaces of libfovea.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "fovea.h"

namespace fovea {

// Sticky device error bits (workspace / memory error word).
enum : int { kErrDepth = 1, kErrTimeout = 2 };

// Bytes at the start of a step workspace: the sticky error word and reserved
// words (fovea_workspace_init zeroes them).
constexpr size_t kWsHeaderBytes = 4096;

// Limit of a bounded mbarrier wait inside the tensor-core kernels (ns).  A
// wait that gives up sets kErrTimeout; the kernel then waits for the work it
// has already issued (copies, MMAs) with fixed limits and unwinds.
constexpr unsigned long long kDefaultWaitLimitNs = 2000000000ull;
// Process-wide limit the GEMM launches pass to their kernels
// (fovea_debug_wait_limit; api.cu).
void set_wait_limit_ns(unsigned long long ns);
unsigned long long wait_limit_ns();

// Depth gate of a draft step: rows whose depth l_n (an invalid depth counts
// as 0, as in the query LN) exceeds l_max are not corrected.  depth == null:
// every row is corrected.
struct DepthGate {
  const int32_t* depth;
  int l_max, max_depth;
};
__device__ __forceinline__ bool row_gated(const DepthGate& g, int n) {
  if (g.depth == nullptr) return false;
  int l = g.depth[n];
  if (l < 0 || l > g.max_depth) l = 0;
  return l > g.l_max;
}

// ---------------------------------------------------------------------------
// Scalar conversions
// ---------------------------------------------------------------------------
__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 x) { return __bfloat162float(x); }

template <class T> __device__ __forceinline__ T from_f32(float x);
template <> __device__ __forceinline__ float from_f32<float>(float x) { return x; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float x) {
  return __float2bfloat16_rn(x);
}

// Logistic sigmoid with the hardware exponential and a correctly rounded
// reciprocal (a few fp32 ulps from the exact value, far below the bf16
// rounding of the activations and the gate's tolerance; exp(-z) = inf for
// z < -88 gives exactly 0, as the zero-gate reading needs).  The activation
// epilogues evaluate it per element, where the full-precision expf and
// division dominated their time.
__device__ __forceinline__ float sigmoidf_(float z) { return __frcp_rn(1.0f + __expf(-z)); }

// Programmatic dependent launch: kernels of the step are launched so that a
// kernel may start while its predecessor finishes.  pdl_wait() blocks until
// the predecessor grid has completed and its writes are visible; a kernel
// calls it before it reads anything the predecessor wrote and before it
// writes anything.  pdl_trigger() lets the successor begin its own prologue.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// 16-byte asynchronous global -> shared copy (both addresses 16-byte
// aligned); cp_async_wait_all() waits for the calling thread's copies.
__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(
                   static_cast<uint32_t>(__cvta_generic_to_shared(smem))),
               "l"(gmem)
               : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;" ::: "memory"); }

// ---------------------------------------------------------------------------
// Reductions (fixed order, so results are run-to-run deterministic)
// ---------------------------------------------------------------------------
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// Block-wide sum / max; `scratch` holds >= 32 floats.  Every thread returns
// the result.  Contains __syncthreads().
__device__ __forceinline__ float block_sum(float v, float* scratch) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  v = warp_sum(v);
  __syncthreads();
  if (lane == 0) scratch[warp] = v;
  __syncthreads();
  float t = lane < nw ? scratch[lane] : 0.0f;
  return warp_sum(t);
}
__device__ __forceinline__ float block_max(float v, float* scratch) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  v = warp_max(v);
  __syncthreads();
  if (lane == 0) scratch[warp] = v;
  __syncthreads();
  float t = lane < nw ? scratch[lane] : -INFINITY;
  return warp_max(t);
}

// ---------------------------------------------------------------------------
// Per-call tables passed by value as kernel parameters
// ---------------------------------------------------------------------------

// One independent sub-problem of a GEMM C = A . B^T: output rows are B rows
// (draft states / tokens), output columns are A rows (features / keys).
struct GemmGroup {
  int a_row0;        // first A row of this group
  int m;             // A rows (output columns) in this group
  int b_row0;        // first B row of this group
  int n;             // B rows (output rows) in this group
  long long c_off;   // output element offset (grouped epilogues)
};

enum EpiKind : int {
  kEpiStore = 0,      // out{0,1}[row * ldc + col] = T(acc), columns split at epi_split
  kEpiScores = 1,     // out0 (fp32)[c_off + n * m + col] = acc * scale * row_scale[row]
  kEpiBiasSilu = 2,   // out0[row * ldc + col] = T(silu(acc + bias{0,1}[col]))
  kEpiBiasF32 = 3,    // out0 (fp32)[row * ldc + col] = acc + bias0[col]
  kEpiStoreHiLo = 4,  // out0 = T(acc), out1 = T(acc - out0): acc carried as two stored values
  kEpiStoreKeys = 5,  // kEpiStore, and columns < epi_split whose acc lies near a bf16
                      // rounding midpoint are listed for an exact recomputation
  kEpiQueryH = 6,     // columns < epi_split as kEpiStoreHiLo; columns >= epi_split:
                      // out2 (fp32)[row * ldc2 + col - epi_split] = acc
  kEpiScoresFolded = 7,  // kEpiScores with one row operand (x_h) against the folded
                         // keys, a hi / lo pair of feature tiles (f_lo_kb), for columns
                         // < epi_split (row stride min(m, epi_split)); columns >=
                         // epi_split: out2 (fp32)[row * ldc2 + col - epi_split] = acc
  kEpiAct = 8,           // the first fusion layer from dense selection weights: the row
                         // operand is the weights' hi / lo pair (B0, B1, both multiplied by
                         // the same feature tile); out0[row * ldc + col] =
                         // T(silu(acc + add_in[row * ldc2 + col] + bias{0,1}[col]))
  kEpiLogits = 9,        // the draft logits: out2 (fp32)[row * ldc2 + col] = acc, and per row
                         // the cand_k largest of the CTA's columns as 64-bit keys (logit order
                         // key << 32 | ~column) into cand[row * cand_ld + slot * cand_k + r],
                         // slot = feature tile * splits + rank, r = 0, 1, ... in descending
                         // key order (zeros last: fewer columns than cand_k)
};

struct KeyFix {       // one listed key element: memory row, feature
  int row, col;
};

struct GemmArgs {
  int k_total;        // contraction length (multiple of 64)
  int a_split;        // A rows >= a_split come from A1 (row - a_split)
  int a_split2;       // tensor-core path: A rows >= a_split2 come from A2 (row - a_split2)
  int r_by_part;      // tensor-core path: output columns from A1 / A2 read B1 at every k
  int b_split;        // contraction index >= b_split comes from B1 (k - b_split)
  int dual_b;         // tensor-core scores: B0 and B1 are the hi / lo parts of one
                      // operand, both multiplied by the same A tile
  int f_lo_kb;        // tensor-core folded scores: the feature operand A0 holds the
                      // hi / lo parts of the folded keys in each row, lo starting
                      // f_lo_kb k-blocks after hi (0: one part)
  // raw operands (SIMT path; the tensor-core path uses tensor maps)
  const void* A0; const void* A1; long long lda0, lda1;
  const void* B0; const void* B1; long long ldb0, ldb1;
  // epilogue
  int epi_split;
  void* out0; void* out1; long long ldc;
  void* out2; long long ldc2;                      // kEpiQueryH
  const void* bias0; const void* bias1;
  const float* row_scale; float scale;
  KeyFix* fix_list; int* fix_count; int fix_cap;   // kEpiStoreKeys
  int splits;         // tensor-core path: CTAs of a cluster sharing one output tile (split K)
  int stages;         // tensor-core path: depth of the shared-memory ring
  int tx_bytes;       // tensor-core path: bytes one ring stage receives (row box + feature tile)
  int kps;            // tensor-core path: k-blocks of 64 per ring stage
  int rbox;           // tensor-core path: rows of a row-operand tile (64 or 128)
  int region;         // tensor-core path: bytes of the ring / partial-tile staging region
  const float* add_in;          // kEpiAct: fp32 term added before the activation
  unsigned long long* cand;     // kEpiLogits: per-row candidate keys
  long long cand_ld;
  int cand_k;
  unsigned long long wait_ns;   // tensor-core path: limit of a bounded mbarrier wait
  int* err;
  // tensor-core path: byte ranges whose share each CTA prefetches into L2 once
  // it has requested its own operands (data a later kernel of the step reads)
  int n_prefetch;
  const void* pf_ptr[4];
  long long pf_bytes[4];
  int ngroups;
  GemmGroup groups[FOVEA_MAX_SEQ];
};

// Per-sequence view of one retrieve_fuse call.
struct SeqTable {
  int B;
  int row_start[FOVEA_MAX_SEQ + 1];
  int key_off[FOVEA_MAX_SEQ];
  int m[FOVEA_MAX_SEQ];
  long long score_off[FOVEA_MAX_SEQ];
};

__device__ __forceinline__ int seq_of_row(const SeqTable& t, int row) {
  int lo = 0, hi = t.B - 1;
  while (lo < hi) {                    // last b with row_start[b] <= row
    int mid = (lo + hi + 1) >> 1;
    if (t.row_start[mid] <= row) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// ---------------------------------------------------------------------------
// Host-side launch interfaces (defined in the kernel translation units)
// ---------------------------------------------------------------------------

// Launches `kern` on `s` with the programmatic-dependent-launch attribute.
template <class... KArgs, class... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

// Sets the message fovea_last_error() returns on this thread (api.cu).
fovea_status report_error(fovea_status st, const char* msg);

cudaError_t launch_ln_rows(int dtype, const void* x, const int32_t* src_row, int rows, int d,
                           const void* gamma, const void* beta, float eps, const void* E,
                           const int32_t* depth, int max_depth, int* err, void* out,
                           cudaStream_t s);
// LN of the draft hidden states plus the depth embedding (rowops.cu), fp32.
cudaError_t launch_ln_query(int dtype, const void* h, int rows, int d, const void* gamma,
                            const void* beta, float eps, const void* E, const int32_t* depth,
                            int max_depth, int* err, void* out, cudaStream_t s);
cudaError_t launch_count_valid(const uint8_t* mask, int B, int M_max, int32_t* counts,
                               cudaStream_t s);
cudaError_t launch_compact(const uint8_t* mask, int B, int M_max, const int32_t* key_off,
                           int32_t* orig_index, int32_t* src_row, cudaStream_t s);
// Selection alone (select.cu): counts, indices, and per row the selected
// compacted memory rows and weights (sel_pos, sel_w, sel_cnt; any may be
// null), and / or the weights as dense bf16 hi / lo rows over the row's
// sequence [N, alpha_ld], zero where not selected (alpha_hi null: none).
cudaError_t launch_select(const float* scores, const SeqTable& tab, int N, const int32_t* orig_index,
                          float rho, int k_min, int k_max, int max_m, const DepthGate& gate,
                          int32_t* counts, int32_t* indices, int32_t* sel_pos, float* sel_w,
                          int32_t* sel_cnt, cudaStream_t s, void* alpha_hi = nullptr,
                          void* alpha_lo = nullptr, int alpha_ld = 0);
cudaError_t launch_readout(int dtype, const void* U, const int32_t* sel_cnt, const int32_t* sel_pos,
                           const float* sel_w, int N, int k_max, int d, float* r_out, void* r_lo,
                           cudaStream_t s);
// Selection fused with the gathers that consume it (select.cu), for rows of
// at most 2048 valid entries and k_max <= 256 (select_readout_fits): the
// readout r (r_out fp32 and / or r_lo, either may be null; U unused when
// both are) and, when P is given, act = SiLU(Gh + sum_t alpha_t P[pi(t)] +
// [b_f1 ; b_g1]) over 2H columns.  p_prefetch_bytes: the first bytes of P the
// CTAs prefetch into L2 before waiting for the scores (0: none).
bool select_readout_fits(int max_m, int k_max);
cudaError_t launch_select_gather(int dtype, const float* scores, const SeqTable& tab, int N,
                                 const int32_t* orig_index, float rho, int k_min, int k_max,
                                 int max_m, const DepthGate& gate, int32_t* counts,
                                 int32_t* indices, const void* U, int d,
                                 float* r_out, void* r_lo, const void* P, int H, const float* Gh,
                                 const void* b_f1, const void* b_g1, void* act, int* err,
                                 cudaStream_t s, long long p_prefetch_bytes = 0);
// Exact rounding of listed key elements: k = sum_l x[row, l] W[col, l]
// evaluated in double-float, rounded once to bf16.  list == nullptr refines
// every element of the [rows, d] key matrix.
// out[c * rows + r] = in[r * cols + c] for a bf16 [rows, cols] matrix, rows
// and cols multiples of 32 (the query folding's W_Q^T, once per memory build).
cudaError_t launch_transpose_bf16(const void* in, int rows, int cols, void* out, cudaStream_t s);

// Images of a memory: first entry and valid count of each (kernel parameter).
struct ImageTable {
  int B;
  int off[FOVEA_MAX_SEQ];
  int m[FOVEA_MAX_SEQ];
};
// out [B, C, ld]: image b's [m_b, C] rows of `in` (from row off_b) transposed,
// zero-padded to ld entries (C and ld multiples of 32).
cudaError_t launch_transpose_images(const void* in, int C, int ld, const ImageTable& tab,
                                    void* out, cudaStream_t s);

// Per row n: the k <= FOVEA_MAX_KC largest of the candidate keys
// cand[n * slots * k .. + slots * k) (logit order key << 32 | ~index) in
// descending order, as token indices and logits.
cudaError_t launch_merge_candidates(const unsigned long long* cand, int N, int slots, int k,
                                    int32_t* top_idx, float* top_val, cudaStream_t s);
// Candidate slots per row the LM-head GEMM writes for this shape (its feature
// tiles times its split-K factor).
int lm_head_slots(int vocab, int d_model, int N);

cudaError_t launch_refine_keys(const void* xv, const void* W, int d, const KeyFix* list,
                               const int* count, int cap, int rows, void* K, cudaStream_t s);
// Rows past the depth gate: h_out = h and gate 0.
cudaError_t launch_finalize(int dtype, const void* h, const float* c, const void* act, int H, int d,
                            const void* w_g2, const void* b_g2, const void* rms_gamma, float eps,
                            int N, const DepthGate& gate, void* h_out, float* gate_out,
                            cudaStream_t s);

// GEMM C = A . B^T with a chosen epilogue.  `tc` selects the tcgen05 path
// (bf16 only); otherwise the SIMT path (fp32 and bf16).
// max_m / max_n bound the per-group extents (grid size).
cudaError_t launch_gemm_simt(int dtype, int epi, const GemmArgs& a, int max_m, int max_n,
                             cudaStream_t s);

struct TmaOperand {     // a row-major [rows, cols] bf16 matrix with a row stride
  const void* base;
  long long rows, cols, ld;   // ld in elements
};
// Tile plan of a tensor-core GEMM: feature tile width, split-K factor and
// the fp32 scratch (partial tiles) that split needs.
struct GemmPlan {
  int bn, splits, stages;
  long long partial_floats;   // global fp32 scratch the launch needs (0: none)
  long long tiles;            // output tiles
  int rbox;                   // rows of a row-operand load (64 or 128)
  int region;                 // bytes of the ring / partial-tile staging region
  int kps;                    // k-blocks of 64 per ring stage
};
GemmPlan plan_gemm_tc(int epi, const GemmArgs& a, int max_m, int max_n);
// Tensor map of a row-major [rows, cols] bf16 matrix (row stride ld
// elements), 128-byte swizzle, box = 64 columns x box_rows rows.
bool encode_bf16_map(CUtensorMap* m, const void* base, long long rows, long long cols,
                     long long ld, int box_rows);
// A2 (optional): the feature operand of output columns >= a_split2.
cudaError_t launch_gemm_tc(int epi, const GemmArgs& a, const TmaOperand& A0, const TmaOperand& A1,
                           const TmaOperand& B0, const TmaOperand& B1, int max_m, int max_n,
                           cudaStream_t s, const TmaOperand& A2 = TmaOperand{nullptr, 0, 0, 0});

}  // namespace fovea
