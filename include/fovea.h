/*
 * fovea.h - C ABI of the FOVEA visual-evidence path on one GB300 (sm_103a).
 *
 * The paper (FOVEA: Focused On-Demand Visual Evidence Adaptation, Sec. 3
 * "Method") defines, for a draft-tree node n with hidden state h_n and depth
 * l_n, the state-conditioned visual readout r_n = R_theta(h_n, l_n, V)
 * (Sec. "Problem formulation") and the corrected scoring representation
 * h_hat_n = RMSNorm(h_n + g_n c_n) (Eq. hidden_correction).  This library
 * computes exactly that path:
 *
 *   fovea_build_memory   - the per-image visual memory M_img = {(k_i, u_i, m_i)},
 *                          k_i = W_K LN(v_i), u_i = W_U LN(v_i)
 *                          (Sec. "Image-specific visual memory").
 *   fovea_retrieve_fuse  - for a batch of draft states: the query
 *                          q_n = W_Q(LN(h_n) + E_dep[l_n]), scores
 *                          s_{n,i} = q_n k_i / sqrt(d_k) over the valid entries,
 *                          the global softmax, the cumulative-mass cardinality
 *                          K_{r,n} (Sec. "State-conditioned top-K_{r,n} visual
 *                          evidence retrieval"), the renormalised readout r_n,
 *                          and the gated residual correction (Sec.
 *                          "Cache-friendly hidden-vector correction"; appendix
 *                          "Visual correction module").
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - All tensors are dense, row-major, contiguous, 16-byte aligned DEVICE
 *   pointers unless a parameter says "host".  Element type is given by
 *   fovea_params.dtype for weights and activations (bf16 or fp32); indices
 *   are int32; the optional readout and gate outputs are fp32.
 * - The caller owns every pointer it passes (weights, inputs, outputs,
 *   workspace).  The library only borrows them for the duration of the
 *   enqueue: kernels read them later, on the given stream, so they must stay
 *   valid until the stream reaches that point.
 * - The library owns fovea_memory handles (device buffers allocated by
 *   fovea_build_memory, released by fovea_memory_destroy).
 * - Work is enqueued on `stream` (a cudaStream_t; NULL = legacy default
 *   stream) of the current device.  fovea_retrieve_fuse never synchronises
 *   the host and never allocates.
 * - Every argument check happens before the first launch; a bad argument
 *   returns FOVEA_ERR_INVALID_ARG (or FOVEA_ERR_UNSUPPORTED for a legal value
 *   outside this build's limits) and enqueues nothing.  A CUDA runtime failure
 *   returns FOVEA_ERR_CUDA.  fovea_last_error() gives the message.  Nothing
 *   aborts the process.
 * - Conditions only the device can see (a depth outside [0, D], a bounded
 *   wait that gave up) set a sticky error word in the workspace; read and
 *   clear it with fovea_sync_errors().
 *
 * Dimensions: d = d_model = d_k = d_u = d_h = d_v (the appendix sets
 * d_k = d_u = d_h; the projector maps visual tokens to the LM width),
 * H = hidden width of the correction and gate networks (512 in the paper),
 * D = maximum tree depth (6 in the paper; E_dep has D + 1 rows).
 */
#ifndef FOVEA_H_
#define FOVEA_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#if defined(__GNUC__)
#define FOVEA_API __attribute__((visibility("default")))
#else
#define FOVEA_API
#endif

typedef enum {
  FOVEA_OK = 0,
  FOVEA_ERR_INVALID_ARG = 1,   /* null pointer, bad size, rho/k range, bad depth (device) */
  FOVEA_ERR_UNSUPPORTED = 2,   /* legal but beyond this build's limits (see FOVEA_MAX_*) */
  FOVEA_ERR_CUDA = 3,          /* a CUDA runtime call failed */
  FOVEA_ERR_OOM = 4,           /* device allocation failed (fovea_build_memory only) */
  FOVEA_ERR_TIMEOUT = 5        /* a bounded device-side wait gave up */
} fovea_status;

typedef enum { FOVEA_BF16 = 0, FOVEA_FP32 = 1 } fovea_dtype;

/* Limits of this build. */
#define FOVEA_MAX_D 8192          /* d_model, also a multiple of 64 */
#define FOVEA_MAX_H 4096          /* hidden width H, a multiple of 128 */
#define FOVEA_MAX_K 1024          /* cap K_max */
#define FOVEA_MAX_ENTRIES 32768   /* valid entries per image */
#define FOVEA_MAX_SEQ 512         /* sequences (images) per call */
#define FOVEA_MAX_KC 32           /* candidate width of fovea_lm_head_topk */

/* Opaque, library-owned, device-resident visual memory of B images. */
typedef struct fovea_memory fovea_memory;

/*
 * Weights theta.  All pointers are device pointers of element type `dtype`,
 * row-major [out, in] for linear maps (y = W x), borrowed per call.
 *   ln_v_gamma, ln_v_beta [d]      LN of visual tokens (Eq. of M_img)
 *   W_K, W_U              [d, d]   key / value projections (Eq. of M_img)
 *   ln_h_gamma, ln_h_beta [d]      LN of draft hidden states (query equation)
 *   E_dep                 [D+1, d] depth embedding
 *   W_Q                   [d, d]   query projection
 *   W_f1 [H, 2d], b_f1 [H], W_f2 [d, H], b_f2 [d]   correction net f_theta
 *   W_g1 [H, 2d], b_g1 [H], w_g2 [H],    b_g2 [1]   gate net g_theta
 *   rms_gamma             [d]      RMSNorm weight (Eq. hidden_correction)
 * f and g read the concatenation [h_n ; r_n] (h first), as printed.
 */
typedef struct fovea_params {
  int d_model;       /* d: multiple of 64, <= FOVEA_MAX_D */
  int mlp_hidden;    /* H: multiple of 128, <= FOVEA_MAX_H (paper: 512) */
  int max_depth;     /* D >= 0 (paper: 6) */
  int dtype;         /* fovea_dtype of every weight and activation */
  float ln_eps;      /* LN epsilon (1e-5 in the workloads here) */
  float rms_eps;     /* RMSNorm epsilon (1e-6 in the workloads here) */
  const void *ln_v_gamma, *ln_v_beta, *W_K, *W_U;
  const void *ln_h_gamma, *ln_h_beta, *E_dep, *W_Q;
  const void *W_f1, *b_f1, *W_f2, *b_f2;
  const void *W_g1, *b_g1, *w_g2, *b_g2;
  const void *rms_gamma;
} fovea_params;

/*
 * Build the visual memory of B images (Sec. "Image-specific visual memory";
 * Algorithm 1, memory construction before the decoding loop):
 * for every valid position i of image b, k_i = W_K LN(v_i), u_i = W_U LN(v_i).
 *   v     [B, M_max, d] device, dtype: projected visual tokens
 *   mask  [B, M_max] device uint8 (1 = valid, 0 = padding), or NULL (all valid)
 * Valid entries are compacted in ascending position; the handle keeps each
 * entry's original position, which is what fovea_retrieve_fuse reports as an
 * index.  An image with no valid entry is allowed (its rows select nothing).
 * bf16 with W_f1 and W_g1 given (and a valid mlp_hidden): the handle also
 * keeps each value through the r-half of the first fusion layer,
 * p_i = [W_f1 ; W_g1][:, d:2d] u_i ([2H], bf16).  The fusion of Eq.
 * hidden_correction is linear in r_n before its SiLU, so a draft step can
 * form [W_f1 ; W_g1][:, d:2d] r_n = sum_t alpha_t p_{pi(t)} from 2H-wide rows
 * instead of d-wide ones.  fovea_retrieve_fuse uses them only when it is
 * given the same W_f1, W_g1 pointers and mlp_hidden; weights changed in
 * place after the build need a new memory (as W_K, W_U already do).
 * bf16 with W_Q given: the handle also keeps the folded keys
 * kappa_i = W_Q^T k_i (query folding).  Since
 * q_n . k_i = (W_Q x_n) . k_i = x_n . kappa_i with x_n = LN(h_n) + E_dep[l_n],
 * a draft step given the same W_Q pointer scores x_n against kappa_i and
 * never streams W_Q.  kappa_i is not rounded to bf16: it is kept as a pair of
 * bf16 values kappa_hi + kappa_lo (about 16 significant bits, the same
 * precision the unfolded scores give q = W_Q x_n), so both score forms
 * follow the paper's q . k to within fp32 accumulation.  Pass W_Q = NULL here
 * to keep the unfolded scores.
 * This call allocates the handle's device buffers and synchronises `stream`
 * once (to size them).  B in [1, FOVEA_MAX_SEQ], M_max in [0, ...],
 * per-image valid count <= FOVEA_MAX_ENTRIES.
 * Errors: INVALID_ARG, UNSUPPORTED, OOM, CUDA; *out is untouched on error.
 */
FOVEA_API fovea_status fovea_build_memory(const fovea_params* p, const void* v,
                                          const uint8_t* mask, int B, int M_max,
                                          void* stream, fovea_memory** out);

/* Release a memory handle (NULL is ignored).  The caller must make sure no
 * enqueued work still reads it (e.g. synchronise the stream first). */
FOVEA_API void fovea_memory_destroy(fovea_memory* mem);

/* Shape of a memory: number of images, total valid entries, and (if
 * valid_counts is non-NULL) the valid count of each image into a HOST array
 * of B ints. */
FOVEA_API fovea_status fovea_memory_info(const fovea_memory* mem, int* B,
                                         int* total_valid, int32_t* valid_counts);

/* Device views of the memory, owned by the handle: keys and values
 * [total_valid, d] (dtype), the original position of each entry
 * [total_valid] int32, and (if non-NULL) the HOST array offsets[B + 1] of
 * each image's first entry.  Any output pointer may be NULL. */
FOVEA_API fovea_status fovea_memory_tensors(const fovea_memory* mem, const void** keys,
                                            const void** values, const int32_t** index,
                                            int64_t* offsets);

/* The folded keys kappa_i = W_Q^T k_i as [total_valid, 2d] bf16 (row i holds
 * kappa_hi then kappa_lo = bf16(kappa - kappa_hi); device, owned by the
 * handle) when the memory holds them for this W_Q pointer, else NULL in
 * *folded: a step given this W_Q scores against them. */
FOVEA_API fovea_status fovea_memory_folded_keys(const fovea_memory* mem, const void* W_Q,
                                                const void** folded);

/*
 * Bytes of workspace fovea_retrieve_fuse needs for this memory, these row
 * offsets (HOST array [B + 1]) and this cap.  The workspace is caller-owned
 * device memory (256-byte aligned) and must be initialised once with
 * fovea_workspace_init before its first use.
 */
FOVEA_API fovea_status fovea_workspace_size(const fovea_params* p, const fovea_memory* mem,
                                            const int32_t* row_offsets, int k_max,
                                            size_t* bytes);

/* Zero the workspace's header (the sticky error word and reserved words;
 * enqueued on `stream`).  One initialisation serves every later call;
 * fovea_sync_errors clears the header again after it reports an error. */
FOVEA_API fovea_status fovea_workspace_init(void* workspace, size_t bytes, void* stream);

/*
 * One draft step over N = row_offsets[B] draft states (Algorithm 1, the loop
 * body over nodes at enabled correction depths; retrieval equations and
 * Eq. hidden_correction).  Rows row_offsets[b] .. row_offsets[b+1]-1 query
 * image b of `mem`.
 *   h           [N, d] device, dtype: draft hidden states h_n
 *   depth       [N] device int32: tree depth l_n in [0, D] (checked on the
 *               device: a bad depth sets INVALID_ARG in the workspace error
 *               word and the row uses depth 0)
 *   row_offsets [B + 1] HOST int32: 0 = row_offsets[0] <= ... , B = mem's B
 *   row_scale   [N] device fp32 or NULL: multiplies the score scale
 *               1/sqrt(d_k) per row (NULL = 1, the paper's scores)
 *   rho         mass threshold, 0 < rho <= 1 (paper: 0.8)
 *   k_min,k_max 1 <= k_min <= k_max <= FOVEA_MAX_K (paper: 32, 256)
 *   l_max       depth gate (the experimental setup corrects nodes at depth
 *               <= 1): a row with l_n > l_max is not corrected: h_out = h,
 *               count 0, indices -1, readout 0, gate 0.  l_max >= D corrects
 *               every row (and reads no depth for the gate).  A depth outside
 *               [0, D] counts as 0 here, as in the query.
 * Outputs (device, caller-owned):
 *   h_out       [N, d] dtype: h_hat_n = RMSNorm(h_n + g_n c_n)   (required)
 *   counts      [N] int32: K_{r,n}                                (or NULL)
 *   indices     [N, k_max] int32: original positions pi_n(1..K) in descending
 *               score order (ties: smaller position first), -1 after K (or NULL)
 *   readout     [N, d] fp32: r_n                                   (or NULL)
 *   gate        [N] fp32: g_n                                      (or NULL)
 * Scores are s = (q . k) / sqrt(d) * row_scale; selection orders by s
 * descending, smaller original position first on ties; K_raw is the first k
 * with cumulative global-softmax mass >= rho (|V| if rounding never reaches
 * it); K = min(|V|, k_max, max(k_min, K_raw)); an image with no valid entry
 * gives K = 0 and r = 0.
 * bf16 path: LN(h) + E_dep, q and the SiLU activations are stored as bf16
 * (with folded keys for this W_Q, q is not formed: the scores are
 * (x_n . kappa_i) / sqrt(d) * row_scale, x_n the stored bf16 LN(h) + E_dep);
 * r enters the fusion as a bf16 vector, or (memory with projected values for
 * these weights, rows of <= 2048 entries, k_max <= 256) through the bf16
 * projected values p_i with the sum kept in fp32; accumulation is fp32
 * throughout.
 * Errors: INVALID_ARG, UNSUPPORTED (nothing enqueued), CUDA.
 */
FOVEA_API fovea_status fovea_retrieve_fuse(const fovea_params* p, const fovea_memory* mem,
                                           const void* h, const int32_t* depth,
                                           const int32_t* row_offsets, const float* row_scale,
                                           float rho, int k_min, int k_max, int l_max,
                                           void* h_out, int32_t* counts, int32_t* indices,
                                           float* readout, float* gate,
                                           void* workspace, size_t workspace_bytes,
                                           void* stream);

/*
 * fovea_retrieve_fuse without a workspace argument, for callers that cannot
 * allocate device memory where they run the draft step: code recorded into a
 * CUDA graph or running inside a runtime with a fixed, pre-planned memory
 * budget (where cudaMalloc is illegal or unavailable), and latency-critical
 * loops that must not take the implicit device synchronisation of
 * cudaMalloc / cudaFree.  The paper has no counterpart: this is an interface
 * convenience of this library.
 *
 * Arguments and outputs are those of fovea_retrieve_fuse.  The scratch is a
 * file-scope device array of FOVEA_NOALLOC_WORKSPACE_BYTES that every GPU
 * loading the library holds until the process exits; the call allocates
 * nothing (no cudaMalloc, cudaFree or allocating library routine).
 * - A call whose scratch need (fovea_workspace_size) exceeds the array returns
 *   FOVEA_ERR_UNSUPPORTED and enqueues nothing.
 * - The first call on a device looks up the array's device address
 *   (cudaGetSymbolAddress, with that device current); make that first call
 *   before any stream capture.
 * - Every call on a device shares the one array: calls that overlap on the GPU
 *   (other streams, other host threads) race and corrupt each other.  Each
 *   call clears the array's reserved header words, not its error word:
 *   device-side conditions (a bad depth, a bounded wait that gave up) stay
 *   in the error word until fovea_noalloc_sync_errors reads and clears it.
 *   This entry point does not report them itself.
 */
#define FOVEA_NOALLOC_WORKSPACE_BYTES (32u << 20)
FOVEA_API fovea_status fovea_retrieve_fuse_noalloc(const fovea_params* p, const fovea_memory* mem,
                                                   const void* h, const int32_t* depth,
                                                   const int32_t* row_offsets,
                                                   const float* row_scale, float rho, int k_min,
                                                   int k_max, int l_max, void* h_out,
                                                   int32_t* counts, int32_t* indices,
                                                   float* readout, float* gate, void* stream);
/* fovea_sync_errors for the static array of fovea_retrieve_fuse_noalloc on
 * the current device: synchronise `stream`, read and clear its error word
 * (FOVEA_OK, FOVEA_ERR_INVALID_ARG for a bad depth, FOVEA_ERR_TIMEOUT). */
FOVEA_API fovea_status fovea_noalloc_sync_errors(void* stream);

/*
 * Draft logits and tree-expansion candidates (Eq. hidden_correction,
 * z_n = W_LM h_hat_n; the experimental setup's candidate width K_c, 6 in
 * the paper): for every row of h_hat, the logits over the vocabulary and the
 * k_c largest of them in descending order, ties broken by the smaller token
 * index.
 *   W_LM      [vocab, d_model] device, dtype, row-major (16-byte aligned)
 *   h_hat     [N, d_model] device, dtype (e.g. fovea_retrieve_fuse's h_out)
 *   logits    [N, vocab] device fp32, caller-owned: z (written), or NULL
 *             when only the candidates are wanted (the 4 N vocab bytes of
 *             logits are then not written)
 *   top_idx   [N, k_c] device int32: token indices (written)
 *   top_val   [N, k_c] device fp32: their logits (or NULL)
 *   workspace device memory of fovea_lm_head_workspace_size bytes (256-byte
 *             aligned), its header initialised with fovea_workspace_init:
 *             the error word, then the candidates (the GEMM's epilogue keeps
 *             each row's k_c largest logits of every tile; a second kernel
 *             merges them)
 * bf16 only (fp32 returns UNSUPPORTED); 1 <= k_c <= FOVEA_MAX_KC <= vocab;
 * accumulation in fp32.  Enqueued on `stream`, no host synchronisation.
 * Enqueued on the stream of a draft step right after fovea_retrieve_fuse, the
 * LM-head GEMM starts streaming W_LM while the step's last kernel runs
 * (programmatic dependent launch): the logits follow the corrected states
 * without a host round trip.
 * Errors: INVALID_ARG, UNSUPPORTED (nothing enqueued), CUDA.
 */
FOVEA_API fovea_status fovea_lm_head_topk(const void* W_LM, int vocab, int d_model, int dtype,
                                          const void* h_hat, int N, int k_c, float* logits,
                                          int32_t* top_idx, float* top_val, void* workspace,
                                          size_t workspace_bytes, void* stream);
/* Workspace bytes of fovea_lm_head_topk for this shape.  Errors: INVALID_ARG. */
FOVEA_API fovea_status fovea_lm_head_workspace_size(int vocab, int d_model, int N, int k_c,
                                                    size_t* bytes);

/* Synchronise `stream`, read and clear the workspace's sticky error word.
 * Returns FOVEA_OK, FOVEA_ERR_INVALID_ARG (a depth outside [0, D] was seen)
 * or FOVEA_ERR_TIMEOUT (a bounded device wait gave up), or FOVEA_ERR_CUDA.
 * After an error the whole header is cleared, as fovea_workspace_init does,
 * so the workspace serves the next call. */
FOVEA_API fovea_status fovea_sync_errors(void* workspace, void* stream);

/* Limit of the bounded mbarrier waits in the tensor-core kernels launched
 * after this call (process-wide; 0 restores the default of about 2 s).  The
 * paper has no counterpart: it exists so that tests can make a wait give up
 * and check that the call reports FOVEA_ERR_TIMEOUT (through
 * fovea_sync_errors) and that the workspace serves the next call.  A wait
 * that gives up still waits, with fixed limits, for the copies and MMAs its
 * kernel issued before the kernel exits; the outputs of that call are
 * undefined. */
FOVEA_API fovea_status fovea_debug_wait_limit(unsigned long long limit_ns);

/* Message of the last non-OK status returned on this thread ("" if none). */
FOVEA_API const char* fovea_last_error(void);

/* Per-kernel timing with CUDA events recorded around every launch of this
 * library (off by default; for measurement only).  fovea_timing_enable(1)
 * clears the records and starts recording; fovea_timing_read synchronises the
 * recorded events and fills up to `capacity` entries of kernel name, total
 * milliseconds and launch count; it returns the number of distinct kernels.
 * Launches recorded while the stream is captured into a CUDA graph become
 * external event nodes of the graph: after each replay, fovea_timing_read
 * returns that replay's durations.  Keep timing enabled (do not call
 * fovea_timing_enable again) while such a graph is still replayed. */
FOVEA_API fovea_status fovea_timing_enable(int enable);
FOVEA_API int fovea_timing_read(const char** names, double* total_ms, int* launches,
                                int capacity);

/* Library ABI version (major * 100 + minor). */
FOVEA_API int fovea_version(void);

#ifdef __cplusplus
}
#endif

#endif /* FOVEA_H_ */
