// C ABI of libfovea (include/fovea.h): argument checks, the memory handle,
// the workspace layout, and the launch sequence of one draft step.
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <algorithm>
#include <mutex>
#include <string>
#include <vector>

#include <atomic>

#include "common.cuh"

using namespace fovea;

// ---------------------------------------------------------------------------
// Errors
// ---------------------------------------------------------------------------
static thread_local std::string g_last_error;

static fovea_status fail(fovea_status st, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return st;
}
namespace fovea {
// Records the message fovea_last_error() returns (for other translation units).
fovea_status report_error(fovea_status st, const char* msg) {
  g_last_error = msg;
  return st;
}
}  // namespace fovea

static fovea_status cuda_fail(cudaError_t e, const char* where) {
  return fail(FOVEA_ERR_CUDA, "%s: %s", where, cudaGetErrorString(e));
}
#define FOVEA_CUDA(call, where)                   \
  do {                                            \
    cudaError_t e_ = (call);                      \
    if (e_ != cudaSuccess) return cuda_fail(e_, where); \
  } while (0)

// ---------------------------------------------------------------------------
// Per-launch timing (CUDA events on the launching stream)
// ---------------------------------------------------------------------------
namespace {
struct TimingRec {
  const char* name;
  cudaEvent_t start, stop;
};
std::mutex g_tmu;
bool g_timing = false;
std::vector<TimingRec> g_recs;
std::vector<cudaEvent_t> g_free_events;

cudaEvent_t take_event() {
  if (!g_free_events.empty()) {
    cudaEvent_t e = g_free_events.back();
    g_free_events.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}

bool capturing(cudaStream_t s) {
  cudaStreamCaptureStatus st = cudaStreamCaptureStatusNone;
  cudaStreamIsCapturing(s, &st);
  return st != cudaStreamCaptureStatusNone;
}

// Records start/stop events around one launch when timing is enabled.  While
// the stream is being captured into a CUDA graph the records become external
// event nodes of the graph, re-recorded by every replay.
struct KernelTimer {
  const char* name;
  cudaStream_t s;
  bool on, graph;
  KernelTimer(const char* n, cudaStream_t st) : name(n), s(st), on(false), graph(false) {
    std::lock_guard<std::mutex> lk(g_tmu);
    if (!g_timing) return;
    graph = capturing(s);
    TimingRec r{name, take_event(), take_event()};
    if (graph) cudaEventRecordWithFlags(r.start, s, cudaEventRecordExternal);
    else cudaEventRecord(r.start, s);
    g_recs.push_back(r);
    on = true;
  }
  ~KernelTimer() {
    if (!on) return;
    std::lock_guard<std::mutex> lk(g_tmu);
    for (auto it = g_recs.rbegin(); it != g_recs.rend(); ++it)
      if (it->name == name) {
        if (graph) cudaEventRecordWithFlags(it->stop, s, cudaEventRecordExternal);
        else cudaEventRecord(it->stop, s);
        break;
      }
  }
};
}  // namespace

// ---------------------------------------------------------------------------
// Memory handle
// ---------------------------------------------------------------------------
struct fovea_memory {
  int device = 0;
  int B = 0, M_max = 0, d = 0, dtype = 0;
  int total = 0;
  std::vector<int32_t> counts;       // valid entries per image (host)
  std::vector<int64_t> offsets;      // first entry of each image, B + 1 (host)
  void* keys = nullptr;              // [total, d]
  void* values = nullptr;            // [total, d]
  int32_t* orig_index = nullptr;     // [total]
  int* err = nullptr;                // device error word
  int refined = 0;                   // key elements re-rounded exactly at build
  // bf16: the values projected through the r-half of the first fusion layer,
  // p_i = [W_f1 ; W_g1][:, d:2d] u_i  ([total, 2H]), and the weights they
  // were built with (a call with other W_f1 / W_g1 pointers or H does not
  // use them)
  void* proj = nullptr;
  // the projected values transposed per image, [B, 2H, proj_ld] with
  // proj_ld = max valid count rounded up to 64 (zero-padded): the feature
  // operand of the weighted-sum GEMM over dense selection weights
  void* projT = nullptr;
  int proj_ld = 0;
  const void* proj_wf1 = nullptr;
  const void* proj_wg1 = nullptr;
  int proj_h = 0;
  // bf16: the keys folded through the query projection, kappa_i = W_Q^T k_i,
  // as a hi / lo pair of bf16 values ([total, 2d]: row i holds kappa_hi then
  // kappa_lo = bf16(kappa - kappa_hi), about 16 significant bits), and the
  // W_Q they were built with: q . k_i = x . kappa_i, so a call with that W_Q
  // scores x = LN(h) + E_dep against them directly
  void* folded = nullptr;
  const void* fold_wq = nullptr;
};

static size_t esize(int dtype) { return dtype == FOVEA_BF16 ? 2 : 4; }
static bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
static size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

static fovea_status check_dims(const fovea_params* p) {
  if (p == nullptr) return fail(FOVEA_ERR_INVALID_ARG, "params is NULL");
  if (p->dtype != FOVEA_BF16 && p->dtype != FOVEA_FP32)
    return fail(FOVEA_ERR_INVALID_ARG, "dtype %d is neither FOVEA_BF16 nor FOVEA_FP32", p->dtype);
  if (p->d_model <= 0 || p->d_model % 64 != 0)
    return fail(FOVEA_ERR_INVALID_ARG, "d_model %d must be a positive multiple of 64", p->d_model);
  if (p->d_model > FOVEA_MAX_D)
    return fail(FOVEA_ERR_UNSUPPORTED, "d_model %d exceeds %d", p->d_model, FOVEA_MAX_D);
  if (!(p->ln_eps > 0.0f) || !(p->rms_eps > 0.0f))
    return fail(FOVEA_ERR_INVALID_ARG, "ln_eps and rms_eps must be > 0");
  return FOVEA_OK;
}

#define NEED_PTR(ptr, name)                                                             \
  do {                                                                                  \
    if ((ptr) == nullptr) return fail(FOVEA_ERR_INVALID_ARG, "%s is NULL", name);       \
    if (!aligned16(ptr)) return fail(FOVEA_ERR_INVALID_ARG, "%s is not 16-byte aligned", name); \
  } while (0)

static fovea_status check_step_params(const fovea_params* p) {
  fovea_status st = check_dims(p);
  if (st != FOVEA_OK) return st;
  if (p->mlp_hidden <= 0 || p->mlp_hidden % 128 != 0)
    return fail(FOVEA_ERR_INVALID_ARG, "mlp_hidden %d must be a positive multiple of 128",
                p->mlp_hidden);
  if (p->mlp_hidden > FOVEA_MAX_H)
    return fail(FOVEA_ERR_UNSUPPORTED, "mlp_hidden %d exceeds %d", p->mlp_hidden, FOVEA_MAX_H);
  if (p->max_depth < 0) return fail(FOVEA_ERR_INVALID_ARG, "max_depth %d < 0", p->max_depth);
  NEED_PTR(p->ln_h_gamma, "ln_h_gamma");
  NEED_PTR(p->ln_h_beta, "ln_h_beta");
  NEED_PTR(p->E_dep, "E_dep");
  NEED_PTR(p->W_Q, "W_Q");
  NEED_PTR(p->W_f1, "W_f1");
  NEED_PTR(p->b_f1, "b_f1");
  NEED_PTR(p->W_f2, "W_f2");
  NEED_PTR(p->b_f2, "b_f2");
  NEED_PTR(p->W_g1, "W_g1");
  NEED_PTR(p->b_g1, "b_g1");
  NEED_PTR(p->w_g2, "w_g2");
  if (p->b_g2 == nullptr) return fail(FOVEA_ERR_INVALID_ARG, "b_g2 is NULL");
  NEED_PTR(p->rms_gamma, "rms_gamma");
  return FOVEA_OK;
}

static fovea_status alloc_dev(void** ptr, size_t bytes, const char* what) {
  *ptr = nullptr;
  if (bytes == 0) return FOVEA_OK;
  const char* fault = getenv("FOVEA_FAULT_ALLOC");
  if (fault != nullptr && fault[0] == '1')
    return fail(FOVEA_ERR_OOM, "allocation of %s (%zu bytes) failed (FOVEA_FAULT_ALLOC=1)", what,
                bytes);
  cudaError_t e = cudaMalloc(ptr, bytes);
  if (e != cudaSuccess) {
    cudaGetLastError();
    *ptr = nullptr;
    return fail(FOVEA_ERR_OOM, "cudaMalloc of %s (%zu bytes): %s", what, bytes,
                cudaGetErrorString(e));
  }
  return FOVEA_OK;
}

static void free_memory(fovea_memory* m) {
  if (m == nullptr) return;
  cudaFree(m->keys);
  cudaFree(m->values);
  cudaFree(m->proj);
  cudaFree(m->projT);
  cudaFree(m->folded);
  cudaFree(m->orig_index);
  cudaFree(m->err);
  delete m;
}

// The bf16 path runs every GEMM on tcgen05 tensor cores; fp32 runs SIMT.
static cudaError_t run_gemm(int dtype, int epi, const GemmArgs& a, const TmaOperand& A0,
                            const TmaOperand& A1, const TmaOperand& B0, const TmaOperand& B1,
                            int max_m, int max_n, cudaStream_t s) {
  if (dtype == FOVEA_BF16) return launch_gemm_tc(epi, a, A0, A1, B0, B1, max_m, max_n, s);
  return launch_gemm_simt(dtype, epi, a, max_m, max_n, s);
}

static void init_args(GemmArgs& a) {
  memset(&a, 0, sizeof(a));
  a.a_split = 0x7fffffff;
  a.a_split2 = 0x7fffffff;
  a.epi_split = 0x7fffffff;
  a.scale = 1.0f;
}

extern "C" {

FOVEA_API const char* fovea_last_error(void) { return g_last_error.c_str(); }

FOVEA_API int fovea_version(void) { return 200; }

FOVEA_API fovea_status fovea_build_memory(const fovea_params* p, const void* v,
                                          const uint8_t* mask, int B, int M_max, void* stream,
                                          fovea_memory** out) {
  g_last_error.clear();
  fovea_status st = check_dims(p);
  if (st != FOVEA_OK) return st;
  if (out == nullptr) return fail(FOVEA_ERR_INVALID_ARG, "out is NULL");
  if (B < 1) return fail(FOVEA_ERR_INVALID_ARG, "B = %d must be >= 1", B);
  if (B > FOVEA_MAX_SEQ) return fail(FOVEA_ERR_UNSUPPORTED, "B = %d exceeds %d", B, FOVEA_MAX_SEQ);
  if (M_max < 0) return fail(FOVEA_ERR_INVALID_ARG, "M_max = %d < 0", M_max);
  if (mask == nullptr && M_max > FOVEA_MAX_ENTRIES)
    return fail(FOVEA_ERR_UNSUPPORTED, "M_max = %d valid entries exceed %d per image", M_max,
                FOVEA_MAX_ENTRIES);
  if ((long long)B * M_max >= (1ll << 31))
    return fail(FOVEA_ERR_UNSUPPORTED, "B * M_max exceeds 2^31 entries");
  if (M_max > 0) NEED_PTR(v, "v");
  NEED_PTR(p->ln_v_gamma, "ln_v_gamma");
  NEED_PTR(p->ln_v_beta, "ln_v_beta");
  NEED_PTR(p->W_K, "W_K");
  NEED_PTR(p->W_U, "W_U");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int d = p->d_model;
  const size_t es = esize(p->dtype);

  fovea_memory* m = new fovea_memory();
  m->B = B;
  m->M_max = M_max;
  m->d = d;
  m->dtype = p->dtype;
  cudaGetDevice(&m->device);
  st = alloc_dev(reinterpret_cast<void**>(&m->err), 256, "error word");
  if (st != FOVEA_OK) { free_memory(m); return st; }
  void* scratch = nullptr;           // counts [B] | key_off [B] (int32)
  st = alloc_dev(&scratch, align_up(2 * B * sizeof(int32_t), 256), "build scratch");
  if (st != FOVEA_OK) { free_memory(m); return st; }
  int32_t* d_counts = static_cast<int32_t*>(scratch);
  int32_t* d_keyoff = d_counts + B;

  auto cleanup = [&](fovea_status code) {
    cudaStreamSynchronize(s);
    cudaFree(scratch);
    free_memory(m);
    return code;
  };
  cudaError_t e = cudaMemsetAsync(m->err, 0, 256, s);
  if (e != cudaSuccess) return cleanup(cuda_fail(e, "cudaMemsetAsync"));

  m->counts.assign(B, M_max);
  if (mask != nullptr && M_max > 0) {
    { KernelTimer t("count_valid", s); e = launch_count_valid(mask, B, M_max, d_counts, s); }
    if (e != cudaSuccess) return cleanup(cuda_fail(e, "count_valid"));
    e = cudaMemcpyAsync(m->counts.data(), d_counts, B * sizeof(int32_t), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cleanup(cuda_fail(e, "reading valid counts"));
  }
  m->offsets.assign(B + 1, 0);
  for (int b = 0; b < B; ++b) {
    if (m->counts[b] > FOVEA_MAX_ENTRIES)
      return cleanup(fail(FOVEA_ERR_UNSUPPORTED, "image %d has %d valid entries (limit %d)", b,
                          m->counts[b], FOVEA_MAX_ENTRIES));
    m->offsets[b + 1] = m->offsets[b] + m->counts[b];
  }
  m->total = (int)m->offsets[B];
  const int total = m->total;
  if (total > 0) {
    std::vector<int32_t> keyoff(B);
    for (int b = 0; b < B; ++b) keyoff[b] = (int32_t)m->offsets[b];
    void* xv = nullptr;
    void* src_row = nullptr;
    void* fix = nullptr;                     // bf16: count word + listed key elements
    const bool bf = p->dtype == FOVEA_BF16;
    const long long fix_cap = bf ? (long long)total * d / 8 + 4096 : 0;
    if ((st = alloc_dev(&m->keys, (size_t)total * d * es, "keys")) != FOVEA_OK ||
        (st = alloc_dev(&m->values, (size_t)total * d * es, "values")) != FOVEA_OK ||
        (st = alloc_dev(reinterpret_cast<void**>(&m->orig_index), total * sizeof(int32_t),
                        "index")) != FOVEA_OK ||
        (st = alloc_dev(&src_row, total * sizeof(int32_t), "source rows")) != FOVEA_OK ||
        (st = alloc_dev(&xv, (size_t)total * d * es, "LN(v)")) != FOVEA_OK ||
        (bf && (st = alloc_dev(&fix, 256 + (size_t)fix_cap * sizeof(KeyFix), "key fix list")) != FOVEA_OK)) {
      cudaFree(xv);
      cudaFree(src_row);
      cudaFree(fix);
      return cleanup(st);
    }
    int* fix_count = static_cast<int*>(fix);
    KeyFix* fix_list = bf ? reinterpret_cast<KeyFix*>(static_cast<uint8_t*>(fix) + 256) : nullptr;
    auto run = [&]() -> fovea_status {
      cudaError_t err = cudaMemcpyAsync(d_keyoff, keyoff.data(), B * sizeof(int32_t),
                                        cudaMemcpyHostToDevice, s);
      if (err != cudaSuccess) return cuda_fail(err, "cudaMemcpyAsync");
      { KernelTimer t("compact", s);
        err = launch_compact(mask, B, M_max, d_keyoff, m->orig_index, (int32_t*)src_row, s); }
      if (err != cudaSuccess) return cuda_fail(err, "compact");
      { KernelTimer t("ln_v", s);
        err = launch_ln_rows(p->dtype, v, (const int32_t*)src_row, total, d, p->ln_v_gamma,
                             p->ln_v_beta, p->ln_eps, nullptr, nullptr, 0, m->err, xv, s); }
      if (err != cudaSuccess) return cuda_fail(err, "ln_v");
      GemmArgs a;
      init_args(a);
      a.k_total = d;
      a.a_split = d;
      a.b_split = d;
      a.A0 = p->W_K; a.A1 = p->W_U; a.lda0 = d; a.lda1 = d;
      a.B0 = xv; a.B1 = xv; a.ldb0 = d; a.ldb1 = d;
      a.epi_split = d;
      a.out0 = m->keys; a.out1 = m->values; a.ldc = d;
      a.err = m->err;
      a.fix_list = fix_list; a.fix_count = fix_count; a.fix_cap = (int)fix_cap;
      a.ngroups = 1;
      a.groups[0] = GemmGroup{0, 2 * d, 0, total, 0};
      TmaOperand A0{p->W_K, d, d, d}, A1{p->W_U, d, d, d}, B0{xv, total, d, d}, B1{nullptr, 0, 0, 0};
      if (bf) {
        err = cudaMemsetAsync(fix_count, 0, sizeof(int), s);
        if (err != cudaSuccess) return cuda_fail(err, "cudaMemsetAsync");
      }
      { KernelTimer t("memory_proj", s);
        err = run_gemm(p->dtype, bf ? kEpiStoreKeys : kEpiStore, a, A0, A1, B0, B1, 2 * d, total, s); }
      if (err != cudaSuccess) return cuda_fail(err, "memory projection");
      if (bf) {
        // keys whose fp32 value sat near a bf16 rounding midpoint: exact recompute
        { KernelTimer t("refine_keys", s);
          err = launch_refine_keys(xv, p->W_K, d, fix_list, fix_count, (int)fix_cap, total, m->keys, s); }
        if (err != cudaSuccess) return cuda_fail(err, "refine_keys");
      }
      int herr[2] = {0, 0};
      err = cudaMemcpyAsync(&herr[0], m->err, sizeof(int), cudaMemcpyDeviceToHost, s);
      if (err == cudaSuccess && bf)
        err = cudaMemcpyAsync(&herr[1], fix_count, sizeof(int), cudaMemcpyDeviceToHost, s);
      if (err == cudaSuccess) err = cudaStreamSynchronize(s);
      if (err != cudaSuccess) return cuda_fail(err, "memory build");
      if (herr[0] & kErrTimeout)
        return fail(FOVEA_ERR_TIMEOUT, "a bounded device wait gave up during the memory build");
      m->refined = herr[1];
      if (bf && herr[1] > fix_cap) {      // list overflowed: refine every key element
        { KernelTimer t("refine_keys", s);
          err = launch_refine_keys(xv, p->W_K, d, nullptr, nullptr, 0, total, m->keys, s); }
        if (err == cudaSuccess) err = cudaStreamSynchronize(s);
        if (err != cudaSuccess) return cuda_fail(err, "refine_keys");
      }
      // bf16 with W_Q given: the folded keys kappa_i = W_Q^T k_i, a GEMM of
      // W_Q^T (transposed once here) with the stored keys, kept as the hi / lo
      // pair of its fp32 accumulator (no bf16 rounding of the query map)
      if (bf && p->W_Q != nullptr && aligned16(p->W_Q)) {
        fovea_status fs = alloc_dev(&m->folded, (size_t)total * 2 * d * 2, "folded keys");
        if (fs != FOVEA_OK) return fs;
        void* wqt = nullptr;
        if ((fs = alloc_dev(&wqt, (size_t)d * d * 2, "transposed W_Q")) != FOVEA_OK) return fs;
        auto fold = [&]() -> fovea_status {
          { KernelTimer t("transpose_wq", s);
            err = launch_transpose_bf16(p->W_Q, d, d, wqt, s); }
          if (err != cudaSuccess) return cuda_fail(err, "transpose W_Q");
          GemmArgs fa;
          init_args(fa);
          fa.k_total = d;
          fa.b_split = d;
          fa.B0 = m->keys; fa.ldb0 = d;
          fa.out0 = m->folded;
          fa.out1 = static_cast<__nv_bfloat16*>(m->folded) + d;
          fa.ldc = 2 * d;
          fa.err = m->err;
          fa.ngroups = 1;
          fa.groups[0] = GemmGroup{0, d, 0, total, 0};
          { KernelTimer t("memory_fold", s);
            err = launch_gemm_tc(kEpiStoreHiLo, fa, TmaOperand{wqt, d, d, d},
                                 TmaOperand{nullptr, 0, 0, 0}, TmaOperand{m->keys, total, d, d},
                                 TmaOperand{nullptr, 0, 0, 0}, d, total, s); }
          if (err != cudaSuccess) return cuda_fail(err, "query folding of the keys");
          int fe = 0;
          err = cudaMemcpyAsync(&fe, m->err, sizeof(int), cudaMemcpyDeviceToHost, s);
          if (err == cudaSuccess) err = cudaStreamSynchronize(s);
          if (err != cudaSuccess) return cuda_fail(err, "query folding");
          if (fe & kErrTimeout)
            return fail(FOVEA_ERR_TIMEOUT, "a bounded device wait gave up while folding the keys");
          return FOVEA_OK;
        };
        fs = fold();
        cudaStreamSynchronize(s);
        cudaFree(wqt);
        if (fs != FOVEA_OK) return fs;
        m->fold_wq = p->W_Q;
      }
      // bf16 with the fusion weights given: p_i = [W_f1 ; W_g1]_r u_i, the
      // first fusion layer's r-half applied to every value once per image
      const int H = p->mlp_hidden;
      if (bf && p->W_f1 != nullptr && p->W_g1 != nullptr && H > 0 && H % 128 == 0 &&
          H <= FOVEA_MAX_H && aligned16(p->W_f1) && aligned16(p->W_g1)) {
        fovea_status ps = alloc_dev(&m->proj, (size_t)total * 2 * H * 2, "projected values");
        if (ps != FOVEA_OK) return ps;
        const __nv_bfloat16* wf1r = static_cast<const __nv_bfloat16*>(p->W_f1) + d;
        const __nv_bfloat16* wg1r = static_cast<const __nv_bfloat16*>(p->W_g1) + d;
        GemmArgs pa;
        init_args(pa);
        pa.k_total = d;
        pa.a_split = H;
        pa.b_split = d;
        pa.B0 = m->values; pa.ldb0 = d;
        pa.out0 = m->proj; pa.ldc = 2 * H;
        pa.err = m->err;
        pa.ngroups = 1;
        pa.groups[0] = GemmGroup{0, 2 * H, 0, total, 0};
        { KernelTimer t("memory_proj_fusion", s);
          err = launch_gemm_tc(kEpiStore, pa, TmaOperand{wf1r, H, d, 2 * d},
                               TmaOperand{wg1r, H, d, 2 * d}, TmaOperand{m->values, total, d, d},
                               TmaOperand{nullptr, 0, 0, 0}, 2 * H, total, s); }
        if (err == cudaSuccess) err = cudaStreamSynchronize(s);
        if (err != cudaSuccess) return cuda_fail(err, "fusion projection of the values");
        int m_max = 0;
        for (int b = 0; b < B; ++b) m_max = std::max(m_max, m->counts[b]);
        const int ld = (m_max + 63) / 64 * 64;
        if ((ps = alloc_dev(&m->projT, (size_t)B * 2 * H * ld * 2, "transposed projected values")) != FOVEA_OK)
          return ps;
        static thread_local ImageTable itab;
        itab.B = B;
        for (int b = 0; b < B; ++b) {
          itab.off[b] = (int)m->offsets[b];
          itab.m[b] = m->counts[b];
        }
        { KernelTimer t("memory_proj_transpose", s);
          err = launch_transpose_images(m->proj, 2 * H, ld, itab, m->projT, s); }
        if (err == cudaSuccess) err = cudaStreamSynchronize(s);
        if (err != cudaSuccess) return cuda_fail(err, "transposing the projected values");
        m->proj_ld = ld;
        m->proj_wf1 = p->W_f1;
        m->proj_wg1 = p->W_g1;
        m->proj_h = H;
      }
      return FOVEA_OK;
    };
    st = run();
    cudaStreamSynchronize(s);
    cudaFree(xv);
    cudaFree(src_row);
    cudaFree(fix);
    if (st != FOVEA_OK) return cleanup(st);
  }
  cudaStreamSynchronize(s);
  cudaFree(scratch);
  *out = m;
  return FOVEA_OK;
}

FOVEA_API void fovea_memory_destroy(fovea_memory* mem) { free_memory(mem); }

FOVEA_API fovea_status fovea_memory_info(const fovea_memory* mem, int* B, int* total_valid,
                                         int32_t* valid_counts) {
  g_last_error.clear();
  if (mem == nullptr) return fail(FOVEA_ERR_INVALID_ARG, "memory is NULL");
  if (B) *B = mem->B;
  if (total_valid) *total_valid = mem->total;
  if (valid_counts) memcpy(valid_counts, mem->counts.data(), mem->B * sizeof(int32_t));
  return FOVEA_OK;
}

FOVEA_API fovea_status fovea_memory_folded_keys(const fovea_memory* mem, const void* W_Q,
                                                const void** folded) {
  g_last_error.clear();
  if (mem == nullptr) return fail(FOVEA_ERR_INVALID_ARG, "memory is NULL");
  if (folded == nullptr) return fail(FOVEA_ERR_INVALID_ARG, "folded is NULL");
  *folded = (mem->folded != nullptr && W_Q != nullptr && mem->fold_wq == W_Q) ? mem->folded : nullptr;
  return FOVEA_OK;
}

FOVEA_API fovea_status fovea_memory_tensors(const fovea_memory* mem, const void** keys,
                                            const void** values, const int32_t** index,
                                            int64_t* offsets) {
  g_last_error.clear();
  if (mem == nullptr) return fail(FOVEA_ERR_INVALID_ARG, "memory is NULL");
  if (keys) *keys = mem->keys;
  if (values) *values = mem->values;
  if (index) *index = mem->orig_index;
  if (offsets) memcpy(offsets, mem->offsets.data(), (mem->B + 1) * sizeof(int64_t));
  return FOVEA_OK;
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Workspace layout (all regions 256-byte aligned)
// ---------------------------------------------------------------------------
namespace {
struct WsLayout {
  size_t err, xh, q, scores, sel_pos, sel_w, sel_cnt, r_lo, act, c, gh, alpha_hi, alpha_lo, total;
};

// LM head workspace: the header, then the candidate keys [N, slots, k_c].
size_t lm_head_ws_bytes(int N, int slots, int k_c) {
  return kWsHeaderBytes + (size_t)N * slots * k_c * sizeof(unsigned long long);
}

int device_sms() {
  static int sms = 0;
  if (sms == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (sms <= 0) sms = 148;
  }
  return sms;
}

// alpha_ld: entries of a dense weight row (the memory's padded per-image
// count when it keeps the transposed projected values, else 0).
WsLayout ws_layout(int dtype, int d, int H, int N, int k_max, long long score_elems, int alpha_ld) {
  WsLayout L;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off = align_up(off + bytes, 256);
    return o;
  };
  const size_t es = esize(dtype);
  L.err = take(kWsHeaderBytes);          // the sticky error word, then reserved words
  L.xh = take((size_t)N * d * es);
  L.q = take((size_t)N * d * es * (dtype == FOVEA_BF16 ? 2 : 1));   // bf16: q_hi | q_lo
  L.scores = take((size_t)score_elems * 4);
  L.sel_pos = take((size_t)N * k_max * 4);
  L.sel_w = take((size_t)N * k_max * 4);
  L.sel_cnt = take((size_t)N * 4);
  L.r_lo = take((size_t)N * d * es);
  L.act = take((size_t)N * 2 * H * es);
  L.c = take((size_t)N * d * 4);
  L.gh = take(dtype == FOVEA_BF16 ? (size_t)N * 2 * H * 4 : 0);   // [W_f1 ; W_g1]_h h, fp32
  L.alpha_hi = take((size_t)N * alpha_ld * 2);                     // dense weights, bf16 hi
  L.alpha_lo = take((size_t)N * alpha_ld * 2);                     // and lo
  L.total = off;
  return L;
}

fovea_status check_rows(const fovea_memory* mem, const int32_t* row_offsets, int* N_out,
                        long long* score_elems, int* max_m, int* max_r, int* ngroups) {
  if (mem == nullptr) return fail(FOVEA_ERR_INVALID_ARG, "memory is NULL");
  if (row_offsets == nullptr) return fail(FOVEA_ERR_INVALID_ARG, "row_offsets is NULL");
  if (row_offsets[0] != 0) return fail(FOVEA_ERR_INVALID_ARG, "row_offsets[0] = %d, expected 0", row_offsets[0]);
  long long se = 0;
  int mm = 0, mr = 0, ng = 0;
  for (int b = 0; b < mem->B; ++b) {
    const int r = row_offsets[b + 1] - row_offsets[b];
    if (r < 0) return fail(FOVEA_ERR_INVALID_ARG, "row_offsets decrease at sequence %d", b);
    se += (long long)r * mem->counts[b];
    if (r > 0 && mem->counts[b] > mm) mm = mem->counts[b];
    if (r > 0 && mem->counts[b] > 0) {
      ++ng;
      if (r > mr) mr = r;
    }
  }
  *N_out = row_offsets[mem->B];
  *score_elems = se;
  *max_m = mm;
  *max_r = mr;
  *ngroups = ng;
  return FOVEA_OK;
}
}  // namespace

extern "C" {

FOVEA_API fovea_status fovea_workspace_size(const fovea_params* p, const fovea_memory* mem,
                                            const int32_t* row_offsets, int k_max,
                                            size_t* bytes) {
  g_last_error.clear();
  fovea_status st = check_dims(p);
  if (st != FOVEA_OK) return st;
  if (bytes == nullptr) return fail(FOVEA_ERR_INVALID_ARG, "bytes is NULL");
  if (p->mlp_hidden <= 0 || p->mlp_hidden % 128 != 0)
    return fail(FOVEA_ERR_INVALID_ARG, "mlp_hidden %d must be a positive multiple of 128",
                p->mlp_hidden);
  if (k_max < 1) return fail(FOVEA_ERR_INVALID_ARG, "k_max = %d < 1", k_max);
  int N, mm, mr, ng;
  long long se;
  if ((st = check_rows(mem, row_offsets, &N, &se, &mm, &mr, &ng)) != FOVEA_OK) return st;
  *bytes = ws_layout(p->dtype, p->d_model, p->mlp_hidden, N, k_max, se,
                     mem->projT != nullptr ? mem->proj_ld : 0).total;
  return FOVEA_OK;
}

FOVEA_API fovea_status fovea_workspace_init(void* workspace, size_t bytes, void* stream) {
  g_last_error.clear();
  if (workspace == nullptr) return fail(FOVEA_ERR_INVALID_ARG, "workspace is NULL");
  if (bytes < kWsHeaderBytes)
    return fail(FOVEA_ERR_INVALID_ARG, "workspace of %zu bytes is too small", bytes);
  FOVEA_CUDA(cudaMemsetAsync(workspace, 0, kWsHeaderBytes, static_cast<cudaStream_t>(stream)),
             "cudaMemsetAsync");
  return FOVEA_OK;
}

FOVEA_API fovea_status fovea_sync_errors(void* workspace, void* stream) {
  g_last_error.clear();
  if (workspace == nullptr) return fail(FOVEA_ERR_INVALID_ARG, "workspace is NULL");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int herr = 0;
  FOVEA_CUDA(cudaMemcpyAsync(&herr, workspace, sizeof(int), cudaMemcpyDeviceToHost, s),
             "cudaMemcpyAsync");
  FOVEA_CUDA(cudaStreamSynchronize(s), "cudaStreamSynchronize");
  // clear the whole header: a kernel that gave up may have left other words set
  FOVEA_CUDA(cudaMemsetAsync(workspace, 0, herr ? kWsHeaderBytes : sizeof(int), s),
             "cudaMemsetAsync");
  FOVEA_CUDA(cudaStreamSynchronize(s), "cudaStreamSynchronize");
  if (herr & kErrTimeout)
    return fail(FOVEA_ERR_TIMEOUT, "a bounded device wait gave up (error word 0x%x)", herr);
  if (herr & kErrDepth)
    return fail(FOVEA_ERR_INVALID_ARG, "a draft state had a depth outside [0, max_depth]");
  return FOVEA_OK;
}

FOVEA_API fovea_status fovea_debug_wait_limit(unsigned long long limit_ns) {
  g_last_error.clear();
  set_wait_limit_ns(limit_ns == 0 ? kDefaultWaitLimitNs : limit_ns);
  return FOVEA_OK;
}

FOVEA_API fovea_status fovea_retrieve_fuse(const fovea_params* p, const fovea_memory* mem,
                                           const void* h, const int32_t* depth,
                                           const int32_t* row_offsets, const float* row_scale,
                                           float rho, int k_min, int k_max, int l_max,
                                           void* h_out, int32_t* counts, int32_t* indices,
                                           float* readout, float* gate, void* workspace,
                                           size_t workspace_bytes, void* stream) {
  g_last_error.clear();
  fovea_status st = check_step_params(p);
  if (st != FOVEA_OK) return st;
  if (!(rho > 0.0f && rho <= 1.0f))
    return fail(FOVEA_ERR_INVALID_ARG, "rho = %g must satisfy 0 < rho <= 1", (double)rho);
  if (k_min < 1 || k_min > k_max)
    return fail(FOVEA_ERR_INVALID_ARG, "need 1 <= k_min (%d) <= k_max (%d)", k_min, k_max);
  if (k_max > FOVEA_MAX_K)
    return fail(FOVEA_ERR_UNSUPPORTED, "k_max = %d exceeds %d", k_max, FOVEA_MAX_K);
  if (mem == nullptr) return fail(FOVEA_ERR_INVALID_ARG, "memory is NULL");
  if (mem->d != p->d_model || mem->dtype != p->dtype)
    return fail(FOVEA_ERR_INVALID_ARG, "memory was built with d=%d dtype=%d, params have d=%d dtype=%d",
                mem->d, mem->dtype, p->d_model, p->dtype);
  int N, max_m, max_r, ngroups;
  long long score_elems;
  if ((st = check_rows(mem, row_offsets, &N, &score_elems, &max_m, &max_r, &ngroups)) != FOVEA_OK)
    return st;
  if (N == 0) return FOVEA_OK;
  NEED_PTR(h, "h");
  NEED_PTR(h_out, "h_out");
  if (depth == nullptr) return fail(FOVEA_ERR_INVALID_ARG, "depth is NULL");
  if (readout != nullptr && !aligned16(readout))
    return fail(FOVEA_ERR_INVALID_ARG, "readout is not 16-byte aligned");
  if (workspace == nullptr) return fail(FOVEA_ERR_INVALID_ARG, "workspace is NULL");
  if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0)
    return fail(FOVEA_ERR_INVALID_ARG, "workspace is not 256-byte aligned");
  const int d = p->d_model, H = p->mlp_hidden, dt = p->dtype;
  const WsLayout L = ws_layout(dt, d, H, N, k_max, score_elems,
                              mem->projT != nullptr ? mem->proj_ld : 0);
  if (workspace_bytes < L.total)
    return fail(FOVEA_ERR_INVALID_ARG, "workspace has %zu bytes, needs %zu", workspace_bytes, L.total);

  cudaStream_t s = static_cast<cudaStream_t>(stream);
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  int* err = reinterpret_cast<int*>(ws + L.err);
  void* xh = ws + L.xh;
  void* q = ws + L.q;
  float* scores = reinterpret_cast<float*>(ws + L.scores);
  int32_t* sel_pos = reinterpret_cast<int32_t*>(ws + L.sel_pos);
  float* sel_w = reinterpret_cast<float*>(ws + L.sel_w);
  int32_t* sel_cnt = reinterpret_cast<int32_t*>(ws + L.sel_cnt);
  void* r_lo = ws + L.r_lo;
  void* act = ws + L.act;
  float* cbuf = reinterpret_cast<float*>(ws + L.c);
  float* gh = reinterpret_cast<float*>(ws + L.gh);
  // depth gate: rows deeper than l_max are not corrected (their selection is
  // empty and h_hat = h); with l_max >= D every row is corrected and the gate
  // reads nothing
  const DepthGate gate_rows{l_max < p->max_depth ? depth : nullptr, l_max, p->max_depth};

  // Per-sequence table (kernel parameter).
  static thread_local SeqTable tab;
  tab.B = mem->B;
  for (int b = 0; b < mem->B; ++b) {
    tab.row_start[b] = row_offsets[b];
    tab.key_off[b] = (int)mem->offsets[b];
    tab.m[b] = mem->counts[b];
  }
  tab.row_start[mem->B] = row_offsets[mem->B];
  {
    long long so = 0;
    for (int b = 0; b < mem->B; ++b) {
      tab.score_off[b] = so;
      so += (long long)(row_offsets[b + 1] - row_offsets[b]) * mem->counts[b];
    }
  }
  cudaError_t e;

  // (1) x_h = LN_h(h) + E_dep[l]
  { KernelTimer t("ln_query", s);
    e = launch_ln_query(dt, h, N, d, p->ln_h_gamma, p->ln_h_beta, p->ln_eps, p->E_dep, depth,
                        p->max_depth, err, xh, s); }
  if (e != cudaSuccess) return cuda_fail(e, "ln_query");

  static thread_local GemmArgs a;
  // (2) q = W_Q x_h  (bf16 path: stored as q_hi + q_lo).  With the memory's
  // projected values valid for these weights, the same launch computes
  // G_h = [W_f1 ; W_g1]_h h (the h-half of the first fusion layer, fp32):
  // the r-half then reduces to a weighted sum of projected values (4).
  // With the memory's folded keys valid for this W_Q, q is never formed:
  // the scores take x_h against the folded keys, and the launch computes
  // G_h alone (or is skipped without the projected values).
  const bool bf = dt == FOVEA_BF16;
  // The r-half of the first fusion layer from the projected values: either
  // gathered row by row in the selection kernel (rows of <= 2048 entries,
  // k_max <= 256, a batch that fills the GPU in about a wave), or, with the
  // selection weights written as dense rows, one GEMM against the memory's
  // transposed projected values (long rows, large caps, large batches).
  const bool have_proj = bf && mem->proj != nullptr && mem->proj_wf1 == p->W_f1 &&
                         mem->proj_wg1 == p->W_g1 && mem->proj_h == H;
  const bool alpha_path = have_proj && mem->projT != nullptr &&
                          (!select_readout_fits(max_m, k_max) || N > 2 * device_sms());
  const bool use_proj = have_proj && (alpha_path || select_readout_fits(max_m, k_max));
  const bool use_fold = bf && mem->folded != nullptr && mem->fold_wq == p->W_Q;
  // the folded keys are [total, 2d] (hi | lo per entry)
  const long long score_key_bytes = (long long)mem->total * d * 2 * (use_fold ? 2 : 1);
  const void* score_keys = use_fold ? mem->folded : mem->keys;
  // With folded keys and projected values, G_h does not depend on the query:
  // when one sequence's keys serve every row (one score group covering all N
  // rows), the score launch computes it too, as two more feature parts
  // against h.
  int gh_seq = -1;
  if (use_fold && use_proj && ngroups == 1) {
    for (int b = 0; b < mem->B; ++b)
      if (row_offsets[b + 1] - row_offsets[b] == N && mem->counts[b] > 0) gh_seq = b;
  }
  const bool gh_in_scores = gh_seq >= 0;
  void* q_lo = bf ? static_cast<void*>(static_cast<uint8_t*>(q) + (size_t)N * d * 2) : nullptr;
  init_args(a);
  a.k_total = d; a.b_split = d;
  a.A0 = p->W_Q; a.lda0 = d;
  a.B0 = xh; a.ldb0 = d;
  a.out0 = q; a.out1 = q_lo; a.ldc = d; a.err = err;
  a.ngroups = 1;
  a.groups[0] = GemmGroup{0, d, 0, N, 0};
  if (use_proj) {
    a.a_split = d; a.a_split2 = d + H;
    a.r_by_part = 1;
    a.epi_split = d;
    a.out2 = gh; a.ldc2 = 2 * H;
    a.groups[0] = GemmGroup{0, d + 2 * H, 0, N, 0};
  }
  // entries selected at most: when they are most of the memory, the value
  // rows are prefetched
  long long m_sel = 0;
  for (int b = 0; b < mem->B; ++b)
    m_sel += std::min<long long>(mem->counts[b], (long long)(row_offsets[b + 1] - row_offsets[b]) * k_max);
  if (bf) {
    // the keys when the score GEMM's own loads before its griddepcontrol.wait
    // (its first ring stages) cannot cover them, and the values when most of
    // their rows will be read by the readout
    if (score_key_bytes > (8ll << 20)) {
      a.pf_ptr[a.n_prefetch] = score_keys;
      a.pf_bytes[a.n_prefetch++] = score_key_bytes;
    }
    if (2 * m_sel >= mem->total) {
      if (!use_proj || readout != nullptr) {
        a.pf_ptr[a.n_prefetch] = mem->values;
        a.pf_bytes[a.n_prefetch++] = (long long)mem->total * d * 2;
      }
    }
  }
  if (use_fold && use_proj && !gh_in_scores) {
    // G_h only: parts W_f1 and W_g1 (h-halves), both against h, fp32 out
    a.A0 = p->W_f1; a.lda0 = 2 * d;
    a.B0 = h;
    a.a_split = H; a.a_split2 = 0x7fffffff;
    a.r_by_part = 0;
    a.epi_split = 0;
    a.out2 = gh; a.ldc2 = 2 * H;
    a.groups[0] = GemmGroup{0, 2 * H, 0, N, 0};
    { KernelTimer t("fusion_h", s);
      e = launch_gemm_tc(kEpiQueryH, a, TmaOperand{p->W_f1, H, d, 2 * d},
                         TmaOperand{p->W_g1, H, d, 2 * d}, TmaOperand{h, N, d, d},
                         TmaOperand{nullptr, 0, 0, 0}, 2 * H, N, s); }
    if (e != cudaSuccess) return cuda_fail(e, "fusion_h");
  } else if (!use_fold) {
    KernelTimer t("query_proj", s);
    if (use_proj)
      e = launch_gemm_tc(kEpiQueryH, a, TmaOperand{p->W_Q, d, d, d}, TmaOperand{p->W_f1, H, d, 2 * d},
                         TmaOperand{xh, N, d, d}, TmaOperand{h, N, d, d}, d + 2 * H, N, s,
                         TmaOperand{p->W_g1, H, d, 2 * d});
    else
      e = run_gemm(dt, bf ? kEpiStoreHiLo : kEpiStore, a, TmaOperand{p->W_Q, d, d, d},
                   TmaOperand{nullptr, 0, 0, 0}, TmaOperand{xh, N, d, d},
                   TmaOperand{nullptr, 0, 0, 0}, d, N, s);
    if (e != cudaSuccess) return cuda_fail(e, "query_proj");
  }

  // (3) s = q k^T / sqrt(d) (* row_scale), per sequence; folded: x_h against
  // kappa_hi and kappa_lo
  if (score_elems > 0) {
    init_args(a);
    a.k_total = d; a.b_split = d;
    a.A0 = score_keys; a.lda0 = use_fold ? 2 * d : d;
    a.B0 = use_fold ? xh : q; a.ldb0 = d;
    a.out0 = scores;
    a.row_scale = row_scale;
    a.scale = (float)(1.0 / sqrt((double)d));
    a.err = err;
    a.f_lo_kb = use_fold ? d / 64 : 0;
    int g = 0;
    for (int b = 0; b < mem->B; ++b) {
      const int r = row_offsets[b + 1] - row_offsets[b];
      if (r == 0 || mem->counts[b] == 0) continue;
      a.groups[g++] = GemmGroup{(int)mem->offsets[b], mem->counts[b], row_offsets[b], r, tab.score_off[b]};
    }
    a.ngroups = g;
    a.dual_b = bf && !use_fold ? 1 : 0;
    if (use_fold && !use_proj && 2 * m_sel >= mem->total) {
      // no query launch carries the value prefetch on this path
      a.pf_ptr[a.n_prefetch] = mem->values;
      a.pf_bytes[a.n_prefetch++] = (long long)mem->total * d * 2;
    }
    if (bf && !use_proj) {
      // the fusion weights, read after selection and readout (with the
      // projected values the selection kernel prefetches them, and the
      // second correction layer's GEMM loads its weights before its
      // griddepcontrol.wait)
      a.pf_ptr[a.n_prefetch] = p->W_f1;
      a.pf_bytes[a.n_prefetch++] = (long long)H * 2 * d * 2;
      a.pf_ptr[a.n_prefetch] = p->W_g1;
      a.pf_bytes[a.n_prefetch++] = (long long)H * 2 * d * 2;
      if (a.n_prefetch < 4) {
        a.pf_ptr[a.n_prefetch] = p->W_f2;
        a.pf_bytes[a.n_prefetch++] = (long long)d * H * 2;
      }
    }
    const TmaOperand folded_op{mem->folded, mem->total, 2 * d, 2 * d};
    if (gh_in_scores) {
      // one group: the sequence's folded keys (scores, against x_h), then the
      // h-halves of W_f1 and W_g1 (G_h, against h)
      const int M = mem->counts[gh_seq];
      a.groups[0] = GemmGroup{(int)mem->offsets[gh_seq], M + 2 * H, 0, N, 0};
      a.a_split = M; a.a_split2 = M + H;
      a.r_by_part = 1;
      a.epi_split = M;
      a.out2 = gh; a.ldc2 = 2 * H;
      if (readout != nullptr && 2 * m_sel >= mem->total && a.n_prefetch < 4) {
        a.pf_ptr[a.n_prefetch] = mem->values;
        a.pf_bytes[a.n_prefetch++] = (long long)mem->total * d * 2;
      }
      KernelTimer t("score_fusion_h", s);
      e = launch_gemm_tc(kEpiScoresFolded, a, folded_op, TmaOperand{p->W_f1, H, d, 2 * d},
                         TmaOperand{xh, N, d, d}, TmaOperand{h, N, d, d}, M + 2 * H, N, s,
                         TmaOperand{p->W_g1, H, d, 2 * d});
    } else if (use_fold) {
      KernelTimer t("score_folded", s);
      e = launch_gemm_tc(kEpiScoresFolded, a, folded_op, TmaOperand{nullptr, 0, 0, 0},
                         TmaOperand{xh, N, d, d}, TmaOperand{nullptr, 0, 0, 0}, max_m, max_r, s);
    } else {
      KernelTimer t("score", s);
      e = run_gemm(dt, kEpiScores, a, TmaOperand{mem->keys, mem->total, d, d},
                   TmaOperand{nullptr, 0, 0, 0}, TmaOperand{q, N, d, d},
                   TmaOperand{q_lo, N, d, d}, max_m, max_r, s);
    }
    if (e != cudaSuccess) return cuda_fail(e, "score");
  }

  // (4) softmax, cumulative-mass cardinality, selected set, renormalised weights;
  // (5) r = sum alpha u; with the projected values, also
  // (6) [a_f | a_g] = SiLU(G_h + sum alpha p + [b_f1 | b_g1])
  if (alpha_path) {
    // the selection writes the weights as dense bf16 hi / lo rows; the
    // readout, when asked for, gathers the values row by row
    void* alpha_hi = ws + L.alpha_hi;
    void* alpha_lo = ws + L.alpha_lo;
    { KernelTimer t("select", s);
      e = launch_select(scores, tab, N, mem->orig_index, rho, k_min, k_max, max_m, gate_rows,
                        counts, indices, readout ? sel_pos : nullptr, readout ? sel_w : nullptr,
                        readout ? sel_cnt : nullptr, s, alpha_hi, alpha_lo, mem->proj_ld); }
    if (e != cudaSuccess) return cuda_fail(e, "select");
    if (readout != nullptr) {
      { KernelTimer t("readout", s);
        e = launch_readout(dt, mem->values, sel_cnt, sel_pos, sel_w, N, k_max, d, readout, r_lo, s); }
      if (e != cudaSuccess) return cuda_fail(e, "readout");
    }
    // [a_f | a_g] = SiLU(G_h + alpha P + [b_f1 | b_g1]): per image, the
    // weights' hi / lo rows against the image's transposed projected values
    init_args(a);
    a.k_total = mem->proj_ld; a.b_split = mem->proj_ld;
    a.A0 = mem->projT; a.lda0 = mem->proj_ld;
    a.B0 = alpha_hi; a.B1 = alpha_lo; a.ldb0 = mem->proj_ld; a.ldb1 = mem->proj_ld;
    a.epi_split = H;
    a.out0 = act; a.ldc = 2 * H;
    a.bias0 = p->b_f1; a.bias1 = p->b_g1;
    a.add_in = gh; a.ldc2 = 2 * H;
    a.err = err;
    int g = 0, max_rows = 0;
    for (int b = 0; b < mem->B; ++b) {
      const int r = row_offsets[b + 1] - row_offsets[b];
      if (r == 0) continue;
      a.groups[g++] = GemmGroup{b * 2 * H, 2 * H, row_offsets[b], r, 0};
      max_rows = std::max(max_rows, r);
    }
    a.ngroups = g;
    { KernelTimer t("act_gemm", s);
      e = launch_gemm_tc(kEpiAct, a, TmaOperand{mem->projT, (long long)mem->B * 2 * H, mem->proj_ld,
                                                mem->proj_ld},
                         TmaOperand{nullptr, 0, 0, 0}, TmaOperand{alpha_hi, N, mem->proj_ld, mem->proj_ld},
                         TmaOperand{alpha_lo, N, mem->proj_ld, mem->proj_ld}, 2 * H, max_rows, s); }
    if (e != cudaSuccess) return cuda_fail(e, "act_gemm");
  } else if (use_proj) {
    { KernelTimer t("select_fuse", s);
      e = launch_select_gather(dt, scores, tab, N, mem->orig_index, rho, k_min, k_max, max_m,
                               gate_rows, counts, indices, mem->values, d, readout, nullptr,
                               mem->proj, H, gh, p->b_f1, p->b_g1, act, err, s,
                               (long long)mem->total * 2 * H * 2); }
    if (e != cudaSuccess) return cuda_fail(e, "select_fuse");
  } else {
    if (select_readout_fits(max_m, k_max)) {
      { KernelTimer t("select_readout", s);
        e = launch_select_gather(dt, scores, tab, N, mem->orig_index, rho, k_min, k_max, max_m,
                                 gate_rows, counts, indices, mem->values, d, readout, r_lo,
                                 nullptr, H, nullptr, nullptr, nullptr, nullptr, err, s); }
      if (e != cudaSuccess) return cuda_fail(e, "select_readout");
    } else {
      { KernelTimer t("select", s);
        e = launch_select(scores, tab, N, mem->orig_index, rho, k_min, k_max, max_m, gate_rows,
                          counts, indices, sel_pos, sel_w, sel_cnt, s); }
      if (e != cudaSuccess) return cuda_fail(e, "select");
      { KernelTimer t("readout", s);
        e = launch_readout(dt, mem->values, sel_cnt, sel_pos, sel_w, N, k_max, d, readout, r_lo, s); }
      if (e != cudaSuccess) return cuda_fail(e, "readout");
    }

    // (6) [a_f | a_g] = SiLU([h; r] [W_f1 | W_g1]^T + [b_f1 | b_g1])
    init_args(a);
    a.k_total = 2 * d;
    a.a_split = H;
    a.b_split = d;
    a.A0 = p->W_f1; a.A1 = p->W_g1; a.lda0 = 2 * d; a.lda1 = 2 * d;
    a.B0 = h; a.B1 = r_lo; a.ldb0 = d; a.ldb1 = d;
    a.epi_split = H;
    a.out0 = act; a.ldc = 2 * H;
    a.bias0 = p->b_f1; a.bias1 = p->b_g1;
    a.err = err;
    a.ngroups = 1;
    a.groups[0] = GemmGroup{0, 2 * H, 0, N, 0};
    { KernelTimer t("fuse_hidden", s);
      e = run_gemm(dt, kEpiBiasSilu, a, TmaOperand{p->W_f1, H, 2 * d, 2 * d},
                   TmaOperand{p->W_g1, H, 2 * d, 2 * d}, TmaOperand{h, N, d, d},
                   TmaOperand{r_lo, N, d, d}, 2 * H, N, s); }
    if (e != cudaSuccess) return cuda_fail(e, "fuse_hidden");
  }

  // (7) c = a_f W_f2^T + b_f2
  init_args(a);
  a.k_total = H; a.b_split = H;
  a.A0 = p->W_f2; a.lda0 = H;
  a.B0 = act; a.ldb0 = 2 * H;
  a.out0 = cbuf; a.ldc = d;
  a.bias0 = p->b_f2;
  a.err = err;
  a.ngroups = 1;
  a.groups[0] = GemmGroup{0, d, 0, N, 0};
  { KernelTimer t("fuse_out", s);
    e = run_gemm(dt, kEpiBiasF32, a, TmaOperand{p->W_f2, d, H, H}, TmaOperand{nullptr, 0, 0, 0},
                 TmaOperand{act, N, H, 2 * H}, TmaOperand{nullptr, 0, 0, 0}, d, N, s); }
  if (e != cudaSuccess) return cuda_fail(e, "fuse_out");

  // (8) g = sigma(a_g w_g2 + b_g2); h_hat = RMSNorm(h + g c); rows past the
  // depth gate: h_hat = h
  { KernelTimer t("finalize", s);
    e = launch_finalize(dt, h, cbuf, act, H, d, p->w_g2, p->b_g2, p->rms_gamma, p->rms_eps, N,
                        gate_rows, h_out, gate, s); }
  if (e != cudaSuccess) return cuda_fail(e, "finalize");
  return FOVEA_OK;
}

FOVEA_API fovea_status fovea_lm_head_topk(const void* W_LM, int vocab, int d_model, int dtype,
                                          const void* h_hat, int N, int k_c, float* logits,
                                          int32_t* top_idx, float* top_val, void* workspace,
                                          size_t workspace_bytes, void* stream) {
  g_last_error.clear();
  if (dtype != FOVEA_BF16 && dtype != FOVEA_FP32)
    return fail(FOVEA_ERR_INVALID_ARG, "dtype %d is neither FOVEA_BF16 nor FOVEA_FP32", dtype);
  if (d_model <= 0 || d_model % 64 != 0 || d_model > FOVEA_MAX_D)
    return fail(FOVEA_ERR_INVALID_ARG, "d_model %d must be a positive multiple of 64 (<= %d)",
                d_model, FOVEA_MAX_D);
  if (N < 0) return fail(FOVEA_ERR_INVALID_ARG, "N = %d < 0", N);
  if (k_c < 1 || k_c > FOVEA_MAX_KC)
    return fail(FOVEA_ERR_INVALID_ARG, "k_c = %d must lie in [1, %d]", k_c, FOVEA_MAX_KC);
  if (vocab < k_c) return fail(FOVEA_ERR_INVALID_ARG, "vocab %d < k_c %d", vocab, k_c);
  NEED_PTR(W_LM, "W_LM");
  NEED_PTR(h_hat, "h_hat");
  if (top_idx == nullptr) return fail(FOVEA_ERR_INVALID_ARG, "top_idx is NULL");
  if (workspace == nullptr || (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0)
    return fail(FOVEA_ERR_INVALID_ARG, "workspace is NULL or not 256-byte aligned");
  if (dtype != FOVEA_BF16)
    return fail(FOVEA_ERR_UNSUPPORTED, "the LM head runs on bf16 weights and states only");
  if (N == 0) return FOVEA_OK;
  const int slots = lm_head_slots(vocab, d_model, N);
  const size_t need = lm_head_ws_bytes(N, slots, k_c);
  if (workspace_bytes < need)
    return fail(FOVEA_ERR_INVALID_ARG, "workspace has %zu bytes, needs %zu "
                "(fovea_lm_head_workspace_size)", workspace_bytes, need);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // z = h_hat W_LM^T: W_LM [vocab, d] is the feature operand, streamed once;
  // every column goes to the fp32 logits, and the epilogue keeps each row's
  // k_c largest of every tile as candidates after the header
  unsigned long long* cand = reinterpret_cast<unsigned long long*>(
      static_cast<uint8_t*>(workspace) + kWsHeaderBytes);
  static thread_local GemmArgs a;
  init_args(a);
  a.k_total = d_model; a.b_split = d_model;
  a.epi_split = 0;
  a.out2 = logits; a.ldc2 = vocab;
  a.cand = cand; a.cand_k = k_c; a.cand_ld = (long long)slots * k_c;
  a.err = static_cast<int*>(workspace);
  a.ngroups = 1;
  a.groups[0] = GemmGroup{0, vocab, 0, N, 0};
  cudaError_t e;
  { KernelTimer t("lm_head", s);
    e = launch_gemm_tc(kEpiLogits, a, TmaOperand{W_LM, vocab, d_model, d_model},
                       TmaOperand{nullptr, 0, 0, 0}, TmaOperand{h_hat, N, d_model, d_model},
                       TmaOperand{nullptr, 0, 0, 0}, vocab, N, s); }
  if (e != cudaSuccess) return cuda_fail(e, "lm_head");
  { KernelTimer t("merge_candidates", s);
    e = launch_merge_candidates(cand, N, slots, k_c, top_idx, top_val, s); }
  if (e != cudaSuccess) return cuda_fail(e, "merge_candidates");
  return FOVEA_OK;
}

FOVEA_API fovea_status fovea_lm_head_workspace_size(int vocab, int d_model, int N, int k_c,
                                                    size_t* bytes) {
  g_last_error.clear();
  if (bytes == nullptr) return fail(FOVEA_ERR_INVALID_ARG, "bytes is NULL");
  if (d_model <= 0 || d_model % 64 != 0 || d_model > FOVEA_MAX_D)
    return fail(FOVEA_ERR_INVALID_ARG, "d_model %d must be a positive multiple of 64 (<= %d)",
                d_model, FOVEA_MAX_D);
  if (N < 0) return fail(FOVEA_ERR_INVALID_ARG, "N = %d < 0", N);
  if (k_c < 1 || k_c > FOVEA_MAX_KC)
    return fail(FOVEA_ERR_INVALID_ARG, "k_c = %d must lie in [1, %d]", k_c, FOVEA_MAX_KC);
  if (vocab < k_c) return fail(FOVEA_ERR_INVALID_ARG, "vocab %d < k_c %d", vocab, k_c);
  *bytes = N == 0 ? kWsHeaderBytes : lm_head_ws_bytes(N, lm_head_slots(vocab, d_model, N), k_c);
  return FOVEA_OK;
}

FOVEA_API fovea_status fovea_timing_enable(int enable) {
  std::lock_guard<std::mutex> lk(g_tmu);
  for (auto& r : g_recs) {
    g_free_events.push_back(r.start);
    g_free_events.push_back(r.stop);
  }
  g_recs.clear();
  g_timing = enable != 0;
  return FOVEA_OK;
}

FOVEA_API int fovea_timing_read(const char** names, double* total_ms, int* launches,
                                int capacity) {
  std::lock_guard<std::mutex> lk(g_tmu);
  std::vector<const char*> nm;
  std::vector<double> ms;
  std::vector<int> cnt;
  for (auto& r : g_recs) {
    if (cudaEventSynchronize(r.stop) != cudaSuccess) continue;
    float t = 0.0f;
    if (cudaEventElapsedTime(&t, r.start, r.stop) != cudaSuccess) continue;
    size_t i = 0;
    while (i < nm.size() && strcmp(nm[i], r.name) != 0) ++i;
    if (i == nm.size()) {
      nm.push_back(r.name);
      ms.push_back(0.0);
      cnt.push_back(0);
    }
    ms[i] += t;
    cnt[i] += 1;
  }
  for (size_t i = 0; i < nm.size() && (int)i < capacity; ++i) {
    if (names) names[i] = nm[i];
    if (total_ms) total_ms[i] = ms[i];
    if (launches) launches[i] = cnt[i];
  }
  return (int)nm.size();
}

}  // extern "C"
