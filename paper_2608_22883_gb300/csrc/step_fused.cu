// Persistent step kernel: one draft step of the FOVEA path (query equation,
// scores, cumulative-mass selection, renormalised readout, fusion layers,
// gated residual and RMSNorm: Sec. 3 and the appendix's correction module)
// as ONE cooperative launch of one CTA per SM, instead of eight kernels.
//
// Why: at the 7B-shaped workload a step moves ~65 MB and is bound by HBM at
// ~10 us, but eight dependent launches cost far more than that in launch
// ramps, tails and split-K bookkeeping.  Here the phases are separated by
// software grid barriers (~1.2 us each on GB300), and the weight streams of
// later phases are requested while earlier phases compute.
//
// Roles (320 threads):
//   warp 0, lane 0   TMA producer.  Walks the k-blocks of every GEMM unit of
//                    every phase in order, keeping a 3-stage shared-memory
//                    ring full.  The feature operand (weights, keys) never
//                    depends on earlier phases, so it is loaded up to three
//                    stages ahead of the row operand, which waits for the
//                    grid barrier that publishes it.  Once the query
//                    projection's weights are requested it prefetches this
//                    CTA's share of the later phases' weights (and the memory
//                    values when selection is dense) into L2.
//   warp 1           owns the tensor memory (two 256-column accumulators);
//                    lane 0 issues the tcgen05 MMAs of each unit.
//   warps 2..9       256 worker threads: LayerNorm, the GEMM epilogues
//                    (accumulator -> fp32 partial tiles), the split-K
//                    reductions, selection, readout and the final RMSNorm.
//
// GEMM units.  A GEMM phase C = R . F^T (rows R = draft states, features F =
// weight rows or memory keys) is cut into units (group, row tile of 128,
// feature tile of bn, K split s); unit u runs on CTA u mod G.  Every unit
// writes its fp32 partial tile row-major to global scratch (staged through
// shared memory so each store instruction writes whole 128-byte lines);
// consumers sum the S partials of an output in split order, so results do
// not depend on timing.  The scores' partials are summed by the selection
// phase and the last fusion layer's by the RMSNorm phase directly.
//
// Grid barriers (one arrival counter each; barrier k is passed when its
// counter reaches G): 1 LN done, 2 query partials, 3 q, 4 score partials,
// 5 selection, 6 readout, 7 fusion-1 partials, 8 activations, 9 fusion-2
// partials.  A CTA with no work in a phase arrives at the next barrier early,
// which is why the barriers do not share one running count.  Every wait is
// bounded (~2 s) and observes an abort word, so a failure unwinds the whole
// grid with kErrTimeout set.  The last CTA to leave resets the counters.
#include "rowmath.cuh"
#include "select_core.cuh"
#include "step_fused.h"
#include "tc_ptx.cuh"

namespace fovea {
namespace fused {

using namespace tc;
typedef __nv_bfloat16 bf16;

constexpr int kThreads = 320;
constexpr int kWorkers = 256;
constexpr int kStages = 3;
constexpr int kRTile = 128 * 64 * 2;          // one row-operand tile (128 rows x 64 bf16)
constexpr int kStageBytes = 48 * 1024;
constexpr int kRingBytes = kStages * kStageBytes;
constexpr int kTmemCols = 512;                // two accumulators of 256 columns
constexpr uint64_t kWaitNs = 2000000000ull;
// words of a.sync: [k] arrivals at grid barrier k (1..kBarriers), then the
// exit counter and the abort word
constexpr int kBarriers = 9;
constexpr int kSyncExit = kBarriers + 1;
constexpr int kSyncAbort = kBarriers + 2;

// scratch region (bytes), reused by the worker phases one after another
constexpr int kScrTranspose = 8 * 4096;       // per worker warp: 32 x 32 fp32
constexpr int kScrUs = 48 * 1024;             // readout: staged value columns
constexpr int kScrSel = 16 * 1024;            // readout: staged positions / weights (each)
constexpr int kScrCnt = 1024;                 // readout: staged counts
constexpr int kScrBytes = kScrUs + 2 * kScrSel + kScrCnt;
constexpr int kBarBytes = 256;
constexpr int kSmemBytes = 1024 + kRingBytes + kScrBytes + kBarBytes;
static_assert(kScrBytes >= kScrTranspose, "scratch");
static_assert(kSmemBytes <= 232448, "shared memory");

// ---------------------------------------------------------------------------
// small helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ void wsync() { asm volatile("bar.sync 1, 256;" ::: "memory"); }
__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}
__device__ __forceinline__ void red_release_add(int* p, int v) {
  asm volatile("red.release.gpu.global.add.s32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void prefetch_l2(const void* p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}
__device__ __forceinline__ uint32_t make_idesc(int bn) {
  // kind::f16: D fp32, A and B bf16, both K-major, N >> 3, M = 128 >> 4
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(bn >> 3) << 17) |
         ((uint32_t)(128 >> 4) << 24);
}
__device__ __forceinline__ float worker_sum(float v, float* red, int wtid) {
  const int lane = wtid & 31, warp = wtid >> 5;
  v = warp_sum(v);
  wsync();
  if (lane == 0) red[warp] = v;
  wsync();
  const float t = lane < kWorkers / 32 ? red[lane] : 0.0f;
  return warp_sum(t);
}

// Spin (bounded) until all G CTAs arrived at grid barrier k; false on
// timeout or abort.  One thread calls it.
__device__ bool spin_barrier(const FusedArgs& a, int k) {
  const int* ctr = a.sync + k;
  const int G = (int)gridDim.x;
  if (ld_acquire_gpu(ctr) >= G) return true;
  const uint64_t t0 = globaltimer_ns();
  while (true) {
    // poll with a short sleep: every SM polls the same line
    for (int i = 0; i < 32; ++i) {
      __nanosleep(40);
      if (ld_acquire_gpu(ctr) >= G) return true;
    }
    if (ld_acquire_gpu(a.sync + kSyncAbort) != 0) return false;
    if (globaltimer_ns() - t0 > kWaitNs) {
      atomicOr(a.err, kErrTimeout);
      atomicExch(a.sync + kSyncAbort, 1);
      return false;
    }
  }
}

struct WorkerCtx {
  int wtid, lane, wwarp;     // worker thread index, lane, worker warp (0..7)
  volatile int* s_ok;        // shared: 0 once this CTA saw an abort
};

// Worker arrival at grid barrier k.
__device__ __forceinline__ void grid_arrive(const FusedArgs& a, const WorkerCtx& w, int k,
                                            bool tma_consumed) {
  if (tma_consumed) fence_proxy_async_global();   // generic writes read by TMA later
  wsync();
  if (w.wtid == 0) {
    __threadfence();
    red_release_add(a.sync + k, 1);
  }
}
// Worker wait for grid barrier k; false after an abort.
__device__ __forceinline__ bool grid_wait(const FusedArgs& a, const WorkerCtx& w, int k) {
  if (w.wtid == 0 && *w.s_ok) {
    if (!spin_barrier(a, k)) *w.s_ok = 0;
  }
  wsync();
  return *w.s_ok != 0;
}

struct UnitPos {
  int g, rt, ft, s;
};
__device__ __forceinline__ UnitPos decode_unit(const PhaseGemm& p, int u) {
  int g = 0;
  while (g + 1 < p.ngroups && p.unit0[g + 1] <= u) ++g;
  const int local = u - p.unit0[g];
  UnitPos r;
  r.g = g;
  r.s = local % p.splits;
  const int tile = local / p.splits;
  r.ft = tile % p.ftiles[g];
  r.rt = tile / p.ftiles[g];
  return r;
}
__device__ __forceinline__ float* partial_tile(const FusedArgs& a, const PhaseGemm& p, int u) {
  return a.partials + (long long)u * 128 * p.bn;
}

// Sum in split order of the S partial float4 at base + s * stride (floats),
// with the loads of up to 16 splits in flight together.
__device__ __forceinline__ float4 sum_splits(const float* base, long long stride, int S) {
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int s0 = 0; s0 < S; s0 += 16) {
    float4 t[16];
#pragma unroll
    for (int i = 0; i < 16; ++i)
      if (s0 + i < S) t[i] = __ldcg(reinterpret_cast<const float4*>(base + (s0 + i) * stride));
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      if (s0 + i < S) {
        if (s0 + i == 0) {
          acc = t[i];
        } else {
          acc.x += t[i].x;
          acc.y += t[i].y;
          acc.z += t[i].z;
          acc.w += t[i].w;
        }
      }
    }
  }
  return acc;
}

// k-block cursor over (phase, unit of this CTA, k-block)
struct Cursor {
  int phase, u, kb, kb_hi;
};
__device__ __forceinline__ void cursor_settle(const FusedArgs& a, Cursor& c) {
  while (c.phase < kPhases && c.u >= a.g[c.phase].units) {
    ++c.phase;
    c.u = blockIdx.x;
  }
  if (c.phase < kPhases) {
    const PhaseGemm& p = a.g[c.phase];
    const int s = (c.u - p.unit0[decode_unit(p, c.u).g]) % p.splits;
    c.kb = (int)((long long)s * p.kb_total / p.splits);
    c.kb_hi = (int)((long long)(s + 1) * p.kb_total / p.splits);
  }
}
__device__ __forceinline__ void cursor_next(const FusedArgs& a, Cursor& c) {
  if (++c.kb >= c.kb_hi) {
    c.u += gridDim.x;
    cursor_settle(a, c);
  }
}

// ---------------------------------------------------------------------------
// producer (one thread)
// ---------------------------------------------------------------------------
__device__ void issue_l2_prefetch(const FusedArgs& a) {
  const int G = gridDim.x;
  for (int i = 0; i < a.n_prefetch; ++i) {
    const long long bytes = a.pf_bytes[i];
    long long chunk = (bytes + G - 1) / G;
    chunk = (chunk + 15) & ~15ll;
    long long beg = chunk * blockIdx.x;
    const long long end = min(bytes, beg + chunk);
    const uint8_t* base = static_cast<const uint8_t*>(a.pf_ptr[i]);
    while (beg < end) {
      const long long n = min(end - beg, 32768ll) & ~15ll;
      if (n <= 0) break;
      prefetch_l2(base + beg, (uint32_t)n);
      beg += n;
    }
  }
}

__device__ void producer(const FusedArgs& a, const FusedMaps& maps, uint8_t* ring, uint64_t* full,
                         uint64_t* empty) {
  volatile int* abort_word = a.sync + kSyncAbort;
  Cursor cf{0, (int)blockIdx.x, 0, 0}, cr{0, (int)blockIdx.x, 0, 0};
  cursor_settle(a, cf);
  cursor_settle(a, cr);
  long long it_f = 0, it_r = 0;
  int passed = 0;
  bool ok = true, prefetched = a.n_prefetch == 0;
  while (ok && cr.phase < kPhases) {
    // feature loads, up to kStages k-blocks ahead of the row loads
    while (cf.phase < kPhases && it_f < it_r + kStages) {
      if (!prefetched && cf.phase > 0) {
        issue_l2_prefetch(a);
        prefetched = true;
      }
      const int st = (int)(it_f % kStages);
      if (it_f >= kStages &&
          !mbar_wait(&empty[st], (uint32_t)((it_f / kStages) & 1) ^ 1u, abort_word)) {
        ok = false;
        break;
      }
      const PhaseGemm& p = a.g[cf.phase];
      const UnitPos up = decode_unit(p, cf.u);
      const int rbytes = p.dual ? 2 * kRTile : kRTile;
      uint8_t* stage = ring + st * kStageBytes;
      mbar_expect_tx(&full[st], (uint32_t)((p.dual ? 2 : 1) * p.rbox * 128 + p.bn * 128));
      const int f = up.ft * p.bn;
      const bool second = f >= p.f_split;
      tma_load_2d(stage + rbytes, &maps.m[second ? p.fmap1 : p.fmap0], &full[st], cf.kb * 64,
                  second ? f - p.f_split : p.a_row0[up.g] + f);
      ++it_f;
      cursor_next(a, cf);
    }
    if (!ok) break;
    // row loads of k-block it_r
    const PhaseGemm& p = a.g[cr.phase];
    const UnitPos up = decode_unit(p, cr.u);
    const int st = (int)(it_r % kStages);
    uint8_t* stage = ring + st * kStageBytes;
    const int ry = p.b_row0[up.g] + up.rt * 128;
    const bool r_second = !p.dual && cr.kb >= p.r_split_kb;
    const int need = r_second ? p.wait_r1 : p.wait_r0;
    if (need > passed) {
      if (!spin_barrier(a, need)) {
        ok = false;
        break;
      }
      fence_proxy_async_global();
      passed = need;
    }
    if (p.dual) {
      tma_load_2d(stage, &maps.m[p.rmap0], &full[st], cr.kb * 64, ry);
      tma_load_2d(stage + kRTile, &maps.m[p.rmap1], &full[st], cr.kb * 64, ry);
    } else if (r_second) {
      tma_load_2d(stage, &maps.m[p.rmap1], &full[st], (cr.kb - p.r_split_kb) * 64, ry);
    } else {
      tma_load_2d(stage, &maps.m[p.rmap0], &full[st], cr.kb * 64, ry);
    }
    ++it_r;
    cursor_next(a, cr);
  }
  if (!ok) {
    atomicOr(a.err, kErrTimeout);
    atomicExch(a.sync + kSyncAbort, 1);
    // complete the stages whose row loads were not issued (in-bounds loads of
    // whatever the buffers hold), then let every copy in flight land
    while (it_r < it_f) {
      const PhaseGemm& p = a.g[cr.phase];
      const UnitPos up = decode_unit(p, cr.u);
      const int st = (int)(it_r % kStages);
      uint8_t* stage = ring + st * kStageBytes;
      const int ry = p.b_row0[up.g] + up.rt * 128;
      if (p.dual) {
        tma_load_2d(stage, &maps.m[p.rmap0], &full[st], cr.kb * 64, ry);
        tma_load_2d(stage + kRTile, &maps.m[p.rmap1], &full[st], cr.kb * 64, ry);
      } else if (cr.kb >= p.r_split_kb) {
        tma_load_2d(stage, &maps.m[p.rmap1], &full[st], (cr.kb - p.r_split_kb) * 64, ry);
      } else {
        tma_load_2d(stage, &maps.m[p.rmap0], &full[st], cr.kb * 64, ry);
      }
      ++it_r;
      cursor_next(a, cr);
    }
  }
  // every copy this thread issued has landed before the CTA can leave (after
  // an abort the MMA thread no longer consumes the stages)
  for (long long i = it_f > kStages ? it_f - kStages : 0; i < it_f; ++i)
    mbar_wait(&full[i % kStages], (uint32_t)((i / kStages) & 1), nullptr, 20000000ull);
}

// ---------------------------------------------------------------------------
// MMA issuer (one thread)
// ---------------------------------------------------------------------------
__device__ void mma_issuer(const FusedArgs& a, uint8_t* ring, uint64_t* full, uint64_t* empty,
                           uint64_t* tfull, uint64_t* tempty, uint64_t* done, uint32_t tmem_base) {
  volatile int* abort_word = a.sync + kSyncAbort;
  long long it = 0;
  int uc = 0;
  bool ok = true;
  for (int ph = 0; ph < kPhases && ok; ++ph) {
    const PhaseGemm& p = a.g[ph];
    const uint32_t idesc = make_idesc(p.bn);
    const int rbytes = p.dual ? 2 * kRTile : kRTile;
    for (int u = blockIdx.x; u < p.units && ok; u += gridDim.x) {
      const UnitPos up = decode_unit(p, u);
      const int kb_lo = (int)((long long)up.s * p.kb_total / p.splits);
      const int kb_hi = (int)((long long)(up.s + 1) * p.kb_total / p.splits);
      const int buf = uc & 1, use = uc >> 1;
      if (use >= 1 && !mbar_wait(&tempty[buf], (uint32_t)((use - 1) & 1), abort_word)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t d_tmem = tmem_base + (uint32_t)(buf * 256);
      for (int kb = kb_lo; kb < kb_hi; ++kb, ++it) {
        const int st = (int)(it % kStages);
        if (!mbar_wait(&full[st], (uint32_t)((it / kStages) & 1), abort_word)) {
          ok = false;
          break;
        }
        // (no tcgen05 fence per k-block: the stage is published by TMA through
        // the mbarrier, and a fence would serialise the MMAs)
        uint8_t* stage = ring + st * kStageBytes;
        const uint64_t adesc = sw128_desc(smem_u32(stage));
        const uint64_t adesc_lo = sw128_desc(smem_u32(stage + kRTile));
        const uint64_t bdesc = sw128_desc(smem_u32(stage + rbytes));
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          umma_bf16(d_tmem, adesc + (uint64_t)(2 * k), bdesc + (uint64_t)(2 * k), idesc,
                    (kb > kb_lo || k > 0) ? 1u : 0u);
          if (p.dual)
            umma_bf16(d_tmem, adesc_lo + (uint64_t)(2 * k), bdesc + (uint64_t)(2 * k), idesc, 1u);
        }
        umma_commit(&empty[st]);
      }
      if (!ok) break;
      umma_commit(&tfull[buf]);
      ++uc;
    }
  }
  if (!ok) {
    atomicOr(a.err, kErrTimeout);
    atomicExch(a.sync + kSyncAbort, 1);
  }
  // every MMA issued by this thread has completed before tensor memory is freed
  umma_commit(done);
  mbar_wait(done, 0, nullptr, 100000000ull);
}

// ---------------------------------------------------------------------------
// worker phases
// ---------------------------------------------------------------------------

// LN_h(h_n) + E_dep[l_n] -> x (bf16), one row per CTA iteration (query
// equation).  The row stays in registers between the statistics and the
// affine map; gamma, beta and the depth embedding are loaded per vector in
// the second pass, so few values are live at once.  Four independent
// double-float accumulators per sum keep the dependency chains short.
__device__ void phase_ln(const FusedArgs& a, const WorkerCtx& w, uint8_t* scr) {
  constexpr int MV = FOVEA_MAX_D / 8 / kWorkers;     // 16-byte vectors per thread
  dfloat* red = reinterpret_cast<dfloat*>(scr);      // [2][8], then mean, rstd
  const int d = a.d, nvec = d / 8;
  for (int n = blockIdx.x; n < a.N; n += gridDim.x) {
    int dep = a.depth[n];
    if (dep < 0 || dep > a.max_depth) {
      if (w.wtid == 0) atomicOr(a.err, kErrDepth);
      dep = 0;
    }
    const bf16* xr = a.h + (long long)n * d;
    const bf16* er = a.E + (long long)dep * d;
    float xv[MV][8];
#pragma unroll
    for (int j = 0; j < MV; ++j) {
      const int vi = w.wtid + j * kWorkers;
      if (vi < nvec) ln_load<bf16>(xr + vi * 8, xv[j]);
    }
    dfloat s1, s2;
    {
      dfloat a1[4], a2[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) a1[q] = a2[q] = dfloat{0.0f, 0.0f};
#pragma unroll
      for (int j = 0; j < MV; ++j) {
        if (w.wtid + j * kWorkers < nvec) {
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            a1[i & 3] = df_add_f(a1[i & 3], xv[j][i]);
            a2[i & 3] = df_add(a2[i & 3], df_two_prod(xv[j][i], xv[j][i]));
          }
        }
      }
      s1 = df_add(df_add(a1[0], a1[1]), df_add(a1[2], a1[3]));
      s2 = df_add(df_add(a2[0], a2[1]), df_add(a2[2], a2[3]));
    }
    s1 = warp_sum_df(s1);
    s2 = warp_sum_df(s2);
    wsync();                     // the previous row's readers of red are done
    if (w.lane == 0) {
      red[w.wwarp] = s1;
      red[8 + w.wwarp] = s2;
    }
    wsync();
    if (w.wwarp == 0) {
      dfloat t1 = w.lane < 8 ? red[w.lane] : dfloat{0.0f, 0.0f};
      dfloat t2 = w.lane < 8 ? red[8 + w.lane] : dfloat{0.0f, 0.0f};
      t1 = warp_sum_df(t1);
      t2 = warp_sum_df(t2);
      if (w.lane == 0) {
        const dfloat mean = df_div_f(t1, (float)d);
        const dfloat ex2 = df_div_f(t2, (float)d);
        const dfloat var = df_add(ex2, df_mul(dfloat{-mean.hi, -mean.lo}, mean));
        red[16] = mean;
        red[17] = df_rsqrt(df_add_f(var, a.ln_eps));
      }
    }
    wsync();
    const dfloat neg_mean = {-red[16].hi, -red[16].lo};
    const dfloat rstd = red[17];
    bf16* o = a.x + (long long)n * d;
#pragma unroll
    for (int j = 0; j < MV; ++j) {
      const int vi = w.wtid + j * kWorkers;
      if (vi < nvec) {
        float gv[8], bv[8], ev[8];
        ln_load<bf16>(a.ln_gamma + vi * 8, gv);
        ln_load<bf16>(a.ln_beta + vi * 8, bv);
        ln_load<bf16>(er + vi * 8, ev);
        bf16 res[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          dfloat y = df_mul(df_add_f(neg_mean, xv[j][i]), rstd);
          y = df_add_f(df_mul_f(y, gv[i]), bv[i]);
          y = df_add_f(y, ev[i]);
          res[i] = df_to_bf16(y);
        }
        *reinterpret_cast<uint4*>(o + vi * 8) = *reinterpret_cast<const uint4*>(res);
      }
    }
  }
}

// Accumulators of this CTA's units of one GEMM phase -> fp32 partial tiles,
// row-major [128][bn].  Worker warp ww reads accumulator lanes (rows)
// 32 (hw_warp % 4) .. +31 and half of the columns; each 32 x 32 block is
// transposed through shared memory so a store instruction writes 4 rows x
// 128 contiguous bytes.
__device__ void phase_epilogue(const FusedArgs& a, const WorkerCtx& w, int ph, uint8_t* scr,
                               uint64_t* tfull, uint64_t* tempty, uint32_t tmem_base, int& uc) {
  const PhaseGemm& p = a.g[ph];
  const int hw_warp = w.wwarp + 2;
  const int quarter = hw_warp & 3;
  const int half = w.wwarp >> 2;
  float* tb = reinterpret_cast<float*>(scr + w.wwarp * 4096);     // [32][32], 16-byte chunks swizzled
  for (int u = blockIdx.x; u < p.units; u += gridDim.x) {
    const UnitPos up = decode_unit(p, u);
    const int buf = uc & 1, use = uc >> 1;
    ++uc;
    bool ok = *w.s_ok != 0;
    if (ok) ok = mbar_wait(&tfull[buf], (uint32_t)(use & 1), a.sync + kSyncAbort);
    ok = __all_sync(0xffffffffu, ok);
    if (!ok && w.lane == 0) {
      atomicOr(a.err, kErrTimeout);
      atomicExch(a.sync + kSyncAbort, 1);
      *w.s_ok = 0;
    }
    tc_fence_after();
    const int rows_real = min(128, p.n[up.g] - up.rt * 128);
    const int cols_real = min(p.bn, p.m[up.g] - up.ft * p.bn);
    const int row0 = quarter * 32;
    if (ok && row0 < rows_real) {
      float* P = partial_tile(a, p, u);
      const int hcols = p.bn >> 1;
      for (int c = 0; c < hcols; c += 32) {
        const int col0 = half * hcols + c;
        if (col0 >= cols_real) break;                    // warp-uniform
        float v[32];
        tmem_ld32(tmem_base + (uint32_t)(buf * 256) + ((uint32_t)row0 << 16) + (uint32_t)col0, v);
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          const int pq = q ^ (w.lane & 7);
          *reinterpret_cast<float4*>(tb + w.lane * 32 + pq * 4) =
              make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
        }
        __syncwarp();
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int r = 4 * i + (w.lane >> 3);
          const int q = w.lane & 7;
          const float4 val = *reinterpret_cast<const float4*>(tb + r * 32 + ((q ^ (r & 7)) * 4));
          if (row0 + r < rows_real)
            __stcg(reinterpret_cast<float4*>(P + (long long)(row0 + r) * p.bn + col0 + 4 * q), val);
        }
        __syncwarp();
      }
    }
    tc_fence_before();
    __syncwarp();
    if (w.lane == 0) mbar_arrive(&tempty[buf]);
  }
}

// Split-K reduction of a row-operand-producing phase (query, fusion layer 1):
// thread item = (row, 4 consecutive features); the S partials are summed in
// split order, then the epilogue (q hi/lo, or bias + SiLU) is applied.
template <int PH>
__device__ void phase_reduce(const FusedArgs& a, const WorkerCtx& w) {
  const PhaseGemm& p = a.g[PH];
  const int F = p.m[0];
  const int q4 = F >> 2;
  const long long items = (long long)a.N * q4;
  const long long stride = (long long)gridDim.x * kWorkers;
  for (long long it = (long long)blockIdx.x * kWorkers + w.wtid; it < items; it += stride) {
    const int n = (int)(it / q4);
    const int c = (int)(it - (long long)n * q4) * 4;
    const int rt = n >> 7, rit = n & 127;
    const int ft = c / p.bn, j = c - ft * p.bn;
    const int u0 = p.unit0[0] + (rt * p.ftiles[0] + ft) * p.splits;
    const float4 acc = sum_splits(partial_tile(a, p, u0) + (long long)rit * p.bn + j,
                                  128ll * p.bn, p.splits);
    const float v[4] = {acc.x, acc.y, acc.z, acc.w};
    if constexpr (PH == kPhaseQuery) {
      bf16 hi[4], lo[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        hi[i] = __float2bfloat16_rn(v[i]);
        lo[i] = __float2bfloat16_rn(v[i] - __bfloat162float(hi[i]));
      }
      *reinterpret_cast<uint2*>(a.q_hi + (long long)n * F + c) = *reinterpret_cast<const uint2*>(hi);
      *reinterpret_cast<uint2*>(a.q_lo + (long long)n * F + c) = *reinterpret_cast<const uint2*>(lo);
    } else {
      bf16 out[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int col = c + i;
        const float bias = col < a.H ? __bfloat162float(a.b_f1[col]) : __bfloat162float(a.b_g1[col - a.H]);
        const float z = v[i] + bias;
        out[i] = __float2bfloat16_rn(z * sigmoidf_(z));
      }
      *reinterpret_cast<uint2*>(a.act + (long long)n * F + c) = *reinterpret_cast<const uint2*>(out);
    }
  }
}

struct WorkerSync {
  __device__ __forceinline__ void operator()() const { wsync(); }
};

// Scores of draft state n summed from the score phase's partial tiles (in
// split order) and scaled, then the cumulative-mass selection.
__device__ void phase_select(const FusedArgs& a, const WorkerCtx& w, uint8_t* scr) {
  SelectSmem& sm = *reinterpret_cast<SelectSmem*>(scr);
  float* s_sc = reinterpret_cast<float*>(scr + ((sizeof(SelectSmem) + 15) & ~(size_t)15));
  const PhaseGemm& p = a.g[kPhaseScore];
  SelectArgs sa{nullptr, a.orig_index, a.rho, a.k_min, a.k_max, a.counts, a.indices,
                a.sel_pos, a.sel_w, a.sel_cnt};
  for (int n = blockIdx.x; n < a.N; n += gridDim.x) {
    int b = 0;
    while (b + 1 < a.B && a.row_start[b + 1] <= n) ++b;
    const int M = a.mseq[b];
    const int g = a.seq_group[b];
    wsync();                      // the previous row's readers of sm / s_sc are done
    if (M == 0 || g < 0) {
      select_empty(sa, n, w.wtid);
      continue;
    }
    const int ln = n - a.row_start[b];
    const int rt = ln >> 7, rit = ln & 127;
    const float rs = a.row_scale ? a.row_scale[n] : 1.0f;
    const int q4 = (M + 3) >> 2;
    for (int q = w.wtid; q < q4; q += kWorkers) {
      const int i0 = q * 4;
      const int ft = i0 / p.bn, j = i0 - ft * p.bn;
      const int u0 = p.unit0[g] + (rt * p.ftiles[g] + ft) * p.splits;
      const float4 acc = sum_splits(partial_tile(a, p, u0) + (long long)rit * p.bn + j,
                                    128ll * p.bn, p.splits);
      const float v[4] = {acc.x, acc.y, acc.z, acc.w};
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        if (i0 + i < M) {
          float sc = v[i] * a.scale * rs;
          if (sc == 0.0f) sc = 0.0f;      // -0 -> +0 so equal scores get equal keys
          s_sc[i0 + i] = sc;
        }
      }
    }
    wsync();
    select_row(sa, n, M, a.key_off[b], s_sc, sm, w.wtid, WorkerSync{});
  }
}

// Readout r_n = sum_{t<K} alpha_t u_{pi(t)} (the alpha / r_n equation).  Item =
// (sequence, a column slice of W features): the slice of every value row of
// the sequence is staged in shared memory once (read from HBM / L2 once), so
// the K_n-fold reuse of a value row by the draft states is served on chip.
__device__ void phase_readout(const FusedArgs& a, const WorkerCtx& w, uint8_t* scr) {
  bf16* us = reinterpret_cast<bf16*>(scr);
  int* spos = reinterpret_cast<int*>(scr + kScrUs);
  float* sw = reinterpret_cast<float*>(scr + kScrUs + kScrSel);
  int* scnt = reinterpret_cast<int*>(scr + kScrUs + 2 * kScrSel);
  const int W = a.ro_w, QW = W >> 2;
  const int chunks = a.d / W;
  const int k_max = a.k_max;
  for (int item = blockIdx.x; item < a.ro_items; item += gridDim.x) {
    const int b = a.ro_seq[item / chunks];
    const int c0 = (item % chunks) * W;
    const int M = a.mseq[b];
    const int row0 = a.row_start[b], R = a.row_start[b + 1] - row0;
    const int koff = a.key_off[b];
    wsync();                          // the previous item's readers are done
    if (M > 0) {
      const int pieces = W >> 3;      // 16-byte pieces per value row slice
      const int tot = M * pieces;
      for (int i0 = w.wtid; i0 < tot; i0 += 8 * kWorkers) {
        uint4 v[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const int i = i0 + k * kWorkers;
          if (i < tot) {
            const int r = i / pieces, pc = i - r * pieces;
            v[k] = __ldg(reinterpret_cast<const uint4*>(a.U + (long long)(koff + r) * a.d + c0 + pc * 8));
          }
        }
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const int i = i0 + k * kWorkers;
          if (i < tot) {
            const int r = i / pieces, pc = i - r * pieces;
            *reinterpret_cast<uint4*>(us + r * W + pc * 8) = v[k];
          }
        }
      }
    }
    for (int rb = 0; rb < R; rb += a.ro_rows) {
      const int nb = min(a.ro_rows, R - rb);
      if (rb > 0) wsync();
      const int tot = nb * k_max;
      const long long g0 = (long long)(row0 + rb) * k_max;
      for (int i0 = w.wtid; i0 < tot; i0 += 8 * kWorkers) {
        int pv[8];
        float wv[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const int i = i0 + k * kWorkers;
          if (i < tot) {
            pv[k] = __ldcg(a.sel_pos + g0 + i);
            wv[k] = __ldcg(a.sel_w + g0 + i);
          }
        }
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const int i = i0 + k * kWorkers;
          if (i < tot) {
            spos[i] = pv[k] - koff;
            sw[i] = wv[k];
          }
        }
      }
      for (int i = w.wtid; i < nb; i += kWorkers) scnt[i] = __ldcg(a.sel_cnt + row0 + rb + i);
      wsync();
      const int rows_per_pass = kWorkers / QW;
      const int cq = w.wtid % QW;
      for (int rr = w.wtid / QW; rr < nb; rr += rows_per_pass) {
        const int K = scnt[rr];
        const int* pp = spos + rr * k_max;
        const float* ww = sw + rr * k_max;
        // four entries per step with their loads issued together; the four
        // partial sums are combined in a fixed order
        float acc4[4][4];
#pragma unroll
        for (int q = 0; q < 4; ++q)
#pragma unroll
          for (int i = 0; i < 4; ++i) acc4[q][i] = 0.f;
        int t = 0;
        for (; t + 4 <= K; t += 4) {
          uint2 raw[4];
          float wt[4];
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            wt[q] = ww[t + q];
            raw[q] = *reinterpret_cast<const uint2*>(us + pp[t + q] * W + cq * 4);
          }
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&raw[q]);
            const float2 f0 = __bfloat1622float2(h2[0]), f1 = __bfloat1622float2(h2[1]);
            acc4[q][0] = fmaf(wt[q], f0.x, acc4[q][0]);
            acc4[q][1] = fmaf(wt[q], f0.y, acc4[q][1]);
            acc4[q][2] = fmaf(wt[q], f1.x, acc4[q][2]);
            acc4[q][3] = fmaf(wt[q], f1.y, acc4[q][3]);
          }
        }
        for (; t < K; ++t) {
          const float wt = ww[t];
          const uint2 raw = *reinterpret_cast<const uint2*>(us + pp[t] * W + cq * 4);
          const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&raw);
          const float2 f0 = __bfloat1622float2(h2[0]), f1 = __bfloat1622float2(h2[1]);
          acc4[0][0] = fmaf(wt, f0.x, acc4[0][0]);
          acc4[0][1] = fmaf(wt, f0.y, acc4[0][1]);
          acc4[0][2] = fmaf(wt, f1.x, acc4[0][2]);
          acc4[0][3] = fmaf(wt, f1.y, acc4[0][3]);
        }
        float acc[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[i] = (acc4[0][i] + acc4[1][i]) + (acc4[2][i] + acc4[3][i]);
        const long long n = row0 + rb + rr;
        const int col = c0 + cq * 4;
        bf16 o[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) o[i] = __float2bfloat16_rn(acc[i]);
        *reinterpret_cast<uint2*>(a.r + n * a.d + col) = *reinterpret_cast<const uint2*>(o);
        if (a.readout)
          *reinterpret_cast<float4*>(a.readout + n * a.d + col) = make_float4(acc[0], acc[1], acc[2], acc[3]);
      }
    }
  }
}

// Gate, gated residual and RMSNorm (Eq. hidden_correction), with c summed
// from the last fusion layer's partial tiles in split order plus b_f2.  The
// gate comes first; y = h + g c stays in registers for the second pass.
__device__ void phase_finalize(const FusedArgs& a, const WorkerCtx& w, uint8_t* scr) {
  constexpr int MV = FOVEA_MAX_D / 8 / kWorkers;
  float* red = reinterpret_cast<float*>(scr);
  const PhaseGemm& p = a.g[kPhaseFuse2];
  const int d = a.d, H = a.H, nvec = d / 8;
  for (int n = blockIdx.x; n < a.N; n += gridDim.x) {
    const int rt = n >> 7, rit = n & 127;
    const bf16* a_g = a.act + (long long)n * 2 * H + H;
    float part = 0.0f;
    for (int k = w.wtid; k < H; k += kWorkers)
      part = fmaf(__bfloat162float(__ldcg(a_g + k)), __bfloat162float(a.w_g2[k]), part);
    const float z = worker_sum(part, red, w.wtid) + __bfloat162float(a.b_g2[0]);
    const float g = sigmoidf_(z);
    // c = sum of the partial tiles in split order (every quad's load of one
    // split in flight together)
    float yv[MV][8];
    for (int s = 0; s < p.splits; ++s) {
      float4 t[MV][2];
#pragma unroll
      for (int j = 0; j < MV; ++j) {
        const int vi = w.wtid + j * kWorkers;
        if (vi < nvec) {
#pragma unroll
          for (int h4 = 0; h4 < 2; ++h4) {
            const int c = vi * 8 + h4 * 4;
            const int ft = c / p.bn, jj = c - ft * p.bn;
            const int u = p.unit0[0] + (rt * p.ftiles[0] + ft) * p.splits + s;
            t[j][h4] = __ldcg(reinterpret_cast<const float4*>(partial_tile(a, p, u) +
                                                               (long long)rit * p.bn + jj));
          }
        }
      }
#pragma unroll
      for (int j = 0; j < MV; ++j) {
        if (w.wtid + j * kWorkers < nvec) {
#pragma unroll
          for (int h4 = 0; h4 < 2; ++h4) {
            const float e[4] = {t[j][h4].x, t[j][h4].y, t[j][h4].z, t[j][h4].w};
#pragma unroll
            for (int i = 0; i < 4; ++i)
              yv[j][h4 * 4 + i] = s == 0 ? e[i] : yv[j][h4 * 4 + i] + e[i];
          }
        }
      }
    }
    float ss = 0.0f;
#pragma unroll
    for (int j = 0; j < MV; ++j) {
      const int vi = w.wtid + j * kWorkers;
      if (vi < nvec) {
        float hv[8], bf[8];
        ln_load<bf16>(a.h + (long long)n * d + vi * 8, hv);
        ln_load<bf16>(a.b_f2 + vi * 8, bf);
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const float c = yv[j][i] + bf[i];
          yv[j][i] = fmaf(g, c, hv[i]);          // y = h + g c
          ss = fmaf(yv[j][i], yv[j][i], ss);
        }
      }
    }
    const float tot = worker_sum(ss, red + 8, w.wtid);
    const float inv = 1.0f / sqrtf(tot / (float)d + a.rms_eps);
    bf16* o = a.h_out + (long long)n * d;
#pragma unroll
    for (int j = 0; j < MV; ++j) {
      const int vi = w.wtid + j * kWorkers;
      if (vi < nvec) {
        float gv[8];
        ln_load<bf16>(a.rms_gamma + vi * 8, gv);
        bf16 res[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) res[i] = __float2bfloat16_rn(yv[j][i] * inv * gv[i]);
        *reinterpret_cast<uint4*>(o + vi * 8) = *reinterpret_cast<const uint4*>(res);
      }
    }
    if (a.gate != nullptr && w.wtid == 0) a.gate[n] = g;
  }
}

// ---------------------------------------------------------------------------
// the kernel
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads, 1)
    step_kernel(const __grid_constant__ FusedMaps maps, const __grid_constant__ FusedArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* ring = smem;
  uint8_t* scr = smem + kRingBytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(scr + kScrBytes);
  uint64_t* full = bars;             // [3]
  uint64_t* empty = bars + 3;        // [3]
  uint64_t* tfull = bars + 6;        // [2]
  uint64_t* tempty = bars + 8;       // [2]
  uint64_t* done = bars + 10;        // [1]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 11);
  volatile int* s_ok = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull[i], 1);
      mbar_init(&tempty[i], kWorkers / 32);
    }
    mbar_init(done, 1);
    *s_ok = ld_acquire_gpu(a.sync + kSyncAbort) == 0 ? 1 : 0;
    if (!*s_ok) atomicOr(a.err, kErrTimeout);       // an earlier launch gave up
    fence_mbar_init();
    for (int i = 0; i < kNumMaps; ++i) prefetch_tmap(&maps.m[i]);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    if (lane == 0 && *s_ok) producer(a, maps, ring, full, empty);
  } else if (warp == 1) {
    if (lane == 0 && *s_ok) mma_issuer(a, ring, full, empty, tfull, tempty, done, tmem_base);
    __syncwarp();
  } else {
    WorkerCtx w;
    w.wtid = threadIdx.x - 64;
    w.lane = lane;
    w.wwarp = warp - 2;
    w.s_ok = s_ok;
    int uc = 0;
    if (*s_ok) phase_ln(a, w, scr);
    grid_arrive(a, w, 1, true);
    phase_epilogue(a, w, kPhaseQuery, scr, tfull, tempty, tmem_base, uc);
    grid_arrive(a, w, 2, false);
    if (grid_wait(a, w, 2)) phase_reduce<kPhaseQuery>(a, w);
    grid_arrive(a, w, 3, true);
    phase_epilogue(a, w, kPhaseScore, scr, tfull, tempty, tmem_base, uc);
    grid_arrive(a, w, 4, false);
    if (grid_wait(a, w, 4)) phase_select(a, w, scr);
    grid_arrive(a, w, 5, false);
    if (grid_wait(a, w, 5)) phase_readout(a, w, scr);
    grid_arrive(a, w, 6, true);
    phase_epilogue(a, w, kPhaseFuse1, scr, tfull, tempty, tmem_base, uc);
    grid_arrive(a, w, 7, false);
    if (grid_wait(a, w, 7)) phase_reduce<kPhaseFuse1>(a, w);
    grid_arrive(a, w, 8, true);
    phase_epilogue(a, w, kPhaseFuse2, scr, tfull, tempty, tmem_base, uc);
    grid_arrive(a, w, 9, false);
    if (grid_wait(a, w, 9)) phase_finalize(a, w, scr);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
  if (threadIdx.x == 0) {
    // the last CTA to leave resets the barrier counters for the next launch
    __threadfence();
    if (atomicAdd(a.sync + kSyncExit, 1) == (int)gridDim.x - 1) {
      for (int k = 1; k <= kBarriers; ++k) atomicExch(a.sync + k, 0);
      atomicExch(a.sync + kSyncExit, 0);
    }
  }
}

}  // namespace fused

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
namespace {

int mma_cycles(int bn) { return bn <= 64 ? 50 : bn <= 128 ? 66 : bn <= 192 ? 98 : 129; }

// Choose (bn, splits) for one phase: estimated unit time (MMA issue vs the
// unit's feature bytes at a per-SM share of HBM, or of L2 when several row
// tiles reuse the same feature tiles) times the waves of units, plus the
// split-K partial traffic.
void plan_phase(fused::PhaseGemm& p, int G, int kb_total, const int* m, const int* n, int ngroups,
                bool dual, int f_split_hint) {
  static const int cands[3] = {256, 128, 64};
  double best = 1e30;
  int best_bn = 64, best_s = 1;
  for (int bn : cands) {
    if (dual && bn > 128) continue;
    if (f_split_hint > 0 && f_split_hint % bn != 0) continue;
    long long tiles = 0, outs = 0;
    int rtiles_max = 0, rows_max = 0;
    for (int g = 0; g < ngroups; ++g) {
      rows_max = std::max(rows_max, n[g]);
      tiles += (long long)((n[g] + 127) / 128) * ((m[g] + bn - 1) / bn);
      outs += (long long)n[g] * m[g];
      rtiles_max = std::max(rtiles_max, (n[g] + 127) / 128);
    }
    if (tiles == 0) continue;
    int S = (int)std::max<long long>(1, G / tiles);
    S = std::min(S, kb_total);
    const long long units = tiles * S;
    const long long waves = (units + G - 1) / G;
    const int nkb = (kb_total + S - 1) / S;
    const double t_mma = nkb * 4.0 * mma_cycles(bn) * (dual ? 2 : 1) / 2000.0;
    // feature bytes from HBM (from L2 when several row tiles reuse them), row
    // bytes from L2; per-SM shares of the bandwidth in bytes per microsecond
    const double rbytes = (dual ? 2.0 : 1.0) * std::min(128, (rows_max + 7) / 8 * 8) * 128.0;
    const double t_bytes = nkb * ((double)bn * 128.0 / (rtiles_max > 1 ? 150e3 : 45e3) +
                                  rbytes / 150e3);
    const double t_red = (double)S * outs * 4.0 / (G * 100e3);
    const double t = waves * std::max(t_mma, t_bytes) + t_red;
    if (t < best - 1e-9) {
      best = t;
      best_bn = bn;
      best_s = S;
    }
  }
  int rows_max = 0;
  for (int g = 0; g < ngroups; ++g) rows_max = std::max(rows_max, n[g]);
  p.rbox = std::min(128, (rows_max + 7) / 8 * 8);
  p.bn = best_bn;
  p.splits = best_s;
  p.kb_total = kb_total;
  p.dual = dual ? 1 : 0;
  p.ngroups = ngroups;
  int u = 0;
  for (int g = 0; g < ngroups; ++g) {
    p.unit0[g] = u;
    p.m[g] = m[g];
    p.n[g] = n[g];
    p.ftiles[g] = (m[g] + best_bn - 1) / best_bn;
    u += ((n[g] + 127) / 128) * p.ftiles[g] * best_s;
  }
  p.unit0[ngroups] = u;
  p.units = u;
}

int sm_count() {
  static int sms = 0;
  if (sms == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (sms <= 0) sms = 1;
  }
  return sms;
}

}  // namespace

bool fused_plan(const FusedShape& sh, FusedPlan* out) {
  FusedPlan pl;
  memset(&pl, 0, sizeof(pl));
  if (!sh.bf16 || sh.N <= 0 || sh.B > fused::kMaxSeq || sh.d % 64 != 0 || sh.d > FOVEA_MAX_D ||
      sh.H % 64 != 0 || sh.k_max > FOVEA_MAX_K || sh.k_max < 1)
    return false;
  int max_m = 0;
  for (int b = 0; b < sh.B; ++b)
    if (sh.row_offsets[b + 1] > sh.row_offsets[b]) max_m = std::max(max_m, sh.m[b]);
  int w = 32;
  while (w > 8 && (long long)max_m * w * 2 > fused::kScrUs) w >>= 1;
  if ((long long)max_m * w * 2 > fused::kScrUs || sh.d % w != 0) return false;
  if (((sizeof(SelectSmem) + 15) & ~(size_t)15) + (size_t)max_m * 4 > (size_t)fused::kScrBytes)
    return false;
  const int G = sm_count();
  pl.G = G;
  pl.ro_w = w;
  pl.ro_rows = std::max(1, std::min(256, fused::kScrSel / 4 / sh.k_max));
  // query: rows N, features d, K d
  {
    int m = sh.d, n = sh.N;
    plan_phase(pl.g[fused::kPhaseQuery], G, sh.d / 64, &m, &n, 1, false, 0);
  }
  // scores: one group per sequence with rows and keys
  {
    int m[fused::kMaxSeq], n[fused::kMaxSeq], ng = 0;
    for (int b = 0; b < sh.B; ++b) {
      const int R = sh.row_offsets[b + 1] - sh.row_offsets[b];
      pl.seq_group[b] = -1;
      if (R > 0 && sh.m[b] > 0) {
        pl.seq_group[b] = ng;
        m[ng] = sh.m[b];
        n[ng] = R;
        ++ng;
      }
    }
    if (ng > 0) {
      plan_phase(pl.g[fused::kPhaseScore], G, sh.d / 64, m, n, ng, true, 0);
    } else {
      pl.g[fused::kPhaseScore].units = 0;
      pl.g[fused::kPhaseScore].bn = 64;
      pl.g[fused::kPhaseScore].splits = 1;
    }
    pl.n_score_groups = ng;
  }
  // fusion layer 1: rows N, features 2H (W_f1 | W_g1), K 2d (h | r)
  {
    int m = 2 * sh.H, n = sh.N;
    plan_phase(pl.g[fused::kPhaseFuse1], G, 2 * sh.d / 64, &m, &n, 1, false, sh.H);
  }
  // fusion layer 2: rows N, features d, K H
  {
    int m = sh.d, n = sh.N;
    plan_phase(pl.g[fused::kPhaseFuse2], G, sh.H / 64, &m, &n, 1, false, 0);
  }
  long long pf = 0;
  for (int ph = 0; ph < fused::kPhases; ++ph)
    pf = std::max(pf, (long long)pl.g[ph].units * 128 * pl.g[ph].bn);
  pl.partial_floats = pf;
  // readout items: (sequence with rows) x column slices
  int ns = 0;
  for (int b = 0; b < sh.B; ++b)
    if (sh.row_offsets[b + 1] > sh.row_offsets[b]) pl.ro_seq[ns++] = b;
  pl.ro_nseq = ns;
  *out = pl;
  return true;
}

cudaError_t launch_fused_step(const FusedPlan& pl, const FusedLaunch& L, cudaStream_t s) {
  using namespace fused;
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(step_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         kSmemBytes);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  static thread_local FusedArgs a;
  static thread_local FusedMaps maps;
  memset(&a, 0, sizeof(a));
  for (int ph = 0; ph < kPhases; ++ph) a.g[ph] = pl.g[ph];
  const int d = L.d, H = L.H, N = L.N;
  // operand tensor maps and per-phase wiring
  struct Op {
    const void* base;
    long long rows, cols, ld;
    int box_rows;
  };
  const int bnQ = pl.g[kPhaseQuery].bn, bnS = pl.g[kPhaseScore].bn, bn1 = pl.g[kPhaseFuse1].bn,
            bn2 = pl.g[kPhaseFuse2].bn;
  const Op ops[kNumMaps] = {
      {L.W_Q, d, d, d, bnQ},                       // 0 F: query weights
      {L.x, N, d, d, pl.g[kPhaseQuery].rbox},      // 1 R: LN(h) + E
      {L.keys, std::max<long long>(L.total_keys, 1), d, d, bnS},   // 2 F: keys
      {L.q_hi, N, d, d, std::max(8, pl.g[kPhaseScore].rbox)},   // 3 R: q hi
      {L.q_lo, N, d, d, std::max(8, pl.g[kPhaseScore].rbox)},   // 4 R: q lo
      {L.W_f1, H, 2 * d, 2 * d, bn1},              // 5 F: W_f1
      {L.W_g1, H, 2 * d, 2 * d, bn1},              // 6 F: W_g1
      {L.h, N, d, d, pl.g[kPhaseFuse1].rbox},      // 7 R: h
      {L.r, N, d, d, pl.g[kPhaseFuse1].rbox},      // 8 R: r
      {L.W_f2, d, H, H, bn2},                      // 9 F: W_f2
      {L.act, N, H, 2 * H, pl.g[kPhaseFuse2].rbox},   // 10 R: a_f (columns 0..H-1 of act)
  };
  for (int i = 0; i < kNumMaps; ++i) {
    if (!encode_bf16_map(&maps.m[i], ops[i].base, ops[i].rows, ops[i].cols, ops[i].ld,
                         ops[i].box_rows))
      return cudaErrorInvalidValue;
  }
  const int INF = 0x7fffffff;
  PhaseGemm& q = a.g[kPhaseQuery];
  q.fmap0 = q.fmap1 = 0; q.rmap0 = q.rmap1 = 1; q.f_split = INF; q.r_split_kb = INF;
  q.a_row0[0] = 0; q.b_row0[0] = 0; q.wait_r0 = q.wait_r1 = 1;
  PhaseGemm& sc = a.g[kPhaseScore];
  sc.fmap0 = sc.fmap1 = 2; sc.rmap0 = 3; sc.rmap1 = 4; sc.f_split = INF; sc.r_split_kb = INF;
  sc.wait_r0 = sc.wait_r1 = 3;
  for (int b = 0; b < L.B; ++b) {
    const int g = pl.seq_group[b];
    if (g >= 0) {
      sc.a_row0[g] = L.key_off[b];
      sc.b_row0[g] = L.row_offsets[b];
    }
  }
  PhaseGemm& f1 = a.g[kPhaseFuse1];
  f1.fmap0 = 5; f1.fmap1 = 6; f1.rmap0 = 7; f1.rmap1 = 8; f1.f_split = H; f1.r_split_kb = d / 64;
  f1.a_row0[0] = 0; f1.b_row0[0] = 0; f1.wait_r0 = 0; f1.wait_r1 = 6;
  PhaseGemm& f2 = a.g[kPhaseFuse2];
  f2.fmap0 = f2.fmap1 = 9; f2.rmap0 = f2.rmap1 = 10; f2.f_split = INF; f2.r_split_kb = INF;
  f2.a_row0[0] = 0; f2.b_row0[0] = 0; f2.wait_r0 = f2.wait_r1 = 8;

  a.N = N; a.d = d; a.H = H; a.B = L.B; a.k_max = L.k_max; a.k_min = L.k_min; a.rho = L.rho;
  a.scale = (float)(1.0 / sqrt((double)d));
  a.ln_eps = L.ln_eps; a.rms_eps = L.rms_eps; a.max_depth = L.max_depth;
  a.h = (const bf16*)L.h; a.depth = L.depth; a.row_scale = L.row_scale;
  a.ln_gamma = (const bf16*)L.ln_gamma; a.ln_beta = (const bf16*)L.ln_beta; a.E = (const bf16*)L.E;
  a.U = (const bf16*)L.values; a.orig_index = L.orig_index;
  a.b_f1 = (const bf16*)L.b_f1; a.b_g1 = (const bf16*)L.b_g1; a.b_f2 = (const bf16*)L.b_f2;
  a.w_g2 = (const bf16*)L.w_g2; a.b_g2 = (const bf16*)L.b_g2; a.rms_gamma = (const bf16*)L.rms_gamma;
  for (int b = 0; b <= L.B; ++b) a.row_start[b] = L.row_offsets[b];
  for (int b = 0; b < L.B; ++b) {
    a.key_off[b] = L.key_off[b];
    a.mseq[b] = L.m[b];
    a.seq_group[b] = pl.seq_group[b];
  }
  a.x = (bf16*)L.x; a.q_hi = (bf16*)L.q_hi; a.q_lo = (bf16*)L.q_lo; a.r = (bf16*)L.r;
  a.act = (bf16*)L.act; a.partials = L.partials;
  a.sel_pos = L.sel_pos; a.sel_w = L.sel_w; a.sel_cnt = L.sel_cnt;
  a.err = L.err; a.sync = L.sync;
  a.h_out = (bf16*)L.h_out; a.counts = L.counts; a.indices = L.indices; a.readout = L.readout;
  a.gate = L.gate;
  a.ro_w = pl.ro_w; a.ro_rows = pl.ro_rows;
  for (int i = 0; i < pl.ro_nseq; ++i) a.ro_seq[i] = pl.ro_seq[i];
  a.ro_items = pl.ro_nseq * (d / pl.ro_w);
  // L2 prefetch (after the query weights are requested): keys, the fusion
  // weights, and the values when the selected sets are dense
  int np = 0;
  if (L.total_keys > 0) {
    a.pf_ptr[np] = L.keys; a.pf_bytes[np] = (long long)L.total_keys * d * 2; ++np;
    if (L.prefetch_values) {
      a.pf_ptr[np] = L.values; a.pf_bytes[np] = (long long)L.total_keys * d * 2; ++np;
    }
  }
  a.pf_ptr[np] = L.W_f1; a.pf_bytes[np] = (long long)H * 2 * d * 2; ++np;
  a.pf_ptr[np] = L.W_g1; a.pf_bytes[np] = (long long)H * 2 * d * 2; ++np;
  a.pf_ptr[np] = L.W_f2; a.pf_bytes[np] = (long long)d * H * 2; ++np;
  a.n_prefetch = np;

  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(pl.G, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = kSmemBytes;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, step_kernel, maps, a);
}

}  // namespace fovea
