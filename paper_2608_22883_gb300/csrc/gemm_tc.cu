// tcgen05 GEMM C = A . B^T for the bf16 path (sm_103a): the memory
// projections k = W_K LN(v), u = W_U LN(v), the query projection W_Q, the
// scores q . k^T per sequence, and the two fusion layers.  For the scores the
// query is carried as a bf16 hi/lo pair (q ~= q_hi + q_lo, about 16
// significant bits) and each key tile meets both parts, so the scores are not
// limited by a bf16 rounding of q.
//
// A (weights or keys) supplies the UMMA M = 128 rows; B (draft states or
// tokens) supplies UMMA N = BN columns, so a 64-row draft batch is one N = 64
// MMA instead of a mostly-empty M tile ("swap AB").  Both operands are
// K-major bf16, staged by TMA into 128-byte-swizzled shared-memory tiles of
// 64 contraction elements; fp32 accumulators live in tensor memory and are
// read back with tcgen05.ld for the epilogue.
//
// Roles (128 threads): warp 0 lane 0 issues TMA loads into a STAGES-deep ring,
// warp 1 owns the tensor-memory allocation and its lane 0 issues the MMAs
// (one elected thread), and all four warps run the epilogue: warp w reads
// accumulator lanes 32w..32w+31.  Every mbarrier wait is bounded (~2 s); a
// wait that gives up sets kErrTimeout in the error word and the CTA unwinds.
#include "gemm_epilogue.cuh"

namespace fovea {
namespace tc {

constexpr int BM = 128;          // UMMA M
constexpr int BK = 64;           // contraction elements per stage (128 bytes bf16)
constexpr int UMMA_K = 16;       // contraction elements per tcgen05.mma (kind::f16)
constexpr int kThreads = 128;
constexpr int kSmemBudget = 200 * 1024;

// DUAL: the B stage holds two tiles (hi and lo parts of one operand), and
// every A tile is multiplied by both into the same accumulator.
template <int BN, bool DUAL = false>
struct Cfg {
  static constexpr int A_BYTES = BM * BK * 2;
  static constexpr int B_TILE = BN * BK * 2;
  static constexpr int B_BYTES = B_TILE * (DUAL ? 2 : 1);
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int STAGES = (kSmemBudget / STAGE_BYTES) < 8 ? (kSmemBudget / STAGE_BYTES) : 8;
  static constexpr int SMEM = STAGES * STAGE_BYTES + 1024 /*alignment*/ + 256 /*barriers*/;
  static constexpr uint32_t TMEM_COLS = BN < 32 ? 32 : BN;
  // Instruction descriptor, kind::f16: D fp32 (bits 4-5 = 1), A bf16 (bits 7-9
  // = 1), B bf16 (bits 10-12 = 1), both K-major (bits 15, 16 = 0), N >> 3 at
  // bits 17-22, M >> 4 at bits 24-28.
  static constexpr uint32_t IDESC = (1u << 4) | (1u << 7) | (1u << 10) |
                                    ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ uint32_t mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok;
}
__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Bounded wait on an mbarrier phase: true when it completed; false after
// `limit_ns` (about 2 s by default) or once another role of the CTA has
// aborted (when abort_flag is given).
__device__ __noinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                       uint64_t limit_ns = 2000000000ull) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  while (true) {
    for (int i = 0; i < 64; ++i)
      if (mbar_try_wait(bar, parity)) return true;
    if (abort_flag != nullptr && *abort_flag) return false;
    if (globaltimer_ns() - t0 > limit_ns) return false;
  }
}

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, uint64_t* bar, int x,
                                            int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(x), "r"(y)
      : "memory");
}
__device__ __forceinline__ void prefetch_tmap(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

__device__ __forceinline__ void tmem_alloc(uint32_t* slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(slot)),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// Shared-memory matrix descriptor of a K-major, 128-byte-swizzled tile whose
// rows are 128 bytes apart and whose 8-row groups are 1024 bytes apart:
// start address >> 4 (bits 0-13), leading offset 1 (unused for this layout,
// bits 16-29), stride offset 1024 >> 4 (bits 32-45), descriptor version 1
// (bits 46-47), swizzle mode 2 = 128B (bits 61-63).
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)1 << 16;
  d |= (uint64_t)(1024 >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

__device__ __forceinline__ void umma_bf16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                          uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(tmem_d),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}

// 32 consecutive fp32 accumulator columns of this thread's lane.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
        "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
        "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// Key epilogue: store bf16(acc); for key columns, list the element when acc
// lies within 2^-14 * max(|acc|, scale) of a bf16 rounding midpoint.  The
// tensor-core fp32 accumulation error measured on d = 4096 keys is about
// 5e-6 of that scale (one tenth of the window), so an element outside the
// window rounds as the exact value would.
__device__ __forceinline__ void store_key(const GemmArgs& a, const GemmGroup& g, int m, int n,
                                          float acc, float scale) {
  const long long row = (long long)g.b_row0 + n;
  const __nv_bfloat16 r = __float2bfloat16_rn(acc);
  if (m >= a.epi_split) {
    static_cast<__nv_bfloat16*>(a.out1)[row * a.ldc + (m - a.epi_split)] = r;
    return;
  }
  static_cast<__nv_bfloat16*>(a.out0)[row * a.ldc + m] = r;
  const unsigned short bits = __bfloat16_as_ushort(r);
  const float rf = __bfloat162float(r);
  const float up = __bfloat162float(__ushort_as_bfloat16((unsigned short)(bits + 1)));
  const float dn = __bfloat162float(__ushort_as_bfloat16((unsigned short)(bits - 1)));
  const float dist = fminf(fabsf(acc - 0.5f * (rf + up)), fabsf(acc - 0.5f * (rf + dn)));
  const float window = ldexpf(fmaxf(fabsf(acc), scale), -14);
  if (!(dist > window)) {
    const int slot = atomicAdd(a.fix_count, 1);
    if (slot < a.fix_cap) a.fix_list[slot] = KeyFix{(int)row, m};
  }
}

template <int BN, int EPI>
__global__ void __launch_bounds__(kThreads, 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap tmA0, const __grid_constant__ CUtensorMap tmA1,
                   const __grid_constant__ CUtensorMap tmB0, const __grid_constant__ CUtensorMap tmB1,
                   const __grid_constant__ GemmArgs args) {
  constexpr bool DUAL = EPI == kEpiScores;
  using C = Cfg<BN, DUAL>;
  const GemmGroup& g = args.groups[blockIdx.z];
  // Output columns [0, a_split) come from A0 and [a_split, m) from A1; each
  // part is tiled on its own so no tile straddles the two operands.
  // (A group smaller than the grid leaves its extra CTAs idle.)
  const int split = args.a_split;
  const bool has_second = split < g.m;
  const int tiles0 = has_second ? (split + BM - 1) / BM : (g.m + BM - 1) / BM;
  const int bx = (int)blockIdx.x;
  if (!has_second && bx >= tiles0) return;    // uniform for the CTA, before any setup
  const bool a_second = has_second && bx >= tiles0;
  const int m0 = a_second ? split + (bx - tiles0) * BM : bx * BM;
  const int m_end = a_second ? g.m : min(g.m, split);
  const int n0 = blockIdx.y * BN;
  if (m0 >= m_end || n0 >= g.n) return;

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + C::STAGES * C::A_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(sB + C::STAGES * C::B_BYTES);
  uint64_t* empty = full + C::STAGES;
  uint64_t* accum = empty + C::STAGES;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(accum + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(accum, 1);
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tmA0);
    prefetch_tmap(&tmB0);
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
  const int b_split_kb = args.b_split / BK;

  if (warp == 0 && lane == 0) {
    // ---- TMA producer ----
    const CUtensorMap* mapA = a_second ? &tmA1 : &tmA0;
    const int ay = a_second ? m0 - split : g.a_row0 + m0;
    const int by = g.b_row0 + n0;
    int issued = 0;
    for (int kb = 0; kb < kb_total; ++kb) {
      const int s = kb % C::STAGES;
      const uint32_t ph = (uint32_t)(kb / C::STAGES) & 1u;
      if (!mbar_wait(&empty[s], ph ^ 1u, abort_flag)) {
        *abort_flag = 1;
        break;
      }
      mbar_expect_tx(&full[s], C::STAGE_BYTES);
      tma_load_2d(sA + s * C::A_BYTES, mapA, &full[s], kb * BK, ay);
      if constexpr (DUAL) {
        tma_load_2d(sB + s * C::B_BYTES, &tmB0, &full[s], kb * BK, by);
        tma_load_2d(sB + s * C::B_BYTES + C::B_TILE, &tmB1, &full[s], kb * BK, by);
      } else {
        const bool b_second = kb >= b_split_kb;
        tma_load_2d(sB + s * C::B_BYTES, b_second ? &tmB1 : &tmB0, &full[s],
                    (b_second ? kb - b_split_kb : kb) * BK, by);
      }
      ++issued;
    }
    if (*abort_flag) {
      // let copies already in flight land before the CTA gives up its shared memory
      for (int kb = issued > C::STAGES ? issued - C::STAGES : 0; kb < issued; ++kb)
        mbar_wait(&full[kb % C::STAGES], (uint32_t)(kb / C::STAGES) & 1u, nullptr, 20000000ull);
    }
  } else if (warp == 1 && lane == 0) {
    // ---- MMA issuer (single elected thread) ----
    for (int kb = 0; kb < kb_total; ++kb) {
      const int s = kb % C::STAGES;
      const uint32_t ph = (uint32_t)(kb / C::STAGES) & 1u;
      if (!mbar_wait(&full[s], ph, abort_flag)) {
        *abort_flag = 1;
        break;
      }
      tc_fence_after();
      const uint64_t adesc = sw128_desc(smem_u32(sA + s * C::A_BYTES));
      const uint64_t bdesc = sw128_desc(smem_u32(sB + s * C::B_BYTES));
#pragma unroll
      for (int k = 0; k < BK / UMMA_K; ++k) {
        // advance the start address by k * 32 bytes inside the swizzle atom
        umma_bf16(tmem_base, adesc + (uint64_t)(2 * k), bdesc + (uint64_t)(2 * k), C::IDESC,
                  (kb > 0 || k > 0) ? 1u : 0u);
        if constexpr (DUAL) {
          const uint64_t bdesc_lo = sw128_desc(smem_u32(sB + s * C::B_BYTES + C::B_TILE));
          umma_bf16(tmem_base, adesc + (uint64_t)(2 * k), bdesc_lo + (uint64_t)(2 * k), C::IDESC,
                    1u);
        }
      }
      umma_commit(&empty[s]);       // frees this stage once its MMAs have read it
    }
    umma_commit(accum);             // all issued MMAs complete -> accumulator ready
  }

  // ---- epilogue: all warps ----
  __syncwarp();
  const bool waited = mbar_wait(accum, 0, abort_flag);
  // warp-uniform decision: tcgen05.ld below is a .sync.aligned instruction
  const bool ok = __all_sync(0xffffffffu, waited && *abort_flag == 0);
  if (!ok) {
    if (lane == 0) atomicOr(args.err, kErrTimeout);
  } else {
    tc_fence_after();
    const int m = m0 + warp * 32 + lane;
    const uint32_t taddr = tmem_base + ((uint32_t)(warp * 32) << 16);
    float key_scale = 0.0f;
    if constexpr (EPI == kEpiStoreKeys) {
      // RMS of this feature over the tile's tokens: the magnitude of the
      // partial sums, which sets the size of the accumulation error
      float ss = 0.0f;
      int cnt = 0;
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 32) {
        if (n0 + c0 >= g.n) break;
        float v[32];
        tmem_ld32(taddr + (uint32_t)c0, v);
#pragma unroll
        for (int j = 0; j < 32; ++j)
          if (n0 + c0 + j < g.n) { ss = fmaf(v[j], v[j], ss); ++cnt; }
      }
      key_scale = sqrtf(ss / (float)max(cnt, 1));
    }
#pragma unroll 1
    for (int c0 = 0; c0 < BN; c0 += 32) {
      if (n0 + c0 >= g.n) break;                    // uniform across the warp
      float v[32];
      tmem_ld32(taddr + (uint32_t)c0, v);
      if (m < m_end) {
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const int n = n0 + c0 + j;
          if (n < g.n) {
            if constexpr (EPI == kEpiStoreKeys) store_key(args, g, m, n, v[j], key_scale);
            else gemm_epilogue<__nv_bfloat16, EPI>(args, g, m, n, v[j]);
          }
        }
      }
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

template <int BN, int EPI>
static cudaError_t launch_tc_inst(const GemmArgs& a, const CUtensorMap* maps, int max_m, int max_n,
                                  cudaStream_t s) {
  using C = tc::Cfg<BN, EPI == kEpiScores>;
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(tc::tc_gemm_kernel<BN, EPI>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  const int tiles_m = a.a_split >= max_m
                          ? (max_m + tc::BM - 1) / tc::BM
                          : (a.a_split + tc::BM - 1) / tc::BM + (max_m - a.a_split + tc::BM - 1) / tc::BM;
  dim3 grid(tiles_m, (max_n + BN - 1) / BN, a.ngroups);
  tc::tc_gemm_kernel<BN, EPI><<<grid, tc::kThreads, C::SMEM, s>>>(maps[0], maps[1], maps[2], maps[3],
                                                                  a);
  return cudaGetLastError();
}

template <int EPI>
static cudaError_t launch_tc_epi(const GemmArgs& a, const CUtensorMap* maps, int bn, int max_m,
                                 int max_n, cudaStream_t s) {
  switch (bn) {
    case 32: return launch_tc_inst<32, EPI>(a, maps, max_m, max_n, s);
    case 64: return launch_tc_inst<64, EPI>(a, maps, max_m, max_n, s);
    case 128: return launch_tc_inst<128, EPI>(a, maps, max_m, max_n, s);
    default: return launch_tc_inst<256, EPI>(a, maps, max_m, max_n, s);
  }
}

cudaError_t launch_gemm_tc(int epi, const GemmArgs& a, const TmaOperand& A0, const TmaOperand& A1,
                           const TmaOperand& B0, const TmaOperand& B1, int max_m, int max_n,
                           cudaStream_t s) {
  if (max_m <= 0 || max_n <= 0 || a.ngroups <= 0) return cudaSuccess;
  const int bn = max_n <= 32 ? 32 : max_n <= 64 ? 64 : max_n <= 128 ? 128 : 256;
  CUtensorMap maps[4];
  const TmaOperand& a1 = A1.base ? A1 : A0;
  const TmaOperand& b1 = B1.base ? B1 : B0;
  if (!make_map(&maps[0], A0, tc::BM) || !make_map(&maps[1], a1, tc::BM) ||
      !make_map(&maps[2], B0, bn) || !make_map(&maps[3], b1, bn))
    return cudaErrorInvalidValue;
  cudaError_t e;
  switch (epi) {
    case kEpiStore: e = launch_tc_epi<kEpiStore>(a, maps, bn, max_m, max_n, s); break;
    case kEpiScores: e = launch_tc_epi<kEpiScores>(a, maps, bn, max_m, max_n, s); break;
    case kEpiBiasSilu: e = launch_tc_epi<kEpiBiasSilu>(a, maps, bn, max_m, max_n, s); break;
    case kEpiStoreHiLo: e = launch_tc_epi<kEpiStoreHiLo>(a, maps, bn, max_m, max_n, s); break;
    case kEpiStoreKeys: e = launch_tc_epi<kEpiStoreKeys>(a, maps, bn, max_m, max_n, s); break;
    default: e = launch_tc_epi<kEpiBiasF32>(a, maps, bn, max_m, max_n, s); break;
  }
  return e;
}

}  // namespace fovea
