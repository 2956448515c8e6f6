// score_tc.cu — a1/a2 on the 5th-generation tensor cores (tcgen05 + TMEM).
//
// The same two passes as score.cu (§4 observation-window score; the log-sum-
// exp of every observation row is needed before any column sum), for the
// observation-row counts R that are multiples of 128 (of 256 above 256):
//   pass 1  D[rows x keys] = Q K^T.  Each epilogue thread owns one row and
//           keeps its online (max, sum) over the CTA's keys without shuffles.
//   pass 2  D[keys x rows] = K Q^T.  Each epilogue thread owns one key and sums
//           exp(l - LSE_row) over the rows of its TMEM lane without shuffles.
// Roles per CTA (one work item = one unit x kKeysPerItem keys):
//   warp 0      TMA producer: Q once, then K tiles of 128 keys (two 128-byte
//               swizzled boxes of 64 dims) into a kStages-deep ring;
//   warp 1      TMEM allocation and the single MMA-issuing thread
//               (tcgen05.mma kind::f16, bf16 x bf16 -> fp32 in TMEM, two
//               accumulator buffers so MMA and epilogue overlap);
//   warps 2..17 epilogue: warp (q, cq) reads TMEM lane quadrant q and the
//               64-column quarter cq of every tile's accumulator buffer
//               (tcgen05.ld), releases the buffer, then does the exp2 and the
//               reductions.
// Every mbarrier wait is bounded; a timeout sets an abort flag and the status
// word, every role then drains and the CTA frees its TMEM before returning.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "../../include/certkv.h"
#include "common.cuh"
#include "internal.cuh"
#include "tma.cuh"

namespace certkv {
namespace tc {

#ifndef CERTKV_TC_STAGES
#define CERTKV_TC_STAGES 4
#endif
#ifndef CERTKV_TC_STAGES1
#define CERTKV_TC_STAGES1 3
#endif
constexpr int kEpiWarps = 16;  // warp (q, cq): TMEM lane quadrant q, 64-column quarter cq
constexpr int kThreads = (2 + kEpiWarps) * 32;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kStatusTimeout = CERTKV_STATUS_TIMEOUT;

// Shared-memory plan of one pass: Q rows staged once, a ring of K tiles, then
// MISC bytes: the barriers (256 B), the TMEM slot and abort flag (256 B) and
// any per-pass scratch.
template <int QROWS, int TKEYS, int STAGES, int MISC>
struct Cfg {
  static constexpr int kQRows = QROWS;
  static constexpr int kTileKeys = TKEYS;
  static constexpr int kStages = STAGES;
  static constexpr int kQBytes = QROWS * 128 * 2;        // two 128-B-wide halves
  static constexpr int kStageBytes = TKEYS * 128 * 2;    // one K tile, two halves
  static constexpr int kBarOff = kQBytes + STAGES * kStageBytes;
  static constexpr int kSmemBytes = kBarOff + MISC + 1024;  // + alignment slack
  static_assert(kSmemBytes <= 232448, "over the 227 KB of shared memory a CTA can have");
};
// pass 1: one 128-row half of Q per CTA, 256-key tiles (M128 x N256 MMAs),
// three stages so that each tile's copy has two tile periods to land; the
// final (max, sum) merge reuses the Q region once every MMA has completed
using Pass1 = Cfg<128, 256, CERTKV_TC_STAGES1, 512>;
// pass 2: all (<= 256) rows of Q, 128-key tiles (M128 x N<=256 MMAs); the
// rows' log-sum-exp values (1 KB) after the barriers
using Pass2 = Cfg<256, 128, CERTKV_TC_STAGES, 512 + 1024>;

// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle, rows of
// 128 B, groups of 8 rows 1024 B apart.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t smem) {
  uint64_t d = 0;
  d |= (uint64_t)((smem >> 4) & 0x3FFFu);
  d |= (uint64_t)1u << 16;             // leading byte offset (unused with this swizzle)
  d |= (uint64_t)(1024u >> 4) << 32;   // stride byte offset: 8 rows x 128 B
  d |= (uint64_t)1u << 46;             // descriptor version
  d |= (uint64_t)2u << 61;             // 128-byte swizzle
  return d;
}

// Instruction descriptor of kind::f16: fp32 accumulate, bf16 A and B, both
// K-major, shape M x N.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) |
         ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ void umma_commit(uint32_t mbar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   mbar)
               : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// 32 consecutive fp32 columns of this warp's 32 TMEM lanes (one per thread).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,"
      "%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
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

// max(a, b, c) in one instruction (sm_100 family); like fmaxf, a NaN operand
// is ignored.
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

// Hardware base-2 exponential (MUFU), flush-to-zero, relative error ~2^-22.
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// 64 consecutive fp32 columns: two 32-column loads issued before one wait.
__device__ __forceinline__ void tmem_ld64(uint32_t taddr, float (&v)[64]) {
  uint32_t r[64];
#define CERTKV_R8(o) "=r"(r[o]), "=r"(r[o + 1]), "=r"(r[o + 2]), "=r"(r[o + 3]), "=r"(r[o + 4]), \
                     "=r"(r[o + 5]), "=r"(r[o + 6]), "=r"(r[o + 7])
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,"
      "%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : CERTKV_R8(0), CERTKV_R8(8), CERTKV_R8(16), CERTKV_R8(24)
      : "r"(taddr));
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,"
      "%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : CERTKV_R8(32), CERTKV_R8(40), CERTKV_R8(48), CERTKV_R8(56)
      : "r"(taddr + 32u));
#undef CERTKV_R8
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 64; ++i) v[i] = __uint_as_float(r[i]);
}

// Named barrier over the epilogue warps only.
__device__ __forceinline__ void epi_sync() {
  asm volatile("bar.sync 1, %0;" ::"n"(kEpiWarps * 32) : "memory");
}

template <class C>
struct Shared {
  char* base;  // 1024-byte aligned
  __device__ uint32_t q() const { return saddr(base); }
  __device__ uint32_t kst(int s) const { return saddr(base + C::kQBytes + s * C::kStageBytes); }
  __device__ uint64_t* bars() const { return reinterpret_cast<uint64_t*>(base + C::kBarOff); }
  __device__ uint32_t full(int s) const { return saddr(bars() + s); }
  __device__ uint32_t empty(int s) const { return saddr(bars() + C::kStages + s); }
  __device__ uint32_t accf(int b) const { return saddr(bars() + 2 * C::kStages + b); }
  __device__ uint32_t acce(int b) const { return saddr(bars() + 2 * C::kStages + 2 + b); }
  __device__ uint32_t qfull() const { return saddr(bars() + 2 * C::kStages + 4); }
  __device__ uint32_t done() const { return saddr(bars() + 2 * C::kStages + 5); }
  __device__ uint32_t* tmem_slot() const {
    return reinterpret_cast<uint32_t*>(base + C::kBarOff + 256);
  }
  __device__ volatile int* abort_flag() const {
    return reinterpret_cast<volatile int*>(base + C::kBarOff + 260);
  }
  // lse[256] of pass 2 after the barriers; the partial (max, sum) of 4 x 128
  // rows of pass 1 in the Q region (written only after the last MMA)
  __device__ float* lse() const { return reinterpret_cast<float*>(base + C::kBarOff + 512); }
  __device__ float* pm() const { return reinterpret_cast<float*>(base); }
  __device__ float* pl() const { return reinterpret_cast<float*>(base + 2048); }
};

template <class C>
__device__ __forceinline__ Shared<C> shared_layout(char* raw) {
  Shared<C> s;
  s.base = reinterpret_cast<char*>((reinterpret_cast<uintptr_t>(raw) + 1023) & ~(uintptr_t)1023);
  return s;
}

// Set-up common to both passes: barriers, TMEM allocation.
template <class C>
__device__ __forceinline__ uint32_t setup(const Shared<C>& sh, int warp) {
  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(sh.full(s), 1);
      mbar_init(sh.empty(s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(sh.accf(b), 1);
      mbar_init(sh.acce(b), kEpiWarps);
    }
    mbar_init(sh.qfull(), 1);
    mbar_init(sh.done(), 1);
    *sh.abort_flag() = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     saddr(sh.tmem_slot())),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  return *sh.tmem_slot();
}

template <class C>
__device__ __forceinline__ void teardown(const Shared<C>& sh, int warp, uint32_t tmem,
                                         uint32_t* status) {
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0 && *sh.abort_flag()) atomicOr(status, kStatusTimeout);
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                 "r"(kTmemCols)
                 : "memory");
  }
}

// Producer: qrows rows of Q once, then the K tiles starting at row krow0.
template <class C>
__device__ __forceinline__ void produce(const Shared<C>& sh, const CUtensorMap* tmK,
                                        const CUtensorMap* tmQ, int qrow0, int qrows, long krow0,
                                        int ntiles) {
  volatile int* ab = sh.abort_flag();
  mbar_expect_tx(sh.qfull(), (uint32_t)qrows * 256u);
  tma_load_2d(sh.q(), tmQ, 0, qrow0, sh.qfull());
  tma_load_2d(sh.q() + C::kQBytes / 2, tmQ, 64, qrow0, sh.qfull());
  int issued = 0;
  for (int t = 0; t < ntiles; ++t) {
    const int s = t % C::kStages;
    if (t >= C::kStages && !mbar_wait(sh.empty(s), ((t / C::kStages) - 1) & 1, ab)) break;
    mbar_expect_tx(sh.full(s), (uint32_t)C::kStageBytes);
    const int y = (int)(krow0 + (long)t * C::kTileKeys);
    tma_load_2d(sh.kst(s), tmK, 0, y, sh.full(s));
    tma_load_2d(sh.kst(s) + C::kStageBytes / 2, tmK, 64, y, sh.full(s));
    issued = t + 1;
  }
  // drain: the copies of the last stages must land before the CTA exits
  for (int t = (issued > C::kStages ? issued - C::kStages : 0); t < issued; ++t) {
    const int s = t % C::kStages;
    volatile int dummy = 0;
    mbar_wait(sh.full(s), (t / C::kStages) & 1, &dummy);
  }
  volatile int dummy = 0;
  mbar_wait(sh.qfull(), 0, &dummy);
}

// The 8 k-steps of one tile as back-to-back MMAs into d: a and b are the
// descriptors of the operands' first k-step; k-step ks starts (ks & 3) * 32
// bytes into the 128-byte swizzled rows of half ks >> 2, which lies ha (hb)
// descriptor units after the first half.  A descriptor's address field is
// the byte address / 16 in its low 14 bits, and no operand reaches 256 KB,
// so the offsets are plain additions.
template <uint32_t ha, uint32_t hb>
__device__ __forceinline__ void umma_tile(uint32_t d, uint64_t a, uint64_t b, uint32_t idesc) {
#define CERTKV_A(ks) (a + (uint64_t)(((ks) >> 2) * ha + ((ks) & 3) * 2))
#define CERTKV_B(ks) (b + (uint64_t)(((ks) >> 2) * hb + ((ks) & 3) * 2))
  asm volatile(
      "{\n .reg .pred p0, p1;\n setp.ne.b32 p0, %17, %17;\n setp.eq.b32 p1, %17, %17;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %18, p0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %3, %4, %18, p1;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %5, %6, %18, p1;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %7, %8, %18, p1;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %9, %10, %18, p1;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %11, %12, %18, p1;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %13, %14, %18, p1;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %15, %16, %18, p1;\n}\n" ::"r"(d),
      "l"(CERTKV_A(0)), "l"(CERTKV_B(0)), "l"(CERTKV_A(1)), "l"(CERTKV_B(1)), "l"(CERTKV_A(2)),
      "l"(CERTKV_B(2)), "l"(CERTKV_A(3)), "l"(CERTKV_B(3)), "l"(CERTKV_A(4)), "l"(CERTKV_B(4)),
      "l"(CERTKV_A(5)), "l"(CERTKV_B(5)), "l"(CERTKV_A(6)), "l"(CERTKV_B(6)), "l"(CERTKV_A(7)),
      "l"(CERTKV_B(7)), "r"(0u), "r"(idesc));
#undef CERTKV_A
#undef CERTKV_B
}

// MMA issuer: for each tile, 8 k-steps of one M128 x N MMA into buffer t & 1.
// kKeysA: the K tile is the A operand (pass 2), else Q is (pass 1).  The
// descriptors are formed once; each tile only adds its stage's offset, so
// the issuing thread (which shares its SM sub-partition with four epilogue
// warps) spends few instructions per tile.
template <class C, bool kKeysA>
__device__ __forceinline__ void issue_mmas(const Shared<C>& sh, uint32_t tmem, uint32_t idesc,
                                           int ntiles) {
  volatile int* ab = sh.abort_flag();
  bool ok = mbar_wait(sh.qfull(), 0, ab);
  tc_fence_after();
  const uint64_t dq = sw128_desc(sh.q());
  const uint64_t dk0 = sw128_desc(sh.kst(0));
  constexpr uint32_t kHalfQ = (uint32_t)(C::kQBytes / 2) >> 4;
  constexpr uint32_t kHalfK = (uint32_t)(C::kStageBytes / 2) >> 4;
  constexpr uint32_t kStep = (uint32_t)C::kStageBytes >> 4;
  for (int t = 0; ok && t < ntiles; ++t) {
    const int s = t % C::kStages, b = t & 1;
    if (!mbar_wait(sh.full(s), (t / C::kStages) & 1, ab)) break;
    if (t >= 2 && !mbar_wait(sh.acce(b), ((t >> 1) - 1) & 1, ab)) break;
    tc_fence_after();
    const uint32_t d = tmem + (uint32_t)(b * 256);
    const uint64_t dk = dk0 + (uint64_t)((uint32_t)s * kStep);
    if (kKeysA) umma_tile<kHalfK, kHalfQ>(d, dk, dq, idesc);
    else umma_tile<kHalfQ, kHalfK>(d, dq, dk, idesc);
    umma_commit(sh.empty(s));
    umma_commit(sh.accf(b));
  }
  umma_commit(sh.done());  // every MMA issued above has finished reading smem
  volatile int dummy = 0;
  mbar_wait(sh.done(), 0, &dummy);
}

// Pass 1.  grid = units * key_splits * halves; adjacent CTAs are the two
// 128-row halves of one key range (they stream the same K tiles, the second
// mostly from L2).  D[rows x 256 keys]; epilogue thread = one row and a
// 64-key quarter of every tile.
__global__ void __launch_bounds__(kThreads, 1) lse_tc_kernel(const __grid_constant__ CUtensorMap tmK,
                                                             const __grid_constant__ CUtensorMap tmQ,
                                                             Prob p, float2* __restrict__ lse_part,
                                                             uint32_t* status) {
  using C = Pass1;
  extern __shared__ char smem_raw[];
  const Shared<C> sh = shared_layout<C>(smem_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int halves = p.R / 128;
  const int half = blockIdx.x % halves;
  const int item = blockIdx.x / halves;
  const int u = item / p.key_splits, split = item % p.key_splits;
  const int n = p.n, R = p.R;
  const int j_begin = split * kKeysPerItemTc;
  const int j_end = min(n, j_begin + kKeysPerItemTc);
  const int ntiles = (j_end - j_begin + C::kTileKeys - 1) / C::kTileKeys;
  const uint32_t tmem = setup<C>(sh, warp);
  volatile int* ab = sh.abort_flag();

  if (warp == 0) {
    if (lane == 0) produce<C>(sh, &tmK, &tmQ, u * R + half * 128, 128, (long)u * n + j_begin, ntiles);
  } else if (warp == 1) {
    if (lane == 0)
      issue_mmas<C, false>(sh, tmem, idesc_bf16(128, C::kTileKeys), ntiles);
  } else {
    // every warp takes every tile: warp (q, cq) owns rows q*32.. of the half
    // (its TMEM lane quadrant) and keys cq*64 .. cq*64+63 of each 256-key tile.
    // It releases the accumulator as soon as its columns are in registers.
    const int ew = warp - 2, q = warp & 3, cq = ew >> 2;
    const int rloc = q * 32 + lane;
    const int row = half * 128 + rloc;
    const int lim = n - p.w + (row % p.w);
    const float sl2 = p.scale_log2;
    float m = -INFINITY, l = 0.f;
    for (int t = 0; t < ntiles; ++t) {
      const int b = t & 1;
      if (!mbar_wait(sh.accf(b), (t >> 1) & 1, ab)) break;
      tc_fence_after();
      float v[64];
      tmem_ld64(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(b * 256 + cq * 64), v);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(sh.acce(b));
      const int jc = j_begin + t * C::kTileKeys + cq * 64;
      const bool interior = (jc + 64 <= j_end) && (jc + 63 <= n - p.w);
      if (interior) {
        // the tile's maximum with three-input maxima (exact, as fmaxf)
        float mx0 = v[0], mx1 = v[1];
#pragma unroll
        for (int i = 2; i < 62; i += 4) {
          mx0 = fmax3(mx0, v[i], v[i + 1]);
          mx1 = fmax3(mx1, v[i + 2], v[i + 3]);
        }
        mx0 = fmax3(mx0, v[62], v[63]);
        const float nm = fmaxf(m, fmaxf(mx0, mx1) * sl2);  // sl2 > 0: max commutes with scaling
        // the scale-and-subtract and the accumulation two-wide (f32x2), each
        // element into acc[i & 7] in order as a one-wide loop would add it
        // (measured: pass 1 3 % faster on C3, 7 % on C5)
        float acc[8];
        {
          const float2 s2 = make_float2(sl2, sl2), m2 = make_float2(-nm, -nm);
          float2 a01 = make_float2(0.f, 0.f), a23 = a01, a45 = a01, a67 = a01;
#pragma unroll
          for (int i = 0; i < 64; i += 8) {
            const float2 x0 = ffma2(make_float2(v[i], v[i + 1]), s2, m2);
            const float2 x1 = ffma2(make_float2(v[i + 2], v[i + 3]), s2, m2);
            const float2 x2 = ffma2(make_float2(v[i + 4], v[i + 5]), s2, m2);
            const float2 x3 = ffma2(make_float2(v[i + 6], v[i + 7]), s2, m2);
            a01 = fadd2(a01, make_float2(ex2(x0.x), ex2(x0.y)));
            a23 = fadd2(a23, make_float2(ex2(x1.x), ex2(x1.y)));
            a45 = fadd2(a45, make_float2(ex2(x2.x), ex2(x2.y)));
            a67 = fadd2(a67, make_float2(ex2(x3.x), ex2(x3.y)));
          }
          acc[0] = a01.x; acc[1] = a01.y; acc[2] = a23.x; acc[3] = a23.y;
          acc[4] = a45.x; acc[5] = a45.y; acc[6] = a67.x; acc[7] = a67.y;
        }
        const float sum = ((acc[0] + acc[1]) + (acc[2] + acc[3])) + ((acc[4] + acc[5]) + (acc[6] + acc[7]));
        l = fmaf(l, ex2(m - nm), sum);
        m = nm;
      } else {
        float cm = -INFINITY;
#pragma unroll
        for (int i = 0; i < 64; ++i) {
          const int j = jc + i;
          v[i] = (j <= lim && j < j_end) ? v[i] * sl2 : -INFINITY;
          cm = fmaxf(cm, v[i]);
        }
        const float nm = fmaxf(m, cm);
        if (nm > -INFINITY) {
          float sum = 0.f;
#pragma unroll
          for (int i = 0; i < 64; ++i) sum += ex2(v[i] - nm);
          l = fmaf(l, ex2(m - nm), sum);
          m = nm;
        }
      }
    }
    // merge the four partial (max, sum) of each row, one per key quarter
    sh.pm()[cq * 128 + rloc] = m;
    sh.pl()[cq * 128 + rloc] = l;
    epi_sync();
    if (cq == 0 && !*ab) {
      float M = -INFINITY;
#pragma unroll
      for (int k = 0; k < 4; ++k) M = fmaxf(M, sh.pm()[k * 128 + rloc]);
      float L = 0.f;
      if (M > -INFINITY) {
#pragma unroll
        for (int k = 0; k < 4; ++k) L += sh.pl()[k * 128 + rloc] * ex2(sh.pm()[k * 128 + rloc] - M);
      }
      lse_part[((size_t)u * R + row) * p.key_splits + split] = make_float2(M, L);
    }
  }
  teardown<C>(sh, warp, tmem, status);
}

// Pass 2.  grid = units * key_splits.  D[128 keys x R rows]; epilogue thread
// = one key, summing exp(l - LSE_row) over a 64-row quarter of its TMEM lane.
template <bool kGrouped>  // R > 256: the rows come in groups of 256, one per CTA
__global__ void __launch_bounds__(kThreads, 1) colsum_tc_kernel(const __grid_constant__ CUtensorMap tmK,
                                                                const __grid_constant__ CUtensorMap tmQ,
                                                                Prob p, const float* __restrict__ lse2,
                                                                float* __restrict__ s_part,
                                                                uint32_t* status) {
  using C = Pass2;
  extern __shared__ char smem_raw[];
  const Shared<C> sh = shared_layout<C>(smem_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // rows come in groups of RG <= 256 (one MMA's N); adjacent CTAs are the
  // groups of one key range and stream the same K tiles
  const int n = p.n, R = p.R;
  const int RG = kGrouped ? 256 : R;
  const int groups = kGrouped ? R / 256 : 1;
  const int grp = kGrouped ? (int)(blockIdx.x % groups) : 0;
  const unsigned item = kGrouped ? blockIdx.x / groups : blockIdx.x;
  const int u = item / p.key_splits, split = item % p.key_splits;
  const int rg0 = grp * RG;
  const int j_begin = split * kKeysPerItemTc;
  const int j_end = min(n, j_begin + kKeysPerItemTc);
  const int ntiles = (j_end - j_begin + C::kTileKeys - 1) / C::kTileKeys;
  for (int r = threadIdx.x; r < RG; r += blockDim.x) sh.lse()[r] = lse2[(size_t)u * R + rg0 + r];
  const uint32_t tmem = setup<C>(sh, warp);
  volatile int* ab = sh.abort_flag();

  if (warp == 0) {
    if (lane == 0) produce<C>(sh, &tmK, &tmQ, u * R + rg0, RG, (long)u * n + j_begin, ntiles);
  } else if (warp == 1) {
    if (lane == 0)
      issue_mmas<C, true>(sh, tmem, idesc_bf16(C::kTileKeys, RG), ntiles);
  } else {
    // every warp takes every tile: warp (q, cq) owns keys q*32.. of the tile
    // (its TMEM lane quadrant) and rows rg0 + cq*64 .. +63, summed into row
    // block grp*4 + cq.  It releases the accumulator as soon as its columns
    // are read.
    const int ew = warp - 2, q = warp & 3, cq = ew >> 2;
    const int key = q * 32 + lane;
    const bool rows_here = cq * 64 < RG;
    const float sl2 = p.scale_log2;
    const int nw = n - p.w;
    float* out = s_part + ((size_t)u * p.row_blocks + grp * 4 + cq) * n;
    const int r0 = cq * 64;
    const float4* L4 = reinterpret_cast<const float4*>(sh.lse() + r0);
    for (int t = 0; t < ntiles; ++t) {
      const int b = t & 1;
      if (!mbar_wait(sh.accf(b), (t >> 1) & 1, ab)) break;
      tc_fence_after();
      float v[64];
      if (rows_here)
        tmem_ld64(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(b * 256 + cq * 64), v);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(sh.acce(b));
      if (!rows_here) continue;
      const int j0 = j_begin + t * C::kTileKeys;
      const int j = j0 + key;
      const bool interior = (j0 + C::kTileKeys <= j_end) && (j0 + C::kTileKeys <= nw);
      float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
      if (interior && q < 2) {
        // TMEM quadrants 0 and 1 run on the SM sub-partitions that also issue
        // the copies and the MMAs, and are this pass's slowest: there the
        // scale-and-subtract and the accumulation go two-wide (f32x2), in the
        // same order as below (measured: 1 % on C3's pass, 2 % on C5's; the
        // two-wide form on every warp was not faster)
        const float2 s2 = make_float2(sl2, sl2);
        float2 a01 = make_float2(0.f, 0.f), a23 = a01, a45 = a01, a67 = a01;
#pragma unroll
        for (int i = 0; i < 64; i += 8) {
          const float4 La = L4[i >> 2], Lb = L4[(i >> 2) + 1];
          const float2 x0 = ffma2(make_float2(v[i], v[i + 1]), s2, make_float2(-La.x, -La.y));
          const float2 x1 = ffma2(make_float2(v[i + 2], v[i + 3]), s2, make_float2(-La.z, -La.w));
          const float2 x2 = ffma2(make_float2(v[i + 4], v[i + 5]), s2, make_float2(-Lb.x, -Lb.y));
          const float2 x3 = ffma2(make_float2(v[i + 6], v[i + 7]), s2, make_float2(-Lb.z, -Lb.w));
          a01 = fadd2(a01, make_float2(ex2(x0.x), ex2(x0.y)));
          a23 = fadd2(a23, make_float2(ex2(x1.x), ex2(x1.y)));
          a45 = fadd2(a45, make_float2(ex2(x2.x), ex2(x2.y)));
          a67 = fadd2(a67, make_float2(ex2(x3.x), ex2(x3.y)));
        }
        acc[0] = a01.x; acc[1] = a01.y; acc[2] = a23.x; acc[3] = a23.y;
        acc[4] = a45.x; acc[5] = a45.y; acc[6] = a67.x; acc[7] = a67.y;
      } else if (interior) {
#pragma unroll
        for (int i = 0; i < 64; i += 4) {
          const float4 L = L4[i >> 2];
          acc[(i + 0) & 7] += ex2(fmaf(v[i], sl2, -L.x));
          acc[(i + 1) & 7] += ex2(fmaf(v[i + 1], sl2, -L.y));
          acc[(i + 2) & 7] += ex2(fmaf(v[i + 2], sl2, -L.z));
          acc[(i + 3) & 7] += ex2(fmaf(v[i + 3], sl2, -L.w));
        }
      } else {
#pragma unroll
        for (int i = 0; i < 64; ++i) {
          const int r = r0 + i;  // row of the group; rg0 + r of the unit
          if (j < j_end && j <= nw + ((rg0 + r) % p.w)) acc[0] += ex2(fmaf(v[i], sl2, -sh.lse()[r]));
        }
      }
      if (j < j_end)
        out[j] = ((acc[0] + acc[1]) + (acc[2] + acc[3])) + ((acc[4] + acc[5]) + (acc[6] + acc[7]));
    }
  }
  teardown<C>(sh, warp, tmem, status);
}

}  // namespace tc

// Self-test of the bounded wait: one thread waits on an mbarrier that nothing
// arrives on (no copy and no MMA is issued), so the wait must give up after
// its poll limit, set the abort flag and report CERTKV_STATUS_TIMEOUT.
__device__ uint32_t g_selftest_result[2];
__global__ void selftest_wait_kernel() {
  uint32_t* result = g_selftest_result;
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    tc::mbar_init(tc::saddr(&bar), 1);
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    const bool done = tc::mbar_wait(tc::saddr(&bar), 0, &abort_flag);
    result[0] = done ? 0u : tc::kStatusTimeout;
    result[1] = (uint32_t)abort_flag;
  }
}

// --------------------------------------------------------------- host ----
namespace {

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  }
  return fn;
}

}  // namespace

bool make_row_map(CUtensorMap* map, const void* base, uint64_t rows, uint32_t box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {128, rows};
  cuuint64_t strides[1] = {256};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// R = G w observation rows per KV head: pass 1 takes 128-row halves, pass 2
// groups of min(R, 256) rows (one MMA's N each).
bool score_tc_supported(const Prob& p) {
  return p.R >= 128 && p.R % 128 == 0 && (p.R <= 256 || p.R % 256 == 0);
}

bool launch_score_tc(const Prob& p, const void* K, const void* Q, float2* lse_part, float* lse2,
                     float* s_part, uint32_t* status, cudaStream_t st) {
  CUtensorMap mk1, mq1, mk2, mq2;
  const uint64_t krows = (uint64_t)p.units * p.n, qrows = (uint64_t)p.units * p.R;
  if (!make_row_map(&mk1, K, krows, tc::Pass1::kTileKeys) || !make_row_map(&mq1, Q, qrows, 128) ||
      !make_row_map(&mk2, K, krows, tc::Pass2::kTileKeys) ||
      !make_row_map(&mq2, Q, qrows, (uint32_t)(p.R < 256 ? p.R : 256)))
    return false;
  static bool attr = false;
  if (!attr) {
    cudaFuncSetAttribute(tc::lse_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         tc::Pass1::kSmemBytes);
    cudaFuncSetAttribute(tc::colsum_tc_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         tc::Pass2::kSmemBytes);
    cudaFuncSetAttribute(tc::colsum_tc_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         tc::Pass2::kSmemBytes);
    attr = true;
  }
  const unsigned items = (unsigned)(p.units * p.key_splits);
  {
    TraceScope ts_("score_pass1", st);
    tc::lse_tc_kernel<<<items * (p.R / 128), tc::kThreads, tc::Pass1::kSmemBytes, st>>>(
        mk1, mq1, p, lse_part, status);
  }
  const size_t rows = (size_t)p.units * p.R;
  {
    TraceScope ts_("lse_merge", st);
    lse_merge_kernel<<<(unsigned)((rows + 255) / 256), 256, 0, st>>>(p, lse_part, lse2);
  }
  {
    TraceScope ts_("score_pass2", st);
    if (p.R <= 256)
      tc::colsum_tc_kernel<false><<<items, tc::kThreads, tc::Pass2::kSmemBytes, st>>>(
          mk2, mq2, p, lse2, s_part, status);
    else
      tc::colsum_tc_kernel<true><<<items * (p.R / 256), tc::kThreads, tc::Pass2::kSmemBytes, st>>>(
          mk2, mq2, p, lse2, s_part, status);
  }
  return true;
}

}  // namespace certkv

extern "C" int certkv_selftest_bounded_wait(void* stream) {
  using namespace certkv;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  uint32_t h[2] = {0u, 0u};
  selftest_wait_kernel<<<1, 32, 0, st>>>();
  if (cudaGetLastError() != cudaSuccess ||
      cudaMemcpyFromSymbolAsync(h, g_selftest_result, sizeof h, 0, cudaMemcpyDeviceToHost, st) !=
          cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess)
    return -1;
  return (h[0] == CERTKV_STATUS_TIMEOUT && h[1] == 1u) ? (int)h[0] : -2;
}
