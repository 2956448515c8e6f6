// decode.cu — a9: decode attention over the packed cache.
//
// For each query head qh of unit u = (b, l, qh / G):
//   out = sum_s softmax_s(scale <q, k_s>) v_s
// over the real_counts[u] real slots plus the tail slot (the "plain slot" of
// the paper's ablation table: the synthetic pair enters as an ordinary KV
// entry).
//
// The per-head budgets of one layer differ by an order of magnitude (the
// allocator gives most heads b_min and a few heads most of the budget), so the
// work is balanced over the global sequence of 32-slot tiles of all units, not
// over units: a plan kernel scans the tile counts, then a persistent split
// kernel gives every CTA an equal contiguous range of that sequence.  In each
// CTA one thread streams the tiles' K and V rows into a ring of shared-memory
// stages with bulk copies, and the consumer warps keep online (max, sum, acc)
// for the G query heads of the current unit: for the logits, 2G lanes share a
// slot and hold their slice of the G queries in registers (so a K row is read
// once, coalesced, with no per-lane query traffic through shared memory); for
// the values, a lane owns four dimensions.  Where a CTA's range crosses into
// the next unit the consumer warps combine their states into one record for
// (CTA, unit).  Every packed K/V byte is read once per step.  A merge kernel
// combines the records of each unit in the log-sum-exp domain.
#include "../../include/certkv.h"
#include "common.cuh"
#include "internal.cuh"
#include "tma.cuh"
#include "headlogits.cuh"

namespace certkv {

#ifndef CERTKV_DEC_STAGES
#define CERTKV_DEC_STAGES 4
#endif
#ifndef CERTKV_DEC_CONSUMERS
#define CERTKV_DEC_CONSUMERS 4
#endif
constexpr int kDecTile = 32;
constexpr int kDecStages = CERTKV_DEC_STAGES;
constexpr int kDecConsumers = CERTKV_DEC_CONSUMERS;  // consumer warps; warp 0 issues the copies
constexpr int kDecThreads = (1 + kDecConsumers) * 32;
// Tile k uses stage k % kDecStages and consumer warp k % kDecConsumers.  A
// consumer waits for a stage's phase by its parity, which is only unambiguous
// when the stage's previous phase is already complete; with the stage count a
// multiple of the consumer count every stage belongs to one warp, which has
// itself waited for that previous phase.
static_assert(kDecStages % kDecConsumers == 0, "each ring stage must belong to one consumer warp");
constexpr int kDecMaxBlocks = 1024;  // records are sized for at most this many split CTAs
constexpr int kDecKBytes = kDecTile * 256;
constexpr int kDecVBytes = kDecTile * 256;
constexpr int kDecStageBytes = kDecKBytes + kDecVBytes;
__host__ __device__ constexpr int decode_smem_bytes(int G) {
  return kDecStages * kDecStageBytes + kDecConsumers * G * (kD + 2) * 4 +
         kDecConsumers * kDecTile * G * 4 + 2 * kDecStages * 8 + 16 + 128;
}
// records: one per (CTA b, unit u) that meet, at index b + u (unique, and the
// records of a unit are consecutive)
__host__ __device__ inline size_t decode_records(int units) { return (size_t)units + kDecMaxBlocks; }

// one block of 1024 threads: T[u] = sum_{u' < u} ceil(slots_u' / 32), T[units] = total
__global__ void __launch_bounds__(1024) decode_plan_kernel(int units,
                                                           const int32_t* __restrict__ counts,
                                                           int tail_slot, int32_t* __restrict__ T) {
  __shared__ int32_t wsum[32];
  __shared__ int32_t carry;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) carry = 0;
  __syncthreads();
  for (int base = 0; base < units; base += 1024) {
    const int u = base + threadIdx.x;
    const int v = u < units ? (counts[u] + tail_slot + kDecTile - 1) / kDecTile : 0;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(kFull, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) wsum[warp] = x;
    __syncthreads();
    if (warp == 0) {
      int w = wsum[lane];
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(kFull, w, o);
        if (lane >= o) w += y;
      }
      wsum[lane] = w;  // inclusive over warps
    }
    __syncthreads();
    const int excl = carry + (warp > 0 ? wsum[warp - 1] : 0) + x - v;
    if (u < units) T[u] = excl;
    __syncthreads();
    if (threadIdx.x == 0) carry += wsum[31];
    __syncthreads();
  }
  if (threadIdx.x == 0) T[units] = carry;
}

__device__ __forceinline__ void consumers_sync() {
  asm volatile("bar.sync 1, %0;" ::"n"(kDecConsumers * 32) : "memory");
}

// grid = NB persistent CTAs, block = kDecThreads.  CTA b takes the global
// tiles [b per, (b + 1) per), per = ceil(T[units] / NB); its k-th tile goes
// through ring stage k % kDecStages (K and V rows as bulk copies) and is
// consumed by consumer warp k % kDecConsumers.  Logits as in DecGeo; the value
// sums with lane = four dimensions and the weights of a row read as one
// broadcast.  Every wait is bounded; after a timeout the CTA skips the
// remaining work but keeps its barrier sequence, and writes NaN records, so
// the affected query heads read NaN.
template <int G>
__global__ void __launch_bounds__(kDecThreads) decode_split_kernel(
    Prob p, const __nv_bfloat16* __restrict__ q, const __nv_bfloat16* __restrict__ pk,
    const __nv_bfloat16* __restrict__ pv, const int64_t* __restrict__ offsets,
    const int32_t* __restrict__ counts, const int32_t* __restrict__ T, int tail_slot,
    float scale_log2, float2* __restrict__ rec_ml, float* __restrict__ rec_acc) {
  using Geo = DecGeo<G>;
  extern __shared__ uint8_t dsm_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>(((uintptr_t)dsm_raw + 127) & ~(uintptr_t)127);
  uint8_t* kst = sm;                                  // [stage][32 rows][256 B]
  uint8_t* vst = sm + kDecStages * kDecKBytes;        // [stage][32 rows][256 B]
  // the regions read or written with 16-byte vectors (wacc: 512 B per warp and
  // head, pw: 128 B per warp and head) start on 16-byte boundaries
  float* wacc = reinterpret_cast<float*>(vst + kDecStages * kDecVBytes);  // [consumers][G][kD]
  float* pw = wacc + kDecConsumers * G * kD;  // [consumers][32 slots][G] softmax weights
  float* wm = pw + kDecConsumers * kDecTile * G;                          // [consumers][G]
  float* wl = wm + kDecConsumers * G;                                     // [consumers][G]
  uint64_t* bars = reinterpret_cast<uint64_t*>(wl + kDecConsumers * G);   // full, empty
  volatile int* abort_flag = reinterpret_cast<volatile int*>(bars + 2 * kDecStages);
  const uint32_t full0 = tc::saddr(bars), empty0 = tc::saddr(bars + kDecStages);

  const int units = p.units;
  const int total = T[units];
  const int per = (total + (int)gridDim.x - 1) / (int)gridDim.x;
  const int g0 = min(total, (int)blockIdx.x * per), g1 = min(total, g0 + per);
  if (g0 >= g1) return;  // uniform over the CTA, before any barrier
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // first unit of the range: the last u with T[u] <= g0
  int lo = 0, hi = units;
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (T[mid] <= g0) lo = mid;
    else hi = mid;
  }
  const int u_first = lo;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kDecStages; ++s) {
      tc::mbar_init(full0 + 8 * s, 1);
      tc::mbar_init(empty0 + 8 * s, 1);
    }
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();

  if (warp == 0) {
    if (lane == 0) {  // producer: tiles g0 .. g1-1 in order, across unit boundaries
      int u = u_first, issued = 0;
      for (int k = 0; k < g1 - g0; ++k) {
        const int gt = g0 + k;
        while (T[u + 1] <= gt) ++u;
        const int s = k % kDecStages;
        if (k >= kDecStages &&
            !tc::mbar_wait(empty0 + 8 * s, ((k / kDecStages) - 1) & 1, abort_flag))
          break;
        const int t = gt - T[u];
        int cnt = min(kDecTile, counts[u] + tail_slot - t * kDecTile);
        const int64_t s0 = offsets[u] + (int64_t)t * kDecTile;
        // (debug builds) a tile outside the packed cache is not copied: the
        // stage completes with no bytes and its outputs are invalid
        if (!CERTKV_IN_BOUNDS(s0 >= 0 && (p.capacity <= 0 || s0 + cnt <= p.capacity), p.status))
          cnt = 0;
        const size_t e0 = (size_t)s0 * kD;
        tc::mbar_expect_tx(full0 + 8 * s, (uint32_t)cnt * 512u);
        if (cnt > 0) {
          tc::bulk_load(tc::saddr(kst + s * kDecKBytes), pk + e0, (uint32_t)cnt * 256u,
                        full0 + 8 * s);
          tc::bulk_load(tc::saddr(vst + s * kDecVBytes), pv + e0, (uint32_t)cnt * 256u,
                        full0 + 8 * s);
        }
        issued = k + 1;
      }
      // the last copies must land before the CTA exits
      for (int k = issued > kDecStages ? issued - kDecStages : 0; k < issued; ++k) {
        volatile int dummy = 0;
        tc::mbar_wait(full0 + 8 * (k % kDecStages), (k / kDecStages) & 1, &dummy);
      }
    }
  } else {  // consumers: one segment per unit met
    const int cw = warp - 1, ct = threadIdx.x - 32;
    const int gi = lane % Geo::LPS;  // lane within its slot group
    const int gs = lane / Geo::LPS;  // slot group: slot = pass * SPP + gs
    const int myg = gi & (G - 1);    // head of the logits this lane ends with
    float* pwarp = pw + cw * kDecTile * G;
    for (int u = u_first; u < units && T[u] < g1; ++u) {
      const int ka = max(g0, T[u]) - g0, kb = min(g1, T[u + 1]) - g0;
      if (ka >= kb) continue;  // a unit without tiles (uniform over the consumers)
      const int bl = u / p.H, h = u - bl * p.H;
      // this lane's dimensions of the group's queries, as fp32 pairs:
      // G <= 8: the 16-byte chunks gi + LPS t of the row; G = 16: dims 4 gi .. 4 gi + 3
      float2 qr[Geo::NPAIR][G];
      load_query_slice<G>(q + ((size_t)bl * p.Hq + (size_t)h * G) * kD, lane, qr);
      const int slots = counts[u] + tail_slot;
      float m[G], l_own = 0.f;
      float2 acc[G][2];  // dimensions (4 lane, 4 lane + 1), (4 lane + 2, 4 lane + 3)
#pragma unroll
      for (int g = 0; g < G; ++g) {
        m[g] = -INFINITY;
        acc[g][0] = acc[g][1] = make_float2(0.f, 0.f);
      }
      for (int k = ka + ((cw - ka % kDecConsumers) + kDecConsumers) % kDecConsumers; k < kb;
           k += kDecConsumers) {
        const int s = k % kDecStages;
        // warp-uniform decision: every lane waits for the stage; a timeout or an
        // abort anywhere skips the tile for the whole warp
        bool skip = __any_sync(kFull, *abort_flag != 0);
        if (!skip) skip = !__all_sync(kFull, tc::mbar_wait(full0 + 8 * s, (k / kDecStages) & 1,
                                                           abort_flag));
        if (skip) continue;
        const int t = g0 + k - T[u];
        const int cnt = min(kDecTile, slots - t * kDecTile);
        // logits of (slot pass * SPP + gs, head myg); rows past cnt were not
        // copied and are masked below
        const uint8_t* kt = kst + s * kDecKBytes;
        float xl[Geo::NP];
#pragma unroll
        for (int ps = 0; ps < Geo::NP; ++ps) {
          const uint8_t* row = kt + (ps * Geo::SPP + gs) * 256;
          float2 x2[G];
#pragma unroll
          for (int g = 0; g < G; ++g) x2[g] = make_float2(0.f, 0.f);
          if constexpr (Geo::DPL >= 8) {
#pragma unroll
            for (int c = 0; c < Geo::DPL / 8; ++c) {
              const uint4 raw = *reinterpret_cast<const uint4*>(row + (gi + Geo::LPS * c) * 16);
              const float2 kp[4] = {make_float2(bf16lo(raw.x), bf16hi(raw.x)),
                                    make_float2(bf16lo(raw.y), bf16hi(raw.y)),
                                    make_float2(bf16lo(raw.z), bf16hi(raw.z)),
                                    make_float2(bf16lo(raw.w), bf16hi(raw.w))};
#pragma unroll
              for (int e = 0; e < 4; ++e)
#pragma unroll
                for (int g = 0; g < G; ++g) x2[g] = ffma2(qr[4 * c + e][g], kp[e], x2[g]);
            }
          } else {
            const uint2 raw = *reinterpret_cast<const uint2*>(row + gi * 8);
            const float2 kp[2] = {make_float2(bf16lo(raw.x), bf16hi(raw.x)),
                                  make_float2(bf16lo(raw.y), bf16hi(raw.y))};
#pragma unroll
            for (int e = 0; e < 2; ++e)
#pragma unroll
              for (int g = 0; g < G; ++g) x2[g] = ffma2(qr[e][g], kp[e], x2[g]);
          }
          float v[G];
#pragma unroll
          for (int g = 0; g < G; ++g) v[g] = x2[g].x + x2[g].y;
          xl[ps] = reduce_heads<G>(v, lane) * scale_log2;
        }
        // tile maximum of head myg, then every head's maximum on every lane
        float tm = -INFINITY;
#pragma unroll
        for (int ps = 0; ps < Geo::NP; ++ps)
          if (ps * Geo::SPP + gs < cnt) tm = fmaxf(tm, xl[ps]);
#pragma unroll
        for (int o = Geo::LPS; o < 32; o <<= 1) tm = fmaxf(tm, __shfl_xor_sync(kFull, tm, o));
        float m_own = 0.f, c_own = 0.f;
#pragma unroll
        for (int g = 0; g < G; ++g) {
          const float nm = fmaxf(m[g], __shfl_sync(kFull, tm, g));  // lane g holds head g
          const float corr = exp2f(m[g] - nm);
          m[g] = nm;
          acc[g][0] = fmul2(acc[g][0], make_float2(corr, corr));
          acc[g][1] = fmul2(acc[g][1], make_float2(corr, corr));
          if (g == myg) {
            m_own = nm;
            c_own = corr;
          }
        }
        l_own *= c_own;
#pragma unroll
        for (int ps = 0; ps < Geo::NP; ++ps) {
          const int slot = ps * Geo::SPP + gs;
          const float pe = slot < cnt ? exp2f(xl[ps] - m_own) : 0.f;
          l_own += pe;
          if (gi < G) pwarp[slot * G + gi] = pe;
        }
        __syncwarp();
        // values: lane = 4 dimensions; only the tile's cnt rows were copied; the
        // weights of a row are one broadcast read
        const uint8_t* vt = vst + s * kDecVBytes + lane * 8;
#pragma unroll 8
        for (int r = 0; r < cnt; ++r) {
          const uint2 raw = *reinterpret_cast<const uint2*>(vt + r * 256);
          const float2 v01 = make_float2(bf16lo(raw.x), bf16hi(raw.x));
          const float2 v23 = make_float2(bf16lo(raw.y), bf16hi(raw.y));
          float pj[G];
          if constexpr (G % 4 == 0) {
#pragma unroll
            for (int g = 0; g < G; g += 4) {
              const float4 w = *reinterpret_cast<const float4*>(pwarp + r * G + g);
              pj[g] = w.x;
              pj[g + 1] = w.y;
              pj[g + 2] = w.z;
              pj[g + 3] = w.w;
            }
          } else {
#pragma unroll
            for (int g = 0; g < G; ++g) pj[g] = pwarp[r * G + g];
          }
#pragma unroll
          for (int g = 0; g < G; ++g) {
            const float2 pp = make_float2(pj[g], pj[g]);
            acc[g][0] = ffma2(pp, v01, acc[g][0]);
            acc[g][1] = ffma2(pp, v23, acc[g][1]);
          }
        }
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(empty0 + 8 * s);
      }
      // the unit's record for this CTA: combine the consumer warps.  The sum of
      // head g: lanes gi = g of every slot group (lanes gi = g + G repeat them).
      float lt = gi < G ? l_own : 0.f;
#pragma unroll
      for (int o = Geo::LPS; o < 32; o <<= 1) lt += __shfl_xor_sync(kFull, lt, o);
#pragma unroll
      for (int g = 0; g < G; ++g) {
        if (lane == g) {
          wm[cw * G + g] = m[g];
          wl[cw * G + g] = lt;
        }
        *reinterpret_cast<float4*>(&wacc[(cw * G + g) * kD + lane * 4]) =
            make_float4(acc[g][0].x, acc[g][0].y, acc[g][1].x, acc[g][1].y);
      }
      consumers_sync();
      const bool failed = *abort_flag != 0;
      const size_t rec = (size_t)blockIdx.x + u;
      for (int idx = ct; idx < G * kD; idx += kDecConsumers * 32) {
        const int g = idx / kD, i = idx - g * kD;
        float M = -INFINITY;
#pragma unroll
        for (int wi = 0; wi < kDecConsumers; ++wi) M = fmaxf(M, wm[wi * G + g]);
        float L = 0.f, A = 0.f;
#pragma unroll
        for (int wi = 0; wi < kDecConsumers; ++wi) {
          if (wm[wi * G + g] > -INFINITY) {
            const float f = exp2f(wm[wi * G + g] - M);
            L += wl[wi * G + g] * f;
            A += wacc[(wi * G + g) * kD + i] * f;
          }
        }
        if (failed) {
          M = 0.f;
          L = A = __int_as_float(0x7fc00000);
        }
        rec_acc[(rec * G + g) * kD + i] = A;
        if (i == 0) rec_ml[rec * G + g] = make_float2(M, L);
      }
      consumers_sync();  // wm / wl / wacc are reused by the next unit
    }
  }
  __syncthreads();
}

// ---------------------------------------------------------------------------
// Tensor-core split kernel for G = 4, 8 and 16 query heads per KV head.  At
// G = 8 the CUDA-core consumer needs ~4 fp32 FMAs per byte of cache; here both
// products run as mma.sync m16n8k16 (bf16 in, fp32 accumulate) with the G
// query heads as the M rows (padded to 16 with zero rows for G = 4 and 8;
// the padded rows' results are dropped): S = Q K^T over 32 slots (4 n-blocks
// x 8 k-steps), online softmax per
// row in the log2 domain, then O += P V (2 k-blocks x 16 n-blocks) with P as a
// bf16 part plus the bf16 rounding of its remainder (fp32-level weights).  The tiles arrive by TMA with 128-byte swizzle (two boxes of
// 64 dimensions x 32 slots for K and for V), so the ldmatrix reads are free of
// bank conflicts; rows past the segment (the next segment's, or zeros past
// the cache) get weight 0.  Work split, records and merge as in
// decode_split_kernel.
constexpr int kTcStageBytes = 4 * 4096;  // K and V, two 64-dimension halves each
template <int G>
__host__ __device__ constexpr int decode_tc_smem_bytes() {
  return kDecStages * kTcStageBytes + kDecConsumers * G * kD * 4 + 2 * kDecConsumers * G * 4 +
         2 * kDecStages * 8 + 16 + 1024;
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                               uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&h);
}
// byte address of (slot, 16-byte chunk c of the 256-byte row) in a tile of 32
// rows stored as two 128-byte-swizzled halves of 4096 bytes
__device__ __forceinline__ uint32_t sw_addr(uint32_t tile, int slot, int c) {
  return tile + (uint32_t)((c >> 3) * 4096 + slot * 128 + (((c & 7) ^ (slot & 7)) << 4));
}

template <int G>
__global__ void __launch_bounds__(kDecThreads) decode_split_tc_kernel(
    const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV, Prob p,
    const __nv_bfloat16* __restrict__ q, const int64_t* __restrict__ offsets,
    const int32_t* __restrict__ counts, const int32_t* __restrict__ T, int tail_slot,
    float scale_log2, float2* __restrict__ rec_ml, float* __restrict__ rec_acc) {
  static_assert(G == 4 || G == 8 || G == 16,
                "the tensor-core decode takes 4, 8 or 16 query heads per KV head");
  constexpr bool kPadded = G < 8;  // rows G..7 of the first fragment row block are zero
  extern __shared__ uint8_t dsm_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>(((uintptr_t)dsm_raw + 1023) & ~(uintptr_t)1023);
  // stage s: K halves at + 0 / 4096, V halves at + 8192 / 12288
  float* wacc = reinterpret_cast<float*>(sm + kDecStages * kTcStageBytes);  // [consumers][G][kD]
  float* wm = wacc + kDecConsumers * G * kD;                                // [consumers][G]
  float* wl = wm + kDecConsumers * G;                                       // [consumers][G]
  uint64_t* bars = reinterpret_cast<uint64_t*>(wl + kDecConsumers * G);     // full, empty
  volatile int* abort_flag = reinterpret_cast<volatile int*>(bars + 2 * kDecStages);
  const uint32_t full0 = tc::saddr(bars), empty0 = tc::saddr(bars + kDecStages);
  const uint32_t stage0 = tc::saddr(sm);

  const int units = p.units;
  const int total = T[units];
  const int per = (total + (int)gridDim.x - 1) / (int)gridDim.x;
  const int g0 = min(total, (int)blockIdx.x * per), g1 = min(total, g0 + per);
  if (g0 >= g1) return;  // uniform over the CTA, before any barrier
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int lo = 0, hi = units;  // first unit of the range: the last u with T[u] <= g0
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (T[mid] <= g0) lo = mid;
    else hi = mid;
  }
  const int u_first = lo;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kDecStages; ++s) {
      tc::mbar_init(full0 + 8 * s, 1);
      tc::mbar_init(empty0 + 8 * s, 1);
    }
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();

  if (warp == 0) {
    if (lane == 0) {  // producer: tiles g0 .. g1-1 in order, four TMA boxes each
      int u = u_first, issued = 0;
      for (int k = 0; k < g1 - g0; ++k) {
        const int gt = g0 + k;
        while (T[u + 1] <= gt) ++u;
        const int s = k % kDecStages;
        if (k >= kDecStages &&
            !tc::mbar_wait(empty0 + 8 * s, ((k / kDecStages) - 1) & 1, abort_flag))
          break;
        const int t = gt - T[u];
        const int64_t s0 = offsets[u] + (int64_t)t * kDecTile;
        const int cnt = min(kDecTile, counts[u] + tail_slot - t * kDecTile);
        const uint32_t st = stage0 + (uint32_t)(s * kTcStageBytes);
        tc::mbar_expect_tx(full0 + 8 * s, (uint32_t)kTcStageBytes);
        // (debug builds) a tile that starts outside the packed cache is not
        // loaded: the boxes are then read at row 0 and weighted 0
        const int y = CERTKV_IN_BOUNDS(s0 >= 0 && (p.capacity <= 0 || s0 + cnt <= p.capacity),
                                       p.status)
                          ? (int)s0
                          : 0;
        tc::tma_load_2d(st, &tmK, 0, y, full0 + 8 * s);
        tc::tma_load_2d(st + 4096, &tmK, 64, y, full0 + 8 * s);
        tc::tma_load_2d(st + 8192, &tmV, 0, y, full0 + 8 * s);
        tc::tma_load_2d(st + 12288, &tmV, 64, y, full0 + 8 * s);
        issued = k + 1;
      }
      // the last copies must land before the CTA exits
      for (int k = issued > kDecStages ? issued - kDecStages : 0; k < issued; ++k) {
        volatile int dummy = 0;
        tc::mbar_wait(full0 + 8 * (k % kDecStages), (k / kDecStages) & 1, &dummy);
      }
    }
  } else {  // consumers: one segment per unit met
    const int cw = warp - 1, ct = threadIdx.x - 32;
    const int qr = lane >> 2, qc = lane & 3;  // fragment row (head), column pair
    // ldmatrix row addresses of this lane: matrix mi = lane / 8, row lane % 8
    const int mi = lane >> 3, mr = lane & 7;
    for (int u = u_first; u < units && T[u] < g1; ++u) {
      const int ka = max(g0, T[u]) - g0, kb = min(g1, T[u + 1]) - g0;
      if (ka >= kb) continue;  // a unit without tiles (uniform over the consumers)
      const int bl = u / p.H, h = u - bl * p.H;
      // Q as the A operand (rows 0..G-1 the group's heads, zero above), 8 k-steps
      const uint32_t* qg = reinterpret_cast<const uint32_t*>(q + ((size_t)bl * p.Hq + (size_t)h * G) * kD);
      uint32_t qa[8][4];
#pragma unroll
      for (int ks = 0; ks < 8; ++ks) {
        const int c0 = (16 * ks + 2 * qc) / 2;  // 32-bit word of dims 16 ks + 2 qc, +1
        const bool row = !kPadded || qr < G;
        qa[ks][0] = row ? __ldg(qg + qr * (kD / 2) + c0) : 0u;
        qa[ks][2] = row ? __ldg(qg + qr * (kD / 2) + c0 + 4) : 0u;
        if (G == 16) {
          qa[ks][1] = __ldg(qg + (qr + 8) * (kD / 2) + c0);
          qa[ks][3] = __ldg(qg + (qr + 8) * (kD / 2) + c0 + 4);
        } else {
          qa[ks][1] = qa[ks][3] = 0u;
        }
      }
      const int slots = counts[u] + tail_slot;
      float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;  // rows qr, qr + 8
      float o[16][4];
#pragma unroll
      for (int nd = 0; nd < 16; ++nd) o[nd][0] = o[nd][1] = o[nd][2] = o[nd][3] = 0.f;
      for (int k = ka + ((cw - ka % kDecConsumers) + kDecConsumers) % kDecConsumers; k < kb;
           k += kDecConsumers) {
        const int s = k % kDecStages;
        bool skip = __any_sync(kFull, *abort_flag != 0);
        if (!skip) skip = !__all_sync(kFull, tc::mbar_wait(full0 + 8 * s, (k / kDecStages) & 1,
                                                           abort_flag));
        if (skip) continue;
        const int t = g0 + k - T[u];
        const int cnt = min(kDecTile, slots - t * kDecTile);
        const uint32_t kt = stage0 + (uint32_t)(s * kTcStageBytes), vt = kt + 8192;
        // S = Q K^T: 4 n-blocks of 8 slots
        float sc[4][4];
#pragma unroll
        for (int nb = 0; nb < 4; ++nb) sc[nb][0] = sc[nb][1] = sc[nb][2] = sc[nb][3] = 0.f;
#pragma unroll
        for (int ks = 0; ks < 8; ++ks) {
#pragma unroll
          for (int np = 0; np < 2; ++np) {  // n-block pair (2 np, 2 np + 1)
            uint32_t b0, b1, b2, b3;
            // matrix mi: slots 8 (2 np + mi / 2) + mr, dims 16 ks + 8 (mi & 1)
            ldsm_x4(sw_addr(kt, 8 * (2 * np + (mi >> 1)) + mr, 2 * ks + (mi & 1)), b0, b1, b2, b3);
            mma_bf16_16816(sc[2 * np], qa[ks], b0, b1);
            mma_bf16_16816(sc[2 * np + 1], qa[ks], b2, b3);
          }
        }
        // online softmax (log2 domain) of rows qr and qr + 8 over the tile
        float tm0 = -INFINITY, tm1 = -INFINITY;
#pragma unroll
        for (int nb = 0; nb < 4; ++nb) {
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            const bool ok = 8 * nb + 2 * qc + e < cnt;
            sc[nb][e] = ok ? sc[nb][e] * scale_log2 : -INFINITY;
            sc[nb][2 + e] = ok ? sc[nb][2 + e] * scale_log2 : -INFINITY;
            tm0 = fmaxf(tm0, sc[nb][e]);
            tm1 = fmaxf(tm1, sc[nb][2 + e]);
          }
        }
        tm0 = fmaxf(tm0, __shfl_xor_sync(kFull, tm0, 1));
        tm0 = fmaxf(tm0, __shfl_xor_sync(kFull, tm0, 2));
        tm1 = fmaxf(tm1, __shfl_xor_sync(kFull, tm1, 1));
        tm1 = fmaxf(tm1, __shfl_xor_sync(kFull, tm1, 2));
        const float n0 = fmaxf(m0, tm0), n1 = fmaxf(m1, tm1);
        const float c0 = exp2f(m0 - n0), c1 = exp2f(m1 - n1);  // both -inf: no slot yet
        m0 = n0;
        m1 = n1;
        // P as the A operand of two k16 blocks, split into a bf16 part and the
        // bf16 rounding of its remainder (P = ph + pl to ~2^-16 relative), so
        // that the weights carry fp32 accuracy into the tensor-core products
        uint32_t ph[2][4], pl[2][4];
        float ps0 = 0.f, ps1 = 0.f;
#pragma unroll
        for (int nb = 0; nb < 4; ++nb) {
          const float p0 = n0 > -INFINITY ? exp2f(sc[nb][0] - n0) : 0.f;
          const float p1 = n0 > -INFINITY ? exp2f(sc[nb][1] - n0) : 0.f;
          const float p2 = n1 > -INFINITY ? exp2f(sc[nb][2] - n1) : 0.f;
          const float p3 = n1 > -INFINITY ? exp2f(sc[nb][3] - n1) : 0.f;
          ps0 += p0 + p1;
          ps1 += p2 + p3;
          const uint32_t h01 = pack_bf16(p0, p1), h23 = pack_bf16(p2, p3);
          const uint32_t l01 = pack_bf16(p0 - bf16lo(h01), p1 - bf16hi(h01));
          const uint32_t l23 = pack_bf16(p2 - bf16lo(h23), p3 - bf16hi(h23));
          ph[nb >> 1][(nb & 1) * 2 + 0] = h01;
          ph[nb >> 1][(nb & 1) * 2 + 1] = h23;
          pl[nb >> 1][(nb & 1) * 2 + 0] = l01;
          pl[nb >> 1][(nb & 1) * 2 + 1] = l23;
        }
        l0 = l0 * (n0 > -INFINITY ? c0 : 1.f) + ps0;
        l1 = l1 * (n1 > -INFINITY ? c1 : 1.f) + ps1;
        const float r0 = n0 > -INFINITY ? c0 : 1.f, r1 = n1 > -INFINITY ? c1 : 1.f;
#pragma unroll
        for (int nd = 0; nd < 16; ++nd) {
          o[nd][0] *= r0;
          o[nd][1] *= r0;
          o[nd][2] *= r1;
          o[nd][3] *= r1;
        }
        // O += P V: k16 blocks of slots, n-block pairs of dimensions
#pragma unroll
        for (int kb2 = 0; kb2 < 2; ++kb2) {
#pragma unroll
          for (int np = 0; np < 8; ++np) {
            uint32_t b0, b1, b2, b3;
            // matrix mi: slots 16 kb2 + 8 (mi & 1) + mr, dims 8 (2 np + mi / 2)
            ldsm_x4_t(sw_addr(vt, 16 * kb2 + 8 * (mi & 1) + mr, 2 * np + (mi >> 1)), b0, b1, b2,
                      b3);
            mma_bf16_16816(o[2 * np], ph[kb2], b0, b1);
            mma_bf16_16816(o[2 * np + 1], ph[kb2], b2, b3);
            mma_bf16_16816(o[2 * np], pl[kb2], b0, b1);
            mma_bf16_16816(o[2 * np + 1], pl[kb2], b2, b3);
          }
        }
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(empty0 + 8 * s);
      }
      // the row sums over the quad, then this warp's record slices
      l0 += __shfl_xor_sync(kFull, l0, 1);
      l0 += __shfl_xor_sync(kFull, l0, 2);
      l1 += __shfl_xor_sync(kFull, l1, 1);
      l1 += __shfl_xor_sync(kFull, l1, 2);
      const bool own_row = !kPadded || qr < G;  // padded rows are not the group's heads
      if (qc == 0 && own_row) {
        wm[cw * G + qr] = m0;
        wl[cw * G + qr] = l0;
        if (G == 16) {
          wm[cw * G + qr + 8] = m1;
          wl[cw * G + qr + 8] = l1;
        }
      }
#pragma unroll
      for (int nd = 0; nd < 16; ++nd) {
        const int d = 8 * nd + 2 * qc;
        if (own_row)
          *reinterpret_cast<float2*>(&wacc[(cw * G + qr) * kD + d]) = make_float2(o[nd][0], o[nd][1]);
        if (G == 16)
          *reinterpret_cast<float2*>(&wacc[(cw * G + qr + 8) * kD + d]) =
              make_float2(o[nd][2], o[nd][3]);
      }
      consumers_sync();
      const bool failed = *abort_flag != 0;
      const size_t rec = (size_t)blockIdx.x + u;
      for (int idx = ct; idx < G * kD; idx += kDecConsumers * 32) {
        const int g = idx / kD, i = idx - g * kD;
        float M = -INFINITY;
#pragma unroll
        for (int wi = 0; wi < kDecConsumers; ++wi) M = fmaxf(M, wm[wi * G + g]);
        float L = 0.f, A = 0.f;
#pragma unroll
        for (int wi = 0; wi < kDecConsumers; ++wi) {
          if (wm[wi * G + g] > -INFINITY) {
            const float f = exp2f(wm[wi * G + g] - M);
            L += wl[wi * G + g] * f;
            A += wacc[(wi * G + g) * kD + i] * f;
          }
        }
        if (failed) {
          M = 0.f;
          L = A = __int_as_float(0x7fc00000);
        }
        rec_acc[(rec * G + g) * kD + i] = A;
        if (i == 0) rec_ml[rec * G + g] = make_float2(M, L);
      }
      consumers_sync();  // wm / wl / wacc are reused by the next unit
    }
  }
  __syncthreads();
}

// The records of unit u, merged for query head g of its group (log2 domain):
// returns the running maximum and sum and this thread's dimension of the sum.
__device__ __forceinline__ void merge_records(const int32_t* __restrict__ T, int units, int nb,
                                              int u, int g, int G, int i,
                                              const float2* __restrict__ rec_ml,
                                              const float* __restrict__ rec_acc, float* M_out,
                                              float* L_out, float* A_out) {
  const int total = T[units];
  const int per = (total + nb - 1) / nb;
  const int ta = T[u], tb = T[u + 1];
  float M = -INFINITY, L = 0.f, A = 0.f;
  if (tb > ta && per > 0) {
    const int b_lo = ta / per, b_hi = (tb - 1) / per;
    for (int b = b_lo; b <= b_hi; ++b) M = fmaxf(M, rec_ml[((size_t)b + u) * G + g].x);
    for (int b = b_lo; b <= b_hi; ++b) {
      const size_t r = ((size_t)b + u) * G + g;
      const float2 ml = rec_ml[r];
      if (ml.x > -INFINITY) {
        const float f = exp2f(ml.x - M);
        L += ml.y * f;
        A += rec_acc[r * kD + i] * f;
      }
    }
  }
  *M_out = M;
  *L_out = L;
  *A_out = A;
}

// grid = units * G, block = 128: merge the records of one query head.
__global__ void __launch_bounds__(128) decode_merge_kernel(Prob p, int G, int nb,
                                                           const int32_t* __restrict__ T,
                                                           const float2* __restrict__ rec_ml,
                                                           const float* __restrict__ rec_acc,
                                                           __nv_bfloat16* __restrict__ out) {
  const int ug = blockIdx.x;
  const int u = ug / G, g = ug - u * G;
  const int i = threadIdx.x;
  float M, L, A;
  merge_records(T, p.units, nb, u, g, G, i, rec_ml, rec_acc, &M, &L, &A);
  // query head index: (b, l, h*G + g) -> [B*L][Hq]
  const int bl = u / p.H, h = u - bl * p.H;
  out[((size_t)bl * p.Hq + (size_t)h * G + g) * kD + i] = __float2bfloat16_rn(A / L);
}

// Sum over the 128 threads of the block (one per dimension).
__device__ __forceinline__ float block_sum128(float x, float* red) {
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) x += __shfl_xor_sync(kFull, x, o);
  __syncthreads();  // red may still be read from the previous reduction
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = x;
  __syncthreads();
  return (red[0] + red[1]) + (red[2] + red[3]);
}

// grid = units * G, block = 128 (thread = dimension): the real-slot records of
// one query head merged as in decode_merge_kernel, then the m cluster
// summaries added with weight n_g e^{lbar_g} (all weights relative to one
// log2-domain shift, to which the bound is invariant), then the certificate.
__global__ void __launch_bounds__(128) decode_certified_merge_kernel(
    Prob p, int G, int m, int tail_slot, float scale, const __nv_bfloat16* __restrict__ q,
    const __nv_bfloat16* __restrict__ pk, const __nv_bfloat16* __restrict__ pv,
    const int64_t* __restrict__ offsets, const int32_t* __restrict__ counts,
    const float4* __restrict__ cluster_meta, const float* __restrict__ kept_vmax, int nb,
    const int32_t* __restrict__ T, const float2* __restrict__ rec_ml,
    const float* __restrict__ rec_acc,
    __nv_bfloat16* __restrict__ out, float* __restrict__ bound, int32_t* __restrict__ certified) {
  __shared__ float red[4];
  __shared__ float s_lam[CERTKV_MAX_CLUSTERS], s_r[CERTKV_MAX_CLUSTERS];
  __shared__ float s_vn[CERTKV_MAX_CLUSTERS], s_rho[CERTKV_MAX_CLUSTERS];
  const int ug = blockIdx.x;
  const int u = ug / G, g = ug - u * G;
  const int i = threadIdx.x;
  const float kLog2e = 1.4426950408889634f;
  // real slots: merge of the records (log2 domain)
  float MS, LS, AS;
  merge_records(T, p.units, nb, u, g, G, i, rec_ml, rec_acc, &MS, &LS, &AS);
  const int bl = u / p.H, h = u - bl * p.H;
  const size_t qi = (size_t)bl * p.Hq + (size_t)h * G + g;
  const float qv = __bfloat162float(q[qi * kD + i]);
  const float qn = sqrtf(block_sum128(qv * qv, red));
  const int64_t s0 = offsets[u] + counts[u] + tail_slot;  // first summary slot
  // clusters: lbar (log2 domain, with log2 n_g), logit radius, ||vbar||, rho
  float M = MS;
  for (int c = 0; c < m; ++c) {
    const float4 meta = cluster_meta[(size_t)u * m + c];
    const float kb = __bfloat162float(pk[(s0 + c) * kD + i]);
    const float vb = __bfloat162float(pv[(s0 + c) * kD + i]);
    const float dot = block_sum128(qv * kb, red);
    const float vn = sqrtf(block_sum128(vb * vb, red));
    const float lam = meta.x > 0.f ? fmaf(dot, scale * kLog2e, log2f(meta.x)) : -INFINITY;
    if (i == 0) {
      s_lam[c] = lam;
      s_r[c] = scale * qn * meta.y;
      s_vn[c] = vn;
      s_rho[c] = meta.z;
    }
    M = fmaxf(M, lam);
  }
  __syncthreads();
  const float fS = MS > -INFINITY ? exp2f(MS - M) : 0.f;
  float num = AS * fS, Z = LS * fS;
  for (int c = 0; c < m; ++c) {
    if (!(s_lam[c] > -INFINITY)) continue;
    const float zg = exp2f(s_lam[c] - M);
    num = fmaf(zg, __bfloat162float(pv[(s0 + c) * kD + i]), num);
    Z += zg;
  }
  out[qi * kD + i] = __float2bfloat16_rn(num / Z);
  if (i == 0) {
    // a few scalars per query head, in float64: e^r (e^r - 1) overflows fp32
    // from r = 44 on, which a strong key in a cluster reaches with a unit
    // query; the bound is stored as fp32 (+inf when it exceeds its range)
    double DZ = 0.0, DN = 0.0, vmax = kept_vmax[u];
    for (int c = 0; c < m; ++c) {
      if (!(s_lam[c] > -INFINITY)) continue;
      const double zg = exp2((double)(s_lam[c] - M));
      const double er = exp((double)s_r[c]);
      DZ += (er - 1.0) * er * zg;
      DN += er * zg * ((er - 1.0) * s_vn[c] + s_rho[c]);
      vmax = fmax(vmax, (double)(s_vn[c] + s_rho[c]));
    }
    bound[qi] = (float)(3.0 / Z * (DN + vmax * DZ));
    certified[qi] = DZ <= Z / 3.0 ? 1 : 0;
  }
}

namespace {
struct DecodeLayout {
  size_t T, ml, acc, total;
};
DecodeLayout decode_layout(const Prob& p) {
  auto a = [](size_t x) { return (x + 255) / 256 * 256; };
  const size_t recs = decode_records(p.units) * p.G;
  DecodeLayout ly;
  ly.T = 0;
  ly.ml = a(((size_t)p.units + 1) * sizeof(int32_t));
  ly.acc = ly.ml + a(recs * sizeof(float2));
  ly.total = ly.acc + recs * kD * sizeof(float);
  return ly;
}

// CTAs of the persistent split kernel: as many as fit on the device at once
// (set up once per device: the shared-memory opt-in and the occupancy query)
constexpr int kDecMaxDevices = 64;
template <int G>
int split_blocks() {
  static int cached[kDecMaxDevices] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 0;
  if (dev < kDecMaxDevices && cached[dev] > 0) return cached[dev];
  int sms = 0, per_sm = 0;
  if (cudaFuncSetAttribute(decode_split_kernel<G>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           decode_smem_bytes(G)) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decode_split_kernel<G>, kDecThreads,
                                                    decode_smem_bytes(G)) != cudaSuccess ||
      per_sm < 1 || sms < 1)
    return 0;
  const int nb = sms * per_sm < kDecMaxBlocks ? sms * per_sm : kDecMaxBlocks;
  if (dev < kDecMaxDevices) cached[dev] = nb;
  return nb;
}

template <int G>
int launch_split(const Prob& p, const __nv_bfloat16* q, const __nv_bfloat16* pk,
                 const __nv_bfloat16* pv, const int64_t* offsets, const int32_t* counts,
                 const int32_t* T, int tail_slot, float sl2, float2* ml, float* acc,
                 cudaStream_t st) {
  const int nb = split_blocks<G>();
  if (nb < 1) return 0;
  TraceScope ts_("decode_split", st);
  decode_split_kernel<G><<<nb, kDecThreads, decode_smem_bytes(G), st>>>(
      p, q, pk, pv, offsets, counts, T, tail_slot, sl2, ml, acc);
  return nb;
}

template <int G>
int split_tc_blocks() {
  static int cached[kDecMaxDevices] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 0;
  if (dev < kDecMaxDevices && cached[dev] > 0) return cached[dev];
  int sms = 0, per_sm = 0;
  if (cudaFuncSetAttribute(decode_split_tc_kernel<G>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           decode_tc_smem_bytes<G>()) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decode_split_tc_kernel<G>,
                                                    kDecThreads, decode_tc_smem_bytes<G>()) !=
          cudaSuccess ||
      per_sm < 1 || sms < 1)
    return 0;
  const int nb = sms * per_sm < kDecMaxBlocks ? sms * per_sm : kDecMaxBlocks;
  if (dev < kDecMaxDevices) cached[dev] = nb;
  return nb;
}

// the tensor-core split kernel (G = 8, 16); 0 if it cannot run (no tensor
// maps for the packed cache, or no occupancy)
template <int G>
int launch_split_tc(const Prob& p, const __nv_bfloat16* q, const void* pk, const void* pv,
                    const int64_t* offsets, const int32_t* counts, const int32_t* T, int tail_slot,
                    float sl2, float2* ml, float* acc, cudaStream_t st) {
  if (p.capacity <= 0) return 0;
  CUtensorMap mk, mv;
  if (!make_row_map(&mk, pk, (uint64_t)p.capacity, kDecTile) ||
      !make_row_map(&mv, pv, (uint64_t)p.capacity, kDecTile))
    return 0;
  const int nb = split_tc_blocks<G>();
  if (nb < 1) return 0;
  TraceScope ts_("decode_split", st);
  decode_split_tc_kernel<G><<<nb, kDecThreads, decode_tc_smem_bytes<G>(), st>>>(
      mk, mv, p, q, offsets, counts, T, tail_slot, sl2, ml, acc);
  return nb;
}

// plan + split kernels; returns the number of split CTAs (0: nothing launched)
int run_splits(const Prob& p, const void* q, const void* pk, const void* pv,
               const int64_t* offsets, const int32_t* counts, int tail_slot, float scale,
               char* ws, cudaStream_t st) {
  const DecodeLayout ly = decode_layout(p);
  int32_t* T = reinterpret_cast<int32_t*>(ws + ly.T);
  float2* ml = reinterpret_cast<float2*>(ws + ly.ml);
  float* acc = reinterpret_cast<float*>(ws + ly.acc);
  {
    TraceScope ts_("decode_plan", st);
    decode_plan_kernel<<<1, 1024, 0, st>>>(p.units, counts, tail_slot, T);
  }
  const float sl2 = scale * 1.4426950408889634f;
  const __nv_bfloat16* qb = reinterpret_cast<const __nv_bfloat16*>(q);
  const __nv_bfloat16* kb = reinterpret_cast<const __nv_bfloat16*>(pk);
  const __nv_bfloat16* vb = reinterpret_cast<const __nv_bfloat16*>(pv);
  switch (p.G) {
    case 1: return launch_split<1>(p, qb, kb, vb, offsets, counts, T, tail_slot, sl2, ml, acc, st);
    case 2: return launch_split<2>(p, qb, kb, vb, offsets, counts, T, tail_slot, sl2, ml, acc, st);
    case 4: {
      const int nb = launch_split_tc<4>(p, qb, pk, pv, offsets, counts, T, tail_slot, sl2, ml, acc, st);
      return nb > 0 ? nb : launch_split<4>(p, qb, kb, vb, offsets, counts, T, tail_slot, sl2, ml, acc, st);
    }
    case 8: {
      const int nb = launch_split_tc<8>(p, qb, pk, pv, offsets, counts, T, tail_slot, sl2, ml, acc, st);
      return nb > 0 ? nb : launch_split<8>(p, qb, kb, vb, offsets, counts, T, tail_slot, sl2, ml, acc, st);
    }
    case 16: {
      const int nb = launch_split_tc<16>(p, qb, pk, pv, offsets, counts, T, tail_slot, sl2, ml, acc, st);
      return nb > 0 ? nb : launch_split<16>(p, qb, kb, vb, offsets, counts, T, tail_slot, sl2, ml, acc, st);
    }
    default: return 0;
  }
}
}  // namespace

size_t decode_workspace(const Prob& p) { return decode_layout(p).total; }

bool launch_decode(const Prob& p, const void* q, const void* pk, const void* pv,
                   const int64_t* offsets, const int32_t* counts, int tail_slot, float scale,
                   void* out, char* ws, cudaStream_t st) {
  const int nb = run_splits(p, q, pk, pv, offsets, counts, tail_slot, scale, ws, st);
  if (nb < 1) return false;
  const DecodeLayout ly = decode_layout(p);
  {
    TraceScope ts_("decode_merge", st);
    decode_merge_kernel<<<p.units * p.G, 128, 0, st>>>(
        p, p.G, nb, reinterpret_cast<const int32_t*>(ws + ly.T),
        reinterpret_cast<const float2*>(ws + ly.ml), reinterpret_cast<const float*>(ws + ly.acc),
        reinterpret_cast<__nv_bfloat16*>(out));
  }
  return true;
}

bool launch_decode_certified(const Prob& p, const void* q, const void* pk, const void* pv,
                             const int64_t* offsets, const int32_t* counts, int tail_slot,
                             int clusters, const float* cluster_meta, const float* kept_vmax,
                             float scale, void* out, float* bound, int32_t* certified, char* ws,
                             cudaStream_t st) {
  // the real slots only: the splits see no tail slot
  const int nb = run_splits(p, q, pk, pv, offsets, counts, 0, scale, ws, st);
  if (nb < 1) return false;
  const DecodeLayout ly = decode_layout(p);
  {
    TraceScope ts_("decode_certified_merge", st);
    decode_certified_merge_kernel<<<p.units * p.G, 128, 0, st>>>(
        p, p.G, clusters, tail_slot, scale, reinterpret_cast<const __nv_bfloat16*>(q),
        reinterpret_cast<const __nv_bfloat16*>(pk), reinterpret_cast<const __nv_bfloat16*>(pv),
        offsets, counts, reinterpret_cast<const float4*>(cluster_meta), kept_vmax, nb,
        reinterpret_cast<const int32_t*>(ws + ly.T), reinterpret_cast<const float2*>(ws + ly.ml),
        reinterpret_cast<const float*>(ws + ly.acc), reinterpret_cast<__nv_bfloat16*>(out), bound,
        certified);
  }
  return true;
}

}  // namespace certkv
