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
// CTA one thread streams the tiles into a ring of shared-memory stages with
// the TMA (K through a 2-D tensor map with the 128-byte swizzle, so that a lane
// reading its own slot's row meets no bank conflict; V as one contiguous bulk
// copy), and the consumer warps keep online (max, sum, acc) for the G query
// heads of the current unit; where the range crosses into the next unit they
// combine their states into one record for (CTA, unit).  Every packed K/V
// byte is read once per step, in whole tiles.  A merge kernel combines the
// records of each unit in the log-sum-exp domain.
#include "../../include/certkv.h"
#include "common.cuh"
#include "internal.cuh"
#include "tma.cuh"

namespace certkv {

#ifndef CERTKV_DEC_STAGES
#define CERTKV_DEC_STAGES 5
#endif
#ifndef CERTKV_DEC_CONSUMERS
#define CERTKV_DEC_CONSUMERS 5
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
constexpr int kDecKBytes = kDecTile * 256;  // two 4 KB boxes of 64 columns
constexpr int kDecVBytes = kDecTile * 256;
constexpr int kDecStageBytes = kDecKBytes + kDecVBytes;
static_assert(kDecKBytes % 1024 == 0 && kDecVBytes % 1024 == 0,
              "the swizzled K boxes need 1024-B alignment");
__host__ __device__ constexpr int decode_smem_bytes(int G) {
  return kDecStages * kDecStageBytes + G * kD * 2 + kDecConsumers * G * (kD + 2) * 4 +
         kDecConsumers * kDecTile * G * 4 + 2 * kDecStages * 8 + 16 + 1024;
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
// through ring stage k % kDecStages and is consumed by consumer warp
// k % kDecConsumers.  A consumer lane owns one slot for the logits (its K row
// read from the swizzled stage, the query broadcast from shared memory) and
// four dimensions for the value sums.  Every wait is bounded; after a timeout
// the CTA skips the remaining work but keeps its barrier sequence, and writes
// NaN records, so the affected query heads read NaN.
template <int G>
__global__ void __launch_bounds__(kDecThreads) decode_split_kernel(
    const __grid_constant__ CUtensorMap map_k, Prob p, const __nv_bfloat16* __restrict__ q,
    const __nv_bfloat16* __restrict__ pv, const int64_t* __restrict__ offsets,
    const int32_t* __restrict__ counts, const int32_t* __restrict__ T, int tail_slot,
    float scale_log2, float2* __restrict__ rec_ml, float* __restrict__ rec_acc) {
  extern __shared__ uint8_t dsm_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>(((uintptr_t)dsm_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* kst = sm;                                                    // [stage][2][32][128 B]
  uint8_t* vst = sm + kDecStages * kDecKBytes;                          // [stage][32][256 B]
  // every region that is read or written with 16-byte vectors starts on a
  // 16-byte boundary: qs (256 B per head), wacc (512 B per warp and head) and pw
  // (128 B per warp and head) come first, the scalar arrays after them
  uint32_t* qs = reinterpret_cast<uint32_t*>(vst + kDecStages * kDecVBytes);  // [G][kD / 2] bf16 pairs
  float* wacc = reinterpret_cast<float*>(qs + G * kD / 2);              // [consumers][G][kD]
  float* pw = wacc + kDecConsumers * G * kD;  // [consumers][32 slots][G] softmax weights
  float* wm = pw + kDecConsumers * kDecTile * G;                        // [consumers][G]
  float* wl = wm + kDecConsumers * G;                                   // [consumers][G]
  uint64_t* bars = reinterpret_cast<uint64_t*>(wl + kDecConsumers * G);  // full, empty (8-B aligned)
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
        const int cnt = min(kDecTile, counts[u] + tail_slot - t * kDecTile);
        const int64_t row0 = offsets[u] + (int64_t)t * kDecTile;
        tc::mbar_expect_tx(full0 + 8 * s, (uint32_t)(kDecKBytes + cnt * 256));
        const uint32_t kd = tc::saddr(kst + s * kDecKBytes);
        tc::tma_load_2d(kd, &map_k, 0, (int)row0, full0 + 8 * s);
        tc::tma_load_2d(kd + kDecKBytes / 2, &map_k, 64, (int)row0, full0 + 8 * s);
        tc::bulk_load(tc::saddr(vst + s * kDecVBytes), pv + row0 * kD, (uint32_t)cnt * 256u,
                      full0 + 8 * s);
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
    const uint4* q4 = reinterpret_cast<const uint4*>(qs);  // 8 bf16 dimensions per load
    for (int u = u_first; u < units && T[u] < g1; ++u) {
      const int ka = max(g0, T[u]) - g0, kb = min(g1, T[u + 1]) - g0;
      if (ka >= kb) continue;  // a unit without tiles (uniform over the consumers)
      const int bl = u / p.H, h = u - bl * p.H;
      // the group's queries as their bf16 pairs (the scale is applied to the dot
      // products)
      const uint32_t* qu =
          reinterpret_cast<const uint32_t*>(q + ((size_t)bl * p.Hq + (size_t)h * G) * kD);
      for (int i = ct; i < G * kD / 2; i += kDecConsumers * 32) qs[i] = qu[i];
      consumers_sync();
      const int slots = counts[u] + tail_slot;
      float m[G], l[G];
      float2 acc[G][2];  // dimensions (4 lane, 4 lane + 1), (4 lane + 2, 4 lane + 3)
#pragma unroll
      for (int g = 0; g < G; ++g) {
        m[g] = -INFINITY;
        l[g] = 0.f;
        acc[g][0] = acc[g][1] = make_float2(0.f, 0.f);
      }
      float* pwarp = pw + cw * kDecTile * G;
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
        const bool ok = lane < cnt;
        // logits: lane = slot; chunk c of the row sits at chunk (c ^ (row & 7))
        // of its 128-byte box row; even and odd dimensions in the two halves of
        // a packed f32x2 accumulator
        const uint8_t* krow = kst + s * kDecKBytes + lane * 128;
        float2 x2[G];
#pragma unroll
        for (int g = 0; g < G; ++g) x2[g] = make_float2(0.f, 0.f);
#pragma unroll
        for (int c = 0; c < 16; ++c) {
          const uint4 raw = *reinterpret_cast<const uint4*>(krow + (c >> 3) * (kDecKBytes / 2) +
                                                            (((c & 7) ^ (lane & 7)) << 4));
          const float2 k0 = make_float2(bf16lo(raw.x), bf16hi(raw.x));
          const float2 k1 = make_float2(bf16lo(raw.y), bf16hi(raw.y));
          const float2 k2 = make_float2(bf16lo(raw.z), bf16hi(raw.z));
          const float2 k3 = make_float2(bf16lo(raw.w), bf16hi(raw.w));
#pragma unroll
          for (int g = 0; g < G; ++g) {
            const uint4 qq = q4[g * (kD / 8) + c];
            x2[g] = ffma2(make_float2(bf16lo(qq.x), bf16hi(qq.x)), k0, x2[g]);
            x2[g] = ffma2(make_float2(bf16lo(qq.y), bf16hi(qq.y)), k1, x2[g]);
            x2[g] = ffma2(make_float2(bf16lo(qq.z), bf16hi(qq.z)), k2, x2[g]);
            x2[g] = ffma2(make_float2(bf16lo(qq.w), bf16hi(qq.w)), k3, x2[g]);
          }
        }
#pragma unroll
        for (int g = 0; g < G; ++g) {
          const float xv = ok ? (x2[g].x + x2[g].y) * scale_log2 : -INFINITY;
          const float nm = fmaxf(m[g], warp_max(xv));
          const float corr = exp2f(m[g] - nm);
          m[g] = nm;
          l[g] *= corr;
          acc[g][0] = fmul2(acc[g][0], make_float2(corr, corr));
          acc[g][1] = fmul2(acc[g][1], make_float2(corr, corr));
          const float pe = ok ? exp2f(xv - nm) : 0.f;
          l[g] += pe;
          pwarp[lane * G + g] = pe;
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
      // the unit's record for this CTA: combine the consumer warps
#pragma unroll
      for (int g = 0; g < G; ++g) {
        float lt = l[g];
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) lt += __shfl_xor_sync(kFull, lt, o);
        if (lane == 0) {
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
      consumers_sync();  // wm / wl / wacc and qs are reused by the next unit
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
    float DZ = 0.f, DN = 0.f, vmax = kept_vmax[u];
    for (int c = 0; c < m; ++c) {
      if (!(s_lam[c] > -INFINITY)) continue;
      const float zg = exp2f(s_lam[c] - M);
      const float er = expf(s_r[c]);
      DZ += (er - 1.f) * er * zg;
      DN += er * zg * ((er - 1.f) * s_vn[c] + s_rho[c]);
      vmax = fmaxf(vmax, s_vn[c] + s_rho[c]);
    }
    bound[qi] = 3.f / Z * (DN + vmax * DZ);
    certified[qi] = DZ <= Z / 3.f ? 1 : 0;
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
int launch_split(const Prob& p, const CUtensorMap& map_k, const __nv_bfloat16* q,
                 const __nv_bfloat16* pv, const int64_t* offsets, const int32_t* counts,
                 const int32_t* T, int tail_slot, float sl2, float2* ml, float* acc,
                 cudaStream_t st) {
  const int nb = split_blocks<G>();
  if (nb < 1) return 0;
  TraceScope ts_("decode_split", st);
  decode_split_kernel<G><<<nb, kDecThreads, decode_smem_bytes(G), st>>>(
      map_k, p, q, pv, offsets, counts, T, tail_slot, sl2, ml, acc);
  return nb;
}

// plan + split kernels; returns the number of split CTAs (0: nothing launched)
int run_splits(const Prob& p, const void* q, const void* pk, const void* pv, int64_t rows,
               const int64_t* offsets, const int32_t* counts, int tail_slot, float scale,
               char* ws, cudaStream_t st) {
  CUtensorMap map_k;
  if (rows < 1 || rows > INT32_MAX || !make_row_map(&map_k, pk, (uint64_t)rows, kDecTile))
    return 0;
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
  const __nv_bfloat16* vb = reinterpret_cast<const __nv_bfloat16*>(pv);
  switch (p.G) {
    case 1: return launch_split<1>(p, map_k, qb, vb, offsets, counts, T, tail_slot, sl2, ml, acc, st);
    case 2: return launch_split<2>(p, map_k, qb, vb, offsets, counts, T, tail_slot, sl2, ml, acc, st);
    case 4: return launch_split<4>(p, map_k, qb, vb, offsets, counts, T, tail_slot, sl2, ml, acc, st);
    case 8: return launch_split<8>(p, map_k, qb, vb, offsets, counts, T, tail_slot, sl2, ml, acc, st);
    case 16: return launch_split<16>(p, map_k, qb, vb, offsets, counts, T, tail_slot, sl2, ml, acc, st);
    default: return 0;
  }
}
}  // namespace

size_t decode_workspace(const Prob& p) { return decode_layout(p).total; }

bool launch_decode(const Prob& p, const void* q, const void* pk, const void* pv, int64_t rows,
                   const int64_t* offsets, const int32_t* counts, int tail_slot, float scale,
                   void* out, char* ws, cudaStream_t st) {
  const int nb = run_splits(p, q, pk, pv, rows, offsets, counts, tail_slot, scale, ws, st);
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
                             int64_t rows, const int64_t* offsets, const int32_t* counts,
                             int tail_slot, int clusters, const float* cluster_meta,
                             const float* kept_vmax, float scale, void* out, float* bound,
                             int32_t* certified, char* ws, cudaStream_t st) {
  // the real slots only: the splits see no tail slot
  const int nb = run_splits(p, q, pk, pv, rows, offsets, counts, 0, scale, ws, st);
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
