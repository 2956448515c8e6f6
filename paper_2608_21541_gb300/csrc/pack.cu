// pack.cu — a6 select, a7 tail slot, a8 packed cache.
//
//   tail    (k*, v*) = sum_{E} a_j (k_j, v_j) / m over the evicted ranks
//           b_h..n-1 (§4: the key and value centroids of the evicted suffix
//           under r_j = a_j / m), from the chunk suffix sums plus the partial
//           chunk, in double-float; rounded once to bf16 into the last slot.
//           The V and m suffix sums come from the curve's prefix kernel; the
//           K ones, needed at this one chunk only, are folded here from the
//           chunk sums in the same order (last chunk down).
//   select  top-b_h real tokens = ranks 0..b_h-1; emitted in ascending
//           position by comparing each token's sort key with the first
//           evicted one (a threshold) and compacting in position order.
//   copy    gathers the kept K and V rows bit-exactly into the packed cache.
#include "common.cuh"
#include "internal.cuh"

namespace certkv {

// stored radii and norms are rounded up by this factor so that they stay upper
// bounds (fp32 sums of 128 squares and square roots are within a few 1e-6)
constexpr float kRadiusRoundUp = 1.0f + 1e-5f;

// grid = units, block = 128 (one thread per dimension)
__global__ void __launch_bounds__(128) tail_kernel(
    Prob p, const uint32_t* __restrict__ keys, const int32_t* __restrict__ perm,
    const __nv_bfloat16* __restrict__ K, const __nv_bfloat16* __restrict__ V,
    const float4* __restrict__ base_mq, const float2* __restrict__ base_v,
    const float* __restrict__ agg_k, const int32_t* __restrict__ counts,
    const int64_t* __restrict__ offsets, __nv_bfloat16* __restrict__ pk,
    __nv_bfloat16* __restrict__ pv, int32_t* __restrict__ positions, float* __restrict__ tail_f32,
    double* __restrict__ tail_mass, uint32_t* status) {
  const int u = blockIdx.x, i = threadIdx.x;
  const int n = p.n;
  const int b = counts[u];
  if (!CERTKV_IN_BOUNDS(b >= 0 && b < n, p.status)) return;
  if (!CERTKV_IN_BOUNDS(p.capacity <= 0 || offsets[u] + b < p.capacity, p.status)) return;
  const uint32_t* ku = keys + (size_t)u * n;
  const int32_t* pu = perm + (size_t)u * n;
  const __nv_bfloat16* Ku = K + (size_t)u * n * kD;
  const __nv_bfloat16* Vu = V + (size_t)u * n * kD;
  const int kb = b / kChunk;
  const int r_end = min(n, (kb + 1) * kChunk);
  const size_t ci = (size_t)u * p.chunks + kb;
  const float4 bmq = base_mq[ci];
  DF m{bmq.x, bmq.y};
  float2 t = base_v[ci * kD + i];
  DF tv{t.x, t.y};
  // the K sums over the chunks after chunk kb, folded from the last chunk
  // down; the next 32 chunks' loads are in flight while 32 are folded
  DF tk = df_make(0.f);
  {
    const float* src = agg_k + (size_t)u * p.chunks * kD + i;
    float nxt[32];
#pragma unroll
    for (int e = 0; e < 32; ++e) {
      const int c = p.chunks - 1 - e;
      nxt[e] = c > kb ? src[(size_t)c * kD] : 0.f;
    }
    for (int top = p.chunks - 1; top > kb; top -= 32) {
      float x[32];
#pragma unroll
      for (int e = 0; e < 32; ++e) {
        x[e] = nxt[e];
        const int c = top - 32 - e;
        nxt[e] = c > kb ? src[(size_t)c * kD] : 0.f;
      }
#pragma unroll
      for (int e = 0; e < 32; ++e)
        if (top - e > kb) tk = df_add_f(tk, x[e]);
    }
  }
  // the partial chunk's scores and token indices staged once; then the K and
  // V values of sixteen ranks at a time in flight, summed in rank order
  __shared__ float s_a[kChunk];
  __shared__ int s_j[kChunk];
  if (b + i < r_end) {
    int j = pu[b + i];
    if (!CERTKV_IN_BOUNDS(j >= 0 && j < n, p.status)) j = 0;
    s_a[i] = key_score(ku[b + i]);
    s_j[i] = j;
  }
  __syncthreads();
  for (int r0 = b; r0 < r_end; r0 += 16) {
    float vv[16], kv[16];
#pragma unroll
    for (int e = 0; e < 16; ++e) {
      vv[e] = kv[e] = 0.f;
      if (r0 + e < r_end) {
        const size_t o = (size_t)s_j[r0 + e - b] * kD + i;
        vv[e] = __bfloat162float(Vu[o]);
        kv[e] = __bfloat162float(Ku[o]);
      }
    }
#pragma unroll
    for (int e = 0; e < 16; ++e) {
      if (r0 + e >= r_end) break;
      const float a = s_a[r0 + e - b];
      m = df_add_f(m, a);
      tv = df_add(tv, two_prod(a, vv[e]));
      tk = df_add(tk, two_prod(a, kv[e]));
    }
  }
  DF ks, vs;
  if (m.hi > 0.0f) {
    ks = df_div(tk, m);
    vs = df_div(tv, m);
  } else {  // zero tail mass in floating point: uniform mean of the tail
    DF sk = df_make(0.f), sv = df_make(0.f);
    for (int r = b; r < n; ++r) {
      int j = pu[r];
      if (!CERTKV_IN_BOUNDS(j >= 0 && j < n, p.status)) j = 0;
      sv = df_add_f(sv, __bfloat162float(Vu[(size_t)j * kD + i]));
      sk = df_add_f(sk, __bfloat162float(Ku[(size_t)j * kD + i]));
    }
    const DF cnt = df_make((float)(n - b));
    ks = df_div(sk, cnt);
    vs = df_div(sv, cnt);
    if (i == 0) raise_status(status, 2u);
  }
  const int64_t slot = offsets[u] + b;
  reinterpret_cast<uint16_t*>(pk)[slot * kD + i] = df_to_bf16(ks.hi, ks.lo);
  reinterpret_cast<uint16_t*>(pv)[slot * kD + i] = df_to_bf16(vs.hi, vs.lo);
  if (i == 0) positions[slot] = -1;
  if (tail_f32) {
    tail_f32[((size_t)u * 2 + 0) * kD + i] = ks.hi;
    tail_f32[((size_t)u * 2 + 1) * kD + i] = vs.hi;
  }
  if (tail_mass && i == 0) tail_mass[u] = df_to_double(m);
}

// grid = units, block = 1024: positions of the kept tokens in ascending order.
__global__ void __launch_bounds__(1024, 2) select_kernel(Prob p, const float* __restrict__ a,
                                                      const uint32_t* __restrict__ keys,
                                                      const int32_t* __restrict__ perm,
                                                      const int32_t* __restrict__ counts,
                                                      const int64_t* __restrict__ offsets,
                                                      int32_t* __restrict__ positions,
                                                      uint32_t* status) {
  // per-warp totals, double-buffered by round: a round's buffer is rewritten
  // two rounds later, after two more barriers, so two barriers per round
  // suffice; every thread keeps the same running offset `carry`
  __shared__ int warp_tot2[2][32];
  int carry = 0;
  const int u = blockIdx.x;
  const int n = p.n;
  const int b = counts[u];
  if (!CERTKV_IN_BOUNDS(b >= 0 && b < n, p.status)) return;
  if (!CERTKV_IN_BOUNDS(p.capacity <= 0 || offsets[u] + b <= p.capacity, p.status)) return;
  const uint32_t kt = keys[(size_t)u * n + b];  // first evicted rank
  const int jt = perm[(size_t)u * n + b];
  const float* au = a + (size_t)u * n;
  int32_t* out = positions + offsets[u];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  constexpr int kPer = 4;
  // the next round's scores are loaded while this round is ranked
  float x[kPer];
#pragma unroll
  for (int e = 0; e < kPer; ++e) {
    const int j = threadIdx.x * kPer + e;
    x[e] = j < n ? au[j] : 0.f;
  }
  for (int base = 0, round = 0; base < n; base += blockDim.x * kPer, ++round) {
    int* warp_tot = warp_tot2[round & 1];
    int j0 = base + threadIdx.x * kPer;
    bool kept[kPer];
    int cnt = 0;
#pragma unroll
    for (int e = 0; e < kPer; ++e) {
      int j = j0 + e;
      bool k = false;
      if (j < n) {
        uint32_t kj = score_key(x[e]);
        k = (kj < kt) || (kj == kt && j < jt);
      }
      kept[e] = k;
      cnt += k;
    }
#pragma unroll
    for (int e = 0; e < kPer; ++e) {
      const int j = j0 + blockDim.x * kPer + e;
      x[e] = j < n ? au[j] : 0.f;
    }
    int incl = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      int y = __shfl_up_sync(kFull, incl, o);
      if (lane >= o) incl += y;
    }
    if (lane == 31) warp_tot[warp] = incl;
    __syncthreads();
    if (warp == 0) {
      int t = lane < (int)(blockDim.x >> 5) ? warp_tot[lane] : 0;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        int y = __shfl_up_sync(kFull, t, o);
        if (lane >= o) t += y;
      }
      warp_tot[lane] = t;
    }
    __syncthreads();
    int pos = carry + (warp > 0 ? warp_tot[warp - 1] : 0) + incl - cnt;
#pragma unroll
    for (int e = 0; e < kPer; ++e)
      if (kept[e]) {
        if (pos < b) out[pos] = j0 + e;
        ++pos;
      }
    carry += warp_tot[(blockDim.x >> 5) - 1];
  }
  if (threadIdx.x == 0 && carry != b) raise_status(status, 1u);
}

// grid = (units, rows_split), block = 256: copy kept rows (16 B per thread-step)
__global__ void __launch_bounds__(256) copy_rows_kernel(Prob p, const __nv_bfloat16* __restrict__ K,
                                                        const __nv_bfloat16* __restrict__ V,
                                                        const int32_t* __restrict__ counts,
                                                        const int64_t* __restrict__ offsets,
                                                        const int32_t* __restrict__ positions,
                                                        __nv_bfloat16* __restrict__ pk,
                                                        __nv_bfloat16* __restrict__ pv,
                                                        float* __restrict__ kept_vmax) {
  const int u = blockIdx.x;
  const int b = counts[u];
  const int64_t off = offsets[u];
  if (!CERTKV_IN_BOUNDS(b >= 0 && b < p.n && off >= 0 && (p.capacity <= 0 || off + b <= p.capacity),
                        p.status))
    return;
  const uint4* Ku = reinterpret_cast<const uint4*>(K + (size_t)u * p.n * kD);
  const uint4* Vu = reinterpret_cast<const uint4*>(V + (size_t)u * p.n * kD);
  uint4* PK = reinterpret_cast<uint4*>(pk);
  uint4* PV = reinterpret_cast<uint4*>(pv);
  // 16 uint4 per row; 256 threads = 16 rows per step, 4 steps' loads in flight
  const int sub = threadIdx.x & 15;
  const int stride = gridDim.y * 16;
  float vmax = 0.f;
  // the loop bound is the warp's first row, so both half-warps run the same
  // iterations (the row-norm shuffles need the whole warp)
  for (int wrow0 = blockIdx.y * 16 + (threadIdx.x >> 5) * 2; wrow0 < b; wrow0 += 4 * stride) {
    const int row0 = wrow0 + ((threadIdx.x >> 4) & 1);
    int j[4];
    uint4 kx[4], vx[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int row = row0 + e * stride;
      j[e] = row < b ? positions[off + row] : -1;
      if (row < b && !CERTKV_IN_BOUNDS(j[e] >= 0 && j[e] < p.n, p.status)) j[e] = -1;
    }
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const bool ok = j[e] >= 0 && j[e] < p.n;  // false only past b (the selection is consistent)
      kx[e] = ok ? __ldg(Ku + (size_t)j[e] * 16 + sub) : make_uint4(0u, 0u, 0u, 0u);
      vx[e] = ok ? __ldg(Vu + (size_t)j[e] * 16 + sub) : make_uint4(0u, 0u, 0u, 0u);
    }
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int row = row0 + e * stride;
      if (j[e] >= 0 && j[e] < p.n) {
        PK[(size_t)(off + row) * 16 + sub] = kx[e];
        PV[(size_t)(off + row) * 16 + sub] = vx[e];
      }
    }
    if (kept_vmax) {  // largest ||v|| of the kept rows (for the clustered-tail bound)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const uint32_t w[4] = {vx[e].x, vx[e].y, vx[e].z, vx[e].w};
        float sq = 0.f;
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          const float a = bf16lo(w[c]), b2 = bf16hi(w[c]);
          sq = fmaf(a, a, fmaf(b2, b2, sq));
        }
#pragma unroll
        for (int o = 8; o >= 1; o >>= 1) sq += __shfl_xor_sync(kFull, sq, o);  // the row's 16 threads
        vmax = fmaxf(vmax, sqrtf(sq));
      }
    }
  }
  if (kept_vmax) {
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) vmax = fmaxf(vmax, __shfl_xor_sync(kFull, vmax, o));
    // non-negative floats order like their bit patterns
    if ((threadIdx.x & 31) == 0)
      atomicMax(reinterpret_cast<unsigned int*>(kept_vmax) + u,
                __float_as_uint(vmax * kRadiusRoundUp));
  }
}

// Clustered-tail summaries (appendix: deterministic output-error bound for
// clustered tail summaries; readings R-C1, R-C2): group g of unit u = ranks
// b + floor(g T / m) .. b + floor((g + 1) T / m) - 1 of the evicted tail
// (T = n - b); stored representatives = the bf16-rounded unweighted means,
// radii = the largest distances of the group's rows to them, rounded up by
// 1e-5 relative (the fp32 sum of 128 squares and the square root are within
// a few 1e-6 of exact).  Each group is cut into kClusterParts contiguous
// parts, one CTA each (warp per row, four rows in flight):
//   cluster_sum     part sums of the keys and values (fp32 over 32 rows,
//                   folded into double-float);
//   cluster_mean    the parts added in a fixed order, the mean rounded and
//                   stored in the summary slot;
//   cluster_radius  part maxima of the distances to the stored means;
//   cluster_meta    the maxima over the parts, rounded up.
constexpr int kClusterParts = 8;
constexpr int kClusterWarps = 8;

namespace {
__device__ __forceinline__ void cluster_rows(const Prob& p, const int32_t* counts, int u, int g,
                                             int part, int& lo, int& hi) {
  const int n = p.n, b = counts[u], m = p.clusters;
  const int T = n - b;
  const int r0 = b + (int)(((int64_t)g * T) / m), r1 = b + (int)(((int64_t)(g + 1) * T) / m);
  const int cnt = r1 - r0;
  lo = r0 + (int)(((int64_t)part * cnt) / kClusterParts);
  hi = r0 + (int)(((int64_t)(part + 1) * cnt) / kClusterParts);
}
__device__ __forceinline__ void load_row4(const uint2* base, int j, int lane, float (&x)[4]) {
  const uint2 raw = __ldg(base + (size_t)j * (kD / 4) + lane);
  x[0] = bf16lo(raw.x);
  x[1] = bf16hi(raw.x);
  x[2] = bf16lo(raw.y);
  x[3] = bf16hi(raw.y);
}
}  // namespace

// grid = (units, m, kClusterParts), block = 32 * kClusterWarps.
// part_sum [u][g][part][2][kD] double-float (hi, lo).
__global__ void __launch_bounds__(kClusterWarps * 32) cluster_sum_kernel(
    Prob p, const int32_t* __restrict__ perm, const __nv_bfloat16* __restrict__ K,
    const __nv_bfloat16* __restrict__ V, const int32_t* __restrict__ counts,
    float2* __restrict__ part_sum) {
  __shared__ DF s_sum[kClusterWarps][2][kD];
  const int u = blockIdx.x, g = blockIdx.y, part = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n = p.n;
  const int32_t* pu = perm + (size_t)u * n;
  const uint2* Ku = reinterpret_cast<const uint2*>(K + (size_t)u * n * kD);
  const uint2* Vu = reinterpret_cast<const uint2*>(V + (size_t)u * n * kD);
  int lo, hi;
  cluster_rows(p, counts, u, g, part, lo, hi);
  DF sk[4], sv[4];
#pragma unroll
  for (int c = 0; c < 4; ++c) sk[c] = sv[c] = df_make(0.f);
  int in_block = 0;
  float fk[4] = {0.f, 0.f, 0.f, 0.f}, fv[4] = {0.f, 0.f, 0.f, 0.f};
  for (int rb = lo + warp; rb < hi; rb += 4 * kClusterWarps) {
    float k4[4][4], v4[4][4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int r = rb + e * kClusterWarps;
      if (r < hi) {
        int j = pu[r];
        if (!CERTKV_IN_BOUNDS(j >= 0 && j < n, p.status)) j = 0;
        load_row4(Ku, j, lane, k4[e]);
        load_row4(Vu, j, lane, v4[e]);
      }
    }
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      if (rb + e * kClusterWarps >= hi) break;
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        fk[c] += k4[e][c];
        fv[c] += v4[e][c];
      }
    }
    in_block += 4;
    if (in_block >= 32) {  // fp32 over 32 rows, then double-float
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        sk[c] = df_add_f(sk[c], fk[c]);
        sv[c] = df_add_f(sv[c], fv[c]);
        fk[c] = fv[c] = 0.f;
      }
      in_block = 0;
    }
  }
#pragma unroll
  for (int c = 0; c < 4; ++c) {
    s_sum[warp][0][lane * 4 + c] = df_add_f(sk[c], fk[c]);
    s_sum[warp][1][lane * 4 + c] = df_add_f(sv[c], fv[c]);
  }
  __syncthreads();
  const int t = threadIdx.x / kD, i = threadIdx.x % kD;  // 256 threads = 2 tensors x kD
  DF sum = df_make(0.f);
  for (int w = 0; w < kClusterWarps; ++w) sum = df_add(sum, s_sum[w][t][i]);
  part_sum[((((size_t)u * p.clusters + g) * kClusterParts + part) * 2 + t) * kD + i] =
      make_float2(sum.hi, sum.lo);
}

// grid = (units, m), block = 256.  means [u][g][2][kD] fp32 = the stored
// bf16 values.
__global__ void __launch_bounds__(256) cluster_mean_kernel(
    Prob p, const int32_t* __restrict__ counts, const int64_t* __restrict__ offsets,
    const float2* __restrict__ part_sum, float* __restrict__ means, __nv_bfloat16* __restrict__ pk,
    __nv_bfloat16* __restrict__ pv, int32_t* __restrict__ positions) {
  const int u = blockIdx.x, g = blockIdx.y, m = p.clusters;
  const int n = p.n, b = counts[u];
  const int T = n - b;
  const int cnt = (int)(((int64_t)(g + 1) * T) / m) - (int)(((int64_t)g * T) / m);
  const int t = threadIdx.x / kD, i = threadIdx.x % kD;
  DF sum = df_make(0.f);
  for (int part = 0; part < kClusterParts; ++part) {
    const float2 x = part_sum[((((size_t)u * m + g) * kClusterParts + part) * 2 + t) * kD + i];
    sum = df_add(sum, DF{x.x, x.y});
  }
  const DF mean = cnt > 0 ? df_div(sum, df_make((float)cnt)) : df_make(0.f);
  const uint16_t bits = df_to_bf16(mean.hi, mean.lo);
  const int64_t slot = offsets[u] + b + p.tail_slot + g;
  if (!CERTKV_IN_BOUNDS(p.capacity <= 0 || (slot >= 0 && slot < p.capacity), p.status)) return;
  reinterpret_cast<uint16_t*>(t == 0 ? pk : pv)[slot * kD + i] = bits;
  means[(((size_t)u * m + g) * 2 + t) * kD + i] = __uint_as_float((uint32_t)bits << 16);
  if (threadIdx.x == 0) positions[slot] = -2 - g;
}

// grid = (units, m, kClusterParts), block = 32 * kClusterWarps.
// part_max [u][g][part] = (largest key distance, largest value distance).
__global__ void __launch_bounds__(kClusterWarps * 32) cluster_radius_kernel(
    Prob p, const int32_t* __restrict__ perm, const __nv_bfloat16* __restrict__ K,
    const __nv_bfloat16* __restrict__ V, const int32_t* __restrict__ counts,
    const float* __restrict__ means, float2* __restrict__ part_max) {
  __shared__ float s_mean[2][kD];
  __shared__ float s_max[kClusterWarps][2];
  const int u = blockIdx.x, g = blockIdx.y, part = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n = p.n;
  const int32_t* pu = perm + (size_t)u * n;
  const uint2* Ku = reinterpret_cast<const uint2*>(K + (size_t)u * n * kD);
  const uint2* Vu = reinterpret_cast<const uint2*>(V + (size_t)u * n * kD);
  (&s_mean[0][0])[threadIdx.x] = means[((size_t)u * p.clusters + g) * 2 * kD + threadIdx.x];
  __syncthreads();
  int lo, hi;
  cluster_rows(p, counts, u, g, part, lo, hi);
  float mk = 0.f, mv = 0.f;
  for (int rb = lo + warp; rb < hi; rb += 4 * kClusterWarps) {
    float k4[4][4], v4[4][4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int r = rb + e * kClusterWarps;
      if (r < hi) {
        int j = pu[r];
        if (!CERTKV_IN_BOUNDS(j >= 0 && j < n, p.status)) j = 0;
        load_row4(Ku, j, lane, k4[e]);
        load_row4(Vu, j, lane, v4[e]);
      }
    }
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      if (rb + e * kClusterWarps >= hi) break;
      float qk = 0.f, qv = 0.f;
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const float dk = k4[e][c] - s_mean[0][lane * 4 + c];
        const float dv = v4[e][c] - s_mean[1][lane * 4 + c];
        qk = fmaf(dk, dk, qk);
        qv = fmaf(dv, dv, qv);
      }
#pragma unroll
      for (int o = 16; o >= 1; o >>= 1) {
        qk += __shfl_xor_sync(kFull, qk, o);
        qv += __shfl_xor_sync(kFull, qv, o);
      }
      mk = fmaxf(mk, sqrtf(qk));
      mv = fmaxf(mv, sqrtf(qv));
    }
  }
  if (lane == 0) {
    s_max[warp][0] = mk;
    s_max[warp][1] = mv;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float a = 0.f, c = 0.f;
    for (int w = 0; w < kClusterWarps; ++w) {
      a = fmaxf(a, s_max[w][0]);
      c = fmaxf(c, s_max[w][1]);
    }
    part_max[((size_t)u * p.clusters + g) * kClusterParts + part] = make_float2(a, c);
  }
}

// grid = units, block = 64 (thread = group g < m)
__global__ void cluster_meta_kernel(Prob p, const int32_t* __restrict__ counts,
                                    const float2* __restrict__ part_max,
                                    float4* __restrict__ cluster_meta) {
  const int u = blockIdx.x, g = threadIdx.x, m = p.clusters;
  if (g >= m) return;
  const int T = p.n - counts[u];
  const int cnt = (int)(((int64_t)(g + 1) * T) / m) - (int)(((int64_t)g * T) / m);
  float a = 0.f, c = 0.f;
  for (int part = 0; part < kClusterParts; ++part) {
    const float2 x = part_max[((size_t)u * m + g) * kClusterParts + part];
    a = fmaxf(a, x.x);
    c = fmaxf(c, x.y);
  }
  cluster_meta[(size_t)u * m + g] =
      make_float4((float)cnt, a * kRadiusRoundUp, c * kRadiusRoundUp, 0.f);
}

void launch_pack(const Prob& p, const Layout& ly, char* ws, const void* K, const void* V,
                 const float* a, void* pk, void* pv, const int64_t* offsets,
                 const int32_t* counts, int32_t* positions, float* tail_f32,
                 double* tail_mass, float* cluster_meta, float* kept_vmax, cudaStream_t st) {
  const uint32_t* keys = reinterpret_cast<const uint32_t*>(ws + ly.keys0);
  const int32_t* perm = reinterpret_cast<const int32_t*>(ws + ly.vals0);
  const __nv_bfloat16* Kb = reinterpret_cast<const __nv_bfloat16*>(K);
  const __nv_bfloat16* Vb = reinterpret_cast<const __nv_bfloat16*>(V);
  __nv_bfloat16* PK = reinterpret_cast<__nv_bfloat16*>(pk);
  __nv_bfloat16* PV = reinterpret_cast<__nv_bfloat16*>(pv);
  uint32_t* status = reinterpret_cast<uint32_t*>(ws + ly.status);
  {
    TraceScope ts("select", st);
    select_kernel<<<p.units, 1024, 0, st>>>(p, a, keys, perm, counts, offsets, positions, status);
  }

  int ysplit = (p.n + 15) / 16;
  if (ysplit > 64) ysplit = 64;
  {
    TraceScope ts("copy_rows", st);
    if (p.clusters > 0) cudaMemsetAsync(kept_vmax, 0, (size_t)p.units * sizeof(float), st);
    copy_rows_kernel<<<dim3(p.units, ysplit), 256, 0, st>>>(
        p, Kb, Vb, counts, offsets, positions, PK, PV, p.clusters > 0 ? kept_vmax : nullptr);
  }
  if (p.clusters > 0) {
    float2* part_sum = reinterpret_cast<float2*>(ws + ly.cl_sum);
    float* means = reinterpret_cast<float*>(ws + ly.cl_mean);
    float2* part_max = reinterpret_cast<float2*>(ws + ly.cl_max);
    const dim3 gp(p.units, p.clusters, kClusterParts);
    {
      TraceScope ts("cluster_sum", st);
      cluster_sum_kernel<<<gp, kClusterWarps * 32, 0, st>>>(p, perm, Kb, Vb, counts, part_sum);
    }
    {
      TraceScope ts("cluster_mean", st);
      cluster_mean_kernel<<<dim3(p.units, p.clusters), 256, 0, st>>>(p, counts, offsets, part_sum,
                                                                     means, PK, PV, positions);
    }
    {
      TraceScope ts("cluster_radius", st);
      cluster_radius_kernel<<<gp, kClusterWarps * 32, 0, st>>>(p, perm, Kb, Vb, counts, means,
                                                               part_max);
    }
    {
      TraceScope ts("cluster_meta", st);
      cluster_meta_kernel<<<p.units, 64, 0, st>>>(p, counts, part_max,
                                                  reinterpret_cast<float4*>(cluster_meta));
    }
  }
  if (p.tail_slot) {
    TraceScope ts("tail", st);
    tail_kernel<<<p.units, 128, 0, st>>>(
        p, keys, perm, Kb, Vb, reinterpret_cast<const float4*>(ws + ly.base_mq),
        reinterpret_cast<const float2*>(ws + ly.base_v),
        reinterpret_cast<const float*>(ws + ly.agg_k), counts, offsets, PK, PV, positions,
        tail_f32, tail_mass, status);
  }
}

}  // namespace certkv
