// decode.cu — a9: decode attention over the packed cache.
//
// For each query head qh of unit u = (b, l, qh / G):
//   out = sum_s softmax_s(scale <q, k_s>) v_s
// over the real_counts[u] real slots plus the tail slot (the "plain slot" of
// the paper's ablation table: the synthetic pair enters as an ordinary KV
// entry).  Split-K: kDecodeSplits CTAs per unit each stream an interleaved
// share of 32-slot tiles and keep online (max, sum, acc) for the G query
// heads that share the unit, so every packed K/V byte is read once per step;
// a merge kernel combines the splits in the log-sum-exp domain.
#include "../../include/certkv.h"
#include "common.cuh"
#include "internal.cuh"

namespace certkv {

struct DecodePart {  // one (unit, split, query head)
  float m, l;
};

// grid = (units, kDecodeSplits), block = 128 (4 warps)
template <int G>
__global__ void __launch_bounds__(128) decode_split_kernel(Prob p, const __nv_bfloat16* __restrict__ q,
                                                           const __nv_bfloat16* __restrict__ pk,
                                                           const __nv_bfloat16* __restrict__ pv,
                                                           const int64_t* __restrict__ offsets,
                                                           const int32_t* __restrict__ counts,
                                                           int tail_slot, float scale_log2,
                                                           float2* __restrict__ part_ml,
                                                           float* __restrict__ part_acc) {
  __shared__ __align__(16) float qs[G][kD];
  __shared__ float wm[4][G], wl[4][G];
  __shared__ float wacc[4][G][kD];
  const int u = blockIdx.x, split = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int bl = u / p.H, h = u - bl * p.H;
  const __nv_bfloat16* qu = q + ((size_t)bl * p.Hq + (size_t)h * G) * kD;
  for (int i = threadIdx.x; i < G * kD; i += blockDim.x)
    (&qs[0][0])[i] = __bfloat162float(qu[i]) * scale_log2;
  __syncthreads();

  const int slots = counts[u] + tail_slot;
  const int64_t off = offsets[u];
  float m[G], l[G], acc[G][4];
#pragma unroll
  for (int g = 0; g < G; ++g) {
    m[g] = -INFINITY;
    l[g] = 0.f;
    acc[g][0] = acc[g][1] = acc[g][2] = acc[g][3] = 0.f;
  }
  const int ntiles = (slots + 31) / 32;
  for (int t = split * 4 + warp; t < ntiles; t += kDecodeSplits * 4) {
    const int s = t * 32 + lane;
    const bool ok = s < slots;
    // scores: lane = slot
    float x[G];
#pragma unroll
    for (int g = 0; g < G; ++g) x[g] = 0.f;
    if (ok) {
      const uint4* kr = reinterpret_cast<const uint4*>(pk + (size_t)(off + s) * kD);
      uint4 krow[16];  // the whole 256-byte row in flight before the dot products
#pragma unroll
      for (int c = 0; c < 16; ++c) krow[c] = __ldg(kr + c);
#pragma unroll
      for (int c = 0; c < 16; ++c) {
        const uint4 raw = krow[c];
        const float kf[8] = {bf16lo(raw.x), bf16hi(raw.x), bf16lo(raw.y), bf16hi(raw.y),
                             bf16lo(raw.z), bf16hi(raw.z), bf16lo(raw.w), bf16hi(raw.w)};
#pragma unroll
        for (int g = 0; g < G; ++g) {
          const float4 q0 = *reinterpret_cast<const float4*>(&qs[g][c * 8]);
          const float4 q1 = *reinterpret_cast<const float4*>(&qs[g][c * 8 + 4]);
          x[g] = fmaf(q0.x, kf[0], x[g]);
          x[g] = fmaf(q0.y, kf[1], x[g]);
          x[g] = fmaf(q0.z, kf[2], x[g]);
          x[g] = fmaf(q0.w, kf[3], x[g]);
          x[g] = fmaf(q1.x, kf[4], x[g]);
          x[g] = fmaf(q1.y, kf[5], x[g]);
          x[g] = fmaf(q1.z, kf[6], x[g]);
          x[g] = fmaf(q1.w, kf[7], x[g]);
        }
      }
    } else {
#pragma unroll
      for (int g = 0; g < G; ++g) x[g] = -INFINITY;
    }
    float pr[G];
#pragma unroll
    for (int g = 0; g < G; ++g) {
      const float tm = warp_max(x[g]);
      const float nm = fmaxf(m[g], tm);
      const float corr = exp2f(m[g] - nm);
      m[g] = nm;
      l[g] *= corr;
#pragma unroll
      for (int i = 0; i < 4; ++i) acc[g][i] *= corr;
      pr[g] = ok ? exp2f(x[g] - nm) : 0.f;
      l[g] += pr[g];
    }
    // values: lane = 4 dims
    const int cnt = min(32, slots - t * 32);
    const uint2* vrow = reinterpret_cast<const uint2*>(pv + (size_t)(off + t * 32) * kD) + lane;
    for (int j0 = 0; j0 < cnt; j0 += 8) {  // 8 rows' loads in flight, then their FMAs
      uint2 raw[8];
#pragma unroll
      for (int e = 0; e < 8; ++e)
        raw[e] = (j0 + e < cnt) ? __ldg(vrow + (size_t)(j0 + e) * (kD / 4)) : make_uint2(0u, 0u);
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        const float v0 = bf16lo(raw[e].x), v1 = bf16hi(raw[e].x), v2 = bf16lo(raw[e].y),
                    v3 = bf16hi(raw[e].y);
#pragma unroll
        for (int g = 0; g < G; ++g) {
          const float pj = __shfl_sync(kFull, pr[g], j0 + e);  // 0 past the last slot
          acc[g][0] = fmaf(pj, v0, acc[g][0]);
          acc[g][1] = fmaf(pj, v1, acc[g][1]);
          acc[g][2] = fmaf(pj, v2, acc[g][2]);
          acc[g][3] = fmaf(pj, v3, acc[g][3]);
        }
      }
    }
  }
  // combine the 4 warps
#pragma unroll
  for (int g = 0; g < G; ++g) {
    float lt = l[g];
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) lt += __shfl_xor_sync(kFull, lt, o);
    if (lane == 0) {
      wm[warp][g] = m[g];
      wl[warp][g] = lt;
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) wacc[warp][g][lane * 4 + i] = acc[g][i];
  }
  __syncthreads();
  for (int idx = threadIdx.x; idx < G * kD; idx += blockDim.x) {
    const int g = idx / kD, i = idx - g * kD;
    float M = -INFINITY;
#pragma unroll
    for (int wi = 0; wi < 4; ++wi) M = fmaxf(M, wm[wi][g]);
    float L = 0.f, A = 0.f;
#pragma unroll
    for (int wi = 0; wi < 4; ++wi) {
      if (wm[wi][g] > -INFINITY) {
        const float f = exp2f(wm[wi][g] - M);
        L += wl[wi][g] * f;
        A += wacc[wi][g][i] * f;
      }
    }
    const size_t pi = ((size_t)u * kDecodeSplits + split) * G + g;
    part_acc[pi * kD + i] = A;
    if (i == 0) part_ml[pi] = make_float2(M, L);
  }
}

// grid = units * G, block = 128: merge the splits of one query head.
__global__ void __launch_bounds__(128) decode_merge_kernel(Prob p, int G,
                                                           const float2* __restrict__ part_ml,
                                                           const float* __restrict__ part_acc,
                                                           __nv_bfloat16* __restrict__ out) {
  const int ug = blockIdx.x;
  const int u = ug / G, g = ug - u * G;
  const int i = threadIdx.x;
  float M = -INFINITY;
  for (int s = 0; s < kDecodeSplits; ++s)
    M = fmaxf(M, part_ml[((size_t)u * kDecodeSplits + s) * G + g].x);
  float L = 0.f, A = 0.f;
  for (int s = 0; s < kDecodeSplits; ++s) {
    const size_t pi = ((size_t)u * kDecodeSplits + s) * G + g;
    const float2 ml = part_ml[pi];
    if (ml.x > -INFINITY) {
      const float f = exp2f(ml.x - M);
      L += ml.y * f;
      A += part_acc[pi * kD + i] * f;
    }
  }
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

// grid = units * G, block = 128 (thread = dimension): the real-slot splits of
// one query head merged as in decode_merge_kernel, then the m cluster
// summaries added with weight n_g e^{lbar_g} (all weights relative to one
// log2-domain shift, to which the bound is invariant), then the certificate.
__global__ void __launch_bounds__(128) decode_certified_merge_kernel(
    Prob p, int G, int m, int tail_slot, float scale, const __nv_bfloat16* __restrict__ q,
    const __nv_bfloat16* __restrict__ pk, const __nv_bfloat16* __restrict__ pv,
    const int64_t* __restrict__ offsets, const int32_t* __restrict__ counts,
    const float4* __restrict__ cluster_meta, const float* __restrict__ kept_vmax,
    const float2* __restrict__ part_ml, const float* __restrict__ part_acc,
    __nv_bfloat16* __restrict__ out, float* __restrict__ bound, int32_t* __restrict__ certified) {
  __shared__ float red[4];
  __shared__ float s_lam[CERTKV_MAX_CLUSTERS], s_r[CERTKV_MAX_CLUSTERS];
  __shared__ float s_vn[CERTKV_MAX_CLUSTERS], s_rho[CERTKV_MAX_CLUSTERS];
  const int ug = blockIdx.x;
  const int u = ug / G, g = ug - u * G;
  const int i = threadIdx.x;
  const float kLog2e = 1.4426950408889634f;
  // real slots: merge of the splits (log2 domain)
  float MS = -INFINITY;
  for (int s = 0; s < kDecodeSplits; ++s)
    MS = fmaxf(MS, part_ml[((size_t)u * kDecodeSplits + s) * G + g].x);
  float LS = 0.f, AS = 0.f;
  for (int s = 0; s < kDecodeSplits; ++s) {
    const size_t pi = ((size_t)u * kDecodeSplits + s) * G + g;
    const float2 ml = part_ml[pi];
    if (ml.x > -INFINITY) {
      const float f = exp2f(ml.x - MS);
      LS += ml.y * f;
      AS += part_acc[pi * kD + i] * f;
    }
  }
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

size_t decode_workspace(const Prob& p) {
  const size_t parts = (size_t)p.units * kDecodeSplits * p.G;
  return parts * sizeof(float2) + parts * kD * sizeof(float) + 512;
}

template <int G>
static void launch_split(const Prob& p, const __nv_bfloat16* q, const __nv_bfloat16* pk,
                         const __nv_bfloat16* pv, const int64_t* offsets, const int32_t* counts,
                         int tail_slot, float sl2, float2* ml, float* acc, cudaStream_t st) {
  {
    TraceScope ts_("decode_split", st);
    decode_split_kernel<G><<<dim3(p.units, kDecodeSplits), 128, 0, st>>>(p, q, pk, pv, offsets,
                                                                         counts, tail_slot, sl2, ml,
                                                                         acc);
  }
}

void launch_decode(const Prob& p, const void* q, const void* pk, const void* pv,
                   const int64_t* offsets, const int32_t* counts, int tail_slot, float scale,
                   void* out, char* ws, cudaStream_t st) {
  const size_t parts = (size_t)p.units * kDecodeSplits * p.G;
  float2* ml = reinterpret_cast<float2*>(ws);
  size_t acc_off = (parts * sizeof(float2) + 255) / 256 * 256;
  float* acc = reinterpret_cast<float*>(ws + acc_off);
  const float sl2 = scale * 1.4426950408889634f;
  const __nv_bfloat16* qb = reinterpret_cast<const __nv_bfloat16*>(q);
  const __nv_bfloat16* kb = reinterpret_cast<const __nv_bfloat16*>(pk);
  const __nv_bfloat16* vb = reinterpret_cast<const __nv_bfloat16*>(pv);
  switch (p.G) {
    case 1: launch_split<1>(p, qb, kb, vb, offsets, counts, tail_slot, sl2, ml, acc, st); break;
    case 2: launch_split<2>(p, qb, kb, vb, offsets, counts, tail_slot, sl2, ml, acc, st); break;
    case 4: launch_split<4>(p, qb, kb, vb, offsets, counts, tail_slot, sl2, ml, acc, st); break;
    case 8: launch_split<8>(p, qb, kb, vb, offsets, counts, tail_slot, sl2, ml, acc, st); break;
    case 16: launch_split<16>(p, qb, kb, vb, offsets, counts, tail_slot, sl2, ml, acc, st); break;
    default: return;
  }
  {
    TraceScope ts_("decode_merge", st);
    decode_merge_kernel<<<p.units * p.G, 128, 0, st>>>(p, p.G, ml, acc,
                                                       reinterpret_cast<__nv_bfloat16*>(out));
  }
}

void launch_decode_certified(const Prob& p, const void* q, const void* pk, const void* pv,
                             const int64_t* offsets, const int32_t* counts, int tail_slot,
                             int clusters, const float* cluster_meta, const float* kept_vmax,
                             float scale, void* out, float* bound, int32_t* certified, char* ws,
                             cudaStream_t st) {
  const size_t parts = (size_t)p.units * kDecodeSplits * p.G;
  float2* ml = reinterpret_cast<float2*>(ws);
  size_t acc_off = (parts * sizeof(float2) + 255) / 256 * 256;
  float* acc = reinterpret_cast<float*>(ws + acc_off);
  const float sl2 = scale * 1.4426950408889634f;
  const __nv_bfloat16* qb = reinterpret_cast<const __nv_bfloat16*>(q);
  const __nv_bfloat16* kb = reinterpret_cast<const __nv_bfloat16*>(pk);
  const __nv_bfloat16* vb = reinterpret_cast<const __nv_bfloat16*>(pv);
  // the real slots only: the splits see no tail slot
  switch (p.G) {
    case 1: launch_split<1>(p, qb, kb, vb, offsets, counts, 0, sl2, ml, acc, st); break;
    case 2: launch_split<2>(p, qb, kb, vb, offsets, counts, 0, sl2, ml, acc, st); break;
    case 4: launch_split<4>(p, qb, kb, vb, offsets, counts, 0, sl2, ml, acc, st); break;
    case 8: launch_split<8>(p, qb, kb, vb, offsets, counts, 0, sl2, ml, acc, st); break;
    case 16: launch_split<16>(p, qb, kb, vb, offsets, counts, 0, sl2, ml, acc, st); break;
    default: return;
  }
  {
    TraceScope ts_("decode_certified_merge", st);
    decode_certified_merge_kernel<<<p.units * p.G, 128, 0, st>>>(
        p, p.G, clusters, tail_slot, scale, qb, kb, vb, offsets, counts,
        reinterpret_cast<const float4*>(cluster_meta), kept_vmax, ml, acc,
        reinterpret_cast<__nv_bfloat16*>(out), bound, certified);
  }
}

}  // namespace certkv
