// diagnose.cu — fixed-row diagnostics over the full cache (an evaluation
// tool: it reads every original K and V row).
//
// For each query head and its realized softmax row A over all n original
// tokens of the unit (Theorem: fixed-row tail factorization), with S = the
// kept real tokens of a packed cache: the kept mass p_S, exact attention O,
// the subset-only output O~_S = sum_S A v / p_S, the fixed-row correction
// u* = sum_{not S} A v, the mass bound 2 V_max (1 - p_S), and the error of
// the compressed decode.  One split-K pass keeps two online softmax states
// (all tokens, kept tokens) under one shared running maximum.
#include "../../include/certkv.h"
#include "common.cuh"
#include "internal.cuh"

namespace certkv {

constexpr int kDiagSplits = 32;

// mask[u][w]: bit j % 32 of word j / 32 set when token j of unit u is kept
__global__ void kept_mask_kernel(Prob p, const int64_t* __restrict__ offsets,
                                 const int32_t* __restrict__ counts,
                                 const int32_t* __restrict__ positions, uint32_t* __restrict__ mask) {
  const int u = blockIdx.x;
  const int words = (p.n + 31) / 32;
  for (int s = threadIdx.x; s < counts[u]; s += blockDim.x) {
    const int j = positions[offsets[u] + s];
    if (j >= 0 && j < p.n) atomicOr(&mask[(size_t)u * words + j / 32], 1u << (j % 32));
  }
}

struct DiagPart {  // one (unit, split, query head)
  float m, l_all, l_kept, vmax;
};

// grid = (units, kDiagSplits), block = 128 (4 warps); 32-token tiles, lane =
// token for the logits, lane = 4 dimensions for the value sums.
template <int G>
__global__ void __launch_bounds__(128) fixed_row_split_kernel(
    Prob p, const __nv_bfloat16* __restrict__ q, const __nv_bfloat16* __restrict__ K,
    const __nv_bfloat16* __restrict__ V, const uint32_t* __restrict__ mask, float scale_log2,
    DiagPart* __restrict__ part, float* __restrict__ part_acc) {
  __shared__ __align__(16) float qs[G][kD];
  __shared__ DiagPart wp[4][G];
  __shared__ float wacc[4][2][kD];  // one query head at a time
  const int u = blockIdx.x, split = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int bl = u / p.H, h = u - bl * p.H;
  const int n = p.n, words = (n + 31) / 32;
  const __nv_bfloat16* qu = q + ((size_t)bl * p.Hq + (size_t)h * G) * kD;
  for (int i = threadIdx.x; i < G * kD; i += blockDim.x)
    (&qs[0][0])[i] = __bfloat162float(qu[i]) * scale_log2;
  __syncthreads();
  const uint4* Ku = reinterpret_cast<const uint4*>(K + (size_t)u * n * kD);
  const uint2* Vu = reinterpret_cast<const uint2*>(V + (size_t)u * n * kD);
  float m[G], la[G], lk[G], aa[G][4], ak[G][4];
#pragma unroll
  for (int g = 0; g < G; ++g) {
    m[g] = -INFINITY;
    la[g] = lk[g] = 0.f;
#pragma unroll
    for (int i = 0; i < 4; ++i) aa[g][i] = ak[g][i] = 0.f;
  }
  float vmax = 0.f;
  const int ntiles = (n + 31) / 32;
  for (int t = split * 4 + warp; t < ntiles; t += kDiagSplits * 4) {
    const int j = t * 32 + lane;
    const bool ok = j < n;
    const bool kept = ok && ((mask[(size_t)u * words + (j >> 5)] >> (j & 31)) & 1u);
    float x[G];
#pragma unroll
    for (int g = 0; g < G; ++g) x[g] = -INFINITY;
    if (ok) {
      uint4 krow[16];
#pragma unroll
      for (int c = 0; c < 16; ++c) krow[c] = __ldg(Ku + (size_t)j * 16 + c);
#pragma unroll
      for (int g = 0; g < G; ++g) x[g] = 0.f;
#pragma unroll
      for (int c = 0; c < 16; ++c) {
        const uint4 raw = krow[c];
        const float kf[8] = {bf16lo(raw.x), bf16hi(raw.x), bf16lo(raw.y), bf16hi(raw.y),
                             bf16lo(raw.z), bf16hi(raw.z), bf16lo(raw.w), bf16hi(raw.w)};
#pragma unroll
        for (int g = 0; g < G; ++g)
#pragma unroll
          for (int e = 0; e < 8; ++e) x[g] = fmaf(qs[g][c * 8 + e], kf[e], x[g]);
      }
    }
    float pa[G], pk[G];
#pragma unroll
    for (int g = 0; g < G; ++g) {
      const float nm = fmaxf(m[g], warp_max(x[g]));
      const float corr = exp2f(m[g] - nm);
      m[g] = nm;
      la[g] *= corr;
      lk[g] *= corr;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        aa[g][i] *= corr;
        ak[g][i] *= corr;
      }
      pa[g] = ok ? exp2f(x[g] - nm) : 0.f;
      pk[g] = kept ? pa[g] : 0.f;
      la[g] += pa[g];
      lk[g] += pk[g];
    }
    const int cnt = min(32, n - t * 32);
    for (int r = 0; r < cnt; ++r) {
      const uint2 raw = __ldg(Vu + (size_t)(t * 32 + r) * (kD / 4) + lane);
      const float v[4] = {bf16lo(raw.x), bf16hi(raw.x), bf16lo(raw.y), bf16hi(raw.y)};
      float sq = fmaf(v[3], v[3], fmaf(v[2], v[2], fmaf(v[1], v[1], v[0] * v[0])));
#pragma unroll
      for (int o = 16; o >= 1; o >>= 1) sq += __shfl_xor_sync(kFull, sq, o);
      vmax = fmaxf(vmax, sqrtf(sq));
#pragma unroll
      for (int g = 0; g < G; ++g) {
        const float wa = __shfl_sync(kFull, pa[g], r), wk = __shfl_sync(kFull, pk[g], r);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          aa[g][i] = fmaf(wa, v[i], aa[g][i]);
          ak[g][i] = fmaf(wk, v[i], ak[g][i]);
        }
      }
    }
  }
  // combine the 4 warps, one query head at a time
#pragma unroll
  for (int g = 0; g < G; ++g) {
    float ta = la[g], tk = lk[g];
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) {
      ta += __shfl_xor_sync(kFull, ta, o);
      tk += __shfl_xor_sync(kFull, tk, o);
    }
    if (lane == 0) wp[warp][g] = DiagPart{m[g], ta, tk, vmax};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      wacc[warp][0][lane * 4 + i] = aa[g][i];
      wacc[warp][1][lane * 4 + i] = ak[g][i];
    }
    __syncthreads();
    const int i = threadIdx.x;  // 128 threads = kD dimensions
    float M = -INFINITY, vm = 0.f;
#pragma unroll
    for (int wi = 0; wi < 4; ++wi) {
      M = fmaxf(M, wp[wi][g].m);
      vm = fmaxf(vm, wp[wi][g].vmax);
    }
    float LA = 0.f, LK = 0.f, A = 0.f, B = 0.f;
#pragma unroll
    for (int wi = 0; wi < 4; ++wi) {
      if (wp[wi][g].m > -INFINITY) {
        const float f = exp2f(wp[wi][g].m - M);
        LA += wp[wi][g].l_all * f;
        LK += wp[wi][g].l_kept * f;
        A += wacc[wi][0][i] * f;
        B += wacc[wi][1][i] * f;
      }
    }
    const size_t pi = ((size_t)u * kDiagSplits + split) * G + g;
    part_acc[(pi * 2 + 0) * kD + i] = A;
    part_acc[(pi * 2 + 1) * kD + i] = B;
    if (i == 0) part[pi] = DiagPart{M, LA, LK, vm};
    __syncthreads();
  }
}

__device__ __forceinline__ float block_sum_128(float x, float* red) {
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) x += __shfl_xor_sync(kFull, x, o);
  __syncthreads();
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = x;
  __syncthreads();
  return (red[0] + red[1]) + (red[2] + red[3]);
}

// grid = units * G, block = 128 (thread = dimension): merge the splits of one
// query head and write its 8 statistics.
__global__ void __launch_bounds__(128) fixed_row_merge_kernel(
    Prob p, int G, const DiagPart* __restrict__ part, const float* __restrict__ part_acc,
    const __nv_bfloat16* __restrict__ ohat, float* __restrict__ stats) {
  __shared__ float red[4];
  const int ug = blockIdx.x;
  const int u = ug / G, g = ug - u * G;
  const int i = threadIdx.x;
  float M = -INFINITY, vm = 0.f;
  for (int s = 0; s < kDiagSplits; ++s) {
    const DiagPart q = part[((size_t)u * kDiagSplits + s) * G + g];
    M = fmaxf(M, q.m);
    vm = fmaxf(vm, q.vmax);
  }
  float LA = 0.f, LK = 0.f, A = 0.f, B = 0.f;
  for (int s = 0; s < kDiagSplits; ++s) {
    const size_t pi = ((size_t)u * kDiagSplits + s) * G + g;
    const DiagPart q = part[pi];
    if (q.m > -INFINITY) {
      const float f = exp2f(q.m - M);
      LA += q.l_all * f;
      LK += q.l_kept * f;
      A += part_acc[(pi * 2 + 0) * kD + i] * f;
      B += part_acc[(pi * 2 + 1) * kD + i] * f;
    }
  }
  const float o = A / LA;                       // exact attention
  const float os = LK > 0.f ? B / LK : 0.f;     // subset-only output
  const float uu = (A - B) / LA;                // fixed-row correction
  const float pS = LK / LA;
  const int bl = u / p.H, h = u - bl * p.H;
  const size_t qi = (size_t)bl * p.Hq + (size_t)h * G + g;
  const float oh = __bfloat162float(ohat[qi * kD + i]);
  const float vbt = pS < 1.f ? uu / (1.f - pS) : 0.f;
  const float f = os + (1.f - pS) * (vbt - os) - o;
  const float nO = block_sum_128(o * o, red);
  const float eS = block_sum_128((os - o) * (os - o), red);
  const float nu = block_sum_128(uu * uu, red);
  const float eh = block_sum_128((oh - o) * (oh - o), red);
  const float res = block_sum_128(f * f, red);
  if (i == 0) {
    float* st = stats + qi * 8;
    st[0] = pS;
    st[1] = sqrtf(nO);
    st[2] = sqrtf(eS);
    st[3] = sqrtf(nu);
    st[4] = 2.f * vm * (1.f - pS);
    st[5] = sqrtf(eh);
    st[6] = vm;
    st[7] = sqrtf(res);
  }
}

size_t fixed_row_workspace(const Prob& p) {
  const size_t words = (size_t)(p.n + 31) / 32;
  const size_t parts = (size_t)p.units * kDiagSplits * p.G;
  auto a = [](size_t x) { return (x + 255) / 256 * 256; };
  return a(p.units * words * 4) + a(parts * sizeof(DiagPart)) + a(parts * 2 * kD * 4) +
         a((size_t)p.units * p.G * kD * 2) + a(decode_workspace(p));
}

void launch_fixed_row(const Prob& p, const void* q, const void* K, const void* V,
                      const int64_t* offsets, const int32_t* counts, const int32_t* positions,
                      const void* pk, const void* pv, int tail_slot, float scale, float* stats,
                      char* ws, cudaStream_t st) {
  const size_t words = (size_t)(p.n + 31) / 32;
  const size_t parts = (size_t)p.units * kDiagSplits * p.G;
  auto a = [](size_t x) { return (x + 255) / 256 * 256; };
  uint32_t* mask = reinterpret_cast<uint32_t*>(ws);
  DiagPart* part = reinterpret_cast<DiagPart*>(ws + a(p.units * words * 4));
  float* acc = reinterpret_cast<float*>(ws + a(p.units * words * 4) + a(parts * sizeof(DiagPart)));
  char* ohat = ws + a(p.units * words * 4) + a(parts * sizeof(DiagPart)) + a(parts * 2 * kD * 4);
  char* dws = ohat + a((size_t)p.units * p.G * kD * 2);
  // the compressed decode's output, for its error against O
  launch_decode(p, q, pk, pv, offsets, counts, tail_slot, scale, ohat, dws, st);
  cudaMemsetAsync(mask, 0, p.units * words * 4, st);
  {
    TraceScope ts_("kept_mask", st);
    kept_mask_kernel<<<p.units, 256, 0, st>>>(p, offsets, counts, positions, mask);
  }
  const float sl2 = scale * 1.4426950408889634f;
  const __nv_bfloat16* qb = reinterpret_cast<const __nv_bfloat16*>(q);
  const __nv_bfloat16* kb = reinterpret_cast<const __nv_bfloat16*>(K);
  const __nv_bfloat16* vb = reinterpret_cast<const __nv_bfloat16*>(V);
  const dim3 grid(p.units, kDiagSplits);
  {
    TraceScope ts_("fixed_row_split", st);
    switch (p.G) {
      case 1: fixed_row_split_kernel<1><<<grid, 128, 0, st>>>(p, qb, kb, vb, mask, sl2, part, acc); break;
      case 2: fixed_row_split_kernel<2><<<grid, 128, 0, st>>>(p, qb, kb, vb, mask, sl2, part, acc); break;
      case 4: fixed_row_split_kernel<4><<<grid, 128, 0, st>>>(p, qb, kb, vb, mask, sl2, part, acc); break;
      case 8: fixed_row_split_kernel<8><<<grid, 128, 0, st>>>(p, qb, kb, vb, mask, sl2, part, acc); break;
      case 16: fixed_row_split_kernel<16><<<grid, 128, 0, st>>>(p, qb, kb, vb, mask, sl2, part, acc); break;
      default: return;
    }
  }
  {
    TraceScope ts_("fixed_row_merge", st);
    fixed_row_merge_kernel<<<p.units * p.G, 128, 0, st>>>(
        p, p.G, part, acc, reinterpret_cast<const __nv_bfloat16*>(ohat), stats);
  }
}

}  // namespace certkv
