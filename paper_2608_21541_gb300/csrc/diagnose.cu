// diagnose.cu — fixed-row diagnostics over the full cache (an evaluation
// tool: it reads every original K and V row).
//
// For each query head and its realized softmax row A over all n original
// tokens of the unit (Theorem: fixed-row tail factorization), with S = the
// kept real tokens of a packed cache and T the evicted ones: the kept mass
// p_S, exact attention O, the subset-only output O~_S = sum_S A v / p_S, the
// fixed-row correction u* = sum_T A v, the mass bound 2 V_max (1 - p_S), and
// the error of the compressed decode; and the quantities of the future-query
// lift (Theorem: future-query lift and summary mismatch): the tail mass p, the
// synthetic slot's compressed weight q, ||a - r||_1 between the exact tail
// distribution and the slot's tail weights, Lambda_T - z*, both of the
// theorem's bounds and the exact lifted L1 mismatch.  One split-K pass keeps
// two online softmax states (kept tokens, evicted tokens) under one shared
// running maximum and stores every logit; the merge reads the logits back for
// the per-token L1 sums.
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
  float m, l_kept, l_tail, vmax;
};

constexpr int kSvStride = kD + 1;  // per (unit, split): sum_T s_j v_j [kD], sum_T s_j

// grid = (units, kDiagSplits), block = 128 (4 warps); 32-token tiles, lane =
// token for the logits, lane = 4 dimensions for the value sums.  With scores
// `sc` (may be null) it also sums s_j v_j and s_j over the evicted tokens, and
// with part_tm (may be null) the evicted values' moments sum_T v_j and
// sum_T ||v_j||^2.  z2[u][g][j] receives every log2-domain logit.
template <int G>
__global__ void __launch_bounds__(128) fixed_row_split_kernel(
    Prob p, const __nv_bfloat16* __restrict__ q, const __nv_bfloat16* __restrict__ K,
    const __nv_bfloat16* __restrict__ V, const uint32_t* __restrict__ mask,
    const float* __restrict__ sc, float scale_log2, DiagPart* __restrict__ part,
    float* __restrict__ part_acc, float* __restrict__ z2, float* __restrict__ part_sv,
    float* __restrict__ part_tm) {
  __shared__ __align__(16) float qs[G][kD];
  __shared__ DiagPart wp[4][G];
  __shared__ float wacc[4][2][kD];  // one query head at a time
  __shared__ float wsv[4][kD];
  __shared__ float wss[4];
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
  float m[G], lk[G], lt[G], ak[G][4], at[G][4];
#pragma unroll
  for (int g = 0; g < G; ++g) {
    m[g] = -INFINITY;
    lk[g] = lt[g] = 0.f;
#pragma unroll
    for (int i = 0; i < 4; ++i) ak[g][i] = at[g][i] = 0.f;
  }
  float vmax = 0.f, ssum = 0.f, sv[4] = {0.f, 0.f, 0.f, 0.f};
  float tv[4] = {0.f, 0.f, 0.f, 0.f}, tq = 0.f;  // evicted values: sum v, sum ||v||^2 (lane part)
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
    if (ok) {
#pragma unroll
      for (int g = 0; g < G; ++g) z2[((size_t)u * G + g) * n + j] = x[g];
    }
    const float sj = (sc != nullptr && ok && !kept) ? sc[(size_t)u * n + j] : 0.f;
    ssum += sj;
    float pk[G], pt[G];
#pragma unroll
    for (int g = 0; g < G; ++g) {
      const float nm = fmaxf(m[g], warp_max(x[g]));
      const float corr = exp2f(m[g] - nm);
      m[g] = nm;
      lk[g] *= corr;
      lt[g] *= corr;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        ak[g][i] *= corr;
        at[g][i] *= corr;
      }
      const float pe = ok ? exp2f(x[g] - nm) : 0.f;
      pk[g] = kept ? pe : 0.f;
      pt[g] = kept ? 0.f : pe;
      lk[g] += pk[g];
      lt[g] += pt[g];
    }
    // value rows of the tile, 8 loads in flight per lane; rows past the end
    // of the unit read as zero and carry zero weight
    const int cnt = min(32, n - t * 32);
    const unsigned tailbits = __ballot_sync(kFull, ok && !kept);
    for (int r0 = 0; r0 < cnt; r0 += 8) {
      uint2 raw[8];
#pragma unroll
      for (int k = 0; k < 8; ++k)
        raw[k] = r0 + k < cnt ? __ldg(Vu + (size_t)(t * 32 + r0 + k) * (kD / 4) + lane)
                              : make_uint2(0u, 0u);
      float sq[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const int r = r0 + k;
        const float v[4] = {bf16lo(raw[k].x), bf16hi(raw[k].x), bf16lo(raw[k].y),
                            bf16hi(raw[k].y)};
        sq[k] = fmaf(v[3], v[3], fmaf(v[2], v[2], fmaf(v[1], v[1], v[0] * v[0])));
#pragma unroll
        for (int g = 0; g < G; ++g) {
          const float wk = __shfl_sync(kFull, pk[g], r), wt = __shfl_sync(kFull, pt[g], r);
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            ak[g][i] = fmaf(wk, v[i], ak[g][i]);
            at[g][i] = fmaf(wt, v[i], at[g][i]);
          }
        }
        if (sc != nullptr) {
          const float ws = __shfl_sync(kFull, sj, r);
#pragma unroll
          for (int i = 0; i < 4; ++i) sv[i] = fmaf(ws, v[i], sv[i]);
        }
        if (part_tm != nullptr && ((tailbits >> r) & 1u)) {
#pragma unroll
          for (int i = 0; i < 4; ++i) tv[i] += v[i];
          tq += sq[k];
        }
      }
      vmax = fmaxf(vmax, sqrtf(reduce8(sq, lane)));  // lane l: row r0 + (l & 7)
    }
  }
  vmax = warp_max(vmax);
  // combine the 4 warps, one query head at a time
  const int i = threadIdx.x;  // 128 threads = kD dimensions
#pragma unroll
  for (int g = 0; g < G; ++g) {
    float tk = lk[g], tt = lt[g];
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) {
      tk += __shfl_xor_sync(kFull, tk, o);
      tt += __shfl_xor_sync(kFull, tt, o);
    }
    if (lane == 0) wp[warp][g] = DiagPart{m[g], tk, tt, vmax};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      wacc[warp][0][lane * 4 + e] = ak[g][e];
      wacc[warp][1][lane * 4 + e] = at[g][e];
    }
    __syncthreads();
    float M = -INFINITY, vm = 0.f;
#pragma unroll
    for (int wi = 0; wi < 4; ++wi) {
      M = fmaxf(M, wp[wi][g].m);
      vm = fmaxf(vm, wp[wi][g].vmax);
    }
    float LK = 0.f, LT = 0.f, A = 0.f, B = 0.f;
#pragma unroll
    for (int wi = 0; wi < 4; ++wi) {
      if (wp[wi][g].m > -INFINITY) {
        const float f = exp2f(wp[wi][g].m - M);
        LK += wp[wi][g].l_kept * f;
        LT += wp[wi][g].l_tail * f;
        A += wacc[wi][0][i] * f;
        B += wacc[wi][1][i] * f;
      }
    }
    const size_t pi = ((size_t)u * kDiagSplits + split) * G + g;
    part_acc[(pi * 2 + 0) * kD + i] = A;
    part_acc[(pi * 2 + 1) * kD + i] = B;
    if (i == 0) part[pi] = DiagPart{M, LK, LT, vm};
    __syncthreads();
  }
  if (sc != nullptr) {  // block-uniform
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) ssum += __shfl_xor_sync(kFull, ssum, o);
#pragma unroll
    for (int e = 0; e < 4; ++e) wsv[warp][lane * 4 + e] = sv[e];
    if (lane == 0) wss[warp] = ssum;
    __syncthreads();
    float* ps = part_sv + ((size_t)u * kDiagSplits + split) * kSvStride;
    ps[i] = (wsv[0][i] + wsv[1][i]) + (wsv[2][i] + wsv[3][i]);
    if (i == 0) ps[kD] = (wss[0] + wss[1]) + (wss[2] + wss[3]);
  }
  if (part_tm != nullptr) {  // block-uniform
    __syncthreads();  // wsv / wss may still be read above
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) tq += __shfl_xor_sync(kFull, tq, o);
#pragma unroll
    for (int e = 0; e < 4; ++e) wsv[warp][lane * 4 + e] = tv[e];
    if (lane == 0) wss[warp] = tq;
    __syncthreads();
    float* pt = part_tm + ((size_t)u * kDiagSplits + split) * kSvStride;
    pt[i] = (wsv[0][i] + wsv[1][i]) + (wsv[2][i] + wsv[3][i]);
    if (i == 0) pt[kD] = (wss[0] + wss[1]) + (wss[2] + wss[3]);
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
// query head, write its fixed-row statistics, then (with scores) sweep the
// stored logits of the evicted tokens for the two L1 sums of the lift.
__global__ void __launch_bounds__(128) fixed_row_merge_kernel(
    Prob p, int G, const DiagPart* __restrict__ part, const float* __restrict__ part_acc,
    const __nv_bfloat16* __restrict__ ohat, const __nv_bfloat16* __restrict__ q,
    const __nv_bfloat16* __restrict__ pk, const __nv_bfloat16* __restrict__ pv,
    const int64_t* __restrict__ offsets, const int32_t* __restrict__ counts, int tail_slot,
    float scale_log2, const float* __restrict__ sc, const float* __restrict__ z2,
    const float* __restrict__ part_sv, const uint32_t* __restrict__ mask,
    float* __restrict__ stats) {
  __shared__ float red[4];
  const int ug = blockIdx.x;
  const int u = ug / G, g = ug - u * G;
  const int i = threadIdx.x;
  const int n = p.n, words = (n + 31) / 32;
  float M = -INFINITY, vm = 0.f;
  for (int s = 0; s < kDiagSplits; ++s) {
    const DiagPart d = part[((size_t)u * kDiagSplits + s) * G + g];
    M = fmaxf(M, d.m);
    vm = fmaxf(vm, d.vmax);
  }
  float LK = 0.f, LT = 0.f, AK = 0.f, AT = 0.f;
  for (int s = 0; s < kDiagSplits; ++s) {
    const size_t pi = ((size_t)u * kDiagSplits + s) * G + g;
    const DiagPart d = part[pi];
    if (d.m > -INFINITY) {
      const float f = exp2f(d.m - M);
      LK += d.l_kept * f;
      LT += d.l_tail * f;
      AK += part_acc[(pi * 2 + 0) * kD + i] * f;
      AT += part_acc[(pi * 2 + 1) * kD + i] * f;
    }
  }
  const float LA = LK + LT;
  const float o = (AK + AT) / LA;               // exact attention
  const float os = LK > 0.f ? AK / LK : 0.f;    // subset-only output
  const float uu = AT / LA;                     // fixed-row correction
  const float pS = LK / LA, pT = LT / LA;
  const int bl = u / p.H, h = u - bl * p.H;
  const size_t qi = (size_t)bl * p.Hq + (size_t)h * G + g;
  const float oh = __bfloat162float(ohat[qi * kD + i]);
  // the tail mass is pT (computed from the tail's own sum), not 1 - pS, which
  // loses it to cancellation when the kept tokens hold almost all the mass
  const float vbt = pT > 0.f ? uu / pT : 0.f;
  const float f = os + pT * (vbt - os) - o;
  const float nO = block_sum_128(o * o, red);
  const float eS = block_sum_128((os - o) * (os - o), red);
  const float nu = block_sum_128(uu * uu, red);
  const float eh = block_sum_128((oh - o) * (oh - o), red);
  const float res = block_sum_128(f * f, red);

  // the synthetic slot: its logit z* (log2 domain), compressed weight q and
  // Lambda_T - z* (natural log units)
  const bool slot = tail_slot != 0;
  float qstar = 0.f, dlam = NAN, dmix = NAN;
  const size_t srow = slot ? (size_t)(offsets[u] + counts[u]) : 0;
  if (slot) {
    const float xs =
        block_sum_128(__bfloat162float(q[qi * kD + i]) * __bfloat162float(pk[srow * kD + i]), red) *
        scale_log2;
    qstar = 1.f / (1.f + exp2f(M + log2f(LK) - xs));
    dlam = 0.6931471805599453f * (M + log2f(LT) - xs);
  }
  float d1 = NAN, d2 = NAN;
  if (sc != nullptr) {
    float ST = 0.f, SV = 0.f;
    for (int s = 0; s < kDiagSplits; ++s) {
      const float* ps = part_sv + ((size_t)u * kDiagSplits + s) * kSvStride;
      SV += ps[i];
      ST += ps[kD];
    }
    if (slot && ST > 0.f) {  // the stored value against the exact r-mixture
      const float e = __bfloat162float(pv[srow * kD + i]) - SV / ST;
      dmix = sqrtf(block_sum_128(e * e, red));
    }
    const int nT = n - counts[u];
    const float invLT = LT > 0.f ? 1.f / LT : 0.f, invLA = 1.f / LA;
    const float invST = ST > 0.f ? 1.f / ST : 0.f, uni = 1.f / (float)nT;
    const float* zz = z2 + ((size_t)u * G + g) * n;
    const float* su = sc + (size_t)u * n;
    const uint32_t* mu = mask + (size_t)u * words;
    float a1 = 0.f, a2 = 0.f;
    for (int j = i; j < n; j += 128) {
      if ((mu[j >> 5] >> (j & 31)) & 1u) continue;
      const float e = exp2f(zz[j] - M);
      const float r = ST > 0.f ? su[j] * invST : uni;
      a1 += fabsf(e * invLT - r);          // |a_j - r_j|
      a2 += fabsf(e * invLA - qstar * r);  // |A_j - q r_j|
    }
    d1 = block_sum_128(a1, red);
    // on S the lifted row is Ahat = A * Z / Zhat, so sum_S |A - Ahat| =
    // |p_S - (1 - q)| = |q - p_T|
    d2 = fabsf(qstar - pT) + block_sum_128(a2, red);
  }
  if (i == 0) {
    float* st = stats + qi * CERTKV_FIXED_ROW_STATS;
    st[0] = pS;
    st[1] = sqrtf(nO);
    st[2] = sqrtf(eS);
    st[3] = sqrtf(nu);
    st[4] = 2.f * vm * pT;
    st[5] = sqrtf(eh);
    st[6] = vm;
    st[7] = sqrtf(res);
    st[8] = pT;
    st[9] = qstar;
    st[10] = d1;
    st[11] = dlam;
    st[12] = sc != nullptr ? vm * (2.f * fabsf(pT - qstar) + fminf(pT, qstar) * d1) : NAN;
    st[13] = slot ? tanhf(0.25f * fabsf(dlam)) : NAN;
    st[14] = d2;
    st[15] = dmix;
  }
}

// ---------------------------------------------- sampled tail compensation --

// grid = units * G, block = 128: merge the splits of one query head into its
// log2-domain maximum and kept / evicted sums, scal[ug] = (M, LK, LT, 0), and
// the fixed-row correction u* = sum_T A_j v_j.
__global__ void __launch_bounds__(128) sampled_merge_kernel(int G, const DiagPart* __restrict__ part,
                                                            const float* __restrict__ part_acc,
                                                            float4* __restrict__ scal,
                                                            float* __restrict__ ustar) {
  const int ug = blockIdx.x;
  const int u = ug / G, g = ug - u * G;
  const int i = threadIdx.x;
  float M = -INFINITY;
  for (int s = 0; s < kDiagSplits; ++s) M = fmaxf(M, part[((size_t)u * kDiagSplits + s) * G + g].m);
  float LK = 0.f, LT = 0.f, AT = 0.f;
  for (int s = 0; s < kDiagSplits; ++s) {
    const size_t pi = ((size_t)u * kDiagSplits + s) * G + g;
    const DiagPart d = part[pi];
    if (d.m > -INFINITY) {
      const float f = exp2f(d.m - M);
      LK += d.l_kept * f;
      LT += d.l_tail * f;
      AT += part_acc[(pi * 2 + 1) * kD + i] * f;
    }
  }
  ustar[(size_t)ug * kD + i] = AT / (LK + LT);
  if (i == 0) scal[ug] = make_float4(M, LK, LT, 0.f);
}

constexpr int kSampThreads = 256;

// grid = units * G, block = kSampThreads: the two sampled estimators of u* for
// one query head (see the proposition on sampled tail compensation).  Thread t
// owns tokens [t CH, (t + 1) CH); the cumulative tail weight is summed in
// float64 in token order, chunk by chunk.
__global__ void __launch_bounds__(kSampThreads) sampled_kernel(
    Prob p, int G, int m, const float* __restrict__ z2, const uint32_t* __restrict__ mask,
    const int32_t* __restrict__ counts, const __nv_bfloat16* __restrict__ V,
    const float4* __restrict__ scal, const float* __restrict__ ustar,
    const float* __restrict__ part_tm, const float* __restrict__ unif,
    int32_t* __restrict__ idx_out, float* __restrict__ stats) {
  __shared__ double cpre[kSampThreads + 1];  // cumulative tail weight before chunk t
  __shared__ int npre[kSampThreads + 1];     // tail tokens before chunk t
  __shared__ double wq[kSampThreads];
  __shared__ int sidx[2 * CERTKV_MAX_SAMPLES];
  __shared__ int srank[CERTKV_MAX_SAMPLES];
  __shared__ float red[8];
  const int ug = blockIdx.x;
  const int u = ug / G;
  const int t = threadIdx.x;
  const int n = p.n, words = (n + 31) / 32;
  const int CH = (n + kSampThreads - 1) / kSampThreads;
  const int j0 = min(n, t * CH), j1 = min(n, j0 + CH);
  const float* zz = z2 + (size_t)ug * n;
  const uint32_t* mu = mask + (size_t)u * words;
  const float4 sc = scal[ug];
  const float M = sc.x, LA = sc.y + sc.z;
  // pass 1: per-chunk tail weight (float64, token order), its squares, tail count
  double c = 0.0, c2 = 0.0;
  int cnt = 0;
  for (int j = j0; j < j1; ++j) {
    if ((mu[j >> 5] >> (j & 31)) & 1u) continue;
    const double w = (double)exp2f(zz[j] - M);
    c += w;
    c2 += w * w;
    ++cnt;
  }
  wq[t] = c2;
  cpre[t + 1] = c;
  npre[t + 1] = cnt;
  __syncthreads();
  if (t == 0) {
    cpre[0] = 0.0;
    npre[0] = 0;
    for (int k = 1; k <= kSampThreads; ++k) {
      cpre[k] += cpre[k - 1];
      npre[k] += npre[k - 1];
    }
    double q2 = 0.0;
    for (int k = 0; k < kSampThreads; ++k) q2 += wq[k];
    wq[0] = q2;
  }
  __syncthreads();
  const double WT = cpre[kSampThreads];
  const int N = npre[kSampThreads];
  if (m > N) {  // fewer evicted tokens than samples: nothing to estimate
    if (idx_out != nullptr && t < 2 * m) idx_out[(size_t)ug * 2 * m + t] = -1;
    if (t < 8) stats[(size_t)ug * 8 + t] = __int_as_float(0x7fc00000);
    return;
  }
  // weight-proportional draws: thread r < m inverts the cumulative weight
  if (t < m) {
    const double target = (double)unif[(size_t)ug * 2 * m + t] * WT;
    int lo = 0, hi = kSampThreads - 1;  // first chunk whose end exceeds the target
    while (lo < hi) {
      const int mid = (lo + hi) >> 1;
      if (cpre[mid + 1] > target) hi = mid;
      else lo = mid + 1;
    }
    if (!(cpre[lo + 1] > target))  // rounding at the very end: the last chunk with tail tokens
      while (lo > 0 && npre[lo + 1] == npre[lo]) --lo;
    const int a = min(n, lo * CH), b = min(n, a + CH);
    double cc = cpre[lo];
    int pick = -1, last = -1;
    for (int j = a; j < b; ++j) {
      if ((mu[j >> 5] >> (j & 31)) & 1u) continue;
      last = j;
      cc += (double)exp2f(zz[j] - M);
      if (cc > target) { pick = j; break; }
    }
    sidx[t] = pick >= 0 ? pick : last;  // rounding at the chunk end: its last tail token
  }
  // uniform subset of the tail ranks (Floyd's algorithm), one thread
  if (t == 0) {
    for (int s2 = 0; s2 < m; ++s2) {
      const int i = N - m + s2;
      int r = (int)floor((double)unif[(size_t)ug * 2 * m + m + s2] * (double)(i + 1));
      if (r > i) r = i;
      bool taken = false;
      for (int e = 0; e < s2; ++e) taken = taken || (srank[e] == r);
      srank[s2] = taken ? i : r;
    }
  }
  __syncthreads();
  // tail rank -> token: thread s < m finds its chunk, then counts within it
  if (t < m) {
    const int r = srank[t];
    int lo = 0, hi = kSampThreads - 1;
    while (lo < hi) {
      const int mid = (lo + hi) >> 1;
      if (npre[mid + 1] > r) hi = mid;
      else lo = mid + 1;
    }
    int k = npre[lo], pick = -1;
    for (int j = min(n, lo * CH); j < min(n, lo * CH + CH); ++j) {
      if ((mu[j >> 5] >> (j & 31)) & 1u) continue;
      if (k == r) { pick = j; break; }
      ++k;
    }
    sidx[m + t] = pick;
  }
  __syncthreads();
  if (idx_out != nullptr && t < 2 * m) idx_out[(size_t)ug * 2 * m + t] = sidx[t];
  // the estimates (threads 0..127: weight-proportional, 128..255: uniform)
  const int dim = t & (kD - 1), half = t >> 7;
  float acc = 0.f;
  for (int r = 0; r < m; ++r) {
    const int j = sidx[half * m + r];
    if (j >= 0) acc += __bfloat162float(V[((size_t)u * n + j) * kD + dim]);
  }
  const float pT = sc.z / LA;
  const float us = ustar[(size_t)ug * kD + dim];
  const float e = acc * (pT / (float)m) - us;
  // block sums: e^2 of each half, ||u*||^2 from the first half
  float x = e * e, y = half == 0 ? us * us : 0.f;
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) {
    x += __shfl_xor_sync(kFull, x, o);
    y += __shfl_xor_sync(kFull, y, o);
  }
  __syncthreads();
  if ((t & 31) == 0) red[t >> 5] = x;
  __syncthreads();
  if (t == 0) {
    const float ew = (red[0] + red[1]) + (red[2] + red[3]);
    const float eu = (red[4] + red[5]) + (red[6] + red[7]);
    red[0] = ew;
    red[1] = eu;
  }
  __syncthreads();
  if ((t & 31) == 0 && t < 128) red[2 + (t >> 5)] = y;
  __syncthreads();
  if (t == 0) {
    const float nu = (red[2] + red[3]) + (red[4] + red[5]);
    // evicted values' per-coordinate variance from the split moments
    double sv2 = 0.0, sq = 0.0;
    for (int d = 0; d < kD; ++d) {
      double sd = 0.0;
      for (int s2 = 0; s2 < kDiagSplits; ++s2)
        sd += part_tm[((size_t)u * kDiagSplits + s2) * kSvStride + d];
      sv2 += sd * sd;
    }
    for (int s2 = 0; s2 < kDiagSplits; ++s2) sq += part_tm[((size_t)u * kDiagSplits + s2) * kSvStride + kD];
    const double s2v = N > 0 ? (sq - sv2 / N) / ((double)kD * N) : 0.0;
    // 1 - p_S as the tail's own mass (no cancellation when p_S is near 1)
    const double pSd = (double)sc.y / (double)LA, pTd = (double)sc.z / (double)LA;
    const double omp2 = pTd * pTd;
    const double QT = wq[0] / ((double)LA * (double)LA);
    const double imb = omp2 > 0.0 ? QT / omp2 : 0.0;
    const double mse_w = kD * s2v * omp2 / m * (1.0 - imb);
    const double mse_u = kD * s2v * omp2 * (1.0 / m - 2.0 / N + imb);
    float* st = stats + (size_t)ug * 8;
    st[0] = (float)pSd;
    st[1] = (float)QT;
    st[2] = sqrtf(nu);
    st[3] = sqrtf(red[0]);
    st[4] = sqrtf(red[1]);
    st[5] = (float)sqrt(mse_w > 0.0 ? mse_w : 0.0);
    st[6] = (float)sqrt(mse_u > 0.0 ? mse_u : 0.0);
    st[7] = (float)s2v;
  }
}

namespace {
struct FixedRowLayout {
  size_t mask, part, acc, z2, sv, ohat, dec, total;
};
FixedRowLayout fixed_row_layout(const Prob& p) {
  const size_t words = (size_t)(p.n + 31) / 32;
  const size_t parts = (size_t)p.units * kDiagSplits * p.G;
  auto a = [](size_t x) { return (x + 255) / 256 * 256; };
  FixedRowLayout ly;
  ly.mask = 0;
  ly.part = ly.mask + a(p.units * words * 4);
  ly.acc = ly.part + a(parts * sizeof(DiagPart));
  ly.z2 = ly.acc + a(parts * 2 * kD * 4);
  ly.sv = ly.z2 + a((size_t)p.units * p.G * p.n * 4);
  ly.ohat = ly.sv + a((size_t)p.units * kDiagSplits * kSvStride * 4);
  ly.dec = ly.ohat + a((size_t)p.units * p.G * kD * 2);
  ly.total = ly.dec + a(decode_workspace(p));
  return ly;
}
struct SampledLayout {
  size_t tm, scal, ustar, total;
};
SampledLayout sampled_layout(const Prob& p) {
  auto a = [](size_t x) { return (x + 255) / 256 * 256; };
  SampledLayout ly;
  ly.tm = fixed_row_layout(p).total;
  ly.scal = ly.tm + a((size_t)p.units * kDiagSplits * kSvStride * 4);
  ly.ustar = ly.scal + a((size_t)p.units * p.G * sizeof(float4));
  ly.total = ly.ustar + a((size_t)p.units * p.G * kD * 4);
  return ly;
}
}  // namespace

size_t sampled_workspace(const Prob& p) { return sampled_layout(p).total; }

bool launch_sampled(const Prob& p, const void* q, const void* K, const void* V,
                    const int64_t* offsets, const int32_t* counts, const int32_t* positions,
                    int m, const float* unif, int32_t* idx_out, float scale, float* stats,
                    char* ws, cudaStream_t st) {
  const FixedRowLayout ly = fixed_row_layout(p);
  const SampledLayout sl = sampled_layout(p);
  const size_t words = (size_t)(p.n + 31) / 32;
  uint32_t* mask = reinterpret_cast<uint32_t*>(ws + ly.mask);
  DiagPart* part = reinterpret_cast<DiagPart*>(ws + ly.part);
  float* acc = reinterpret_cast<float*>(ws + ly.acc);
  float* z2 = reinterpret_cast<float*>(ws + ly.z2);
  float* psv = reinterpret_cast<float*>(ws + ly.sv);
  float* ptm = reinterpret_cast<float*>(ws + sl.tm);
  float4* scal = reinterpret_cast<float4*>(ws + sl.scal);
  float* ustar = reinterpret_cast<float*>(ws + sl.ustar);
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
#define CERTKV_SC_SPLIT(GG)                                                                  \
  fixed_row_split_kernel<GG><<<grid, 128, 0, st>>>(p, qb, kb, vb, mask, nullptr, sl2, part, acc, \
                                                  z2, psv, ptm)
    switch (p.G) {
      case 1: CERTKV_SC_SPLIT(1); break;
      case 2: CERTKV_SC_SPLIT(2); break;
      case 4: CERTKV_SC_SPLIT(4); break;
      case 8: CERTKV_SC_SPLIT(8); break;
      case 16: CERTKV_SC_SPLIT(16); break;
      default: return false;
    }
#undef CERTKV_SC_SPLIT
  }
  {
    TraceScope ts_("sampled_merge", st);
    sampled_merge_kernel<<<p.units * p.G, 128, 0, st>>>(p.G, part, acc, scal, ustar);
  }
  {
    TraceScope ts_("sampled", st);
    sampled_kernel<<<p.units * p.G, kSampThreads, 0, st>>>(p, p.G, m, z2, mask, counts, vb, scal,
                                                          ustar, ptm, unif, idx_out, stats);
  }
  return true;
}

size_t fixed_row_workspace(const Prob& p) { return fixed_row_layout(p).total; }

bool launch_fixed_row(const Prob& p, const void* q, const void* K, const void* V,
                      const float* scores, const int64_t* offsets, const int32_t* counts,
                      const int32_t* positions, const void* pk, const void* pv, int tail_slot,
                      float scale, float* stats, char* ws, cudaStream_t st) {
  const FixedRowLayout ly = fixed_row_layout(p);
  const size_t words = (size_t)(p.n + 31) / 32;
  uint32_t* mask = reinterpret_cast<uint32_t*>(ws + ly.mask);
  DiagPart* part = reinterpret_cast<DiagPart*>(ws + ly.part);
  float* acc = reinterpret_cast<float*>(ws + ly.acc);
  float* z2 = reinterpret_cast<float*>(ws + ly.z2);
  float* psv = reinterpret_cast<float*>(ws + ly.sv);
  char* ohat = ws + ly.ohat;
  // the compressed decode's output, for its error against O
  if (!launch_decode(p, q, pk, pv, offsets, counts, tail_slot, scale, ohat, ws + ly.dec, st))
    return false;
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
#define CERTKV_FR_SPLIT(GG)                                                                  \
  fixed_row_split_kernel<GG><<<grid, 128, 0, st>>>(p, qb, kb, vb, mask, scores, sl2, part, acc, \
                                                  z2, psv, nullptr)
    switch (p.G) {
      case 1: CERTKV_FR_SPLIT(1); break;
      case 2: CERTKV_FR_SPLIT(2); break;
      case 4: CERTKV_FR_SPLIT(4); break;
      case 8: CERTKV_FR_SPLIT(8); break;
      case 16: CERTKV_FR_SPLIT(16); break;
      default: return false;
    }
#undef CERTKV_FR_SPLIT
  }
  {
    TraceScope ts_("fixed_row_merge", st);
    fixed_row_merge_kernel<<<p.units * p.G, 128, 0, st>>>(
        p, p.G, part, acc, reinterpret_cast<const __nv_bfloat16*>(ohat), qb,
        reinterpret_cast<const __nv_bfloat16*>(pk), reinterpret_cast<const __nv_bfloat16*>(pv),
        offsets, counts, tail_slot, sl2, scores, z2, psv, mask, stats);
  }
  return true;
}

}  // namespace certkv
