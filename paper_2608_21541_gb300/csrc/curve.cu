// curve.cu — a4: suffix moments and the allocation curve of every unit.
//
// Implementation appendix (and Eq. certkv-curve): over the score-sorted axis,
// for the evicted suffix E(b) = ranks b..n-1,
//   m(b) = sum a_j,  W(b) = sum a_j v_j,  Q(b) = sum a_j ||v_j||^2,
//   c(b)^2 = (m(b) Q(b) - ||W(b)||^2)_+ .
// The ranks are cut into chunks of kChunk; one warp owns a chunk.
//   agg     gathers V (and K, for the tail slot) in rank order and writes the
//           chunk sums of a, a||v||^2 (double-float), a v and a k (fp32), and
//           ||v||^2 per rank;
//   prefix  suffix-sums the chunk sums over chunks in double-float;
//   curve   walks each chunk from its last rank down, W(b) = W_base + P(b)
//           with P the in-chunk partial, and evaluates
//           c^2 = m Q - (||W_base||^2 + <2 W_base + P, P>) in double-float.
// The scalar sums that dominate c^2 (m, Q, ||W_base||^2) are carried in
// double-float so that c(b) agrees with a float64 evaluation to ~1e-13; the
// small in-chunk vector terms stay in fp32.
#include "common.cuh"
#include "internal.cuh"

namespace certkv {

namespace {

// As reduce8 (common.cuh), in double-float.
__device__ __forceinline__ DF reduce8_df(DF (&v)[8], int lane) {
#pragma unroll
  for (int o = 4; o >= 1; o >>= 1) {
    const bool upper = (lane & o) != 0;
#pragma unroll
    for (int i = 0; i < o; ++i) {
      const DF keep = upper ? v[i + o] : v[i];
      const DF send = upper ? v[i] : v[i + o];
      v[i] = df_add(keep, shfl_xor_df(send, o));
    }
  }
  DF x = v[0];
  x = df_add(x, shfl_xor_df(x, 8));
  x = df_add(x, shfl_xor_df(x, 16));
  return x;
}

// As reduce8, from fp32 inputs, in double-float (the first level is an
// error-free two_sum).
__device__ __forceinline__ DF reduce8_f2df(float (&v)[8], int lane) {
  DF w[4];
  {
    const bool upper = (lane & 4) != 0;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float keep = upper ? v[i + 4] : v[i];
      const float send = upper ? v[i] : v[i + 4];
      w[i] = two_sum(keep, __shfl_xor_sync(kFull, send, 4));
    }
  }
#pragma unroll
  for (int o = 2; o >= 1; o >>= 1) {
    const bool upper = (lane & o) != 0;
#pragma unroll
    for (int i = 0; i < o; ++i) {
      const DF keep = upper ? w[i + o] : w[i];
      const DF send = upper ? w[i] : w[i + o];
      w[i] = df_add(keep, shfl_xor_df(send, o));
    }
  }
  DF x = w[0];
  x = df_add(x, shfl_xor_df(x, 8));
  x = df_add(x, shfl_xor_df(x, 16));
  return x;
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}

constexpr int kEvalGroup = 8;                  // V rows per staged group
constexpr int kEvalAhead = 2;                  // groups in flight ahead of the one in use
constexpr int kEvalRing = kEvalAhead + 1;
constexpr int kEvalGroupBytes = kEvalGroup * kD * 2;

}  // namespace

constexpr int kAggAhead = 2;                   // groups in flight ahead of the one in use
constexpr int kAggRing = kAggAhead + 1;
constexpr int kAggRingBytes = 4 * kAggRing * 2 * kEvalGroupBytes;  // [warp][slot][V, K]
constexpr int kAggSmemBytes = kAggRingBytes + 4 * kChunk * 8;      // + a and token per rank

// grid = (ceil(chunks / 4), units), block = 128 (one warp per chunk), dynamic
// shared memory kAggSmemBytes.  The V (and K) rows of a chunk are staged in
// groups of 8 ranks (ascending) through a per-warp ring, kAggAhead groups
// ahead of their use.  Chunk sums of a and a||v||^2 are carried per lane in
// double-float and summed over the warp once at the end.
__global__ void __launch_bounds__(128) curve_agg_kernel(Prob p, const uint32_t* __restrict__ keys,
                                                        const int32_t* __restrict__ perm,
                                                        const __nv_bfloat16* __restrict__ K,
                                                        const __nv_bfloat16* __restrict__ V,
                                                        bool need_k, float4* __restrict__ agg_mq,
                                                        float* __restrict__ agg_v,
                                                        float* __restrict__ agg_k,
                                                        float2* __restrict__ yrank) {
  extern __shared__ __align__(16) unsigned char agg_smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int chunk = blockIdx.x * 4 + warp;
  const int u = blockIdx.y;
  if (chunk >= p.chunks) return;
  const int n = p.n;
  const int r0 = chunk * kChunk, r1 = min(n, r0 + kChunk);
  const uint32_t* ku = keys + (size_t)u * n;
  const int32_t* pu = perm + (size_t)u * n;
  const unsigned char* Vu = reinterpret_cast<const unsigned char*>(V + (size_t)u * n * kD);
  const unsigned char* Ku = reinterpret_cast<const unsigned char*>(K + (size_t)u * n * kD);
  unsigned char* ring_w = agg_smem + warp * (kAggRing * 2 * kEvalGroupBytes);
  const uint32_t ring = (uint32_t)__cvta_generic_to_shared(ring_w);
  float* sa = reinterpret_cast<float*>(agg_smem + kAggRingBytes) + warp * kChunk;
  int* sj = reinterpret_cast<int*>(agg_smem + kAggRingBytes + 4 * kChunk * 4) + warp * kChunk;

#pragma unroll
  for (int e = 0; e < kChunk / 32; ++e) {
    const int r = r0 + e * 32 + lane;
    const bool ok = r < r1;
    int j = ok ? pu[r] : 0;
    if (!CERTKV_IN_BOUNDS(j >= 0 && j < n, p.status)) j = 0;
    sa[e * 32 + lane] = ok ? key_score(ku[r]) : 0.f;
    sj[e * 32 + lane] = j;
  }
  __syncwarp();
  const int ngroups = (r1 - r0 + kEvalGroup - 1) / kEvalGroup;  // group g: chunk ranks 8g .. 8g+7
  // lane l copies 16-byte piece (l & 15) of rows (l >> 4) + 2k, k = 0..3
  auto stage = [&](int g) {
    if (g < ngroups) {
      const uint32_t dst = ring + (uint32_t)((g % kAggRing) * 2 * kEvalGroupBytes);
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int t = (lane >> 4) + 2 * k;
        const int rl = kEvalGroup * g + t;
        if (r0 + rl < r1) {
          const size_t src = (size_t)sj[rl] * (kD * 2) + (lane & 15) * 16;
          const uint32_t off = t * (kD * 2) + (lane & 15) * 16;
          cp_async16(dst + off, Vu + src);
          if (need_k) cp_async16(dst + kEvalGroupBytes + off, Ku + src);
        }
      }
    }
    cp_async_commit();
  };
#pragma unroll
  for (int g = 0; g < kAggAhead; ++g) stage(g);

  float sv[4] = {0.f, 0.f, 0.f, 0.f}, sk[4] = {0.f, 0.f, 0.f, 0.f};
  DF ml = df_make(0.f), ql = df_make(0.f);
  DF ylane = df_make(0.f);  // lane r: ||v||^2 of rank r of the current batch
  for (int g = 0; g < ngroups; ++g) {
    stage(g + kAggAhead);
    asm volatile("cp.async.wait_group %0;" ::"n"(kAggAhead) : "memory");
    __syncwarp();
    const unsigned char* rows = ring_w + (g % kAggRing) * 2 * kEvalGroupBytes;
    const int rl0 = kEvalGroup * g;
    const int cnt = r1 - (r0 + rl0);
    // ||v||^2: per lane the 4 squares of bf16 values (each exact in fp32) are
    // summed in fp32, the 32 lane partials in double-float.
    float yp[8];
#pragma unroll
    for (int t = 0; t < 8; ++t) {
      const float as = sa[rl0 + t];
      float v[4] = {0.f, 0.f, 0.f, 0.f}, k4[4] = {0.f, 0.f, 0.f, 0.f};
      if (t < cnt) {
        const uint2 rv = *reinterpret_cast<const uint2*>(rows + t * (kD * 2) + lane * 8);
        v[0] = bf16lo(rv.x);
        v[1] = bf16hi(rv.x);
        v[2] = bf16lo(rv.y);
        v[3] = bf16hi(rv.y);
        if (need_k) {
          const uint2 rk =
              *reinterpret_cast<const uint2*>(rows + kEvalGroupBytes + t * (kD * 2) + lane * 8);
          k4[0] = bf16lo(rk.x);
          k4[1] = bf16hi(rk.x);
          k4[2] = bf16lo(rk.y);
          k4[3] = bf16hi(rk.y);
        }
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        sv[i] = fmaf(as, v[i], sv[i]);
        sk[i] = fmaf(as, k4[i], sk[i]);
      }
      yp[t] = fmaf(v[3], v[3], fmaf(v[2], v[2], fmaf(v[1], v[1], v[0] * v[0])));
    }
    const DF y = reduce8_f2df(yp, lane);
    if ((lane >> 3) == (g & 3)) ylane = y;
    __syncwarp();  // the ring slot of group g is free once every lane has read it
    if ((g & 3) == 3 || g == ngroups - 1) {  // end of batch g / 4
      const int rl = 32 * (g >> 2) + lane;
      const bool ok = r0 + rl < r1;
      const float at = sa[rl];
      if (ok) {
        yrank[(size_t)u * n + r0 + rl] = make_float2(ylane.hi, ylane.lo);
        ml = df_add_f(ml, at);
        ql = df_add(ql, df_mul_f(ylane, at));
      }
    }
  }
  asm volatile("cp.async.wait_all;" ::: "memory");
  const DF m = warp_sum_df(ml), q = warp_sum_df(ql);
  const size_t ci = (size_t)u * p.chunks + chunk;
  reinterpret_cast<float4*>(agg_v + ci * kD)[lane] = make_float4(sv[0], sv[1], sv[2], sv[3]);
  if (need_k)
    reinterpret_cast<float4*>(agg_k + ci * kD)[lane] = make_float4(sk[0], sk[1], sk[2], sk[3]);
  if (lane == 0) agg_mq[ci] = make_float4(m.hi, m.lo, q.hi, q.lo);
}

// One warp evaluates chunk `chunk` of unit u.  The V rows of the chunk are
// staged in groups of 8 ranks (descending) through the warp's ring in shared
// memory (ring_w, kEvalRing groups), kEvalAhead groups ahead of the
// evaluation; sa, sj hold the chunk's scores and token indices.  Each lane
// loads the ||v||^2 of its rank of a 32-rank batch into a register at the
// batch's first group; it is used at the batch's end.
// kLast: the unit's last chunk (W_base = 0), in double-float.
struct EvalArgs {
  const uint32_t* keys;
  const int32_t* perm;
  const __nv_bfloat16* V;
  const float2* yrank;
  const float4* base_mq;
  const float2* base_v;
  float2* curve;
  unsigned long long* cmax;
  uint32_t* status;
};
template <bool kLast>
__device__ __forceinline__ void eval_chunk(const Prob& p, const EvalArgs& ea, int chunk, int u,
                                           int lane, unsigned char* ring_w, float* sa, int* sj) {
  const uint32_t* __restrict__ keys = ea.keys;
  const int32_t* __restrict__ perm = ea.perm;
  const __nv_bfloat16* __restrict__ V = ea.V;
  const float2* __restrict__ yrank = ea.yrank;
  const float4* __restrict__ base_mq = ea.base_mq;
  const float2* __restrict__ base_v = ea.base_v;
  float2* __restrict__ curve = ea.curve;
  unsigned long long* __restrict__ cmax = ea.cmax;
  uint32_t* status = ea.status;
  const int n = p.n;
  const int r0 = chunk * kChunk, r1 = min(n, r0 + kChunk);
  const uint32_t* ku = keys + (size_t)u * n;
  const int32_t* pu = perm + (size_t)u * n;
  const unsigned char* Vu = reinterpret_cast<const unsigned char*>(V + (size_t)u * n * kD);
  const size_t ci = (size_t)u * p.chunks + chunk;
  const uint32_t ring = (uint32_t)__cvta_generic_to_shared(ring_w);

  // per-rank scalars of the whole chunk (zero past the end)
#pragma unroll
  for (int e = 0; e < kChunk / 32; ++e) {
    const int r = r0 + e * 32 + lane;
    const bool ok = r < r1;
    int j = ok ? pu[r] : 0;
    if (!CERTKV_IN_BOUNDS(j >= 0 && j < n, p.status)) j = 0;
    sa[e * 32 + lane] = ok ? key_score(ku[r]) : 0.f;
    sj[e * 32 + lane] = j;
  }
  __syncwarp();
  const int nb = (r1 - r0 + 31) / 32;
  const int ngroups = nb * 4;  // group g: ranks r0 + 32*(nb-1-g/4) + 24 - 8*(g%4) + 0..7
  // lane l copies 16-byte piece (l & 15) of rows (l >> 4) + 2k, k = 0..3
  const bool full = r1 - r0 == kChunk;  // every chunk but a partial last one
  auto stage = [&](int g) {
    if (g < ngroups) {
      const int rl = 32 * (nb - 1 - g / 4) + 24 - 8 * (g % 4);  // first rank of the group, chunk-local
      const uint32_t dst = ring + (uint32_t)((g % kEvalRing) * kEvalGroupBytes);
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int t = (lane >> 4) + 2 * k;
        if (full || r0 + rl + t < r1)
          cp_async16(dst + t * (kD * 2) + (lane & 15) * 16,
                     Vu + (size_t)sj[rl + t] * (kD * 2) + (lane & 15) * 16);
      }
    }
    cp_async_commit();
  };
#pragma unroll
  for (int g = 0; g < kEvalAhead; ++g) stage(g);

  // the sums over the ranks after the chunk (zero after the last chunk, which
  // runs alongside the kernel that writes them and so must not read them)
  const float4 bmq = kLast ? make_float4(0.f, 0.f, 0.f, 0.f) : base_mq[ci];
  const DF M0{bmq.x, bmq.y}, Q0{bmq.z, bmq.w};
  float wb2x[4] = {0.f, 0.f, 0.f, 0.f};
  DF wb2 = df_make(0.f);
  if constexpr (!kLast) {
    const float4* bv = reinterpret_cast<const float4*>(base_v + ci * kD) + lane * 2;
    float4 x0 = bv[0], x1 = bv[1];
    const float hi[4] = {x0.x, x0.z, x1.x, x1.z}, lo[4] = {x0.y, x0.w, x1.y, x1.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      wb2x[i] = 2.0f * hi[i];
      DF sq = two_prod(hi[i], hi[i]);
      sq = df_add_f(sq, 2.0f * hi[i] * lo[i]);
      wb2 = df_add(wb2, sq);
    }
    wb2 = warp_sum_df(wb2);
  }
  // The last chunk has W_base = 0 and a vanishing tail, so c(b)^2 there is a
  // small difference of small terms: its partial sums run in double-float.
  constexpr bool exact = kLast;  // the last chunk: W_base = 0, in double-float
  float P[4] = {0.f, 0.f, 0.f, 0.f};
  DF Pd[4] = {df_make(0.f), df_make(0.f), df_make(0.f), df_make(0.f)};
  DF base_m = M0, base_q = Q0;  // sums over the ranks after the current batch
  unsigned long long best = 0ull;
  bool bad = false;
  DF xt = df_make(0.f);  // lane r: ||W_base + P(b)||^2 - ||W_base||^2 for rank r of the batch
  DF yt = df_make(0.f);  // lane r: ||v||^2 of rank r of the batch (last chunk only)
  float2 yv = make_float2(0.f, 0.f);  // lane r: ||v||^2 of rank r of the batch (as staged)
  for (int g = 0; g < ngroups; ++g) {
    stage(g + kEvalAhead);
    const int bi = nb - 1 - g / 4;
    const int s0 = 24 - 8 * (g % 4);
    if (!exact && s0 == 24) {  // the batch's first group: its ranks' ||v||^2, used at its end
      const int r = r0 + 32 * bi + lane;
      yv = r < r1 ? yrank[(size_t)u * n + r] : make_float2(0.f, 0.f);
    }
    asm volatile("cp.async.wait_group %0;" ::"n"(kEvalAhead) : "memory");
    __syncwarp();
    const int rl = 32 * bi + s0;
    const int cnt = r1 - (r0 + rl);  // rows of the group that exist (may exceed 8)
    const unsigned char* rows = ring_w + (g % kEvalRing) * kEvalGroupBytes;
    if constexpr (!exact) {
      // dimension pairs (0,1) and (2,3) of this lane in two-wide arithmetic
      float2 P01 = make_float2(P[0], P[1]), P23 = make_float2(P[2], P[3]);
      const float2 W01 = make_float2(wb2x[0], wb2x[1]), W23 = make_float2(wb2x[2], wb2x[3]);
      float xg[8];
      if (cnt >= 8) {  // a whole group (every group but a partial chunk's): no per-rank tests
        const float4 alo = *reinterpret_cast<const float4*>(sa + rl);
        const float4 ahi = *reinterpret_cast<const float4*>(sa + rl + 4);
        const float as8[8] = {alo.x, alo.y, alo.z, alo.w, ahi.x, ahi.y, ahi.z, ahi.w};
#pragma unroll
        for (int t = 7; t >= 0; --t) {
          const uint2 raw = *reinterpret_cast<const uint2*>(rows + t * (kD * 2) + lane * 8);
          const float2 a2 = make_float2(as8[t], as8[t]);
          P01 = ffma2(a2, make_float2(bf16lo(raw.x), bf16hi(raw.x)), P01);
          P23 = ffma2(a2, make_float2(bf16lo(raw.y), bf16hi(raw.y)), P23);
          const float2 acc = ffma2(fadd2(W23, P23), P23, fmul2(fadd2(W01, P01), P01));
          xg[t] = acc.x + acc.y;
        }
      } else {
#pragma unroll
        for (int t = 7; t >= 0; --t) {
          const float as = sa[rl + t];
          uint2 raw = make_uint2(0u, 0u);
          if (t < cnt) raw = *reinterpret_cast<const uint2*>(rows + t * (kD * 2) + lane * 8);
          const float2 a2 = make_float2(as, as);
          P01 = ffma2(a2, make_float2(bf16lo(raw.x), bf16hi(raw.x)), P01);
          P23 = ffma2(a2, make_float2(bf16lo(raw.y), bf16hi(raw.y)), P23);
          const float2 acc = ffma2(fadd2(W23, P23), P23, fmul2(fadd2(W01, P01), P01));
          xg[t] = (t < cnt) ? acc.x + acc.y : 0.f;
        }
      }
      P[0] = P01.x;
      P[1] = P01.y;
      P[2] = P23.x;
      P[3] = P23.y;
      const float x = reduce8(xg, lane);
      if ((lane >> 3) == (s0 >> 3)) xt = df_make(x);
    } else {
      // ||v||^2 is also recomputed here in double-float (the per-rank values
      // of curve_agg sum each lane's four squares in fp32, which rounds when
      // their magnitudes spread over more than 24 bits): near b = n - 1 the
      // tail holds a few tokens and m Q - ||W||^2 cancels to ~0, so Q and W
      // must see the same ||v||^2
      DF xg[8], yg[8];
#pragma unroll
      for (int t = 7; t >= 0; --t) {
        const float as = sa[rl + t];
        xg[t] = df_make(0.f);
        yg[t] = df_make(0.f);
        if (t < cnt) {
          const uint2 raw = *reinterpret_cast<const uint2*>(rows + t * (kD * 2) + lane * 8);
          const float v[4] = {bf16lo(raw.x), bf16hi(raw.x), bf16lo(raw.y), bf16hi(raw.y)};
          DF acc = df_make(0.f);
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            Pd[i] = df_add(Pd[i], two_prod(as, v[i]));
            acc = df_add(acc, df_mul(Pd[i], Pd[i]));
          }
          xg[t] = acc;
          // squares of bf16 values are exact in fp32
          yg[t] = df_add(two_sum(v[0] * v[0], v[1] * v[1]), two_sum(v[2] * v[2], v[3] * v[3]));
        }
      }
      const DF x = reduce8_df(xg, lane);
      const DF y = reduce8_df(yg, lane);
      if ((lane >> 3) == (s0 >> 3)) {
        xt = x;
        yt = y;
      }
    }
    __syncwarp();  // the ring slot of group g is free once every lane has read it
    if (s0 != 0) continue;

    // ---- end of batch bi: the curve at its 32 ranks ----
    const int r = r0 + 32 * bi + lane;
    const bool ok = r < r1;
    const float at = sa[32 * bi + lane];
    // in-batch inclusive suffix sums over lanes >= t (a and a||v||^2 are
    // non-negative: same-sign double-float additions)
    DF sm = df_make(at);
    DF sq = ok ? df_mul_f(exact ? yt : DF{yv.x, yv.y}, at) : df_make(0.f);
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      DF om{__shfl_down_sync(kFull, sm.hi, o), __shfl_down_sync(kFull, sm.lo, o)};
      DF oq{__shfl_down_sync(kFull, sq.hi, o), __shfl_down_sync(kFull, sq.lo, o)};
      if (lane + o < 32) {
        sm = df_add_same_sign(sm, om);
        sq = df_add_same_sign(sq, oq);
      }
    }
    const DF Mt = df_add_same_sign(base_m, sm);
    const DF Qt = df_add_same_sign(base_q, sq);
    DF c, arg = df_make(0.f);
    if (p.statistic == 2) {
      c = Mt;
    } else if (p.statistic == 1) {
      arg = df_mul(Mt, Qt);
      c = df_sqrt_newton(arg);
    } else {
      const DF W2 = df_add(wb2, xt);
      arg = df_add(df_mul(Mt, Qt), df_neg(W2));
      c = df_sqrt_newton(arg);
    }
    if (ok) {
      curve[(size_t)u * n + r] = make_float2(c.hi, c.lo);
      // a non-finite value (the square root maps a NaN argument, such as
      // inf - inf from an infinite value row, to 0, so test the argument too)
      if (!(c.hi <= 3.0e38f) || arg.hi != arg.hi) bad = true;
      unsigned long long k = df_order_key(c);
      best = k > best ? k : best;
    }
    base_m = df_add_same_sign(base_m, shfl_df(sm, 0));
    base_q = df_add_same_sign(base_q, shfl_df(sq, 0));
  }
  asm volatile("cp.async.wait_all;" ::: "memory");
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) {
    unsigned long long other = __shfl_xor_sync(kFull, best, o);
    best = other > best ? other : best;
  }
  if (lane == 0) atomicMax(cmax + u, best);
  if (__any_sync(kFull, bad) && lane == 0) raise_status(status, 1u);
}

// grid = (ceil(chunks / 4), units), block = 128: warp w of block x takes chunk
// 4x + w, every chunk but the last (curve_prefix_kernel takes the last ones).
__global__ void __launch_bounds__(128, 7)  // seven CTAs per SM: 69 registers, no spills
curve_eval_kernel(Prob p, EvalArgs ea) {
  __shared__ __align__(16) unsigned char s_ring[4][kEvalRing][kEvalGroupBytes];
  __shared__ __align__(16) float s_a[4][kChunk];  // read as float4 by whole groups
  __shared__ int s_j[4][kChunk];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int chunk = blockIdx.x * 4 + warp;
  if (chunk >= p.chunks - 1) return;
  eval_chunk<false>(p, ea, chunk, blockIdx.y, lane, s_ring[warp][0], s_a[warp], s_j[warp]);
}

// grid = (units, 2), block = 160: exclusive suffix sums over chunks in
// double-float, folded from the last chunk down in chunk order.  In
// blockIdx.y = 0, threads 0..127 take one dimension of the V sums, with the
// next kPrefixBlock chunks' loads in flight while the current ones are
// folded, and warp 4 the scalar sums m and Q, one chunk per lane per round.
// In blockIdx.y = 1, warp 0 evaluates the unit's last chunk of ranks instead
// (its W_base, m and Q bases are zero, so it needs none of these sums), in
// double-float, alongside.  The K sums are needed at one chunk per unit only
// (the tail slot's), so the tail kernel folds them itself.
constexpr int kPrefixBlock = 32;
__global__ void __launch_bounds__(160) curve_prefix_kernel(Prob p, const float4* __restrict__ agg_mq,
                                                           const float* __restrict__ agg_v,
                                                           float4* __restrict__ base_mq,
                                                           float2* __restrict__ base_v,
                                                           EvalArgs ea) {
  const int u = blockIdx.x;
  if (blockIdx.y == gridDim.y - 1) {
    __shared__ __align__(16) unsigned char l_ring[kEvalRing][kEvalGroupBytes];
    __shared__ __align__(16) float l_a[kChunk];
    __shared__ int l_j[kChunk];
    if (threadIdx.x < 32) eval_chunk<true>(p, ea, p.chunks - 1, u, threadIdx.x, l_ring[0], l_a, l_j);
    return;
  }
  const int chunks = p.chunks;
  const size_t c0 = (size_t)u * chunks;
  if (threadIdx.x >= kD) {
    const int lane = threadIdx.x & 31;
    DF rm = df_make(0.f), rq = df_make(0.f);
    float4 nxt = make_float4(0.f, 0.f, 0.f, 0.f);
    if (chunks - 1 - lane >= 0) nxt = agg_mq[c0 + chunks - 1 - lane];
    for (int top = chunks - 1; top >= 0; top -= 32) {
      const float4 cur = nxt;
      if (top - 32 - lane >= 0) nxt = agg_mq[c0 + top - 32 - lane];
      for (int e = 0; e < 32 && top - e >= 0; ++e) {
        if (lane == e) base_mq[c0 + top - e] = make_float4(rm.hi, rm.lo, rq.hi, rq.lo);
        const float mh = __shfl_sync(kFull, cur.x, e), ml = __shfl_sync(kFull, cur.y, e);
        const float qh = __shfl_sync(kFull, cur.z, e), ql = __shfl_sync(kFull, cur.w, e);
        rm = df_add(rm, DF{mh, ml});
        rq = df_add(rq, DF{qh, ql});
      }
    }
    return;
  }
  const int i = threadIdx.x;
  const float* src = agg_v + c0 * kD + i;
  float2* dst = base_v + c0 * kD + i;
  DF r = df_make(0.f);
  float nxt[kPrefixBlock];
#pragma unroll
  for (int e = 0; e < kPrefixBlock; ++e) {
    const int c = chunks - 1 - e;
    nxt[e] = c >= 0 ? src[(size_t)c * kD] : 0.f;
  }
  for (int top = chunks - 1; top >= 0; top -= kPrefixBlock) {
    float cur[kPrefixBlock];
#pragma unroll
    for (int e = 0; e < kPrefixBlock; ++e) {
      cur[e] = nxt[e];
      const int c = top - kPrefixBlock - e;
      nxt[e] = c >= 0 ? src[(size_t)c * kD] : 0.f;
    }
#pragma unroll
    for (int e = 0; e < kPrefixBlock; ++e) {
      const int c = top - e;
      if (c < 0) break;
      dst[(size_t)c * kD] = make_float2(r.hi, r.lo);
      r = df_add_f(r, cur[e]);
    }
  }
}

__global__ void cmax_clear_kernel(unsigned long long* cmax, int units) {
  int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < units) cmax[i] = 0ull;
}

__global__ void export_curves_kernel(Prob p, const int32_t* __restrict__ perm,
                                     const float2* __restrict__ curve, int32_t* __restrict__ perm_out,
                                     double* __restrict__ c_out) {
  const size_t total = (size_t)p.units * p.n;
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (size_t)gridDim.x * blockDim.x) {
    if (perm_out) perm_out[i] = perm[i];
    if (c_out) {
      float2 c = curve[i];
      c_out[i] = (double)c.x + (double)c.y;
    }
  }
}

void launch_curves(const Prob& p, const Layout& ly, char* ws, const void* K, const void* V,
                   bool need_k, cudaStream_t st) {
  const uint32_t* keys = reinterpret_cast<const uint32_t*>(ws + ly.keys0);
  const int32_t* perm = reinterpret_cast<const int32_t*>(ws + ly.vals0);
  const __nv_bfloat16* Kb = reinterpret_cast<const __nv_bfloat16*>(K);
  const __nv_bfloat16* Vb = reinterpret_cast<const __nv_bfloat16*>(V);
  float4* agg_mq = reinterpret_cast<float4*>(ws + ly.agg_mq);
  float* agg_v = reinterpret_cast<float*>(ws + ly.agg_v);
  float* agg_k = reinterpret_cast<float*>(ws + ly.agg_k);
  float2* yrank = reinterpret_cast<float2*>(ws + ly.yrank);
  float4* base_mq = reinterpret_cast<float4*>(ws + ly.base_mq);
  float2* base_v = reinterpret_cast<float2*>(ws + ly.base_v);
  float2* curve = reinterpret_cast<float2*>(ws + ly.curve);
  unsigned long long* cmax = reinterpret_cast<unsigned long long*>(ws + ly.cmax);
  dim3 grid((p.chunks + 3) / 4, p.units);
  {
    TraceScope ts_("cmax_clear", st);
    cmax_clear_kernel<<<(p.units + 255) / 256, 256, 0, st>>>(cmax, p.units);
  }
  static bool attr = false;
  if (!attr) {
    cudaFuncSetAttribute(curve_agg_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         kAggSmemBytes);
    attr = true;
  }
  {
    TraceScope ts_("curve_agg", st);
    curve_agg_kernel<<<grid, 128, kAggSmemBytes, st>>>(p, keys, perm, Kb, Vb, need_k, agg_mq, agg_v, agg_k,
                                           yrank);
  }
  const EvalArgs ea{keys,    perm,  Vb,   yrank, base_mq, base_v,
                    curve,   cmax,  reinterpret_cast<uint32_t*>(ws + ly.status)};
  {
    TraceScope ts_("curve_prefix", st);
    curve_prefix_kernel<<<dim3(p.units, 2), 160, 0, st>>>(p, agg_mq, agg_v, base_mq, base_v, ea);
  }
  {
    TraceScope ts_("curve_eval", st);
    curve_eval_kernel<<<grid, 128, 0, st>>>(p, ea);
  }
}

void launch_export_curves(const Prob& p, const Layout& ly, char* ws, int32_t* perm_out,
                          double* c_out, cudaStream_t st) {
  {
    TraceScope ts_("export_curves", st);
    export_curves_kernel<<<1024, 256, 0, st>>>(p, reinterpret_cast<const int32_t*>(ws + ly.vals0),
                                               reinterpret_cast<const float2*>(ws + ly.curve),
                                               perm_out, c_out);
  }
}

}  // namespace certkv
