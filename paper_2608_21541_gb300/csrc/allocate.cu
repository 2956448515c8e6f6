// allocate.cu — a5: exact-budget split of B_real real-token slots over the H
// heads of every (sequence, layer) (Algorithm 1; implementation appendix).
//
// The paper's per-step argmin_b c_h(b) + lambda b over every b in
// [b_min, n-1] is answered on a candidate subset that provably contains every
// minimiser: the smallest minimiser of c(b) + lambda b for any lambda is a
// vertex of the lower convex hull of the points (b, c(b)).  The candidates are
//   hull_seg    per segment of kHullSeg points, a monotone-chain lower hull
//               in fp32 that only drops a point when it lies above a chord by
//               more than a rounding bound, so true hull vertices survive;
//   hull_merge  the same tolerant chain over the concatenated survivors.
// The bisection then evaluates c(b) + lambda b in float64 on the candidates
// with the same expression and rounding as a direct scan (smallest b on
// ties), so the result matches the algorithm as stated.  The best-marginal
// repair walks one token at a time with the heads' upcoming curve values
// staged in shared memory.
#include <float.h>
#include <limits.h>

#include "common.cuh"
#include "internal.cuh"

namespace certkv {

namespace {

// Should middle point B be dropped from the lower hull, i.e. is it above the
// chord from A to C by more than the fp32 rounding of this test can explain?
__device__ __forceinline__ bool clearly_above(int xa, float ya, int xb, float yb, int xc, float yc) {
  const float dx1 = (float)(xb - xa), dx2 = (float)(xc - xa);
  const float dy1 = yb - ya, dy2 = yc - ya;
  const float cross = dx1 * dy2 - dy1 * dx2;
  const float ymax = fmaxf(fmaxf(fabsf(ya), fabsf(yb)), fabsf(yc));
  const float eps = 16.0f * 5.9604645e-8f * ymax * (dx1 + dx2);  // 16 * 2^-24 * ...
  return cross < -eps;
}

__device__ __forceinline__ double curve_at(const float2* c, int b) {
  float2 v = c[b];
  return (double)v.x + (double)v.y;
}

}  // namespace

// grid = (ceil(hull_segs / 128), units), one thread per segment.
__global__ void __launch_bounds__(128) hull_seg_kernel(Prob p, const float2* __restrict__ curve,
                                                       int32_t* __restrict__ cand,
                                                       int32_t* __restrict__ ncand) {
  const int seg = blockIdx.x * blockDim.x + threadIdx.x;
  const int u = blockIdx.y;
  if (seg >= p.hull_segs) return;
  const int n = p.n;
  const float2* cu = curve + (size_t)u * n;
  int32_t* st = cand + (size_t)u * n + (size_t)seg * kHullSeg;  // private stack
  const int b0 = p.b_min + seg * kHullSeg;
  const int b1 = min(n, b0 + kHullSeg);
  int top = 0;
  int xa = 0, xb = 0;
  float ya = 0.f, yb = 0.f;
  for (int b = b0; b < b1; ++b) {
    const float y = cu[b].x;
    while (top >= 2 && clearly_above(xa, ya, xb, yb, b, y)) {
      --top;
      xb = xa;
      yb = ya;
      if (top >= 2) {
        xa = st[top - 2];
        ya = cu[xa].x;
      }
    }
    st[top++] = b;
    xa = xb;
    ya = yb;
    xb = b;
    yb = y;
  }
  ncand[(size_t)u * (p.hull_segs + 1) + seg] = top;
}

// grid = ceil(units / 128), one thread per unit: merge the segment survivors
// in place into the front of the unit's candidate list.
__global__ void __launch_bounds__(128) hull_merge_kernel(Prob p, const float2* __restrict__ curve,
                                                         int32_t* __restrict__ cand,
                                                         int32_t* __restrict__ ncand) {
  const int u = blockIdx.x * blockDim.x + threadIdx.x;
  if (u >= p.units) return;
  const int n = p.n;
  const float2* cu = curve + (size_t)u * n;
  int32_t* cl = cand + (size_t)u * n;
  int32_t* nc = ncand + (size_t)u * (p.hull_segs + 1);
  int top = 0;
  int xa = 0, xb = 0;
  float ya = 0.f, yb = 0.f;
  for (int s = 0; s < p.hull_segs; ++s) {
    const int cnt = nc[s];
    const int32_t* src = cl + (size_t)s * kHullSeg;
    for (int i = 0; i < cnt; ++i) {
      const int b = src[i];
      const float y = cu[b].x;
      while (top >= 2 && clearly_above(xa, ya, xb, yb, b, y)) {
        --top;
        xb = xa;
        yb = ya;
        if (top >= 2) {
          xa = cl[top - 2];
          ya = cu[xa].x;
        }
      }
      cl[top++] = b;
      xa = xb;
      ya = yb;
      xb = b;
      yb = y;
    }
  }
  nc[p.hull_segs] = top;
}

namespace {
// warp-wide lexicographic argmin of (f, b)
__device__ __forceinline__ void warp_argmin(double& f, int& b) {
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) {
    double of = __shfl_xor_sync(kFull, f, o);
    int ob = __shfl_xor_sync(kFull, b, o);
    if (of < f || (of == f && ob < b)) {
      f = of;
      b = ob;
    }
  }
}
}  // namespace

// grid = B*L, block = 256: bisection, repair, counts and offsets of one
// (sequence, layer).
__global__ void __launch_bounds__(256) bisect_repair_kernel(Prob p, const float2* __restrict__ curve,
                                                            const int32_t* __restrict__ cand,
                                                            const int32_t* __restrict__ ncand,
                                                            const unsigned long long* __restrict__ cmax,
                                                            int32_t* __restrict__ counts,
                                                            int64_t* __restrict__ offsets) {
  __shared__ int bsel[32];
  __shared__ double lam_sh[2];
  __shared__ double win[32][64];
  const int bl = blockIdx.x;
  const int H = p.H, n = p.n;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nwarps = blockDim.x >> 5;
  const int64_t B_real = p.B_real;

  if (threadIdx.x == 0) {
    double mx = 0.0;
    for (int h = 0; h < H; ++h) {
      double v = df_to_double(df_from_order_key(cmax[(size_t)bl * H + h]));
      mx = v > mx ? v : mx;
    }
    lam_sh[0] = 0.0;
    lam_sh[1] = __dadd_rn(__dmul_rn(2.0, mx), 1.0);
  }
  __syncthreads();

  auto argmin_heads = [&](double lam) {
    for (int h = warp; h < H; h += nwarps) {
      const int u = bl * H + h;
      const float2* cu = curve + (size_t)u * n;
      const int32_t* cl = cand + (size_t)u * n;
      const int cnt = ncand[(size_t)u * (p.hull_segs + 1) + p.hull_segs];
      double bf = INFINITY;
      int bb = INT_MAX;
      for (int k = lane; k < cnt; k += 32) {
        const int b = cl[k];
        const double f = __dadd_rn(curve_at(cu, b), __dmul_rn(lam, (double)b));
        if (f < bf || (f == bf && b < bb)) {
          bf = f;
          bb = b;
        }
      }
      warp_argmin(bf, bb);
      if (lane == 0) bsel[h] = (bb == INT_MAX) ? p.b_min : bb;
    }
  };

  for (int t = 0; t < p.T; ++t) {
    const double lam = __dmul_rn(__dadd_rn(lam_sh[0], lam_sh[1]), 0.5);
    argmin_heads(lam);
    __syncthreads();
    if (threadIdx.x == 0) {
      int64_t tot = 0;
      for (int h = 0; h < H; ++h) tot += bsel[h];
      if (tot > B_real) lam_sh[0] = lam; else lam_sh[1] = lam;
    }
    __syncthreads();
  }
  argmin_heads(lam_sh[1]);
  __syncthreads();

  if (warp == 0) {
    const int h = lane;
    const bool live = h < H;
    int b = live ? bsel[h] : 0;
    const float2* cu = curve + (size_t)(bl * H + (live ? h : 0)) * n;
    int64_t tot = 0;
    for (int i = 0; i < H; ++i) tot += bsel[i];
    // surplus (not reachable from lambda_hi, kept for robustness): remove one
    while (tot > B_real) {
      double mg = INFINITY;
      if (live && b > p.b_min) {
        double d = curve_at(cu, b - 1) - curve_at(cu, b);
        mg = (d == d) ? d : DBL_MAX;
      }
      int who = lane;
      warp_argmin(mg, who);
      if (lane == who) --b;
      --tot;
    }
    // best-marginal repair: add one token at a time
    double cb = live ? curve_at(cu, b) : 0.0;
    int wpos = 64;
    while (tot < B_real) {
      double mg = INFINITY;
      if (live && b < n - 1) {
        if (wpos == 64) {
          for (int k = 0; k < 64; ++k) win[h][k] = (b + 1 + k < n) ? curve_at(cu, b + 1 + k) : 0.0;
          wpos = 0;
        }
        const double d = win[h][wpos] - cb;
        mg = (d == d) ? d : DBL_MAX;
      }
      int who = lane;
      warp_argmin(mg, who);
      if (lane == who) {
        cb = win[h][wpos];
        ++wpos;
        ++b;
      }
      ++tot;
    }
    // counts and offsets: segment = b_h real slots (+ 1 tail slot)
    int seg = live ? b + p.tail_slot : 0;
    int incl = seg;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      int y = __shfl_up_sync(kFull, incl, o);
      if (lane >= o) incl += y;
    }
    if (live) {
      counts[(size_t)bl * H + h] = b;
      offsets[(size_t)bl * H + h] = (int64_t)bl * p.B_live + (incl - seg);
    }
    if (bl == p.bl - 1 && lane == 0) offsets[(size_t)p.bl * H] = (int64_t)p.bl * p.B_live;
  }
}

void launch_allocate(const Prob& p, const Layout& ly, char* ws, int32_t* counts,
                     int64_t* offsets, cudaStream_t st) {
  const float2* curve = reinterpret_cast<const float2*>(ws + ly.curve);
  int32_t* cand = reinterpret_cast<int32_t*>(ws + ly.cand);
  int32_t* ncand = reinterpret_cast<int32_t*>(ws + ly.ncand);
  dim3 g1((p.hull_segs + 127) / 128, p.units);
  {
    TraceScope ts_("hull_seg", st);
    hull_seg_kernel<<<g1, 128, 0, st>>>(p, curve, cand, ncand);
  }
  {
    TraceScope ts_("hull_merge", st);
    hull_merge_kernel<<<(p.units + 127) / 128, 128, 0, st>>>(p, curve, cand, ncand);
  }
  {
    TraceScope ts_("bisect_repair", st);
    bisect_repair_kernel<<<p.bl, 256, 0, st>>>(
        p, curve, cand, ncand, reinterpret_cast<const unsigned long long*>(ws + ly.cmax), counts,
        offsets);
  }
}

}  // namespace certkv
