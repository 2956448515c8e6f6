// allocate.cu — a5: exact-budget split of B_real real-token slots over the H
// heads of every (sequence, layer) (Algorithm 1; implementation appendix).
//
// The paper's per-step argmin_b c_h(b) + lambda b over every b in
// [b_min, n-1] is answered on a candidate subset that contains every
// minimiser: the smallest minimiser of c(b) + lambda b, for any lambda, is a
// vertex of the lower convex hull of the points (b, c(b)).  Candidates come
// from two levels of filtering, both in parallel:
//   hull_seg    one thread per segment of kHullSeg points;
//   hull_group  one thread per group of kGroupSegs segments, over the
//               segment survivors.
// Each level shears its points by the chord of its range (the lower hull is
// invariant under adding a linear function; the chord is computed in
// double-float) so that fp32 only resolves the small residual, and runs a
// monotone chain that drops a point only when it is above a chord by more
// than the rounding of the test can explain.  True hull vertices therefore
// always survive.
// The bisection (T steps on the shared multiplier, smallest b on ties) and
// the one-token best-marginal repair then run in double-float on the fp32
// pipe; the multiplier itself is bisected in float64 as the paper states.
#include <float.h>
#include <limits.h>

#include "../../include/certkv.h"
#include "common.cuh"
#include "internal.cuh"

namespace certkv {

namespace {

__device__ __forceinline__ DF curve_df(const float2* c, int b) {
  const float2 v = c[b];
  return DF{v.x, v.y};
}

__device__ __forceinline__ bool df_less(DF x, DF y) {
  return x.hi < y.hi || (x.hi == y.hi && x.lo < y.lo);
}

// Drop the middle point B of sheared values y only if it lies above the chord
// A-C by more than the fp32 rounding of this test plus the error `dy` of the
// sheared values can explain.
__device__ __forceinline__ bool clearly_above(int xa, float ya, int xb, float yb, int xc, float yc,
                                              float dy) {
  const float dx1 = (float)(xb - xa), dx2 = (float)(xc - xa);
  const float cross = dx1 * (yc - ya) - (yb - ya) * dx2;
  const float ymax = fmaxf(fmaxf(fabsf(ya), fabsf(yb)), fabsf(yc));
  const float eps = (dx1 + dx2) * (16.0f * 5.9604645e-8f * ymax + 8.0f * dy);
  return cross < -eps;
}

// c(b) minus the chord through (b0, c0) with slope `slope`, in fp32, and a
// bound on its error (2^-40 |c|, far above the double-float rounding).
struct Shear {
  const float2* cu;
  int b0;
  DF c0, slope;
  __device__ __forceinline__ void at(int b, float& y, float& dy) const {
    at_value(b, cu[b], y, dy);
  }
  // the same for a curve value c(b) already loaded
  __device__ __forceinline__ void at_value(int b, float2 v, float& y, float& dy) const {
    const DF cb{v.x, v.y};
    const DF line = df_add(c0, df_mul_f(slope, (float)(b - b0)));
    y = df_add(cb, df_neg(line)).hi;
    dy = 9.094947e-13f * fmaxf(fabsf(cb.hi), fabsf(line.hi));
  }
};

__device__ __forceinline__ Shear make_shear(const float2* cu, int b0, int b1) {
  Shear s;
  s.cu = cu;
  s.b0 = b0;
  s.c0 = curve_df(cu, b0);
  const DF c1 = curve_df(cu, b1);
  s.slope = (b1 > b0) ? df_div(df_add(c1, df_neg(s.c0)), df_make((float)(b1 - b0))) : df_make(0.f);
  return s;
}

// Candidate counts per unit: [hull_segs] segment counts, then [groups] group
// counts (see Layout::ncand).
__device__ __forceinline__ int groups_of(const Prob& p) {
  return (p.hull_segs + kGroupSegs - 1) / kGroupSegs;
}
__device__ __forceinline__ size_t ncand_stride(const Prob& p) {
  return (size_t)p.hull_segs + groups_of(p);
}

// warp-wide lexicographic argmin of (f, b)
__device__ __forceinline__ void warp_argmin_df(DF& f, int& b) {
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) {
    const DF of = shfl_xor_df(f, o);
    const int ob = __shfl_xor_sync(kFull, b, o);
    if (df_less(of, f) || (of.hi == f.hi && of.lo == f.lo && ob < b)) {
      f = of;
      b = ob;
    }
  }
}

__device__ __forceinline__ DF df_from_double(double x) {
  const float hi = __double2float_rn(x);
  return DF{hi, __double2float_rn(x - (double)hi)};
}

}  // namespace

// Stack slots per hull_seg thread held in shared memory (8 B each).
constexpr int kHullWin = 16;

// grid = (ceil(hull_segs / 128), units), block = 128 (the window's thread
// dimension), one thread per segment.
__global__ void __launch_bounds__(128) hull_seg_kernel(Prob p, const float2* __restrict__ curve,
                                                       int32_t* __restrict__ cand,
                                                       int32_t* __restrict__ ncand) {
  const int seg = blockIdx.x * blockDim.x + threadIdx.x;
  const int u = blockIdx.y;
  if (seg >= p.hull_segs) return;
  const int n = p.n;
  const float2* cu = curve + (size_t)u * n;
  int32_t* out = cand + (size_t)u * n + (size_t)seg * kHullSeg;
  const int b0 = p.b_min + seg * kHullSeg;
  const int b1 = min(n, b0 + kHullSeg);
  const Shear sh = make_shear(cu, b0, b1 - 1);
  // tolerant monotone chain (a point is dropped only when clearly_above says
  // so), with the sheared values of eight consecutive points evaluated ahead
  // (their curve loads in flight together) and kept on the thread-private
  // stack next to b (as its offset in the segment), so that a pop needs no
  // curve reload.  The top two entries are held in registers (xa, ya: entry
  // top - 2; xb, yb: entry top - 1), so a point that pops nothing reads no
  // stack memory.  Entries [spill, top) live in a window of kHullWin slots per
  // thread in shared memory (slot = entry mod kHullWin, one bank per lane
  // whatever the entries the lanes touch); older entries [0, spill) move to
  // the local arrays when the window is full (the stack stays within 18
  // entries on C3-shaped curves, so that is rare).  Each test takes the
  // largest error bound of the points seen so far, at least that of its own
  // three points: the filter can only keep more.
  static_assert(kHullSeg <= 256, "segment offsets are stored in one byte");
  static_assert((kHullWin & (kHullWin - 1)) == 0 && kHullWin >= 2, "window slots by mask");
  __shared__ int win_b[kHullWin][128];
  __shared__ float win_y[kHullWin][128];
  const int tid = threadIdx.x;
  uint8_t st[kHullSeg];
  float sty[kHullSeg];
  float dmax = 0.f;
  int top = 0, spill = 0;
  int xa = 0, xb = 0;
  float ya = 0.f, yb = 0.f;
  const int count = b1 - b0;
  // the curve values of the next eight points are loaded while the chain
  // takes the current eight
  float2 nxt[8];
#pragma unroll
  for (int k = 0; k < 8; ++k) nxt[k] = k < count ? cu[b0 + k] : make_float2(0.f, 0.f);
  for (int i0 = 0; i0 < count; i0 += 8) {
    float yv[8], dv[8];
#pragma unroll
    for (int k = 0; k < 8; ++k)
      if (i0 + k < count) sh.at_value(b0 + i0 + k, nxt[k], yv[k], dv[k]);
#pragma unroll
    for (int k = 0; k < 8; ++k)
      nxt[k] = i0 + 8 + k < count ? cu[b0 + i0 + 8 + k] : make_float2(0.f, 0.f);
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      if (i0 + k >= count) break;
      const int i = i0 + k;
      dmax = fmaxf(dmax, dv[k]);
      while (top >= 2 && clearly_above(xa, ya, xb, yb, i, yv[k], dmax)) {
        --top;
        if (top < spill) spill = top;
        xb = xa;
        yb = ya;
        if (top >= 2) {
          const int e = top - 2;
          if (e >= spill) {
            xa = win_b[e & (kHullWin - 1)][tid];
            ya = win_y[e & (kHullWin - 1)][tid];
          } else {
            xa = st[e];
            ya = sty[e];
          }
        }
      }
      if (top - spill == kHullWin) {  // window full: its oldest entry to local memory
        st[spill] = (uint8_t)win_b[spill & (kHullWin - 1)][tid];
        sty[spill] = win_y[spill & (kHullWin - 1)][tid];
        ++spill;
      }
      win_b[top & (kHullWin - 1)][tid] = i;
      win_y[top & (kHullWin - 1)][tid] = yv[k];
      ++top;
      xa = xb;
      ya = yb;
      xb = i;
      yb = yv[k];
    }
  }
  for (int e = 0; e < top; ++e) out[e] = b0 + (e < spill ? (int)st[e] : win_b[e & (kHullWin - 1)][tid]);
  ncand[(size_t)u * ncand_stride(p) + seg] = top;
}

// grid = (ceil(groups / 128), units), block = 128 (the window's thread
// dimension), one thread per group of segments.  The
// tolerant chain over the segment survivors in order, eight points at a time:
// their b, then their sheared values, each batch of loads in flight together.
// The stack is the group's own candidate list (it never overtakes the read
// position); a pop below the shared-memory window reloads the new top and
// recomputes its sheared value.  Each test takes
// the largest error bound seen so far (the filter can only keep more).
__global__ void __launch_bounds__(128) hull_group_kernel(Prob p, const float2* __restrict__ curve,
                                                         int32_t* __restrict__ cand,
                                                         int32_t* __restrict__ ncand) {
  const int g = blockIdx.x * blockDim.x + threadIdx.x;
  const int u = blockIdx.y;
  if (g >= groups_of(p)) return;
  const int n = p.n;
  const float2* cu = curve + (size_t)u * n;
  int32_t* cl = cand + (size_t)u * n;
  int32_t* nc = ncand + (size_t)u * ncand_stride(p);
  const int s0 = g * kGroupSegs, s1 = min(p.hull_segs, s0 + kGroupSegs);
  const int b0 = p.b_min + s0 * kHullSeg;
  const int b1 = min(n, p.b_min + s1 * kHullSeg) - 1;
  const Shear sh = make_shear(cu, b0, b1);
  int32_t* st = cl + (size_t)s0 * kHullSeg;
  // entries [spill, top) also in a window of kHullWin slots per thread in
  // shared memory with their sheared values (one bank per lane), so that a
  // pop within it reads neither the list nor the curve again
  __shared__ int win_b[kHullWin][128];
  __shared__ float win_y[kHullWin][128];
  const int tid = threadIdx.x;
  int top = 0, spill = 0;
  int xa = 0, xb = 0;
  float ya = 0.f, yb = 0.f, dmax = 0.f;
  for (int s = s0; s < s1; ++s) {
    const int cnt = nc[s];
    const int32_t* src = cl + (size_t)s * kHullSeg;
    for (int i0 = 0; i0 < cnt; i0 += 8) {
      int bv[8];
      float yv[8], dv[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) bv[k] = (i0 + k < cnt) ? src[i0 + k] : 0;
#pragma unroll
      for (int k = 0; k < 8; ++k)
        if (i0 + k < cnt) sh.at(bv[k], yv[k], dv[k]);
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        if (i0 + k >= cnt) break;
        const int b = bv[k];
        dmax = fmaxf(dmax, dv[k]);
        while (top >= 2 && clearly_above(xa, ya, xb, yb, b, yv[k], dmax)) {
          --top;
          if (top < spill) spill = top;
          xb = xa;
          yb = ya;
          if (top >= 2) {
            const int e = top - 2;
            if (e >= spill) {
              xa = win_b[e & (kHullWin - 1)][tid];
              ya = win_y[e & (kHullWin - 1)][tid];
            } else {
              xa = st[e];
              float d;
              sh.at(xa, ya, d);
            }
          }
        }
        if (top - spill == kHullWin) ++spill;  // the oldest window entry stays in the list only
        win_b[top & (kHullWin - 1)][tid] = b;
        win_y[top & (kHullWin - 1)][tid] = yv[k];
        st[top++] = b;  // top <= the points read so far: never past the read position
        xa = xb;
        ya = yb;
        xb = b;
        yb = yv[k];
      }
    }
  }
  nc[p.hull_segs + g] = top;
}

// grid = B*L, block = 1024: bisection, repair, counts and offsets of one
// (sequence, layer).  Candidates are staged in shared memory when they fit;
// the repair keeps a 64-value window of each head's upcoming curve values in
// shared memory, refilled by the whole warp.
constexpr int kCandCap = 12288;  // staged candidates: 96 KB of values + 48 KB of b (dynamic smem)
constexpr int kScan = 2048;      // curve values per round of a block extension (16 KB)
constexpr float kFilterTol = 9.5367432e-7f;  // 2^-20, eight times the fp32 error bound of f

__global__ void __launch_bounds__(1024) bisect_repair_kernel(Prob p, const float2* __restrict__ curve,
                                                            const int32_t* __restrict__ cand,
                                                            const int32_t* __restrict__ ncand,
                                                            const unsigned long long* __restrict__ cmax,
                                                            int32_t* __restrict__ counts,
                                                            int64_t* __restrict__ offsets) {
  __shared__ int bsel[32];
  __shared__ int coff[33];
  __shared__ int htot[32];
  __shared__ int klo[32], khi[32];  // per head: staged index range that holds b_h(lambda)
  __shared__ int blo[32], bhi[32];  // the same range as values of b
  __shared__ DF wbest_f[32];  // per-warp argmin, combined per head
  __shared__ int wbest_b[32], wbest_k[32];
  __shared__ double lam_sh[2];
  __shared__ DF lam_node[7];  // a round's multipliers as double-float, for every warp
  __shared__ float2 win[32][64];
  __shared__ float2 scanbuf[kScan];
  extern __shared__ __align__(16) char dyn[];
  float2* cy = reinterpret_cast<float2*>(dyn);
  int32_t* cb_ = reinterpret_cast<int32_t*>(dyn + kCandCap * sizeof(float2));
  const int bl = blockIdx.x;
  const int H = p.H, n = p.n;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nwarps = blockDim.x >> 5;
  const int64_t B_real = p.B_real;
  const int groups = groups_of(p);
  const size_t stride = ncand_stride(p);

  const bool lagrangian = p.allocator == CERTKV_ALLOC_LAGRANGIAN;  // the hull filter ran only for it
  // Candidate offsets: warp h scans head h's group counts into gpre[h][g]
  // (exclusive, gpre[h][groups] = the head's total), kept in the repair's
  // scan buffer, which is free until the repair.
  int* gpre = reinterpret_cast<int*>(scanbuf);
  const int gstride = groups + 1;
  const bool gfit = H * gstride <= (int)(sizeof(scanbuf) / sizeof(int));
  if (lagrangian && gfit) {
    for (int h = warp; h < H; h += nwarps) {
      const int32_t* nc = ncand + (size_t)(bl * H + h) * stride + p.hull_segs;
      int carry = 0;
      for (int g0 = 0; g0 < groups; g0 += 32) {
        const int g = g0 + lane;
        const int v = g < groups ? nc[g] : 0;
        int x = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int y = __shfl_up_sync(kFull, x, o);
          if (lane >= o) x += y;
        }
        if (g < groups) gpre[h * gstride + g] = carry + x - v;
        carry += __shfl_sync(kFull, x, 31);
      }
      if (lane == 0) {
        gpre[h * gstride + groups] = carry;
        htot[h] = carry;
      }
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    double mx = 0.0;
    int acc = 0;
    for (int h = 0; h < H; ++h) {
      const double v = df_to_double(df_from_order_key(cmax[(size_t)bl * H + h]));
      mx = v > mx ? v : mx;
      coff[h] = acc;
      if (lagrangian) {
        if (gfit) {
          acc += htot[h];
        } else {
          const int32_t* nc = ncand + (size_t)(bl * H + h) * stride + p.hull_segs;
          for (int g = 0; g < groups; ++g) acc += nc[g];
        }
      }
    }
    coff[H] = acc;
    lam_sh[0] = 0.0;
    lam_sh[1] = __dadd_rn(__dmul_rn(2.0, mx), 1.0);
  }
  if (threadIdx.x < H) {
    blo[threadIdx.x] = 0;
    bhi[threadIdx.x] = INT_MAX;
  }
  __syncthreads();
  const bool staged = lagrangian && gfit && coff[H] <= kCandCap;
  if (staged) {
    // gather the group survivors of every head, in order: one thread per
    // candidate finds its head and group and loads b and c(b)
    for (int k = threadIdx.x; k < coff[H]; k += blockDim.x) {
      int h = 0;
      while (coff[h + 1] <= k) ++h;
      const int r = k - coff[h];
      const int* gp = gpre + h * gstride;
      int lo = 0, hi = groups - 1;  // the last group g with gp[g] <= r
      while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (gp[mid] <= r) lo = mid; else hi = mid - 1;
      }
      const int u = bl * H + h;
      const int b = cand[(size_t)u * n + (size_t)lo * kGroupSegs * kHullSeg + (r - gp[lo])];
      cb_[k] = b;
      cy[k] = curve[(size_t)u * n + b];
    }
  }
  if (threadIdx.x < H) {
    klo[threadIdx.x] = coff[threadIdx.x];
    khi[threadIdx.x] = coff[threadIdx.x + 1] - 1;
  }
  __syncthreads();

  // Head h is scanned by warps h * wph .. h * wph + wph - 1 (wph = warps per
  // head); the lexicographic (value, b) minimum does not depend on the split.
  // The smallest minimiser of c(b) + lambda b does not increase with lambda,
  // so for lambda inside the bracket (lo, hi) it lies between the minimisers
  // found at hi and at lo: each head scans only that range of its candidates
  // (blo..bhi, as staged indices klo..khi).
  // Each round evaluates the next `levels` bisection steps at once: the
  // 2^levels - 1 midpoints they can visit (node 0 the bracket's midpoint, the
  // children of node j the midpoints of its two half-brackets), computed from
  // the round's bracket by the same float64 operations as one step at a time;
  // warp 0 then follows the decisions down the tree.  Warps are shared out
  // over (node, head) pairs, wpp warps per pair.
  int max_levels = 1;
  while (max_levels < 3 && ((2 << max_levels) - 1) * H <= nwarps) ++max_levels;
  auto scan_heads = [&](int nodes) {
    const int pairs = nodes * H, wpp = nwarps / pairs;
    const int pi = warp / wpp, sub = warp - pi * wpp;
    if (pi < pairs) {
      const int node = pi / H, h = pi - node * H;
      const DF ld = lam_node[node];
      const int u = bl * H + h;
      DF bf{INFINITY, 0.f};
      int bb = INT_MAX, bk = -1;
      auto consider = [&](int b, float2 c, int k) {
        const DF f = df_add(DF{c.x, c.y}, df_mul_f(ld, (float)b));
        if (df_less(f, bf) || (f.hi == bf.hi && f.lo == bf.lo && b < bb)) {
          bf = f;
          bb = b;
          bk = k;
        }
      };
      if (staged) {
        // f = c(b) + lambda b >= 0; fp32 of the high parts is within 2^-23 f
        // of it, so only candidates whose fp32 lower bound reaches the
        // warp's least fp32 upper bound can be the warp's minimiser
        const int k0 = klo[h] + sub * 32 + lane, k1 = khi[h];
        float ub = INFINITY;
        for (int k = k0; k <= k1; k += wpp * 32)
          ub = fminf(ub, fmaf(ld.hi, (float)cb_[k], cy[k].x) * (1.0f + kFilterTol));
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) ub = fminf(ub, __shfl_xor_sync(kFull, ub, o));
        for (int k = k0; k <= k1; k += wpp * 32) {
          const int b = cb_[k];
          const float2 c = cy[k];
          if (fmaf(ld.hi, (float)b, c.x) * (1.0f - kFilterTol) <= ub) consider(b, c, k);
        }
      } else {
        const int32_t* nc = ncand + (size_t)u * stride + p.hull_segs;
        const int32_t* cl = cand + (size_t)u * n;
        const int b_lo = blo[h], b_hi = bhi[h];
        for (int g = 0; g < groups; ++g)
          for (int k = sub * 32 + lane; k < nc[g]; k += wpp * 32) {
            const int b = cl[(size_t)g * kGroupSegs * kHullSeg + k];
            if (b >= b_lo && b <= b_hi) consider(b, curve[(size_t)u * n + b], -1);
          }
      }
      const int own_b = bb, own_k = bk;
      warp_argmin_df(bf, bb);
      // b is unique within a head: the winner's index is held by the lane
      // whose own best was bb
      const unsigned holder = __ballot_sync(kFull, bb != INT_MAX && own_b == bb);
      const int kw = holder ? __shfl_sync(kFull, own_k, __ffs(holder) - 1) : -1;
      if (lane == 0) {
        wbest_f[warp] = bf;
        wbest_b[warp] = bb;
        wbest_k[warp] = kw;
      }
    }
  };
  // warp 0, lane = head, after a scan: the head's minimiser b at node `node`
  // (b_min when it has no candidate) and its staged index k (-2: no
  // candidate; -1: not staged)
  auto combine = [&](int nodes, int node, int& b_out, int& k_out) {
    const int wpp = nwarps / (nodes * H);
    DF bf{INFINITY, 0.f};
    int bb = INT_MAX, kk = -2;
    if (lane < H) {
      const int w0 = (node * H + lane) * wpp;
      for (int w = w0; w < w0 + wpp; ++w) {
        const DF f = wbest_f[w];
        const int b = wbest_b[w];
        if (df_less(f, bf) || (f.hi == bf.hi && f.lo == bf.lo && b < bb)) {
          bf = f;
          bb = b;
          kk = wbest_k[w];
        }
      }
    }
    b_out = (bb == INT_MAX) ? p.b_min : bb;
    k_out = (bb == INT_MAX) ? -2 : kk;
  };
  auto mid = [](double x, double y) { return __dmul_rn(__dadd_rn(x, y), 0.5); };

  // the bracket lives in warp 0 (every lane holds the same values)
  double lam_lo = lam_sh[0], lam_hi = lam_sh[1];
  double node_lam[7];
  for (int t = 0; lagrangian && t < p.T;) {
    const int levels = min(max_levels, p.T - t);
    const int nodes = (1 << levels) - 1;
    if (warp == 0) {
      node_lam[0] = mid(lam_lo, lam_hi);
      if (levels >= 2) {
        node_lam[1] = mid(lam_lo, node_lam[0]);
        node_lam[2] = mid(node_lam[0], lam_hi);
      }
      if (levels >= 3) {
        node_lam[3] = mid(lam_lo, node_lam[1]);
        node_lam[4] = mid(node_lam[1], node_lam[0]);
        node_lam[5] = mid(node_lam[0], node_lam[2]);
        node_lam[6] = mid(node_lam[2], lam_hi);
      }
      if (lane == 0)
        for (int j = 0; j < nodes; ++j) lam_node[j] = df_from_double(node_lam[j]);
    }
    __syncthreads();
    scan_heads(nodes);
    __syncthreads();
    if (warp == 0) {
      int j = 0;
      for (int l = 0; l < levels; ++l) {
        int bh, kh;
        combine(nodes, j, bh, kh);
        long long tot = lane < H ? bh : 0;
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) tot += __shfl_xor_sync(kFull, tot, o);
        const bool up = tot > B_real;
        if (up) lam_lo = node_lam[j]; else lam_hi = node_lam[j];
        // the new bracket end's minimisers bound the next scans
        if (lane < H && kh != -2) {
          if (up) {
            bhi[lane] = bh;
            if (staged) khi[lane] = kh;
          } else {
            blo[lane] = bh;
            if (staged) klo[lane] = kh;
          }
        }
        j = 2 * j + (up ? 2 : 1);
      }
    }
    t += levels;
    __syncthreads();
  }
  if (lagrangian) {  // the minimisers at lambda_hi
    if (threadIdx.x == 0) lam_node[0] = df_from_double(lam_hi);
    __syncthreads();
    scan_heads(1);
    __syncthreads();
    if (warp == 0) {
      int bh, kh;
      combine(1, 0, bh, kh);
      if (lane < H) bsel[lane] = bh;
    }
  } else if (threadIdx.x < H) {  // the allocator ablations' starting points
    const int h = threadIdx.x;
    bsel[h] = (p.allocator == CERTKV_ALLOC_UNIFORM)
                  ? (int)(B_real / H + (h < B_real % H ? 1 : 0))  // already sums to B_real
                  : p.b_min;  // greedy: the repair below adds the rest
  }
  __syncthreads();

  if (warp == 0) {
    const int h = lane;
    const bool live = h < H;
    int b = live ? bsel[h] : 0;
    const float2* cu = curve + (size_t)(bl * H + (live ? h : 0)) * n;
    int64_t tot = 0;
    for (int i = 0; i < H; ++i) tot += bsel[i];
    const DF kNone{INFINITY, 0.f}, kBad{FLT_MAX, 0.f};
    // surplus (not reachable from lambda_hi, kept for robustness): remove one
    while (tot > B_real) {
      DF mg = kNone;
      if (live && b > p.b_min) {
        const DF d = df_add(curve_df(cu, b - 1), df_neg(curve_df(cu, b)));
        mg = (d.hi == d.hi) ? d : kBad;
      }
      int who = lane;
      warp_argmin_df(mg, who);
      if (lane == who) --b;
      --tot;
    }
    // best-marginal repair: add one token at a time.  win[h][k] = c_h(base_h + k)
    DF cur = live ? curve_df(cu, b) : df_make(0.f);
    int base = b + 1;
    for (int hh = 0; hh < H; ++hh) {
      const int bh = __shfl_sync(kFull, b, hh);
      const float2* ch = curve + (size_t)(bl * H + hh) * n;
      for (int k = lane; k < 64; k += 32)
        win[hh][k] = (bh + 1 + k < n) ? ch[bh + 1 + k] : make_float2(0.f, 0.f);
    }
    __syncwarp();
    while (tot < B_real) {
      DF mg = kNone;
      if (live && b < n - 1) {
        const float2 w = win[h][b + 1 - base];
        const DF d = df_add(DF{w.x, w.y}, df_neg(cur));
        mg = (d.hi == d.hi) ? d : kBad;
      }
      int who = lane;
      warp_argmin_df(mg, who);
      const int nb = __shfl_sync(kFull, b, who) + 1;  // the winner's new count
      const int wbase = __shfl_sync(kFull, base, who);
      if (lane == who) {
        const float2 w = win[h][nb - base];
        cur = DF{w.x, w.y};
        b = nb;
      }
      ++tot;
      const float2* ch = curve + (size_t)(bl * H + who) * n;
      // The winner keeps every following marginal strictly below its leading
      // one: those would be picked next one at a time anyway (each is below
      // every other head's front), so the whole run is taken at once.
      int bw = nb;
      DF cw = shfl_df(cur, who);
      bool more = false;
      if (tot < B_real && bw < n - 1) {
        int nbase = wbase;
        if (bw + 1 - nbase >= 64) nbase = -1;  // next value not in the window
        DF d1 = kNone;
        if (nbase >= 0) {
          const float2 w = win[who][bw + 1 - nbase];
          d1 = df_add(DF{w.x, w.y}, df_neg(cw));
        } else {
          const float2 w = ch[bw + 1];
          d1 = df_add(DF{w.x, w.y}, df_neg(cw));
        }
        more = df_less(d1, mg);
      }
      // the run inside the winner's window first (no global loads): lane e
      // checks marginal c(bw+1+e) - c(bw+e) for window positions, 32 at a time
      if (more && bw + 1 - wbase < 64) {
        const int i0 = bw + 1 - wbase;  // window index of c(bw + 1); c(bw) sits at i0 - 1
        int run = 64 - i0;              // whole rest of the window, unless a check fails
        for (int e0 = 0; e0 < 64 - i0; e0 += 32) {
          const int e = e0 + lane, i = i0 + e;
          bool stop = false;
          if (i < 64) {
            const float2 pv = win[who][i - 1], nv = win[who][i];
            const DF d = df_add(DF{nv.x, nv.y}, df_neg(DF{pv.x, pv.y}));
            stop = (bw + e >= n - 1) || !df_less(d, mg);
          }
          const unsigned stops = __ballot_sync(kFull, stop);
          if (stops) {
            run = e0 + __ffs(stops) - 1;
            break;
          }
        }
        const int64_t room = B_real - tot;
        if ((int64_t)run > room) run = (int)room;
        const bool whole = (run == 64 - i0);
        if (run > 0) {
          const float2 last = win[who][i0 + run - 1];
          cw = DF{last.x, last.y};
        }
        bw += run;
        tot += run;
        more = whole && tot < B_real && bw < n - 1;
        if (more) {  // does the run go on past the window?
          const float2 w = ch[bw + 1];
          more = df_less(df_add(DF{w.x, w.y}, df_neg(cw)), mg);
        }
      }
      bool extended = false;
      while (more) {  // warp-cooperative scan, kScan values per round
        extended = true;
        __syncwarp();
        // every value of the round in flight at once (8-byte asynchronous copies)
        const uint32_t sbuf = (uint32_t)__cvta_generic_to_shared(scanbuf);
        for (int k = lane; k < kScan; k += 32) {
          if (bw + 1 + k < n)
            asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"(sbuf + (uint32_t)k * 8u),
                         "l"(ch + bw + 1 + k)
                         : "memory");
          else
            scanbuf[k] = make_float2(0.f, 0.f);
        }
        asm volatile("cp.async.commit_group;\n\tcp.async.wait_all;" ::: "memory");
        __syncwarp();
        // positions e = 32 i + lane in order, 32 per ballot, up to the first
        // marginal c(bw+e+1) - c(bw+e) that is not below the front
        int run = kScan;
        for (int i = 0; i < kScan / 32; ++i) {
          const int e = i * 32 + lane;
          const float2 pv = (e == 0) ? make_float2(cw.hi, cw.lo) : scanbuf[e - 1];
          const float2 nv = scanbuf[e];
          const DF d = df_add(DF{nv.x, nv.y}, df_neg(DF{pv.x, pv.y}));
          const bool stop = (bw + e >= n - 1) || !df_less(d, mg);
          const unsigned stops = __ballot_sync(kFull, stop);
          if (stops) {
            run = i * 32 + __ffs(stops) - 1;
            break;
          }
        }
        const int64_t room = B_real - tot;
        if ((int64_t)run > room) run = (int)room;
        if (run > 0) {
          const float2 last = scanbuf[run - 1];
          cw = DF{last.x, last.y};
        }
        bw += run;
        tot += run;
        more = (run == kScan) && tot < B_real && bw < n - 1;
      }
      if (lane == who && bw > nb) {
        b = bw;
        cur = cw;
      }
      if (bw + 1 - wbase >= 64 || extended) {  // refill the winner's window
        if (bw < n - 1) {
          __syncwarp();
          for (int k = lane; k < 64; k += 32)
            win[who][k] = (bw + 1 + k < n) ? ch[bw + 1 + k] : make_float2(0.f, 0.f);
          if (lane == who) base = bw + 1;
          __syncwarp();
        }
      }
    }
    // counts and offsets: segment = b_h real slots (+ 1 tail slot) (+ m cluster summaries)
    const int seg = live ? b + p.tail_slot + p.clusters : 0;
    int incl = seg;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(kFull, incl, o);
      if (lane >= o) incl += y;
    }
    if (live) {
      // the budget within [b_min, n - 1] and the segments within B_live
      CERTKV_IN_BOUNDS(b >= p.b_min && b <= p.n - 1, p.status);
      CERTKV_IN_BOUNDS(incl <= p.B_live, p.status);
      counts[(size_t)bl * H + h] = b;
      offsets[(size_t)bl * H + h] = p.slot_base + (int64_t)bl * p.B_live + (incl - seg);
    }
    if (bl == p.bl - 1 && lane == 0) offsets[(size_t)p.bl * H] = p.slot_base + (int64_t)p.bl * p.B_live;
  }
}

void launch_allocate(const Prob& p, const Layout& ly, char* ws, int32_t* counts,
                     int64_t* offsets, cudaStream_t st) {
  const float2* curve = reinterpret_cast<const float2*>(ws + ly.curve);
  int32_t* cand = reinterpret_cast<int32_t*>(ws + ly.cand);
  int32_t* ncand = reinterpret_cast<int32_t*>(ws + ly.ncand);
  const int groups = (p.hull_segs + kGroupSegs - 1) / kGroupSegs;
  if (p.allocator == CERTKV_ALLOC_LAGRANGIAN) {  // candidates for the bisection only
  {
    TraceScope ts_("hull_seg", st);
    hull_seg_kernel<<<dim3((p.hull_segs + 127) / 128, p.units), 128, 0, st>>>(p, curve, cand,
                                                                             ncand);
  }
  {
    TraceScope ts_("hull_group", st);
    hull_group_kernel<<<dim3((groups + 127) / 128, p.units), 128, 0, st>>>(p, curve, cand, ncand);
  }
  }
  {
    TraceScope ts_("bisect_repair", st);
    const size_t smem = kCandCap * (sizeof(float2) + sizeof(int32_t));
    static bool attr = false;
    if (!attr) {
      cudaFuncSetAttribute(bisect_repair_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)smem);
      attr = true;
    }
    bisect_repair_kernel<<<p.bl, 1024, smem, st>>>(
        p, curve, cand, ncand, reinterpret_cast<const unsigned long long*>(ws + ly.cmax), counts,
        offsets);
  }
}

}  // namespace certkv
