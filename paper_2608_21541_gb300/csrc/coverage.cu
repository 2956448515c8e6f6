// coverage.cu — coverage profile of realized query rows (an evaluation
// instrument, §3 "count sparsity does not imply coverage sparsity" and the
// appendix's gap-profile instrument, which recomputes the row logits in fp32).
//
// For each query row (one per decode query head) over the n keys of its KV
// head: the logits z_j = scale <q, k_j> in fp32, their order pi (descending,
// ties by lower index), the ranked gap profile G(j) = z_(1) - z_(j), the
// coverage budgets K_eta = min{k : sum_{j<=k} A_(j) >= 1 - eta}, the
// relative-weight counts #{j : A_j > eps A_(1)} and the calibrated counts
// #{j : A_j > eps}.  The order is the segmented radix sort of the compression
// pass run over rows instead of units; the ranked softmax mass is accumulated
// in float64 in one fixed order, so every K_eta is decided on one sequence of
// partial sums.
#include "../../include/certkv.h"
#include "common.cuh"
#include "internal.cuh"
#include "headlogits.cuh"

namespace certkv {

namespace {

constexpr int kCovSplits = 32;

// order-preserving map of a float to uint32 (ascending), then complemented so
// that an ascending sort of the key is a descending order of the logit
__device__ __forceinline__ uint32_t desc_key(float z) {
  const uint32_t b = __float_as_uint(z + 0.0f);  // -0 -> +0
  const uint32_t ord = (b & 0x80000000u) ? ~b : (b | 0x80000000u);
  return ~ord;
}
__device__ __forceinline__ float key_logit(uint32_t key) {
  const uint32_t ord = ~key;
  return __uint_as_float((ord & 0x80000000u) ? (ord & 0x7fffffffu) : ~ord);
}

// grid = (units, kCovSplits), block = 128: each warp takes 32-token tiles; the
// G query heads of the unit's group are dotted with each K row by 2G lanes
// (coalesced), then lane = token writes its keys, [u * G + g][n] (the sort's
// first pass takes the token indices as its values).
template <int G>
__global__ void __launch_bounds__(128) coverage_logits_kernel(
    Prob p, const __nv_bfloat16* __restrict__ q, const __nv_bfloat16* __restrict__ K,
    float scale, uint32_t* __restrict__ keys) {
  __shared__ float xs[4][32 * G];
  const int u = blockIdx.x, split = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int bl = u / p.H, h = u - bl * p.H;
  const int n = p.n;
  float2 qr[DecGeo<G>::NPAIR][G];
  load_query_slice<G>(q + ((size_t)bl * p.Hq + (size_t)h * G) * kD, lane, qr);
  const __nv_bfloat16* Ku = K + (size_t)u * n * kD;
  const int ntiles = (n + 31) / 32;
  for (int t = split * 4 + warp; t < ntiles; t += kCovSplits * 4) {
    tile_head_logits<G>(Ku + (size_t)t * 32 * kD, min(32, n - t * 32), qr, lane, xs[warp]);
    const int j = t * 32 + lane;
    if (j < n) {
#pragma unroll
      for (int g = 0; g < G; ++g)
        keys[((size_t)u * G + g) * n + j] = desc_key(xs[warp][lane * G + g] * scale);
    }
    __syncwarp();  // xs is rewritten by the next tile
  }
}

struct CovThresholds {
  int n_eta, n_rel, n_abs;
  double eta[CERTKV_COVERAGE_MAX_THRESHOLDS];
  float rel_log[CERTKV_COVERAGE_MAX_THRESHOLDS];  // log eps, fp32
  double abs_log[CERTKV_COVERAGE_MAX_THRESHOLDS];  // log eps, fp64
};

// one 32-rank step of a warp's running sum of the ranked weights: *incl = the
// inclusive partial sum at this lane's rank; returns the sum after the step
// (the same fp64 operations in every call, so a re-scan reproduces each
// partial sum bit for bit)
__device__ __forceinline__ double ranked_mass_step(double e, int lane, double carry,
                                                   double* incl) {
  double s = e;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const double y = __shfl_up_sync(kFull, s, o);
    if (lane >= o) s += y;
  }
  *incl = carry + s;
  return carry + __shfl_sync(kFull, s, 31);
}

// first rank r (0-based) in [lo, hi) whose predicate z_(r) - z1 > thr fails,
// over the row's sorted keys (the predicate is monotone along the ranks)
__device__ int first_fail(const uint32_t* __restrict__ kr, int lo, int hi, float z1, float thr) {
  while (lo < hi) {
    const int mid = (lo + hi) >> 1;
    if (key_logit(kr[mid]) - z1 > thr) lo = mid + 1;
    else hi = mid;
  }
  return lo;
}

// grid = rows, block = 1024 (32 warps, warp w owns ranks [w seg, (w+1) seg)).
__global__ void __launch_bounds__(1024) coverage_profile_kernel(
    int n, CovThresholds th, const uint32_t* __restrict__ keys, const int32_t* __restrict__ vals,
    int32_t* __restrict__ K_eta, int32_t* __restrict__ rel, int32_t* __restrict__ abs_,
    float* __restrict__ top, int32_t* __restrict__ order, float* __restrict__ gap) {
  __shared__ double wtot[32], wpre[32];
  __shared__ double Zs;
  const int row = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t* kr = keys + (size_t)row * n;
  const int seg = ((n + 1023) / 1024) * 32;
  const int r0 = min(n, warp * seg), r1 = min(n, r0 + seg);
  const float z1 = key_logit(kr[0]);
  double carry = 0.0, incl;
  for (int b = r0; b < r1; b += 32) {
    const int r = b + lane;
    float e = 0.f;
    if (r < r1) {
      const float z = key_logit(kr[r]);
      e = expf(z - z1);
      if (gap) gap[(size_t)row * n + r] = z1 - z;
      if (order) order[(size_t)row * n + r] = vals[(size_t)row * n + r];
    }
    carry = ranked_mass_step((double)e, lane, carry, &incl);
  }
  if (lane == 0) wtot[warp] = carry;
  __syncthreads();
  if (threadIdx.x == 0) {
    double acc = 0.0;
    for (int w = 0; w < 32; ++w) {
      wpre[w] = acc;
      acc += wtot[w];
    }
    Zs = acc;
  }
  __syncthreads();
  const double Z = Zs;
  // K_eta: the warp whose ranks contain the first crossing re-scans them
  for (int e = 0; e < th.n_eta; ++e) {
    const double T = (1.0 - th.eta[e]) * Z;
    const double pre = wpre[warp];
    const bool last = (warp == 31);
    const double end = last ? Z : wpre[warp + 1];
    if (r0 < r1 && pre < T && end >= T) {
      double c = 0.0;
      int found = -1;
      for (int b = r0; b < r1 && found < 0; b += 32) {
        const int r = b + lane;
        const float ev = r < r1 ? expf(key_logit(kr[r]) - z1) : 0.f;
        c = ranked_mass_step((double)ev, lane, c, &incl);
        const unsigned hit = __ballot_sync(kFull, r < r1 && pre + incl >= T);
        if (hit) found = b + __ffs(hit) - 1;
      }
      if (lane == 0) K_eta[(size_t)row * th.n_eta + e] = (found >= 0 ? found : r1 - 1) + 1;
    }
  }
  // counts: A_j > eps A_(1)  <=>  z_j - z_(1) > log eps;  A_j > eps  <=>
  // z_j - z_(1) > log eps + log Z
  const double logZ = log(Z);
  if (threadIdx.x < th.n_rel)
    rel[(size_t)row * th.n_rel + threadIdx.x] = first_fail(kr, 0, n, z1, th.rel_log[threadIdx.x]);
  if (threadIdx.x >= 32 && threadIdx.x < 32 + th.n_abs) {
    const int e = threadIdx.x - 32;
    abs_[(size_t)row * th.n_abs + e] = first_fail(kr, 0, n, z1, (float)(th.abs_log[e] + logZ));
  }
  if (threadIdx.x == 0) {
    top[(size_t)row * 2 + 0] = z1;
    top[(size_t)row * 2 + 1] = (float)((double)z1 + logZ);
  }
}

struct CovLayout {
  size_t keys0, keys1, vals0, vals1, hist, total;
};
CovLayout cov_layout(const Prob& p) {
  const size_t rows = (size_t)p.units * p.G, n = (size_t)p.n;
  auto a = [](size_t x) { return (x + 255) / 256 * 256; };
  CovLayout ly;
  ly.keys0 = 0;
  ly.keys1 = ly.keys0 + a(rows * n * 4);
  ly.vals0 = ly.keys1 + a(rows * n * 4);
  ly.vals1 = ly.vals0 + a(rows * n * 4);
  ly.hist = ly.vals1 + a(rows * n * 4);
  ly.total = ly.hist + a(rows * 256 * (size_t)p.sort_tiles * 4);
  return ly;
}

}  // namespace

size_t coverage_workspace(const Prob& p) { return cov_layout(p).total; }

void launch_coverage(const Prob& p, const void* q, const void* K, float scale,
                     const double* eta, int n_eta, const double* rel_eps, int n_rel,
                     const double* abs_eps, int n_abs, int32_t* K_eta, int32_t* rel,
                     int32_t* abs_, float* top, int32_t* order, float* gap, char* ws,
                     cudaStream_t st) {
  const CovLayout cl = cov_layout(p);
  uint32_t* k0 = reinterpret_cast<uint32_t*>(ws + cl.keys0);
  int32_t* v0 = reinterpret_cast<int32_t*>(ws + cl.vals0);
  const __nv_bfloat16* qb = reinterpret_cast<const __nv_bfloat16*>(q);
  const __nv_bfloat16* kb = reinterpret_cast<const __nv_bfloat16*>(K);
  const dim3 grid(p.units, kCovSplits);
  {
    TraceScope ts_("coverage_logits", st);
#define CERTKV_COV_LOGITS(GG) \
  coverage_logits_kernel<GG><<<grid, 128, 0, st>>>(p, qb, kb, scale, k0)
    switch (p.G) {
      case 1: CERTKV_COV_LOGITS(1); break;
      case 2: CERTKV_COV_LOGITS(2); break;
      case 4: CERTKV_COV_LOGITS(4); break;
      case 8: CERTKV_COV_LOGITS(8); break;
      case 16: CERTKV_COV_LOGITS(16); break;
      default: return;
    }
#undef CERTKV_COV_LOGITS
  }
  // the compression pass's segmented radix sort, one segment per row
  Prob ps = p;
  ps.units = p.units * p.G;
  Layout ly{};
  ly.keys0 = cl.keys0;
  ly.keys1 = cl.keys1;
  ly.vals0 = cl.vals0;
  ly.vals1 = cl.vals1;
  ly.hist = cl.hist;
  launch_sort(ps, ly, ws, nullptr, st);
  CovThresholds th{};
  th.n_eta = n_eta;
  th.n_rel = n_rel;
  th.n_abs = n_abs;
  for (int e = 0; e < n_eta; ++e) th.eta[e] = eta[e];
  for (int e = 0; e < n_rel; ++e) th.rel_log[e] = (float)log(rel_eps[e]);
  for (int e = 0; e < n_abs; ++e) th.abs_log[e] = log(abs_eps[e]);
  {
    TraceScope ts_("coverage_profile", st);
    coverage_profile_kernel<<<ps.units, 1024, 0, st>>>(p.n, th, k0, v0, K_eta, rel, abs_, top,
                                                       order, gap);
  }
}

}  // namespace certkv
