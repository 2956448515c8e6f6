// sort.cu — a3: per-unit stable order of the scores (descending, ties by
// lower index; Algorithm 1 "sort by s_h descending").
//
// Segmented LSD radix sort over all units at once: 32-bit keys
// (~bits(a), ascending = a descending), 8-bit digits, 4 passes.  Each pass is
// histogram -> per-unit exclusive scan in (digit, tile) order -> stable
// scatter.  The input of pass 0 is in index order and its values are the
// indices themselves (not read), so stability yields the lower-index
// tie-break.
#include "common.cuh"
#include "internal.cuh"

namespace certkv {

namespace {
constexpr int kWarps = kSortThreads / 32;
constexpr int kPerLane = kSortTile / kSortThreads;  // 8 keys per lane, striped per warp

// Lanes of the warp whose 8-bit digit equals this lane's, among the lanes with
// `ok` set (0 for a lane without it): one ballot per digit bit.
__device__ __forceinline__ uint32_t same_digit_lanes(uint32_t dgt, bool ok) {
  uint32_t peers = __ballot_sync(kFull, ok);
#pragma unroll
  for (int b = 0; b < 8; ++b) {
    const uint32_t bit = (dgt >> b) & 1u;
    const uint32_t bal = __ballot_sync(kFull, bit != 0u);
    peers &= bit ? bal : ~bal;
  }
  return ok ? peers : 0u;
}
}  // namespace

// grid = (tiles, units): per-tile digit histogram, stored [u][digit][tile].
__global__ void __launch_bounds__(kSortThreads) radix_hist_kernel(const uint32_t* __restrict__ keys,
                                                                  int n, int tiles, int shift,
                                                                  uint32_t* __restrict__ hist) {
  __shared__ uint32_t cnt[256];
  const int tile = blockIdx.x, u = blockIdx.y;
  cnt[threadIdx.x] = 0;
  __syncthreads();
  const uint32_t* ku = keys + (size_t)u * n;
  const int base = tile * kSortTile;
  uint32_t k[kPerLane];
#pragma unroll
  for (int e = 0; e < kPerLane; ++e) {  // all loads in flight before the counting
    const int j = base + e * kSortThreads + threadIdx.x;
    k[e] = j < n ? ku[j] : 0u;
  }
#pragma unroll
  for (int e = 0; e < kPerLane; ++e)
    if (base + e * kSortThreads + (int)threadIdx.x < n) atomicAdd(&cnt[(k[e] >> shift) & 255u], 1u);
  __syncthreads();
  hist[((size_t)u * 256 + threadIdx.x) * tiles + tile] = cnt[threadIdx.x];
}

// grid = units, block = 1024: exclusive scan of the unit's 256 * tiles
// counters, 16 consecutive counters per thread per round (four 16-byte loads;
// 256 * tiles is a multiple of 16).
constexpr int kScanPer = 16;
__global__ void __launch_bounds__(1024) radix_scan_kernel(uint32_t* __restrict__ hist, int tiles) {
  __shared__ uint32_t warp_tot[32];
  uint32_t* h = hist + (size_t)blockIdx.x * 256 * tiles;
  const int total = 256 * tiles;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t carry = 0;
  for (int base = 0; base < total; base += kScanPer * 1024) {
    const int i0 = base + kScanPer * (int)threadIdx.x;
    const bool mine = i0 < total;
    uint4 v[kScanPer / 4];
#pragma unroll
    for (int e = 0; e < kScanPer / 4; ++e)
      v[e] = mine ? reinterpret_cast<const uint4*>(h + i0)[e] : make_uint4(0u, 0u, 0u, 0u);
    uint32_t s = 0;
#pragma unroll
    for (int e = 0; e < kScanPer / 4; ++e) s += v[e].x + v[e].y + v[e].z + v[e].w;
    uint32_t x = s;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(kFull, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) warp_tot[warp] = x;
    __syncthreads();
    if (warp == 0) {
      uint32_t t = warp_tot[lane];
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(kFull, t, o);
        if (lane >= o) t += y;
      }
      warp_tot[lane] = t;  // inclusive
    }
    __syncthreads();
    uint32_t run = carry + (warp > 0 ? warp_tot[warp - 1] : 0u) + x - s;
    if (mine) {
#pragma unroll
      for (int e = 0; e < kScanPer / 4; ++e) {
        uint4 o;
        o.x = run;
        run += v[e].x;
        o.y = run;
        run += v[e].y;
        o.z = run;
        run += v[e].z;
        o.w = run;
        run += v[e].w;
        reinterpret_cast<uint4*>(h + i0)[e] = o;
      }
    }
    carry += warp_tot[31];
    __syncthreads();  // warp_tot is rewritten by the next round
  }
}

// grid = (tiles, units): stable scatter of one tile.  The tile is first
// ordered by digit in shared memory (stable ranks from per-warp counts), then
// written out so that consecutive threads store consecutive positions of a
// digit's run.  kFirst: the values are the key indices (vin is not read).
template <bool kFirst>  // at most 48 registers: five CTAs per SM to hide the load latency
__global__ void __launch_bounds__(kSortThreads, 5) radix_scatter_kernel(
    const uint32_t* __restrict__ kin, const int32_t* __restrict__ vin, uint32_t* __restrict__ kout,
    int32_t* __restrict__ vout, int n, int tiles, int shift, const uint32_t* __restrict__ hist,
    uint32_t* status) {
  __shared__ uint32_t wcnt[kWarps][256];
  __shared__ uint32_t gbase[256];
  __shared__ uint32_t tstart[256];
  __shared__ uint32_t wsum[kWarps];
  __shared__ uint32_t skey[kSortTile];
  __shared__ int32_t sval[kSortTile];
  const int tile = blockIdx.x, u = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // the tile's keys and values, its digit offsets and the counter reset all
  // in flight together
  const uint32_t* ku = kin + (size_t)u * n;
  const int32_t* vu = vin + (size_t)u * n;
  const int wbase = tile * kSortTile + warp * (kSortTile / kWarps);
  uint32_t key[kPerLane];
  int32_t val[kPerLane];
#pragma unroll
  for (int i = 0; i < kPerLane; ++i) {
    int j = wbase + i * 32 + lane;
    bool ok = j < n;
    key[i] = ok ? ku[j] : 0u;
    val[i] = kFirst ? j : (ok ? vu[j] : 0);
  }
  gbase[threadIdx.x] = hist[((size_t)u * 256 + threadIdx.x) * tiles + tile];
  for (int i = threadIdx.x; i < kWarps * 256; i += kSortThreads) (&wcnt[0][0])[i] = 0;
  __syncthreads();
  const uint32_t lt = (1u << lane) - 1u;
  // 1. per-warp digit counts; peers[i] = lanes holding the same digit
  uint32_t peers[kPerLane];
#pragma unroll
  for (int i = 0; i < kPerLane; ++i) {
    const int j = wbase + i * 32 + lane;
    const bool ok = j < n;
    const uint32_t dgt = (key[i] >> shift) & 255u;
    peers[i] = same_digit_lanes(dgt, ok);
    if (ok && (peers[i] & lt) == 0u) wcnt[warp][dgt] += __popc(peers[i]);
    __syncwarp();
  }
  __syncthreads();
  // 2. per digit: exclusive scan across warps, then over digits (tile start)
  {
    const int d = threadIdx.x;
    uint32_t run = 0;
#pragma unroll
    for (int wi = 0; wi < kWarps; ++wi) {
      uint32_t t = wcnt[wi][d];
      wcnt[wi][d] = run;
      run += t;
    }
    uint32_t x = run;  // inclusive scan over digits: warp level, then warp totals
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      uint32_t y = __shfl_up_sync(kFull, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) wsum[warp] = x;
    __syncthreads();
    uint32_t before = 0;
#pragma unroll
    for (int wi = 0; wi < kWarps; ++wi)
      if (wi < warp) before += wsum[wi];
    const uint32_t start = before + x - run;
    tstart[d] = start;
#pragma unroll
    for (int wi = 0; wi < kWarps; ++wi) wcnt[wi][d] += start;
  }
  __syncthreads();
  // 3. stable tile-local ranks -> shared memory, in digit order
#pragma unroll
  for (int i = 0; i < kPerLane; ++i) {
    const int j = wbase + i * 32 + lane;
    const bool ok = j < n;
    const uint32_t dgt = (key[i] >> shift) & 255u;
    uint32_t before = 0;
    if (ok) before = wcnt[warp][dgt];
    __syncwarp();
    if (ok) {
      const uint32_t pos = before + __popc(peers[i] & lt);
      skey[pos] = key[i];
      sval[pos] = val[i];
      if ((peers[i] & lt) == 0u) wcnt[warp][dgt] = before + __popc(peers[i]);
    }
    __syncwarp();
  }
  __syncthreads();
  // 4. coalesced write-out of the digit runs
  uint32_t* ko = kout + (size_t)u * n;
  int32_t* vo = vout + (size_t)u * n;
  const int count = min(kSortTile, n - tile * kSortTile);
  for (int i = threadIdx.x; i < count; i += kSortThreads) {
    const uint32_t k = skey[i];
    const uint32_t d = (k >> shift) & 255u;
    const uint32_t pos = gbase[d] + (uint32_t)i - tstart[d];
    if (!CERTKV_IN_BOUNDS(pos < (uint32_t)n, status)) continue;
    ko[pos] = k;
    vo[pos] = sval[i];
  }
}

void launch_sort(const Prob& p, const Layout& ly, char* ws, const float* /*a*/, cudaStream_t st) {
  uint32_t* k0 = reinterpret_cast<uint32_t*>(ws + ly.keys0);
  uint32_t* k1 = reinterpret_cast<uint32_t*>(ws + ly.keys1);
  int32_t* v0 = reinterpret_cast<int32_t*>(ws + ly.vals0);
  int32_t* v1 = reinterpret_cast<int32_t*>(ws + ly.vals1);
  uint32_t* hist = reinterpret_cast<uint32_t*>(ws + ly.hist);
  dim3 grid(p.sort_tiles, p.units);
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = pass * 8;
    const uint32_t* kin = (pass & 1) ? k1 : k0;
    const int32_t* vin = (pass & 1) ? v1 : v0;
    uint32_t* kout = (pass & 1) ? k0 : k1;
    int32_t* vout = (pass & 1) ? v0 : v1;
    {
      TraceScope ts_("sort_hist", st);
      radix_hist_kernel<<<grid, kSortThreads, 0, st>>>(kin, p.n, p.sort_tiles, shift, hist);
    }
    {
      TraceScope ts_("sort_scan", st);
      radix_scan_kernel<<<p.units, 1024, 0, st>>>(hist, p.sort_tiles);
    }
    {
      TraceScope ts_("sort_scatter", st);
      if (pass == 0)
        radix_scatter_kernel<true><<<grid, kSortThreads, 0, st>>>(kin, vin, kout, vout, p.n,
                                                                  p.sort_tiles, shift, hist,
                                                                  p.status);
      else
        radix_scatter_kernel<false><<<grid, kSortThreads, 0, st>>>(kin, vin, kout, vout, p.n,
                                                                   p.sort_tiles, shift, hist,
                                                                   p.status);
    }
  }
  // after 4 passes the sorted keys / permutation are back in keys0 / vals0
}

}  // namespace certkv
