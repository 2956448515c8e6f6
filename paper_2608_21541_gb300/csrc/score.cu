// score.cu — a1/a2: observation-window scores on tensor cores.
//
// For every unit (sequence, layer, KV head) the R = G*w observation rows of
// the G query heads that read the KV head are scored against all n keys
// (§4: SnapKV's observation-window score; the implementation appendix keeps
// the scorer unchanged and normalises a_j = (s_j)_+ / sum_i (s_i)_+).  The
// softmax column sums need each row's log-sum-exp before any probability, so
// the keys are streamed twice:
//   pass 1  logits -> per-row online (max, sum) per key split
//   merge   splits -> LSE per row
//   pass 2  logits again -> p = exp(l - LSE) -> column sums over the rows
//   final   mean over rows, average pool, window protection, normalisation,
//           plus the radix-sort keys of the scores
// Logits are bf16 x bf16 -> fp32 products on the tensor cores
// (mma.sync.m16n8k16); K tiles are staged in swizzled shared memory by
// cp.async and read with ldmatrix.
#include "common.cuh"
#include "internal.cuh"

namespace certkv {

namespace {

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem, bool valid) {
  unsigned s = (unsigned)__cvta_generic_to_shared(smem);
  int bytes = valid ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(s), "l"(gmem), "r"(bytes));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
__device__ __forceinline__ void cp_async_wait_1() { asm volatile("cp.async.wait_group 1;\n" ::); }
__device__ __forceinline__ void cp_async_wait_0() { asm volatile("cp.async.wait_group 0;\n" ::); }

__device__ __forceinline__ void ldmatrix_x4(uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3,
                                            const void* smem) {
  unsigned s = (unsigned)__cvta_generic_to_shared(smem);
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(s));
}

__device__ __forceinline__ void mma_bf16(float (&c)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Byte offset of 16-byte chunk `c` of key row `r` in a swizzled 64 x 256 B tile.
__device__ __forceinline__ int tile_off(int r, int c) { return r * 256 + ((c ^ (r & 7)) << 4); }

// Stage keys [j0, j0 + 64) of one unit into `tile` (zero-filled past n).
__device__ __forceinline__ void stage_tile(char* tile, const __nv_bfloat16* Ku, int j0, int n,
                                           int tid, int nthreads) {
  for (int i = tid; i < kScoreTileKeys * 16; i += nthreads) {
    int r = i >> 4, c = i & 15;
    int j = j0 + r;
    bool ok = j < n;
    const char* src = reinterpret_cast<const char*>(Ku + (size_t)(ok ? j : 0) * kD) + c * 16;
    cp_async16(tile + tile_off(r, c), src, ok);
  }
}

}  // namespace

// Pass 1 (PASS2 = false) and pass 2 (PASS2 = true) over one key split and one
// row block of one unit.  grid = (key_splits, row_blocks, units).
template <bool PASS2>
__global__ void __launch_bounds__(512) score_pass_kernel(const __nv_bfloat16* __restrict__ K,
                                                         const __nv_bfloat16* __restrict__ Q,
                                                         Prob p, const float* __restrict__ lse2,
                                                         float2* __restrict__ lse_part,
                                                         float* __restrict__ s_part) {
  extern __shared__ __align__(128) char smem[];
  char* tiles = smem;                                   // 2 x 16 KB
  float* colsum = reinterpret_cast<float*>(smem + 2 * kScoreTileKeys * 256);  // [warps][64]

  const int split = blockIdx.x, rb = blockIdx.y, u = blockIdx.z;
  const int warps = blockDim.x >> 5;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gid = lane >> 2, tig = lane & 3;
  const int n = p.n, w = p.w, R = p.R;
  const int bl = u / p.H, h = u - bl * p.H;

  const __nv_bfloat16* Ku = K + (size_t)u * n * kD;
  const __nv_bfloat16* Qu = Q + ((size_t)bl * p.Hq + (size_t)h * p.G) * w * kD;

  // rows handled by this warp
  const int r_base = rb * warps * 16 + warp * 16;
  const int rA = r_base + gid, rB = rA + 8;
  const bool okA = rA < R, okB = rB < R;

  // A fragments of the warp's 16 rows over d = 128 (8 k-steps)
  uint32_t afrag[8][4];
  {
    const uint32_t* qa = reinterpret_cast<const uint32_t*>(Qu + (size_t)(okA ? rA : 0) * kD);
    const uint32_t* qb = reinterpret_cast<const uint32_t*>(Qu + (size_t)(okB ? rB : 0) * kD);
#pragma unroll
    for (int ks = 0; ks < 8; ++ks) {
      int c0 = ks * 8 + tig;  // 32-bit word index of k = 16 ks + 2 tig
      afrag[ks][0] = okA ? __ldg(qa + c0) : 0u;
      afrag[ks][1] = okB ? __ldg(qb + c0) : 0u;
      afrag[ks][2] = okA ? __ldg(qa + c0 + 4) : 0u;
      afrag[ks][3] = okB ? __ldg(qb + c0 + 4) : 0u;
    }
  }
  // visibility limits: row r (window position r % w) sees keys j <= n - w + r % w
  const int limA = okA ? (n - w + rA % w) : -1;
  const int limB = okB ? (n - w + rB % w) : -1;
  float lseA = 0.f, lseB = 0.f;
  if (PASS2) {
    lseA = okA ? lse2[(size_t)u * R + rA] : __int_as_float(0x7f800000);
    lseB = okB ? lse2[(size_t)u * R + rB] : __int_as_float(0x7f800000);
  }
  const float sl2 = p.scale_log2;

  float mA = -INFINITY, mB = -INFINITY, lA = 0.f, lB = 0.f;  // pass 1 running stats

  const int j_begin = split * kScoreKeysPerCta;
  const int j_end = min(n, j_begin + kScoreKeysPerCta);
  const int ntiles = (j_end - j_begin + kScoreTileKeys - 1) / kScoreTileKeys;

  stage_tile(tiles, Ku, j_begin, n, threadIdx.x, blockDim.x);
  cp_async_commit();

  for (int t = 0; t < ntiles; ++t) {
    const int j0 = j_begin + t * kScoreTileKeys;
    char* cur = tiles + (t & 1) * (kScoreTileKeys * 256);
    if (t + 1 < ntiles) {
      stage_tile(tiles + ((t + 1) & 1) * (kScoreTileKeys * 256), Ku, j0 + kScoreTileKeys, n,
                 threadIdx.x, blockDim.x);
      cp_async_commit();
      cp_async_wait_1();
    } else {
      cp_async_wait_0();
    }
    __syncthreads();

    float acc[8][4];
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) acc[nt][0] = acc[nt][1] = acc[nt][2] = acc[nt][3] = 0.f;
#pragma unroll
    for (int ks = 0; ks < 8; ++ks) {
#pragma unroll
      for (int np = 0; np < 4; ++np) {  // pairs of n8 tiles
        int key = np * 16 + ((lane >> 4) << 3) + (lane & 7);
        int chunk = ks * 2 + ((lane >> 3) & 1);
        uint32_t b0, b1, b2, b3;
        ldmatrix_x4(b0, b1, b2, b3, cur + tile_off(key, chunk));
        mma_bf16(acc[2 * np], afrag[ks], b0, b1);
        mma_bf16(acc[2 * np + 1], afrag[ks], b2, b3);
      }
    }

    // logits in the log2 domain with the causal / range mask
    const bool need_mask = (j0 + kScoreTileKeys - 1 > n - w) || (j0 + kScoreTileKeys > n);
    float xa[16], xb[16];
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        int j = j0 + nt * 8 + tig * 2 + e;
        float va = acc[nt][e] * sl2, vb = acc[nt][2 + e] * sl2;
        if (need_mask) {
          if (j > limA || j >= n) va = -INFINITY;
          if (j > limB || j >= n) vb = -INFINITY;
        }
        xa[nt * 2 + e] = va;
        xb[nt * 2 + e] = vb;
      }
    }

    if (!PASS2) {
      float tA = xa[0], tB = xb[0];
#pragma unroll
      for (int i = 1; i < 16; ++i) { tA = fmaxf(tA, xa[i]); tB = fmaxf(tB, xb[i]); }
      tA = fmaxf(tA, __shfl_xor_sync(kFull, tA, 1));
      tA = fmaxf(tA, __shfl_xor_sync(kFull, tA, 2));
      tB = fmaxf(tB, __shfl_xor_sync(kFull, tB, 1));
      tB = fmaxf(tB, __shfl_xor_sync(kFull, tB, 2));
      float nA = fmaxf(mA, tA), nB = fmaxf(mB, tB);
      if (nA > -INFINITY) {
        float s = 0.f;
#pragma unroll
        for (int i = 0; i < 16; ++i) s += exp2f(xa[i] - nA);
        lA = lA * exp2f(mA - nA) + s;
        mA = nA;
      }
      if (nB > -INFINITY) {
        float s = 0.f;
#pragma unroll
        for (int i = 0; i < 16; ++i) s += exp2f(xb[i] - nB);
        lB = lB * exp2f(mB - nB) + s;
        mB = nB;
      }
    } else {
      // column sums over this warp's 16 rows
      float cs[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) cs[i] = exp2f(xa[i] - lseA) + exp2f(xb[i] - lseB);
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        cs[i] += __shfl_xor_sync(kFull, cs[i], 4);
        cs[i] += __shfl_xor_sync(kFull, cs[i], 8);
        cs[i] += __shfl_xor_sync(kFull, cs[i], 16);
      }
      float* cw = colsum + (t & 1) * warps * 64 + warp * 64;
      if (gid == 0) {
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) {
          cw[nt * 8 + tig * 2] = cs[nt * 2];
          cw[nt * 8 + tig * 2 + 1] = cs[nt * 2 + 1];
        }
      }
    }
    __syncthreads();  // tile buffer and column sums are complete
    if (PASS2) {
      const float* cb = colsum + (t & 1) * warps * 64;
      for (int c = threadIdx.x; c < kScoreTileKeys; c += blockDim.x) {
        float s = 0.f;
        for (int wi = 0; wi < warps; ++wi) s += cb[wi * 64 + c];
        const int j = j0 + c;
        if (j < n) s_part[((size_t)u * p.row_blocks + rb) * n + j] = s;
      }
    }
  }

  if (!PASS2) {
    lA += __shfl_xor_sync(kFull, lA, 1);
    lA += __shfl_xor_sync(kFull, lA, 2);
    lB += __shfl_xor_sync(kFull, lB, 1);
    lB += __shfl_xor_sync(kFull, lB, 2);
    if (tig == 0) {
      if (okA) lse_part[((size_t)u * R + rA) * p.key_splits + split] = make_float2(mA, lA);
      if (okB) lse_part[((size_t)u * R + rB) * p.key_splits + split] = make_float2(mB, lB);
    }
  }
}

// LSE (log2 domain) of every observation row from the per-split partials.
__global__ void lse_merge_kernel(Prob p, const float2* __restrict__ part, float* __restrict__ lse2) {
  const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  const size_t total = (size_t)p.units * p.R;
  if (i >= total) return;
  const float2* pr = part + i * p.key_splits;
  float M = -INFINITY;
  for (int s = 0; s < p.key_splits; ++s) M = fmaxf(M, pr[s].x);
  float L = 0.f;
  for (int s = 0; s < p.key_splits; ++s)
    if (pr[s].x > -INFINITY) L += pr[s].y * exp2f(pr[s].x - M);
  lse2[i] = M + log2f(L);
}

// Finalize (a2), in two position-parallel kernels over slices of
// kFinSpan keys.  pool: s_j = (1/R) sum of the row blocks, average-pooled
// over non-window keys (zero padding, divided by the width; the slice loads a
// halo of pool/2 keys on each side), written to s_pool; per slice the max of
// the pooled scores and the double-float sum of the clipped ones.
// scale: the unit's max and total from its slices (window keys count as the
// max when protected), then a_j = (s_j)+ / total, the sort keys and indices.
__global__ void __launch_bounds__(256) score_pool_kernel(Prob p, const float* __restrict__ s_part,
                                                         float* __restrict__ s_pool,
                                                         float4* __restrict__ fin_part,
                                                         uint32_t* status) {
  extern __shared__ __align__(16) float s_win[];  // s over [lo, lo + window), lo <= j0 - half
  __shared__ float red_max[8];
  __shared__ DF red_sum[8];
  const int slice = blockIdx.x, u = blockIdx.y;
  const int n = p.n, nw = n - p.w, half = p.pool / 2;
  const int j0 = slice * kFinSpan, j1 = min(n, j0 + kFinSpan);
  const float invR = 1.0f / (float)p.R;
  const float invPool = 1.0f / (float)p.pool;
  // the row-block partials summed in row-block order
  const float* sb = s_part + (size_t)u * p.row_blocks * n;
  int lo = j0 - half, cnt = (j1 + half) - lo;
  if ((n & 3) == 0) {
    // rows of s_part 16-byte aligned: the window widened to whole float4s
    // ([lo, lo + cnt) rounded out to multiples of 4; j0 is one), each float4
    // either wholly inside [0, n) or wholly outside; two float4s per thread
    // and iteration with four row blocks unrolled, so that eight 16-byte loads
    // are in flight together
    lo = -(((half - j0) + 3) >> 2) * 4;  // floor to a multiple of 4 of j0 - half
    if (j0 - half >= 0) lo = (j0 - half) & ~3;
    const int hi = (j1 + half + 3) & ~3;
    const int nv = (hi - lo) >> 2;
    const float4* sb4 = reinterpret_cast<const float4*>(sb);
    const int rs4 = n >> 2;  // row stride in float4s
    for (int t0 = threadIdx.x; t0 < nv; t0 += 2 * blockDim.x) {
      float4 s[2] = {make_float4(0.f, 0.f, 0.f, 0.f), make_float4(0.f, 0.f, 0.f, 0.f)};
      int i4[2];
      bool in[2];
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int t = t0 + e * (int)blockDim.x;
        i4[e] = (lo >> 2) + t;
        in[e] = t < nv && i4[e] >= 0 && i4[e] < rs4;
      }
#pragma unroll 4
      for (int rb = 0; rb < p.row_blocks; ++rb) {
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const float4 x = in[e] ? sb4[(size_t)rb * rs4 + i4[e]] : make_float4(0.f, 0.f, 0.f, 0.f);
          s[e].x += x.x;
          s[e].y += x.y;
          s[e].z += x.z;
          s[e].w += x.w;
        }
      }
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int t = t0 + e * (int)blockDim.x;
        if (t < nv)
          reinterpret_cast<float4*>(s_win)[t] =
              make_float4(s[e].x * invR, s[e].y * invR, s[e].z * invR, s[e].w * invR);
      }
    }
    cnt = 0;  // the scalar loop below has nothing left to do
  }
  // four window positions per thread and iteration, so that their loads are
  // in flight together
  for (int t0 = threadIdx.x; t0 < cnt; t0 += 4 * blockDim.x) {
    float s[4] = {0.f, 0.f, 0.f, 0.f};
    for (int rb = 0; rb < p.row_blocks; ++rb) {
      float x[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int i = lo + t0 + e * (int)blockDim.x;
        x[e] = (t0 + e * (int)blockDim.x < cnt && i >= 0 && i < n) ? sb[(size_t)rb * n + i] : 0.f;
      }
#pragma unroll
      for (int e = 0; e < 4; ++e) s[e] += x[e];
    }
#pragma unroll
    for (int e = 0; e < 4; ++e)
      if (t0 + e * (int)blockDim.x < cnt) s_win[t0 + e * blockDim.x] = s[e] * invR;
  }
  __syncthreads();
  float* sp = s_pool + (size_t)u * n;
  float mx = -INFINITY;
  DF tot = df_make(0.f);
  bool bad = false;
  for (int j = j0 + threadIdx.x; j < j1; j += blockDim.x) {
    float v;
    if (j < nw) {
      if (p.pool == 1) {
        v = s_win[j - lo];
      } else if (p.pool == 5 && j >= 2 && j + 2 < nw) {  // the default width, window inside
        const float* w5 = s_win + (j - 2 - lo);          // the same additions, in order
        float acc = 0.f;
        acc += w5[0];
        acc += w5[1];
        acc += w5[2];
        acc += w5[3];
        acc += w5[4];
        v = acc * invPool;
      } else {
        float acc = 0.f;
        for (int i = j - half; i <= j + half; ++i)
          if (i >= 0 && i < nw) acc += s_win[i - lo];
        v = acc * invPool;
      }
      mx = fmaxf(mx, v);
    } else {
      if (p.protect) continue;  // the unit's max, known only after every slice
      v = s_win[j - lo];
    }
    sp[j] = v;
    if (!(fabsf(v) <= 3.0e38f)) bad = true;  // NaN or Inf
    tot = df_add_f(tot, v > 0.f ? v : 0.f);
  }
  if (bad) raise_status(status, 1u);
  mx = warp_max(mx);
  tot = warp_sum_df(tot);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) {
    red_max[warp] = mx;
    red_sum[warp] = tot;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float m = -INFINITY;
    DF t = df_make(0.f);
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) {
      m = fmaxf(m, red_max[w]);
      t = df_add(t, red_sum[w]);
    }
    fin_part[(size_t)u * gridDim.x + slice] = make_float4(m, t.hi, t.lo, 0.f);
  }
}

__global__ void __launch_bounds__(256) score_scale_kernel(Prob p, const float* __restrict__ s_pool,
                                                          const float4* __restrict__ fin_part,
                                                          float* __restrict__ a_out,
                                                          uint32_t* __restrict__ keys,
                                                          uint32_t* status) {
  const int slice = blockIdx.x, u = blockIdx.y;
  const int n = p.n, nw = n - p.w;
  float smax = -INFINITY;
  DF tot = df_make(0.f);
  for (int k = 0; k < (int)gridDim.x; ++k) {  // every thread, same order
    const float4 f = fin_part[(size_t)u * gridDim.x + k];
    smax = fmaxf(smax, f.x);
    tot = df_add(tot, DF{f.y, f.z});
  }
  if (p.protect) {
    if (!(fabsf(smax) <= 3.0e38f) && slice == 0 && threadIdx.x == 0) raise_status(status, 1u);
    tot = df_add(tot, two_prod(smax > 0.f ? smax : 0.f, (float)p.w));
  }
  const float total = tot.hi;
  const float* sp = s_pool + (size_t)u * n;
  float* au = a_out + (size_t)u * n;
  const int j0 = slice * kFinSpan, j1 = min(n, j0 + kFinSpan);
  for (int jb = j0 + threadIdx.x; jb < j1; jb += 4 * blockDim.x) {
    float v[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {  // four loads in flight
      const int j = jb + e * (int)blockDim.x;
      v[e] = j < j1 ? ((j >= nw && p.protect) ? smax : sp[j]) : 0.f;
    }
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int j = jb + e * (int)blockDim.x;
      if (j >= j1) break;
      const float x = v[e] > 0.f ? v[e] : 0.f;
      const float a = __fdiv_rn(x, total);
      au[j] = a;
      if (keys) keys[(size_t)u * n + j] = score_key(a);
    }
  }
}

void launch_score(const Prob& p, const Layout& ly, char* ws, const void* K, const void* Q,
                  float* a_out, cudaStream_t st) {
  const __nv_bfloat16* Kb = reinterpret_cast<const __nv_bfloat16*>(K);
  const __nv_bfloat16* Qb = reinterpret_cast<const __nv_bfloat16*>(Q);
  float2* lse_part = reinterpret_cast<float2*>(ws + ly.lse_part);
  float* lse2 = reinterpret_cast<float*>(ws + ly.lse);
  float* s_part = reinterpret_cast<float*>(ws + ly.s_part);
  const int threads = p.score_warps * 32;
  const size_t smem = 2 * kScoreTileKeys * 256 + 2 * p.score_warps * 64 * sizeof(float);
  static bool attr_set = false;
  if (!attr_set) {
    cudaFuncSetAttribute(score_pass_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, 96 * 1024);
    cudaFuncSetAttribute(score_pass_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, 96 * 1024);
    attr_set = true;
  }
  bool done = false;
  if (p.score_tc)
    done = launch_score_tc(p, K, Q, lse_part, lse2, s_part,
                           reinterpret_cast<uint32_t*>(ws + ly.status), st);
  dim3 grid(p.key_splits, p.row_blocks, p.units);
  if (!done) {
  {
    TraceScope ts_("score_pass1", st);
    score_pass_kernel<false><<<grid, threads, smem, st>>>(Kb, Qb, p, nullptr, lse_part, nullptr);
  }
  const size_t rows = (size_t)p.units * p.R;
  {
    TraceScope ts_("lse_merge", st);
    lse_merge_kernel<<<(unsigned)((rows + 255) / 256), 256, 0, st>>>(p, lse_part, lse2);
  }
  {
    TraceScope ts_("score_pass2", st);
    score_pass_kernel<true><<<grid, threads, smem, st>>>(Kb, Qb, p, lse2, nullptr, s_part);
  }
  }
  const dim3 fgrid((p.n + kFinSpan - 1) / kFinSpan, p.units);
  float* s_pool = reinterpret_cast<float*>(ws + ly.s_tmp);
  float4* fin_part = reinterpret_cast<float4*>(ws + ly.fin_part);
  uint32_t* status = reinterpret_cast<uint32_t*>(ws + ly.status);
  {
    TraceScope ts_("score_pool", st);
    // the window [j0 - half, j1 + half), widened by up to 3 keys on each side
    const size_t fsmem = (size_t)(kFinSpan + p.pool + 8) * sizeof(float);
    score_pool_kernel<<<fgrid, 256, fsmem, st>>>(p, s_part, s_pool, fin_part, status);
  }
  {
    TraceScope ts_("score_scale", st);
    score_scale_kernel<<<fgrid, 256, 0, st>>>(
        p, s_pool, fin_part, a_out, reinterpret_cast<uint32_t*>(ws + ly.keys0), status);
  }
}

}  // namespace certkv
