// internal.cuh — problem description and kernel launchers shared by the
// translation units of the CertKV library.  Not part of the public ABI.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "../../include/certkv.h"

namespace certkv {

// One compress/decode call, after host-side validation.
struct Prob {
  int B, L, Hq, H, n, d, w, G, R;  // R = G * w observation rows per KV head
  int units;                       // B * L * H
  int bl;                          // B * L
  float scale;                     // softmax scale
  float scale_log2;                // scale * log2(e)
  int pool, protect;
  int alpha_num, alpha_den, T, statistic, tail_slot;
  int allocator;  // CERTKV_ALLOC_*
  int clusters;   // m cluster summaries per head over the evicted tail (0 = none)
  int64_t B_live, B_real;
  int b_min;
  int64_t slot_base;  // packed slot of this problem's first (sequence, layer): offsets are global
  int64_t capacity;   // packed-cache slots the caller gave (0: not known to the kernels)
  uint32_t* status;   // the workspace status word (bounds reports of debug builds; may be null)
  // derived launch geometry
  int score_tc;     // 1: tcgen05 scorer (R in {128, 256}); 0: mma.sync scorer
  int score_warps;  // warps per score CTA (16 rows each)
  int row_blocks;   // ceil(R / (16 * score_warps))
  int key_splits;   // ceil(n / kScoreKeysPerCta)
  int sort_tiles;   // ceil(n / kSortTile)
  int chunks;       // ceil(n / kChunk)
  int hull_segs;    // ceil((n - b_min) / kHullSeg)
};

constexpr int kScoreKeysPerCta = 1024;   // keys per CTA of the mma.sync scorer
constexpr int kKeysPerItemTc = 16384;    // keys per CTA of the tcgen05 scorer
constexpr int kScoreTileKeys = 64;
constexpr int kFinSpan = 8192;           // keys per CTA of the score finalize kernels

// Workspace carve-up (byte offsets from the workspace base, 256-B aligned).
struct Layout {
  size_t status;     // uint32 status word (+ padding)
  size_t lse_part;   // float2 [U][R][key_splits]
  size_t lse;        // float  [U][R]   log2-domain LSE of each observation row
  size_t s_part;     // float  [U][row_blocks][n]
  size_t s_tmp;      // float  [U][n]   pooled scores
  size_t fin_part;   // float4 [U][ceil(n / kFinSpan)]  per-slice (max, sum.hi, sum.lo, 0)
  size_t a;          // float  [U][n]   scores (when the caller gives none)
  size_t keys0, keys1, vals0, vals1;  // uint32/int32 [U][n]
  size_t hist;       // uint32 [U][256][sort_tiles]
  size_t yrank;      // float2 [U][n]  ||v||^2 per rank, double-float
  size_t agg_mq;     // float4 [U][chunks]  (m.hi, m.lo, q.hi, q.lo)
  size_t agg_v;      // float  [U][chunks][d]
  size_t agg_k;      // float  [U][chunks][d]
  size_t base_mq;    // float4 [U][chunks]  suffix after the chunk
  size_t base_v;     // float2 [U][chunks][d]
  size_t curve;      // float2 [U][n]  c(b) as hi + lo
  size_t cmax;       // uint64 [U]     order key of max_b c(b)
  size_t cand;       // int32  [U][n]  allocator candidates
  size_t ncand;      // int32  [U][hull_segs + groups] survivors per segment, per group
  size_t cl_sum;     // float2 [U][m][8 parts][2][d]  cluster part sums (m = clusters)
  size_t cl_mean;    // float  [U][m][2][d]           stored cluster means
  size_t cl_max;     // float2 [U][m][8 parts]        cluster part radii
  size_t total;
  // 16-byte guard words after the regions (certkv_workspace_guard_*)
  static constexpr int kMaxGuards = 32;
  size_t guard[kMaxGuards];
  int nguards;
};

Layout make_layout(const Prob& p);

// Validation shared by the decode entry points (certkv_decode_attn and
// certkv_decode_attn_noalloc), so that both accept exactly the same calls.
// decode_prob: the shape (as every entry point checks it) -> the problem
// description of a decode call.  decode_args: query, packed cache and output
// pointers (non-null, 16-byte aligned), tail_slot in {0, 1}, a finite scale
// >= 0 -> the effective softmax scale (0 selects 1/sqrt(d)).  Both return
// CERTKV_OK or CERTKV_EINVAL and launch nothing.
int decode_prob(const certkv_shape* shape, Prob* p);
int decode_args(const certkv_shape* shape, const void* q, const certkv_packed* packed,
                float scale, int32_t tail_slot, const void* out, float* sc);

// ---- launchers (all asynchronous on `st`) --------------------------------
__global__ void lse_merge_kernel(Prob p, const float2* __restrict__ part, float* __restrict__ lse2);
bool score_tc_supported(const Prob& p);
bool launch_score_tc(const Prob& p, const void* K, const void* Q, float2* lse_part, float* lse2,
                     float* s_part, uint32_t* status, cudaStream_t st);
void launch_score(const Prob& p, const Layout& ly, char* ws, const void* K, const void* Q,
                  float* a_out, cudaStream_t st);
void launch_sort(const Prob& p, const Layout& ly, char* ws, const float* a, cudaStream_t st);
void launch_curves(const Prob& p, const Layout& ly, char* ws, const void* K, const void* V,
                   bool need_k, cudaStream_t st);
void launch_allocate(const Prob& p, const Layout& ly, char* ws, int32_t* counts,
                     int64_t* offsets, cudaStream_t st);
void launch_pack(const Prob& p, const Layout& ly, char* ws, const void* K, const void* V,
                 const float* a, void* pk, void* pv, const int64_t* offsets,
                 const int32_t* counts, int32_t* positions, float* tail_f32,
                 double* tail_mass, float* cluster_meta, float* kept_vmax, cudaStream_t st);
void launch_export_curves(const Prob& p, const Layout& ly, char* ws, int32_t* perm_out,
                          double* c_out, cudaStream_t st);
// Decode launchers: false if nothing could be launched (the device query of
// the persistent grid failed).
bool launch_decode(const Prob& p, const void* q, const void* pk, const void* pv,
                   const int64_t* offsets, const int32_t* counts, int tail_slot, float scale,
                   void* out, char* ws, cudaStream_t st);
size_t decode_workspace(const Prob& p);
size_t fixed_row_workspace(const Prob& p);
size_t coverage_workspace(const Prob& p);
size_t sampled_workspace(const Prob& p);
bool launch_sampled(const Prob& p, const void* q, const void* K, const void* V,
                    const int64_t* offsets, const int32_t* counts, const int32_t* positions,
                    int m, const float* unif, int32_t* idx_out, float scale, float* stats,
                    char* ws, cudaStream_t st);
void launch_coverage(const Prob& p, const void* q, const void* K, float scale,
                     const double* eta, int n_eta, const double* rel_eps, int n_rel,
                     const double* abs_eps, int n_abs, int32_t* K_eta, int32_t* rel,
                     int32_t* abs_, float* top, int32_t* order, float* gap, char* ws,
                     cudaStream_t st);
bool launch_fixed_row(const Prob& p, const void* q, const void* K, const void* V,
                      const float* scores, const int64_t* offsets, const int32_t* counts,
                      const int32_t* positions,
                      const void* pk, const void* pv, int tail_slot, float scale, float* stats,
                      char* ws, cudaStream_t st);
bool launch_decode_certified(const Prob& p, const void* q, const void* pk, const void* pv,
                             const int64_t* offsets, const int32_t* counts, int tail_slot,
                             int clusters, const float* cluster_meta, const float* kept_vmax,
                             float scale, void* out, float* bound, int32_t* certified, char* ws,
                             cudaStream_t st);

// ---- optional kernel timing (off by default) ------------------------------
// When enabled with certkv_trace_enable(), every kernel launch is bracketed
// by a pair of CUDA events recorded on the launching stream.
void trace_begin(const char* name, cudaStream_t st);
void trace_end(cudaStream_t st);

struct TraceScope {
  cudaStream_t st;
  TraceScope(const char* name, cudaStream_t s) : st(s) { trace_begin(name, s); }
  ~TraceScope() { trace_end(st); }
};

}  // namespace certkv
