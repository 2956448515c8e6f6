// api.cu — the C ABI (include/certkv.h): host-side validation, workspace
// carve-up and the launch sequence of each entry point.  Validation runs
// before any launch; a call that returns an error has enqueued nothing.
#include <math.h>
#include <stdint.h>
#include <string.h>

#include "../../include/certkv.h"
#include "common.cuh"
#include "internal.cuh"

namespace certkv {

namespace {

size_t align256(size_t x) { return (x + 255) / 256 * 256; }

bool is_pow2_le16(int g) { return g == 1 || g == 2 || g == 4 || g == 8 || g == 16; }

int check_shape(const certkv_shape* s) {
  if (!s) return CERTKV_EINVAL;
  if (s->batch < 1 || s->layers < 1 || s->hq < 1 || s->hkv < 1) return CERTKV_EINVAL;
  if (s->d != kD) return CERTKV_EINVAL;
  if (s->hkv > 32 || s->hq % s->hkv != 0) return CERTKV_EINVAL;
  if (!is_pow2_le16(s->hq / s->hkv)) return CERTKV_EINVAL;
  if (s->w < 1 || s->w >= s->n || s->n > (1 << 24)) return CERTKV_EINVAL;
  const long long units = (long long)s->batch * s->layers * s->hkv;
  if (units > (1LL << 24)) return CERTKV_EINVAL;
  return CERTKV_OK;
}

int check_params(const certkv_params* q) {
  if (!q) return CERTKV_EINVAL;
  if (!(q->scale >= 0.0f) || !isfinite(q->scale)) return CERTKV_EINVAL;
  if (q->pool_kernel < 1 || (q->pool_kernel & 1) == 0 || q->pool_kernel > 255) return CERTKV_EINVAL;
  if (q->protect_window != 0 && q->protect_window != 1) return CERTKV_EINVAL;
  if (q->alpha_den < 1 || q->alpha_num < 0 || q->alpha_num > q->alpha_den) return CERTKV_EINVAL;
  if (q->bisect_steps < 0 || q->bisect_steps > 200) return CERTKV_EINVAL;
  if (q->statistic < 0 || q->statistic > 2) return CERTKV_EINVAL;
  if (q->tail_slot != 0 && q->tail_slot != 1) return CERTKV_EINVAL;
  if (q->allocator < CERTKV_ALLOC_LAGRANGIAN || q->allocator > CERTKV_ALLOC_GREEDY) return CERTKV_EINVAL;
  if (q->tail_clusters < 0 || q->tail_clusters > CERTKV_MAX_CLUSTERS) return CERTKV_EINVAL;
  return CERTKV_OK;
}

// Fill the problem description; budget_live < 0 means "no budget needed".
int make_prob(const certkv_shape* s, const certkv_params* q, int64_t budget_live, Prob* p) {
  int rc = check_shape(s);
  if (rc) return rc;
  rc = check_params(q);
  if (rc) return rc;
  Prob& P = *p;
  memset(&P, 0, sizeof P);
  P.B = s->batch; P.L = s->layers; P.Hq = s->hq; P.H = s->hkv; P.n = s->n; P.d = s->d;
  P.w = s->w; P.G = s->hq / s->hkv; P.R = P.G * P.w;
  P.units = P.B * P.L * P.H;
  P.bl = P.B * P.L;
  P.scale = q->scale > 0.0f ? q->scale : (float)(1.0 / sqrt((double)s->d));
  P.scale_log2 = P.scale * 1.4426950408889634f;
  P.pool = q->pool_kernel; P.protect = q->protect_window;
  P.alpha_num = q->alpha_num; P.alpha_den = q->alpha_den; P.T = q->bisect_steps;
  P.statistic = q->statistic; P.tail_slot = q->tail_slot; P.allocator = q->allocator;
  P.clusters = q->tail_clusters;
  P.score_warps = (P.R + 15) / 16 < 16 ? (P.R + 15) / 16 : 16;
  P.row_blocks = (P.R + 16 * P.score_warps - 1) / (16 * P.score_warps);
  if (score_tc_supported(P)) P.row_blocks = P.R / 64;  // one per 64-row quarter of the tcgen05 pass 2
  P.score_tc = score_tc_supported(P) ? 1 : 0;
  P.key_splits = P.score_tc ? (P.n + kKeysPerItemTc - 1) / kKeysPerItemTc
                            : (P.n + kScoreKeysPerCta - 1) / kScoreKeysPerCta;
  P.sort_tiles = (P.n + kSortTile - 1) / kSortTile;
  P.chunks = (P.n + kChunk - 1) / kChunk;
  if (budget_live >= 0) {
    const int64_t H = P.H;
    const int64_t charged = H * ((P.tail_slot ? 1 : 0) + P.clusters);  // summary slots
    if (budget_live < charged + H || budget_live > H * (int64_t)P.n) return CERTKV_EBUDGET;
    P.B_live = budget_live;
    P.B_real = budget_live - charged;
    int64_t bmin = ((int64_t)P.alpha_num * P.B_real) / ((int64_t)P.alpha_den * H);
    if (bmin < 1) bmin = 1;
    if (P.B_real < H * bmin || P.B_real > H * (int64_t)(P.n - 1)) return CERTKV_EBUDGET;
    P.b_min = (int)bmin;
  } else {
    P.b_min = 1;
  }
  P.hull_segs = (P.n - P.b_min + kHullSeg - 1) / kHullSeg;
  return CERTKV_OK;
}

}  // namespace

Layout make_layout(const Prob& p) {
  Layout ly;
  ly.nguards = 0;
  size_t off = 0;
  // each region is followed by a 16-byte guard (after its bytes rounded up to
  // 16) that no kernel writes
  auto take = [&](size_t bytes) {
    size_t o = off;
    const size_t g = o + (bytes + 15) / 16 * 16;
    if (ly.nguards < Layout::kMaxGuards) ly.guard[ly.nguards++] = g;
    off = align256(g + 16);
    return o;
  };
  const size_t U = (size_t)p.units, n = (size_t)p.n;
  ly.status = take(256);
  ly.lse_part = take(U * p.R * p.key_splits * sizeof(float2));
  ly.lse = take(U * p.R * sizeof(float));
  ly.s_part = take(U * p.row_blocks * n * sizeof(float));
  ly.s_tmp = take(U * n * sizeof(float));
  ly.fin_part = take(U * ((n + kFinSpan - 1) / kFinSpan) * sizeof(float4));
  ly.a = take(U * n * sizeof(float));
  ly.keys0 = take(U * n * 4);
  ly.keys1 = take(U * n * 4);
  ly.vals0 = take(U * n * 4);
  ly.vals1 = take(U * n * 4);
  ly.hist = take(U * 256 * p.sort_tiles * 4);
  ly.yrank = take(U * n * sizeof(float2));
  ly.agg_mq = take(U * p.chunks * sizeof(float4));
  ly.agg_v = take(U * p.chunks * kD * sizeof(float));
  ly.agg_k = take(U * p.chunks * kD * sizeof(float));
  ly.base_mq = take(U * p.chunks * sizeof(float4));
  ly.base_v = take(U * p.chunks * kD * sizeof(float2));
  ly.curve = take(U * n * sizeof(float2));
  ly.cmax = take(U * sizeof(unsigned long long));
  ly.cand = take(U * n * sizeof(int32_t));
  // the candidate counts are sized for the smallest b_min (1) so that one
  // workspace size serves every budget of a shape
  const size_t segs = (size_t)((p.n - 1 + kHullSeg - 1) / kHullSeg);
  const size_t groups = (segs + kGroupSegs - 1) / kGroupSegs;
  ly.ncand = take(U * (segs + groups) * sizeof(int32_t));
  const size_t mc = (size_t)p.clusters;
  ly.cl_sum = take(U * mc * 8 * 2 * kD * sizeof(float) * 2);
  ly.cl_mean = take(U * mc * 2 * kD * sizeof(float));
  ly.cl_max = take(U * mc * 8 * sizeof(float) * 2);
  ly.total = off;
  return ly;
}

}  // namespace certkv

namespace certkv {

int decode_prob(const certkv_shape* shape, Prob* p) {
  int rc = check_shape(shape);
  if (rc) return rc;
  certkv_params prm;
  certkv_default_params(&prm);
  return make_prob(shape, &prm, -1, p);
}

int decode_args(const certkv_shape* shape, const void* q, const certkv_packed* packed,
                float scale, int32_t tail_slot, const void* out, float* sc) {
  if (!q || !packed || !packed->k || !packed->v || !packed->offsets || !packed->real_counts || !out)
    return CERTKV_EINVAL;
  if (((uintptr_t)packed->k | (uintptr_t)packed->v | (uintptr_t)q) % 16 != 0) return CERTKV_EINVAL;
  if (tail_slot != 0 && tail_slot != 1) return CERTKV_EINVAL;
  if (!(scale >= 0.0f) || !isfinite(scale)) return CERTKV_EINVAL;
  *sc = scale > 0.0f ? scale : (float)(1.0 / sqrt((double)shape->d));
  return CERTKV_OK;
}

}  // namespace certkv

namespace certkv_api {

using namespace certkv;

int cuda_ok(cudaError_t e) { return e == cudaSuccess ? CERTKV_OK : CERTKV_ECUDA; }

bool aligned(const void* ptr, size_t a) { return ((uintptr_t)ptr % a) == 0; }

// key-init for caller-given scores: keys0 = ~bits(a) (the sort's first pass
// takes the indices as its values); flags negative or non-finite scores.
__global__ void key_init_kernel(Prob p, const float* __restrict__ a, uint32_t* __restrict__ keys,
                                uint32_t* status) {
  const size_t total = (size_t)p.units * p.n;
  bool bad = false;
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (size_t)gridDim.x * blockDim.x) {
    const float x = a[i];
    if (!(x >= 0.0f && x <= 3.0e38f)) bad = true;
    keys[i] = score_key(x > 0.0f ? x : 0.0f);
  }
  if (bad) raise_status(status, CERTKV_STATUS_NONFINITE);
}

// The guard words written after every workspace region (a fixed pattern).
__device__ __constant__ uint32_t kGuard[4] = {0x9E3779B9u, 0x7F4A7C15u, 0xF39CC060u, 0x5CEDC834u};
struct GuardSet {
  size_t off[Layout::kMaxGuards];
  int n;
};
GuardSet guard_set(const Layout& ly) {
  GuardSet g;
  g.n = ly.nguards;
  for (int i = 0; i < Layout::kMaxGuards; ++i) g.off[i] = i < ly.nguards ? ly.guard[i] : 0;
  return g;
}
__global__ void guard_arm_kernel(char* ws, GuardSet g) {
  const int i = threadIdx.x;
  if (i < g.n)
    *reinterpret_cast<uint4*>(ws + g.off[i]) = make_uint4(kGuard[0], kGuard[1], kGuard[2], kGuard[3]);
}
__global__ void guard_check_kernel(const char* ws, GuardSet g, uint32_t* count) {
  const int i = threadIdx.x;
  if (i < g.n) {
    const uint4 x = *reinterpret_cast<const uint4*>(ws + g.off[i]);
    if (x.x != kGuard[0] || x.y != kGuard[1] || x.z != kGuard[2] || x.w != kGuard[3])
      atomicAdd(count, 1u);
  }
}

int check_ws(const Prob& p, void* ws, size_t ws_bytes, Layout* ly) {
  *ly = make_layout(p);
  if (!ws || !aligned(ws, 256) || ws_bytes < ly->total) return CERTKV_EWORKSPACE;
  return CERTKV_OK;
}

int check_packed(const Prob& p, const certkv_packed* out) {
  if (!out || !out->k || !out->v || !out->offsets || !out->real_counts || !out->positions)
    return CERTKV_EINVAL;
  if (!aligned(out->k, 16) || !aligned(out->v, 16)) return CERTKV_EINVAL;
  if (out->capacity_slots < (int64_t)p.bl * p.B_live) return CERTKV_ECAPACITY;
  if (p.clusters > 0 && (!out->cluster_meta || !out->kept_vmax)) return CERTKV_EINVAL;
  return CERTKV_OK;
}

int run_scored(const Prob& p, const Layout& ly, char* ws, const void* K, const void* V,
               const float* a, certkv_packed* out, cudaStream_t st) {
  launch_sort(p, ly, ws, a, st);
  launch_curves(p, ly, ws, K, V, p.tail_slot != 0, st);
  launch_allocate(p, ly, ws, out->real_counts, out->offsets, st);
  launch_pack(p, ly, ws, K, V, a, out->k, out->v, out->offsets, out->real_counts, out->positions,
              out->tail_f32, out->tail_mass, out->cluster_meta, out->kept_vmax, st);
  return cuda_ok(cudaGetLastError());
}

}  // namespace certkv_api

using namespace certkv;
using namespace certkv_api;

extern "C" {

void certkv_default_params(certkv_params* p) {
  if (!p) return;
  p->scale = 0.0f;
  p->pool_kernel = 5;
  p->protect_window = 1;
  p->alpha_num = 1;
  p->alpha_den = 5;
  p->bisect_steps = 40;
  p->statistic = CERTKV_STAT_CENTERED;
  p->tail_slot = 1;
  p->allocator = CERTKV_ALLOC_LAGRANGIAN;
  p->tail_clusters = 0;
}

int64_t certkv_live_budget(int32_t n, int32_t hkv, int64_t keep_num, int64_t keep_den) {
  if (n < 1 || hkv < 1 || keep_num < 0 || keep_den < 1 || keep_num > keep_den) return -1;
  return (int64_t)hkv * (((int64_t)n * keep_num) / keep_den);
}

size_t certkv_workspace_bytes(const certkv_shape* shape, const certkv_params* params) {
  Prob p;
  if (make_prob(shape, params, -1, &p)) return 0;
  return make_layout(p).total;
}

size_t certkv_decode_workspace_bytes(const certkv_shape* shape) {
  if (check_shape(shape)) return 0;
  certkv_params q;
  certkv_default_params(&q);
  Prob p;
  if (make_prob(shape, &q, -1, &p)) return 0;
  return decode_workspace(p);
}

int certkv_score(const certkv_shape* shape, const void* K, const void* Q_obs,
                 const certkv_params* params, float* a_out, void* workspace,
                 size_t workspace_bytes, void* stream) {
  Prob p;
  int rc = make_prob(shape, params, -1, &p);
  if (rc) return rc;
  if (!K || !Q_obs || !a_out) return CERTKV_EINVAL;
  if (!aligned(K, 16) || !aligned(Q_obs, 16)) return CERTKV_EINVAL;
  Layout ly;
  if ((rc = check_ws(p, workspace, workspace_bytes, &ly))) return rc;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  char* ws = reinterpret_cast<char*>(workspace);
  p.status = reinterpret_cast<uint32_t*>(ws + ly.status);
  if ((rc = cuda_ok(cudaMemsetAsync(ws + ly.status, 0, 256, st)))) return rc;
  launch_score(p, ly, ws, K, Q_obs, a_out, st);
  return cuda_ok(cudaGetLastError());
}

int certkv_curves(const certkv_shape* shape, const void* V, const float* a,
                  const certkv_params* params, int32_t* perm_out, double* c_out, void* workspace,
                  size_t workspace_bytes, void* stream) {
  Prob p;
  int rc = make_prob(shape, params, -1, &p);
  if (rc) return rc;
  if (!V || !a || (!perm_out && !c_out)) return CERTKV_EINVAL;
  if (!aligned(V, 16)) return CERTKV_EINVAL;
  Layout ly;
  if ((rc = check_ws(p, workspace, workspace_bytes, &ly))) return rc;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  char* ws = reinterpret_cast<char*>(workspace);
  p.status = reinterpret_cast<uint32_t*>(ws + ly.status);
  if ((rc = cuda_ok(cudaMemsetAsync(ws + ly.status, 0, 256, st)))) return rc;
  {
    TraceScope ts_("key_init", st);
    key_init_kernel<<<1024, 256, 0, st>>>(p, a, reinterpret_cast<uint32_t*>(ws + ly.keys0),
                                          reinterpret_cast<uint32_t*>(ws + ly.status));
  }
  launch_sort(p, ly, ws, a, st);
  launch_curves(p, ly, ws, V, V, false, st);
  launch_export_curves(p, ly, ws, perm_out, c_out, st);
  return cuda_ok(cudaGetLastError());
}

int certkv_compress_scored(const certkv_shape* shape, const void* K, const void* V,
                           const float* a, int64_t budget_live, const certkv_params* params,
                           certkv_packed* out, void* workspace, size_t workspace_bytes,
                           void* stream) {
  Prob p;
  if (budget_live < 0) return CERTKV_EBUDGET;
  int rc = make_prob(shape, params, budget_live, &p);
  if (rc) return rc;
  if (!K || !V || !a) return CERTKV_EINVAL;
  if (!aligned(K, 16) || !aligned(V, 16)) return CERTKV_EINVAL;
  if ((rc = check_packed(p, out))) return rc;
  p.capacity = out->capacity_slots;
  Layout ly;
  if ((rc = check_ws(p, workspace, workspace_bytes, &ly))) return rc;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  char* ws = reinterpret_cast<char*>(workspace);
  p.status = reinterpret_cast<uint32_t*>(ws + ly.status);
  if ((rc = cuda_ok(cudaMemsetAsync(ws + ly.status, 0, 256, st)))) return rc;
  {
    TraceScope ts_("key_init", st);
    key_init_kernel<<<1024, 256, 0, st>>>(p, a, reinterpret_cast<uint32_t*>(ws + ly.keys0),
                                          reinterpret_cast<uint32_t*>(ws + ly.status));
  }
  return run_scored(p, ly, ws, K, V, a, out, st);
}

namespace {
// (sequence, layer) pairs per chunk of certkv_compress_host: 0 picks about
// 1 GiB of K and V per chunk (at least 1 pair, at most all of them).
int host_chunk(const Prob& p, int32_t chunk) {
  if (chunk > 0) return chunk < p.bl ? chunk : p.bl;
  const size_t per_bl = (size_t)2 * p.H * p.n * kD * 2;
  size_t c = ((size_t)1 << 30) / per_bl;
  if (c < 1) c = 1;
  if (c > (size_t)p.bl) c = (size_t)p.bl;
  return (int)c;
}
// Shape of a chunk of `cnt` consecutive (sequence, layer) pairs: one
// sequence with cnt layers (the pairs are independent).
certkv_shape chunk_shape(const certkv_shape* s, int cnt) {
  certkv_shape c = *s;
  c.batch = 1;
  c.layers = cnt;
  return c;
}
struct HostPlan {
  Prob full, sub;
  int chunk;
  size_t ws_sub, stage_k, stage_q, stage, total;
};
int host_plan(const certkv_shape* shape, const certkv_params* params, int64_t budget, int32_t chunk,
              HostPlan* hp) {
  int rc = make_prob(shape, params, budget, &hp->full);
  if (rc) return rc;
  hp->chunk = host_chunk(hp->full, chunk);
  const certkv_shape cs = chunk_shape(shape, hp->chunk);
  if ((rc = make_prob(&cs, params, budget, &hp->sub))) return rc;
  hp->ws_sub = align256(make_layout(hp->sub).total);
  hp->stage_k = align256((size_t)hp->chunk * hp->full.H * hp->full.n * kD * 2);
  hp->stage_q = align256((size_t)hp->chunk * hp->full.Hq * hp->full.w * kD * 2);
  hp->stage = 2 * hp->stage_k + hp->stage_q;
  hp->total = hp->ws_sub + 2 * hp->stage;
  return CERTKV_OK;
}
}  // namespace

size_t certkv_host_workspace_bytes(const certkv_shape* shape, const certkv_params* params,
                                   int32_t chunk) {
  HostPlan hp;
  if (chunk < 0 || host_plan(shape, params, -1, chunk, &hp)) return 0;
  return hp.total;
}

namespace {
// certkv_compress_host, and with host_out the chunk-by-chunk copy back of the
// packed cache on a third stream
int compress_host_impl(const certkv_shape* shape, const void* hK, const void* hV,
                       const void* hQ_obs, int64_t budget_live, const certkv_params* params,
                       int32_t chunk, certkv_packed* out, certkv_packed* host_out,
                       void* workspace, size_t workspace_bytes, void* stream) {
  if (budget_live < 0) return CERTKV_EBUDGET;
  if (chunk < 0) return CERTKV_EINVAL;
  HostPlan hp;
  int rc = host_plan(shape, params, budget_live, chunk, &hp);
  if (rc) return rc;
  if (!hK || !hV || !hQ_obs) return CERTKV_EINVAL;
  if ((rc = check_packed(hp.full, out))) return rc;
  if (host_out && (!host_out->k || !host_out->v || !host_out->offsets ||
                   !host_out->real_counts || !host_out->positions ||
                   host_out->capacity_slots < (int64_t)hp.full.bl * hp.full.B_live))
    return CERTKV_EINVAL;
  if (!workspace || !aligned(workspace, 256) || workspace_bytes < hp.total) return CERTKV_EWORKSPACE;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  char* ws = reinterpret_cast<char*>(workspace);
  char* stage[2] = {ws + hp.ws_sub, ws + hp.ws_sub + hp.stage};
  // private copy streams (in; back) and their events, released when their
  // work is done
  cudaStream_t cs = nullptr, ds = nullptr;
  cudaEvent_t start = nullptr, staged[2] = {nullptr, nullptr}, freed[2] = {nullptr, nullptr};
  cudaEvent_t packed_ev = nullptr, back_done = nullptr;
  auto release = [&]() {
    for (int i = 0; i < 2; ++i) {
      if (staged[i]) cudaEventDestroy(staged[i]);
      if (freed[i]) cudaEventDestroy(freed[i]);
    }
    if (start) cudaEventDestroy(start);
    if (packed_ev) cudaEventDestroy(packed_ev);
    if (back_done) cudaEventDestroy(back_done);
    if (cs) cudaStreamDestroy(cs);
    if (ds) cudaStreamDestroy(ds);
  };
  if (cudaStreamCreateWithFlags(&cs, cudaStreamNonBlocking) != cudaSuccess ||
      cudaEventCreateWithFlags(&start, cudaEventDisableTiming) != cudaSuccess) {
    release();
    return CERTKV_ECUDA;
  }
  if (host_out && (cudaStreamCreateWithFlags(&ds, cudaStreamNonBlocking) != cudaSuccess ||
                   cudaEventCreateWithFlags(&packed_ev, cudaEventDisableTiming) != cudaSuccess ||
                   cudaEventCreateWithFlags(&back_done, cudaEventDisableTiming) != cudaSuccess)) {
    release();
    return CERTKV_ECUDA;
  }
  for (int i = 0; i < 2; ++i)
    if (cudaEventCreateWithFlags(&staged[i], cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&freed[i], cudaEventDisableTiming) != cudaSuccess) {
      release();
      return CERTKV_ECUDA;
    }
  const Prob& F = hp.full;
  const size_t kv_bl = (size_t)F.H * F.n * kD * 2, q_bl = (size_t)F.Hq * F.w * kD * 2;
  const Layout ly_sub = make_layout(hp.sub);
  rc = cuda_ok(cudaMemsetAsync(ws + ly_sub.status, 0, 256, st));
  if (!rc) rc = cuda_ok(cudaEventRecord(start, st));
  if (!rc) rc = cuda_ok(cudaStreamWaitEvent(cs, start, 0));
  for (int bl0 = 0, c = 0; !rc && bl0 < F.bl; bl0 += hp.chunk, ++c) {
    const int cnt = (F.bl - bl0) < hp.chunk ? (F.bl - bl0) : hp.chunk;
    const int s = c & 1;
    char* sK = stage[s];
    char* sV = stage[s] + hp.stage_k;
    char* sQ = stage[s] + 2 * hp.stage_k;
    // copy stream: wait until chunk c - 2 has left this half, then stage chunk c
    if (c >= 2) rc = cuda_ok(cudaStreamWaitEvent(cs, freed[s], 0));
    if (!rc) rc = cuda_ok(cudaMemcpyAsync(sK, (const char*)hK + bl0 * kv_bl, cnt * kv_bl,
                                          cudaMemcpyHostToDevice, cs));
    if (!rc) rc = cuda_ok(cudaMemcpyAsync(sV, (const char*)hV + bl0 * kv_bl, cnt * kv_bl,
                                          cudaMemcpyHostToDevice, cs));
    if (!rc) rc = cuda_ok(cudaMemcpyAsync(sQ, (const char*)hQ_obs + bl0 * q_bl, cnt * q_bl,
                                          cudaMemcpyHostToDevice, cs));
    if (!rc) rc = cuda_ok(cudaEventRecord(staged[s], cs));
    if (!rc) rc = cuda_ok(cudaStreamWaitEvent(st, staged[s], 0));
    if (rc) break;
    // compute stream: the chunk as its own problem, writing global slots
    Prob p;
    certkv_shape csub = chunk_shape(shape, cnt);
    if ((rc = make_prob(&csub, params, budget_live, &p))) break;
    p.slot_base = (int64_t)bl0 * F.B_live;
    p.capacity = out->capacity_slots;
    const Layout ly = make_layout(p);
    p.status = reinterpret_cast<uint32_t*>(ws + ly.status);
    certkv_packed o = *out;
    o.offsets = out->offsets + (size_t)bl0 * F.H;
    o.real_counts = out->real_counts + (size_t)bl0 * F.H;
    if (out->tail_f32) o.tail_f32 = out->tail_f32 + (size_t)bl0 * F.H * 2 * kD;
    if (out->tail_mass) o.tail_mass = out->tail_mass + (size_t)bl0 * F.H;
    if (out->cluster_meta) o.cluster_meta = out->cluster_meta + (size_t)bl0 * F.H * F.clusters * 4;
    if (out->kept_vmax) o.kept_vmax = out->kept_vmax + (size_t)bl0 * F.H;
    float* a = reinterpret_cast<float*>(ws + ly.a);
    launch_score(p, ly, ws, sK, sQ, a, st);
    rc = run_scored(p, ly, ws, sK, sV, a, &o, st);
    if (!rc) rc = cuda_ok(cudaEventRecord(freed[s], st));
    if (!rc && host_out) {  // this chunk's part of the packed cache back to the host
      const size_t s0 = (size_t)bl0 * F.B_live, ns = (size_t)cnt * F.B_live;
      const size_t u0 = (size_t)bl0 * F.H, nu = (size_t)cnt * F.H;
      const size_t row = (size_t)kD * 2;
      const bool last = bl0 + cnt == F.bl;
      rc = cuda_ok(cudaEventRecord(packed_ev, st));
      if (!rc) rc = cuda_ok(cudaStreamWaitEvent(ds, packed_ev, 0));
      if (!rc) rc = cuda_ok(cudaMemcpyAsync((char*)host_out->k + s0 * row, (const char*)out->k + s0 * row,
                                            ns * row, cudaMemcpyDeviceToHost, ds));
      if (!rc) rc = cuda_ok(cudaMemcpyAsync((char*)host_out->v + s0 * row, (const char*)out->v + s0 * row,
                                            ns * row, cudaMemcpyDeviceToHost, ds));
      if (!rc) rc = cuda_ok(cudaMemcpyAsync(host_out->positions + s0, out->positions + s0,
                                            ns * sizeof(int32_t), cudaMemcpyDeviceToHost, ds));
      if (!rc) rc = cuda_ok(cudaMemcpyAsync(host_out->real_counts + u0, out->real_counts + u0,
                                            nu * sizeof(int32_t), cudaMemcpyDeviceToHost, ds));
      if (!rc) rc = cuda_ok(cudaMemcpyAsync(host_out->offsets + u0, out->offsets + u0,
                                            (nu + (last ? 1 : 0)) * sizeof(int64_t),
                                            cudaMemcpyDeviceToHost, ds));
    }
  }
  if (!rc && host_out) {  // the call completes on `stream` with its copies back
    rc = cuda_ok(cudaEventRecord(back_done, ds));
    if (!rc) rc = cuda_ok(cudaStreamWaitEvent(st, back_done, 0));
  }
  release();
  return rc;
}
}  // namespace

int certkv_compress_host(const certkv_shape* shape, const void* hK, const void* hV,
                         const void* hQ_obs, int64_t budget_live, const certkv_params* params,
                         int32_t chunk, certkv_packed* out, void* workspace,
                         size_t workspace_bytes, void* stream) {
  return compress_host_impl(shape, hK, hV, hQ_obs, budget_live, params, chunk, out, nullptr,
                            workspace, workspace_bytes, stream);
}

int certkv_compress_host_copyback(const certkv_shape* shape, const void* hK, const void* hV,
                                  const void* hQ_obs, int64_t budget_live,
                                  const certkv_params* params, int32_t chunk, certkv_packed* out,
                                  certkv_packed* host_out, void* workspace,
                                  size_t workspace_bytes, void* stream) {
  if (!host_out) return CERTKV_EINVAL;
  return compress_host_impl(shape, hK, hV, hQ_obs, budget_live, params, chunk, out, host_out,
                            workspace, workspace_bytes, stream);
}

int certkv_compress(const certkv_shape* shape, const void* K, const void* V, const void* Q_obs,
                    int64_t budget_live, const certkv_params* params, certkv_packed* out,
                    void* workspace, size_t workspace_bytes, void* stream) {
  Prob p;
  if (budget_live < 0) return CERTKV_EBUDGET;
  int rc = make_prob(shape, params, budget_live, &p);
  if (rc) return rc;
  if (!K || !V || !Q_obs) return CERTKV_EINVAL;
  if (!aligned(K, 16) || !aligned(V, 16) || !aligned(Q_obs, 16)) return CERTKV_EINVAL;
  if ((rc = check_packed(p, out))) return rc;
  p.capacity = out->capacity_slots;
  Layout ly;
  if ((rc = check_ws(p, workspace, workspace_bytes, &ly))) return rc;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  char* ws = reinterpret_cast<char*>(workspace);
  p.status = reinterpret_cast<uint32_t*>(ws + ly.status);
  if ((rc = cuda_ok(cudaMemsetAsync(ws + ly.status, 0, 256, st)))) return rc;
  float* a = reinterpret_cast<float*>(ws + ly.a);
  launch_score(p, ly, ws, K, Q_obs, a, st);
  return run_scored(p, ly, ws, K, V, a, out, st);
}

int certkv_decode_attn(const certkv_shape* shape, const void* q, const certkv_packed* packed,
                       float scale, int32_t tail_slot, void* out, void* workspace,
                       size_t workspace_bytes, void* stream) {
  Prob p;
  int rc = decode_prob(shape, &p);
  if (rc) return rc;
  float sc = 0.0f;
  if ((rc = decode_args(shape, q, packed, scale, tail_slot, out, &sc))) return rc;
  if (!workspace || !aligned(workspace, 256) || workspace_bytes < decode_workspace(p))
    return CERTKV_EWORKSPACE;
  p.capacity = packed->capacity_slots;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (!launch_decode(p, q, packed->k, packed->v, packed->offsets, packed->real_counts, tail_slot,
                     sc, out, reinterpret_cast<char*>(workspace), st))
    return CERTKV_ECUDA;
  return cuda_ok(cudaGetLastError());
}

int certkv_decode_certified(const certkv_shape* shape, const void* q, const certkv_packed* packed,
                            float scale, int32_t tail_slot, int32_t clusters, void* out,
                            float* bound, int32_t* certified, void* workspace,
                            size_t workspace_bytes, void* stream) {
  int rc = check_shape(shape);
  if (rc) return rc;
  if (!q || !packed || !packed->k || !packed->v || !packed->offsets || !packed->real_counts ||
      !packed->cluster_meta || !packed->kept_vmax || !out || !bound || !certified)
    return CERTKV_EINVAL;
  if (!aligned(packed->k, 16) || !aligned(packed->v, 16) || !aligned(q, 16)) return CERTKV_EINVAL;
  if (tail_slot != 0 && tail_slot != 1) return CERTKV_EINVAL;
  if (clusters < 1 || clusters > CERTKV_MAX_CLUSTERS) return CERTKV_EINVAL;
  if (!(scale >= 0.0f) || !isfinite(scale)) return CERTKV_EINVAL;
  certkv_params prm;
  certkv_default_params(&prm);
  Prob p;
  if ((rc = make_prob(shape, &prm, -1, &p))) return rc;
  if (!workspace || !aligned(workspace, 256) || workspace_bytes < decode_workspace(p))
    return CERTKV_EWORKSPACE;
  p.capacity = packed->capacity_slots;
  const float sc = scale > 0.0f ? scale : (float)(1.0 / sqrt((double)shape->d));
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (!launch_decode_certified(p, q, packed->k, packed->v, packed->offsets,
                               packed->real_counts, tail_slot, clusters, packed->cluster_meta,
                               packed->kept_vmax, sc, out, bound, certified,
                               reinterpret_cast<char*>(workspace), st))
    return CERTKV_ECUDA;
  return cuda_ok(cudaGetLastError());
}

size_t certkv_fixed_row_workspace_bytes(const certkv_shape* shape) {
  certkv_params prm;
  certkv_default_params(&prm);
  Prob p;
  if (make_prob(shape, &prm, -1, &p)) return 0;
  return fixed_row_workspace(p);
}

int certkv_fixed_row_stats(const certkv_shape* shape, const void* q, const void* K, const void* V,
                           const float* scores, const certkv_packed* packed, float scale,
                           int32_t tail_slot, float* stats, void* workspace,
                           size_t workspace_bytes, void* stream) {
  certkv_params prm;
  certkv_default_params(&prm);
  Prob p;
  int rc = make_prob(shape, &prm, -1, &p);
  if (rc) return rc;
  if (!q || !K || !V || !packed || !packed->k || !packed->v || !packed->offsets ||
      !packed->real_counts || !packed->positions || !stats)
    return CERTKV_EINVAL;
  if (!aligned(q, 16) || !aligned(K, 16) || !aligned(V, 16) || !aligned(packed->k, 16) ||
      !aligned(packed->v, 16) || !aligned(scores, 4))
    return CERTKV_EINVAL;
  if (tail_slot != 0 && tail_slot != 1) return CERTKV_EINVAL;
  if (!(scale >= 0.0f) || !isfinite(scale)) return CERTKV_EINVAL;
  if (!workspace || !aligned(workspace, 256) || workspace_bytes < fixed_row_workspace(p))
    return CERTKV_EWORKSPACE;
  p.capacity = packed->capacity_slots;  // its decode runs as certkv_decode_attn does
  const float sc = scale > 0.0f ? scale : (float)(1.0 / sqrt((double)shape->d));
  if (!launch_fixed_row(p, q, K, V, scores, packed->offsets, packed->real_counts,
                        packed->positions, packed->k, packed->v, tail_slot, sc, stats,
                        reinterpret_cast<char*>(workspace), reinterpret_cast<cudaStream_t>(stream)))
    return CERTKV_ECUDA;
  return cuda_ok(cudaGetLastError());
}

size_t certkv_sampled_workspace_bytes(const certkv_shape* shape) {
  certkv_params prm;
  certkv_default_params(&prm);
  Prob p;
  if (make_prob(shape, &prm, -1, &p)) return 0;
  return sampled_workspace(p);
}

int certkv_sampled_compensation(const certkv_shape* shape, const void* q, const void* K,
                                const void* V, const certkv_packed* packed, float scale,
                                int32_t m, const float* unif, int32_t* idx_out, float* stats,
                                void* workspace, size_t workspace_bytes, void* stream) {
  certkv_params prm;
  certkv_default_params(&prm);
  Prob p;
  int rc = make_prob(shape, &prm, -1, &p);
  if (rc) return rc;
  if (!q || !K || !V || !packed || !packed->offsets || !packed->real_counts ||
      !packed->positions || !unif || !stats)
    return CERTKV_EINVAL;
  if (!aligned(q, 16) || !aligned(K, 16) || !aligned(V, 16) || !aligned(unif, 4)) return CERTKV_EINVAL;
  if (m < 1 || m > CERTKV_MAX_SAMPLES) return CERTKV_EINVAL;
  if (!(scale >= 0.0f) || !isfinite(scale)) return CERTKV_EINVAL;
  if (!workspace || !aligned(workspace, 256) || workspace_bytes < sampled_workspace(p))
    return CERTKV_EWORKSPACE;
  p.capacity = packed->capacity_slots;
  const float sc = scale > 0.0f ? scale : (float)(1.0 / sqrt((double)shape->d));
  if (!launch_sampled(p, q, K, V, packed->offsets, packed->real_counts, packed->positions, m, unif,
                      idx_out, sc, stats, reinterpret_cast<char*>(workspace),
                      reinterpret_cast<cudaStream_t>(stream)))
    return CERTKV_EINVAL;
  return cuda_ok(cudaGetLastError());
}

size_t certkv_coverage_workspace_bytes(const certkv_shape* shape) {
  certkv_params prm;
  certkv_default_params(&prm);
  Prob p;
  if (make_prob(shape, &prm, -1, &p)) return 0;
  return coverage_workspace(p);
}

namespace {
bool thresholds_ok(const double* x, int32_t cnt, bool below_one, const void* out) {
  if (cnt < 0 || cnt > CERTKV_COVERAGE_MAX_THRESHOLDS) return false;
  if (cnt == 0) return true;
  if (!x || !out) return false;
  for (int32_t e = 0; e < cnt; ++e)
    if (!(x[e] > 0.0) || !isfinite(x[e]) || (below_one && !(x[e] < 1.0))) return false;
  return true;
}
}  // namespace

int certkv_coverage_profile(const certkv_shape* shape, const void* q, const void* K, float scale,
                            const double* eta, int32_t n_eta, const double* rel_eps,
                            int32_t n_rel, const double* abs_eps, int32_t n_abs, int32_t* K_eta,
                            int32_t* rel_counts, int32_t* abs_counts, float* top, int32_t* order,
                            float* gap, void* workspace, size_t workspace_bytes, void* stream) {
  certkv_params prm;
  certkv_default_params(&prm);
  Prob p;
  int rc = make_prob(shape, &prm, -1, &p);
  if (rc) return rc;
  if (!q || !K || !top || !aligned(q, 16) || !aligned(K, 16)) return CERTKV_EINVAL;
  if (!thresholds_ok(eta, n_eta, true, K_eta) || !thresholds_ok(rel_eps, n_rel, false, rel_counts) ||
      !thresholds_ok(abs_eps, n_abs, false, abs_counts))
    return CERTKV_EINVAL;
  if (!(scale >= 0.0f) || !isfinite(scale)) return CERTKV_EINVAL;
  if (!workspace || !aligned(workspace, 256) || workspace_bytes < coverage_workspace(p))
    return CERTKV_EWORKSPACE;
  const float sc = scale > 0.0f ? scale : (float)(1.0 / sqrt((double)shape->d));
  launch_coverage(p, q, K, sc, eta, n_eta, rel_eps, n_rel, abs_eps, n_abs, K_eta, rel_counts,
                  abs_counts, top, order, gap, reinterpret_cast<char*>(workspace),
                  reinterpret_cast<cudaStream_t>(stream));
  return cuda_ok(cudaGetLastError());
}

int certkv_workspace_guard_arm(const certkv_shape* shape, const certkv_params* params,
                               void* workspace, size_t workspace_bytes, void* stream) {
  Prob p;
  if (make_prob(shape, params, -1, &p)) return -1;
  Layout ly;
  if (check_ws(p, workspace, workspace_bytes, &ly)) return -1;
  guard_arm_kernel<<<1, Layout::kMaxGuards, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
      reinterpret_cast<char*>(workspace), guard_set(ly));
  return cudaGetLastError() == cudaSuccess ? 0 : -1;
}

int certkv_workspace_guard_check(const certkv_shape* shape, const certkv_params* params,
                                 void* workspace, size_t workspace_bytes, void* stream) {
  Prob p;
  if (make_prob(shape, params, -1, &p)) return -1;
  Layout ly;
  if (check_ws(p, workspace, workspace_bytes, &ly)) return -1;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  char* ws = reinterpret_cast<char*>(workspace);
  uint32_t* count = reinterpret_cast<uint32_t*>(ws + ly.status + 4);  // beside the status word
  if (cudaMemsetAsync(count, 0, sizeof(uint32_t), st) != cudaSuccess) return -1;
  guard_check_kernel<<<1, Layout::kMaxGuards, 0, st>>>(ws, guard_set(ly), count);
  uint32_t v = 0;
  if (cudaGetLastError() != cudaSuccess || cudaStreamSynchronize(st) != cudaSuccess ||
      cudaMemcpy(&v, count, sizeof v, cudaMemcpyDeviceToHost) != cudaSuccess)
    return -1;
  return (int)v;
}

int certkv_read_status(const void* workspace, void* stream) {
  if (!workspace) return -1;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(st) != cudaSuccess) return -1;
  uint32_t v = 0;
  if (cudaMemcpy(&v, workspace, sizeof v, cudaMemcpyDeviceToHost) != cudaSuccess) return -1;
  return (int)v;
}

const char* certkv_strerror(int code) {
  switch (code) {
    case CERTKV_OK: return "ok";
    case CERTKV_EINVAL: return "invalid shape, pointer or parameter";
    case CERTKV_EBUDGET: return "infeasible budget (need 2H <= B_live <= H*n with a tail slot)";
    case CERTKV_EWORKSPACE: return "workspace missing, misaligned or too small";
    case CERTKV_ECAPACITY: return "packed-cache capacity below B*L*B_live slots";
    case CERTKV_ECUDA: return "CUDA runtime error";
    case CERTKV_ETOOLARGE:
      return "problem exceeds the fixed 16 MiB scratch of certkv_decode_attn_noalloc "
             "(about (B*L*H + 1024)*G <= 32000); split the call";
    default: return "unknown error";
  }
}

}  // extern "C"
