/*
 * certkv.h — C ABI of the CertKV exact-budget KV-cache compressor and of
 * decode attention over the packed cache it produces, for NVIDIA GB300
 * (sm_103a).
 *
 * The method is the one of "Beyond Sparse Weights: When Is Attention
 * Compressible?", §4 (CertKV: value-aware compression under exact budgets),
 * Eq. (certkv-curve), Algorithm 1 and the appendix "CertKV: implementation and
 * exact-budget protocol".  Once per (sequence, layer), after prefill:
 *
 *   a1/a2  score   observation-window softmax mass per cached token and KV head
 *                  (the SnapKV observation-window scorer the paper keeps
 *                  unchanged), normalised to a_j = (s_j)_+ / sum_i (s_i)_+;
 *   a3     order   per-head stable order by a descending, ties by lower index;
 *   a4     curve   suffix moments m_h(b), W_h(b), Q_h(b) over the evicted
 *                  ranks and the centred-dispersion curve
 *                  c_h(b) = sqrt((m_h(b) Q_h(b) - ||W_h(b)||^2)_+), b = 0..n-1;
 *   a5     budget  B_real = B_live - H, b_min = max{1, floor(alpha B_real / H)},
 *                  T-step Lagrangian bisection on a shared multiplier, then
 *                  best-marginal repair until sum_h b_h = B_real;
 *   a6     select  the top-b_h real tokens of each head;
 *   a7     tail    one synthetic pair per head: the mass-weighted key and value
 *                  centroids (k*, v*) of the evicted suffix;
 *   a8     pack    a ragged bf16 cache holding exactly B_live live slots per
 *                  (sequence, layer): b_h real slots + 1 tail slot per head.
 *   a9     decode  softmax attention over the b_h + 1 slots of each head
 *                  (the "plain slot" of the paper's ablation table).
 *
 * Conventions shared by every entry point
 *   - Pointers named in the argument lists are DEVICE pointers unless a
 *     comment says otherwise.  The caller owns every buffer: the library never
 *     allocates or frees memory.
 *   - All work is enqueued on the caller's stream `stream` (a cudaStream_t
 *     passed as void*; NULL = the legacy default stream) and the calls return
 *     without synchronising.  Arguments are validated on the host before any
 *     launch; a call that returns non-zero has enqueued nothing.
 *   - Tensors are dense, row-major, with these layouts (B = batch, L = layers,
 *     Hq query heads, H = hkv KV heads, G = Hq / H, n context, d head dim,
 *     w observation window):
 *         K, V   bf16  [B][L][H][n][d]
 *         Q_obs  bf16  [B][L][Hq][w][d]   the last w prefill queries
 *         q      bf16  [B][L][Hq][d]      one decode query per head
 *     Query head qh reads KV head qh / G.  Observation row t of a query head
 *     sits at absolute position n - w + t and sees keys j <= n - w + t.
 *     Every tensor pointer must be 16-byte aligned (CERTKV_EINVAL otherwise).
 *   - A "unit" is one (sequence, layer, KV head): u = (b * L + l) * H + h.
 *   - Device-side problems (non-finite scores, an evicted suffix with zero
 *     mass) are recorded in a status word inside the workspace; read it with
 *     certkv_read_status().  No kernel traps.
 *   - Supported sizes: d = 128; 1 <= H <= 32; G = Hq / H an integer with
 *     1 <= G <= 16; 1 <= w < n; n <= 2^24; B * L * H <= 2^24.
 */
#ifndef CERTKV_H
#define CERTKV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- return codes -------------------------------------------------------- */
#define CERTKV_OK          0
#define CERTKV_EINVAL      1  /* bad shape, pointer or parameter                 */
#define CERTKV_EBUDGET     2  /* budget infeasible: B_live < 2H or B_live > H*n  */
#define CERTKV_EWORKSPACE  3  /* workspace missing, misaligned or too small      */
#define CERTKV_ECAPACITY   4  /* packed-cache capacity below B * L * B_live      */
#define CERTKV_ECUDA       5  /* a CUDA runtime call failed                      */
#define CERTKV_ETOOLARGE   6  /* problem exceeds the fixed scratch of
                                 certkv_decode_attn_noalloc                     */

/* bits of the device status word returned by certkv_read_status() */
#define CERTKV_STATUS_NONFINITE   1u  /* a score or curve value was NaN/Inf     */
#define CERTKV_STATUS_ZERO_TAIL   2u  /* an evicted suffix had zero mass: its
                                         tail slot is the uniform mean instead */
#define CERTKV_STATUS_TIMEOUT     4u  /* a bounded wait inside a tensor-core
                                         kernel gave up; its outputs are invalid */
#define CERTKV_STATUS_BOUNDS      8u  /* only in a library built with
                                         CERTKV_DEBUG: a ragged index or offset
                                         (a token of the order, a kept position,
                                         a slot, a radix destination, a budget)
                                         was outside its extent; the access was
                                         skipped, the outputs are invalid      */

/* ---- problem description ------------------------------------------------- */
typedef struct {
  int32_t batch;   /* B  sequences                                   */
  int32_t layers;  /* L  layers compressed in this call              */
  int32_t hq;      /* Hq query heads                                 */
  int32_t hkv;     /* H  KV heads                                    */
  int32_t n;       /* context length (cached tokens per KV head)     */
  int32_t d;       /* head dimension (128)                           */
  int32_t w;       /* observation window (last w prefill queries)    */
} certkv_shape;

/* Statistic used for the allocation curve (paper: one-factor ablations). */
#define CERTKV_STAT_CENTERED    0  /* c = sqrt((m Q - ||W||^2)_+)  (default, Eq. certkv-curve) */
#define CERTKV_STAT_UNCENTERED  1  /* c = sqrt(m Q)                                             */
#define CERTKV_STAT_TAIL_MASS   2  /* c = m                                                     */

typedef struct {
  float   scale;          /* softmax scale for <q,k>; 0 selects 1/sqrt(d)            */
  int32_t pool_kernel;    /* observation-score average-pool width, odd >= 1; 5 default;
                             zero padding, divided by the width, window keys excluded  */
  int32_t protect_window; /* 1 (default): the w window keys get the head's maximum
                             pooled score; 0: their own mean causal probability       */
  int32_t alpha_num;      /* safeguard alpha = alpha_num / alpha_den (default 1 / 5), */
  int32_t alpha_den;      /*   0 <= alpha <= 1, exact rational                        */
  int32_t bisect_steps;   /* T, number of bisection steps (default 40), 0..200        */
  int32_t statistic;      /* CERTKV_STAT_* (default CERTKV_STAT_CENTERED)             */
  int32_t tail_slot;      /* 1 (default): one synthetic tail slot per head is charged
                             to the budget; 0: no slot, the slot goes to a real token */
  int32_t allocator;      /* CERTKV_ALLOC_* (default CERTKV_ALLOC_LAGRANGIAN)          */
  int32_t tail_clusters;  /* m >= 0 (default 0): cluster summaries of each head's evicted
                             tail, for certkv_decode_certified; each costs one slot of
                             the budget (B_real = B_live - H (tail_slot + m)); at most
                             CERTKV_MAX_CLUSTERS                                       */
} certkv_params;

#define CERTKV_MAX_CLUSTERS 64

/* Cross-head allocator (paper: one-factor ablations, "Allocator" block).  The
 * paper names the two ablations without defining them; the readings used:
 * UNIFORM gives every head floor(B_real / H) real tokens and one more to each
 * of the lowest (B_real mod H) heads; GREEDY starts every head at b_min and
 * adds one token at a time to the head with the smallest c_h(b_h+1) - c_h(b_h)
 * (lowest head on ties), the repair rule of Algorithm 1 run from b_min. */
#define CERTKV_ALLOC_LAGRANGIAN 0  /* T-step bisection on lambda + repair (Algorithm 1) */
#define CERTKV_ALLOC_UNIFORM    1
#define CERTKV_ALLOC_GREEDY     2

/* Ragged packed cache.  Segment u (one per unit) holds real_counts[u] real
 * slots in ascending original position followed, when params.tail_slot = 1,
 * by the tail slot, then, when params.tail_clusters = m > 0, by m cluster
 * summary slots (positions -2 - g; k, v = the bf16-rounded unweighted means of
 * cluster g of the evicted ranks, which is ranks b + floor(g T / m) ..
 * b + floor((g + 1) T / m) - 1 with T = n - b); offsets[u] is its first slot.
 * Each (sequence, layer) owns exactly B_live consecutive slots:
 * offsets[(b*L+l)*H] = (b*L+l)*B_live. */
typedef struct {
  void*    k;               /* bf16 [capacity_slots][d]                          */
  void*    v;               /* bf16 [capacity_slots][d]                          */
  int64_t* offsets;         /* [B*L*H + 1] first slot of each segment            */
  int32_t* real_counts;     /* [B*L*H] b_h, real slots per segment               */
  int32_t* positions;       /* [capacity_slots] original token index; -1 = tail  */
  int64_t  capacity_slots;  /* slots available in k, v and positions             */
  float*   tail_f32;        /* optional (NULL = skip) [B*L*H][2][d]: k*, v* in fp32
                               before rounding to bf16                            */
  double*  tail_mass;       /* optional (NULL = skip) [B*L*H]: m_h(b_h)          */
  float*   cluster_meta;    /* with params.tail_clusters = m > 0 (else NULL):
                               [B*L*H][m][4] = (count n_g, key radius R_g, value
                               radius rho_g, 0) of each cluster summary slot     */
  float*   kept_vmax;       /* with m > 0: [B*L*H] largest ||v|| of the real slots */
} certkv_packed;

/* Fill `p` with the defaults listed above.  Host call. */
void certkv_default_params(certkv_params* p);

/* Live-slot budget of the paper's exact-budget protocol for a kept fraction
 * keep_num / keep_den: H * floor(n * keep_num / keep_den), computed in exact
 * integer arithmetic (the paper writes B_live = H floor(n (1 - r)) for an
 * evicted fraction r).  Returns -1 for invalid arguments.  Host call. */
int64_t certkv_live_budget(int32_t n, int32_t hkv, int64_t keep_num, int64_t keep_den);

/* Workspace bytes needed by certkv_compress / certkv_compress_scored /
 * certkv_score / certkv_curves for this shape (an upper bound for all four),
 * and by certkv_decode_attn.  0 if the shape or parameters are invalid. */
size_t certkv_workspace_bytes(const certkv_shape* shape, const certkv_params* params);
size_t certkv_decode_workspace_bytes(const certkv_shape* shape);

/* a1-a2: observation-window scores.  a_out: fp32 [B*L*H][n], each row a
 * probability vector (a_j >= 0, sum 1) — §4 and the implementation appendix
 * ("we normalize directly, rather than re-softmaxing").  K: bf16 as above;
 * Q_obs: bf16 [B][L][Hq][w][d]. */
int certkv_score(const certkv_shape* shape, const void* K, const void* Q_obs,
                 const certkv_params* params, float* a_out,
                 void* workspace, size_t workspace_bytes, void* stream);

/* a3-a4: per-unit order and allocation curve, exposed for inspection.
 * a: fp32 [B*L*H][n] scores (e.g. from certkv_score); V bf16 as above.
 * perm_out: int32 [B*L*H][n], perm_out[u][r] = token at rank r (rank 0 =
 * highest score, ties by lower index).  c_out: fp64 [B*L*H][n],
 * c_out[u][b] = c_h(b) for the evicted suffix of ranks b..n-1 (Algorithm 1,
 * suffix-scan and curve lines). */
int certkv_curves(const certkv_shape* shape, const void* V, const float* a,
                  const certkv_params* params, int32_t* perm_out, double* c_out,
                  void* workspace, size_t workspace_bytes, void* stream);

/* a3-a8 from given scores `a` (fp32 [B*L*H][n], e.g. from certkv_score):
 * order, curves, exact-budget allocation, selection, tail slot and packing.
 * budget_live = B_live, live slots per (sequence, layer); it must satisfy
 * 2H <= B_live <= H*n when tail_slot = 1 and H <= B_live <= H*n when
 * tail_slot = 0 (else CERTKV_EBUDGET). */
int certkv_compress_scored(const certkv_shape* shape, const void* K, const void* V,
                           const float* a, int64_t budget_live,
                           const certkv_params* params, certkv_packed* out,
                           void* workspace, size_t workspace_bytes, void* stream);

/* a1-a8: the whole compression pass (Algorithm 1 with the observation-window
 * scorer in front).  Same contract as certkv_compress_scored. */
int certkv_compress(const certkv_shape* shape, const void* K, const void* V,
                    const void* Q_obs, int64_t budget_live,
                    const certkv_params* params, certkv_packed* out,
                    void* workspace, size_t workspace_bytes, void* stream);

/* a1-a8 from HOST inputs, with the host->device copies overlapped with the
 * compression (a runtime convenience; the paper's method is certkv_compress).
 * hK, hV, hQ_obs: host memory in the layouts above; page-locked (pinned)
 * memory makes the copies asynchronous, pageable memory works but its copies
 * block the calling thread.  The (sequence, layer) pairs are processed
 * `chunk` at a time (0: about 1 GiB of K and V per chunk): chunk c + 1 is
 * copied into the other half of a double-buffered staging area inside the
 * workspace, on a stream of the library's own, while chunk c compresses on
 * `stream`.  Each pair is compressed independently, so `out` (device memory,
 * as for certkv_compress) receives exactly what certkv_compress writes for the
 * whole problem.  The host buffers must stay valid and unchanged until the
 * work enqueued on `stream` has finished.  Workspace:
 * certkv_host_workspace_bytes(shape, params, chunk) bytes, 256-byte aligned;
 * certkv_read_status reads it as for the other entry points.  Returns the
 * codes of certkv_compress; CERTKV_EINVAL also for chunk < 0. */
size_t certkv_host_workspace_bytes(const certkv_shape* shape, const certkv_params* params,
                                   int32_t chunk);
int certkv_compress_host(const certkv_shape* shape, const void* hK, const void* hV,
                         const void* hQ_obs, int64_t budget_live, const certkv_params* params,
                         int32_t chunk, certkv_packed* out, void* workspace,
                         size_t workspace_bytes, void* stream);

/* certkv_compress_host, with the packed cache also copied back to host memory
 * chunk by chunk (a runtime convenience): as soon as a chunk of (sequence,
 * layer) pairs is compressed, its slots [bl0 * budget_live, (bl0 + cnt) *
 * budget_live) of k, v and positions, and its entries of real_counts and
 * offsets (with the final offset after the last chunk), are copied to
 * `host_out` on a third stream of the library's own, so that these copies run
 * while later chunks are copied in and compressed.  `out` (device memory)
 * receives the same as from certkv_compress_host.  host_out: k, v,
 * real_counts, offsets and positions are HOST pointers sized as out's
 * (page-locked memory for asynchronous copies); its other fields are ignored
 * (the optional device outputs of `out` are not copied back).  The copies
 * complete on `stream`, like the rest of the call.  Workspace and return
 * codes as for certkv_compress_host; CERTKV_EINVAL also when host_out or one
 * of its five pointers is NULL, or when host_out->capacity_slots is below
 * budget_live * batch * layers. */
int certkv_compress_host_copyback(const certkv_shape* shape, const void* hK, const void* hV,
                                  const void* hQ_obs, int64_t budget_live,
                                  const certkv_params* params, int32_t chunk, certkv_packed* out,
                                  certkv_packed* host_out, void* workspace,
                                  size_t workspace_bytes, void* stream);

/* a9: decode attention over the packed cache: for every query head qh of
 * unit u = (b, l, qh / G), out[b][l][qh] = sum_s softmax_s(scale <q, k_s>) v_s
 * over the real_counts[u] (+ 1 tail) slots of segment u.  q, out: bf16
 * [B][L][Hq][d].  `packed` must come from certkv_compress* with the same
 * shape and tail_slot; scale 0 selects 1/sqrt(d). */
int certkv_decode_attn(const certkv_shape* shape, const void* q,
                       const certkv_packed* packed, float scale, int32_t tail_slot,
                       void* out, void* workspace, size_t workspace_bytes,
                       void* stream);

/* Clustered-tail decode with its runtime output-error bound (appendix:
 * deterministic output-error bound for clustered tail summaries, theorem and
 * runtime remark).  For each query head: O-hat = (sum over the real slots of
 * e^l v + sum_g n_g e^{lbar_g} vbar_g) / Z-hat with lbar_g = scale <q, kbar_g>
 * (the plain tail slot, if present, is not used), and
 * bound = (3 / Z-hat) (D_N + V'max D_Z), D_Z = sum_g (e^{r_g} - 1) e^{r_g} Zhat_g,
 * D_N = sum_g e^{r_g} Zhat_g ((e^{r_g} - 1) ||vbar_g|| + rho_g),
 * V'max = max(kept_vmax, max_g ||vbar_g|| + rho_g), with logit radius
 * r_g = scale ||q|| R_g (Cauchy-Schwarz).  certified = 1 when D_Z <= Z-hat / 3,
 * the condition under which ||O-hat - O|| <= bound for exact attention O over
 * every original token.  packed comes from a compression with
 * params.tail_clusters = clusters and params.tail_slot = tail_slot.
 * out: bf16 [B][L][Hq][d]; bound: fp32 [B][L][Hq]; certified: int32 [B][L][Hq].
 * Workspace: certkv_decode_workspace_bytes(shape). */
int certkv_decode_certified(const certkv_shape* shape, const void* q, const certkv_packed* packed,
                            float scale, int32_t tail_slot, int32_t clusters, void* out,
                            float* bound, int32_t* certified, void* workspace,
                            size_t workspace_bytes, void* stream);

/* Fixed-row diagnostics (an evaluation tool: it reads the full original K and
 * V, like the paper's fixed-row experiments).  For every query head qh of unit
 * u with its decode query q, the realized logits z_j = scale <q, k_j> and
 * softmax row A_j over all n original tokens, S = the real tokens kept in
 * `packed` and T = the evicted ones, writes stats fp32
 * [B][L][Hq][CERTKV_FIXED_ROW_STATS]:
 *   Theorem (fixed-row tail factorization):
 *   0  p_S = sum_{j in S} A_j (kept mass)
 *   1  ||O||_2 of exact attention O = sum_j A_j v_j
 *   2  ||O~_S - O||_2, O~_S = sum_{j in S} A_j v_j / p_S (subset-only output)
 *   3  ||u*||_2, u* = sum_{j in T} A_j v_j (the fixed-row correction)
 *   4  2 V_max (1 - p_S), V_max = max_j ||v_j||_2 (the theorem's mass bound)
 *   5  ||O-hat - O||_2 for O-hat = certkv_decode_attn(q, packed, tail_slot)
 *   6  V_max
 *   7  ||p_S O~_S + (1 - p_S) V-bar_T - O||_2, the factorization residual
 *   Theorem (future-query lift and summary mismatch), with Ahat the softmax
 *   over S and the synthetic slot (logit z* = scale <q, k*>), and the slot's
 *   tail weights r_j = s_j / sum_T s (uniform 1/|T| when that sum is 0):
 *   8  p = A(T), the tail mass (computed from the evicted tokens, not 1 - p_S)
 *   9  q = Ahat_star, the slot's compressed weight (0 when tail_slot = 0)
 *   10 ||a - r||_1 over T, a = A_T / p (a = 0 when p = 0)
 *   11 Lambda_T - z*, Lambda_T = log sum_{j in T} e^{z_j} (NaN without a slot)
 *   12 V_max (2 |p - q| + min(p, q) ||a - r||_1), the theorem's bound on
 *      ||O - O-hat|| for a slot value equal to the r-mixture
 *   13 tanh(|Lambda_T - z*| / 4), the theorem's bound on |p - q| (NaN without a slot)
 *   14 ||A - Abar||_1 for the lifted row Abar (Ahat on S, q r_j on T)
 *   15 ||v*_stored - sum_T r_j v_j||_2, the packed slot value against the
 *      exact mixture (bf16 rounding; NaN without a slot or when sum_T s = 0)
 * Fields 10, 12, 14 and 15 need `scores` (fp32 [B*L*H][n], the a_j the
 * compression used, e.g. from certkv_score with the same inputs and params);
 * with scores = NULL they are NaN.  q bf16 [B][L][Hq][d]; K, V as for
 * certkv_compress; workspace: certkv_fixed_row_workspace_bytes(shape) (it
 * holds every logit, 4 (B*L*Hq) n bytes). */
#define CERTKV_FIXED_ROW_STATS 16
size_t certkv_fixed_row_workspace_bytes(const certkv_shape* shape);
int certkv_fixed_row_stats(const certkv_shape* shape, const void* q, const void* K, const void* V,
                           const float* scores, const certkv_packed* packed, float scale,
                           int32_t tail_slot, float* stats, void* workspace,
                           size_t workspace_bytes, void* stream);

/* Sampled tail compensation (an evaluation tool over the full K and V; appendix:
 * proposition on sampled tail compensation).  For every query head qh of unit
 * u with its decode query q, the realized softmax row A over all n original
 * tokens, S = the real tokens kept in `packed` and T the N evicted ones, the
 * fixed-row correction u* = sum_T A_j v_j is estimated from m tail tokens:
 *   weight-proportional: token j_r (r < m) is the first evicted token, in
 *     index order, whose cumulative tail weight exceeds unif[r] * A(T) (the
 *     cumulative weight summed in float64); u_w = (1 - p_S)/m sum_r v_{j_r}
 *   uniform subset: Floyd's algorithm over the tail ranks, for i = N - m .. N - 1
 *     rank floor(unif[m + i - N + m] * (i + 1)) unless already taken, else i
 *     (float64 products); u_u = (1 - p_S)/m sum of the subset's values.
 * unif: fp32 [B][L][Hq][2m] uniforms in [0, 1) (device); idx_out: int32
 * [B][L][Hq][2m] the drawn token indices (may be NULL); stats fp32
 * [B][L][Hq][8]: 0 p_S, 1 Q_T = sum_T A_j^2, 2 ||u*||, 3 ||u_w - u*||,
 * 4 ||u_u - u*||, 5 the proposition's root-mean-square error of u_w,
 * sqrt(d s2 (1 - p_S)^2/m (1 - Q_T/(1 - p_S)^2)), 6 that of u_u,
 * sqrt(d s2 (1 - p_S)^2 (1/m - 2/N + Q_T/(1 - p_S)^2)), 7 s2 = the evicted
 * values' per-coordinate variance (standing for sigma_V^2).  1 <= m <=
 * CERTKV_MAX_SAMPLES; a head with fewer than m evicted tokens gets NaN stats
 * and -1 indices.  q bf16 [B][L][Hq][d]; K, V as for certkv_compress;
 * workspace: certkv_sampled_workspace_bytes(shape). */
#define CERTKV_MAX_SAMPLES 64
size_t certkv_sampled_workspace_bytes(const certkv_shape* shape);
int certkv_sampled_compensation(const certkv_shape* shape, const void* q, const void* K,
                                const void* V, const certkv_packed* packed, float scale,
                                int32_t m, const float* unif, int32_t* idx_out, float* stats,
                                void* workspace, size_t workspace_bytes, void* stream);

/* Coverage profile of realized query rows (an evaluation instrument: §3,
 * "count sparsity does not imply coverage sparsity", with the ranked gap
 * profile G(j) = z_(1) - z_(j) and the coverage budget K_eta; the appendix's
 * gap-profile instrument recomputes the row logits in fp32, as here).  One row
 * per query head qh of each (sequence, layer), over the n keys of KV head
 * qh / G: z_j = scale <q, k_j> (fp32), A = softmax(z), pi the order of the
 * logits, descending, ties by lower index.  Per row r = (b L + l) Hq + qh:
 *   K_eta[r][e]      = min{k : sum_{j <= k} A_(j) >= 1 - eta[e]}  (int32)
 *   rel_counts[r][e] = #{j : A_j > rel_eps[e] A_(1)}  (relative-weight count)
 *   abs_counts[r][e] = #{j : A_j > abs_eps[e]}        (calibrated count k(eps))
 *   top[r][0] = z_(1), top[r][1] = log sum_j e^{z_j}  (fp32)
 *   order[r][i] = pi(i + 1), the token at rank i (int32 [rows][n], may be NULL)
 *   gap[r][i]   = G(i + 1) (fp32 [rows][n], may be NULL)
 * The ranked mass is summed in float64 in one fixed order from fp32 weights
 * e^{z_(j) - z_(1)}; the counts compare fp32 logit differences with log eps.
 * eta, rel_eps, abs_eps: HOST arrays of n_eta, n_rel, n_abs values (each count
 * 0..CERTKV_COVERAGE_MAX_THRESHOLDS; 0 < eta < 1; eps > 0, finite); an output
 * array may be NULL when its count is 0.  q bf16 [B][L][Hq][d], K bf16 as for
 * certkv_compress; scale 0 selects 1/sqrt(d).  Workspace:
 * certkv_coverage_workspace_bytes(shape) (16 n bytes per row plus the sort's
 * tile histograms). */
#define CERTKV_COVERAGE_MAX_THRESHOLDS 16
size_t certkv_coverage_workspace_bytes(const certkv_shape* shape);
int certkv_coverage_profile(const certkv_shape* shape, const void* q, const void* K, float scale,
                            const double* eta, int32_t n_eta, const double* rel_eps,
                            int32_t n_rel, const double* abs_eps, int32_t n_abs, int32_t* K_eta,
                            int32_t* rel_counts, int32_t* abs_counts, float* top, int32_t* order,
                            float* gap, void* workspace, size_t workspace_bytes, void* stream);

/* Decode attention that allocates nothing.  The paper has no counterpart: this
 * entry point exists for callers that cannot hand the library a scratch
 * buffer, for example a plugin that an inference server gives only its input
 * and output tensors, or a per-token decode loop that must not call cudaMalloc
 * because cudaMalloc can wait for the whole device and breaks a memory plan
 * fixed at start-up.  It computes exactly what certkv_decode_attn computes
 * (same kernels, same arguments minus the workspace); its split-K scratch is a
 * fixed array of CERTKV_NOALLOC_SCRATCH_BYTES in the library's own device
 * memory, present on every GPU that loads the library until the process exits.
 *   - Limit: certkv_decode_workspace_bytes(shape) must fit in the array: with
 *     U = B * L * H, 4 (U + 1) bytes of tile offsets and (U + 1024) * G split
 *     records of 520 bytes, about (U + 1024) * G <= 32000 (eight 32-layer,
 *     8-KV-head, G = 4 sequences per call); larger calls return
 *     CERTKV_ETOOLARGE and enqueue nothing.  Split a larger batch into
 *     several calls.
 *   - The first call on each device looks up the array's device address (with
 *     that device current); make that first call before any stream capture.
 *   - Every call on a device shares the one array, and each call rewrites every
 *     scratch record before reading it, so nothing has to start at zero; calls
 *     that overlap on the GPU (different streams, threads or processes sharing
 *     the context) race on the array: order them, e.g. on one stream.
 *   - No cudaMalloc, cudaFree or allocating library routine is called.
 * Returns CERTKV_OK, CERTKV_EINVAL, CERTKV_ETOOLARGE or CERTKV_ECUDA. */
#define CERTKV_NOALLOC_SCRATCH_BYTES (16u << 20)
int certkv_decode_attn_noalloc(const certkv_shape* shape, const void* q,
                               const certkv_packed* packed, float scale, int32_t tail_slot,
                               void* out, void* stream);

/* Guard words of a compression workspace (a debugging aid with no
 * counterpart in the paper).  Every region of the workspace that
 * certkv_workspace_bytes(shape, params) describes is followed by 16 bytes of
 * padding that no kernel writes.  certkv_workspace_guard_arm fills them with a
 * fixed pattern (asynchronously, on `stream`); after any number of
 * certkv_score / certkv_curves / certkv_compress_scored / certkv_compress
 * calls with the same shape and params on that workspace,
 * certkv_workspace_guard_check synchronises `stream` and returns how many
 * guards no longer hold the pattern: 0 means no kernel wrote past the end of
 * its region.  Both return -1 for an invalid shape, params or workspace (NULL,
 * misaligned or smaller than certkv_workspace_bytes) or a CUDA error; the
 * check also writes the count into the status region (it does not change the
 * status word). */
int certkv_workspace_guard_arm(const certkv_shape* shape, const certkv_params* params,
                               void* workspace, size_t workspace_bytes, void* stream);
int certkv_workspace_guard_check(const certkv_shape* shape, const certkv_params* params,
                                 void* workspace, size_t workspace_bytes, void* stream);

/* Self-test of the bounded waits the kernels use (a debugging aid with no
 * counterpart in the paper): one thread waits on an mbarrier that nothing
 * arrives on, with no copy and no MMA in flight.  The wait must give up after
 * its poll limit (a few seconds at most) and report a timeout without any
 * fault.  Synchronises `stream` and returns CERTKV_STATUS_TIMEOUT when it
 * did; -2 if the wait did not give up as designed; -1 on a CUDA error.  Its
 * result sits in a small array of the library's own device memory: calls
 * that overlap on the GPU race on it. */
int certkv_selftest_bounded_wait(void* stream);

/* Synchronise `stream`, then return the device status word (CERTKV_STATUS_*
 * bits, 0 = clean) that the last compress call on `workspace` left, or -1 if
 * a CUDA call failed.  Host pointer args: none. */
int certkv_read_status(const void* workspace, void* stream);

/* Profiling aid, not part of the paper's method: when enabled (on = 1) every
 * kernel launch of the library is bracketed by two CUDA events recorded on
 * its stream (a pool of events is created once, by the first enable call on
 * the current device); certkv_trace_report() synchronises, writes one line
 * "name launches total_ms" per kernel into the host buffer `buf` (len bytes),
 * clears the records and returns the bytes written, or -1 if the buffer is too
 * small or a CUDA call failed.  certkv_trace_enable returns CERTKV_OK or
 * CERTKV_ECUDA. */
int certkv_trace_enable(int on);
int certkv_trace_report(char* buf, size_t len);

/* Static description of a return code. */
const char* certkv_strerror(int code);

#ifdef __cplusplus
}
#endif
#endif /* CERTKV_H */
