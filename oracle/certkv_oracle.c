/*
 * certkv_oracle.c — TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, float64 CPU restatement of the CertKV compression pass and of
 * decode attention over its packed cache, written from "Beyond Sparse Weights:
 * When Is Attention Compressible?" (§4, Eq. (certkv-curve), Algorithm 1 and the
 * appendix "CertKV: implementation and exact-budget protocol").  It exists to
 * check the CUDA library against; only the tests, the package's smoke check and
 * the benchmark's CPU-baseline leg may load it.  It shares no code, header or
 * table with the CUDA library.
 *
 * Every step is written in the paper's order with naive loops; the only library
 * primitive is qsort (the per-head sort).  Inputs are the raw bf16 bytes the
 * GPU consumed, widened exactly to float64.  Readings of points where the paper
 * is silent are marked READING and listed in the design notes:
 *   R-A1 scorer constants (mean over the G*w observation rows; causal mask in
 *        the window; average pool of width `pool`, zero padding, divided by the
 *        width, over non-window keys only; window keys get the unit's maximum
 *        pooled score);
 *   R-A2 ties in the order are broken by the lower token index;
 *   R-A3 b counts kept tokens, the evicted suffix E(b) is ranks b..n-1;
 *   R-A5/A6 B_live is given as an integer, alpha as an exact rational;
 *   R-A7 lambda_hi = 2 max over every b in [0, n-1] and every head + 1;
 *   R-A8 argmin ties go to the smallest b;
 *   R-A9 repair adds one token to the head with the smallest marginal
 *        c(b+1) - c(b) (lowest head index on ties), or, for a surplus, removes
 *        one from the head with the smallest c(b-1) - c(b);
 *   R-A10 the tail slot stores the centroids k* = sum a k / m, v* = sum a v / m;
 *   R-A11 if m == 0 in floating point the slot is the uniform tail mean;
 *   R-A12 the tail slot enters decode as a plain key/value pair (no logit bias);
 *   R-A15 / R-A16 the "true uniform" and "greedy marginal" allocator ablations
 *        (see oracle_allocate_mode).
 *
 * Build: cc -O2 -ffp-contract=off -fPIC -shared (no fused multiply-add, so that
 * x86 and Arm builds round identically).
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* ---------------------------------------------------------------- bf16 ---- */

static double bf16_to_f64(uint16_t h) {
  uint32_t u = (uint32_t)h << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

/* Round a double to the nearest bf16, ties to even, in one rounding step. */
uint16_t oracle_f64_to_bf16(double x) {
  uint16_t sign = signbit(x) ? 0x8000u : 0u;
  double ax = fabs(x);
  if (isnan(x)) return (uint16_t)(sign | 0x7FC0u);
  if (isinf(x)) return (uint16_t)(sign | 0x7F80u);
  if (ax == 0.0) return sign;
  const double min_normal = ldexp(1.0, -126);
  if (ax < min_normal) {
    /* subnormal bf16: quantum 2^-133 */
    double r = nearbyint(ldexp(ax, 133)); /* default rounding: to nearest even */
    return (uint16_t)(sign | (uint16_t)r); /* r == 128 encodes the min normal */
  }
  int e;
  double f = frexp(ax, &e);          /* ax = f * 2^e, f in [0.5, 1) */
  double r = nearbyint(ldexp(f, 8)); /* 8 significant bits: r in [128, 256] */
  if (r == 256.0) { r = 128.0; e += 1; }
  int biased = e - 1 + 127;          /* value = (r/128) * 2^(e-1) */
  if (biased >= 255) return (uint16_t)(sign | 0x7F80u);
  return (uint16_t)(sign | (uint16_t)(biased << 7) | (uint16_t)((int)r - 128));
}

/* ------------------------------------------------------------- scoring ---- */

/*
 * Observation-window scores of one unit (a1-a2; §4 "SnapKV's observation-window
 * score", implementation appendix: a_j = (s_j)_+ / sum_i (s_i)_+).
 *   K  [n][d]  keys of KV head h;  Qg [G][w][d] observation queries of the G
 *   query heads that read h.  Writes a[n] (float64).  Returns 0.
 */
int oracle_scores(const uint16_t* K, const uint16_t* Qg, int n, int d, int w, int G,
                  double scale, int pool, int protect, double* a) {
  const int R = G * w;
  const int nw = n - w; /* keys outside the observation window */
  double* s = (double*)calloc((size_t)n, sizeof(double));
  double* logit = (double*)malloc((size_t)n * sizeof(double));
  double* qrow = (double*)malloc((size_t)d * sizeof(double));
  double* st = (double*)malloc((size_t)n * sizeof(double));
  if (!s || !logit || !qrow || !st) { free(s); free(logit); free(qrow); free(st); return -1; }

  for (int g = 0; g < G; ++g) {
    for (int t = 0; t < w; ++t) {
      const uint16_t* q = Qg + ((size_t)g * w + t) * d;
      for (int i = 0; i < d; ++i) qrow[i] = bf16_to_f64(q[i]);
      const int visible = nw + t + 1; /* causal: row at position n-w+t sees j <= n-w+t */
      double mx = -INFINITY;
      for (int j = 0; j < visible; ++j) {
        const uint16_t* k = K + (size_t)j * d;
        double dot = 0.0;
        for (int i = 0; i < d; ++i) dot += qrow[i] * bf16_to_f64(k[i]);
        logit[j] = scale * dot;
        if (logit[j] > mx) mx = logit[j];
      }
      double sum = 0.0;
      for (int j = 0; j < visible; ++j) sum += exp(logit[j] - mx);
      const double lse = mx + log(sum);
      for (int j = 0; j < visible; ++j) s[j] += exp(logit[j] - lse);
    }
  }
  for (int j = 0; j < n; ++j) s[j] /= (double)R; /* mean over the R observation rows */

  /* average pool over the non-window keys, zero padding, divided by the width */
  const int half = pool / 2;
  double smax = -INFINITY;
  for (int j = 0; j < nw; ++j) {
    double acc = 0.0;
    for (int i = j - half; i <= j + half; ++i)
      if (i >= 0 && i < nw) acc += s[i];
    st[j] = acc / (double)pool;
    if (st[j] > smax) smax = st[j];
  }
  for (int j = nw; j < n; ++j) st[j] = protect ? smax : s[j];

  double total = 0.0;
  for (int j = 0; j < n; ++j) total += (st[j] > 0.0 ? st[j] : 0.0);
  for (int j = 0; j < n; ++j) a[j] = (st[j] > 0.0 ? st[j] : 0.0) / total;

  free(s); free(logit); free(qrow); free(st);
  return 0;
}

/* ------------------------------------------------------------- order ----- */

typedef struct { double a; int32_t j; } scored_t;

static int cmp_desc_then_index(const void* x, const void* y) {
  const scored_t* p = (const scored_t*)x;
  const scored_t* q = (const scored_t*)y;
  if (p->a > q->a) return -1;
  if (p->a < q->a) return 1;
  return (p->j < q->j) ? -1 : (p->j > q->j);
}

/* a3: perm[r] = token at rank r, scores descending, ties by lower index. */
void oracle_order(const double* a, int n, int32_t* perm) {
  scored_t* tmp = (scored_t*)malloc((size_t)n * sizeof(scored_t));
  for (int j = 0; j < n; ++j) { tmp[j].a = a[j]; tmp[j].j = j; }
  qsort(tmp, (size_t)n, sizeof(scored_t), cmp_desc_then_index);
  for (int r = 0; r < n; ++r) perm[r] = tmp[r].j;
  free(tmp);
}

/* ------------------------------------------------------------- curves ---- */

/*
 * a4: allocation curve of one unit (implementation appendix: suffix moments
 * m(b) = sum a_j, W(b) = sum a_j v_j, Q(b) = sum a_j ||v_j||^2 over the evicted
 * ranks b..n-1, and c(b)^2 = (m(b) Q(b) - ||W(b)||^2)_+ ; Eq. (certkv-curve)).
 * statistic 0: centred, 1: sqrt(m Q) (uncentred ablation), 2: m (tail mass).
 */
void oracle_curve(const double* a, const uint16_t* V, const int32_t* perm, int n, int d,
                  int statistic, double* c) {
  double* W = (double*)calloc((size_t)d, sizeof(double));
  double m = 0.0, Q = 0.0;
  for (int b = n - 1; b >= 0; --b) {
    const int j = perm[b];
    const double aj = a[j];
    const uint16_t* v = V + (size_t)j * d;
    double vv = 0.0;
    for (int i = 0; i < d; ++i) {
      const double x = bf16_to_f64(v[i]);
      W[i] += aj * x;
      vv += x * x;
    }
    m += aj;
    Q += aj * vv;
    if (statistic == 2) { c[b] = m; continue; }
    if (statistic == 1) { c[b] = sqrt(m * Q); continue; }
    double ww = 0.0;
    for (int i = 0; i < d; ++i) ww += W[i] * W[i];
    const double c2 = m * Q - ww;
    c[b] = sqrt(c2 > 0.0 ? c2 : 0.0);
  }
  free(W);
}

/* ---------------------------------------------------------- allocation ---- */

/* b_min of the exact-budget protocol: max{1, floor(alpha * B_real / H)}. */
int64_t oracle_b_min(int64_t B_real, int H, int64_t alpha_num, int64_t alpha_den) {
  int64_t v = (alpha_num * B_real) / (alpha_den * (int64_t)H);
  return v < 1 ? 1 : v;
}

/* smallest argmin over b in [lo, hi] of c[b] + lambda * b */
static int argmin_penalised(const double* c, int lo, int hi, double lambda) {
  int best_b = lo;
  double best = c[lo] + lambda * (double)lo;
  for (int b = lo + 1; b <= hi; ++b) {
    const double f = c[b] + lambda * (double)b;
    if (f < best) { best = f; best_b = b; }
  }
  return best_b;
}

/*
 * a5: split B_real real-token slots across H heads (Algorithm 1: b_min,
 * lambda bisection for T steps, b_h = b_h(lambda_hi), then one-token repair).
 * curves[h] points at c_h(0..n-1).  B_real is the real-token budget (B_live - H
 * when one tail slot per head is charged).  Writes b[H]; *repairs = number of
 * one-token repairs.  Returns 0, or 2 if the budget is infeasible.
 */
int oracle_allocate_mode(const double* const* curves, int H, int n, int64_t B_real,
                         int64_t alpha_num, int64_t alpha_den, int T, int mode, int32_t* b,
                         int64_t* repairs);

int oracle_allocate(const double* const* curves, int H, int n, int64_t B_real,
                    int64_t alpha_num, int64_t alpha_den, int T, int32_t* b,
                    int64_t* repairs) {
  return oracle_allocate_mode(curves, H, n, B_real, alpha_num, alpha_den, T, 0, b, repairs);
}

/*
 * The one-factor allocator ablations (ablation table, "Allocator" block),
 * with `mode`:
 *   0  Lagrangian bisection + repair (the method, above);
 *   1  true uniform: READING R-A15, b_h = floor(B_real / H), the remainder
 *      going one token each to the lowest-index heads;
 *   2  greedy marginal: READING R-A16, every head starts at b_min and the
 *      repair rule above (smallest c_h(b_h+1) - c_h(b_h), lowest head on
 *      ties) adds one token at a time until B_real.
 */
int oracle_allocate_mode(const double* const* curves, int H, int n, int64_t B_real,
                         int64_t alpha_num, int64_t alpha_den, int T, int mode, int32_t* b,
                         int64_t* repairs) {
  const int64_t bmin = oracle_b_min(B_real, H, alpha_num, alpha_den);
  if (B_real < (int64_t)H * bmin || B_real > (int64_t)H * (n - 1)) return 2;
  const int lo_b = (int)bmin, hi_b = n - 1;
  if (mode == 1) {
    for (int h = 0; h < H; ++h) b[h] = (int32_t)(B_real / H + (h < B_real % H ? 1 : 0));
    if (repairs) *repairs = 0;
    return 0;
  }

  double cmax = 0.0;
  for (int h = 0; h < H; ++h)
    for (int bb = 0; bb < n; ++bb)
      if (curves[h][bb] > cmax) cmax = curves[h][bb];
  double lam_lo = 0.0, lam_hi = 2.0 * cmax + 1.0;

  int64_t total = 0;
  if (mode == 2) {
    for (int h = 0; h < H; ++h) b[h] = lo_b;
    total = (int64_t)H * lo_b;
  } else {
    for (int t = 0; t < T; ++t) {
      const double lam = (lam_lo + lam_hi) / 2.0;
      total = 0;
      for (int h = 0; h < H; ++h) total += argmin_penalised(curves[h], lo_b, hi_b, lam);
      if (total > B_real) lam_lo = lam; else lam_hi = lam;
    }
    total = 0;
    for (int h = 0; h < H; ++h) {
      b[h] = argmin_penalised(curves[h], lo_b, hi_b, lam_hi);
      total += b[h];
    }
  }
  int64_t steps = 0;
  while (total < B_real) { /* best-marginal repair: add one token */
    int best_h = -1;
    double best = INFINITY;
    for (int h = 0; h < H; ++h) {
      if (b[h] >= hi_b) continue;
      const double delta = curves[h][b[h] + 1] - curves[h][b[h]];
      if (best_h < 0 || delta < best) { best = delta; best_h = h; }
    }
    b[best_h] += 1; total += 1; steps += 1;
  }
  while (total > B_real) { /* surplus (not reachable from lambda_hi): remove one */
    int best_h = -1;
    double best = INFINITY;
    for (int h = 0; h < H; ++h) {
      if (b[h] <= lo_b) continue;
      const double delta = curves[h][b[h] - 1] - curves[h][b[h]];
      if (best_h < 0 || delta < best) { best = delta; best_h = h; }
    }
    b[best_h] -= 1; total -= 1; steps += 1;
  }
  if (repairs) *repairs = steps;
  return 0;
}

/* --------------------------------------------------- selection and tail ---- */

static int cmp_int32(const void* x, const void* y) {
  const int32_t p = *(const int32_t*)x, q = *(const int32_t*)y;
  return (p > q) - (p < q);
}

/* a6: kept set = ranks 0..b-1, emitted in ascending token position. */
void oracle_select(const int32_t* perm, int b, int32_t* kept) {
  memcpy(kept, perm, (size_t)b * sizeof(int32_t));
  qsort(kept, (size_t)b, sizeof(int32_t), cmp_int32);
}

/*
 * a7: synthetic tail pair over the evicted ranks b..n-1 (§4: r_j = a_j / m,
 * (k*, v*) = E_{j~r}[(k_j, v_j)]).  Writes kstar[d], vstar[d]; returns m, and
 * sets *zero_mass when m == 0 (then the uniform tail mean is stored).
 */
double oracle_tail(const double* a, const uint16_t* K, const uint16_t* V,
                   const int32_t* perm, int n, int d, int b, double* kstar,
                   double* vstar, int* zero_mass) {
  double m = 0.0;
  for (int i = 0; i < d; ++i) { kstar[i] = 0.0; vstar[i] = 0.0; }
  for (int r = b; r < n; ++r) {
    const int j = perm[r];
    m += a[j];
    for (int i = 0; i < d; ++i) {
      kstar[i] += a[j] * bf16_to_f64(K[(size_t)j * d + i]);
      vstar[i] += a[j] * bf16_to_f64(V[(size_t)j * d + i]);
    }
  }
  *zero_mass = 0;
  if (m > 0.0) {
    for (int i = 0; i < d; ++i) { kstar[i] /= m; vstar[i] /= m; }
  } else {
    *zero_mass = 1;
    for (int i = 0; i < d; ++i) { kstar[i] = 0.0; vstar[i] = 0.0; }
    for (int r = b; r < n; ++r) {
      const int j = perm[r];
      for (int i = 0; i < d; ++i) {
        kstar[i] += bf16_to_f64(K[(size_t)j * d + i]);
        vstar[i] += bf16_to_f64(V[(size_t)j * d + i]);
      }
    }
    for (int i = 0; i < d; ++i) { kstar[i] /= (double)(n - b); vstar[i] /= (double)(n - b); }
  }
  return m;
}

void oracle_tail_clusters(const uint16_t* K, const uint16_t* V, const int32_t* perm, int n, int d,
                          int b, int m, uint16_t* kbar_bits, uint16_t* vbar_bits,
                          int32_t* count, double* rk, double* rv, double* kept_vmax);

/* -------------------------------------------------------- whole pass ----- */

typedef struct {
  int B, L, Hq, H, n, d, w;
  double scale;
  int pool, protect, alpha_num, alpha_den, T, statistic, tail_slot, allocator, clusters;
  int64_t B_live;
} oracle_cfg;

typedef struct {
  const oracle_cfg* cfg;
  const uint16_t *K, *V, *Q;
  const float* a_in;       /* optional: scores to start from (conditioned mode) */
  double* a;               /* [units][n] */
  int32_t* perm;           /* [units][n] */
  double* c;               /* [units][n] */
  int32_t* counts;         /* [units] */
  double* tail;            /* [units][2][d] */
  double* tail_mass;       /* [units] */
  int64_t* repairs;        /* [B*L] */
  int* status;             /* [units] */
  int phase;
  int next;                /* work counter */
  pthread_mutex_t lock;
} job_t;

static int take(job_t* jb, int limit) {
  pthread_mutex_lock(&jb->lock);
  int i = jb->next < limit ? jb->next++ : -1;
  pthread_mutex_unlock(&jb->lock);
  return i;
}

static void* worker(void* arg) {
  job_t* jb = (job_t*)arg;
  const oracle_cfg* g = jb->cfg;
  const int units = g->B * g->L * g->H;
  const int G = g->Hq / g->H;
  const size_t n = (size_t)g->n, d = (size_t)g->d;
  if (jb->phase == 0) { /* scores, order and curve per unit */
    for (int u; (u = take(jb, units)) >= 0;) {
      const int bl = u / g->H, h = u % g->H;
      double* a = jb->a + (size_t)u * n;
      if (jb->a_in) {
        for (size_t j = 0; j < n; ++j) a[j] = (double)jb->a_in[(size_t)u * n + j];
      } else {
        const uint16_t* Qg = jb->Q + ((size_t)bl * g->Hq + (size_t)h * G) * g->w * d;
        oracle_scores(jb->K + (size_t)u * n * d, Qg, g->n, g->d, g->w, G, g->scale,
                      g->pool, g->protect, a);
      }
      oracle_order(a, g->n, jb->perm + (size_t)u * n);
      oracle_curve(a, jb->V + (size_t)u * n * d, jb->perm + (size_t)u * n, g->n, g->d,
                   g->statistic, jb->c + (size_t)u * n);
    }
  } else if (jb->phase == 1) { /* allocation per (sequence, layer) */
    for (int bl; (bl = take(jb, g->B * g->L)) >= 0;) {
      const double* curves[64];
      for (int h = 0; h < g->H; ++h) curves[h] = jb->c + ((size_t)bl * g->H + h) * n;
      /* every head is charged its tail slot and its cluster summaries */
      const int64_t B_real = g->B_live - (int64_t)g->H * ((g->tail_slot ? 1 : 0) + g->clusters);
      int rc = oracle_allocate_mode(curves, g->H, g->n, B_real, g->alpha_num, g->alpha_den,
                                    g->T, g->allocator, jb->counts + (size_t)bl * g->H,
                                    jb->repairs + bl);
      for (int h = 0; h < g->H; ++h) jb->status[bl * g->H + h] = rc;
    }
  } else { /* tail per unit */
    for (int u; (u = take(jb, units)) >= 0;) {
      if (!g->tail_slot) { jb->tail_mass[u] = 0.0; continue; }
      int zero = 0;
      jb->tail_mass[u] = oracle_tail(jb->a + (size_t)u * n, jb->K + (size_t)u * n * d,
                                     jb->V + (size_t)u * n * d, jb->perm + (size_t)u * n,
                                     g->n, g->d, jb->counts[u],
                                     jb->tail + (size_t)u * 2 * d,
                                     jb->tail + (size_t)u * 2 * d + d, &zero);
      if (zero) jb->status[u] |= 0x100;
    }
  }
  return NULL;
}

static void run_phase(job_t* jb, int phase, int threads) {
  jb->phase = phase;
  jb->next = 0;
  if (threads <= 1) { worker(jb); return; }
  pthread_t* tid = (pthread_t*)malloc((size_t)threads * sizeof(pthread_t));
  for (int i = 0; i < threads; ++i) pthread_create(&tid[i], NULL, worker, jb);
  for (int i = 0; i < threads; ++i) pthread_join(tid[i], NULL);
  free(tid);
}

/*
 * The whole compression pass over B*L*H units plus the packed cache, in the
 * library's packed layout.  cfg_i holds {B, L, Hq, H, n, d, w, pool, protect,
 * alpha_num, alpha_den, T, statistic, tail_slot, allocator, clusters}; scale and
 * B_live separately.  With clusters = m > 0 each segment ends with m summary
 * slots (stored representatives, positions -2 - g), cl_meta [units][m][3]
 * receives (count, key radius, value radius) and kept_vmax [units] the largest
 * kept value norm (both may be NULL when m = 0).
 * a_in (fp32 [units][n]) may be NULL; when given, scoring is skipped and the
 * pass starts from these scores (conditioned mode).  Outputs (all required):
 *   a [units][n], perm [units][n], c [units][n], counts [units],
 *   offsets [units+1], positions [B*L*B_live], pk, pv bf16 [B*L*B_live][d],
 *   tail [units][2][d] (k*, v* before rounding), tail_mass [units],
 *   repairs [B*L].
 * Returns 0, 2 (infeasible budget) or 0x100 bit set if some tail had zero mass.
 */
int oracle_compress(const int32_t* cfg_i, double scale, int64_t B_live,
                    const uint16_t* K, const uint16_t* V, const uint16_t* Q,
                    const float* a_in, int threads,
                    double* a, int32_t* perm, double* c, int32_t* counts,
                    int64_t* offsets, int32_t* positions, uint16_t* pk, uint16_t* pv,
                    double* tail, double* tail_mass, int64_t* repairs,
                    double* cl_meta, double* kept_vmax) {
  oracle_cfg g;
  g.B = cfg_i[0]; g.L = cfg_i[1]; g.Hq = cfg_i[2]; g.H = cfg_i[3]; g.n = cfg_i[4];
  g.d = cfg_i[5]; g.w = cfg_i[6]; g.pool = cfg_i[7]; g.protect = cfg_i[8];
  g.alpha_num = cfg_i[9]; g.alpha_den = cfg_i[10]; g.T = cfg_i[11];
  g.statistic = cfg_i[12]; g.tail_slot = cfg_i[13]; g.allocator = cfg_i[14];
  g.clusters = cfg_i[15];
  g.scale = scale; g.B_live = B_live;
  if (g.H > 64) return 1;
  const int units = g.B * g.L * g.H;
  const size_t n = (size_t)g.n, d = (size_t)g.d;

  job_t jb;
  memset(&jb, 0, sizeof jb);
  jb.cfg = &g; jb.K = K; jb.V = V; jb.Q = Q; jb.a_in = a_in;
  jb.a = a; jb.perm = perm; jb.c = c; jb.counts = counts; jb.tail = tail;
  jb.tail_mass = tail_mass; jb.repairs = repairs;
  jb.status = (int*)calloc((size_t)units, sizeof(int));
  pthread_mutex_init(&jb.lock, NULL);

  run_phase(&jb, 0, threads);
  run_phase(&jb, 1, threads);
  int rc = 0;
  for (int u = 0; u < units; ++u) if (jb.status[u] == 2) rc = 2;
  if (rc == 0) run_phase(&jb, 2, threads);
  for (int u = 0; u < units && rc == 0; ++u) if (jb.status[u] & 0x100) rc = 0x100;
  pthread_mutex_destroy(&jb.lock);
  free(jb.status);
  if (rc == 2) return rc;

  /* a8: pack.  Segment u: counts[u] real slots (ascending position) + tail slot. */
  int32_t* kept = (int32_t*)malloc(n * sizeof(int32_t));
  int64_t off = 0;
  for (int u = 0; u < units; ++u) {
    if (u % g.H == 0) off = (int64_t)(u / g.H) * g.B_live;
    offsets[u] = off;
    const int bu = counts[u];
    oracle_select(perm + (size_t)u * n, bu, kept);
    for (int s = 0; s < bu; ++s) {
      const size_t src = ((size_t)u * n + (size_t)kept[s]) * d;
      memcpy(pk + (size_t)(off + s) * d, K + src, d * sizeof(uint16_t));
      memcpy(pv + (size_t)(off + s) * d, V + src, d * sizeof(uint16_t));
      positions[off + s] = kept[s];
    }
    off += bu;
    if (g.tail_slot) {
      for (size_t i = 0; i < d; ++i) {
        pk[(size_t)off * d + i] = oracle_f64_to_bf16(tail[(size_t)u * 2 * d + i]);
        pv[(size_t)off * d + i] = oracle_f64_to_bf16(tail[(size_t)u * 2 * d + d + i]);
      }
      positions[off] = -1;
      off += 1;
    }
    if (g.clusters > 0) {  /* the m summary slots (clustered-tail certificate) */
      const int m = g.clusters;
      int32_t* cnt = (int32_t*)malloc((size_t)m * sizeof(int32_t));
      double* rk = (double*)malloc((size_t)m * 2 * sizeof(double));
      oracle_tail_clusters(K + (size_t)u * n * d, V + (size_t)u * n * d, perm + (size_t)u * n,
                           g.n, g.d, bu, m, pk + (size_t)off * d, pv + (size_t)off * d, cnt, rk,
                           rk + m, kept_vmax + u);
      for (int c = 0; c < m; ++c) {
        positions[off + c] = -2 - c;
        cl_meta[((size_t)u * m + c) * 3 + 0] = (double)cnt[c];
        cl_meta[((size_t)u * m + c) * 3 + 1] = rk[c];
        cl_meta[((size_t)u * m + c) * 3 + 2] = rk[m + c];
      }
      off += m;
      free(cnt);
      free(rk);
    }
  }
  offsets[units] = (int64_t)g.B * g.L * g.B_live;
  free(kept);
  return rc;
}

/* ---------------------------------------------------------------- decode -- */

/*
 * a9: out[b][l][qh][:] = sum_s softmax_s(scale <q, k_s>) v_s over the slots of
 * segment (b, l, qh / G), in float64 from the packed bf16 bytes.
 */
void oracle_decode(const int32_t* cfg_i, double scale, const uint16_t* q,
                   const uint16_t* pk, const uint16_t* pv, const int64_t* offsets,
                   const int32_t* counts, int tail_slot, double* out) {
  const int B = cfg_i[0], L = cfg_i[1], Hq = cfg_i[2], H = cfg_i[3], d = cfg_i[5];
  const int G = Hq / H;
  for (int bl = 0; bl < B * L; ++bl) {
    for (int qh = 0; qh < Hq; ++qh) {
      const int u = bl * H + qh / G;
      const int64_t off = offsets[u];
      const int slots = counts[u] + (tail_slot ? 1 : 0);
      const uint16_t* qv = q + ((size_t)bl * Hq + qh) * d;
      double* o = out + ((size_t)bl * Hq + qh) * d;
      double* lg = (double*)malloc((size_t)slots * sizeof(double));
      double mx = -INFINITY;
      for (int s = 0; s < slots; ++s) {
        double dot = 0.0;
        for (int i = 0; i < d; ++i)
          dot += bf16_to_f64(qv[i]) * bf16_to_f64(pk[(size_t)(off + s) * d + i]);
        lg[s] = scale * dot;
        if (lg[s] > mx) mx = lg[s];
      }
      double z = 0.0;
      for (int s = 0; s < slots; ++s) z += exp(lg[s] - mx);
      for (int i = 0; i < d; ++i) o[i] = 0.0;
      for (int s = 0; s < slots; ++s) {
        const double p = exp(lg[s] - mx) / z;
        for (int i = 0; i < d; ++i) o[i] += p * bf16_to_f64(pv[(size_t)(off + s) * d + i]);
      }
      free(lg);
    }
  }
}

/* ------------------------------------------- clustered tail summaries ---- */

/*
 * Summaries of the evicted ranks b..n-1 of one unit for the clustered-tail
 * output-error bound (appendix: deterministic output-error bound for
 * clustered tail summaries, Eq. (cluster-summaries), (cluster-radii)).
 * READING R-C1: m groups of consecutive ranks, group g = ranks
 * b + floor(g T / m) .. b + floor((g + 1) T / m) - 1 with T = n - b (an empty
 * group has count 0).  READING R-C2: the representatives are the unweighted
 * means of the group's keys and values, rounded to bf16 as they are stored
 * (kbar_bits, vbar_bits [m][d]); the radii are the largest Euclidean distances
 * of the group's rows to those stored representatives.  kept_vmax = max over
 * the kept ranks 0..b-1 of ||v_j||_2.
 */
void oracle_tail_clusters(const uint16_t* K, const uint16_t* V, const int32_t* perm, int n, int d,
                          int b, int m, uint16_t* kbar_bits, uint16_t* vbar_bits,
                          int32_t* count, double* rk, double* rv, double* kept_vmax) {
  const int T = n - b;
  double* mk = (double*)malloc((size_t)d * sizeof(double));
  double* mv = (double*)malloc((size_t)d * sizeof(double));
  for (int g = 0; g < m; ++g) {
    const int r0 = b + (int)(((int64_t)g * T) / m), r1 = b + (int)(((int64_t)(g + 1) * T) / m);
    count[g] = r1 - r0;
    for (int i = 0; i < d; ++i) { mk[i] = 0.0; mv[i] = 0.0; }
    for (int r = r0; r < r1; ++r) {
      const int j = perm[r];
      for (int i = 0; i < d; ++i) {
        mk[i] += bf16_to_f64(K[(size_t)j * d + i]);
        mv[i] += bf16_to_f64(V[(size_t)j * d + i]);
      }
    }
    for (int i = 0; i < d; ++i) {
      const double ck = count[g] > 0 ? mk[i] / count[g] : 0.0;
      const double cv = count[g] > 0 ? mv[i] / count[g] : 0.0;
      kbar_bits[(size_t)g * d + i] = oracle_f64_to_bf16(ck);
      vbar_bits[(size_t)g * d + i] = oracle_f64_to_bf16(cv);
    }
    double rkg = 0.0, rvg = 0.0;
    for (int r = r0; r < r1; ++r) {
      const int j = perm[r];
      double sk = 0.0, sv = 0.0;
      for (int i = 0; i < d; ++i) {
        const double dk = bf16_to_f64(K[(size_t)j * d + i]) - bf16_to_f64(kbar_bits[(size_t)g * d + i]);
        const double dv = bf16_to_f64(V[(size_t)j * d + i]) - bf16_to_f64(vbar_bits[(size_t)g * d + i]);
        sk += dk * dk;
        sv += dv * dv;
      }
      if (sqrt(sk) > rkg) rkg = sqrt(sk);
      if (sqrt(sv) > rvg) rvg = sqrt(sv);
    }
    rk[g] = rkg;
    rv[g] = rvg;
  }
  double vm = 0.0;
  for (int r = 0; r < b; ++r) {
    const int j = perm[r];
    double s = 0.0;
    for (int i = 0; i < d; ++i) s += bf16_to_f64(V[(size_t)j * d + i]) * bf16_to_f64(V[(size_t)j * d + i]);
    if (sqrt(s) > vm) vm = sqrt(s);
  }
  *kept_vmax = vm;
  free(mk);
  free(mv);
}

/*
 * Certified decode of one query head (Theorem: runtime-computable output-error
 * bound for clustered tail summaries, Eq. (certificate-estimator),
 * (certificate-quantities), (certificate-bound), (certificate-structure)).
 * Kept set S = the b packed real rows pk, pv [b][d]; clusters g = 0..m-1 with
 * stored representatives kbar, vbar (bf16 bits [m][d]), counts, key radii rk
 * and value radii rv.  READING R-C3: the representative logit is
 * scale <q, kbar_g> and the logit radius r_g = scale ||q||_2 rk_g
 * (Cauchy-Schwarz, the paper's runtime remark).  Empty clusters are skipped.
 * Writes O-hat [d]; returns the bound (3 / Zhat)(D_N + V'max D_Z); *certified
 * = (D_Z <= Zhat / 3); *structural = the bound's structural form.  Every
 * exponential is taken relative to one shift, to which the bound is invariant.
 */
double oracle_decode_certified(const uint16_t* q, const uint16_t* pk, const uint16_t* pv, int b,
                               int d, double scale, const uint16_t* kbar, const uint16_t* vbar,
                               const int32_t* count, const double* rk, const double* rv, int m,
                               double* out, int* certified, double* structural) {
  double qn = 0.0;
  for (int i = 0; i < d; ++i) qn += bf16_to_f64(q[i]) * bf16_to_f64(q[i]);
  qn = sqrt(qn);
  double* lg = (double*)malloc((size_t)(b + m) * sizeof(double));
  double M = -INFINITY;
  for (int s = 0; s < b; ++s) {
    double dot = 0.0;
    for (int i = 0; i < d; ++i) dot += bf16_to_f64(q[i]) * bf16_to_f64(pk[(size_t)s * d + i]);
    lg[s] = scale * dot;
    if (lg[s] > M) M = lg[s];
  }
  for (int g = 0; g < m; ++g) {  /* log of n_g e^{lbar_g} */
    double dot = 0.0;
    for (int i = 0; i < d; ++i) dot += bf16_to_f64(q[i]) * bf16_to_f64(kbar[(size_t)g * d + i]);
    lg[b + g] = count[g] > 0 ? scale * dot + log((double)count[g]) : -INFINITY;
    if (lg[b + g] > M) M = lg[b + g];
  }
  double Z = 0.0, ZS = 0.0, DZ = 0.0, DN = 0.0, vmax = 0.0, smax = 0.0;
  for (int i = 0; i < d; ++i) out[i] = 0.0;
  for (int s = 0; s < b; ++s) {
    const double w = exp(lg[s] - M);
    Z += w;
    ZS += w;
    double vv = 0.0;
    for (int i = 0; i < d; ++i) {
      const double x = bf16_to_f64(pv[(size_t)s * d + i]);
      out[i] += w * x;
      vv += x * x;
    }
    if (sqrt(vv) > vmax) vmax = sqrt(vv);
  }
  for (int g = 0; g < m; ++g) {
    if (count[g] <= 0) continue;
    const double zg = exp(lg[b + g] - M);
    const double r = scale * qn * rk[g];
    const double er = exp(r);
    double vn = 0.0;
    for (int i = 0; i < d; ++i) {
      const double x = bf16_to_f64(vbar[(size_t)g * d + i]);
      out[i] += zg * x;
      vn += x * x;
    }
    vn = sqrt(vn);
    Z += zg;
    DZ += (er - 1.0) * er * zg;
    DN += er * zg * ((er - 1.0) * vn + rv[g]);
    if (vn + rv[g] > vmax) vmax = vn + rv[g];
  }
  for (int i = 0; i < d; ++i) out[i] /= Z;
  for (int g = 0; g < m; ++g) {
    if (count[g] <= 0) continue;
    const double er = exp(scale * qn * rk[g]);
    const double t = er * (2.0 * vmax * (er - 1.0) + rv[g]);
    if (t > smax) smax = t;
  }
  *certified = DZ <= Z / 3.0;
  *structural = 3.0 * (1.0 - ZS / Z) * smax;
  free(lg);
  return 3.0 / Z * (DN + vmax * DZ);
}

/* ------------------------------------------------ coverage profile ------ */

/*
 * Coverage profile of one realized query row over n keys (§3: the ranked gap
 * profile and the coverage budget; the count definitions; appendix: the
 * gap-profile instrument, which recomputes row logits).  z_j = scale <q, k_j>,
 * A = softmax(z).  pi orders the logits nonincreasingly, ties by lower index.
 * Writes
 *   order[r]  = pi(r + 1), the token at rank r (0-based ranks; NULL: skipped)
 *   gap[r]    = G(r + 1) = z_(1) - z_(r+1) (NULL: skipped)
 *   K_eta[e]  = min{k : sum_{j <= k} A_(j) >= 1 - eta[e]}
 *   rel[e]    = #{j : A_j > rel_eps[e] A_(1)} (relative-weight count)
 *   abs_[e]   = #{j : A_j > abs_eps[e]} (calibrated count k(eps))
 *   top[0] = z_(1), top[1] = log sum_j e^{z_j}
 */
void oracle_coverage_profile(const uint16_t* q, const uint16_t* K, int n, int d, double scale,
                             const double* eta, int n_eta, const double* rel_eps, int n_rel,
                             const double* abs_eps, int n_abs, int32_t* order, double* gap,
                             int32_t* K_eta, int32_t* rel, int32_t* abs_, double* top) {
  scored_t* t = (scored_t*)malloc((size_t)n * sizeof(scored_t));
  for (int j = 0; j < n; ++j) {
    double dot = 0.0;
    for (int i = 0; i < d; ++i) dot += bf16_to_f64(q[i]) * bf16_to_f64(K[(size_t)j * d + i]);
    t[j].a = scale * dot;
    t[j].j = j;
  }
  qsort(t, (size_t)n, sizeof(scored_t), cmp_desc_then_index);
  const double z1 = t[0].a;
  double Z = 0.0;
  for (int r = 0; r < n; ++r) Z += exp(t[r].a - z1);
  for (int r = 0; r < n; ++r) {
    if (order) order[r] = t[r].j;
    if (gap) gap[r] = z1 - t[r].a;
  }
  for (int e = 0; e < n_eta; ++e) {
    double c = 0.0;
    int k = n;
    for (int r = 0; r < n; ++r) {
      c += exp(t[r].a - z1) / Z;
      if (c >= 1.0 - eta[e]) { k = r + 1; break; }
    }
    K_eta[e] = k;
  }
  const double A1 = 1.0 / Z;
  for (int e = 0; e < n_rel; ++e) {
    int cnt = 0;
    for (int r = 0; r < n; ++r)
      if (exp(t[r].a - z1) / Z > rel_eps[e] * A1) ++cnt;
    rel[e] = cnt;
  }
  for (int e = 0; e < n_abs; ++e) {
    int cnt = 0;
    for (int r = 0; r < n; ++r)
      if (exp(t[r].a - z1) / Z > abs_eps[e]) ++cnt;
    abs_[e] = cnt;
  }
  top[0] = z1;
  top[1] = z1 + log(Z);
  free(t);
}

/* ------------------------------------------------- fixed-row diagnostics ---- */

/*
 * Fixed-row quantities of one realized query row over all n original tokens
 * of a unit (Theorem: fixed-row tail factorization).  A_j = softmax_j(scale
 * <q, k_j>); S = the tokens with kept[j] != 0.  Writes stats[8]:
 *   0 p_S = sum_{j in S} A_j
 *   1 ||O||_2, O = sum_j A_j v_j (exact attention)
 *   2 ||O~_S - O||_2, O~_S = sum_{j in S} A_j v_j / p_S (subset-only output)
 *   3 ||u*||_2, u* = sum_{j not in S} A_j v_j (the unique fixed-row correction)
 *   4 2 V_max (1 - p_S), V_max = max_j ||v_j||_2 (the theorem's mass bound)
 *   5 ||ohat - O||_2 for the given output ohat [d] (NULL: 0)
 *   6 V_max
 *   7 ||O~_S + (1 - p_S) (V-bar_T - O~_S) - O||_2, the factorization residual
 *     (0 up to rounding; V-bar_T = u* / (1 - p_S))
 */
void oracle_fixed_row(const uint16_t* q, const uint16_t* K, const uint16_t* V,
                      const uint8_t* kept, int n, int d, double scale, const double* ohat,
                      double* stats) {
  double* lg = (double*)malloc((size_t)n * sizeof(double));
  double* O = (double*)calloc((size_t)d, sizeof(double));
  double* OS = (double*)calloc((size_t)d, sizeof(double));
  double mx = -INFINITY, vmax = 0.0;
  for (int j = 0; j < n; ++j) {
    double dot = 0.0, vv = 0.0;
    for (int i = 0; i < d; ++i) {
      dot += bf16_to_f64(q[i]) * bf16_to_f64(K[(size_t)j * d + i]);
      vv += bf16_to_f64(V[(size_t)j * d + i]) * bf16_to_f64(V[(size_t)j * d + i]);
    }
    lg[j] = scale * dot;
    if (lg[j] > mx) mx = lg[j];
    if (sqrt(vv) > vmax) vmax = sqrt(vv);
  }
  double Z = 0.0, ZS = 0.0;
  for (int j = 0; j < n; ++j) {
    const double w = exp(lg[j] - mx);
    Z += w;
    if (kept[j]) ZS += w;
    for (int i = 0; i < d; ++i) {
      const double x = w * bf16_to_f64(V[(size_t)j * d + i]);
      O[i] += x;
      if (kept[j]) OS[i] += x;
    }
  }
  const double pS = ZS / Z;
  double nO = 0.0, eS = 0.0, nu = 0.0, eh = 0.0, res = 0.0;
  for (int i = 0; i < d; ++i) {
    const double o = O[i] / Z;
    const double os = ZS > 0.0 ? OS[i] / ZS : 0.0;
    const double u = (O[i] - OS[i]) / Z;
    const double vbt = pS < 1.0 ? u / (1.0 - pS) : 0.0;
    nO += o * o;
    eS += (os - o) * (os - o);
    nu += u * u;
    if (ohat) eh += (ohat[i] - o) * (ohat[i] - o);
    const double f = os + (1.0 - pS) * (vbt - os) - o;
    res += f * f;
  }
  stats[0] = pS;
  stats[1] = sqrt(nO);
  stats[2] = sqrt(eS);
  stats[3] = sqrt(nu);
  stats[4] = 2.0 * vmax * (1.0 - pS);
  stats[5] = sqrt(eh);
  stats[6] = vmax;
  stats[7] = sqrt(res);
  free(lg);
  free(O);
  free(OS);
}

/*
 * Future-query lift and summary mismatch (Theorem: future-query lift), for
 * one realized query row over all n original tokens of a unit.  S = the
 * tokens with kept[j] != 0, T = the others (nonempty); the compressed cache
 * holds S and, when kstar != NULL, one synthetic slot (kstar, vstar) whose
 * value stands for the mixture sum_T r_j v_j with r_j = s_j / sum_T s (the
 * uniform 1/|T| when that sum is 0).  z_j = scale <q, k_j>, A = softmax(z)
 * over all n tokens, Ahat = softmax over S and the slot.  Writes stats[8]:
 *   0 p = A(T), the exact attention mass of the tail
 *   1 q = Ahat_star, the slot's weight in compressed attention (0 without a slot)
 *   2 ||a - r||_1 over T with a = A_T / p (a = 0 when p = 0)
 *   3 Lambda_T - z_star, Lambda_T = log sum_T e^{z_j}, z_star = scale <q, kstar>
 *     (NaN without a slot)
 *   4 V_max (2 |p - q| + min(p, q) ||a - r||_1), the theorem's bound on
 *     ||O - Ohat|| when the slot value is the exact mixture
 *   5 tanh(|Lambda_T - z_star| / 4), the theorem's bound on |p - q| (NaN without a slot)
 *   6 ||A - Abar||_1, Abar = Ahat on S and q r_j on T (the lifted distribution)
 *   7 ||vstar - sum_T r_j v_j||_2, the stored slot value against the exact
 *     mixture (NaN without a slot or when sum_T s = 0)
 */
void oracle_future_query_lift(const uint16_t* q, const uint16_t* K, const uint16_t* V,
                              const uint8_t* kept, const float* s, const uint16_t* kstar,
                              const uint16_t* vstar, int n, int d, double scale,
                              double* stats) {
  double* z = (double*)malloc((size_t)n * sizeof(double));
  double zmax = -INFINITY, zmaxS = -INFINITY, zmaxT = -INFINITY, vmax = 0.0, sT = 0.0;
  int nT = 0;
  for (int j = 0; j < n; ++j) {
    double dot = 0.0, vv = 0.0;
    for (int i = 0; i < d; ++i) {
      dot += bf16_to_f64(q[i]) * bf16_to_f64(K[(size_t)j * d + i]);
      vv += bf16_to_f64(V[(size_t)j * d + i]) * bf16_to_f64(V[(size_t)j * d + i]);
    }
    z[j] = scale * dot;
    if (z[j] > zmax) zmax = z[j];
    if (kept[j]) { if (z[j] > zmaxS) zmaxS = z[j]; }
    else { if (z[j] > zmaxT) zmaxT = z[j]; sT += (double)s[j]; ++nT; }
    if (sqrt(vv) > vmax) vmax = sqrt(vv);
  }
  /* exact attention and the tail mass p */
  double Z = 0.0, ZT = 0.0;
  for (int j = 0; j < n; ++j) {
    const double w = exp(z[j] - zmax);
    Z += w;
    if (!kept[j]) ZT += w;
  }
  const double p = ZT / Z;
  /* compressed attention over S and the slot */
  const int slot = kstar != NULL;
  double zstar = 0.0;
  if (slot) {
    for (int i = 0; i < d; ++i) zstar += bf16_to_f64(q[i]) * bf16_to_f64(kstar[i]);
    zstar *= scale;
  }
  const double c = (slot && zstar > zmaxS) ? zstar : zmaxS;
  double Zhat = slot ? exp(zstar - c) : 0.0;
  for (int j = 0; j < n; ++j)
    if (kept[j]) Zhat += exp(z[j] - c);
  const double qstar = slot ? exp(zstar - c) / Zhat : 0.0;
  /* tail log-partition */
  double sumT = 0.0;
  for (int j = 0; j < n; ++j)
    if (!kept[j]) sumT += exp(z[j] - zmaxT);
  const double LamT = zmaxT + log(sumT);
  /* the tail distributions a and r, and the lifted distribution Abar */
  double l1_ar = 0.0, l1_lift = 0.0;
  double* mix = (double*)calloc((size_t)d, sizeof(double));
  for (int j = 0; j < n; ++j) {
    const double A = exp(z[j] - zmax) / Z;
    if (kept[j]) {
      const double Ahat = exp(z[j] - c) / Zhat;
      l1_lift += fabs(A - Ahat);
    } else {
      const double r = sT > 0.0 ? (double)s[j] / sT : 1.0 / nT;
      const double a = p > 0.0 ? A / p : 0.0;
      l1_ar += fabs(a - r);
      l1_lift += fabs(A - qstar * r);
      for (int i = 0; i < d; ++i) mix[i] += r * bf16_to_f64(V[(size_t)j * d + i]);
    }
  }
  double dv = 0.0;
  if (slot)
    for (int i = 0; i < d; ++i) {
      const double e = bf16_to_f64(vstar[i]) - mix[i];
      dv += e * e;
    }
  const double dpq = fabs(p - qstar);
  stats[0] = p;
  stats[1] = qstar;
  stats[2] = l1_ar;
  stats[3] = slot ? LamT - zstar : NAN;
  stats[4] = vmax * (2.0 * dpq + (p < qstar ? p : qstar) * l1_ar);
  stats[5] = slot ? tanh(fabs(LamT - zstar) / 4.0) : NAN;
  stats[6] = l1_lift;
  stats[7] = (slot && sT > 0.0) ? sqrt(dv) : NAN;
  free(mix);
  free(z);
}

/*
 * Sampled tail compensation (appendix: proposition on sampled tail
 * compensation) for one realized query row over all n original tokens of a
 * unit.  A = softmax(scale <q, k_j>), S = tokens with kept[j] != 0, T the
 * others (|T| = N >= 1), p_S = A(S), u* = sum_T A_j v_j, Q_T = sum_T A_j^2.
 * Two estimators of u* from m tail tokens, with the 2m uniforms u[0..2m-1] in
 * [0, 1) as the only randomness:
 *   weight-proportional: for r < m, j_r = the first tail token (in index
 *     order) whose cumulative tail weight exceeds u[r] * A(T);
 *     u_w = (1 - p_S)/m sum_r v_{j_r}
 *   uniform m-subset (Floyd's algorithm, m <= N): for i = N - m .. N - 1,
 *     t = floor(u[m + i - (N - m)] * (i + 1)); take tail rank t unless already
 *     taken, else rank i; u_u = (1 - p_S)/m sum over the subset of v_j
 *     (tail rank t = the t-th tail token in index order)
 * forced_idx (2m token indices, or NULL) replaces both draws.  Writes the
 * sampled token indices to idx[2m] and stats[8]:
 *   0 p_S   1 Q_T   2 ||u*||   3 ||u_w - u*||   4 ||u_u - u*||
 *   5 sqrt(d s2 (1 - p_S)^2 / m (1 - Q_T / (1 - p_S)^2))       (part (i))
 *   6 sqrt(d s2 (1 - p_S)^2 (1/m - 2/N + Q_T / (1 - p_S)^2))  (part (ii))
 *   7 s2 = sum_T ||v_j - vbar_T||^2 / (d N), the per-coordinate variance of
 *     the tail values (unweighted mean vbar_T), which stands for sigma_V^2
 */
void oracle_sampled_compensation(const uint16_t* q, const uint16_t* K, const uint16_t* V,
                                 const uint8_t* kept, int n, int d, double scale, int m,
                                 const float* u, const int32_t* forced_idx, int32_t* idx,
                                 double* stats) {
  double* w = (double*)malloc((size_t)n * sizeof(double));
  int32_t* tail = (int32_t*)malloc((size_t)n * sizeof(int32_t));
  double* ustar = (double*)calloc((size_t)d, sizeof(double));
  double* uw = (double*)calloc((size_t)d, sizeof(double));
  double* uu = (double*)calloc((size_t)d, sizeof(double));
  double* vbar = (double*)calloc((size_t)d, sizeof(double));
  double zmax = -INFINITY;
  for (int j = 0; j < n; ++j) {
    double dot = 0.0;
    for (int i = 0; i < d; ++i) dot += bf16_to_f64(q[i]) * bf16_to_f64(K[(size_t)j * d + i]);
    w[j] = scale * dot;
    if (w[j] > zmax) zmax = w[j];
  }
  double Z = 0.0;
  for (int j = 0; j < n; ++j) {
    w[j] = exp(w[j] - zmax);
    Z += w[j];
  }
  int N = 0;
  double pT = 0.0, QT = 0.0;
  for (int j = 0; j < n; ++j) {
    w[j] /= Z; /* A_j */
    if (!kept[j]) {
      tail[N++] = j;
      pT += w[j];
      QT += w[j] * w[j];
      for (int i = 0; i < d; ++i) {
        const double v = bf16_to_f64(V[(size_t)j * d + i]);
        ustar[i] += w[j] * v;
        vbar[i] += v;
      }
    }
  }
  const double pS = 1.0 - pT;
  /* weight-proportional draws by the inverse of the cumulative tail weight */
  for (int r = 0; r < m; ++r) {
    if (forced_idx) {
      idx[r] = forced_idx[r];
      continue;
    }
    const double target = (double)u[r] * pT;
    double c = 0.0;
    int pick = tail[N - 1];
    for (int t = 0; t < N; ++t) {
      c += w[tail[t]];
      if (c > target) { pick = tail[t]; break; }
    }
    idx[r] = pick;
  }
  /* uniform m-subset of the tail ranks, Floyd's algorithm */
  for (int s = 0; s < m; ++s) {
    if (forced_idx) {
      idx[m + s] = forced_idx[m + s];
      continue;
    }
    const int i = N - m + s;
    int t = (int)floor((double)u[m + s] * (double)(i + 1));
    if (t > i) t = i;
    int taken = 0;
    for (int e = 0; e < s; ++e)
      if (idx[m + e] == tail[t]) taken = 1;
    idx[m + s] = taken ? tail[i] : tail[t];
  }
  for (int r = 0; r < m; ++r)
    for (int i = 0; i < d; ++i) {
      uw[i] += bf16_to_f64(V[(size_t)idx[r] * d + i]);
      uu[i] += bf16_to_f64(V[(size_t)idx[m + r] * d + i]);
    }
  double nu = 0.0, ew = 0.0, eu = 0.0, var = 0.0;
  for (int i = 0; i < d; ++i) {
    vbar[i] /= N;
    uw[i] *= (1.0 - pS) / m;
    uu[i] *= (1.0 - pS) / m;
    nu += ustar[i] * ustar[i];
    ew += (uw[i] - ustar[i]) * (uw[i] - ustar[i]);
    eu += (uu[i] - ustar[i]) * (uu[i] - ustar[i]);
  }
  for (int t = 0; t < N; ++t)
    for (int i = 0; i < d; ++i) {
      const double e = bf16_to_f64(V[(size_t)tail[t] * d + i]) - vbar[i];
      var += e * e;
    }
  const double s2 = var / ((double)d * N);
  const double omp2 = (1.0 - pS) * (1.0 - pS);
  const double imb = omp2 > 0.0 ? QT / omp2 : 0.0;
  const double mse_w = d * s2 * omp2 / m * (1.0 - imb);
  const double mse_u = d * s2 * omp2 * (1.0 / m - 2.0 / N + imb);
  stats[0] = pS;
  stats[1] = QT;
  stats[2] = sqrt(nu);
  stats[3] = sqrt(ew);
  stats[4] = sqrt(eu);
  stats[5] = sqrt(mse_w > 0.0 ? mse_w : 0.0);
  stats[6] = sqrt(mse_u > 0.0 ? mse_u : 0.0);
  stats[7] = s2;
  free(w); free(tail); free(ustar); free(uw); free(uu); free(vbar);
}
