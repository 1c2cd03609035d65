/*
 * dc_oracle.c -- plain fp64 CPU oracle of the DistillCache decode/evict step.
 *
 * TEST INFRASTRUCTURE ONLY (see dc_oracle.h): the product path never includes,
 * links or calls this file. It is written for clarity, not speed: every
 * quantity is computed from its definition, in the paper's order, in double
 * precision, with no blocking or fusion.
 *
 * Readings of the paper where it is silent or ambiguous (each one is a choice,
 * listed with the others in the design notes):
 *   - alpha_i averages over the G query heads of this KV group (per-row
 *     selection); alpha_mode 1 sums that average over all steps since the token
 *     was inserted (cumulative attention, as H2O-style scorers do).
 *   - sigma_i is the population variance over the G heads of this step.
 *   - H_i pools (query step, head) pairs: Z_i = sum over the last min(w, steps)
 *     decode steps and the G heads of a_{q,h}(i), S_i the same sum weighted by
 *     each head's entropy; H_i = S_i / Z_i, or 0 when Z_i = 0. The window
 *     includes the current step; a token absent at step q contributes 0.
 *     Natural logarithm; 0 * log 0 = 0.
 *   - pos_i = p_i / max(p_newest, 1), p the absolute position (tokens seen).
 *   - softmax scale 1/sqrt(d); the new token attends to itself.
 *   - MLP: Linear(5, H) -> LayerNorm(H, eps 1e-5, biased variance) -> ReLU ->
 *     Linear(H, 1); without LayerNorm when layernorm == 0.
 *   - ties in the top-B selection go to the lower position; -0 equals +0; NaN
 *     ranks below every number.
 */
#include "dc_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

typedef struct {
  int n;          /* tokens present at that step */
  int64_t* pos;   /* [n], ascending */
  double* a;      /* [n][G]: attention weight of head h on token i */
  double* H;      /* [G]: entropy of head h's distribution */
} win_entry;

struct dco_row {
  int d, G, w, alpha_mode, cap;
  int n;
  int64_t seen;     /* tokens ever appended = next position */
  uint16_t *kb, *vb; /* [cap][d] bf16 bits */
  double *k, *v;     /* [cap][d] exact widenings */
  int64_t* pos;      /* [cap] */
  double* acc;       /* [cap] cumulative alpha (alpha_mode 1) */
  double *S, *Z;     /* [cap] window sums of the last step */
  double *Sp, *Zp;   /* [cap] the same without the last step's query */
  double* score;     /* [cap] scores of the last step */
  int have_scores;
  win_entry* win;    /* ring of w entries */
  int win_count, win_next;
};

static double bf16_to_double(uint16_t b) {
  uint32_t u = ((uint32_t)b) << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

dco_row* dco_row_new(int d, int G, int w, int alpha_mode, int cap) {
  if (d <= 0 || G <= 0 || w <= 0 || cap <= 0 || (alpha_mode != 0 && alpha_mode != 1)) return NULL;
  dco_row* r = (dco_row*)calloc(1, sizeof *r);
  if (!r) return NULL;
  r->d = d; r->G = G; r->w = w; r->alpha_mode = alpha_mode; r->cap = cap;
  size_t nd = (size_t)cap * (size_t)d;
  r->kb = (uint16_t*)calloc(nd, sizeof(uint16_t));
  r->vb = (uint16_t*)calloc(nd, sizeof(uint16_t));
  r->k = (double*)calloc(nd, sizeof(double));
  r->v = (double*)calloc(nd, sizeof(double));
  r->pos = (int64_t*)calloc((size_t)cap, sizeof(int64_t));
  r->acc = (double*)calloc((size_t)cap, sizeof(double));
  r->S = (double*)calloc((size_t)cap, sizeof(double));
  r->Z = (double*)calloc((size_t)cap, sizeof(double));
  r->Sp = (double*)calloc((size_t)cap, sizeof(double));
  r->Zp = (double*)calloc((size_t)cap, sizeof(double));
  r->score = (double*)calloc((size_t)cap, sizeof(double));
  r->win = (win_entry*)calloc((size_t)w, sizeof(win_entry));
  if (!r->kb || !r->vb || !r->k || !r->v || !r->pos || !r->acc || !r->S || !r->Z || !r->Sp ||
      !r->Zp || !r->score ||
      !r->win) {
    dco_row_free(r);
    return NULL;
  }
  return r;
}

static void win_entry_clear(win_entry* e) {
  free(e->pos); free(e->a); free(e->H);
  memset(e, 0, sizeof *e);
}

void dco_row_free(dco_row* r) {
  if (!r) return;
  if (r->win)
    for (int i = 0; i < r->w; ++i) win_entry_clear(&r->win[i]);
  free(r->win); free(r->kb); free(r->vb); free(r->k); free(r->v); free(r->pos);
  free(r->acc); free(r->S); free(r->Z); free(r->Sp); free(r->Zp); free(r->score);
  free(r);
}

static void put_token(dco_row* r, const uint16_t* k, const uint16_t* v) {
  int i = r->n, d = r->d;
  for (int c = 0; c < d; ++c) {
    r->kb[(size_t)i * d + c] = k[c];
    r->vb[(size_t)i * d + c] = v[c];
    r->k[(size_t)i * d + c] = bf16_to_double(k[c]);
    r->v[(size_t)i * d + c] = bf16_to_double(v[c]);
  }
  r->pos[i] = r->seen;
  r->acc[i] = 0.0;
  r->n += 1;
  r->seen += 1;
}

int dco_row_append(dco_row* r, const uint16_t* k, const uint16_t* v, int T) {
  if (T < 0 || r->n + T > r->cap) return -1;
  for (int t = 0; t < T; ++t) put_token(r, k + (size_t)t * r->d, v + (size_t)t * r->d);
  r->have_scores = 0;
  return 0;
}

/* Softmax attention of G heads over the n keys of K/V (fp64 rows):
 * a [n][G] (may be NULL), o [G][d], Hq [G]. */
static void attend_rows(const double* q, const double* K, const double* V, int n, int d, int G,
                        double* a, double* o, double* Hq) {
  double* s = (double*)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
  double scale = 1.0 / sqrt((double)d);
  for (int h = 0; h < G; ++h) {
    const double* qh = q + (size_t)h * d;
    double m = -INFINITY;
    for (int i = 0; i < n; ++i) {
      double dot = 0.0;
      for (int c = 0; c < d; ++c) dot += qh[c] * K[(size_t)i * d + c];
      s[i] = dot * scale;
      if (s[i] > m) m = s[i];
    }
    double l = 0.0;
    for (int i = 0; i < n; ++i) l += exp(s[i] - m);
    double H = 0.0;
    for (int c = 0; c < d; ++c) o[(size_t)h * d + c] = 0.0;
    for (int i = 0; i < n; ++i) {
      double ai = exp(s[i] - m) / l;
      if (a) a[(size_t)i * G + h] = ai;
      if (ai > 0.0) H -= ai * log(ai);
      for (int c = 0; c < d; ++c) o[(size_t)h * d + c] += ai * V[(size_t)i * d + c];
    }
    if (Hq) Hq[h] = H;
  }
  free(s);
}

void dco_attend(const uint16_t* q, const uint16_t* k, const uint16_t* v, int n, int d, int G,
                double* o, double* Hq) {
  double* qd = (double*)malloc(sizeof(double) * (size_t)G * d);
  double* K = (double*)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1) * d);
  double* V = (double*)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1) * d);
  for (int i = 0; i < G * d; ++i) qd[i] = bf16_to_double(q[i]);
  for (size_t i = 0; i < (size_t)n * d; ++i) { K[i] = bf16_to_double(k[i]); V[i] = bf16_to_double(v[i]); }
  attend_rows(qd, K, V, n, d, G, NULL, o, Hq);
  free(qd); free(K); free(V);
}

/* Policy network f_phi [Sec. 3.1.2; App. D]. */
void dco_policy(const double* x, int m, const float* mlp, int hidden, int layernorm, double* score) {
  const float* W1 = mlp;
  const float* b1 = W1 + 5 * hidden;
  const float* gamma = b1 + hidden;
  const float* beta = gamma + hidden;
  const float* w2 = beta + hidden;
  double b2 = (double)w2[hidden];
  double* h = (double*)malloc(sizeof(double) * (size_t)hidden);
  for (int t = 0; t < m; ++t) {
    const double* xt = x + (size_t)t * 5;
    for (int j = 0; j < hidden; ++j) {
      double acc = (double)b1[j];
      for (int c = 0; c < 5; ++c) acc += (double)W1[j * 5 + c] * xt[c];
      h[j] = acc;
    }
    if (layernorm) {
      double mu = 0.0, var = 0.0;
      for (int j = 0; j < hidden; ++j) mu += h[j];
      mu /= hidden;
      for (int j = 0; j < hidden; ++j) var += (h[j] - mu) * (h[j] - mu);
      var /= hidden;
      double inv = 1.0 / sqrt(var + 1e-5);
      for (int j = 0; j < hidden; ++j) h[j] = (h[j] - mu) * inv * (double)gamma[j] + (double)beta[j];
    }
    double out = b2;
    for (int j = 0; j < hidden; ++j) out += (double)w2[j] * (h[j] > 0.0 ? h[j] : 0.0);
    score[t] = out;
  }
  free(h);
}

/* Index of position p in an ascending array, or -1. */
static int find_pos(const int64_t* arr, int n, int64_t p) {
  int lo = 0, hi = n - 1;
  while (lo <= hi) {
    int mid = lo + (hi - lo) / 2;
    if (arr[mid] == p) return mid;
    if (arr[mid] < p) lo = mid + 1; else hi = mid - 1;
  }
  return -1;
}

int dco_row_step(dco_row* r, const uint16_t* q, const uint16_t* k_new, const uint16_t* v_new,
                 const float* mlp, int hidden, int layernorm,
                 double* o, double* Hq, double* feat, double* score) {
  int d = r->d, G = r->G;
  if (r->n + 1 > r->cap) return -1;
  /* Algorithm 1: the forward pass's cache C_t already holds the new pair. */
  put_token(r, k_new, v_new);
  int n = r->n;

  double* qd = (double*)malloc(sizeof(double) * (size_t)G * d);
  for (int i = 0; i < G * d; ++i) qd[i] = bf16_to_double(q[i]);
  double* a = (double*)malloc(sizeof(double) * (size_t)n * G);
  double* oo = (double*)malloc(sizeof(double) * (size_t)G * d);
  double* HH = (double*)malloc(sizeof(double) * (size_t)G);
  attend_rows(qd, r->k, r->v, n, d, G, a, oo, HH);
  if (o) memcpy(o, oo, sizeof(double) * (size_t)G * d);
  if (Hq) memcpy(Hq, HH, sizeof(double) * (size_t)G);

  /* Record this step's attention distributions (keyed by position) in the
   * window of the last w queries [Sec. 3.1.1, H_i]. */
  win_entry* e = &r->win[r->win_next];
  win_entry_clear(e);
  e->n = n;
  e->pos = (int64_t*)malloc(sizeof(int64_t) * (size_t)n);
  e->a = (double*)malloc(sizeof(double) * (size_t)n * G);
  e->H = (double*)malloc(sizeof(double) * (size_t)G);
  memcpy(e->pos, r->pos, sizeof(int64_t) * (size_t)n);
  memcpy(e->a, a, sizeof(double) * (size_t)n * G);
  memcpy(e->H, HH, sizeof(double) * (size_t)G);
  r->win_next = (r->win_next + 1) % r->w;
  if (r->win_count < r->w) r->win_count += 1;

  double* x = (double*)malloc(sizeof(double) * (size_t)n * 5);
  int64_t newest = r->pos[n - 1];
  double pos_den = (double)(newest > 1 ? newest : 1);
  for (int i = 0; i < n; ++i) {
    /* alpha_i: mean over heads of the mass token i receives. */
    double mean = 0.0;
    for (int h = 0; h < G; ++h) mean += a[(size_t)i * G + h];
    mean /= G;
    double alpha = mean;
    if (r->alpha_mode == 1) {
      r->acc[i] += mean;
      alpha = r->acc[i];
    }
    /* sigma_i: population variance across heads. */
    double var = 0.0;
    for (int h = 0; h < G; ++h) {
      double dv = a[(size_t)i * G + h] - mean;
      var += dv * dv;
    }
    var /= G;
    /* |v_i|_2 */
    double vn = 0.0;
    for (int c = 0; c < d; ++c) vn += r->v[(size_t)i * d + c] * r->v[(size_t)i * d + c];
    vn = sqrt(vn);
    /* H_i = S_i / Z_i over the window of recent queries. */
    double S = 0.0, Z = 0.0, Sp = 0.0, Zp = 0.0;
    int newest_entry = (r->win_next + r->w - 1) % r->w;
    for (int qi = 0; qi < r->win_count; ++qi) {
      const win_entry* we = &r->win[qi];
      int j = find_pos(we->pos, we->n, r->pos[i]);
      if (j < 0) continue; /* not yet in the cache at that step */
      for (int h = 0; h < G; ++h) {
        Z += we->a[(size_t)j * G + h];
        S += we->a[(size_t)j * G + h] * we->H[h];
        if (qi != newest_entry) {
          Zp += we->a[(size_t)j * G + h];
          Sp += we->a[(size_t)j * G + h] * we->H[h];
        }
      }
    }
    r->S[i] = S;
    r->Z[i] = Z;
    r->Sp[i] = Sp;
    r->Zp[i] = Zp;
    double Hi = Z > 0.0 ? S / Z : 0.0;
    double posn = (double)r->pos[i] / pos_den;
    x[(size_t)i * 5 + 0] = alpha;
    x[(size_t)i * 5 + 1] = vn;
    x[(size_t)i * 5 + 2] = var;
    x[(size_t)i * 5 + 3] = Hi;
    x[(size_t)i * 5 + 4] = posn;
  }
  dco_policy(x, n, mlp, hidden, layernorm, r->score);
  r->have_scores = 1;
  if (feat) memcpy(feat, x, sizeof(double) * (size_t)n * 5);
  if (score) memcpy(score, r->score, sizeof(double) * (size_t)n);
  free(qd); free(a); free(oo); free(HH); free(x);
  return n;
}

/* Ranking of tokens for argtop_B: score descending, then position ascending;
 * a NaN score ranks below every number. */
typedef struct { double s; int64_t p; int i; } rank_item;

static int rank_cmp(const void* pa, const void* pb) {
  const rank_item* x = (const rank_item*)pa;
  const rank_item* y = (const rank_item*)pb;
  int nx = isnan(x->s), ny = isnan(y->s);
  if (nx != ny) return nx ? 1 : -1;
  if (!nx && x->s != y->s) return x->s > y->s ? -1 : 1;
  return (x->p > y->p) - (x->p < y->p);
}

int dco_row_evict(dco_row* r, int budget, const float* scores_f32) {
  int n = r->n, d = r->d;
  if (!scores_f32 && !r->have_scores) return -1;
  int keep_n = budget < n ? budget : n;
  if (keep_n < 0) keep_n = 0;
  rank_item* it = (rank_item*)malloc(sizeof(rank_item) * (size_t)(n > 0 ? n : 1));
  for (int i = 0; i < n; ++i) {
    it[i].s = scores_f32 ? (double)scores_f32[i] : r->score[i];
    it[i].p = r->pos[i];
    it[i].i = i;
  }
  /* argtop_B [Algorithm 1]: sort by the ranking, keep the first keep_n. */
  qsort(it, (size_t)n, sizeof(rank_item), rank_cmp);
  char* keep = (char*)calloc((size_t)(n > 0 ? n : 1), 1);
  for (int j = 0; j < keep_n; ++j) keep[it[j].i] = 1;
  /* Prune: survivors stay in ascending position order with their state. */
  int w = 0;
  for (int i = 0; i < n; ++i) {
    if (!keep[i]) continue;
    if (w != i) {
      memmove(r->kb + (size_t)w * d, r->kb + (size_t)i * d, sizeof(uint16_t) * d);
      memmove(r->vb + (size_t)w * d, r->vb + (size_t)i * d, sizeof(uint16_t) * d);
      memmove(r->k + (size_t)w * d, r->k + (size_t)i * d, sizeof(double) * d);
      memmove(r->v + (size_t)w * d, r->v + (size_t)i * d, sizeof(double) * d);
      r->pos[w] = r->pos[i];
      r->acc[w] = r->acc[i];
      r->S[w] = r->S[i];
      r->Z[w] = r->Z[i];
      r->Sp[w] = r->Sp[i];
      r->Zp[w] = r->Zp[i];
      r->score[w] = r->score[i];
    }
    w++;
  }
  r->n = w;
  r->have_scores = 0;
  free(it); free(keep);
  return w;
}

int dco_row_len(const dco_row* r) { return r->n; }

void dco_row_positions(const dco_row* r, int64_t* pos) {
  memcpy(pos, r->pos, sizeof(int64_t) * (size_t)r->n);
}

void dco_row_kv_bits(const dco_row* r, uint16_t* k, uint16_t* v) {
  memcpy(k, r->kb, sizeof(uint16_t) * (size_t)r->n * r->d);
  memcpy(v, r->vb, sizeof(uint16_t) * (size_t)r->n * r->d);
}

void dco_row_window_sums(const dco_row* r, double* S, double* Z, double* acc) {
  if (S) memcpy(S, r->S, sizeof(double) * (size_t)r->n);
  if (Z) memcpy(Z, r->Z, sizeof(double) * (size_t)r->n);
  if (acc) memcpy(acc, r->acc, sizeof(double) * (size_t)r->n);
}

/* Heuristic scorers on the same path (the baselines the paper compares with,
 * Sec. 2 and Sec. 4): scorer 1, H2O: the cumulative attention mass each token
 * received since insertion (needs alpha_mode 1); scorer 2, StreamingLLM: the
 * first n_sinks positions rank first (score 3e38, ties by position), then the
 * most recent tokens (score = position - newest position). Scores are for the
 * row as the last decode step left it (ascending positions). Returns 0, or -1
 * for an unknown scorer or scorer 1 without cumulative mass. */
int dco_row_heuristic_scores(const dco_row* r, int scorer, int n_sinks, double* score) {
  if (scorer == 1) {
    if (r->alpha_mode != 1) return -1;
    for (int i = 0; i < r->n; ++i) score[i] = r->acc[i];
    return 0;
  }
  if (scorer == 2) {
    const int64_t newest = r->seen - 1;
    for (int i = 0; i < r->n; ++i)
      score[i] = r->pos[i] < (int64_t)n_sinks ? 3.0e38 : (double)(r->pos[i] - newest);
    return 0;
  }
  return -1;
}

void dco_row_window_sums_prior(const dco_row* r, double* S, double* Z) {
  if (S) memcpy(S, r->Sp, sizeof(double) * (size_t)r->n);
  if (Z) memcpy(Z, r->Zp, sizeof(double) * (size_t)r->n);
}

/* ------------------------------------------------------------------------
 * Training side (App. C): the Plackett-Luce log-partition over size-B subsets
 * and Gumbel-top-B selection.
 * ---------------------------------------------------------------------- */

/* log Z = log sum_{|a| = B} exp(sum_{i in a} s_i / tau), as the log of the
 * elementary symmetric polynomial e_B(x) of x_i = exp(s_i / tau): items are
 * added one at a time, e_k <- e_k + x_i e_{k-1} (highest k first), in log
 * space. Returns -inf when B > L. */
static double log_add(double a, double b) {
  if (a == -INFINITY) return b;
  if (b == -INFINITY) return a;
  const double m = a > b ? a : b;
  return m + log1p(exp(-fabs(a - b)));
}

double dco_pl_logz(const double* s, int L, int B, double tau) {
  if (B < 0 || L < 0) return NAN;
  double* e = (double*)malloc(sizeof(double) * (size_t)(B + 1));
  if (!e) return NAN;
  e[0] = 0.0;
  for (int k = 1; k <= B; ++k) e[k] = -INFINITY;
  for (int i = 0; i < L; ++i) {
    const double y = s[i] / tau;
    for (int k = B; k >= 1; --k) e[k] = log_add(e[k], y + e[k - 1]);
  }
  const double out = e[B];
  free(e);
  return out;
}

/* Gumbel-top-B: the perturbed scores v_i = fl32(fl32(s_i / tau) + g_i) (each
 * operation rounded to fp32, as the device computes them), sorted by (value
 * descending, index ascending); the first B indices, written ascending. A NaN
 * value ranks below every number. Returns 0, or -1 on bad arguments. */
typedef struct {
  float v;
  int i;
} gt_item;

static int gt_cmp(const void* pa, const void* pb) {
  const gt_item* a = (const gt_item*)pa;
  const gt_item* b = (const gt_item*)pb;
  const int an = a->v != a->v, bn = b->v != b->v;
  if (an != bn) return an - bn; /* NaN last */
  if (!an) {
    if (a->v > b->v) return -1;
    if (a->v < b->v) return 1;
  }
  return (a->i > b->i) - (a->i < b->i);
}

static int int_cmp(const void* pa, const void* pb) {
  const int a = *(const int*)pa, b = *(const int*)pb;
  return (a > b) - (a < b);
}

int dco_gumbel_topb(const float* s, const float* g, int L, int B, float tau, int* idx) {
  if (L < 1 || B < 1 || B > L || !(tau > 0.f)) return -1;
  gt_item* it = (gt_item*)malloc(sizeof(gt_item) * (size_t)L);
  if (!it) return -1;
  for (int i = 0; i < L; ++i) {
    volatile float y = s[i] / tau; /* fp32 quotient */
    volatile float v = y + g[i];   /* fp32 sum */
    it[i].v = v == 0.f ? 0.f : v;  /* -0 ranks as +0 */
    it[i].i = i;
  }
  qsort(it, (size_t)L, sizeof *it, gt_cmp);
  for (int k = 0; k < B; ++k) idx[k] = it[k].i;
  qsort(idx, (size_t)B, sizeof(int), int_cmp);
  free(it);
  return 0;
}

/* ------------------------------------------------------------------------
 * Global token mode (Sec. 3.1.1: the features of a token pool all heads and
 * layers; one policy, one argtop_B per sequence). A sequence is R rows (its
 * layers x KV heads) sharing one token set: the same positions in the same
 * order in every row.
 * ---------------------------------------------------------------------- */

typedef struct {
  int n;
  int64_t* pos;  /* [n] ascending */
  double* za;    /* [n]: sum over the sequence's (row, head) pairs of a */
  double* sa;    /* [n]: the same sum weighted by each head's entropy */
} seq_win;

struct dco_seq {
  int R, d, G, w, alpha_mode, cap;
  int n;
  int64_t seen;
  uint16_t *kb, *vb; /* [R][cap][d] */
  double *k, *v;     /* [R][cap][d] */
  int64_t* pos;      /* [cap] */
  double* acc;       /* [cap] cumulative alpha */
  double *S, *Z, *Sp, *Zp;
  double* score;
  int have_scores;
  seq_win* win;
  int win_count, win_next;
};

static void seq_win_clear(seq_win* e) {
  free(e->pos); free(e->za); free(e->sa);
  memset(e, 0, sizeof *e);
}

void dco_seq_free(dco_seq* s) {
  if (!s) return;
  if (s->win)
    for (int i = 0; i < s->w; ++i) seq_win_clear(&s->win[i]);
  free(s->win); free(s->kb); free(s->vb); free(s->k); free(s->v); free(s->pos); free(s->acc);
  free(s->S); free(s->Z); free(s->Sp); free(s->Zp); free(s->score);
  free(s);
}

dco_seq* dco_seq_new(int R, int d, int G, int w, int alpha_mode, int cap) {
  if (R <= 0 || d <= 0 || G <= 0 || w <= 0 || cap <= 0 || (alpha_mode != 0 && alpha_mode != 1)) return NULL;
  dco_seq* s = (dco_seq*)calloc(1, sizeof *s);
  if (!s) return NULL;
  s->R = R; s->d = d; s->G = G; s->w = w; s->alpha_mode = alpha_mode; s->cap = cap;
  const size_t kv = (size_t)R * cap * d;
  s->kb = (uint16_t*)calloc(kv, sizeof(uint16_t));
  s->vb = (uint16_t*)calloc(kv, sizeof(uint16_t));
  s->k = (double*)calloc(kv, sizeof(double));
  s->v = (double*)calloc(kv, sizeof(double));
  s->pos = (int64_t*)calloc((size_t)cap, sizeof(int64_t));
  s->acc = (double*)calloc((size_t)cap, sizeof(double));
  s->S = (double*)calloc((size_t)cap, sizeof(double));
  s->Z = (double*)calloc((size_t)cap, sizeof(double));
  s->Sp = (double*)calloc((size_t)cap, sizeof(double));
  s->Zp = (double*)calloc((size_t)cap, sizeof(double));
  s->score = (double*)calloc((size_t)cap, sizeof(double));
  s->win = (seq_win*)calloc((size_t)w, sizeof(seq_win));
  if (!s->kb || !s->vb || !s->k || !s->v || !s->pos || !s->acc || !s->S || !s->Z || !s->Sp || !s->Zp ||
      !s->score || !s->win) {
    dco_seq_free(s);
    return NULL;
  }
  return s;
}

/* The token of row r at slot i. */
static void seq_put(dco_seq* s, int r, int i, const uint16_t* k, const uint16_t* v) {
  const size_t o = ((size_t)r * s->cap + i) * s->d;
  for (int c = 0; c < s->d; ++c) {
    s->kb[o + c] = k[c];
    s->vb[o + c] = v[c];
    s->k[o + c] = bf16_to_double(k[c]);
    s->v[o + c] = bf16_to_double(v[c]);
  }
}

int dco_seq_append(dco_seq* s, const uint16_t* k, const uint16_t* v, int T) {
  if (T < 0 || s->n + T > s->cap) return -1;
  for (int t = 0; t < T; ++t) {
    for (int r = 0; r < s->R; ++r)
      seq_put(s, r, s->n, k + ((size_t)r * T + t) * s->d, v + ((size_t)r * T + t) * s->d);
    s->pos[s->n] = s->seen;
    s->acc[s->n] = 0.0;
    s->n += 1;
    s->seen += 1;
  }
  s->have_scores = 0;
  return 0;
}

int dco_seq_step(dco_seq* s, const uint16_t* q, const uint16_t* k_new, const uint16_t* v_new,
                 const float* mlp, int hidden, int layernorm, double* o, double* feat, double* score) {
  const int R = s->R, d = s->d, G = s->G;
  if (s->n + 1 > s->cap) return -1;
  /* Algorithm 1: every row's cache already holds the new pair. */
  for (int r = 0; r < R; ++r) seq_put(s, r, s->n, k_new + (size_t)r * d, v_new + (size_t)r * d);
  s->pos[s->n] = s->seen;
  s->acc[s->n] = 0.0;
  s->n += 1;
  s->seen += 1;
  const int n = s->n;
  const int N = R * G; /* attention heads pooled per token */
  double* a = (double*)malloc(sizeof(double) * (size_t)R * n * G);
  double* Hh = (double*)malloc(sizeof(double) * (size_t)R * G);
  double* qd = (double*)malloc(sizeof(double) * (size_t)G * d);
  double* oo = (double*)malloc(sizeof(double) * (size_t)G * d);
  double* Kr = (double*)malloc(sizeof(double) * (size_t)n * d);
  double* Vr = (double*)malloc(sizeof(double) * (size_t)n * d);
  for (int r = 0; r < R; ++r) {
    for (int i = 0; i < G * d; ++i) qd[i] = bf16_to_double(q[(size_t)r * G * d + i]);
    memcpy(Kr, s->k + (size_t)r * s->cap * d, sizeof(double) * (size_t)n * d);
    memcpy(Vr, s->v + (size_t)r * s->cap * d, sizeof(double) * (size_t)n * d);
    attend_rows(qd, Kr, Vr, n, d, G, a + (size_t)r * n * G, oo, Hh + (size_t)r * G);
    if (o) memcpy(o + (size_t)r * G * d, oo, sizeof(double) * (size_t)G * d);
  }
  /* This step's pooled mass and entropy-weighted mass per token, kept (keyed
   * by position) in the window of the last w steps [Sec. 3.1.1, H_i]. */
  seq_win* e = &s->win[s->win_next];
  seq_win_clear(e);
  e->n = n;
  e->pos = (int64_t*)malloc(sizeof(int64_t) * (size_t)n);
  e->za = (double*)calloc((size_t)n, sizeof(double));
  e->sa = (double*)calloc((size_t)n, sizeof(double));
  memcpy(e->pos, s->pos, sizeof(int64_t) * (size_t)n);
  for (int i = 0; i < n; ++i)
    for (int r = 0; r < R; ++r)
      for (int h = 0; h < G; ++h) {
        const double ah = a[((size_t)r * n + i) * G + h];
        e->za[i] += ah;
        e->sa[i] += ah * Hh[(size_t)r * G + h];
      }
  s->win_next = (s->win_next + 1) % s->w;
  if (s->win_count < s->w) s->win_count += 1;
  const int newest_entry = (s->win_next + s->w - 1) % s->w;

  double* x = (double*)malloc(sizeof(double) * (size_t)n * 5);
  const int64_t newest = s->pos[n - 1];
  const double pos_den = (double)(newest > 1 ? newest : 1);
  for (int i = 0; i < n; ++i) {
    /* alpha_i: mean over every (row, head) pair of the mass token i receives */
    double mean = 0.0;
    for (int r = 0; r < R; ++r)
      for (int h = 0; h < G; ++h) mean += a[((size_t)r * n + i) * G + h];
    mean /= N;
    double alpha = mean;
    if (s->alpha_mode == 1) {
      s->acc[i] += mean;
      alpha = s->acc[i];
    }
    /* sigma_i: population variance over the same pairs */
    double var = 0.0;
    for (int r = 0; r < R; ++r)
      for (int h = 0; h < G; ++h) {
        const double dv = a[((size_t)r * n + i) * G + h] - mean;
        var += dv * dv;
      }
    var /= N;
    /* |v_i|: mean over the rows of the value norm */
    double vn = 0.0;
    for (int r = 0; r < R; ++r) {
      double ss = 0.0;
      const double* vv = s->v + ((size_t)r * s->cap + i) * d;
      for (int c = 0; c < d; ++c) ss += vv[c] * vv[c];
      vn += sqrt(ss);
    }
    vn /= R;
    /* H_i over the window of recent steps, pooled */
    double S = 0.0, Z = 0.0, Sp = 0.0, Zp = 0.0;
    for (int qi = 0; qi < s->win_count; ++qi) {
      const seq_win* we = &s->win[qi];
      const int j = find_pos(we->pos, we->n, s->pos[i]);
      if (j < 0) continue;
      Z += we->za[j];
      S += we->sa[j];
      if (qi != newest_entry) {
        Zp += we->za[j];
        Sp += we->sa[j];
      }
    }
    s->S[i] = S; s->Z[i] = Z; s->Sp[i] = Sp; s->Zp[i] = Zp;
    x[(size_t)i * 5 + 0] = alpha;
    x[(size_t)i * 5 + 1] = vn;
    x[(size_t)i * 5 + 2] = var;
    x[(size_t)i * 5 + 3] = Z > 0.0 ? S / Z : 0.0;
    x[(size_t)i * 5 + 4] = (double)s->pos[i] / pos_den;
  }
  dco_policy(x, n, mlp, hidden, layernorm, s->score);
  s->have_scores = 1;
  if (feat) memcpy(feat, x, sizeof(double) * (size_t)n * 5);
  if (score) memcpy(score, s->score, sizeof(double) * (size_t)n);
  free(a); free(Hh); free(qd); free(oo); free(Kr); free(Vr); free(x);
  return n;
}

int dco_seq_evict(dco_seq* s, int budget, const float* scores_f32) {
  const int n = s->n, d = s->d;
  if (!scores_f32 && !s->have_scores) return -1;
  int keep_n = budget < n ? budget : n;
  if (keep_n < 0) keep_n = 0;
  rank_item* it = (rank_item*)malloc(sizeof(rank_item) * (size_t)(n > 0 ? n : 1));
  for (int i = 0; i < n; ++i) {
    it[i].s = scores_f32 ? (double)scores_f32[i] : s->score[i];
    it[i].p = s->pos[i];
    it[i].i = i;
  }
  /* one argtop_B for the whole sequence [Algorithm 1] */
  qsort(it, (size_t)n, sizeof(rank_item), rank_cmp);
  char* keep = (char*)calloc((size_t)(n > 0 ? n : 1), 1);
  for (int j = 0; j < keep_n; ++j) keep[it[j].i] = 1;
  /* prune every row the same way: survivors in ascending position order */
  int w = 0;
  for (int i = 0; i < n; ++i) {
    if (!keep[i]) continue;
    if (w != i) {
      for (int r = 0; r < s->R; ++r) {
        const size_t src = ((size_t)r * s->cap + i) * d, dst = ((size_t)r * s->cap + w) * d;
        memmove(s->kb + dst, s->kb + src, sizeof(uint16_t) * (size_t)d);
        memmove(s->vb + dst, s->vb + src, sizeof(uint16_t) * (size_t)d);
        memmove(s->k + dst, s->k + src, sizeof(double) * (size_t)d);
        memmove(s->v + dst, s->v + src, sizeof(double) * (size_t)d);
      }
      s->pos[w] = s->pos[i];
      s->acc[w] = s->acc[i];
      s->S[w] = s->S[i]; s->Z[w] = s->Z[i]; s->Sp[w] = s->Sp[i]; s->Zp[w] = s->Zp[i];
      s->score[w] = s->score[i];
    }
    ++w;
  }
  s->n = w;
  s->have_scores = 0;
  free(it);
  free(keep);
  return w;
}

int dco_seq_len(const dco_seq* s) { return s->n; }

void dco_seq_positions(const dco_seq* s, int64_t* pos) { memcpy(pos, s->pos, sizeof(int64_t) * (size_t)s->n); }

void dco_seq_kv_bits(const dco_seq* s, int r, uint16_t* k, uint16_t* v) {
  const size_t o = (size_t)r * s->cap * s->d, m = (size_t)s->n * s->d;
  memcpy(k, s->kb + o, sizeof(uint16_t) * m);
  memcpy(v, s->vb + o, sizeof(uint16_t) * m);
}

void dco_seq_window_sums_prior(const dco_seq* s, double* S, double* Z) {
  if (S) memcpy(S, s->Sp, sizeof(double) * (size_t)s->n);
  if (Z) memcpy(Z, s->Zp, sizeof(double) * (size_t)s->n);
}
