/*
 * Float64 CPU oracle for the token-aware verifier (Pro-Router, Section 3.1).
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the slow, plain reference that the
 * GPU path is checked against.  Only the tests, the smoke check and the CPU
 * baseline leg of the benchmark may load it; the product path never does.  It
 * shares no source, header, table or helper with the CUDA library.
 *
 * Every quantity is the textbook definition written out in double precision:
 *
 *   per generated token t (one logit row x over a vocabulary of V tokens),
 *   Eq. 3 and the text under it:
 *     p_t(v)  = exp(x_v) / sum_u exp(x_u)           softmax of the stored row
 *     l_t     = log p_t(y_t)                         emitted-token log-prob
 *     m_t     = max_v p_t(v)                         max probability
 *     H_t^K   = -sum_{v in top-K} p_t(v) log p_t(v)  top-K entropy, K = 20
 *     h_t     = -H_t^K                               negative top-K entropy
 *     rho_t   = t / T                                position fraction (t 1-based)
 *   plus the statistics the verifier's data path also reports:
 *     margin  = p(i1) - p(i2)   (first and second token in the order
 *                                "value descending, index ascending")
 *     H       = -sum_v p log p  full-vocabulary entropy, 0 log 0 := 0
 *     LSE     = log sum_v exp(x_v),  x1 = x_{i1}
 *
 *   per request (a ragged run of T rows), mean pool of Section 3.1 read as a
 *   linear scorer over pooled features:
 *     a = [mean l, min l, mean m, min m, mean margin, min margin,
 *          mean(-H), min(-H), mean h, min h, mean rho]
 *     z = w . a + b,  score = sigmoid(z),  ship iff score >= tau  (Section 3.1,
 *     "ships when p >= tau").
 *
 * Readings where the paper is silent (they are listed with their reasons in
 * the design notes of this repository):
 *   - top-K uses the raw softmax probabilities (renorm = 0); renorm = 1 gives
 *     the variant renormalised over the K kept tokens;
 *   - ties in the token order are broken by the lower index;
 *   - a row holding NaN or +inf, or no finite value at all, is "non-finite":
 *     its features are NaN and its indices -1; -inf is a masked token (p = 0);
 *   - a chosen id outside [0, V) gives l = NaN;
 *   - a request with a non-finite or bad-chosen row has NaN aggregates, NaN
 *     score and does not ship; an empty request (T = 0) has NaN aggregates,
 *     score 0 and does not ship.
 *
 * Parity of this oracle is pinned by closed forms (uniform row, one-hot row,
 * two-way tie), by brute force against library routines on tiny rows and by
 * invariances; see the oracle pin tests.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define OR_DTYPE_F32 0
#define OR_DTYPE_BF16 1

#define OR_FLAG_NONFINITE 1u
#define OR_FLAG_BAD_CHOSEN 2u
#define OR_FLAG_EMPTY_REQ 4u
#define OR_FLAG_BAD_OFFSETS 8u

#define OR_NFEAT 8
#define OR_NAGG 11

/* feature slots of one row record */
#define F_LOGP 0
#define F_MAXP 1
#define F_MARGIN 2
#define F_ENT 3
#define F_TOPK 4
#define F_RHO 5
#define F_LSE 6
#define F_X1 7

/* ---- reading one element ------------------------------------------------ */

static double read_elem(const void* row, int dtype, int64_t v) {
  if (dtype == OR_DTYPE_BF16) {
    /* bfloat16 is the high half of an IEEE binary32 */
    uint16_t h = ((const uint16_t*)row)[v];
    uint32_t bits = ((uint32_t)h) << 16;
    float f;
    memcpy(&f, &bits, sizeof f);
    return (double)f;
  }
  return (double)((const float*)row)[v];
}

/* a comes before b in the order "value descending, index ascending" */
static int before(double xa, int64_t ia, double xb, int64_t ib) {
  if (xa > xb) return 1;
  if (xa < xb) return 0;
  return ia < ib;
}

/* ---- one row: Eq. 3 -------------------------------------------------------- */

int oracle_row_features(const void* row, int dtype, int64_t V, int32_t chosen,
                        int32_t K, int32_t renorm, double* feat, int32_t* idx,
                        uint32_t* flags_out) {
  uint32_t flags = 0;
  for (int j = 0; j < OR_NFEAT; ++j) feat[j] = NAN;
  idx[0] = -1;
  idx[1] = -1;
  if (V <= 0 || K <= 0 || (dtype != OR_DTYPE_F32 && dtype != OR_DTYPE_BF16))
    return -1;

  /* the row as doubles */
  double* x = (double*)malloc((size_t)V * sizeof(double));
  if (!x) return -4;
  int any_finite = 0, bad = 0;
  for (int64_t v = 0; v < V; ++v) {
    x[v] = read_elem(row, dtype, v);
    if (isnan(x[v]) || (isinf(x[v]) && x[v] > 0)) bad = 1;
    if (isfinite(x[v])) any_finite = 1;
  }
  if (chosen < 0 || (int64_t)chosen >= V) flags |= OR_FLAG_BAD_CHOSEN;
  if (bad || !any_finite) {
    flags |= OR_FLAG_NONFINITE;
    free(x);
    *flags_out = flags;
    return 0;
  }

  /* log-sum-exp: LSE = max + log sum exp(x - max) */
  double xmax = -INFINITY;
  for (int64_t v = 0; v < V; ++v)
    if (x[v] > xmax) xmax = x[v];
  double sum = 0.0;
  for (int64_t v = 0; v < V; ++v) sum += exp(x[v] - xmax);
  double lse = xmax + log(sum);

  /* full entropy H = -sum p log p with p = exp(x - LSE), 0 log 0 = 0 */
  double H = 0.0;
  for (int64_t v = 0; v < V; ++v) {
    double p = exp(x[v] - lse);
    if (p > 0.0) H -= p * log(p);
  }

  /* the top-Kc tokens in the order (value desc, index asc), by insertion into
     a sorted list; Kc covers both top-K and top-2 */
  int64_t Kc = K > 2 ? K : 2;
  if (Kc > V) Kc = V;
  double* tv = (double*)malloc((size_t)Kc * sizeof(double));
  int64_t* ti = (int64_t*)malloc((size_t)Kc * sizeof(int64_t));
  if (!tv || !ti) {
    free(x);
    free(tv);
    free(ti);
    return -4;
  }
  int64_t n = 0;
  for (int64_t v = 0; v < V; ++v) {
    if (n == Kc && !before(x[v], v, tv[Kc - 1], ti[Kc - 1])) continue;
    int64_t pos = (n < Kc) ? n : Kc - 1;
    while (pos > 0 && before(x[v], v, tv[pos - 1], ti[pos - 1])) {
      tv[pos] = tv[pos - 1];
      ti[pos] = ti[pos - 1];
      --pos;
    }
    tv[pos] = x[v];
    ti[pos] = v;
    if (n < Kc) ++n;
  }

  double p1 = exp(tv[0] - lse);
  double p2 = (V >= 2) ? exp(tv[1] - lse) : 0.0;
  idx[0] = (int32_t)ti[0];
  idx[1] = (V >= 2) ? (int32_t)ti[1] : -1;

  /* top-K entropy over the K most probable tokens (raw p, or renormalised) */
  int64_t kk = (int64_t)K < V ? (int64_t)K : V;
  double topk_mass = 0.0;
  for (int64_t k = 0; k < kk; ++k) topk_mass += exp(tv[k] - lse);
  double HK = 0.0;
  for (int64_t k = 0; k < kk; ++k) {
    double p = exp(tv[k] - lse);
    if (renorm) p = p / topk_mass;
    if (p > 0.0) HK -= p * log(p);
  }

  feat[F_LOGP] = (flags & OR_FLAG_BAD_CHOSEN) ? NAN : x[chosen] - lse;
  feat[F_MAXP] = p1;
  feat[F_MARGIN] = p1 - p2;
  feat[F_ENT] = H;
  feat[F_TOPK] = -HK;
  feat[F_RHO] = 0.0; /* filled by the caller, which knows t and T */
  feat[F_LSE] = lse;
  feat[F_X1] = tv[0];

  free(x);
  free(tv);
  free(ti);
  *flags_out = flags;
  return 0;
}

/* ---- one request: pool, score, threshold --------------------------------- */

static double nan_min(double a, double b) {
  if (isnan(a) || isnan(b)) return NAN;
  return a < b ? a : b;
}

int oracle_request_score(const double* feat, int64_t T, const uint32_t* row_flags,
                         const double* w, double b, double tau, double* agg,
                         double* score, uint8_t* ship, uint32_t* req_flags) {
  uint32_t flags = 0;
  for (int j = 0; j < OR_NAGG; ++j) agg[j] = NAN;
  if (T <= 0) {
    *req_flags = OR_FLAG_EMPTY_REQ;
    *score = 0.0;
    *ship = 0;
    return 0;
  }
  for (int64_t t = 0; t < T; ++t) flags |= row_flags[t];
  if (flags & (OR_FLAG_NONFINITE | OR_FLAG_BAD_CHOSEN)) {
    *req_flags = flags;
    *score = NAN;
    *ship = 0;
    return 0;
  }
  /* five pooled features: l, m, margin, -H, h */
  static const int src[5] = {F_LOGP, F_MAXP, F_MARGIN, F_ENT, F_TOPK};
  static const double sgn[5] = {1.0, 1.0, 1.0, -1.0, 1.0};
  for (int f = 0; f < 5; ++f) {
    double s = 0.0, mn = INFINITY;
    for (int64_t t = 0; t < T; ++t) {
      double val = sgn[f] * feat[t * OR_NFEAT + src[f]];
      s += val;
      mn = nan_min(mn, val);
    }
    agg[2 * f] = s / (double)T;
    agg[2 * f + 1] = mn;
  }
  double srho = 0.0;
  for (int64_t t = 0; t < T; ++t) srho += feat[t * OR_NFEAT + F_RHO];
  agg[10] = srho / (double)T;

  double z = b;
  for (int j = 0; j < OR_NAGG; ++j) z += w[j] * agg[j];
  double s = 1.0 / (1.0 + exp(-z));
  *score = s;
  *ship = (s >= tau) ? 1 : 0;
  *req_flags = flags;
  return 0;
}

/* ---- a batch: rows -> requests ------------------------------------------- */

typedef struct {
  const void* logits;
  int dtype;
  int64_t n_rows, V, row_stride;
  const int32_t* chosen;
  int32_t K, renorm;
  double* feat;
  int32_t* idx;
  uint32_t* row_flags;
  int64_t lo, hi;
  int status;
} row_job;

static void* run_rows(void* arg) {
  row_job* j = (row_job*)arg;
  size_t esz = (j->dtype == OR_DTYPE_BF16) ? 2 : 4;
  for (int64_t r = j->lo; r < j->hi; ++r) {
    const char* row = (const char*)j->logits + (size_t)r * (size_t)j->row_stride * esz;
    int st = oracle_row_features(row, j->dtype, j->V, j->chosen[r], j->K, j->renorm,
                                 j->feat + r * OR_NFEAT, j->idx + 2 * r,
                                 j->row_flags + r);
    if (st != 0) j->status = st;
  }
  return NULL;
}

/*
 * Full-response verification of a batch: n_rows logit rows (row-major, stride
 * row_stride elements), request r owning rows [offsets[r], offsets[r+1]).
 * Rows are spread over n_threads POSIX threads; everything else is serial.
 */
int oracle_route(const void* logits, int dtype, int64_t n_rows, int64_t V,
                 int64_t row_stride, const int32_t* chosen, const int64_t* offsets,
                 int32_t n_req, int32_t K, int32_t renorm, const double* w, double b,
                 double tau, int32_t n_threads, double* feat, int32_t* idx,
                 uint32_t* row_flags, double* agg, double* score, uint8_t* ship,
                 uint32_t* req_flags) {
  if (n_rows < 0 || V <= 0 || row_stride < V || n_req < 0 || n_threads <= 0)
    return -1;
  if (n_threads > 256) n_threads = 256;
  if (n_threads > n_rows && n_rows > 0) n_threads = (int32_t)n_rows;

  row_job jobs[256];
  pthread_t th[256];
  int nt = n_rows > 0 ? n_threads : 0;
  for (int i = 0; i < nt; ++i) {
    row_job* j = &jobs[i];
    j->logits = logits;
    j->dtype = dtype;
    j->n_rows = n_rows;
    j->V = V;
    j->row_stride = row_stride;
    j->chosen = chosen;
    j->K = K;
    j->renorm = renorm;
    j->feat = feat;
    j->idx = idx;
    j->row_flags = row_flags;
    j->lo = n_rows * i / nt;
    j->hi = n_rows * (i + 1) / nt;
    j->status = 0;
  }
  for (int i = 1; i < nt; ++i) pthread_create(&th[i], NULL, run_rows, &jobs[i]);
  if (nt > 0) run_rows(&jobs[0]);
  for (int i = 1; i < nt; ++i) pthread_join(th[i], NULL);
  for (int i = 0; i < nt; ++i)
    if (jobs[i].status != 0) return jobs[i].status;

  /* requests: position fraction, then pool and score */
  for (int32_t r = 0; r < n_req; ++r) {
    int64_t lo = offsets[r], hi = offsets[r + 1];
    if (lo < 0 || hi < lo || hi > n_rows) {
      for (int j = 0; j < OR_NAGG; ++j) agg[(int64_t)r * OR_NAGG + j] = NAN;
      score[r] = NAN;
      ship[r] = 0;
      req_flags[r] = OR_FLAG_BAD_OFFSETS;
      continue;
    }
    int64_t T = hi - lo;
    for (int64_t t = 1; t <= T; ++t) {
      double* f = feat + (lo + t - 1) * OR_NFEAT;
      if (!(row_flags[lo + t - 1] & OR_FLAG_NONFINITE)) f[F_RHO] = (double)t / (double)T;
    }
    oracle_request_score(feat + lo * OR_NFEAT, T, row_flags + lo, w, b, tau,
                         agg + (int64_t)r * OR_NAGG, score + r, ship + r, req_flags + r);
  }
  return 0;
}
