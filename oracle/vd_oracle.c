/*
 * vd_oracle.c -- fp64 CPU oracle for ValueDiff KV-cache eviction.
 *
 * TEST INFRASTRUCTURE ONLY: the plain definition the CUDA path is checked
 * against.  No blocking, fusion or reordering beyond what the definitions
 * state; each function names the passage of the paper it writes out.
 * Shares nothing with the CUDA library.
 *
 * Parity pins (tests/): closed-form fixtures, the law-of-cosines identity
 * (Eq. decomp), the uniform-attention reconstruction error (Eq. recon_error),
 * the Dirichlet(1,...,1) expectation (App. A), translation/scale/permutation
 * properties, and a brute-force O(n^2) ranking for top-N.
 */
#include "vd_oracle.h"

#include <math.h>
#include <pthread.h>
#include <stdlib.h>
#include <string.h>

double vdo_bf16_to_double(uint16_t bits) {
  /* A bf16 value is the upper half of an IEEE binary32 value. */
  uint32_t w = (uint32_t)bits << 16;
  float f;
  memcpy(&f, &w, sizeof f);
  return (double)f;
}

/* Neumaier's improved Kahan-Babuska summation (Neumaier 1974): a running sum
 * plus a correction term that collects the low-order bits each add loses. */
void vdo_sum_rows(const uint16_t* v, int64_t n, int64_t d, double* out) {
  for (int64_t c = 0; c < d; ++c) {
    double sum = 0.0, corr = 0.0;
    for (int64_t i = 0; i < n; ++i) {
      double x = vdo_bf16_to_double(v[i * d + c]);
      double t = sum + x;
      if (fabs(sum) >= fabs(x))
        corr += (sum - t) + x;
      else
        corr += (x - t) + sum;
      sum = t;
    }
    out[c] = sum + corr;
  }
}

/* Eq. (vd), right half: the cache mean over the n cached tokens. */
void vdo_mean(const uint16_t* v, int64_t n, int64_t d, double* out) {
  vdo_sum_rows(v, n, d, out);
  for (int64_t c = 0; c < d; ++c) out[c] /= (double)n;
}

/* Eq. (vd), left half, and the two endpoint variants of Sec. 3.2:
 *   L2   s_j = sqrt(sum_c (v_jc - mean_c)^2)          (Euclidean norm)
 *   DIR  s_j = 1 - <v_j, mean> / (||v_j|| ||mean||)   (directional)
 *   NORM s_j = ||v_j||                                 (magnitude)       */
void vdo_scores(const uint16_t* v, int64_t n, int64_t d, int variant, double* out) {
  double* mean = NULL;
  double mean_norm = 0.0;
  if (variant != VDO_NORM) {
    mean = (double*)malloc((size_t)d * sizeof(double));
    vdo_mean(v, n, d, mean);
    double mm = 0.0;
    for (int64_t c = 0; c < d; ++c) mm += mean[c] * mean[c];
    mean_norm = sqrt(mm);
  }
  for (int64_t j = 0; j < n; ++j) {
    const uint16_t* row = v + j * d;
    if (variant == VDO_L2) {
      double acc = 0.0;
      for (int64_t c = 0; c < d; ++c) {
        double diff = vdo_bf16_to_double(row[c]) - mean[c];
        acc += diff * diff;
      }
      out[j] = sqrt(acc);
    } else if (variant == VDO_DIR) {
      double dot = 0.0, vv = 0.0;
      for (int64_t c = 0; c < d; ++c) {
        double x = vdo_bf16_to_double(row[c]);
        dot += x * mean[c];
        vv += x * x;
      }
      double vnorm = sqrt(vv);
      /* The paper leaves cos undefined for a zero vector; cos := 0 here. */
      double cosv = (vnorm == 0.0 || mean_norm == 0.0) ? 0.0 : dot / (vnorm * mean_norm);
      out[j] = 1.0 - cosv;
    } else {
      double vv = 0.0;
      for (int64_t c = 0; c < d; ++c) {
        double x = vdo_bf16_to_double(row[c]);
        vv += x * x;
      }
      out[j] = sqrt(vv);
    }
  }
  free(mean);
}

/* App. A, Eq. (app_fastcaote): FastCAOTE evaluates the renormalisation
 * identity at an observed attention vector and replaces the attention output
 * by the cache mean, which leaves a_j / (1 - a_j) times the distance from the
 * mean. */
void vdo_scores_weighted(const uint16_t* v, int64_t n, int64_t d, int variant, const double* a,
                         double* out) {
  vdo_scores(v, n, d, variant, out);
  for (int64_t j = 0; j < n; ++j) {
    if (a[j] >= 0.0 && a[j] < 1.0)
      out[j] *= a[j] / (1.0 - a[j]);
    else
      out[j] = NAN;
  }
}

/* Sec. 3.1: the standard deviation over tokens of the L2 distance from the
 * cache mean (divisor n), from a compensated two-pass computation. */
double vdo_dispersion(const uint16_t* x, int64_t n, int64_t d) {
  double* s = (double*)malloc((size_t)n * sizeof(double));
  vdo_scores(x, n, d, VDO_L2, s);
  double sum = 0.0, corr = 0.0;
  for (int64_t j = 0; j < n; ++j) {
    double t = sum + s[j];
    corr += fabs(sum) >= fabs(s[j]) ? (sum - t) + s[j] : (s[j] - t) + sum;
    sum = t;
  }
  const double m = (sum + corr) / (double)n;
  double ss = 0.0;
  for (int64_t j = 0; j < n; ++j) ss += (s[j] - m) * (s[j] - m);
  free(s);
  return sqrt(ss / (double)n);
}

typedef struct {
  double score;
  int32_t index;
} vdo_ranked;

/* Order of Eq. (eviction)'s top-N: higher score first; among equal scores the
 * lower (earlier) cache slot first.  A NaN score (only an invalid input makes
 * one) ranks below every number, so it is evicted first; NaNs tie among
 * themselves.  -0 and +0 are equal. */
static int vdo_rank_cmp(const void* pa, const void* pb) {
  const vdo_ranked* a = (const vdo_ranked*)pa;
  const vdo_ranked* b = (const vdo_ranked*)pb;
  const int a_nan = isnan(a->score), b_nan = isnan(b->score);
  if (a_nan != b_nan) return a_nan - b_nan;
  if (a->score > b->score) return -1;
  if (a->score < b->score) return 1;
  return (a->index > b->index) - (a->index < b->index);
}

static int vdo_int_cmp(const void* pa, const void* pb) {
  int32_t a = *(const int32_t*)pa, b = *(const int32_t*)pb;
  return (a > b) - (a < b);
}

/* Eq. (eviction): S = top-N(s(C)).  Sort all n tokens by the order above,
 * take the first N, and return them in ascending slot order (the order
 * gather(.) keeps them in). */
int64_t vdo_select_top_n(const double* scores, int64_t n, int64_t N, int32_t* kept) {
  if (n <= N) {
    for (int64_t j = 0; j < n; ++j) kept[j] = (int32_t)j;
    return n;
  }
  vdo_ranked* r = (vdo_ranked*)malloc((size_t)n * sizeof(vdo_ranked));
  for (int64_t j = 0; j < n; ++j) {
    r[j].score = scores[j];
    r[j].index = (int32_t)j;
  }
  qsort(r, (size_t)n, sizeof(vdo_ranked), vdo_rank_cmp);
  for (int64_t i = 0; i < N; ++i) kept[i] = r[i].index;
  qsort(kept, (size_t)N, sizeof(int32_t), vdo_int_cmp);
  free(r);
  return N;
}

/* pi_N of Sec. 2.1: evict only when the cache exceeds the budget, then
 * K' = gather(K, S), V' = gather(V, S) -- written out of place first so the
 * gather never reads a row it already overwrote. */
int64_t vdo_evict_unit(uint16_t* k, uint16_t* v, int64_t n, int64_t d, int64_t N,
                       int variant, int32_t* kept, double* scores) {
  if (n <= N) {
    if (kept)
      for (int64_t j = 0; j < n; ++j) kept[j] = (int32_t)j;
    return n;
  }
  double* s = scores ? scores : (double*)malloc((size_t)n * sizeof(double));
  int32_t* idx = (int32_t*)malloc((size_t)N * sizeof(int32_t));
  vdo_scores(v, n, d, variant, s);
  vdo_select_top_n(s, n, N, idx);

  size_t row_bytes = (size_t)d * sizeof(uint16_t);
  uint16_t* kk = (uint16_t*)malloc((size_t)N * row_bytes);
  uint16_t* vv = (uint16_t*)malloc((size_t)N * row_bytes);
  for (int64_t r = 0; r < N; ++r) {
    memcpy(kk + r * d, k + (int64_t)idx[r] * d, row_bytes);
    memcpy(vv + r * d, v + (int64_t)idx[r] * d, row_bytes);
  }
  memcpy(k, kk, (size_t)N * row_bytes);
  memcpy(v, vv, (size_t)N * row_bytes);
  if (kept) memcpy(kept, idx, (size_t)N * sizeof(int32_t));

  free(kk);
  free(vv);
  free(idx);
  if (!scores) free(s);
  return N;
}

typedef struct {
  uint16_t* k;
  uint16_t* v;
  const int32_t* len;
  const int32_t* N_per_seq;
  int64_t u0, u1, units_per_seq, capacity, d, kept_stride;
  int variant;
  int32_t* kept;
} vdo_job;

static void* vdo_worker(void* arg) {
  vdo_job* j = (vdo_job*)arg;
  for (int64_t u = j->u0; u < j->u1; ++u) {
    int64_t s = u / j->units_per_seq;
    int64_t base = u * j->capacity * j->d;
    vdo_evict_unit(j->k + base, j->v + base, j->len[s], j->d, j->N_per_seq[s], j->variant,
                   j->kept ? j->kept + u * j->kept_stride : NULL, NULL);
  }
  return NULL;
}

int vdo_evict_units(uint16_t* k, uint16_t* v, const int32_t* len, const int32_t* N_per_seq,
                    int64_t n_units, int64_t units_per_seq, int64_t capacity, int64_t d,
                    int variant, int32_t* kept, int64_t kept_stride, int nthreads) {
  if (nthreads < 1) nthreads = 1;
  if (nthreads > n_units) nthreads = (int)(n_units > 0 ? n_units : 1);
  pthread_t* th = (pthread_t*)malloc((size_t)nthreads * sizeof(pthread_t));
  vdo_job* jobs = (vdo_job*)malloc((size_t)nthreads * sizeof(vdo_job));
  int started = 0, rc = 0;
  for (int t = 0; t < nthreads; ++t) {
    vdo_job j = {k, v, len, N_per_seq,
                 n_units * t / nthreads, n_units * (t + 1) / nthreads,
                 units_per_seq, capacity, d, kept_stride, variant, kept};
    jobs[t] = j;
    if (pthread_create(&th[t], NULL, vdo_worker, &jobs[t]) != 0) {
      rc = -1;
      break;
    }
    ++started;
  }
  for (int t = 0; t < started; ++t) pthread_join(th[t], NULL);
  free(th);
  free(jobs);
  return rc;
}
