/*
 * evict_example.c -- a C caller of libvd.so, with no Python in the process.
 *
 * It allocates a small cache with the CUDA runtime, runs one fused block
 * boundary (vd_append_evict_block: N + B -> N, Sec. 2.2 Eq. block_processing)
 * and one fused decode step (vd_append_evict_decode: N + 1 -> N) through the
 * C ABI of include/vd.h, and checks every unit against the fp64 oracle
 * (oracle/vd_oracle.c, test infrastructure) on the same bytes: ValueDiff
 * scores (Sec. 3.2 Eq. vd) within 1e-5 relative plus the fp32 rounding floor,
 * the kept set of Eq. (eviction) outside near ties, the compacted K and V
 * rows bit for bit, and len == N.  Exit status 0: every check passed.
 *
 * Built and run by tests/test_gpu_c_abi.py (gcc, the CUDA runtime, libvd.so
 * and the oracle's C source).
 */
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <cuda_runtime_api.h>

#include "vd.h"
#include "vd_oracle.h"

enum { N_SEQ = 2, N_LAYER = 2, N_HEAD = 2, D = 128, N = 300, B = 64, CAP = N + B };
enum { UNITS = N_SEQ * N_LAYER * N_HEAD, PER_SEQ = N_LAYER * N_HEAD };

static int failures = 0;

#define CHECK(cond, ...)                                   \
  do {                                                     \
    if (!(cond)) {                                         \
      fprintf(stderr, "FAIL %s:%d: ", __FILE__, __LINE__); \
      fprintf(stderr, __VA_ARGS__);                        \
      fprintf(stderr, "\n");                               \
      ++failures;                                          \
    }                                                      \
  } while (0)

#define CUDA(call)                                                          \
  do {                                                                      \
    cudaError_t e_ = (call);                                                \
    if (e_ != cudaSuccess) {                                                \
      fprintf(stderr, "CUDA error %s at %s:%d\n", cudaGetErrorString(e_),   \
              __FILE__, __LINE__);                                          \
      exit(2);                                                              \
    }                                                                       \
  } while (0)

/* xorshift64*: a fixed stream of pseudo-random numbers for the inputs. */
static uint64_t rng_state = 0x9e3779b97f4a7c15ull;
static double uniform(void) {
  rng_state ^= rng_state >> 12;
  rng_state ^= rng_state << 25;
  rng_state ^= rng_state >> 27;
  return (double)((rng_state * 0x2545f4914f6cdd1dull) >> 11) / 9007199254740992.0;
}

/* fp32 -> bf16 bit pattern, round to nearest even (finite inputs only). */
static uint16_t to_bf16(float f) {
  uint32_t x;
  memcpy(&x, &f, sizeof x);
  x += 0x7fffu + ((x >> 16) & 1u);
  return (uint16_t)(x >> 16);
}

/* A row around a per-unit centre: centre + noise (sum of four uniforms). */
static void fill_row(uint16_t* row, const float* centre) {
  for (int c = 0; c < D; ++c) {
    const double z = uniform() + uniform() + uniform() + uniform() - 2.0;
    row[c] = to_bf16((float)(centre[c] + 1.5 * z));
  }
}

static double row_norm(const uint16_t* row) {
  double s = 0.0;
  for (int c = 0; c < D; ++c) {
    const double x = vdo_bf16_to_double(row[c]);
    s += x * x;
  }
  return sqrt(s);
}

static int cmp_desc(const void* a, const void* b) {
  const double x = *(const double*)a, y = *(const double*)b;
  return (x < y) - (x > y);
}

/* One unit, one event.  pre: the n rows (K, V) the event saw, in slot order;
 * post: rows [0, N) after it; kept_gpu: the GPU's kept slots (NULL for
 * decode, which reports evicted instead); scores_gpu: [n] or NULL. */
static void check_unit(int u, const uint16_t* pre_k, const uint16_t* pre_v, int n,
                       const uint16_t* post_k, const uint16_t* post_v, const int32_t* kept_gpu,
                       int evicted_gpu, const float* scores_gpu) {
  double* s = malloc(sizeof(double) * n);
  double* sorted = malloc(sizeof(double) * n);
  double mean[D];
  int32_t* kept_ora = malloc(sizeof(int32_t) * N);
  int32_t* kept = malloc(sizeof(int32_t) * N);
  vdo_scores(pre_v, n, D, VDO_L2, s);
  vdo_mean(pre_v, n, D, mean);
  double mnorm = 0.0;
  for (int c = 0; c < D; ++c) mnorm += mean[c] * mean[c];
  mnorm = sqrt(mnorm);
  if (scores_gpu) {
    for (int j = 0; j < n; ++j) {
      const double tol = 1e-5 * s[j] + 2e-6 * (row_norm(pre_v + (size_t)j * D) + mnorm);
      CHECK(fabs((double)scores_gpu[j] - s[j]) <= tol, "unit %d score %d: %.9g vs %.9g", u, j,
            (double)scores_gpu[j], s[j]);
    }
  }
  vdo_select_top_n(s, n, N, kept_ora);
  /* the GPU's kept slots: given (block), or every slot but the evicted one */
  if (kept_gpu) {
    memcpy(kept, kept_gpu, sizeof(int32_t) * N);
  } else {
    CHECK(evicted_gpu >= 0 && evicted_gpu < n, "unit %d evicted slot %d", u, evicted_gpu);
    for (int r = 0, i = 0; r < n; ++r)
      if (r != evicted_gpu && i < N) kept[i++] = r;
  }
  memcpy(sorted, s, sizeof(double) * n);
  qsort(sorted, (size_t)n, sizeof(double), cmp_desc);
  const double s_n = sorted[N - 1];
  for (int i = 0; i < N; ++i) {
    CHECK(kept[i] >= 0 && kept[i] < n && (i == 0 || kept[i] > kept[i - 1]),
          "unit %d kept[%d] = %d not ascending in range", u, i, kept[i]);
    if (kept[i] < 0 || kept[i] >= n) continue;
    /* a slot the oracle did not keep is acceptable only inside the near-tie band */
    int in_ora = 0;
    for (int k = 0; k < N && !in_ora; ++k) in_ora = kept_ora[k] == kept[i];
    if (!in_ora)
      CHECK(fabs(s[kept[i]] - s_n) <= 1e-5 * s_n + 1e-12, "unit %d keeps slot %d (score %.9g, "
            "N-th %.9g)", u, kept[i], s[kept[i]], s_n);
    CHECK(!memcmp(post_k + (size_t)i * D, pre_k + (size_t)kept[i] * D, sizeof(uint16_t) * D) &&
              !memcmp(post_v + (size_t)i * D, pre_v + (size_t)kept[i] * D, sizeof(uint16_t) * D),
          "unit %d row %d is not the bytes of slot %d", u, i, kept[i]);
  }
  free(s);
  free(sorted);
  free(kept_ora);
  free(kept);
}

int main(void) {
  const size_t rows = (size_t)UNITS * CAP * D;
  uint16_t* hk = calloc(rows, sizeof(uint16_t));
  uint16_t* hv = calloc(rows, sizeof(uint16_t));
  uint16_t* hk_new = malloc(sizeof(uint16_t) * UNITS * B * D);
  uint16_t* hv_new = malloc(sizeof(uint16_t) * UNITS * B * D);
  int32_t hlen[N_SEQ] = {N, N - 40};
  float centre[UNITS][D];
  for (int u = 0; u < UNITS; ++u)
    for (int c = 0; c < D; ++c) centre[u][c] = (float)(4.0 * (uniform() - 0.5));
  for (int u = 0; u < UNITS; ++u)
    for (int r = 0; r < hlen[u / PER_SEQ]; ++r) {
      fill_row(hk + ((size_t)u * CAP + r) * D, centre[u]);
      fill_row(hv + ((size_t)u * CAP + r) * D, centre[u]);
    }
  for (int u = 0; u < UNITS; ++u)
    for (int r = 0; r < B; ++r) {
      fill_row(hk_new + ((size_t)u * B + r) * D, centre[u]);
      fill_row(hv_new + ((size_t)u * B + r) * D, centre[u]);
    }

  void *dk, *dv, *dk_new, *dv_new;
  int32_t *dlen, *dkept, *devicted;
  float* dscores;
  CUDA(cudaMalloc(&dk, rows * 2));
  CUDA(cudaMalloc(&dv, rows * 2));
  CUDA(cudaMalloc(&dk_new, (size_t)UNITS * B * D * 2));
  CUDA(cudaMalloc(&dv_new, (size_t)UNITS * B * D * 2));
  CUDA(cudaMalloc((void**)&dlen, sizeof hlen));
  CUDA(cudaMalloc((void**)&dkept, sizeof(int32_t) * UNITS * N));
  CUDA(cudaMalloc((void**)&devicted, sizeof(int32_t) * UNITS));
  CUDA(cudaMalloc((void**)&dscores, sizeof(float) * UNITS * CAP));
  CUDA(cudaMemcpy(dk, hk, rows * 2, cudaMemcpyHostToDevice));
  CUDA(cudaMemcpy(dv, hv, rows * 2, cudaMemcpyHostToDevice));
  CUDA(cudaMemcpy(dk_new, hk_new, (size_t)UNITS * B * D * 2, cudaMemcpyHostToDevice));
  CUDA(cudaMemcpy(dv_new, hv_new, (size_t)UNITS * B * D * 2, cudaMemcpyHostToDevice));
  CUDA(cudaMemcpy(dlen, hlen, sizeof hlen, cudaMemcpyHostToDevice));

  vd_cache cache = {dk, dv, dlen, N_SEQ, N_LAYER, N_HEAD, D, CAP};

  /* ---- block boundary: append B rows, evict to N ---------------------- */
  vd_status st = vd_append_evict_block(&cache, dk_new, dv_new, B, N, NULL, VD_SCORE_L2,
                                       VD_MU_RECOMPUTE, NULL, NULL, NULL, dkept, dscores, NULL);
  CHECK(st == VD_OK, "vd_append_evict_block: %s", vd_status_string(st));
  st = vd_get_device_status(NULL);
  CHECK(st == VD_OK, "device status after the block event: %s", vd_status_string(st));
  if (failures) return 1;

  uint16_t* pk = malloc(rows * 2);
  uint16_t* pv = malloc(rows * 2);
  int32_t* kept = malloc(sizeof(int32_t) * UNITS * N);
  float* scores = malloc(sizeof(float) * UNITS * CAP);
  int32_t len_after[N_SEQ];
  CUDA(cudaMemcpy(pk, dk, rows * 2, cudaMemcpyDeviceToHost));
  CUDA(cudaMemcpy(pv, dv, rows * 2, cudaMemcpyDeviceToHost));
  CUDA(cudaMemcpy(kept, dkept, sizeof(int32_t) * UNITS * N, cudaMemcpyDeviceToHost));
  CUDA(cudaMemcpy(scores, dscores, sizeof(float) * UNITS * CAP, cudaMemcpyDeviceToHost));
  CUDA(cudaMemcpy(len_after, dlen, sizeof len_after, cudaMemcpyDeviceToHost));
  uint16_t* pre_k = malloc(sizeof(uint16_t) * CAP * D);
  uint16_t* pre_v = malloc(sizeof(uint16_t) * CAP * D);
  for (int u = 0; u < UNITS; ++u) {
    const int len0 = hlen[u / PER_SEQ], n = len0 + B;
    CHECK(len_after[u / PER_SEQ] == N, "seq %d len %d after the block event", u / PER_SEQ,
          len_after[u / PER_SEQ]);
    memcpy(pre_k, hk + (size_t)u * CAP * D, sizeof(uint16_t) * len0 * D);
    memcpy(pre_v, hv + (size_t)u * CAP * D, sizeof(uint16_t) * len0 * D);
    memcpy(pre_k + (size_t)len0 * D, hk_new + (size_t)u * B * D, sizeof(uint16_t) * B * D);
    memcpy(pre_v + (size_t)len0 * D, hv_new + (size_t)u * B * D, sizeof(uint16_t) * B * D);
    check_unit(u, pre_k, pre_v, n, pk + (size_t)u * CAP * D, pv + (size_t)u * CAP * D,
               kept + (size_t)u * N, -1, scores + (size_t)u * CAP);
  }

  /* ---- decode step: one token in, one out ----------------------------- */
  for (int u = 0; u < UNITS; ++u) {
    fill_row(hk_new + (size_t)u * D, centre[u]);
    fill_row(hv_new + (size_t)u * D, centre[u]);
  }
  CUDA(cudaMemcpy(dk_new, hk_new, (size_t)UNITS * D * 2, cudaMemcpyHostToDevice));
  CUDA(cudaMemcpy(dv_new, hv_new, (size_t)UNITS * D * 2, cudaMemcpyHostToDevice));
  st = vd_append_evict_decode(&cache, dk_new, dv_new, N, NULL, VD_SCORE_L2, VD_MU_RECOMPUTE,
                              NULL, NULL, NULL, devicted, NULL, NULL, NULL);
  CHECK(st == VD_OK, "vd_append_evict_decode: %s", vd_status_string(st));
  st = vd_get_device_status(NULL);
  CHECK(st == VD_OK, "device status after the decode step: %s", vd_status_string(st));
  if (failures) return 1;
  uint16_t* qk = malloc(rows * 2);
  uint16_t* qv = malloc(rows * 2);
  int32_t evicted[UNITS];
  CUDA(cudaMemcpy(qk, dk, rows * 2, cudaMemcpyDeviceToHost));
  CUDA(cudaMemcpy(qv, dv, rows * 2, cudaMemcpyDeviceToHost));
  CUDA(cudaMemcpy(evicted, devicted, sizeof evicted, cudaMemcpyDeviceToHost));
  CUDA(cudaMemcpy(len_after, dlen, sizeof len_after, cudaMemcpyDeviceToHost));
  for (int u = 0; u < UNITS; ++u) {
    CHECK(len_after[u / PER_SEQ] == N, "seq %d len %d after the decode step", u / PER_SEQ,
          len_after[u / PER_SEQ]);
    memcpy(pre_k, pk + (size_t)u * CAP * D, sizeof(uint16_t) * N * D);
    memcpy(pre_v, pv + (size_t)u * CAP * D, sizeof(uint16_t) * N * D);
    memcpy(pre_k + (size_t)N * D, hk_new + (size_t)u * D, sizeof(uint16_t) * D);
    memcpy(pre_v + (size_t)N * D, hv_new + (size_t)u * D, sizeof(uint16_t) * D);
    check_unit(u, pre_k, pre_v, N + 1, qk + (size_t)u * CAP * D, qv + (size_t)u * CAP * D, NULL,
               evicted[u], NULL);
  }

  cudaFree(dk);
  cudaFree(dv);
  cudaFree(dk_new);
  cudaFree(dv_new);
  cudaFree(dlen);
  cudaFree(dkept);
  cudaFree(devicted);
  cudaFree(dscores);
  if (failures) {
    fprintf(stderr, "%d checks failed\n", failures);
    return 1;
  }
  printf("c abi example: %d units, block event and decode step match the oracle\n", UNITS);
  return 0;
}
