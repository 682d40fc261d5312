/*
 * vd_oracle.h -- fp64 CPU oracle for ValueDiff KV-cache eviction.
 *
 * TEST INFRASTRUCTURE ONLY.  This is the slow, plain reference that the
 * CUDA path is checked against.  Only the test suite, the smoke check and
 * the benchmark's CPU-baseline leg may load it.  It shares no code, header,
 * table or constant with the CUDA library and never calls it.
 *
 * Every function follows a passage of the paper ("ValueDiff: Value-Geometric
 * KV Cache Eviction for Sink-Suppressed LLMs"):
 *   - cache mean and score ............ Sec. 3.2, Eq. (vd), Eq. (decomp)
 *   - Dir / Norm variants ............. Sec. 3.2 (last paragraph)
 *   - top-N and gather ................ Sec. 2.1, Eq. (eviction)
 *   - eviction trigger "exceeds N" .... Sec. 2.1
 *
 * Values are bf16 bit patterns (uint16_t), widened exactly to double.
 * Row-major [n][d] per (sequence, layer, KV head) unit.
 */
#ifndef VD_ORACLE_H
#define VD_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Scoring rules of Sec. 3.2: L2 = ||v_j - mean||, DIR = 1 - cos(v_j, mean),
 * NORM = ||v_j||. */
enum { VDO_L2 = 0, VDO_DIR = 1, VDO_NORM = 2 };

/* Exact widening of one bf16 bit pattern. */
double vdo_bf16_to_double(uint16_t bits);

/* Sum of the n rows of v ([n][d] bf16) per column, Neumaier-compensated fp64.
 * out: [d]. */
void vdo_sum_rows(const uint16_t* v, int64_t n, int64_t d, double* out);

/* Cache mean of Eq. (vd): mean_c = (1/n) sum_i v_ic.  out: [d].  n >= 1. */
void vdo_mean(const uint16_t* v, int64_t n, int64_t d, double* out);

/* Per-token scores s_j for j < n under `variant`.  out: [n].
 * DIR with a zero-norm v_j or a zero-norm mean takes cos := 0 (score 1). */
void vdo_scores(const uint16_t* v, int64_t n, int64_t d, int variant, double* out);

/* App. A, Eq. (app_fastcaote): the attention-weighted score
 * a_j / (1 - a_j) * s_j, with s_j the `variant` score of vdo_scores and a_j
 * the caller's attention weight (a_j in [0, 1); outside -> NaN).  out: [n]. */
void vdo_scores_weighted(const uint16_t* v, int64_t n, int64_t d, int variant, const double* a,
                         double* out);

/* Sec. 3.1 (and App. C): sigma = std_i || x_i - mean ||_2 over the n rows of
 * one unit (population standard deviation).  Returns sigma. */
double vdo_dispersion(const uint16_t* x, int64_t n, int64_t d);

/* Eq. (eviction): keep the N highest scores, ties to the lower index.
 * Writes the kept indices in ascending order to kept[0..min(n,N)).
 * Returns the number kept (min(n, N)); n <= N keeps everything. */
int64_t vdo_select_top_n(const double* scores, int64_t n, int64_t N, int32_t* kept);

/* One eviction event on one unit: if n > N, score, select and gather K and V
 * in ascending kept order into rows [0, N) (slots >= N are left as they
 * were).  kept: [min(n,N)] (nullable), scores: [n] (nullable; written only
 * when n > N).  Returns the new length. */
int64_t vdo_evict_unit(uint16_t* k, uint16_t* v, int64_t n, int64_t d, int64_t N,
                       int variant, int32_t* kept, double* scores);

/* Many units at once (the CPU baseline).  Unit u's rows start at
 * u * capacity * d; its length is len[u / units_per_seq] and its budget
 * N_per_seq[u / units_per_seq].  Units are split over `nthreads` POSIX
 * threads (units are independent).  kept: [n_units][kept_stride] (nullable).
 * The caller updates len afterwards.  Returns 0, or -1 if a thread could not
 * be started. */
int vdo_evict_units(uint16_t* k, uint16_t* v, const int32_t* len, const int32_t* N_per_seq,
                    int64_t n_units, int64_t units_per_seq, int64_t capacity, int64_t d,
                    int variant, int32_t* kept, int64_t kept_stride, int nthreads);

#ifdef __cplusplus
}
#endif

#endif /* VD_ORACLE_H */
