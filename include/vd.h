/*
 * vd.h -- C ABI of the GB300 (sm_103a) ValueDiff KV-cache eviction library
 * (libvd.so).
 *
 * ValueDiff (Sec. 3.2, Eq. vd) scores every cached token of one
 * (sequence, layer, KV head) "unit" by how far its value vector lies from the
 * cache mean,  s_j = || v_j - mean ||_2,  mean = (1/n) sum_i v_i,  and the
 * eviction policy pi_N of Sec. 2.1, Eq. (eviction) keeps the N highest-scoring
 * tokens and gathers K and V to them.  pi_N runs at every block boundary of
 * block prompt processing (Sec. 2.2, Eq. block_processing: cache N+B -> N)
 * and at every decode step (abstract; Sec. 4 protocol: cache N+1 -> N).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - All buffers are caller-owned DEVICE memory unless stated otherwise.  The
 *   library allocates no device memory; its only device state is one status
 *   word per device (a static __device__ variable).
 * - Calls are asynchronous on `stream` (a cudaStream_t; NULL = legacy default
 *   stream).  Host-side validation happens before any launch: a call that
 *   returns an error launched nothing and changed nothing.
 * - Layout: K and V are bf16, [n_seq][n_layer][n_kv_head][capacity][head_dim]
 *   row-major, so one unit's rows are contiguous.  Unit index
 *   u = (seq * n_layer + layer) * n_kv_head + head.
 * - len is a device int32 [n_seq]: every layer and head of a sequence holds
 *   the same number of tokens.  Slots >= len are never read.
 * - Top-N ties are broken toward the LOWER slot index (the earlier token; the
 *   paper does not fix a tie rule).  Compaction keeps the surviving tokens in
 *   their original (ascending slot) order.  Slots >= N after an eviction hold
 *   unspecified bytes.
 * - Anomalies found on the device (len > capacity, a per-sequence budget out
 *   of range, a non-finite score, a decode call with more than one token over
 *   budget) never trap: the kernel records the first one in the device status
 *   word (read it with vd_get_device_status) and leaves the affected unit
 *   untouched, except VD_ERR_NONFINITE, which is recorded while the unit is
 *   still evicted with NaN scores ranked lowest.
 * - Precision: scores are computed in fp32 from bf16 inputs against the
 *   cache mean carried as an fp32 part plus its fp32 remainder; the mean is
 *   accumulated with exact (TwoSum) fp32 sums, or from the fp64 running sum,
 *   to about 1e-12 of the data's scale.  Every score's rounding error is
 *   relative to the score itself (a few 1e-7 in practice).  Ranking: a NaN
 *   score ranks below every number, +0 and -0 are equal.
 * - Launches: one eviction kernel per call, plus a one-thread-per-sequence
 *   length update (a programmatic dependent launch of the eviction, all on
 *   `stream`).  A hole-fill block eviction or a score-only call that fits
 *   one wave at one CTA per unit but has more units than the GPU has SMs
 *   runs the eviction kernel as two launches over disjoint units, the second
 *   a programmatic dependent of the first, so that no SM carries a whole
 *   unit more than the others.  A short cache (capacity <= 1024,
 *   4 * capacity * head_dim <= 64 KB, at most 16 units per sequence, at most
 *   two units per SM) takes a kernel that keeps the unit in shared memory
 *   and updates the lengths itself: one launch in all.  Results follow the
 *   same rules either way, and every call can be captured in a CUDA graph.
 */
#ifndef VD_H
#define VD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t. */
typedef struct CUstream_st* vd_stream_t;

typedef enum {
  VD_OK = 0,
  VD_ERR_INVALID_ARG = 1, /* null pointer, non-positive size, N out of range, ... */
  VD_ERR_ALIGNMENT = 2,   /* K/V not 16-byte aligned, or head_dim % 8 != 0 */
  VD_ERR_UNSUPPORTED = 3, /* shape beyond what the kernels handle: head_dim > 256;
                             block eviction with capacity > 65536 (16-bit slot
                             lists) or whose on-chip keys and slot lists do not
                             fit one CTA's shared memory at any cluster size
                             (about 41 KB + capacity * (2 + 4 / C) bytes <= 227 KB,
                             C <= head_dim / 4): at head_dim >= 64 every
                             capacity up to 65536 fits */
  VD_ERR_NONFINITE = 4,   /* device: a score was NaN or infinite */
  VD_ERR_TIMEOUT = 5,     /* device: a bounded wait for a bulk copy gave up (score-only
                             kernels); that call's outputs are unspecified */
  VD_ERR_CUDA = 6,        /* a CUDA runtime call failed (launch error, ...) */
  VD_ERR_DEVICE_LEN = 7,  /* device: len[s] out of [0, capacity], or len + B > capacity
                             on append, or B > len in running-sum mode */
  VD_ERR_DEVICE_BUDGET = 8, /* device: N_dev[s] out of [1, N], or a decode call found
                               len > N + 1 */
  VD_ERR_NO_DEVICE = 9,   /* no CUDA device, or not an sm_103 device */
  VD_ERR_INTERNAL = 10    /* device: a kernel's self-check found an inconsistent slot
                             list (never expected); the access was skipped */
} vd_status;

/* Scoring rules of Sec. 3.2.  Higher scores are kept.
 *   VD_SCORE_L2   s_j = || v_j - mean ||_2           (ValueDiff, Eq. vd)
 *   VD_SCORE_DIR  s_j = 1 - cos(v_j, mean)           (ValueDiff-Dir; cos := 0 when
 *                                                     v_j or the mean is zero)
 *   VD_SCORE_NORM s_j = || v_j ||_2                  (ValueDiff-Norm; keeps the
 *                                                     largest norms) */
typedef enum { VD_SCORE_L2 = 0, VD_SCORE_DIR = 1, VD_SCORE_NORM = 2 } vd_variant;

/* How the cache mean is obtained.
 *   VD_MU_RECOMPUTE  sum every cached row at every event (reads V twice per
 *                    event unless the cache slice fits on chip).
 *   VD_MU_RUNNING    keep S = sum of the cached V rows as fp64 [unit][head_dim]
 *                    across events; the mean is S / n.  V is read once.
 *                    Not in the paper: an exact incremental form of its mean. */
typedef enum { VD_MU_RECOMPUTE = 0, VD_MU_RUNNING = 1 } vd_mu_mode;

typedef struct {
  void* k;          /* bf16 device, [n_seq][n_layer][n_kv_head][capacity][head_dim], 16-B aligned */
  void* v;          /* bf16 device, same layout as k, 16-B aligned */
  int32_t* len;     /* device int32 [n_seq]: current number of cached tokens */
  int32_t n_seq, n_layer, n_kv_head;
  int32_t head_dim; /* multiple of 8, at most 256 */
  int32_t capacity; /* slots per unit; the kernels size on-chip buffers by it */
} vd_cache;

/* Scores only (Eq. vd and its Sec. 3.2 variants), mean recomputed from the
 * cache.  scores_out: fp32 device [n_seq][n_layer][n_kv_head][capacity]; rows
 * j < len[s] are written, rows >= len[s] untouched.  The cache is not
 * modified. */
vd_status vd_score(const vd_cache* c, vd_variant var, float* scores_out, vd_stream_t stream);

/* Block-boundary eviction (Sec. 2.2, Eq. block_processing): the caller has
 * already appended B rows (len = old + B).  For every unit whose sequence has
 * len > N_s: score, keep the top N_s (Sec. 2.1, Eq. eviction), compact K and V
 * in place in ascending slot order and set len = N_s.  Sequences with
 * len <= N_s are left as they are ("evict whenever the cache exceeds N").
 *   N            scalar budget, 1 <= N <= capacity; also the row stride of
 *                kept_idx_out and the upper bound of N_dev values.
 *   N_dev        nullable device int32 [n_seq]: per-sequence budgets N_s in
 *                [1, N] (e.g. a budget that grows with length); NULL -> N_s = N.
 *   B            rows appended since the previous call, 0 <= B <= capacity;
 *                used only by VD_MU_RUNNING.
 *   running_sum  fp64 device [n_seq][n_layer][n_kv_head][head_dim], required
 *                when mu == VD_MU_RUNNING: on entry the sum of V rows
 *                [0, len - B) (the rows present after the previous call), on
 *                exit the sum of the rows [0, new len).  Initialise it with
 *                vd_running_sum_init.  Ignored for VD_MU_RECOMPUTE.
 *   kept_idx_out nullable int32 device [n_seq][n_layer][n_kv_head][N]: the
 *                pre-eviction slot of every surviving token, ascending; for a
 *                unit that did not evict, 0..len-1 followed by -1.
 *   scores_out   nullable fp32 device [..][capacity]: the scores of the
 *                pre-eviction rows, written only for units that evicted. */
vd_status vd_evict_block(const vd_cache* c, int32_t N, const int32_t* N_dev, int32_t B,
                         vd_variant var, vd_mu_mode mu, double* running_sum,
                         int32_t* kept_idx_out, float* scores_out, vd_stream_t stream);

/* One step of block prompt processing (Sec. 2.2, Eq. block_processing:
 * C_i = pi_N([C_{i-1} || block_i])) with the append fused into the
 * eviction kernel: the same result as
 * vd_append(c, k_new, v_new, B) followed by vd_evict_block(c, N, N_dev, B,
 * var, mu, running_sum, kept_idx_out, scores_out) -- the same kept slots,
 * scores, compacted K/V bytes in slots [0, new len), running sum and len --
 * but the new rows are read straight from the caller's buffers, and only
 * the ones that survive are written into the cache (appended rows that are
 * evicted at once are never stored).  Block path, either layout.
 *   k_new, v_new  bf16 device [n_seq][n_layer][n_kv_head][B][head_dim],
 *                 16-byte aligned, read only; B >= 1.
 *   len           on entry the rows already cached (the new ones excluded);
 *                 on exit min(len + B, N_s) -- or len + B where no eviction
 *                 happens.
 *   running_sum   (VD_MU_RUNNING) on entry the sum of rows [0, len), on exit
 *                 the sum of rows [0, new len).
 *   pos, pos_first_new  both null: ordered layout (vd_evict_block); both
 *                 given: the hole-fill layout, as vd_append followed by
 *                 vd_evict_block_holefill (arguments as there, pos_first_new
 *                 the position of the first new row).
 * Other arguments as in vd_evict_block.  A sequence with len + B > capacity
 * is left untouched and records VD_ERR_DEVICE_LEN.  Slots at or above the new
 * len hold unspecified bytes. */
vd_status vd_append_evict_block(const vd_cache* c, const void* k_new, const void* v_new,
                                int32_t B, int32_t N, const int32_t* N_dev, vd_variant var,
                                vd_mu_mode mu, double* running_sum, int32_t* pos,
                                const int32_t* pos_first_new, int32_t* kept_idx_out,
                                float* scores_out, vd_stream_t stream);

/* Decode-step eviction (per-token eviction of the abstract and the Sec. 4
 * protocol; Eq. block_processing with B = 1): the caller has appended one
 * token, so len <= N_s + 1.  Units with len = N_s + 1 evict exactly one token
 * (the lowest score; among tied minima the highest slot) and compact.
 * Arguments as in vd_evict_block with B = 1, plus
 *   evicted_out  nullable int32 device [n_seq][n_layer][n_kv_head]: the
 *                evicted pre-eviction slot, or -1 where nothing was evicted.
 * A sequence found with len > N_s + 1 is left untouched and records
 * VD_ERR_DEVICE_BUDGET. */
vd_status vd_evict_decode(const vd_cache* c, int32_t N, const int32_t* N_dev, vd_variant var,
                          vd_mu_mode mu, double* running_sum, int32_t* evicted_out,
                          int32_t* kept_idx_out, float* scores_out, vd_stream_t stream);

/* One decode step, the append fused into the eviction kernel: the same
 * result as vd_append(c, k_new, v_new, 1) followed by vd_evict_decode (or,
 * with pos and pos_first_new, by vd_evict_decode_holefill), with the new
 * token read straight from the
 * caller's buffers and written into the cache only if it survives.
 *   k_new, v_new  bf16 device [n_seq][n_layer][n_kv_head][1][head_dim],
 *                 16-byte aligned, read only.
 *   len           on entry the cached tokens (the new one excluded), on exit
 *                 min(len + 1, N_s).
 *   running_sum   (VD_MU_RUNNING) on entry the sum of rows [0, len).
 * Other arguments as in vd_evict_decode / vd_evict_decode_holefill.  A
 * sequence with len + 1 > capacity is left untouched (VD_ERR_DEVICE_LEN). */
vd_status vd_append_evict_decode(const vd_cache* c, const void* k_new, const void* v_new,
                                 int32_t N, const int32_t* N_dev, vd_variant var, vd_mu_mode mu,
                                 double* running_sum, int32_t* pos, const int32_t* pos_first_new,
                                 int32_t* evicted_out, int32_t* kept_idx_out, float* scores_out,
                                 vd_stream_t stream);

/* Scores with options, no eviction.
 *   score_keys      0: V rows (ValueDiff and its variants, Sec. 3.2); 1: the
 *                   same rules on K rows, with the mean of K (the key-side
 *                   signals of the Sec. 4 baselines: L2 = distance from the key
 *                   centroid, Dir = cosine distance from the mean key).
 *   scores_out      nullable fp32 [..][capacity] (rows >= len untouched).
 *   dispersion_out  nullable fp32 [n_seq][n_layer][n_kv_head]: per unit, the
 *                   standard deviation over its len tokens of the L2 distance
 *                   from the mean -- sigma_V (or sigma_K with score_keys) of
 *                   Sec. 3.1 (population std).  Requires var == VD_SCORE_L2.
 *   mu, running_sum  VD_MU_RECOMPUTE: the mean is summed from the len rows
 *                   (every row is read twice).  VD_MU_RUNNING: the mean is
 *                   running_sum / len (fp64 [n_seq][n_layer][n_kv_head]
 *                   [head_dim], read only: the sums of the len rows of the
 *                   scored tensor that the eviction calls maintain), so the
 *                   rows are read once.  running_sum must be non-null then.
 * At least one of the two outputs must be given. */
vd_status vd_score_ex(const vd_cache* c, vd_variant var, vd_mu_mode mu,
                      const double* running_sum, int32_t score_keys, float* scores_out,
                      float* dispersion_out, vd_stream_t stream);

/* vd_evict_block with scoring options:
 *   score_keys  1: select on the K-side rule (mean of K).  With
 *               VD_MU_RUNNING, running_sum holds sums of K rows (seed it with
 *               vd_running_sum_init_ex(c, 1, ...)).  K and V are still both
 *               compacted.
 *   attn        nullable fp32 device [..][capacity]: an attention weight a_j
 *               in [0, 1) per cached token; the score becomes
 *               a_j / (1 - a_j) * s_j, the FastCAOTE form of App. A
 *               Eq. (app_fastcaote) (with VD_SCORE_L2).  A weight outside
 *               [0, 1) gives a NaN score (ranked lowest, VD_ERR_NONFINITE).
 *               scores_out then holds the weighted scores.
 *   dispersion_out  nullable fp32 device [n_seq][n_layer][n_kv_head]: sigma of
 *               Sec. 3.1 over the len pre-eviction rows (sigma_V, or sigma_K
 *               with score_keys), from the same score pass (no extra read);
 *               the unweighted L2 distances; requires var == VD_SCORE_L2
 *               (else VD_ERR_INVALID_ARG).  Written only for units that
 *               evicted, like scores_out.
 * Other arguments as in vd_evict_block.  A weighted decode step is this call
 * with B = 1. */
vd_status vd_evict_block_ex(const vd_cache* c, int32_t N, const int32_t* N_dev, int32_t B,
                            vd_variant var, vd_mu_mode mu, double* running_sum,
                            int32_t score_keys, const float* attn, int32_t* kept_idx_out,
                            float* scores_out, float* dispersion_out, vd_stream_t stream);

/* vd_append followed by vd_evict_block_ex with the append fused into the
 * eviction kernel, as
 * vd_append_evict_block is for vd_evict_block (one step of Sec. 2.2,
 * Eq. block_processing, with the scoring options above): k_new, v_new are
 * bf16 device [n_seq][n_layer][n_kv_head][B][head_dim], 16-byte aligned,
 * read straight from the caller's buffers, and only surviving rows are
 * written.  len does not count the new rows before the call; during the
 * event they occupy slots len .. len + B - 1, which is where attn, the
 * scores and the kept slots refer to them.  Results are identical to
 * vd_append followed by vd_evict_block_ex.  Ordered layout; errors as
 * vd_append_evict_block and vd_evict_block_ex. */
vd_status vd_append_evict_block_ex(const vd_cache* c, const void* k_new, const void* v_new,
                                   int32_t B, int32_t N, const int32_t* N_dev, vd_variant var,
                                   vd_mu_mode mu, double* running_sum, int32_t score_keys,
                                   const float* attn, int32_t* kept_idx_out, float* scores_out,
                                   float* dispersion_out, vd_stream_t stream);

/* Hole-fill layout (not in the paper; its eviction rule with a cache layout
 * that moves as few rows as possible).  Same policy as vd_evict_block /
 * vd_evict_decode (Sec. 2.1, Eq. eviction; Sec. 2.2, Eq. block_processing),
 * but surviving rows are not kept in slot order: after the call, the kept
 * rows that sat at or above the budget N_s (the appended ones) have moved
 * into the evicted slots below N_s (paired in ascending order), every other
 * kept row stays where it was, and slots [0, N_s) hold the surviving tokens
 * in no particular order.  The tie-break is by token position instead of
 * slot: among equal scores the lower position (earlier token) survives.
 *   pos            int32 device [n_seq][n_layer][n_kv_head][capacity]: the
 *                  sequence position of the token in each slot.  On entry,
 *                  valid for rows [0, len - B); on exit, for rows [0, new len)
 *                  (the kernel writes the positions of the appended rows and
 *                  of every moved row).  Positions within a unit must be
 *                  distinct and non-negative.
 *   pos_first_new  int32 device [n_seq]: the position of the first appended
 *                  row (slot len - B); appended row i has position
 *                  pos_first_new[s] + i.
 *   kept_idx_out   [..][N]: for every slot r < N_s, the pre-eviction slot of
 *                  the token now in slot r (r itself unless r was refilled).
 * A decode step therefore moves at most one row instead of shifting the cache
 * tail; a block boundary moves at most B rows. */
vd_status vd_evict_block_holefill(const vd_cache* c, int32_t N, const int32_t* N_dev, int32_t B,
                                  vd_variant var, vd_mu_mode mu, double* running_sum,
                                  int32_t* pos, const int32_t* pos_first_new,
                                  int32_t* kept_idx_out, float* scores_out, vd_stream_t stream);

vd_status vd_evict_decode_holefill(const vd_cache* c, int32_t N, const int32_t* N_dev,
                                   vd_variant var, vd_mu_mode mu, double* running_sum,
                                   int32_t* pos, const int32_t* pos_first_new,
                                   int32_t* evicted_out, int32_t* kept_idx_out, float* scores_out,
                                   vd_stream_t stream);

/* Append B new rows per unit at slots [len, len + B) and set len += B (the
 * block append of Eq. block_processing).  k_new, v_new: bf16 device
 * [n_seq][n_layer][n_kv_head][B][head_dim], 16-B aligned.  A sequence with
 * len + B > capacity is left untouched and records VD_ERR_DEVICE_LEN.  The
 * running sum, if any, is NOT touched here: vd_evict_* adds the appended rows
 * (pass the same B). */
vd_status vd_append(const vd_cache* c, const void* k_new, const void* v_new, int32_t B,
                    vd_stream_t stream);

/* running_sum[u][:] = sum of V rows [0, len) of unit u, from scratch (fp64
 * [n_seq][n_layer][n_kv_head][head_dim], device). */
vd_status vd_running_sum_init(const vd_cache* c, double* running_sum, vd_stream_t stream);

/* vd_running_sum_init for the tensor a running mean tracks: of_keys = 0 the V
 * rows (ValueDiff and its variants), 1 the K rows (the key-side rules of
 * vd_evict_block_ex with score_keys = 1).  Same layout and errors. */
vd_status vd_running_sum_init_ex(const vd_cache* c, int32_t of_keys, double* running_sum,
                                 vd_stream_t stream);

/* Device scratch the calls need beyond their arguments: always 0 (the fused
 * kernels keep every intermediate on chip). */
size_t vd_workspace_size(const vd_cache* c);

/* Static English text for a status code (never NULL). */
const char* vd_status_string(vd_status st);

/* Synchronises `stream`, returns the first device-side anomaly recorded since
 * the previous call (VD_OK if none) and clears it.  A sticky CUDA error on
 * the stream is returned as VD_ERR_CUDA. */
vd_status vd_get_device_status(vd_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* VD_H */
