// vd_evict.cuh -- the fused ValueDiff eviction kernel for GB300 (sm_103a).
//
// One thread-block cluster of C CTAs owns one (sequence, layer, KV head) unit
// and runs pi_N of Sec. 2.1, Eq. (eviction) on it in a single launch.  CTA r
// of the cluster scores the rows [r*R, (r+1)*R) (R = ceil(n / C)) and moves
// the column slice r of the concatenated [K | V] row.
//
//   1. mean   mean = (1/n) sum_i v_i (Sec. 3.2, Eq. vd) as double-float
//             (hi + lo) fp32 column sums; the C partials are added in rank
//             order through distributed shared memory (DSMEM), so every CTA
//             holds the same mean, kept as an fp32 part plus its remainder.
//             Running-sum mode adds only the appended rows (spread over the
//             cluster) to the caller's fp64 sum S.
//   2. score  rows stream, last to first, through a per-thread ring of
//             asynchronous 16-byte copies (cp.async, 4 stages); d/8 lanes per row, warp
//             shuffle reduction of the squared deviation (L2, as
//             ((v - hi) - lo)^2 against the two-part mean), of the norm
//             (Norm), or of |w|^2 / (2 |v|^2) with w = v - (|v|/|mean|) mean
//             (Dir: equals 1 - cos without cancellation).  Every score's
//             rounding error is relative to the score itself.
//             For d = 64, 128, 256 (L2, Norm) each lane keeps
//             a batch of 8 rows' partial sums (packed f32x2 arithmetic) and
//             the batch is reduced with a transposed butterfly
//             (score_rows_fast).  Scores become order-preserving uint32 keys.
//   3. select block prompt processing (N+B -> N): a 4-pass 8-bit radix select
//             for the N-th largest key t; every CTA histograms only its own
//             rows and the cluster adds the C histograms through DSMEM.
//             Keys > t are kept, and the keys == t with the lowest slots fill
//             the rest (the lower-index tie-break).  Decode (N+1 -> N): a
//             cluster arg-min over (key, -slot) finds the one evicted slot.
//   4. list   per-CTA counts (> t, == t) are exchanged, each CTA ranks its own
//             rows with block prefix sums and scatters them into every CTA's
//             perm[] (uint16): kept slots ascending in [0, N), then the
//             evicted slots ascending.
//   5. sum    running-sum mode: S += sum(appended rows) - sum(evicted rows)
//             over the columns of the scored tensor (V, or K for the key-side
//             rule) this CTA moves, before it moves them.
//   6. move   K' = gather(K, perm), V' = gather(V, perm), in place, for the
//             rows r = first evicted .. N-1 of this CTA's column slice.  Tiles
//             of rows stream through the cp.async ring; tile t is stored only
//             after every thread's copies of tile t have landed (one
//             __syncthreads), while tiles t+1.. are already in flight.  Since
//             perm[r] >= r, a tile's destinations lie below every source a
//             later tile reads, so the ascending order is hazard-free, and
//             column slices make the CTAs of a unit independent.
//
// Template flags select the rest at compile time: DECODE (the arg-min path),
// HF (hole-fill layout: ties broken by token position, and only the kept rows
// at or above N move, into the evicted slots below N) and FUSED (the rows at
// or above len are read from the caller's staging buffers and written only
// if they survive: the append of Eq. block_processing fused into the event).
//
// Nothing waits on a flag; the only cross-CTA synchronisation is the hardware
// cluster barrier, which every CTA of a cluster reaches the same number of
// times (every branch below depends only on per-sequence values that all
// CTAs of the cluster read identically).
#pragma once

#include <climits>
#include <cstdint>
#include <type_traits>

#include "vd_device.cuh"

namespace vd {

// cp.async rings: STAGES stages of ITEMS 16-byte copies per thread.  The
// block kernels (which also hold keys and slot lists in shared memory) and
// the decode / score-only kernels (which hold neither, so they can afford a
// deeper ring) have their own shapes; overridable at build time for tuning
// sweeps.
#ifndef VD_RING_STAGES
#define VD_RING_STAGES 4
#endif
#ifndef VD_RING_ITEMS
#define VD_RING_ITEMS 2
#endif
#ifndef VD_DECODE_RING_STAGES
#define VD_DECODE_RING_STAGES VD_RING_STAGES
#endif
#ifndef VD_DECODE_RING_ITEMS
#define VD_DECODE_RING_ITEMS VD_RING_ITEMS
#endif
// Resident CTAs per SM the block and decode kernels are compiled for (caps
// registers per thread at 65536 / (256 * n)).
#ifndef VD_BLOCK_MIN_CTAS
#define VD_BLOCK_MIN_CTAS 4
#endif
// Hole-fill block eviction: its one-CTA-per-unit launches hold the unit's
// keys and slot list, which at prefill sizes already limit it to 3 CTAs per
// SM, so it takes the registers of 3 (85 per thread): room for the
// double-float retirement sums in its move stream.
#ifndef VD_HF_BLOCK_MIN_CTAS
#define VD_HF_BLOCK_MIN_CTAS 3
#endif
#ifndef VD_DECODE_MIN_CTAS
#define VD_DECODE_MIN_CTAS 4
#endif
// Score-only launches (vd_score, vd_score_ex) have their own instantiation:
// no select, slot lists or compaction, so a deeper ring fits at a lower
// occupancy.
#ifndef VD_SCORE_RING_STAGES
#define VD_SCORE_RING_STAGES 8
#endif
#ifndef VD_SCORE_RING_ITEMS
#define VD_SCORE_RING_ITEMS 2
#endif
#ifndef VD_SCORE_MIN_CTAS
#define VD_SCORE_MIN_CTAS 3
#endif
// Score-only launches at head dims 64, 128, 256 (L2, Norm) stream through a
// ring of bulk copies instead: VD_SCORE_BULK_STAGES stages of 32 KB.
#ifndef VD_SCORE_BULK_STAGES
#define VD_SCORE_BULK_STAGES 2
#endif
template <int STAGES, int ITEMS>
struct RingShape {
  static constexpr int kStages = STAGES;
  static constexpr int kItems = ITEMS;
  static constexpr int kBytes = STAGES * ITEMS * kThreads * 16;
};
using BlockRing = RingShape<VD_RING_STAGES, VD_RING_ITEMS>;
using DecodeRing = RingShape<VD_DECODE_RING_STAGES, VD_DECODE_RING_ITEMS>;
using ScoreRing = RingShape<VD_SCORE_RING_STAGES, VD_SCORE_RING_ITEMS>;

// Launch kinds, which size the shared memory: decode eviction, block
// eviction (the select's keys and the slot list too), score-only.
constexpr int kKindDecode = 0, kKindBlock = 1, kKindScore = 2, kKindScoreBulk = 3;
constexpr int kBulkStages = VD_SCORE_BULK_STAGES;
constexpr int kBulkStageBytes = 32768;

__host__ __device__ constexpr int ring_bytes(int kind) {
  return kind == kKindBlock        ? BlockRing::kBytes
         : kind == kKindScore      ? ScoreRing::kBytes
         : kind == kKindScoreBulk  ? kBulkStages * kBulkStageBytes
                                   : DecodeRing::kBytes;
}

// Whether a score-only launch takes the bulk ring: the batched L2 / Norm
// score pass, whose stage of 32 KB is exactly one batch of rows per lane group.
__host__ __device__ constexpr bool score_bulk(int var, int d) {
  return var != 1 && (d == 64 || d == 128 || d == 256);
}

struct EvictArgs {
  uint16_t* k;            // bf16 [U][capacity][d]
  uint16_t* v;            // bf16 [U][capacity][d]
  int32_t* len;           // [n_seq] (written only by the short-cache kernel)
  const int32_t* N_dev;   // nullable [n_seq]
  double* running_sum;    // [U][d] (running mode)
  int32_t* kept_out;      // nullable [U][N]
  int32_t* evicted_out;   // nullable [U] (decode)
  float* scores_out;      // nullable [U][capacity]
  unsigned* status;       // device status word
  int32_t units_per_seq;  // n_layer * n_kv_head
  int32_t d;              // head_dim (multiple of 8, <= 256)
  int32_t lpr;            // lanes per row: next power of two >= d / 8
  int32_t capacity;
  int32_t N;              // scalar budget, kept_out stride, N_dev bound
  int32_t B;              // rows appended since the previous eviction
  int32_t mu_running;     // 1: mean from running_sum + appended rows
  int32_t score_only;     // 1: vd_score / vd_score_ex (the kernels take it from SCORE)
  int32_t cluster;        // C, CTAs per unit
  int32_t* pos;            // hole-fill layout: token positions [U][capacity]
  const int32_t* pos_new;  // hole-fill layout: position of row len - B, [n_seq]
  int32_t holefill;        // 1: hole-fill layout (ties by position), 0: ordered
  int32_t score_k;         // 1: mean and scores from K (key-side rules)
  const float* weights;    // nullable [U][capacity]: attention weights a_j (block path)
  float* disp_out;         // nullable [U]: std of the L2 scores of the scored rows
  // fused append (block or decode, either layout): the B new rows are read
  // from these staging buffers ([U][B][d] bf16 each) instead of the cache,
  // len does not count them yet, and only the kept ones are written
  // (nullable: the rows were appended beforehand)
  const uint16_t* k_new;
  const uint16_t* v_new;
  // split launch (two launches over disjoint units): the units before this
  // launch's first one.  Only the sequence index adds it; every per-unit
  // pointer above comes offset to the launch's first unit.
  int32_t unit_base;
};

// Fixed part of the dynamic shared memory.  After it (16-byte aligned): the
// cp.async ring, then (block eviction only) this CTA's keys [R] and the
// unit's perm [capacity] (uint16).
struct Smem {
  float mu[256];    // the mean rounded to fp32 ...
  float mulo[256];  // ... and its remainder (mean = mu + mulo to ~2^-44 relative),
                    // pair-transposed: column c at lo_index(c, d / 8)
  float acc_hi[256];  // this CTA's partial column sums (read by peer CTAs)
  float acc_lo[256];
  double snew[256];       // running mode: the running sum plus the appended rows
  uint32_t hist[2][256];  // this CTA's radix histograms (read by peers)
  uint32_t ghist[256];
  int scan[kWarps];
  float fsh[kWarps];
  unsigned long long best;  // decode: this CTA's (key, -tie-break) minimum
  unsigned long long wbest[kWarps];
  int sel_digit, sel_above, sel_cnt;
  uint32_t sel_t;  // rank resolution: the threshold key
  int ncand;       // rank resolution: this CTA's candidates (in ghist, read by peers)
  int cnt_gt, cnt_eq;  // this CTA's keys > t and == t (read by peers)
  int mu_zero;
  int best_slot;       // hole-fill decode: the slot of `best`
  int wslot[kWarps];
  int holes;           // hole-fill: evicted slots below N
  float inv_mnorm;     // Dir: 1 / |mean|
  float disp[4];       // dispersion partials: sum s (hi, lo), sum s^2 (hi, lo)
  float dsc[4 * kWarps];  // dispersion: per-warp partials (block-private)
  unsigned long long bar[4];  // bulk ring: one mbarrier per stage (score-only)
};

__host__ __device__ constexpr size_t align16(size_t x) { return (x + 15) & ~(size_t)15; }

// Slot of column c of the mean's remainder in Smem::mulo (d8 = d / 8 chunks
// of 8 columns): the pairs (2k, 2k + 1) of every chunk are stored together,
// pair k of chunk ci at floats 2 * (k * d8 + ci) and + 1.
__device__ __forceinline__ int lo_index(int c, int d8) {
  return 2 * (((c & 7) >> 1) * d8 + (c >> 3)) + (c & 1);
}

// Byte offsets of the variable parts; the host sizes the launch with the same
// function.  The ring starts on a 128-byte boundary: a warp's 16-byte copies
// then fill whole 32-byte shared-memory sectors (an offset that is only
// 16-byte aligned splits every pair of slots across two sectors, which
// measured 8-13% slower on GB300).
struct SmemLayout {
  size_t ring, keys, perm, total;
};

__host__ __device__ inline SmemLayout smem_layout(int capacity, int cluster, int kind) {
  const bool with_select = kind == kKindBlock;
  SmemLayout l;
  l.ring = (sizeof(Smem) + 127) & ~(size_t)127;
  l.keys = l.ring + (size_t)ring_bytes(kind);
  const size_t rows = with_select ? (size_t)((capacity + cluster - 1) / cluster) : 0;
  l.perm = l.keys + align16(rows * 4);
  l.total = l.perm + (with_select ? align16((size_t)capacity * 2) : 0);
  return l;
}

// Streams items [0, count) through a thread-private cp.async ring.  Item i is
// the row that starts at row_ptr(i); in every group of P lanes (P a power of
// two >= nchunks) lane ci copies 16-byte chunk chunk0 + ci of it.
// Thread group g takes items g, g + ng, g + 2 ng, ...  All threads run the
// same number of steps, so consume() may use warp shuffles; it receives every
// item slot with `in` = item < count and the chunk (zeros for idle lanes).
// A thread only reuses a ring slot after its own consume() used the data.
template <class Ring, class RowPtr, class Consume>
__device__ __forceinline__ void stream_rows(int chunk0, int nchunks, int P, int count,
                                            RowPtr row_ptr, Consume consume, uint32_t ring) {
  const int tid = threadIdx.x, lane = tid & 31;
  const int ci = lane & (P - 1);
  const bool active = ci < nchunks;
  const int ng = kThreads / P, g = tid / P;
  constexpr int kRingStages = Ring::kStages, kRingItems = Ring::kItems;
  const int per_stage = ng * kRingItems;
  const int nst = count > 0 ? (count + per_stage - 1) / per_stage : 0;
  const uint32_t my = ring + (uint32_t)tid * 16u;
  const int coff = (chunk0 + ci) * 8;
  auto slot = [&](int s, int u) {
    return my + (uint32_t)((s * kRingItems + u) * kThreads * 16);
  };
  auto issue = [&](int st) {
    if (st < nst) {
#pragma unroll
      for (int u = 0; u < kRingItems; ++u) {
        const int item = g + (st * kRingItems + u) * ng;
        if (active && item < count) cp_async16(slot(st % kRingStages, u), row_ptr(item) + coff);
      }
    }
    cp_async_commit();
  };
  for (int st = 0; st < kRingStages; ++st) issue(st);
  for (int st = 0; st < nst; ++st) {
    cp_async_wait<kRingStages - 1>();
#pragma unroll
    for (int u = 0; u < kRingItems; ++u) {
      const int item = g + (st * kRingItems + u) * ng;
      const bool in = item < count;
      uint4 q = make_uint4(0, 0, 0, 0);
      if (active && in) q = ld_shared16(slot(st % kRingStages, u));
      consume(item, in, q);
    }
    issue(st + kRingStages);
  }
  cp_async_wait<0>();
}

// Squared norm of one 16-byte chunk (8 bf16 values) of a row: of v - mean
// for VAR 0, of v itself for VAR 2.  The chunk's mean arrives as packed
// pairs of its fp32 part m2 and remainder l2: (x - m2) - l2 is rounded
// relative to x - mean itself, so the score's error is relative to the
// score (with the fp32 mean alone it would carry an absolute 2^-24 |mean|).
template <int VAR, int LPR>
__device__ __forceinline__ float chunk_sq(const uint4& q, const unsigned long long (&m2)[4],
                                          uint32_t lo_addr) {
  const uint32_t w[4] = {q.x, q.y, q.z, q.w};
  unsigned long long acc = 0ull;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const unsigned long long x = bf16x2_to_f2(w[k]);
    if (VAR == 0) {
      // the remainder pair is read from shared memory at each use rather
      // than held in registers (the kernels sit at their register limit)
      const unsigned long long l2 = ld_shared_b64(lo_addr + (uint32_t)(k * LPR * 8));
      const unsigned long long dv = f2_sub(f2_sub(x, m2[k]), l2);
      acc = f2_fma(dv, dv, acc);
    } else {
      acc = f2_fma(x, x, acc);
    }
  }
  return f2_hsum(acc);
}

// Score pass over R contiguous rows (row stride d = 8 * LPR elements, LPR in
// {8, 16, 32} lanes per row) for the L2 (VAR 0) and Norm (VAR 2) rules.
// Rows stream through the thread-private cp.async ring; each lane keeps its
// chunk's partial sums for a batch of kBatch rows and the LPR lanes of a row
// group reduce the batch with a transposed butterfly (kBatch - 1 exchanges
// for kBatch rows, then log2(LPR / kBatch) plain steps), after which lane
// ci holds row ci / (LPR / kBatch) of the batch: the lanes with
// ci % (LPR / kBatch) == 0 call finish(j, s) for the batch's valid rows (j is
// the row's index in [0, R)).  Same arithmetic per element as the general
// path; only the order of the fp32 additions differs.  Rows are visited from
// the last to the first (see the score pass in evict_kernel).
// R >= 1 (callers skip empty ranges).
template <int VAR, int LPR, class Ring, int BATCH, class Finish>
__device__ __forceinline__ void score_rows_fast(const uint16_t* __restrict__ rows, int R,
                                                const float* mu, const float* mulo,
                                                Finish finish, uint32_t ring) {
  constexpr int kStages = Ring::kStages, kItems = Ring::kItems;
  constexpr int kBatch = BATCH;
  constexpr int kLogBatch = kBatch == 8 ? 3 : kBatch == 4 ? 2 : 1;
  static_assert((1 << kLogBatch) == kBatch && kBatch % kItems == 0 && LPR >= kBatch,
                "batch shape");
  constexpr int kStagesPerBatch = kBatch / kItems;
  constexpr int kGroups = kThreads / LPR;
  constexpr int kD = LPR * 8;
  constexpr int kSpread = LPR / kBatch;  // lanes per row after the transposed steps
  const int tid = threadIdx.x, lane = tid & 31, ci = lane & (LPR - 1), g = tid / LPR;
  unsigned long long m2[4];
#pragma unroll
  for (int k = 0; k < 4; ++k)
    m2[k] = VAR == 0 ? f2_pack(mu[ci * 8 + 2 * k], mu[ci * 8 + 2 * k + 1]) : 0ull;
  // mulo is in the pair-transposed layout (lo_index): pair k of chunk ci at
  // float 2 * (k * LPR + ci), so a warp's loads of one pair hit distinct banks
  const uint32_t lo_addr = smem_addr(mulo) + (uint32_t)ci * 8u;
  const int per_stage = kGroups * kItems;
  const int nst = (R + per_stage - 1) / per_stage;
  const uint32_t my = ring + (uint32_t)tid * 16u;
  // visit k of group g reads row R - 1 - (g + k * kGroups)
  const uint16_t* p0 = rows + (size_t)(R - 1) * kD + ci * 8;
  auto slot = [&](int s, int u) {
    return my + (uint32_t)((s * kItems + u) * kThreads * 16);
  };
  auto issue = [&](int st) {
    if (st < nst) {
#pragma unroll
      for (int u = 0; u < kItems; ++u) {
        const int k = st * kItems + u;  // this group's k-th row: g + k * kGroups
        const int i = g + k * kGroups;
        if (i < R) cp_async16(slot(st % kStages, u), p0 - (size_t)i * kD);
      }
    }
    cp_async_commit();
  };
  for (int st = 0; st < kStages; ++st) issue(st);
  const int nbatch = (nst + kStagesPerBatch - 1) / kStagesPerBatch;
  for (int b = 0; b < nbatch; ++b) {
    float part[kBatch];
#pragma unroll
    for (int sb = 0; sb < kStagesPerBatch; ++sb) {
      const int st = b * kStagesPerBatch + sb;
      cp_async_wait<kStages - 1>();
#pragma unroll
      for (int u = 0; u < kItems; ++u) {
        const int k = st * kItems + u;
        uint4 q = make_uint4(0u, 0u, 0u, 0u);
        if (g + k * kGroups < R) q = ld_shared16(slot(st % kStages, u));
        part[sb * kItems + u] = chunk_sq<VAR, LPR>(q, m2, lo_addr);
      }
      issue(st + kStages);
    }
    // transposed steps over lane offsets LPR/2, LPR/4, LPR/8
#pragma unroll
    for (int j = 0; j < kLogBatch; ++j) {
      const int h = kBatch >> (j + 1), off = LPR >> (j + 1);
      const bool upper = (ci & off) != 0;
#pragma unroll
      for (int k = 0; k < h; ++k) {
        const float send = upper ? part[k] : part[k + h];
        const float keep = upper ? part[k + h] : part[k];
        part[k] = keep + __shfl_xor_sync(kFull, send, off);
      }
    }
#pragma unroll
    for (int off = kSpread / 2; off >= 1; off >>= 1) part[0] += __shfl_xor_sync(kFull, part[0], off);
    if (ci % kSpread == 0) {
      const int j = g + (b * kBatch + ci / kSpread) * kGroups;
      if (j < R) finish(R - 1 - j, sqrtf(part[0]));
    }
  }
  cp_async_wait<0>();
}

// Merges every thread's double-float column partials (8 columns from column
// `col`, lanes grouped P per row) into acc_hi/acc_lo (zeroed by the caller),
// across the warp with TwoSum shuffles and across warps in a fixed order.
__device__ __forceinline__ void merge_columns(float (&hi)[8], float (&lo)[8], int P, bool active,
                                              int col, float* acc_hi, float* acc_lo) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  ff p[8];
#pragma unroll
  for (int k = 0; k < 8; ++k) p[k] = ff_add(ff{hi[k], 0.f}, ff{0.f, lo[k]});
  for (int off = P; off < 32; off <<= 1) {
#pragma unroll
    for (int k = 0; k < 8; ++k) p[k] = ff_add(p[k], ff_shfl_xor(p[k], off));
  }
  for (int w = 0; w < kWarps; ++w) {
    if (warp == w && lane < P && active) {
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const ff a = ff_add(ff{acc_hi[col + k], acc_lo[col + k]}, p[k]);
        acc_hi[col + k] = a.hi;
        acc_lo[col + k] = a.lo;
      }
    }
    __syncthreads();
  }
}

// acc (zeroed here) <- sum over items [0, count) of sign(item) * (the row at
// row_ptr(item)), restricted to 16-byte column chunks [chunk0, chunk0 +
// nchunks).
// PACKED: TwoSum on packed fp32 pairs (half the instructions); the scalar
// form gives bit-identical sums and is kept where the packed one would not
// fit the kernel's register budget (the Dir block kernels).
template <class Ring, bool PACKED = true, class RowPtr, class SignOf>
__device__ __forceinline__ void sum_rows(int chunk0, int nchunks, int P, int count,
                                         RowPtr row_ptr, SignOf sign_of, Smem& S, uint32_t ring) {
  S.acc_hi[threadIdx.x] = 0.f;
  S.acc_lo[threadIdx.x] = 0.f;
  __syncthreads();
  const int ci = (threadIdx.x & 31) & (P - 1);
  const bool active = ci < nchunks;
  // the columns of this lane's chunk as packed pairs (2k, 2k + 1); each
  // element enters with TwoSum (ff2_accumulate), a row of sign -1 with its
  // sign bits flipped (exactly sign_of(item) * x)
  float hi[8], lo[8];
  if constexpr (PACKED) {
    unsigned long long hi2[4], lo2[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) hi2[k] = lo2[k] = 0ull;
    stream_rows<Ring>(chunk0, nchunks, P, count, row_ptr,
                      [&](int item, bool in, const uint4& q) {
                        if (in && active) {
                          const uint32_t flip = sign_of(item) < 0.f ? 0x80008000u : 0u;
                          const uint32_t w[4] = {q.x ^ flip, q.y ^ flip, q.z ^ flip, q.w ^ flip};
#pragma unroll
                          for (int k = 0; k < 4; ++k)
                            ff2_accumulate(hi2[k], lo2[k], bf16x2_to_f2(w[k]));
                        }
                      },
                      ring);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      f2_unpack(hi2[k], hi[2 * k], hi[2 * k + 1]);
      f2_unpack(lo2[k], lo[2 * k], lo[2 * k + 1]);
    }
  } else {
#pragma unroll
    for (int k = 0; k < 8; ++k) hi[k] = lo[k] = 0.f;
    stream_rows<Ring>(chunk0, nchunks, P, count, row_ptr,
                      [&](int item, bool in, const uint4& q) {
                        if (in && active) {
                          float x[8];
                          unpack8(q, x);
                          const float sg = sign_of(item);
#pragma unroll
                          for (int k = 0; k < 8; ++k) ff_accumulate(hi[k], lo[k], sg * x[k]);
                        }
                      },
                      ring);
  }
  merge_columns(hi, lo, P, active, (chunk0 + ci) * 8, S.acc_hi, S.acc_lo);
}

static_assert(kBulkStages >= 2 && kBulkStages <= 4, "bulk ring: 2 to 4 stages (Smem::bar)");

// A ring of bulk copies over this CTA's ring region: kBulkStages slots of
// kBulkStageBytes, slot s completing on mbarrier Smem::bar[s].  gst counts
// the stages started by every stream of the launch so far (the same value in
// every thread): stage g uses slot g % S and waits for parity (g / S) & 1.
struct BulkRing {
  uint32_t ring, bar0;
  int gst;
};

__device__ __forceinline__ BulkRing bulk_ring_init(uint32_t ring, Smem& S) {
  const uint32_t bar0 = smem_addr(&S.bar[0]);
  if (threadIdx.x == 0) {
    for (int sl = 0; sl < kBulkStages; ++sl) mbar_init(bar0 + 8u * (uint32_t)sl, 1);
    fence_mbar_init();
  }
  __syncthreads();
  return {ring, bar0, 0};
}

// Streams nst stages of the rows at `base` (row_bytes each); stage_rows(i,
// first, count) names stage i's rows [first, first + count).  Thread 0 issues
// each stage as one bulk copy; every thread waits for it, consume(first,
// count, stage address) reads it, and a block barrier frees the slot before
// thread 0 refills it.
template <class StageRows, class Consume>
__device__ __forceinline__ void bulk_stream(BulkRing& br, const uint16_t* base, int nst,
                                            int row_bytes, StageRows stage_rows, Consume consume,
                                            unsigned* status) {
  auto issue = [&](int i) {
    int first, count;
    stage_rows(i, first, count);
    const uint32_t sl = (uint32_t)((br.gst + i) % kBulkStages);
    const uint32_t bar = br.bar0 + 8u * sl;
    const uint32_t bytes = (uint32_t)(count * row_bytes);
    fence_proxy_async_smem();  // the slot's previous contents were read by generic loads
    mbar_expect_tx(bar, bytes);
    bulk_g2s(br.ring + sl * (uint32_t)kBulkStageBytes,
             reinterpret_cast<const char*>(base) + (size_t)first * row_bytes, bytes, bar);
  };
  if (threadIdx.x == 0)
    for (int i = 0; i < nst && i < kBulkStages; ++i) issue(i);
  for (int i = 0; i < nst; ++i) {
    const int g = br.gst + i;
    const uint32_t sl = (uint32_t)(g % kBulkStages);
    mbar_wait(br.bar0 + 8u * sl, (uint32_t)(g / kBulkStages) & 1u, status);
    int first, count;
    stage_rows(i, first, count);
    consume(first, count, br.ring + sl * (uint32_t)kBulkStageBytes);
    __syncthreads();  // every thread is done with the slot
    if (threadIdx.x == 0 && i + kBulkStages < nst) issue(i + kBulkStages);
  }
  br.gst += nst;
}

// sum_rows over the contiguous rows [0, count) at `rows` (all d columns, P =
// d / 8 lanes per row), streamed through the bulk ring in ascending order.
// Lane group g takes rows g, g + 256/P, ... (a stage holds a whole number of
// such strides), as sum_rows does, so the sums are bit-identical to it.
__device__ __forceinline__ void sum_rows_bulk(BulkRing& br, const uint16_t* rows, int count,
                                              int d, int P, Smem& S, unsigned* status) {
  S.acc_hi[threadIdx.x] = 0.f;
  S.acc_lo[threadIdx.x] = 0.f;
  __syncthreads();
  const int row_bytes = d * 2, srows = kBulkStageBytes / row_bytes;
  const int ci = (threadIdx.x & 31) & (P - 1), g = threadIdx.x / P, ng = kThreads / P;
  const bool active = ci < (d >> 3);
  unsigned long long hi2[4], lo2[4];
#pragma unroll
  for (int k = 0; k < 4; ++k) hi2[k] = lo2[k] = 0ull;
  bulk_stream(
      br, rows, (count + srows - 1) / srows, row_bytes,
      [&](int i, int& first, int& cnt) {
        first = i * srows;
        cnt = min(srows, count - first);
      },
      [&](int, int cnt, uint32_t st) {
        if (!active) return;
        for (int r = g; r < cnt; r += ng) {
          const uint4 q = ld_shared16(st + (uint32_t)(r * row_bytes + ci * 16));
          const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
          for (int k = 0; k < 4; ++k) ff2_accumulate(hi2[k], lo2[k], bf16x2_to_f2(w[k]));
        }
      },
      status);
  float hi[8], lo[8];
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    f2_unpack(hi2[k], hi[2 * k], hi[2 * k + 1]);
    f2_unpack(lo2[k], lo[2 * k], lo[2 * k + 1]);
  }
  merge_columns(hi, lo, P, active, ci * 8, S.acc_hi, S.acc_lo);
}

// score_rows_fast through the bulk ring: a stage is one batch of 8 rows per
// lane group (32 KB at d = 64, 128, 256), taken from the last rows to the
// first; per row the same arithmetic as score_rows_fast.
template <int VAR, int LPR, class Finish>
__device__ __forceinline__ void score_rows_bulk(BulkRing& br, const uint16_t* rows, int R,
                                                const float* mu, const float* mulo,
                                                Finish finish, unsigned* status) {
  constexpr int kBatch = 8, kGroups = kThreads / LPR, kD = LPR * 8, kSpread = LPR / kBatch;
  constexpr int kRowBytes = kD * 2, kSRows = kBulkStageBytes / kRowBytes;
  static_assert(kSRows == kGroups * kBatch, "one batch per lane group per stage");
  const int tid = threadIdx.x, lane = tid & 31, ci = lane & (LPR - 1), g = tid / LPR;
  unsigned long long m2[4];
#pragma unroll
  for (int k = 0; k < 4; ++k)
    m2[k] = VAR == 0 ? f2_pack(mu[ci * 8 + 2 * k], mu[ci * 8 + 2 * k + 1]) : 0ull;
  const uint32_t lo_addr = smem_addr(mulo) + (uint32_t)ci * 8u;
  bulk_stream(
      br, rows, (R + kSRows - 1) / kSRows, kRowBytes,
      [&](int i, int& first, int& cnt) {
        const int end = R - i * kSRows;
        first = max(0, end - kSRows);
        cnt = end - first;
      },
      [&](int first, int cnt, uint32_t st) {
        float part[kBatch];
#pragma unroll
        for (int k = 0; k < kBatch; ++k) {
          const int r = g + k * kGroups;
          uint4 q = make_uint4(0u, 0u, 0u, 0u);
          if (r < cnt) q = ld_shared16(st + (uint32_t)(r * kRowBytes + ci * 16));
          part[k] = chunk_sq<VAR, LPR>(q, m2, lo_addr);
        }
#pragma unroll
        for (int j = 0; j < 3; ++j) {
          const int h = kBatch >> (j + 1), off = LPR >> (j + 1);
          const bool upper = (ci & off) != 0;
#pragma unroll
          for (int k = 0; k < h; ++k) {
            const float send = upper ? part[k] : part[k + h];
            const float keep = upper ? part[k + h] : part[k];
            part[k] = keep + __shfl_xor_sync(kFull, send, off);
          }
        }
#pragma unroll
        for (int off = kSpread / 2; off >= 1; off >>= 1)
          part[0] += __shfl_xor_sync(kFull, part[0], off);
        if (ci % kSpread == 0) {
          const int r = g + (ci / kSpread) * kGroups;
          if (r < cnt) finish(first + r, sqrtf(part[0]));
        }
      },
      status);
}

// Order-preserving key of a score (scores are never negative): a positive
// score maps to its bit pattern + 1 (+inf to 0x7f800001), +0 and -0 both to
// 1, and NaN to 0, strictly below every number, so a NaN ranks lowest and
// never ties with a zero score.  `bad` reports a NaN or infinite score.
__device__ __forceinline__ uint32_t score_key(float s, bool& bad) {
  bad = !(s == s) || s == __int_as_float(0x7f800000);
  return s > 0.f ? __float_as_uint(s) + 1u : (s == 0.f ? 1u : 0u);
}

// The score a key came from (+0 for either zero, NaN for key 0).
__device__ __forceinline__ float key_score(uint32_t key) {
  return key ? __uint_as_float(key - 1u) : __int_as_float(0x7fc00000);
}

// Dispersion of the L2 scores over a unit (Sec. 3.1: sigma = std_j s_j):
// every thread's double-float sums of s and s^2 are merged in a fixed order
// into this CTA's S.disp (ends with a block barrier).  wsc: 4 * kWarps floats
// of block-private scratch (peer CTAs may still be reading S.acc_*).
__device__ __forceinline__ void disp_reduce_cta(float ds_hi, float ds_lo, float dq_hi,
                                                float dq_lo, float* wsc, Smem& S) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  ff a1 = ff_add(ff{ds_hi, 0.f}, ff{0.f, ds_lo});
  ff a2 = ff_add(ff{dq_hi, 0.f}, ff{0.f, dq_lo});
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    a1 = ff_add(a1, ff_shfl_xor(a1, off));
    a2 = ff_add(a2, ff_shfl_xor(a2, off));
  }
  if (lane == 0) {
    wsc[warp] = a1.hi;
    wsc[kWarps + warp] = a1.lo;
    wsc[2 * kWarps + warp] = a2.hi;
    wsc[3 * kWarps + warp] = a2.lo;
  }
  __syncthreads();
  if (tid == 0) {
    ff t1{0.f, 0.f}, t2{0.f, 0.f};
    for (int w = 0; w < kWarps; ++w) {
      t1 = ff_add(t1, ff{wsc[w], wsc[kWarps + w]});
      t2 = ff_add(t2, ff{wsc[2 * kWarps + w], wsc[3 * kWarps + w]});
    }
    S.disp[0] = t1.hi;
    S.disp[1] = t1.lo;
    S.disp[2] = t2.hi;
    S.disp[3] = t2.lo;
  }
  __syncthreads();
}

// sigma = sqrt(E[s^2] - E[s]^2) from the S.disp of the cluster's C CTAs, in
// rank order (one thread; every CTA's S.disp must be complete and its CTA
// still resident).
__device__ __forceinline__ float disp_finish(Smem& S, int C, int n) {
  double s1 = 0.0, s2 = 0.0;
  const uint32_t base = smem_addr(&S.disp[0]);
  for (int rr = 0; rr < C; ++rr) {
    float v[4];
    for (int k = 0; k < 4; ++k)
      v[k] = C > 1 ? ld_cluster_f32(mapa(base + 4u * (unsigned)k, (unsigned)rr)) : S.disp[k];
    s1 += (double)v[0] + (double)v[1];
    s2 += (double)v[2] + (double)v[3];
  }
  const double m = s1 / (double)n;
  const double var = s2 / (double)n - m * m;
  return (float)sqrt(var > 0.0 ? var : 0.0);
}

// Radix select over the keys of the whole cluster: t = the N-th largest key
// (1-based), keep_eq = how many keys equal to t survive, cnt_eq = how many
// keys equal t.  key_of(j, ok) gives the key of this CTA's j-th row (j < R)
// and whether the row takes part.
struct Selection {
  uint32_t t;
  int keep_eq;
  int cnt_eq;
};

// first_ready: S.hist[0] already holds this CTA's counts of the keys' top
// byte (built by the score pass), so the first pass skips its counting loop,
// and S.hist[1] was zeroed with it, so the second pass does not zero it.
//
// As soon as a pass leaves at most kThreads keys in the cluster that share
// the threshold's prefix (the candidates), the remaining passes are replaced
// by ranking the candidates directly: every CTA compacts its own candidates
// (into ghist, which peers then read), gathers the cluster's candidates, and
// each thread counts how many candidates are greater than and equal to its
// own.  The threshold is the candidate with g < need <= g + e.  Candidate
// counts come from the cluster-summed histogram, so every CTA of the cluster
// takes the same branch.
template <class KeyOf>
__device__ __forceinline__ Selection cluster_radix_select(KeyOf key_of, int R, int N, int C,
                                                          Smem& S, bool first_ready = false) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint32_t prefix = 0, pmask = 0;
  int need = N, cnt = 0;
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 24 - 8 * pass;
    uint32_t* h = S.hist[pass & 1];
    const bool counted = pass == 0 && first_ready;
    if (!(first_ready && pass <= 1)) {
      h[tid] = 0;
      __syncthreads();
    }
    for (int base = 0; !counted && base < R; base += kThreads) {
      const int j = base + tid;
      bool ok = false;
      uint32_t key = 0u;
      if (j < R) key = key_of(j, ok);
      const bool match = ok && (key & pmask) == prefix;
      const uint32_t dig = (key >> shift) & 255u;
      if (pass == 0) {
        // the top bytes of nearby scores coincide: one atomic per distinct digit
        const unsigned act = __ballot_sync(kFull, match);
        if (match) {
          const unsigned peers = __match_any_sync(act, dig);
          if (lane == __ffs(peers) - 1) atomicAdd(&h[dig], (uint32_t)__popc(peers));
        }
      } else if (match) {
        atomicAdd(&h[dig], 1u);  // later digits are spread: plain shared atomics
      }
    }
    if (C > 1) cluster_sync(); else __syncthreads();
    {
      uint32_t tot = 0;
      if (C > 1) {
        const uint32_t a = smem_addr(&h[tid]);
        for (int rr = 0; rr < C; ++rr) tot += ld_cluster_u32(mapa(a, (unsigned)rr));
      } else {
        tot = h[tid];
      }
      S.ghist[tid] = tot;
    }
    __syncthreads();
    if (warp == 0) {
      int c[8];
      int sum = 0;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        c[i] = (int)S.ghist[255 - (lane * 8 + i)];
        sum += c[i];
      }
      int incl = sum;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const int y = __shfl_up_sync(kFull, incl, off);
        if (lane >= off) incl += y;
      }
      const int excl = incl - sum;
      if (excl < need && need <= incl) {
        int cum = excl;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          if (cum + c[i] >= need) {
            S.sel_digit = 255 - (lane * 8 + i);
            S.sel_above = cum;
            S.sel_cnt = c[i];
            break;
          }
          cum += c[i];
        }
      }
    }
    __syncthreads();
    need -= S.sel_above;
    prefix |= (uint32_t)S.sel_digit << shift;
    pmask |= 255u << shift;
    cnt = S.sel_cnt;
    if (pass == 3 || cnt > kThreads) continue;

    // ---- rank resolution among the cnt candidates -------------------------
    // (ghist is free once every thread has read the scan's result above)
    if (tid == 0) S.ncand = 0;
    __syncthreads();
    for (int base = 0; base < R; base += kThreads) {
      const int j = base + tid;
      bool ok = false;
      uint32_t key = 0u;
      if (j < R) key = key_of(j, ok);
      const bool match = ok && (key & pmask) == prefix;
      const unsigned act = __ballot_sync(kFull, match);
      int at = 0;
      if (lane == 0 && act) at = atomicAdd(&S.ncand, __popc(act));
      at = __shfl_sync(kFull, at, 0);
      if (match) S.ghist[at + __popc(act & ((1u << lane) - 1u))] = key;
    }
    if (C > 1) cluster_sync(); else __syncthreads();
    // every CTA gathers the cluster's candidates, in rank order, into the
    // histogram buffer that no peer reads any more (the other pass's)
    uint32_t* all = S.hist[(pass + 1) & 1];
    uint32_t mine = 0u;
    {
      int off = 0;
      for (int rr = 0; rr < C; ++rr) {
        const int nc = C > 1 ? (int)ld_cluster_u32(mapa(smem_addr(&S.ncand), (unsigned)rr))
                             : S.ncand;
        if (tid >= off && tid < off + nc)
          mine = C > 1 ? ld_cluster_u32(mapa(smem_addr(&S.ghist[tid - off]), (unsigned)rr))
                       : S.ghist[tid - off];
        off += nc;
      }
    }
    if (tid < cnt) all[tid] = mine;
    __syncthreads();
    if (tid < cnt) {
      int g = 0, e = 0;
      for (int i = 0; i < cnt; ++i) {
        const uint32_t o = all[i];
        g += o > mine;
        e += o == mine;
      }
      if (g < need && need <= g + e) {  // every candidate equal to t writes the same
        S.sel_t = mine;
        S.sel_above = need - g;
        S.sel_cnt = e;
      }
    }
    __syncthreads();
    // peers read this CTA's candidates (ghist) until they pass the caller's
    // next cluster barrier; nothing writes ghist before it
    return {S.sel_t, S.sel_above, S.sel_cnt};
  }
  return {prefix, need, cnt};
}

// Ranks this CTA's rows [r0, r0 + R) against the selection and scatters them
// into perm[] of every CTA of the cluster: kept slots ascending at [0, N),
// evicted slots ascending at [N, n).  Threads own contiguous row chunks, so
// prefix sums follow slot order (ties go to the lower slot).  Ends with the
// cluster barrier after which every CTA's perm[] is complete.  A position
// outside [0, n) (impossible for a consistent selection) is skipped and
// recorded as kStInternal.
template <bool by_tiekey, class TieKey>
__device__ __forceinline__ void cluster_build_perm(const uint32_t* keys, int r0, int R, int N,
                                                   int n, Selection sel, uint32_t t2,
                                                   TieKey tiekey, int C, unsigned rank,
                                                   uint16_t* perm, unsigned* status, Smem& S) {
  const int tid = threadIdx.x;
  const int ch = (R + kThreads - 1) / kThreads;
  const int c0 = min(R, tid * ch), c1 = min(R, c0 + ch);
  const uint32_t t = sel.t;
  // ordered layout: ties go to the lowest slots (prefix counts below);
  // hole-fill layout: a tied row survives iff tiekey(j) >= t2
  int ngt = 0, neq = 0;
  for (int j = c0; j < c1; ++j) {
    ngt += keys[j] > t;
    if (keys[j] == t) neq += by_tiekey ? (tiekey(j) >= t2) : 1;
  }
  int tot_gt, tot_eq;
  const int gt_ex = block_exclusive_scan(ngt, S.scan, tot_gt);
  const int eq_ex = block_exclusive_scan(neq, S.scan, tot_eq);
  if (tid == 0) {
    S.cnt_gt = tot_gt;
    S.cnt_eq = tot_eq;
  }
  if (C > 1) cluster_sync(); else __syncthreads();
  // ties and kept rows of the lower-ranked CTAs
  const int q = sel.keep_eq;
  int tie_off = 0, kept_off = 0;
  for (int rr = 0; rr < (int)rank; ++rr) {
    const int g = (int)ld_cluster_u32(mapa(smem_addr(&S.cnt_gt), rr));
    const int e = (int)ld_cluster_u32(mapa(smem_addr(&S.cnt_eq), rr));
    kept_off += g + (by_tiekey ? e : min(max(q - tie_off, 0), e));
    tie_off += e;
  }
  const int my_tie_quota = max(q - tie_off, 0);  // ties this CTA may still keep
  int tie_rank = eq_ex;                          // ties of this CTA before the chunk
  int kp = kept_off + gt_ex + (by_tiekey ? eq_ex : min(my_tie_quota, eq_ex));
  const uint32_t perm_addr = smem_addr(perm);
  for (int j = c0; j < c1; ++j) {
    const uint32_t key = keys[j];
    const bool eq = key == t;
    const bool keep =
        key > t || (eq && (by_tiekey ? tiekey(j) >= t2 : tie_rank < my_tie_quota));
    tie_rank += eq;
    const int row = r0 + j;
    const int pos = keep ? kp : N + (row - kp);
    kp += keep;
    if ((unsigned)pos >= (unsigned)n) {  // self-check: a consistent selection never gets here
      record_status(status, kStInternal);
      continue;
    }
    if (C > 1) {
      for (int cc = 0; cc < C; ++cc)
        st_cluster_u16(mapa(perm_addr + 2u * (unsigned)pos, (unsigned)cc), (uint16_t)row);
    } else {
      perm[pos] = (uint16_t)row;
    }
  }
  if (C > 1) cluster_sync(); else __syncthreads();
}

// In-place, order-preserving move of rows [r_begin, r_end) of the column
// slice [chunk0, chunk0 + cps) of the concatenated [K | V] row: row r takes
// source row perm[r] (or r + 1 when perm is null: the decode shift).  A
// source at or above n (impossible for a consistent slot list) is not read
// and is recorded as kStInternal (its row then holds unspecified bytes).
// STAGED (fused append): sources at or above first_stage are rows of the
// staging buffers kn / vn ([B][d] per unit) and stream through the same
// ring; they are never cache rows, so the order stays hazard-free.
template <class Ring, bool STAGED>
__device__ __forceinline__ void compact_slice(uint16_t* kb, uint16_t* vb, int d, int chunk0,
                                              int cps, int r_begin, int r_end, int n,
                                              const uint16_t* perm, unsigned* status,
                                              uint32_t ring, const uint16_t* kn,
                                              const uint16_t* vn, int first_stage) {
  const int tid = threadIdx.x;
  const int d8 = d >> 3;
  const int rs = kThreads / cps;
  const bool on = tid < rs * cps;
  const int my_ch = chunk0 + tid % cps;
  const int my_off = tid / cps;
  uint16_t* col = my_ch < d8 ? kb + my_ch * 8 : vb + (my_ch - d8) * 8;
  const uint16_t* scol = nullptr;  // this thread's column of the staging rows
  if constexpr (STAGED) scol = my_ch < d8 ? kn + my_ch * 8 : vn + (my_ch - d8) * 8;
  constexpr int kRingStages = Ring::kStages, kRingItems = Ring::kItems;
  const int tile = rs * kRingItems;
  const int ntiles = r_end > r_begin ? (r_end - r_begin + tile - 1) / tile : 0;
  const uint32_t my = ring + (uint32_t)tid * 16u;
  auto slot = [&](int s, int u) {
    return my + (uint32_t)((s * kRingItems + u) * kThreads * 16);
  };
  auto issue = [&](int t) {
    if (t < ntiles) {
#pragma unroll
      for (int u = 0; u < kRingItems; ++u) {
        const int r = r_begin + t * tile + u * rs + my_off;
        if (on && r < r_end) {
          const int src = perm ? (int)perm[r] : r + 1;
          if (src < n) {
            const uint16_t* sp = col + (size_t)src * d;
            if constexpr (STAGED)
              if (src >= first_stage) sp = scol + (size_t)(src - first_stage) * d;
            cp_async16(slot(t % kRingStages, u), sp);
          } else {
            record_status(status, kStInternal);
          }
        }
      }
    }
    cp_async_commit();
  };
  for (int t = 0; t < kRingStages; ++t) issue(t);
  for (int t = 0; t < ntiles; ++t) {
    cp_async_wait<kRingStages - 1>();
    __syncthreads();  // every source of tile t is in shared memory
#pragma unroll
    for (int u = 0; u < kRingItems; ++u) {
      const int r = r_begin + t * tile + u * rs + my_off;
      if (on && r < r_end) st16(col + (size_t)r * d, ld_shared16(slot(t % kRingStages, u)));
    }
    issue(t + kRingStages);
  }
  cp_async_wait<0>();
}

// Fused append of a unit that does not evict: staging rows [0, B) go to
// cache rows [first, first + B), this CTA's column slice [chunk0, chunk0 +
// cps) of [K | V].
__device__ __forceinline__ void copy_new_rows(uint16_t* kb, uint16_t* vb, const uint16_t* kn,
                                              const uint16_t* vn, int d, int chunk0, int cps,
                                              int first, int B) {
  const int d8 = d >> 3;
  const int items = B * cps;
  constexpr int U = 4;
  for (int base = threadIdx.x; base < items; base += kThreads * U) {
    uint4 q[U];
    uint16_t* dstp[U];
#pragma unroll
    for (int k = 0; k < U; ++k) {
      const int it = base + k * kThreads;
      dstp[k] = nullptr;
      if (it < items) {
        const int i = it / cps, c = chunk0 + it % cps;
        q[k] = ld_cg16((c < d8 ? kn + c * 8 : vn + (c - d8) * 8) + (size_t)i * d);
        dstp[k] = (c < d8 ? kb + c * 8 : vb + (c - d8) * 8) + (size_t)(first + i) * d;
      }
    }
#pragma unroll
    for (int k = 0; k < U; ++k)
      if (dstp[k]) st16(dstp[k], q[k]);
  }
}

// Hole-fill layout: move h rows, row src_of(i) -> row dst_of(i), of the
// column slice [chunk0, chunk0 + cps) of [K | V].  Every source lies at or
// above N and every destination below it, so the moves are independent.  A
// row outside [0, n) (impossible for a consistent slot list) is skipped and
// recorded as kStInternal.
template <class SrcOf, class DstOf>
__device__ __forceinline__ void move_rows(uint16_t* kb, uint16_t* vb, int d, int chunk0, int cps,
                                          int h, int n, SrcOf src_of, DstOf dst_of,
                                          unsigned* status, const uint16_t* kn = nullptr,
                                          const uint16_t* vn = nullptr,
                                          int first_stage = INT_MAX) {
  const int d8 = d >> 3;
  const int items = h * cps;
  constexpr int U = 4;
  for (int base = threadIdx.x; base < items; base += kThreads * U) {
    uint4 q[U];
    uint16_t* dstp[U];
#pragma unroll
    for (int k = 0; k < U; ++k) {
      const int it = base + k * kThreads;
      dstp[k] = nullptr;
      if (it < items) {
        const int i = it / cps, c = chunk0 + it % cps;
        uint16_t* col = c < d8 ? kb + c * 8 : vb + (c - d8) * 8;
        const int sr = src_of(i), dr = dst_of(i);
        if ((unsigned)sr < (unsigned)n && (unsigned)dr < (unsigned)n) {
          // fused append: sources at or above first_stage are staging rows
          q[k] = ld_cg16(sr >= first_stage
                             ? (c < d8 ? kn + c * 8 : vn + (c - d8) * 8) + (size_t)(sr - first_stage) * d
                             : col + (size_t)sr * d);
          dstp[k] = col + (size_t)dr * d;
        } else {
          record_status(status, kStInternal);
        }
      }
    }
#pragma unroll
    for (int k = 0; k < U; ++k)
      if (dstp[k]) st16(dstp[k], q[k]);
  }
}

// move_rows through this CTA's cp.async ring (block hole-fill events, which
// move up to B rows): item i of the h * cps (row, chunk) items is copied from
// row src_of(i / cps) to row dst_of(i / cps) of the column slice.  Sources
// lie at or above N and destinations below it, so no copy can read what
// another writes: each thread stores what it loaded itself, with no barrier
// between tiles, and keeps kStages x kItems copies in flight.  A row
// outside [0, n) is skipped and recorded as kStInternal.
template <class Ring, class SrcOf, class DstOf>
__device__ __forceinline__ void move_rows_ring(uint16_t* kb, uint16_t* vb, int d, int chunk0,
                                               int cps, int h, int n, SrcOf src_of, DstOf dst_of,
                                               unsigned* status, const uint16_t* kn,
                                               const uint16_t* vn, int first_stage,
                                               uint32_t ring) {
  constexpr int kStages = Ring::kStages, kItems = Ring::kItems;
  const int d8 = d >> 3;
  const int items = h * cps;
  const int per_stage = kThreads * kItems;
  const int nst = (items + per_stage - 1) / per_stage;
  const uint32_t my = ring + (uint32_t)threadIdx.x * 16u;
  auto slot = [&](int st, int u) {
    return my + (uint32_t)((st * kItems + u) * kThreads * 16);
  };
  // item of this thread's u-th copy of stage st, and its destination
  auto item_of = [&](int st, int u) { return (st * kItems + u) * kThreads + (int)threadIdx.x; };
  auto dst_ptr = [&](int it) -> uint16_t* {
    const int i = it / cps, c = chunk0 + it % cps;
    const int dr = dst_of(i), sr = src_of(i);
    if ((unsigned)sr >= (unsigned)n || (unsigned)dr >= (unsigned)n) return nullptr;
    return (c < d8 ? kb + c * 8 : vb + (c - d8) * 8) + (size_t)dr * d;
  };
  auto issue = [&](int st) {
    if (st < nst) {
#pragma unroll
      for (int u = 0; u < kItems; ++u) {
        const int it = item_of(st, u);
        if (it < items) {
          const int i = it / cps, c = chunk0 + it % cps;
          const int sr = src_of(i), dr = dst_of(i);
          if ((unsigned)sr < (unsigned)n && (unsigned)dr < (unsigned)n) {
            const uint16_t* sp = sr >= first_stage
                                     ? (c < d8 ? kn + c * 8 : vn + (c - d8) * 8) +
                                           (size_t)(sr - first_stage) * d
                                     : (c < d8 ? kb + c * 8 : vb + (c - d8) * 8) + (size_t)sr * d;
            cp_async16(slot(st % kStages, u), sp);
          } else {
            record_status(status, kStInternal);
          }
        }
      }
    }
    cp_async_commit();
  };
  for (int st = 0; st < kStages; ++st) issue(st);
  for (int st = 0; st < nst; ++st) {
    cp_async_wait<kStages - 1>();
#pragma unroll 1
    for (int u = 0; u < kItems; ++u) {
      const int it = item_of(st, u);
      if (it < items) {
        uint16_t* dp = dst_ptr(it);
        if (dp) st16(dp, ld_shared16(slot(st % kStages, u)));
      }
    }
    issue(st + kStages);
  }
  cp_async_wait<0>();
}

// Hole-fill block events: the kept rows at or above N move into the evicted
// slots below N, and, with the running mean, the evicted rows leave the
// running sum in the same stream.  ev_of(i), i < ne = n - N, lists the
// evicted rows ascending: the first h are the holes below N, which receive
// the movers src_of(i); the rest lie at or above N and are only subtracted.
// Threads keep one 16-byte column chunk of [K | V] (compact_slice's
// mapping), so each thread reads a hole's old bytes and writes the mover's
// into it itself, after both copies have landed, and no barrier is needed
// between ring stages; sources and holes never overlap.  Thread chunks in the
// scored tensor ([sc_lo, sc_hi) of [K | V], when `retire`) accumulate minus
// the evicted rows in double-float; the partials are added per column in a
// fixed order and base[c] plus them is written to rsum_out[c] for this CTA's
// columns of the scored tensor (tchunk0, tchunks).  Rows at or above
// first_stage are read from the staging buffers kn / vn.  A row outside
// [0, n) is skipped and recorded as kStInternal.
template <class Ring, bool PACKED, class SrcOf, class EvOf>
__device__ __forceinline__ void move_rows_retire(uint16_t* kb, uint16_t* vb, int d, int chunk0,
                                                 int cps, int h, int ne, int n, SrcOf src_of,
                                                 EvOf ev_of, unsigned* status, const uint16_t* kn,
                                                 const uint16_t* vn, int first_stage,
                                                 uint32_t ring, bool retire, int sc_lo,
                                                 int sc_hi, int tchunk0, int tchunks,
                                                 uint32_t base, double* rsum_out) {
  static_assert(Ring::kItems >= 2, "one ring slot for the mover, one for the evicted row");
  constexpr int kStages = Ring::kStages;
  const int tid = threadIdx.x, d8 = d >> 3;
  const int rs = kThreads / cps;
  const bool on = tid < rs * cps;
  const int my_ch = chunk0 + tid % cps, my_off = tid / cps;
  const bool scored = retire && on && my_ch >= sc_lo && my_ch < sc_hi;
  uint16_t* col = my_ch < d8 ? kb + my_ch * 8 : vb + (my_ch - d8) * 8;
  const uint16_t* scol = my_ch < d8 ? kn + my_ch * 8 : vn + (my_ch - d8) * 8;
  auto rowp = [&](int r) -> const uint16_t* {
    return r >= first_stage ? scol + (size_t)(r - first_stage) * d : col + (size_t)r * d;
  };
  // this thread's rows: my_off, my_off + rs, ... below h (moves) or ne (retired)
  const int lim = scored ? ne : h;
  const int cnt = on && lim > my_off ? (lim - my_off + rs - 1) / rs : 0;
  const uint32_t my = ring + (uint32_t)tid * 16u;
  auto slot = [&](int st, int k) { return my + (uint32_t)((st * Ring::kItems + k) * kThreads * 16); };
  auto issue = [&](int j) {
    if (j < cnt) {
      const int i = my_off + j * rs;
      const int ev = ev_of(i);
      if ((unsigned)ev < (unsigned)n) {
        if (i < h) {
          const int sr = src_of(i);
          if ((unsigned)sr < (unsigned)n) cp_async16(slot(j % kStages, 0), rowp(sr));
          else record_status(status, kStInternal);
        }
        if (scored) cp_async16(slot(j % kStages, 1), rowp(ev));
      } else {
        record_status(status, kStInternal);
      }
    }
    cp_async_commit();
  };
  float hi[8], lo[8];
  unsigned long long hi2[4], lo2[4];
#pragma unroll
  for (int k = 0; k < 8; ++k) hi[k] = lo[k] = 0.f;
#pragma unroll
  for (int k = 0; k < 4; ++k) hi2[k] = lo2[k] = 0ull;
  for (int j = 0; j < kStages; ++j) issue(j);
  for (int j = 0; j < cnt; ++j) {
    cp_async_wait<kStages - 1>();
    const int i = my_off + j * rs;
    const int ev = ev_of(i);
    if ((unsigned)ev < (unsigned)n) {
      if (scored) {  // minus the evicted row: its sign bits flipped (exact)
        const uint4 q = ld_shared16(slot(j % kStages, 1));
        const uint32_t w[4] = {q.x ^ 0x80008000u, q.y ^ 0x80008000u, q.z ^ 0x80008000u,
                               q.w ^ 0x80008000u};
        if constexpr (PACKED) {
#pragma unroll
          for (int k = 0; k < 4; ++k) ff2_accumulate(hi2[k], lo2[k], bf16x2_to_f2(w[k]));
        } else {
          float x[8];
          unpack8(uint4{w[0], w[1], w[2], w[3]}, x);
#pragma unroll
          for (int k = 0; k < 8; ++k) ff_accumulate(hi[k], lo[k], x[k]);
        }
      }
      if (i < h && (unsigned)src_of(i) < (unsigned)n)
        st16(col + (size_t)ev * d, ld_shared16(slot(j % kStages, 0)));
    }
    issue(j + kStages);
  }
  cp_async_wait<0>();
  if (!retire) return;
  if constexpr (PACKED) {
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      f2_unpack(hi2[k], hi[2 * k], hi[2 * k + 1]);
      f2_unpack(lo2[k], lo[2 * k], lo[2 * k + 1]);
    }
  }
  // per-column partials of the rs threads that share a chunk (in the ring,
  // free once every copy has landed: hi parts, then lo parts, 4 bytes per
  // column), then their sum in the order of the threads
  __syncthreads();
  const uint32_t w = (uint32_t)cps * 32u;  // bytes of one thread row of partials
  const uint32_t lo_off = (uint32_t)rs * w;
  if (scored) {
    const uint32_t at = ring + (uint32_t)my_off * w + (uint32_t)(my_ch - chunk0) * 32u;
    st_shared16(at, uint4{__float_as_uint(hi[0]), __float_as_uint(hi[1]), __float_as_uint(hi[2]),
                          __float_as_uint(hi[3])});
    st_shared16(at + 16u, uint4{__float_as_uint(hi[4]), __float_as_uint(hi[5]),
                                __float_as_uint(hi[6]), __float_as_uint(hi[7])});
    st_shared16(at + lo_off, uint4{__float_as_uint(lo[0]), __float_as_uint(lo[1]),
                                   __float_as_uint(lo[2]), __float_as_uint(lo[3])});
    st_shared16(at + lo_off + 16u, uint4{__float_as_uint(lo[4]), __float_as_uint(lo[5]),
                                         __float_as_uint(lo[6]), __float_as_uint(lo[7])});
  }
  __syncthreads();
  if (tid < tchunks * 8) {
    const int c = tchunk0 * 8 + tid;           // column of the scored tensor
    const int lc = c + sc_lo * 8 - chunk0 * 8;  // its column within this CTA's slice
    ff t{0.f, 0.f};
    for (int o = 0; o < rs; ++o) {
      const uint32_t at = ring + (uint32_t)o * w + (uint32_t)lc * 4u;
      t = ff_add(t, ff{ld_shared_f32(at), ld_shared_f32(at + lo_off)});
    }
    rsum_out[c] = ld_shared_f64(base + (uint32_t)c * 8u) + (double)t.hi + (double)t.lo;
  }
}

// VAR: 0 L2, 1 Dir, 2 Norm.  DECODE: one-token eviction (arg-min) instead of
// the radix select.  HF: hole-fill layout (compiled separately, so the ordered
// layout carries none of its code).  FUSED: the new rows are read from the
// caller's staging buffers (vd_append_evict_*); the other kernels carry none
// of that code.  SCORE: the score-only launches (vd_score, vd_score_ex:
// mean, scores and sigma, nothing evicted), instantiated with DECODE set
// and their own ring and occupancy.
template <int VAR, bool DECODE, bool HF, bool FUSED, bool SCORE>
__device__ __forceinline__ void evict_unit(const EvictArgs& a) {
  static_assert(!SCORE || (DECODE && !HF && !FUSED), "score-only instantiation");
  extern __shared__ __align__(16) unsigned char smem_raw[];
  Smem& S = *reinterpret_cast<Smem*>(smem_raw);
  using Ring = RingShape<SCORE ? ScoreRing::kStages : DECODE ? DecodeRing::kStages
                                                             : BlockRing::kStages,
                         SCORE ? ScoreRing::kItems : DECODE ? DecodeRing::kItems
                                                            : BlockRing::kItems>;
  constexpr bool score_only = SCORE;
  const int C = a.cluster;
  // score-only at head dims 64, 128, 256 (L2, Norm): the bulk-copy ring
  const bool bulk = SCORE && score_bulk(VAR, a.d);
  const int kind = SCORE ? (bulk ? kKindScoreBulk : kKindScore) : DECODE ? kKindDecode : kKindBlock;
  const SmemLayout L = smem_layout(a.capacity, C, kind);
  const uint32_t ring = smem_addr(smem_raw + L.ring);
  uint32_t* keys = reinterpret_cast<uint32_t*>(smem_raw + L.keys);
  uint16_t* perm = reinterpret_cast<uint16_t*>(smem_raw + L.perm);

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const unsigned rank = C > 1 ? cluster_ctarank() : 0u;
  const int u = C > 1 ? (int)cluster_id_x() : (int)blockIdx.x;
  const int d = a.d, d8 = d >> 3;
  const int seq = (u + a.unit_base) / a.units_per_seq;  // unit pointers come pre-offset
  constexpr bool fused = FUSED;  // the new rows are still in the staging buffers
  // packed-pair row sums everywhere but the Dir block kernels (register budget)
  constexpr bool kPackedSum = !(VAR == 1 && !DECODE);
  const int len0 = a.len[seq];
  const int n = len0 + (fused ? a.B : 0);
  const int Nb = a.N_dev ? a.N_dev[seq] : a.N;
  const size_t ubase = (size_t)u * a.capacity * d;
  uint16_t* kb = a.k + ubase;
  uint16_t* vb = a.v + ubase;
  const uint16_t* sb = a.score_k ? kb : vb;  // rows the mean and the scores come from
  // fused append: rows at or above first_stage come from the staging buffers
  // (srow: a row of the scored tensor, V or K)
  const uint16_t* knu = fused ? a.k_new + (size_t)u * a.B * d : nullptr;
  const uint16_t* vnu = fused ? a.v_new + (size_t)u * a.B * d : nullptr;
  const uint16_t* snu = a.score_k ? knu : vnu;
  const int first_stage = fused ? n - a.B : INT_MAX;
  auto srow = [&](int r) -> const uint16_t* {
    return r >= first_stage ? snu + (size_t)(r - first_stage) * d : sb + (size_t)r * d;
  };
  // the start of a range [r, r + m) of rows that lies on one side of
  // first_stage (nullptr when it straddles it: then srow per row)
  auto srange = [&](int r, int m) -> const uint16_t* {
    if (r + m <= first_stage) return sb + (size_t)r * d;
    if (r >= first_stage) return snu + (size_t)(r - first_stage) * d;
    return nullptr;
  };

  // ---- validation: uniform across the cluster (per-sequence values only) ---
  if (len0 < 0 || n > a.capacity || (a.mu_running && !score_only && a.B > n)) {
    if (rank == 0 && tid == 0) record_status(a.status, kStDeviceLen);
    return;
  }
  if (!score_only && (Nb < 1 || Nb > a.N)) {
    if (rank == 0 && tid == 0) record_status(a.status, kStDeviceBudget);
    return;
  }
  const bool evict = !score_only && n > Nb;
  if (DECODE && evict && n > Nb + 1) {
    if (rank == 0 && tid == 0) record_status(a.status, kStDeviceBudget);
    return;
  }
  if (score_only && n == 0) return;
  BulkRing br{0u, 0u, 0};
  if constexpr (SCORE) {
    if (bulk) br = bulk_ring_init(ring, S);
  }

  // column slice of [K | V] this CTA compacts; the running sum is kept for
  // the part of it that lies in the scored tensor (V, or K for the key-side
  // rule): its chunks [tchunk0, tchunk0 + tchunks) of that tensor
  const int cps = (2 * d8) / C;
  const int chunk0 = (int)rank * cps;
  const int tchunk0 = a.score_k ? min(chunk0, d8) : max(chunk0, d8) - d8;
  const int tchunks = a.score_k ? max(0, min(chunk0 + cps, d8) - chunk0)
                                : max(0, chunk0 + cps - max(chunk0, d8));
  int tp = 1;
  while (tp < tchunks) tp <<= 1;
  const int first_new = n - a.B;
  // hole-fill layout: token positions (rows at or above first_new are the
  // appended ones, numbered from pos_new)
  constexpr bool hf = HF;
  int32_t* posu = hf && !score_only ? a.pos + (size_t)u * a.capacity : nullptr;
  const int pnew = hf && !score_only ? a.pos_new[seq] : 0;
  auto pos_of = [&](int r) -> int { return r < first_new ? posu[r] : pnew + (r - first_new); };

  if (!evict && !score_only) {
    if (fused) copy_new_rows(kb, vb, knu, vnu, d, chunk0, cps, first_stage, a.B);
    if (hf && rank == 0)
      for (int r = max(first_new, 0) + tid; r < n; r += kThreads) posu[r] = pnew + (r - first_new);
    // ---- nothing to evict: identity outputs, running sum += appended rows ---
    if (a.kept_out)
      for (int i = (int)rank * kThreads + tid; i < a.N; i += C * kThreads)
        a.kept_out[(size_t)u * a.N + i] = i < n ? i : -1;
    if (DECODE && a.evicted_out && rank == 0 && tid == 0) a.evicted_out[u] = -1;
    if (a.mu_running && a.B > 0 && tchunks > 0) {
      const uint16_t* nb = srange(first_new, a.B);  // the new rows lie on one side
      sum_rows<Ring, kPackedSum>(tchunk0, tchunks, tp, a.B, [&](int i) { return nb + (size_t)i * d; },
               [](int) { return 1.f; }, S, ring);
      if (tid < tchunks * 8) {
        const int c = tchunk0 * 8 + tid;
        double* sp = a.running_sum + (size_t)u * d + c;
        *sp = *sp + (double)S.acc_hi[c] + (double)S.acc_lo[c];
      }
    }
    return;
  }

  // block eviction without attention weights: the score pass counts the
  // keys' top byte for the select's first radix pass as it writes them
  const bool hist_pre = !DECODE && !score_only && a.weights == nullptr;
  if (hist_pre) {
    S.hist[0][tid] = 0;
    S.hist[1][tid] = 0;  // the select's second pass counts into it without zeroing
    __syncthreads();
  }
  // ---- 1. mean ---------------------------------------------------------
  const int rows_per = (n + C - 1) / C;
  const int r0 = min(n, (int)rank * rows_per), r1 = min(n, r0 + rows_per);
  const int lpr = a.lpr;
  if (VAR != 2) {
    // running mean: S plus the appended rows (none for score-only calls)
    const bool run = a.mu_running;
    int p0, p1;
    if (run) {  // the appended rows, spread over the cluster
      const int per = (a.B + C - 1) / C;
      p0 = min(n, first_new + (int)rank * per);
      p1 = min(n, p0 + per);
    } else {
      p0 = r0;
      p1 = r1;
    }
    const int cnt = max(0, p1 - p0);
    // the running sum is loaded before the row sum, whose latency hides it
    const double rs_own = run && tid < d ? a.running_sum[(size_t)u * d + tid] : 0.0;
    const uint16_t* pb = srange(p0, cnt);  // nullptr only where the range straddles
    bool summed = false;
    if constexpr (SCORE) {
      if (bulk) {  // score-only rows are never staged: one contiguous range
        sum_rows_bulk(br, pb, cnt, d, lpr, S, a.status);
        summed = true;
      }
    }
    if (!summed)
      sum_rows<Ring, kPackedSum>(0, d8, lpr, cnt,
                     [&](int i) -> const uint16_t* {
                       if constexpr (FUSED) return pb ? pb + (size_t)i * d : srow(p0 + i);
                       else return pb + (size_t)i * d;
                     },
                     [](int) { return 1.f; }, S, ring);
    if (C > 1) cluster_sync(); else __syncthreads();
    if (tid < d) {
      ff t{0.f, 0.f};
      for (int rr = 0; rr < C; ++rr) {
        ff p;
        if (C > 1) {
          p.hi = ld_cluster_f32(mapa(smem_addr(&S.acc_hi[tid]), rr));
          p.lo = ld_cluster_f32(mapa(smem_addr(&S.acc_lo[tid]), rr));
        } else {
          p = ff{S.acc_hi[tid], S.acc_lo[tid]};
        }
        t = ff_add(t, p);
      }
      double sum = (double)t.hi + (double)t.lo;
      if (run) {
        sum += rs_own;
        S.snew[tid] = sum;  // phase 5 starts from it
      }
      const double m = sum / (double)n;
      const float mh = (float)m;
      S.mu[tid] = mh;
      S.mulo[lo_index(tid, d8)] = (float)(m - (double)mh);
    }
    __syncthreads();
    if (VAR == 1) {
      const float m = tid < d ? S.mu[tid] : 0.f;
      const float nrm2 = block_sum_f32(m * m, S.fsh);
      if (tid == 0) {
        S.mu_zero = !(nrm2 > 0.f);
        S.inv_mnorm = nrm2 > 0.f ? 1.f / sqrtf(nrm2) : 0.f;
      }
      __syncthreads();
    }
  }
  // vd_score reads peer partial sums above and nothing after: release that
  // barrier phase now, wait for it before exiting (peers may still be reading)
  const bool score_split = C > 1 && score_only && VAR != 2;
  if (score_split) cluster_arrive();

  // ---- 2. scores -------------------------------------------------------
  // The rows are visited from the last to the first: the mean's row sum
  // (recomputed mean) and the appended rows (running mean) were read in
  // ascending order just before, so the first rows scored are the ones most
  // recently brought into L2, and the compaction, which walks up from the
  // first evicted slot, starts with the rows scored last.
  // sigma of the L2 scores (host-checked; compiled into the L2 kernels only)
  const bool disp = VAR == 0 && a.disp_out != nullptr;
  {
    const int ci = lane & (lpr - 1);
    const bool active = ci < d8;
    float m8[8];  // this lane's columns of the mean (fp32 part)
#pragma unroll
    for (int k = 0; k < 8; ++k) m8[k] = (VAR != 2 && active) ? S.mu[ci * 8 + k] : 0.f;
    // ... and of its remainder, read in pairs at each use (see chunk_sq)
    const uint32_t lo_addr = smem_addr(S.mulo) + (uint32_t)(active ? ci : 0) * 8u;
    auto lo_pair = [&](int k, float& l0, float& l1) {
      const unsigned long long p = ld_shared_b64(lo_addr + (uint32_t)(k * d8 * 8));
      l0 = __uint_as_float((uint32_t)p);
      l1 = __uint_as_float((uint32_t)(p >> 32));
      if (!active) l0 = l1 = 0.f;
    };
    const bool mu_zero = VAR == 1 && S.mu_zero;
    const float inv_mnorm = VAR == 1 ? S.inv_mnorm : 0.f;
    const bool weighted = !DECODE && a.weights != nullptr;
    float ds_hi = 0.f, ds_lo = 0.f, dq_hi = 0.f, dq_lo = 0.f;  // dispersion sums
    unsigned long long best = ~0ull;  // (key, tie-break) of this thread's minimum
    unsigned best_key = 0xffffffffu;   // hole-fill: key of this thread's minimum
    int best_slot = -1;
    float* sc_out = a.scores_out ? a.scores_out + (size_t)u * a.capacity : nullptr;
    // everything a row's score feeds: the output, sigma, its key
    auto finish_row = [&](int item, float s) {
      const int r = r0 + item;
      if (sc_out && !weighted) sc_out[r] = s;
      if (VAR == 0 && disp) {  // sum s and s^2 (the square split exactly by an FMA)
        ff_accumulate(ds_hi, ds_lo, s);
        const float q2 = s * s;
        ff_accumulate(dq_hi, dq_lo, q2);
        dq_lo += fmaf(s, s, -q2);
      }
      if (!score_only) {
        bool bad;
        const uint32_t key = score_key(s, bad);
        if (bad) record_status(a.status, kStNonfinite);
        if (DECODE) {
          // lowest score first; among equal scores the latest token
          // (highest slot, or highest position in the hole-fill layout,
          // whose positions are read only to settle an exact tie)
          if constexpr (!HF) {
            const unsigned long long pk = ((unsigned long long)key << 32) |
                                          (unsigned long long)(0xffffffffu - (unsigned)r);
            best = pk < best ? pk : best;
          } else if (key < best_key || (key == best_key && pos_of(r) > pos_of(best_slot))) {
            best_key = key;
            best_slot = r;
          }
        } else {
          keys[item] = key;
          if (hist_pre) atomicAdd(&S.hist[0][key >> 24], 1u);  // the select's first pass
        }
      }
    };
    bool fast = false;
    // rows per batch: 4 in the ordered decode kernels, whose other live state
    // (the running arg-min, the staged-row pointers) leaves no room for 8
    // rows' partial sums within 64 registers without spilling
    constexpr int kScoreBatch = DECODE && !HF ? 4 : 8;
    if constexpr (VAR != 1) {  // head dims 64, 128, 256: one 16-byte chunk per lane
      // cache rows [r0, c_end), then (fused append) staging rows [c_end, r1)
      const int c_end = min(r1, max(r0, first_stage));
      auto run = [&](auto lanes) {
        constexpr int LPR = decltype(lanes)::value;
        if constexpr (SCORE) {
          if (bulk) {
            score_rows_bulk<VAR, LPR>(br, sb + (size_t)r0 * d, r1 - r0, S.mu, S.mulo, finish_row,
                                      a.status);
            return;
          }
        }
        if (r1 > c_end)
          score_rows_fast<VAR, LPR, Ring, kScoreBatch>(
              snu + (size_t)(c_end - first_stage) * d, r1 - c_end, S.mu, S.mulo,
              [&](int j, float s) { finish_row(j + (c_end - r0), s); }, ring);
        if (c_end > r0)
          score_rows_fast<VAR, LPR, Ring, kScoreBatch>(sb + (size_t)r0 * d, c_end - r0, S.mu,
                                                       S.mulo, finish_row, ring);
      };
      fast = true;
      if (d == 128) run(std::integral_constant<int, 16>{});
      else if (d == 256) run(std::integral_constant<int, 32>{});
      else if (d == 64) run(std::integral_constant<int, 8>{});
      else fast = false;
    }
    const uint16_t* rb = srange(r0, r1 - r0);  // nullptr only where the range straddles
    const int nr = r1 - r0;  // rows visited last to first, as in score_rows_fast
    if (!fast) stream_rows<Ring>(
        0, d8, lpr, nr,
        [&](int i) -> const uint16_t* {
          if constexpr (FUSED) return rb ? rb + (size_t)(nr - 1 - i) * d : srow(r1 - 1 - i);
          else return rb + (size_t)(nr - 1 - i) * d;
        },
        [&](int item, bool in, const uint4& q) {
          float x[8];
          unpack8(q, x);
          float s;
          if (VAR == 0) {
            float acc = 0.f;
#pragma unroll
            for (int k = 0; k < 8; k += 2) {
              float l0, l1;
              lo_pair(k >> 1, l0, l1);
              const float dv0 = (x[k] - m8[k]) - l0;
              const float dv1 = (x[k + 1] - m8[k + 1]) - l1;
              acc = fmaf(dv0, dv0, acc);
              acc = fmaf(dv1, dv1, acc);
            }
            for (int off = 1; off < lpr; off <<= 1) acc += __shfl_xor_sync(kFull, acc, off);
            s = sqrtf(acc);
          } else if (VAR == 2) {
            float acc = 0.f;
#pragma unroll
            for (int k = 0; k < 8; ++k) acc = fmaf(x[k], x[k], acc);
            for (int off = 1; off < lpr; off <<= 1) acc += __shfl_xor_sync(kFull, acc, off);
            s = sqrtf(acc);
          } else {
            // 1 - cos(v, m) = |w|^2 / (2 |v|^2) with w = v - (|v| / |m|) m:
            // each w_c is one fused multiply-add of the row and the
            // double-float mean, rounded relative to w_c itself, so the
            // score's error stays relative to the score even where v and m
            // are nearly parallel (1 - cos computed directly would cancel)
            float nv = 0.f;
#pragma unroll
            for (int k = 0; k < 8; ++k) nv = fmaf(x[k], x[k], nv);
            for (int off = 1; off < lpr; off <<= 1) nv += __shfl_xor_sync(kFull, nv, off);
            const float lam = sqrtf(nv) * inv_mnorm;
            float acc = 0.f;
#pragma unroll
            for (int k = 0; k < 8; k += 2) {
              float l0, l1;
              lo_pair(k >> 1, l0, l1);
              const float w0 = fmaf(-lam, l0, fmaf(-lam, m8[k], x[k]));
              const float w1 = fmaf(-lam, l1, fmaf(-lam, m8[k + 1], x[k + 1]));
              acc = fmaf(w0, w0, acc);
              acc = fmaf(w1, w1, acc);
            }
            for (int off = 1; off < lpr; off <<= 1) acc += __shfl_xor_sync(kFull, acc, off);
            s = (nv > 0.f && !mu_zero) ? (0.5f * acc) / nv : 1.f;
          }
          if (in && ci == 0) finish_row(nr - 1 - item, s);
        },
        ring);
    if constexpr (VAR == 0) {
      if (disp) disp_reduce_cta(ds_hi, ds_lo, dq_hi, dq_lo, S.dsc, S);
    }
    if (score_only) {
      if (score_split) cluster_wait();
      if constexpr (VAR == 0) {
        if (disp) {
          if (C > 1) cluster_sync();
          if (rank == 0 && tid == 0) a.disp_out[u] = disp_finish(S, C, n);
          if (C > 1) cluster_sync();  // peers stay until rank 0 has read them
        }
      }
      return;
    }
    if (DECODE) {
      if constexpr (HF) {
        if (best_slot >= 0)
          best = ((unsigned long long)best_key << 32) |
                 (unsigned long long)(0xffffffffu - (unsigned)pos_of(best_slot));
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
          const unsigned long long o = __shfl_xor_sync(kFull, best, off);
          const int os = __shfl_xor_sync(kFull, best_slot, off);
          if (o < best) {
            best = o;
            best_slot = os;
          }
        }
      } else {
        best = warp_min_u64(best);
      }
      if (lane == 0) {
        S.wbest[warp] = best;
        if (HF) S.wslot[warp] = best_slot;
      }
      __syncthreads();
      if (tid == 0) {
        unsigned long long b = ~0ull;
        int bs = 0;
        for (int w = 0; w < kWarps; ++w)
          if (S.wbest[w] < b) {
            b = S.wbest[w];
            if (HF) bs = S.wslot[w];
          }
        S.best = b;
        S.best_slot = bs;
      }
    }
  }

  // ---- 3./4. select and kept list --------------------------------------
  int e_first;
  if (DECODE) {
    if (C > 1) cluster_sync(); else __syncthreads();
    unsigned long long b = ~0ull;
    int bs = 0;
    for (int rr = 0; rr < C; ++rr) {
      const unsigned long long o =
          C > 1 ? ld_cluster_u64(mapa(smem_addr(&S.best), rr)) : S.best;
      if (o < b) {
        b = o;
        if (HF) bs = C > 1 ? (int)ld_cluster_u32(mapa(smem_addr(&S.best_slot), rr)) : S.best_slot;
      }
    }
    if (C > 1) cluster_arrive();  // last peer access of this CTA; wait before exit
    // ordered layout: the tie-break field is the slot itself
    e_first = HF ? bs : (int)(0xffffffffu - (unsigned)(b & 0xffffffffull));
  } else {
    __syncthreads();  // own keys complete
    const int R = r1 - r0;
    if (a.weights) {
      // attention-weighted score (the FastCAOTE form of App. A):
      // s'_j = a_j / (1 - a_j) * s_j, for weights a_j in [0, 1)
      const float* wu = a.weights + (size_t)u * a.capacity;
      float* sc_out = a.scores_out ? a.scores_out + (size_t)u * a.capacity : nullptr;
      for (int j = tid; j < R; j += kThreads) {
        const float w = wu[r0 + j];
        const float f = (w >= 0.f && w < 1.f) ? w / (1.f - w) : __int_as_float(0x7fc00000);
        const float sw = key_score(keys[j]) * f;
        bool bad;
        keys[j] = score_key(sw, bad);
        if (bad) record_status(a.status, kStNonfinite);
        if (sc_out) sc_out[r0 + j] = sw;
      }
      __syncthreads();
    }
    const Selection sel = cluster_radix_select(
        [&](int j, bool& ok) {
          ok = true;
          return keys[j];
        },
        R, Nb, C, S, hist_pre);
    if constexpr (VAR == 0) {
      if (disp && rank == 0 && tid == 0) a.disp_out[u] = disp_finish(S, C, n);
    }
    // hole-fill layout: the surviving ties are the lowest positions, found
    // by a second select over the complemented positions of the tied rows
    uint32_t t2 = 0u;
    if (HF && sel.cnt_eq > sel.keep_eq) {
      const Selection s2 = cluster_radix_select(
          [&](int j, bool& ok) {
            ok = keys[j] == sel.t;
            return ~(uint32_t)pos_of(r0 + j);
          },
          R, sel.keep_eq, C, S);
      t2 = s2.t;
    }
    cluster_build_perm<HF>(keys, r0, R, Nb, n, sel, t2,
                           [&](int j) { return ~(uint32_t)pos_of(r0 + j); }, C, rank, perm,
                           a.status, S);
    e_first = perm[Nb];
  }

  // ---- outputs -----------------------------------------------------------
  if (a.kept_out && !hf) {
    int32_t* ko = a.kept_out + (size_t)u * a.N;
    for (int i = (int)rank * kThreads + tid; i < a.N; i += C * kThreads) {
      int val = -1;
      if (i < Nb) val = DECODE ? (i < e_first ? i : i + 1) : (int)perm[i];
      ko[i] = val;
    }
  }
  if (DECODE && a.evicted_out && rank == 0 && tid == 0) a.evicted_out[u] = e_first;

  // ---- 5. running sum: S += appended rows - evicted rows (own columns of
  // the scored tensor).  The appended rows were already summed for the mean
  // (all but Norm: S plus them is in S.snew); only the evicted rows are read
  // again.  Norm loads S before the row sum, whose latency hides it.
  // Hole-fill block events retire the evicted rows in the move stream
  // (move_rows_retire) instead: here Norm only adds the appended rows, into
  // S.snew, the base the move stream subtracts from.
  constexpr bool kRetire = HF && !DECODE;
  if (a.mu_running && tchunks > 0 && !(kRetire && VAR != 2)) {
    const int B = VAR != 2 ? 0 : a.B;
    const int ne = kRetire ? 0 : n - Nb;
    double base = 0.0;
    if (tid < tchunks * 8) {
      const int c = tchunk0 * 8 + tid;
      base = VAR != 2 ? S.snew[c] : a.running_sum[(size_t)u * d + c] + 0.0;
    }
    sum_rows<Ring, kPackedSum>(tchunk0, tchunks, tp, B + ne,
             [&](int i) {
               const int r =
                   i < B ? first_new + i : (DECODE ? e_first : (int)perm[Nb + (i - B)]);
               if ((unsigned)r < (unsigned)n) return srow(r);
               record_status(a.status, kStInternal);  // self-check: never expected
               return srow(0);
             },
             [&](int i) { return i < B ? 1.f : -1.f; }, S, ring);
    if (tid < tchunks * 8) {
      const int c = tchunk0 * 8 + tid;
      const double v = base + (double)S.acc_hi[c] + (double)S.acc_lo[c];
      if (kRetire) S.snew[c] = v;
      else a.running_sum[(size_t)u * d + c] = v;
    }
  }

  // ---- 6. in-place compaction of this CTA's column slice ---------------
  if constexpr (!HF) {
    // fused append: kept new rows below the budget are written too, read
    // from the staging rows in the same stream (their slots, the suffix of
    // the kept list, come last)
    const int r_begin = min(e_first, first_stage);
    compact_slice<Ring, FUSED>(kb, vb, d, chunk0, cps, r_begin, Nb, n, DECODE ? nullptr : perm,
                               a.status, ring, knu, vnu, first_stage);
  } else {
    // hole-fill: the kept rows at or above N move into the evicted slots
    // below N, in ascending order (movers: the tail of the kept list; holes:
    // the head of the evicted list)
    int h;
    if (DECODE) {
      h = e_first < Nb ? 1 : 0;
    } else {
      if (tid == 0) {
        int lo = 0, hi = n - Nb;
        while (lo < hi) {
          const int mid = (lo + hi) >> 1;
          if ((int)perm[Nb + mid] < Nb) lo = mid + 1; else hi = mid;
        }
        S.holes = lo;
      }
      __syncthreads();
      h = S.holes;
    }
    auto src = [&](int i) { return DECODE ? n - 1 : (int)perm[Nb - h + i]; };
    auto dst = [&](int i) { return DECODE ? e_first : (int)perm[Nb + i]; };
    if (fused && Nb > first_stage) {
      // fused append: new rows below the budget stay in their slots (the
      // evicted ones among them are refilled just below)
      copy_new_rows(kb, vb, knu, vnu, d, chunk0, cps, first_stage, Nb - first_stage);
      __syncthreads();
    }
    if constexpr (DECODE) {
      move_rows(kb, vb, d, chunk0, cps, h, n, src, dst, a.status, knu, vnu, first_stage);
    } else {
      // the scored tensor's chunks of [K | V]: K's [0, d8) or V's [d8, 2 d8)
      const int sc_lo = a.score_k ? 0 : d8;
      move_rows_retire<Ring, kPackedSum>(
          kb, vb, d, chunk0, cps, h, n - Nb, n, src, dst, a.status, knu, vnu, first_stage, ring,
          a.mu_running && tchunks > 0, sc_lo, sc_lo + d8, tchunk0, tchunks, smem_addr(S.snew),
          a.running_sum + (size_t)u * d);
    }
    if (rank == 0) {
      for (int r = max(first_new, 0) + tid; r < Nb; r += kThreads) posu[r] = pnew + (r - first_new);
      int32_t* ko = a.kept_out ? a.kept_out + (size_t)u * a.N : nullptr;
      if (ko)
        for (int r = tid; r < a.N; r += kThreads) ko[r] = r < Nb ? r : -1;
      __syncthreads();
      for (int i = tid; i < h; i += kThreads) {
        const int sr = src(i), dr = dst(i);
        if ((unsigned)sr >= (unsigned)n || (unsigned)dr >= (unsigned)n) continue;  // recorded
        posu[dr] = pos_of(sr);
        if (ko) ko[dr] = sr;
      }
    }
  }

  if (DECODE && C > 1) cluster_wait();
}

// One unit per cluster of C CTAs (evict_unit).  Split launches (the host's
// split_plan) run the units in two launches on one stream, the second a
// programmatic dependent launch whose CTAs take the slots the first leaves
// free.  So every kernel lets its dependents be scheduled at once.  The two
// parts touch disjoint units, so the second reads nothing the first writes;
// it waits for the first only before it ends (griddepcontrol.wait, a no-op
// in a normal launch), so that work queued after it on the stream also
// follows the first.
template <int VAR, bool DECODE, bool HF, bool FUSED, bool SCORE = false>
__global__ void __launch_bounds__(kThreads, SCORE    ? VD_SCORE_MIN_CTAS
                                            : DECODE ? VD_DECODE_MIN_CTAS
                                            : HF     ? VD_HF_BLOCK_MIN_CTAS
                                                     : VD_BLOCK_MIN_CTAS)
    evict_kernel(const EvictArgs a) {
  grid_launch_dependents();
  evict_unit<VAR, DECODE, HF, FUSED, SCORE>(a);
  grid_dependency_wait();
}

}  // namespace vd
