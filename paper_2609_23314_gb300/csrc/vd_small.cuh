// vd_small.cuh -- pi_N of Sec. 2.1 Eq. (eviction) for short caches, where the
// fused kernel's machinery (multi-pass radix select, streaming rings, the
// separate length update) costs more than the work itself.
//
// One CTA per (sequence, layer, KV head) unit; the CTAs of one sequence form
// one thread-block cluster (units_per_seq <= 16), so that after a cluster
// barrier the sequence's length can be written by the kernel itself: one
// launch per event.  The unit's n rows of K and V are copied into shared
// memory once; everything after that reads shared memory:
//
//   1. mean    double-float column sums (running mode: the caller's fp64 sum
//              S plus the appended rows), kept as an fp32 part and remainder
//   2. score   L2 ((v - hi) - lo)^2, Dir |w|^2 / (2 |v|^2) with
//              w = v - (|v|/|m|) m, Norm |v|^2, as in the fused kernel
//   3. select  rank_j = #{i : key_i > key_j} + #{i < j : key_i == key_j};
//              row j survives iff rank_j < N (Eq. eviction, ties to the
//              lower slot), O(n^2 / 256) comparisons per thread
//   4. list    kept slots ascending (a block prefix sum), then the evicted
//   5. sum     running mode: S + sum(appended rows) - sum(evicted rows)
//   6. move    rows [first moved, N) written from the shared-memory copy,
//              so the in-place gather has no read-after-write hazard
//
// Same validation, outputs and status codes as the fused kernel; no
// hole-fill layout, attention weights, sigma or key-side rule (those calls
// take the fused kernel).
#pragma once

#include <cstdint>

#include "vd_evict.cuh"

namespace vd {

constexpr int kSmallMaxRows = 1024;

struct SmallSmem {
  float mu[256];
  float mulo[256];     // mean = mu + mulo (natural column order)
  float part_hi[256];  // column-sum partials, [part][column]
  float part_lo[256];
  int scan[kWarps];
  float fsh[kWarps];
  float inv_mnorm;
  int mu_zero;
  int e_first;
};

struct SmallLayout {
  size_t v, k, keys, perm, total;
};

// rows: the capacity (every row the unit may hold); d: head_dim
__host__ __device__ inline SmallLayout small_layout(int capacity, int d) {
  SmallLayout l;
  l.v = (sizeof(SmallSmem) + 127) & ~(size_t)127;
  l.k = l.v + align16((size_t)capacity * d * 2);
  l.keys = l.k + align16((size_t)capacity * d * 2);
  l.perm = l.keys + align16((size_t)capacity * 4);
  l.total = l.perm + align16((size_t)capacity * 2);
  return l;
}

// acc (S.mu as hi, S.mulo as lo, natural columns) <- sum over list items
// [0, count) of sign(i) * row(i), exact per element (TwoSum); P = 256 / d
// threads per column, each summing items p, p + P, ...; the P partials are
// added in a fixed order.  Returns through hi/lo of threads t < d.
template <class RowOf, class SignOf>
__device__ __forceinline__ ff small_column_sum(int d, int count, RowOf row_of, SignOf sign_of,
                                               SmallSmem& S) {
  const int tid = threadIdx.x;
  const int P = kThreads / d;
  const int col = tid % d, part = tid / d;
  float hi = 0.f, lo = 0.f;
  if (part < P)
    for (int i = part; i < count; i += P)
      ff_accumulate(hi, lo, sign_of(i) * __uint_as_float((uint32_t)row_of(i)[col] << 16));
  if (part < P) {
    S.part_hi[part * d + col] = hi;
    S.part_lo[part * d + col] = lo;
  }
  __syncthreads();
  ff t{0.f, 0.f};
  if (tid < d)
    for (int p = 0; p < P; ++p) t = ff_add(t, ff{S.part_hi[p * d + tid], S.part_lo[p * d + tid]});
  __syncthreads();
  return t;
}

// The kernel's parameters: the fused kernel's, plus the number of units.
struct SmallArgs {
  EvictArgs e;
  int32_t n_units;  // n_seq * units_per_seq: the grid's CTAs
};

// VAR: 0 L2, 1 Dir, 2 Norm.  DECODE: the decode entry points (n <= N + 1);
// the selection is the same.  FUSED: rows at or above len come from the
// caller's staging buffers (the append of Eq. block_processing).
// a.cluster = units per sequence (the cluster size), a.capacity <= kSmallMaxRows.
template <int VAR, bool DECODE, bool FUSED>
__global__ void __launch_bounds__(kThreads, 1) small_evict_kernel(const SmallArgs sa) {
  const EvictArgs& a = sa.e;
  // launched as a programmatic dependent: wait for the previous kernel on the
  // stream before reading anything, and let the next one be scheduled
  grid_dependency_wait();
  grid_launch_dependents();
  extern __shared__ __align__(16) unsigned char smem_raw[];
  SmallSmem& S = *reinterpret_cast<SmallSmem*>(smem_raw);
  const int d = a.d, d8 = d >> 3, cap = a.capacity;
  const SmallLayout L = small_layout(cap, d);
  uint16_t* Vs = reinterpret_cast<uint16_t*>(smem_raw + L.v);
  uint16_t* Ks = reinterpret_cast<uint16_t*>(smem_raw + L.k);
  uint32_t* keys = reinterpret_cast<uint32_t*>(smem_raw + L.keys);
  uint16_t* perm = reinterpret_cast<uint16_t*>(smem_raw + L.perm);
  const int tid = threadIdx.x, lane = tid & 31;
  const int C = a.cluster;
  const unsigned rank = C > 1 ? cluster_ctarank() : 0u;
  const int u = (int)blockIdx.x;
  // a CTA past the last unit (impossible for the host's grid) reads and
  // writes nothing but still reaches the cluster barrier
  const bool unit_ok = u < sa.n_units;
  const int seq = unit_ok ? u / a.units_per_seq : 0;
  const int len0 = unit_ok ? a.len[seq] : -1;
  const int n = len0 + (FUSED ? a.B : 0);
  const int Nb = unit_ok ? (a.N_dev ? a.N_dev[seq] : a.N) : 0;
  const size_t ubase = (size_t)u * cap * d;
  uint16_t* kb = a.k + ubase;
  uint16_t* vb = a.v + ubase;
  const uint16_t* knu = FUSED ? a.k_new + (size_t)u * a.B * d : nullptr;
  const uint16_t* vnu = FUSED ? a.v_new + (size_t)u * a.B * d : nullptr;

  // ---- validation: the same per-sequence checks as the fused kernel -------
  bool ok = unit_ok;
  if (!unit_ok) {
    if (tid == 0) record_status(a.status, kStInternal);
  } else if (len0 < 0 || n > cap || (a.mu_running && a.B > n)) {
    if (rank == 0 && tid == 0 && u % a.units_per_seq == 0) record_status(a.status, kStDeviceLen);
    ok = false;
  } else if (Nb < 1 || Nb > a.N || (DECODE && n > Nb + 1)) {
    if (rank == 0 && tid == 0 && u % a.units_per_seq == 0)
      record_status(a.status, kStDeviceBudget);
    ok = false;
  }
  const bool evict = ok && n > Nb;
  const int first_new = n - a.B;

  if (ok) {
    // ---- the unit's rows into shared memory (cache rows below len0, the
    // staging rows above it when fused) ---------------------------------
    const uint32_t vs_a = smem_addr(Vs), ks_a = smem_addr(Ks);
    for (int c = tid; c < n * d8; c += kThreads) {
      const int r = c / d8, col = (c - r * d8) * 8;
      const bool staged = FUSED && r >= len0;
      const size_t go = (size_t)(staged ? r - len0 : r) * d + col;
      cp_async16(vs_a + (uint32_t)(r * d + col) * 2u, (staged ? vnu : vb) + go);
      cp_async16(ks_a + (uint32_t)(r * d + col) * 2u, (staged ? knu : kb) + go);
    }
    cp_async_commit();
    cp_async_wait<0>();
    __syncthreads();
    auto vrow = [&](int r) { return Vs + (size_t)r * d; };
    double* rsu = a.mu_running ? a.running_sum + (size_t)u * d : nullptr;

    if (!evict) {
      // ---- nothing to evict: append (fused), running sum += appended rows --
      if (FUSED)
        for (int c = tid; c < a.B * d8; c += kThreads) {
          const int r = len0 + c / d8, col = (c % d8) * 8;
          st16(kb + (size_t)r * d + col, ld_shared16(ks_a + (uint32_t)(r * d + col) * 2u));
          st16(vb + (size_t)r * d + col, ld_shared16(vs_a + (uint32_t)(r * d + col) * 2u));
        }
      if (a.kept_out)
        for (int i = tid; i < a.N; i += kThreads) a.kept_out[(size_t)u * a.N + i] = i < n ? i : -1;
      if (DECODE && a.evicted_out && tid == 0) a.evicted_out[u] = -1;
      if (rsu && a.B > 0) {
        const ff t = small_column_sum(d, a.B, [&](int i) { return vrow(first_new + i); },
                                      [](int) { return 1.f; }, S);
        if (tid < d) rsu[tid] = rsu[tid] + (double)t.hi + (double)t.lo;
      }
    } else {
      // ---- 1. mean ----------------------------------------------------
      double s_app = 0.0;  // running mode: the caller's sum plus the appended rows
      if (VAR != 2 || rsu) {
        const bool run = rsu != nullptr;
        const int cnt = run ? a.B : n;
        const int r0 = run ? first_new : 0;
        const ff t = small_column_sum(d, cnt, [&](int i) { return vrow(r0 + i); },
                                      [](int) { return 1.f; }, S);
        if (tid < d) {
          double sum = (double)t.hi + (double)t.lo;
          if (run) sum += rsu[tid];
          s_app = sum;
          const double m = sum / (double)n;
          const float mh = (float)m;
          S.mu[tid] = mh;
          S.mulo[tid] = (float)(m - (double)mh);
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
      // ---- 2. scores: lpr lanes per row, one 16-byte chunk each ----------
      const int lpr = a.lpr, ci = lane & (lpr - 1), g = tid / lpr, ng = kThreads / lpr;
      const bool active = ci < d8;
      float m8[8], l8[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        m8[k] = (VAR != 2 && active) ? S.mu[ci * 8 + k] : 0.f;
        l8[k] = (VAR != 2 && active) ? S.mulo[ci * 8 + k] : 0.f;
      }
      const bool mu_zero = VAR == 1 && S.mu_zero;
      const float inv_mnorm = VAR == 1 ? S.inv_mnorm : 0.f;
      float* sc_out = a.scores_out ? a.scores_out + (size_t)u * cap : nullptr;
      for (int base = 0; base < n; base += ng) {
        const int j = base + g;
        const bool in = j < n;
        uint4 q = make_uint4(0u, 0u, 0u, 0u);
        if (in && active) q = ld_shared16(vs_a + (uint32_t)(j * d + ci * 8) * 2u);
        float x[8];
        unpack8(q, x);
        float sc;
        if (VAR == 0) {
          float acc = 0.f;
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const float dv = (x[k] - m8[k]) - l8[k];
            acc = fmaf(dv, dv, acc);
          }
          for (int off = 1; off < lpr; off <<= 1) acc += __shfl_xor_sync(kFull, acc, off);
          sc = sqrtf(acc);
        } else if (VAR == 2) {
          float acc = 0.f;
#pragma unroll
          for (int k = 0; k < 8; ++k) acc = fmaf(x[k], x[k], acc);
          for (int off = 1; off < lpr; off <<= 1) acc += __shfl_xor_sync(kFull, acc, off);
          sc = sqrtf(acc);
        } else {
          float nv = 0.f;
#pragma unroll
          for (int k = 0; k < 8; ++k) nv = fmaf(x[k], x[k], nv);
          for (int off = 1; off < lpr; off <<= 1) nv += __shfl_xor_sync(kFull, nv, off);
          const float lam = sqrtf(nv) * inv_mnorm;
          float acc = 0.f;
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const float w = fmaf(-lam, l8[k], fmaf(-lam, m8[k], x[k]));
            acc = fmaf(w, w, acc);
          }
          for (int off = 1; off < lpr; off <<= 1) acc += __shfl_xor_sync(kFull, acc, off);
          sc = (nv > 0.f && !mu_zero) ? (0.5f * acc) / nv : 1.f;
        }
        if (in && ci == 0) {
          bool bad;
          keys[j] = score_key(sc, bad);
          if (bad) record_status(a.status, kStNonfinite);
          if (sc_out) sc_out[j] = sc;
        }
      }
      __syncthreads();

      // ---- 3./4. rank select and the kept list -------------------------
      // thread t owns rows [t * ch, t * ch + ch), so prefix sums follow slot
      // order (ties go to the lower slot)
      const int ch = (n + kThreads - 1) / kThreads;
      const int c0 = min(n, tid * ch), c1 = min(n, c0 + ch);
      unsigned keep_bits = 0u;  // ch <= kSmallMaxRows / kThreads = 4
      int nkeep = 0;
      for (int j = c0; j < c1; ++j) {
        const uint32_t kj = keys[j];
        int rank_j = 0;
        for (int i = 0; i < n; ++i) {
          const uint32_t ki = keys[i];
          rank_j += (ki > kj) | ((ki == kj) & (i < j));
        }
        if (rank_j < Nb) {
          keep_bits |= 1u << (j - c0);
          ++nkeep;
        }
      }
      int total_kept;
      int kp = block_exclusive_scan(nkeep, S.scan, total_kept);
      for (int j = c0; j < c1; ++j) {
        const bool keep = (keep_bits >> (j - c0)) & 1u;
        const int pos = keep ? kp : Nb + (j - kp);
        kp += keep;
        if ((unsigned)pos >= (unsigned)n || total_kept != Nb) {  // self-check
          record_status(a.status, kStInternal);
          continue;
        }
        perm[pos] = (uint16_t)j;
      }
      __syncthreads();
      // perm entries index the shared-memory copy: clamped to [0, n) so that
      // even after a failed self-check no access leaves it
      auto slot = [&](int i) { return min((int)perm[i], n - 1); };
      const int e_first = slot(Nb);  // the lowest evicted slot

      // ---- outputs --------------------------------------------------------
      if (a.kept_out)
        for (int i = tid; i < a.N; i += kThreads)
          a.kept_out[(size_t)u * a.N + i] = i < Nb ? slot(i) : -1;
      if (DECODE && a.evicted_out && tid == 0) a.evicted_out[u] = e_first;

      // ---- 5. running sum: (S + appended) - evicted rows ------------------
      if (rsu) {
        const ff t = small_column_sum(d, n - Nb, [&](int i) { return vrow(slot(Nb + i)); },
                                      [](int) { return -1.f; }, S);
        if (tid < d) rsu[tid] = s_app + (double)t.hi + (double)t.lo;
      }

      // ---- 6. compaction from the shared-memory copy ---------------------
      // (fused: the kept new rows below the budget are written too)
      const int r_begin = FUSED ? min(e_first, len0) : e_first;
      for (int c = tid; c < (Nb - r_begin) * d8; c += kThreads) {
        const int r = r_begin + c / d8, col = (c % d8) * 8;
        const int src = slot(r);
        st16(kb + (size_t)r * d + col, ld_shared16(ks_a + (uint32_t)(src * d + col) * 2u));
        st16(vb + (size_t)r * d + col, ld_shared16(vs_a + (uint32_t)(src * d + col) * 2u));
      }
    }
  }

  // ---- the sequence's new length, once every unit of it has read len -----
  if (C > 1) cluster_sync(); else __syncthreads();
  if (ok && (evict || FUSED) && rank == 0 && tid == 0 && u + C <= sa.n_units)
    a.len[seq] = evict ? Nb : n;
}

}  // namespace vd
