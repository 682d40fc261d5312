// vd_evict.cuh -- the fused ValueDiff eviction kernel for GB300 (sm_103a).
//
// One thread-block cluster of C CTAs owns one (sequence, layer, KV head) unit
// and runs pi_N of Sec. 2.1, Eq. (eviction) on it in a single launch:
//
//   1. mean   mean = (1/n) sum_i v_i (Sec. 3.2, Eq. vd).  Each CTA sums its
//             row range as double-float (hi + lo) fp32 pairs per column, and the cluster adds the C partials
//             in rank order through distributed shared memory, so every CTA
//             holds the same mean.  Running-sum mode adds only the appended
//             rows to the caller's fp64 sum S.
//   2. score  16-byte bf16 loads, d/8 lanes per row, warp-shuffle reduction
//             of the row's squared deviation (L2), its norm (Norm) or its
//             normalised difference (Dir, as 1/2 |v/|v| - mean/|mean||^2,
//             which equals 1 - cos without cancellation).
//   3. select block prompt processing (N+B -> N): every CTA receives all n
//             fp32 scores (as order-preserving uint32 keys) through DSMEM
//             and runs a 4-pass 8-bit radix select for the N-th largest key t;
//             keys > t are kept and the keys == t with the lowest slot
//             indices fill the rest.  Decode (N+1 -> N): a cluster arg-min
//             over (key, -index) finds the one evicted slot.
//   4. list   block prefix sums turn the keep flags into perm: the kept slots
//             ascending in perm[0, N), the evicted ones after them.
//   5. sum    running-sum mode: S += sum(appended rows) - sum(evicted rows),
//             for the V columns this CTA compacts, before it moves them.
//   6. move   K' = gather(K, perm), V' = gather(V, perm) in place.  CTA r
//             owns a disjoint column slice of [K | V] and walks the rows
//             r = first evicted .. N-1 upward in register tiles: a tile's
//             sources are all loaded before any of its destinations is
//             stored (one __syncthreads), and the next tile's loads are
//             issued before this tile's stores.  Because perm[r] >= r, a
//             store never hits a row a later tile still has to read.
//
// Nothing waits on a flag; the only cross-CTA synchronisation is the hardware
// cluster barrier, which every CTA of a cluster reaches the same number of
// times (every branch below depends only on per-sequence values that all
// CTAs of the cluster read identically).
#pragma once

#include <climits>
#include <cstdint>

#include "vd_device.cuh"

namespace vd {

struct EvictArgs {
  uint16_t* k;            // bf16 [U][capacity][d]
  uint16_t* v;            // bf16 [U][capacity][d]
  const int32_t* len;     // [n_seq]
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
  int32_t score_only;     // 1: vd_score (mean recomputed, no eviction)
  int32_t cluster;        // C, CTAs per unit
};

// Fixed part of the dynamic shared memory; the general (block) kernel appends
// keys[capacity] and perm[capacity].
struct Smem {
  float mu[256];
  float muhat[256];
  float acc_hi[256];  // this CTA's partial column sums (read by peer CTAs)
  float acc_lo[256];
  uint32_t hist[256];
  int scan[kWarps];
  float fsh[kWarps];
  unsigned long long best;  // decode: this CTA's (key, -index) minimum
  unsigned long long wbest[kWarps];
  int sel_digit, sel_above, sel_cnt;
  int e_first;
  int mu_zero;
};

// Sums rows of one unit's V, restricted to 16-byte column chunks
// [chunk0, chunk0 + nchunks), into acc_hi/acc_lo (which the caller zeroed).
// Item i contributes sign(i) * V[row(i)].  Lanes are grouped P per row
// (P = power of two >= nchunks); partials merge across the warp with TwoSum
// shuffles and across warps in a fixed order, so the result is deterministic.
template <class RowOf>
__device__ __forceinline__ void accumulate_rows(const uint16_t* __restrict__ vbase, int d,
                                                int chunk0, int nchunks, int P, int count,
                                                RowOf row_of, float* acc_hi, float* acc_lo) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int ci = lane & (P - 1);
  const bool active = ci < nchunks;
  const int ng = kThreads / P;
  const int g = tid / P;
  const int col = (chunk0 + ci) * 8;
  float s[8], c[8];
#pragma unroll
  for (int k = 0; k < 8; ++k) s[k] = c[k] = 0.f;
  constexpr int U = 4;
  for (int base = g; base < count; base += ng * U) {
    uint4 q[U];
    float sg[U];
#pragma unroll
    for (int i = 0; i < U; ++i) {
      const int it = base + i * ng;
      q[i] = make_uint4(0, 0, 0, 0);
      sg[i] = 0.f;
      if (active && it < count) {
        int row;
        float sign;
        row_of(it, row, sign);
        q[i] = ld_cg16(vbase + (size_t)row * d + col);
        sg[i] = sign;
      }
    }
#pragma unroll
    for (int i = 0; i < U; ++i) {
      if (sg[i] != 0.f) {
        float x[8];
        unpack8(q[i], x);
#pragma unroll
        for (int k = 0; k < 8; ++k) ff_accumulate(s[k], c[k], sg[i] * x[k]);
      }
    }
  }
  ff p[8];
#pragma unroll
  for (int k = 0; k < 8; ++k) p[k] = ff_add(ff{s[k], 0.f}, ff{0.f, c[k]});
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

__device__ __forceinline__ void zero_acc(Smem& S) {
  S.acc_hi[threadIdx.x] = 0.f;
  S.acc_lo[threadIdx.x] = 0.f;
  __syncthreads();
}

// Order-preserving key of a non-negative score; NaN ranks lowest.  `bad`
// reports a NaN or infinite score.
__device__ __forceinline__ uint32_t score_key(float s, bool& bad) {
  bad = !(s == s) || s == __int_as_float(0x7f800000);
  return (s == s) ? __float_as_uint(s) : 0u;
}

// Radix select over keys[0, n): t = the N-th largest key (1-based), keep_eq =
// how many keys equal to t survive, cnt_eq = how many keys equal t.
struct Selection {
  uint32_t t;
  int keep_eq;
  int cnt_eq;
};

__device__ __forceinline__ Selection radix_select(const uint32_t* keys, int n, int N, Smem& S) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint32_t prefix = 0, pmask = 0;
  int need = N, cnt = n;
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 24 - 8 * pass;
    S.hist[tid] = 0;
    __syncthreads();
    for (int base = 0; base < n; base += kThreads) {
      const int j = base + tid;
      const uint32_t key = j < n ? keys[j] : 0u;
      const bool match = j < n && (key & pmask) == prefix;
      const unsigned act = __ballot_sync(kFull, match);
      if (match) {
        const uint32_t dig = (key >> shift) & 255u;
        const unsigned peers = __match_any_sync(act, dig);
        if (lane == __ffs(peers) - 1) atomicAdd(&S.hist[dig], (uint32_t)__popc(peers));
      }
    }
    __syncthreads();
    if (warp == 0) {
      int c[8];
      int sum = 0;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        c[i] = (int)S.hist[255 - (lane * 8 + i)];
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
  }
  return {prefix, need, cnt};
}

// Keep flags -> perm (kept slots ascending, then evicted slots ascending) and
// the first evicted slot.  Threads own contiguous index chunks so the prefix
// sums follow slot order, which is what gives ties to the lower index.
__device__ __forceinline__ void build_perm(const uint32_t* keys, int n, int N, Selection sel, int* perm,
                           Smem& S) {
  const int tid = threadIdx.x;
  const int ch = (n + kThreads - 1) / kThreads;
  const int c0 = min(n, tid * ch), c1 = min(n, c0 + ch);
  const uint32_t t = sel.t;
  const bool scan_ties = sel.cnt_eq > sel.keep_eq;
  const int q = scan_ties ? sel.keep_eq : INT_MAX;
  int total;
  int tie_ex = 0;
  if (scan_ties) {
    int nt = 0;
    for (int j = c0; j < c1; ++j) nt += keys[j] == t;
    tie_ex = block_exclusive_scan(nt, S.scan, total);
  }
  int nk = 0;
  {
    int tr = tie_ex;
    for (int j = c0; j < c1; ++j) {
      const uint32_t key = keys[j];
      const bool eq = key == t;
      nk += (key > t) || (eq && tr < q);
      tr += eq;
    }
  }
  if (tid == 0) S.e_first = INT_MAX;
  const int kept_ex = block_exclusive_scan(nk, S.scan, total);
  int kp = kept_ex, tr = tie_ex, ef = INT_MAX;
  for (int j = c0; j < c1; ++j) {
    const uint32_t key = keys[j];
    const bool eq = key == t;
    const bool keep = (key > t) || (eq && tr < q);
    tr += eq;
    if (keep) {
      perm[kp++] = j;
    } else {
      perm[N + (j - kp)] = j;
      ef = min(ef, j);
    }
  }
  if (ef != INT_MAX) atomicMin(&S.e_first, ef);
  __syncthreads();
}

// In-place, order-preserving move of rows [r_begin, r_end) of the column
// slice [chunk0, chunk0 + cps) of the concatenated [K | V] row: row r takes
// source row perm[r] (or r + 1 when perm is null: the decode shift).
template <int UC>
__device__ __forceinline__ void compact_slice(uint16_t* kb, uint16_t* vb, int d, int chunk0,
                                              int cps, int r_begin, int r_end,
                                              const int* perm) {
  const int d8 = d >> 3;
  const int rs = kThreads / cps;
  const bool on = (int)threadIdx.x < rs * cps;
  const int my_ch = chunk0 + (int)threadIdx.x % cps;
  const int my_off = (int)threadIdx.x / cps;
  uint16_t* col = my_ch < d8 ? kb + my_ch * 8 : vb + (my_ch - d8) * 8;
  const int tile = rs * UC;
  const int ntiles = r_end > r_begin ? (r_end - r_begin + tile - 1) / tile : 0;
  uint4 A[UC], Bq[UC];

  auto load = [&](uint4 (&X)[UC], int t) {
#pragma unroll
    for (int i = 0; i < UC; ++i) {
      const int r = r_begin + t * tile + i * rs + my_off;
      if (on && r < r_end) {
        const int src = perm ? perm[r] : r + 1;
        X[i] = ld_cg16(col + (size_t)src * d);
      }
    }
  };
  auto store = [&](const uint4 (&X)[UC], int t) {
#pragma unroll
    for (int i = 0; i < UC; ++i) {
      const int r = r_begin + t * tile + i * rs + my_off;
      if (on && r < r_end) st16(col + (size_t)r * d, X[i]);
    }
  };

  if (ntiles > 0) load(A, 0);
  for (int t = 0; t < ntiles; t += 2) {
    __syncthreads();  // every source of tile t has been loaded
    if (t + 1 < ntiles) load(Bq, t + 1);
    store(A, t);
    if (t + 1 >= ntiles) break;
    __syncthreads();  // every source of tile t + 1 has been loaded
    if (t + 2 < ntiles) load(A, t + 2);
    store(Bq, t + 1);
  }
}

template <int VAR, bool DECODE>
__global__ void __launch_bounds__(kThreads, 4) evict_kernel(const EvictArgs a) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  Smem& S = *reinterpret_cast<Smem*>(smem_raw);
  uint32_t* keys = reinterpret_cast<uint32_t*>(smem_raw + sizeof(Smem));
  int* perm = reinterpret_cast<int*>(keys + a.capacity);

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int C = a.cluster;
  const unsigned rank = C > 1 ? cluster_ctarank() : 0u;
  const int u = C > 1 ? (int)cluster_id_x() : (int)blockIdx.x;
  const int d = a.d, d8 = d >> 3;
  const int seq = u / a.units_per_seq;
  const int n = a.len[seq];
  const int Nb = a.N_dev ? a.N_dev[seq] : a.N;
  const size_t ubase = (size_t)u * a.capacity * d;
  uint16_t* kb = a.k + ubase;
  uint16_t* vb = a.v + ubase;

  // ---- validation: uniform across the cluster (per-sequence values only) ---
  if (n < 0 || n > a.capacity || (a.mu_running && !a.score_only && a.B > n)) {
    if (rank == 0 && tid == 0) record_status(a.status, kStDeviceLen);
    return;
  }
  if (!a.score_only && (Nb < 1 || Nb > a.N)) {
    if (rank == 0 && tid == 0) record_status(a.status, kStDeviceBudget);
    return;
  }
  const bool evict = !a.score_only && n > Nb;
  if (DECODE && evict && n > Nb + 1) {
    if (rank == 0 && tid == 0) record_status(a.status, kStDeviceBudget);
    return;
  }
  if (a.score_only && n == 0) return;

  // column slice of [K | V] this CTA compacts and keeps the running sum of
  const int cps = (2 * d8) / C;
  const int chunk0 = (int)rank * cps;
  const int vchunk0 = max(chunk0, d8) - d8;
  const int vchunks = max(0, chunk0 + cps - max(chunk0, d8));
  int vp = 1;
  while (vp < vchunks) vp <<= 1;

  if (!evict && !a.score_only) {
    // ---- nothing to evict: identity outputs, running sum += appended rows ---
    if (a.kept_out)
      for (int i = (int)rank * kThreads + tid; i < a.N; i += C * kThreads)
        a.kept_out[(size_t)u * a.N + i] = i < n ? i : -1;
    if (DECODE && a.evicted_out && rank == 0 && tid == 0) a.evicted_out[u] = -1;
    if (a.mu_running && a.B > 0 && vchunks > 0) {
      zero_acc(S);
      const int first_new = n - a.B;
      accumulate_rows(vb, d, vchunk0, vchunks, vp, a.B,
                      [&](int i, int& row, float& sign) { row = first_new + i; sign = 1.f; },
                      S.acc_hi, S.acc_lo);
      if (tid < vchunks * 8) {
        const int c = vchunk0 * 8 + tid;
        double* sp = a.running_sum + (size_t)u * d + c;
        *sp = *sp + (double)S.acc_hi[c] + (double)S.acc_lo[c];
      }
    }
    return;
  }

  // ---- 1. mean ---------------------------------------------------------
  const int rows_per = (n + C - 1) / C;
  const int r0 = min(n, (int)rank * rows_per), r1 = min(n, r0 + rows_per);
  const int lpr = a.lpr;
  if (VAR != 2) {
    const bool run = a.mu_running && !a.score_only;
    const int p0 = run ? max(r0, n - a.B) : r0;
    zero_acc(S);
    accumulate_rows(vb, d, 0, d8, lpr, max(0, r1 - p0),
                    [&](int i, int& row, float& sign) { row = p0 + i; sign = 1.f; },
                    S.acc_hi, S.acc_lo);
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
      if (run) sum += a.running_sum[(size_t)u * d + tid];
      S.mu[tid] = (float)(sum / (double)n);
    }
    __syncthreads();
    if (VAR == 1) {
      const float m = tid < d ? S.mu[tid] : 0.f;
      const float nrm2 = block_sum_f32(m * m, S.fsh);
      if (tid < d) S.muhat[tid] = nrm2 > 0.f ? m / sqrtf(nrm2) : 0.f;
      if (tid == 0) S.mu_zero = !(nrm2 > 0.f);
      __syncthreads();
    }
  }
  // score-only and decode read peer shared memory below or above; release
  // the cluster barrier phase once the last peer access is done
  const bool split_exit = C > 1 && (a.score_only || DECODE) && VAR != 2;

  // ---- 2. scores -------------------------------------------------------
  {
    const int ci = lane & (lpr - 1);
    const bool active = ci < d8;
    const int ng = kThreads / lpr;
    const int g = tid / lpr;
    float m8[8], h8[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      m8[k] = (VAR == 0 && active) ? S.mu[ci * 8 + k] : 0.f;
      h8[k] = (VAR == 1 && active) ? S.muhat[ci * 8 + k] : 0.f;
    }
    const bool mu_zero = VAR == 1 && S.mu_zero;
    const uint32_t keys_addr = smem_addr(keys);
    unsigned long long best = ~0ull;
    float* sc_out = a.scores_out ? a.scores_out + (size_t)u * a.capacity : nullptr;
    constexpr int U = 4;
    // trip count uniform over the CTA: the row reductions below shuffle
    for (int b0 = r0; b0 < r1; b0 += ng * U) {
      uint4 q[U];
#pragma unroll
      for (int i = 0; i < U; ++i) {
        const int r = b0 + g + i * ng;
        q[i] = (active && r < r1) ? ld_cg16(vb + (size_t)r * d + ci * 8) : make_uint4(0, 0, 0, 0);
      }
#pragma unroll
      for (int i = 0; i < U; ++i) {
        const int r = b0 + g + i * ng;
        float x[8];
        unpack8(q[i], x);
        float s;
        if (VAR == 0) {
          float acc = 0.f;
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const float dv = x[k] - m8[k];
            acc = fmaf(dv, dv, acc);
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
          float nv = 0.f;
#pragma unroll
          for (int k = 0; k < 8; ++k) nv = fmaf(x[k], x[k], nv);
          for (int off = 1; off < lpr; off <<= 1) nv += __shfl_xor_sync(kFull, nv, off);
          const float inv = nv > 0.f ? 1.f / sqrtf(nv) : 0.f;
          float acc = 0.f;
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const float dv = x[k] * inv - h8[k];
            acc = fmaf(dv, dv, acc);
          }
          for (int off = 1; off < lpr; off <<= 1) acc += __shfl_xor_sync(kFull, acc, off);
          s = (nv > 0.f && !mu_zero) ? 0.5f * acc : 1.f;
        }
        if (r < r1) {
          if (ci == 0 && sc_out) sc_out[r] = s;
          if (!a.score_only) {
            bool bad;
            const uint32_t key = score_key(s, bad);
            if (bad && ci == 0) record_status(a.status, kStNonfinite);
            if (DECODE) {
              const unsigned long long pk =
                  ((unsigned long long)key << 32) | (unsigned long long)(0xffffffffu - (unsigned)r);
              best = pk < best ? pk : best;
            } else if (C == 1) {
              if (ci == 0) keys[r] = key;
            } else {
              for (int cc = ci; cc < C; cc += lpr)
                st_cluster_u32(mapa(keys_addr + 4u * (unsigned)r, (unsigned)cc), key);
            }
          }
        }
      }
    }
    if (a.score_only) {
      if (split_exit) {
        cluster_arrive();
        cluster_wait();
      }
      return;
    }
    if (DECODE) {
      best = warp_min_u64(best);
      if (lane == 0) S.wbest[warp] = best;
      __syncthreads();
      if (tid == 0) {
        unsigned long long b = ~0ull;
        for (int w = 0; w < kWarps; ++w) b = S.wbest[w] < b ? S.wbest[w] : b;
        S.best = b;
      }
    }
  }
  if (C > 1) cluster_sync(); else __syncthreads();

  // ---- 3./4. select and kept list --------------------------------------
  int e_first;
  if (DECODE) {
    unsigned long long b = ~0ull;
    for (int rr = 0; rr < C; ++rr) {
      const unsigned long long o =
          C > 1 ? ld_cluster_u64(mapa(smem_addr(&S.best), rr)) : S.best;
      b = o < b ? o : b;
    }
    if (split_exit || C > 1) cluster_arrive();  // last peer access of this CTA
    e_first = (int)(0xffffffffu - (unsigned)(b & 0xffffffffull));
  } else {
    const Selection sel = radix_select(keys, n, Nb, S);
    build_perm(keys, n, Nb, sel, perm, S);
    e_first = S.e_first;
  }

  // ---- outputs -----------------------------------------------------------
  if (a.kept_out) {
    int32_t* ko = a.kept_out + (size_t)u * a.N;
    for (int i = (int)rank * kThreads + tid; i < a.N; i += C * kThreads) {
      int val = -1;
      if (i < Nb) val = DECODE ? (i < e_first ? i : i + 1) : perm[i];
      ko[i] = val;
    }
  }
  if (DECODE && a.evicted_out && rank == 0 && tid == 0) a.evicted_out[u] = e_first;

  // ---- 5. running sum: S += appended rows - evicted rows (own V columns) --
  if (a.mu_running && vchunks > 0) {
    zero_acc(S);
    const int first_new = n - a.B;
    const int nev = n - Nb;
    accumulate_rows(vb, d, vchunk0, vchunks, vp, a.B + nev,
                    [&](int i, int& row, float& sign) {
                      if (i < a.B) {
                        row = first_new + i;
                        sign = 1.f;
                      } else {
                        row = DECODE ? e_first : perm[Nb + (i - a.B)];
                        sign = -1.f;
                      }
                    },
                    S.acc_hi, S.acc_lo);
    if (tid < vchunks * 8) {
      const int c = vchunk0 * 8 + tid;
      double* sp = a.running_sum + (size_t)u * d + c;
      *sp = *sp + (double)S.acc_hi[c] + (double)S.acc_lo[c];
    }
  }

  // ---- 6. in-place compaction of this CTA's column slice ---------------
  compact_slice<4>(kb, vb, d, chunk0, cps, e_first, Nb, DECODE ? nullptr : perm);

  if (DECODE && C > 1) cluster_wait();
}

}  // namespace vd
