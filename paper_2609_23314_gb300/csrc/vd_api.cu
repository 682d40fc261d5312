// vd_api.cu -- host side of libvd.so: the C ABI declared in include/vd.h.
//
// Validates arguments before any launch, sizes the thread-block cluster per
// unit, launches the fused eviction kernel with cudaLaunchKernelExC on the
// caller's stream, and owns the device status word (a static __device__
// variable: the library allocates no device memory).
#include <cuda_runtime.h>

#include <algorithm>
#include <climits>
#include <cmath>
#include <cstdint>
#include <cstdlib>
#include <mutex>

#include "vd.h"
#include "vd_evict.cuh"
#include "vd_small.cuh"

namespace vd {
const void* evict_kernel_l2(bool decode, bool holefill, bool fused);
const void* evict_kernel_dir(bool decode, bool holefill, bool fused);
const void* evict_kernel_norm(bool decode, bool holefill, bool fused);
const void* small_kernel_l2(bool decode, bool fused);
const void* small_kernel_dir(bool decode, bool fused);
const void* small_kernel_norm(bool decode, bool fused);
const void* score_kernel_l2();
const void* score_kernel_dir();
const void* score_kernel_norm();
}  // namespace vd

using vd::kThreads;

// First device-side anomaly since the last vd_get_device_status (0 = none).
static __device__ unsigned g_vd_status;

// ---------------------------------------------------------------------------
// small kernels: append (Eq. block_processing's concatenation), length
// update after an eviction, and the from-scratch running sum
// ---------------------------------------------------------------------------
__global__ void vd_append_kernel(uint16_t* __restrict__ k, uint16_t* __restrict__ v,
                                 const uint16_t* __restrict__ kn, const uint16_t* __restrict__ vn,
                                 const int32_t* __restrict__ len, int units_per_seq,
                                 long long n_units, int cap, int d, int B, unsigned* status) {
  const int d8 = d >> 3;
  const long long total = n_units * (long long)B * d8;
  for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < total;
       idx += (long long)gridDim.x * blockDim.x) {
    const int c = (int)(idx % d8);
    const long long ub = idx / d8;
    const int b = (int)(ub % B);
    const long long u = ub / B;
    const int n = len[u / units_per_seq];
    if (n < 0 || n > cap - B) {
      if (b == 0 && c == 0 && u % units_per_seq == 0) vd::record_status(status, vd::kStDeviceLen);
      continue;
    }
    const size_t src = (size_t)ub * d + (size_t)c * 8;
    const size_t dst = ((size_t)u * cap + (size_t)(n + b)) * d + (size_t)c * 8;
    vd::st16(k + dst, vd::ld_cg16(kn + src));
    vd::st16(v + dst, vd::ld_cg16(vn + src));
  }
}

__global__ void vd_len_add_kernel(int32_t* len, int n_seq, int cap, int B) {
  const int s = blockIdx.x * blockDim.x + threadIdx.x;
  if (s >= n_seq) return;
  const int n = len[s];
  if (n >= 0 && n <= cap - B) len[s] = n + B;
}

// Mirrors the eviction kernel's per-sequence decision exactly.  added: the
// rows a fused append adds to len (0 when they were appended beforehand).
// Launched as a programmatic dependent of the eviction (which lets its
// dependents be scheduled at once): it is resident before the eviction ends
// and waits for it to complete before reading or writing len.
__global__ void vd_len_clamp_kernel(int32_t* len, const int32_t* N_dev, int N, int n_seq,
                                    int cap, int B, int running, int decode, int added) {
  vd::grid_dependency_wait();
  const int s = blockIdx.x * blockDim.x + threadIdx.x;
  if (s >= n_seq) return;
  const int n0 = len[s];
  const int n = n0 + added;
  const int Nb = N_dev ? N_dev[s] : N;
  if (n0 < 0 || n > cap || (running && B > n)) return;
  if (Nb < 1 || Nb > N) return;
  if (n <= Nb) {
    if (added) len[s] = n;
    return;
  }
  if (decode && n > Nb + 1) return;
  len[s] = Nb;
}

__global__ void __launch_bounds__(kThreads) vd_rsum_init_kernel(const uint16_t* __restrict__ v,
                                                                const int32_t* __restrict__ len,
                                                                double* rs, int units_per_seq,
                                                                int cap, int d, int lpr,
                                                                unsigned* status) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  vd::Smem& S = *reinterpret_cast<vd::Smem*>(smem_raw);
  const uint32_t ring = vd::smem_addr(smem_raw + vd::smem_layout(cap, 1, vd::kKindDecode).ring);
  const int u = blockIdx.x;
  const int n = len[u / units_per_seq];
  if (n < 0 || n > cap) {
    if (threadIdx.x == 0 && u % units_per_seq == 0) vd::record_status(status, vd::kStDeviceLen);
    return;
  }
  const uint16_t* vb = v + (size_t)u * cap * d;
  vd::sum_rows<vd::DecodeRing>(0, d >> 3, lpr, n, [&](int i) { return vb + (size_t)i * d; },
                               [](int) { return 1.f; }, S, ring);
  if ((int)threadIdx.x < d)
    rs[(size_t)u * d + threadIdx.x] = (double)S.acc_hi[threadIdx.x] + (double)S.acc_lo[threadIdx.x];
}

// ---------------------------------------------------------------------------
// per-device state
// ---------------------------------------------------------------------------
namespace {

// A cluster-size decision for one launch shape (the occupancy queries behind
// it cost more host time than a small eviction takes on the device).
struct ClusterChoice {
  const void* kern;
  long long units;
  int d, capacity, kind, want, c;  // kind: vd::kKind*, or kFitsKind (cached_fits)
  size_t smem;
  long long solo, want_solo;       // split launch: units run one CTA each (split_plan)
};
constexpr int kChoiceSlots = 32;

struct DeviceState {
  bool ready = false;
  unsigned* status = nullptr;
  int sms = 0;
  int smem_optin = 0;
  ClusterChoice choice[kChoiceSlots];  // guarded by g_mu; replaced round-robin
  int n_choice = 0, next_choice = 0;
};

constexpr int kMaxDevices = 64;
std::mutex g_mu;
DeviceState g_dev[kMaxDevices];

const void* evict_kernel(vd_variant var, bool decode, bool holefill, bool fused) {
  switch (var) {
    case VD_SCORE_L2: return vd::evict_kernel_l2(decode, holefill, fused);
    case VD_SCORE_DIR: return vd::evict_kernel_dir(decode, holefill, fused);
    default: return vd::evict_kernel_norm(decode, holefill, fused);
  }
}

const void* score_kernel(vd_variant var) {
  switch (var) {
    case VD_SCORE_L2: return vd::score_kernel_l2();
    case VD_SCORE_DIR: return vd::score_kernel_dir();
    default: return vd::score_kernel_norm();
  }
}

const void* small_kernel(vd_variant var, bool decode, bool fused) {
  switch (var) {
    case VD_SCORE_L2: return vd::small_kernel_l2(decode, fused);
    case VD_SCORE_DIR: return vd::small_kernel_dir(decode, fused);
    default: return vd::small_kernel_norm(decode, fused);
  }
}

vd_status device_state(DeviceState** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    cudaGetLastError();
    return VD_ERR_NO_DEVICE;
  }
  std::lock_guard<std::mutex> lk(g_mu);
  DeviceState& st = g_dev[dev];
  if (!st.ready) {
    cudaDeviceProp p;
    if (cudaGetDeviceProperties(&p, dev) != cudaSuccess) {
      cudaGetLastError();
      return VD_ERR_NO_DEVICE;
    }
    if (p.major != 10 || p.minor != 3) return VD_ERR_NO_DEVICE;  // built for sm_103a only
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_vd_status) != cudaSuccess) return VD_ERR_CUDA;
    st.status = static_cast<unsigned*>(ptr);
    st.sms = p.multiProcessorCount;
    st.smem_optin = (int)p.sharedMemPerBlockOptin;
    if (cudaFuncSetAttribute(reinterpret_cast<const void*>(&vd_rsum_init_kernel),
                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                             st.smem_optin) != cudaSuccess)
      return VD_ERR_CUDA;
    for (int var = 0; var < 3; ++var)
      for (int kind = 0; kind < 8; ++kind) {
        const void* kern =
            evict_kernel((vd_variant)var, (kind & 1) != 0, (kind & 2) != 0, (kind & 4) != 0);
        if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 st.smem_optin) != cudaSuccess ||
            cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) !=
                cudaSuccess)
          return VD_ERR_CUDA;
      }
    for (int var = 0; var < 3; ++var)
      for (int kind = 0; kind < 5; ++kind) {
        const void* kern = kind == 4 ? score_kernel((vd_variant)var)
                                     : small_kernel((vd_variant)var, (kind & 1) != 0,
                                                    (kind & 2) != 0);
        if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 st.smem_optin) != cudaSuccess ||
            cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) !=
                cudaSuccess)
          return VD_ERR_CUDA;
      }
    st.ready = true;
  }
  *out = &st;
  return VD_OK;
}

vd_status validate_cache(const vd_cache* c) {
  if (!c || !c->k || !c->v || !c->len) return VD_ERR_INVALID_ARG;
  if (c->n_seq < 1 || c->n_layer < 1 || c->n_kv_head < 1 || c->capacity < 1 || c->head_dim < 1)
    return VD_ERR_INVALID_ARG;
  if (c->head_dim % 8 != 0) return VD_ERR_ALIGNMENT;
  if (c->head_dim > 256) return VD_ERR_UNSUPPORTED;
  if ((reinterpret_cast<uintptr_t>(c->k) | reinterpret_cast<uintptr_t>(c->v)) & 15u)
    return VD_ERR_ALIGNMENT;
  const long long units = (long long)c->n_seq * c->n_layer * c->n_kv_head;
  if (units * 16 > INT_MAX) return VD_ERR_UNSUPPORTED;  // grid of units x cluster CTAs
  return VD_OK;
}

int lanes_per_row(int d) {
  int p = 1;
  while (p < d / 8) p <<= 1;
  return p;
}

bool cluster_fits(const void* kern, long long groups, int c, size_t smem) {
  if (c == 1) return true;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(groups * c));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeClusterDimension;
  attr.val.clusterDim.x = (unsigned)c;
  attr.val.clusterDim.y = 1;
  attr.val.clusterDim.z = 1;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  int ncl = 0;
  if (cudaOccupancyMaxActiveClusters(&ncl, kern, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return ncl > 0;
}

bool cluster_allowed(int c, int d) {
  const int total_chunks = 2 * (d / 8);
  return c == 1 || (total_chunks % c == 0 && total_chunks / c >= 4);
}

// CTAs per unit: C in {1, 2, 4, 8, 16}, keeping row segments of at least 64
// bytes of [K | V].  Waves = CTAs / resident slots at that C's shared-memory
// size.  Decode and score-only launches: the smallest C whose CTAs form one
// nearly full wave (0.85-1) or at least two waves, so that no short tail
// wave runs alone.  Ordered block eviction (moves most of the cache): the
// smallest C with 0.85-1 waves or at least four, else the decode rule.
// Hole-fill block eviction (moves few rows, so the select's cluster
// synchronisation dominates and grows with C): the smallest C with at least
// 0.4 of a wave (one short wave beats a long tail and more cluster barriers:
// prefill_wide C=1, 0.74 waves, 0.211-0.216 ms vs C=2, 1.47 waves,
// 0.216-0.221; prefill_gqa8b C=1, 0.47 waves, 0.064 ms vs C=2, 0.95 waves,
// 0.069).  Score-only launches on the bulk-copy ring: the smallest C with at
// least half a wave (fewer, longer contiguous slices: the prefill_wide sigma
// pass at C=1, 0.74 waves, 0.115 ms vs C=2 0.131, C=4 0.139; 2 ring stages at
// 3 CTAs per SM; 3 stages 0.141 ms, 4 stages 0.149).  With none such (few
// units), the largest allowed C that
// leaves every CTA at least kMinRowsPerCta rows of the capacity, else the
// smallest allowed C: below that, the cluster barriers cost more than the
// split saves.  (Measured on GB300: prefill_wide ordered C=8 (4.4 waves)
// 0.574 ms vs C=4 (2.2) 0.586; hole-fill C=2 (1.47 waves) 0.205 vs C=4
// 0.216; decode C=1; two units of 160 rows C=1 16.8 us vs C=4 18.5, of 600
// rows C=4 20.9 vs C=1 26.4, of 2400 rows C=8 27.9 vs C=1 75.7.)  Where no C
// with 64-byte segments fits the shared memory (a large capacity at a small
// head dim), the smallest C that fits.  want
// (VD_CLUSTER_SIZE: 1, 2, 4, 8 or 16) overrides the choice, for tuning.
constexpr int kMinRowsPerCta = 128;

int choose_cluster(const void* kern, long long units, int d, int capacity, int kind,
                   bool holefill, int want, const DeviceState& st, size_t* smem_out) {
  const bool with_select = kind == vd::kKindBlock;
  int chosen = 0, fallback = 0, roomy = 0, smallest = 0, narrow = 0;
  for (int c = 1; c <= 16; c *= 2) {
    if (want >= 1 && c != want) continue;
    if ((d / 8 * 2) % c) continue;
    const size_t smem = vd::smem_layout(capacity, c, kind).total;
    if (smem > (size_t)st.smem_optin) continue;
    int occ = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, kern, kThreads, smem) != cudaSuccess) {
      cudaGetLastError();
      continue;
    }
    if (occ < 1 || !cluster_fits(kern, units, c, smem)) continue;
    if (want < 1 && !cluster_allowed(c, d)) {
      // narrower row segments than preferred: only when nothing else fits
      // (a large capacity at a small head dim)
      if (narrow == 0) narrow = c;
      continue;
    }
    if (smallest == 0) smallest = c;
    if ((capacity + c - 1) / c >= kMinRowsPerCta) roomy = c;
    const double waves = (double)(units * c) / ((double)st.sms * occ);
    const bool full_wave = waves >= 0.85 && waves <= 1.0;
    bool ok;
    if (want >= 1)
      ok = true;
    else if (with_select && holefill)
      ok = waves >= 0.4;
    else if (kind == vd::kKindScoreBulk)
      ok = waves >= 0.5;
    else if (with_select)
      ok = full_wave || waves >= 4.0;
    else
      ok = full_wave || waves >= 2.0;
    if (ok) {
      chosen = c;
      break;
    }
    if (fallback == 0 && (full_wave || waves >= 2.0)) fallback = c;
  }
  if (chosen == 0)
    chosen = fallback ? fallback : roomy ? roomy : smallest ? smallest : narrow ? narrow : 1;
  *smem_out = vd::smem_layout(capacity, chosen, kind).total;
  return chosen;
}

// Split launch, for launches that fit one wave of one CTA per unit and
// carry more units than the GPU has SMs.  The block scheduler hands CTAs out
// breadth-first, so with U = k P + L units on P SMs (0 < L < P), L SMs run
// k + 1 whole units and the rest k, and the launch lasts as long as the
// busiest SMs (prefill_wide in the hole-fill layout, 336 units on 152 SMs:
// the CTAs of the 32 SMs that held three finished 28 us after the median).
// Instead, a first launch runs the first k P units (rounded down to a
// multiple of c) one CTA each, and a second launch, a programmatic dependent
// of the first, runs each remaining unit on a cluster of c CTAs: its CTAs
// take the slots the first leaves free, so an SM carries at most
// k + ceil(L c / P) / c units.  c in {2, 4, 8, 16} is the one with the
// smallest such load whose CTAs still form one wave; the split is taken when
// it lowers the load by at least a quarter of a unit.  Used by hole-fill
// block eviction and the score-only launches (each reads its units once and
// moves few rows, so a unit's time is its share of the read bandwidth);
// VD_SPLIT_LAUNCH=0 turns it off.  Returns the number of units of the first
// launch (0: no split) and sets *c_out and *smem_out for the second.
long long split_plan(const void* kern, long long units, int d, int capacity, int kind,
                     const DeviceState& st, int* c_out, size_t* smem_out) {
  const long long P = st.sms;
  if (P < 1 || units <= P) return 0;
  const size_t smem1 = vd::smem_layout(capacity, 1, kind).total;
  if (smem1 > (size_t)st.smem_optin) return 0;
  int occ = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, kern, kThreads, smem1) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  if (occ < 1 || units > P * occ) return 0;  // more than one wave: CTAs balance themselves
  const long long k = units / P;
  if (units % P == 0) return 0;
  double best = (double)(k + 1) - 0.25;
  long long best_solo = 0;
  for (int c = 2; c <= 16; c *= 2) {
    if (!cluster_allowed(c, d)) continue;
    const long long solo = (k * P) / c * c;
    const long long joint = units - solo;
    if (solo + joint * c > P * occ) continue;  // one wave
    const double load = (double)((solo + P - 1) / P) + (double)((joint * c + P - 1) / P) / c;
    const size_t smem_c = vd::smem_layout(capacity, c, kind).total;
    if (load < best && cluster_fits(kern, joint, c, smem_c)) {
      best = load;
      best_solo = solo;
      *c_out = c;
      *smem_out = smem_c;
    }
  }
  return best_solo;
}

// choose_cluster (and split_plan), remembered per launch shape.  A forced
// cluster size (VD_CLUSTER_SIZE) turns the automatic split off;
// VD_SOLO_UNITS with it forces a split whose first launch runs that many
// units (at most all but one) one CTA each, for tests.
int cached_cluster(const void* kern, long long units, int d, int capacity, int kind,
                   bool holefill, DeviceState& st, size_t* smem_out, long long* solo_out) {
  const char* env = std::getenv("VD_CLUSTER_SIZE");
  const int want = env ? std::atoi(env) : 0;
  // want_solo: the forced first part (VD_SOLO_UNITS, with a forced cluster
  // size), else 0 when the split is turned off, else -1 (automatic)
  long long want_solo = -1;
  if (want >= 1) {
    const char* senv = std::getenv("VD_SOLO_UNITS");
    if (senv) want_solo = std::atoll(senv);
  } else {
    const char* off = std::getenv("VD_SPLIT_LAUNCH");
    if (off && std::atoi(off) == 0) want_solo = 0;
  }
  {
    std::lock_guard<std::mutex> lk(g_mu);
    for (int i = 0; i < st.n_choice; ++i) {
      const ClusterChoice& e = st.choice[i];
      if (e.kern == kern && e.units == units && e.d == d && e.capacity == capacity &&
          e.kind == kind && e.want == want && e.want_solo == want_solo) {
        *smem_out = e.smem;
        *solo_out = e.solo;
        return e.c;
      }
    }
  }
  int c = choose_cluster(kern, units, d, capacity, kind, holefill, want, st, smem_out);
  long long solo = 0;
  if (want >= 1 && want_solo > 0) {
    solo = std::min(want_solo, units - 1);
  } else if (want < 1 && want_solo != 0 &&
             ((kind == vd::kKindBlock && holefill) || kind == vd::kKindScore ||
              kind == vd::kKindScoreBulk)) {
    int cs = c;
    size_t sm = *smem_out;
    solo = split_plan(kern, units, d, capacity, kind, st, &cs, &sm);
    if (solo > 0) {
      c = cs;
      *smem_out = sm;
    }
  }
  std::lock_guard<std::mutex> lk(g_mu);
  st.choice[st.next_choice] =
      ClusterChoice{kern, units, d, capacity, kind, want, c, *smem_out, solo, want_solo};
  st.next_choice = (st.next_choice + 1) % kChoiceSlots;
  if (st.n_choice < kChoiceSlots) ++st.n_choice;
  *solo_out = solo;
  return c;
}

// The short-cache kernel (vd_small.cuh) takes a block or decode event when
// the unit's K and V rows fit in shared memory with room to spare
// (capacity * head_dim * 4 bytes <= kSmallRowBytes, capacity <= 1024), a
// sequence's units fit in one cluster (<= 16), the launch is at most two
// waves of one CTA per SM, and no scoring option, hole-fill layout or forced
// cluster size (VD_CLUSTER_SIZE) is asked for.  VD_SMALL_PATH=0 turns it
// off.  The choice depends on the shape only, so the fused and two-call
// forms, block and decode, take the same kernel.
constexpr size_t kSmallRowBytes = 64 * 1024;

bool cluster_fits(const void* kern, long long groups, int c, size_t smem);

bool use_small(const vd_cache* c, bool score_only, bool holefill, const float* weights,
               const float* disp_out, int score_k, const DeviceState& st) {
  if (score_only || holefill || weights || disp_out || score_k) return false;
  const char* off = std::getenv("VD_SMALL_PATH");
  if ((off && std::atoi(off) == 0) || std::getenv("VD_CLUSTER_SIZE")) return false;
  const int ups = c->n_layer * c->n_kv_head;
  const long long units = (long long)c->n_seq * ups;
  if (ups > 16 || c->capacity > vd::kSmallMaxRows || units > 2LL * st.sms) return false;
  if ((size_t)c->capacity * c->head_dim * 4 > kSmallRowBytes) return false;
  return vd::small_layout(c->capacity, c->head_dim).total <= (size_t)st.smem_optin;
}

// groups clusters of c CTAs: the fused kernel's grid is units x c CTAs (a
// cluster per unit), the short-cache kernel's n_seq x units_per_seq (a
// cluster per sequence, a CTA per unit)
// cluster_fits, remembered per launch shape (the occupancy query costs
// several microseconds of host time, as much as a short-cache event takes on
// the device); entries are marked kind == kFitsKind in the choice cache.
constexpr int kFitsKind = 3;
bool cached_fits(const void* kern, long long groups, int c, size_t smem, DeviceState& st) {
  {
    std::lock_guard<std::mutex> lk(g_mu);
    for (int i = 0; i < st.n_choice; ++i) {
      const ClusterChoice& e = st.choice[i];
      if (e.kern == kern && e.units == groups && e.kind == kFitsKind && e.want == c &&
          e.smem == smem)
        return e.c != 0;
    }
  }
  const bool fits = c == 1 || cluster_fits(kern, groups, c, smem);
  std::lock_guard<std::mutex> lk(g_mu);
  st.choice[st.next_choice] =
      ClusterChoice{kern, groups, 0, 0, kFitsKind, c, fits ? c : 0, smem, 0, 0};
  st.next_choice = (st.next_choice + 1) % kChoiceSlots;
  if (st.n_choice < kChoiceSlots) ++st.n_choice;
  return fits;
}

vd_status launch(const void* kern, long long groups, int c, size_t smem, const void* params,
                 cudaStream_t s, bool dependent = false) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(groups * c));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)c;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  // a programmatic dependent launch (the kernel waits in griddepcontrol.wait)
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = dependent ? 2 : 1;
  void* args[] = {const_cast<void*>(params)};
  if (cudaLaunchKernelExC(&cfg, kern, args) != cudaSuccess) {
    cudaGetLastError();
    return VD_ERR_CUDA;
  }
  return VD_OK;
}

vd_status run(const vd_cache* c, int32_t N, const int32_t* N_dev, int32_t B, vd_variant var,
              vd_mu_mode mu, double* running_sum, int32_t* evicted_out, int32_t* kept_idx_out,
              float* scores_out, cudaStream_t s, bool decode, bool score_only,
              int32_t* pos = nullptr, const int32_t* pos_new = nullptr, int score_k = 0,
              const float* weights = nullptr, float* disp_out = nullptr,
              const void* k_new = nullptr, const void* v_new = nullptr) {
  vd_status r = validate_cache(c);
  if (r != VD_OK) return r;
  if (var != VD_SCORE_L2 && var != VD_SCORE_DIR && var != VD_SCORE_NORM) return VD_ERR_INVALID_ARG;
  if (mu != VD_MU_RECOMPUTE && mu != VD_MU_RUNNING) return VD_ERR_INVALID_ARG;
  if (!score_only) {
    if (N < 1 || N > c->capacity) return VD_ERR_INVALID_ARG;
    if (B < 0 || B > c->capacity) return VD_ERR_INVALID_ARG;
    if (mu == VD_MU_RUNNING && !running_sum) return VD_ERR_INVALID_ARG;
  } else if (!scores_out && !disp_out) {
    return VD_ERR_INVALID_ARG;
  }
  if (disp_out && (decode || var != VD_SCORE_L2)) return VD_ERR_INVALID_ARG;
  if (weights && (score_only || decode)) return VD_ERR_INVALID_ARG;
  const bool holefill = pos != nullptr || pos_new != nullptr;
  if (holefill && (!pos || !pos_new)) return VD_ERR_INVALID_ARG;
  const bool fused = k_new != nullptr || v_new != nullptr;
  if (fused) {
    if (!k_new || !v_new || B < 1 || score_only) return VD_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(k_new) | reinterpret_cast<uintptr_t>(v_new)) & 15u)
      return VD_ERR_ALIGNMENT;
  }
  DeviceState* st = nullptr;
  r = device_state(&st);
  if (r != VD_OK) return r;

  // score-only launches have their own instantiation (no per-token buffers)
  const int kind = score_only ? (vd::score_bulk((int)var, c->head_dim) ? vd::kKindScoreBulk
                                                                       : vd::kKindScore)
                 : decode     ? vd::kKindDecode
                              : vd::kKindBlock;
  if (kind == vd::kKindBlock && c->capacity > 65536) return VD_ERR_UNSUPPORTED;  // 16-bit lists
  if (vd::smem_layout(c->capacity, 16, kind).total > (size_t)st->smem_optin)
    return VD_ERR_UNSUPPORTED;
  const void* kern = score_only ? score_kernel(var) : evict_kernel(var, decode, holefill, fused);
  const long long units = (long long)c->n_seq * c->n_layer * c->n_kv_head;

  vd::EvictArgs a;
  a.k = static_cast<uint16_t*>(c->k);
  a.v = static_cast<uint16_t*>(c->v);
  a.len = c->len;
  a.N_dev = score_only ? nullptr : N_dev;
  a.running_sum = running_sum;
  a.kept_out = score_only ? nullptr : kept_idx_out;
  a.evicted_out = decode ? evicted_out : nullptr;
  a.scores_out = scores_out;
  a.status = st->status;
  a.units_per_seq = c->n_layer * c->n_kv_head;
  a.d = c->head_dim;
  a.lpr = lanes_per_row(c->head_dim);
  a.capacity = c->capacity;
  a.N = score_only ? 1 : N;
  a.B = decode ? 1 : B;
  a.mu_running = mu == VD_MU_RUNNING ? 1 : 0;
  a.score_only = score_only ? 1 : 0;
  a.pos = pos;
  a.pos_new = pos_new;
  a.holefill = holefill ? 1 : 0;
  a.score_k = score_k ? 1 : 0;
  a.weights = weights;
  a.disp_out = disp_out;
  a.k_new = static_cast<const uint16_t*>(k_new);
  a.v_new = static_cast<const uint16_t*>(v_new);
  a.unit_base = 0;
  if (use_small(c, score_only, holefill, weights, disp_out, score_k, *st)) {
    // one launch: the kernel also sets the sequences' lengths
    // grid: n_seq clusters of units_per_seq CTAs, one CTA per unit
    const void* sk = small_kernel(var, decode, fused);
    const size_t ssmem = vd::small_layout(c->capacity, c->head_dim).total;
    a.cluster = a.units_per_seq;
    if (cached_fits(sk, c->n_seq, a.cluster, ssmem, *st)) {
      const vd::SmallArgs sa{a, (int32_t)units};
      return launch(sk, c->n_seq, a.cluster, ssmem, &sa, s, true);
    }
  }
  size_t smem = 0;
  long long solo = 0;
  a.cluster =
      cached_cluster(kern, units, c->head_dim, c->capacity, kind, holefill, *st, &smem, &solo);
  if (smem > (size_t)st->smem_optin) return VD_ERR_UNSUPPORTED;

  if (solo > 0) {
    // split launch: units [0, solo) one CTA each, then the rest on clusters,
    // as a programmatic dependent of the first part
    vd::EvictArgs a1 = a;
    a1.cluster = 1;
    const size_t smem1 = vd::smem_layout(c->capacity, 1, kind).total;
    if (smem1 > (size_t)st->smem_optin) return VD_ERR_UNSUPPORTED;
    r = launch(kern, solo, 1, smem1, &a1, s);
    if (r != VD_OK) return r;
    // the second part's per-unit pointers start at unit `solo`
    const size_t rows = (size_t)solo * c->capacity, dd = (size_t)c->head_dim;
    a.unit_base = (int32_t)solo;
    a.k += rows * dd;
    a.v += rows * dd;
    if (a.running_sum) a.running_sum += (size_t)solo * dd;
    if (a.kept_out) a.kept_out += (size_t)solo * a.N;
    if (a.evicted_out) a.evicted_out += solo;
    if (a.scores_out) a.scores_out += rows;
    if (a.pos) a.pos += rows;
    if (a.weights) a.weights += rows;
    if (a.disp_out) a.disp_out += solo;
    if (a.k_new) a.k_new += (size_t)solo * a.B * dd;
    if (a.v_new) a.v_new += (size_t)solo * a.B * dd;
    r = launch(kern, units - solo, a.cluster, smem, &a, s, true);
  } else {
    r = launch(kern, units, a.cluster, smem, &a, s);
  }
  if (r != VD_OK || score_only) return r;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)((c->n_seq + kThreads - 1) / kThreads));
  cfg.blockDim = dim3(kThreads);
  cfg.stream = s;
  cudaLaunchAttribute pdl;
  pdl.id = cudaLaunchAttributeProgrammaticStreamSerialization;
  pdl.val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = &pdl;
  cfg.numAttrs = 1;
  if (cudaLaunchKernelEx(&cfg, vd_len_clamp_kernel, c->len, N_dev, N, c->n_seq, c->capacity,
                         (int)a.B, (int)a.mu_running, decode ? 1 : 0, fused ? (int)a.B : 0) !=
      cudaSuccess) {
    cudaGetLastError();
    return VD_ERR_CUDA;
  }
  return VD_OK;
}

}  // namespace

// ---------------------------------------------------------------------------
// C ABI
// ---------------------------------------------------------------------------
extern "C" {

vd_status vd_score(const vd_cache* c, vd_variant var, float* scores_out, vd_stream_t stream) {
  return run(c, 1, nullptr, 0, var, VD_MU_RECOMPUTE, nullptr, nullptr, nullptr, scores_out,
             reinterpret_cast<cudaStream_t>(stream), false, true);
}

vd_status vd_append_evict_block(const vd_cache* c, const void* k_new, const void* v_new,
                                int32_t B, int32_t N, const int32_t* N_dev, vd_variant var,
                                vd_mu_mode mu, double* running_sum, int32_t* pos,
                                const int32_t* pos_first_new, int32_t* kept_idx_out,
                                float* scores_out, vd_stream_t stream) {
  return run(c, N, N_dev, B, var, mu, running_sum, nullptr, kept_idx_out, scores_out,
             reinterpret_cast<cudaStream_t>(stream), false, false, pos, pos_first_new, 0,
             nullptr, nullptr, k_new, v_new);
}

vd_status vd_append_evict_decode(const vd_cache* c, const void* k_new, const void* v_new,
                                 int32_t N, const int32_t* N_dev, vd_variant var, vd_mu_mode mu,
                                 double* running_sum, int32_t* pos, const int32_t* pos_first_new,
                                 int32_t* evicted_out, int32_t* kept_idx_out, float* scores_out,
                                 vd_stream_t stream) {
  return run(c, N, N_dev, 1, var, mu, running_sum, evicted_out, kept_idx_out, scores_out,
             reinterpret_cast<cudaStream_t>(stream), true, false, pos, pos_first_new, 0, nullptr,
             nullptr, k_new, v_new);
}

vd_status vd_evict_block(const vd_cache* c, int32_t N, const int32_t* N_dev, int32_t B,
                         vd_variant var, vd_mu_mode mu, double* running_sum,
                         int32_t* kept_idx_out, float* scores_out, vd_stream_t stream) {
  return run(c, N, N_dev, B, var, mu, running_sum, nullptr, kept_idx_out, scores_out,
             reinterpret_cast<cudaStream_t>(stream), false, false);
}

vd_status vd_evict_decode(const vd_cache* c, int32_t N, const int32_t* N_dev, vd_variant var,
                          vd_mu_mode mu, double* running_sum, int32_t* evicted_out,
                          int32_t* kept_idx_out, float* scores_out, vd_stream_t stream) {
  return run(c, N, N_dev, 1, var, mu, running_sum, evicted_out, kept_idx_out, scores_out,
             reinterpret_cast<cudaStream_t>(stream), true, false);
}

vd_status vd_score_ex(const vd_cache* c, vd_variant var, vd_mu_mode mu,
                      const double* running_sum, int32_t score_keys, float* scores_out,
                      float* dispersion_out, vd_stream_t stream) {
  if (mu == VD_MU_RUNNING && !running_sum) return VD_ERR_INVALID_ARG;
  // the score-only kernel reads the running sum and never writes it
  return run(c, 1, nullptr, 0, var, mu, const_cast<double*>(running_sum), nullptr, nullptr,
             scores_out, reinterpret_cast<cudaStream_t>(stream), false, true, nullptr, nullptr,
             score_keys, nullptr, dispersion_out);
}

vd_status vd_evict_block_ex(const vd_cache* c, int32_t N, const int32_t* N_dev, int32_t B,
                            vd_variant var, vd_mu_mode mu, double* running_sum,
                            int32_t score_keys, const float* attn, int32_t* kept_idx_out,
                            float* scores_out, float* dispersion_out, vd_stream_t stream) {
  return run(c, N, N_dev, B, var, mu, running_sum, nullptr, kept_idx_out, scores_out,
             reinterpret_cast<cudaStream_t>(stream), false, false, nullptr, nullptr, score_keys,
             attn, dispersion_out);
}

vd_status vd_append_evict_block_ex(const vd_cache* c, const void* k_new, const void* v_new,
                                   int32_t B, int32_t N, const int32_t* N_dev, vd_variant var,
                                   vd_mu_mode mu, double* running_sum, int32_t score_keys,
                                   const float* attn, int32_t* kept_idx_out, float* scores_out,
                                   float* dispersion_out, vd_stream_t stream) {
  return run(c, N, N_dev, B, var, mu, running_sum, nullptr, kept_idx_out, scores_out,
             reinterpret_cast<cudaStream_t>(stream), false, false, nullptr, nullptr, score_keys,
             attn, dispersion_out, k_new, v_new);
}

vd_status vd_evict_block_holefill(const vd_cache* c, int32_t N, const int32_t* N_dev, int32_t B,
                                  vd_variant var, vd_mu_mode mu, double* running_sum,
                                  int32_t* pos, const int32_t* pos_first_new,
                                  int32_t* kept_idx_out, float* scores_out, vd_stream_t stream) {
  if (!pos || !pos_first_new) return VD_ERR_INVALID_ARG;
  return run(c, N, N_dev, B, var, mu, running_sum, nullptr, kept_idx_out, scores_out,
             reinterpret_cast<cudaStream_t>(stream), false, false, pos, pos_first_new);
}

vd_status vd_evict_decode_holefill(const vd_cache* c, int32_t N, const int32_t* N_dev,
                                   vd_variant var, vd_mu_mode mu, double* running_sum,
                                   int32_t* pos, const int32_t* pos_first_new,
                                   int32_t* evicted_out, int32_t* kept_idx_out, float* scores_out,
                                   vd_stream_t stream) {
  if (!pos || !pos_first_new) return VD_ERR_INVALID_ARG;
  return run(c, N, N_dev, 1, var, mu, running_sum, evicted_out, kept_idx_out, scores_out,
             reinterpret_cast<cudaStream_t>(stream), true, false, pos, pos_first_new);
}

vd_status vd_append(const vd_cache* c, const void* k_new, const void* v_new, int32_t B,
                    vd_stream_t stream) {
  vd_status r = validate_cache(c);
  if (r != VD_OK) return r;
  if (!k_new || !v_new || B < 0 || B > c->capacity) return VD_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(k_new) | reinterpret_cast<uintptr_t>(v_new)) & 15u)
    return VD_ERR_ALIGNMENT;
  if (B == 0) return VD_OK;
  DeviceState* st = nullptr;
  r = device_state(&st);
  if (r != VD_OK) return r;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const long long units = (long long)c->n_seq * c->n_layer * c->n_kv_head;
  const long long work = units * B * (c->head_dim / 8);
  const long long want = (work + 255) / 256;
  const int blocks = (int)(want < (long long)st->sms * 32 ? want : (long long)st->sms * 32);
  vd_append_kernel<<<blocks, 256, 0, s>>>(
      static_cast<uint16_t*>(c->k), static_cast<uint16_t*>(c->v),
      static_cast<const uint16_t*>(k_new), static_cast<const uint16_t*>(v_new), c->len,
      c->n_layer * c->n_kv_head, units, c->capacity, c->head_dim, B, st->status);
  vd_len_add_kernel<<<(c->n_seq + 255) / 256, 256, 0, s>>>(c->len, c->n_seq, c->capacity, B);
  if (cudaGetLastError() != cudaSuccess) return VD_ERR_CUDA;
  return VD_OK;
}

vd_status vd_running_sum_init(const vd_cache* c, double* running_sum, vd_stream_t stream) {
  return vd_running_sum_init_ex(c, 0, running_sum, stream);
}

vd_status vd_running_sum_init_ex(const vd_cache* c, int32_t of_keys, double* running_sum,
                                 vd_stream_t stream) {
  vd_status r = validate_cache(c);
  if (r != VD_OK) return r;
  if (!running_sum) return VD_ERR_INVALID_ARG;
  DeviceState* st = nullptr;
  r = device_state(&st);
  if (r != VD_OK) return r;
  const long long units = (long long)c->n_seq * c->n_layer * c->n_kv_head;
  const size_t smem = vd::smem_layout(c->capacity, 1, vd::kKindDecode).total;
  vd_rsum_init_kernel<<<(unsigned)units, kThreads, smem, reinterpret_cast<cudaStream_t>(stream)>>>(
      static_cast<const uint16_t*>(of_keys ? c->k : c->v), c->len, running_sum,
      c->n_layer * c->n_kv_head,
      c->capacity, c->head_dim, lanes_per_row(c->head_dim), st->status);
  if (cudaGetLastError() != cudaSuccess) return VD_ERR_CUDA;
  return VD_OK;
}

size_t vd_workspace_size(const vd_cache* c) {
  (void)c;
  return 0;
}

const char* vd_status_string(vd_status st) {
  switch (st) {
    case VD_OK: return "ok";
    case VD_ERR_INVALID_ARG: return "invalid argument";
    case VD_ERR_ALIGNMENT: return "misaligned pointer or head_dim not a multiple of 8";
    case VD_ERR_UNSUPPORTED: return "unsupported shape";
    case VD_ERR_NONFINITE: return "non-finite score on the device";
    case VD_ERR_TIMEOUT: return "device wait timed out";
    case VD_ERR_CUDA: return "CUDA runtime error";
    case VD_ERR_DEVICE_LEN: return "device: sequence length out of range";
    case VD_ERR_DEVICE_BUDGET: return "device: budget out of range or decode over budget";
    case VD_ERR_NO_DEVICE: return "no sm_103 CUDA device";
    case VD_ERR_INTERNAL: return "device: inconsistent slot list (internal self-check)";
    default: return "unknown status";
  }
}

vd_status vd_get_device_status(vd_stream_t stream) {
  DeviceState* st = nullptr;
  vd_status r = device_state(&st);
  if (r != VD_OK) return r;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(s) != cudaSuccess) {
    cudaGetLastError();
    return VD_ERR_CUDA;
  }
  unsigned w = 0;
  const unsigned z = 0;
  if (cudaMemcpyFromSymbolAsync(&w, g_vd_status, sizeof w, 0, cudaMemcpyDeviceToHost, s) !=
          cudaSuccess ||
      cudaMemcpyToSymbolAsync(g_vd_status, &z, sizeof z, 0, cudaMemcpyHostToDevice, s) !=
          cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess) {
    cudaGetLastError();
    return VD_ERR_CUDA;
  }
  return static_cast<vd_status>(w);
}

}  // extern "C"
