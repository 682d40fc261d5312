// vd_device.cuh -- device-side building blocks of the GB300 (sm_103a) ValueDiff
// eviction kernels: bf16 unpacking, asynchronous copies, double-float sums,
// thread-block
// cluster primitives (distributed shared memory, hardware cluster barrier) and
// block-wide scans/reductions for a 256-thread CTA.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace vd {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr unsigned kFull = 0xffffffffu;

// Device status codes (the values of vd_status in include/vd.h).
constexpr unsigned kStNonfinite = 4;
constexpr unsigned kStTimeout = 5;
constexpr unsigned kStDeviceLen = 7;
constexpr unsigned kStDeviceBudget = 8;
constexpr unsigned kStInternal = 10;

// First anomaly wins; later ones are dropped.  Never traps.
__device__ __forceinline__ void record_status(unsigned* st, unsigned code) {
  atomicCAS(st, 0u, code);
}

// ---------------------------------------------------------------------------
// bf16 <-> fp32.  A bf16 value is the upper half of an fp32 bit pattern, so
// widening is a shift; eight values arrive per 16-byte vector.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void unpack8(const uint4& q, float (&x)[8]) {
  x[0] = __uint_as_float(q.x << 16);
  x[1] = __uint_as_float(q.x & 0xffff0000u);
  x[2] = __uint_as_float(q.y << 16);
  x[3] = __uint_as_float(q.y & 0xffff0000u);
  x[4] = __uint_as_float(q.z << 16);
  x[5] = __uint_as_float(q.z & 0xffff0000u);
  x[6] = __uint_as_float(q.w << 16);
  x[7] = __uint_as_float(q.w & 0xffff0000u);
}

// ---------------------------------------------------------------------------
// Packed fp32 pairs: the sm_100-family f32x2 add/fma instructions do two
// fp32 operations (each rounded as the scalar one) per issue slot.  A pair
// is a 64-bit register: low half = first element, high half = second.
// ---------------------------------------------------------------------------
__device__ __forceinline__ unsigned long long f2_pack(float lo, float hi) {
  unsigned long long r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}

__device__ __forceinline__ float f2_hsum(unsigned long long v) {
  float lo, hi;
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
  return lo + hi;
}

__device__ __forceinline__ void f2_unpack(unsigned long long v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}

__device__ __forceinline__ unsigned long long f2_add(unsigned long long a, unsigned long long b) {
  unsigned long long r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}

__device__ __forceinline__ unsigned long long f2_sub(unsigned long long a, unsigned long long b) {
  unsigned long long r;
  asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}

__device__ __forceinline__ unsigned long long f2_fma(unsigned long long a, unsigned long long b,
                                                     unsigned long long c) {
  unsigned long long r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
  return r;
}

// Two bf16 values (one 32-bit word, first element in the low half) widened
// to a packed fp32 pair.
__device__ __forceinline__ unsigned long long bf16x2_to_f2(uint32_t w) {
  return f2_pack(__uint_as_float(w << 16), __uint_as_float(w & 0xffff0000u));
}

// 16-byte global load through L2 only.  The "memory" clobber keeps it in
// program order with the plain C++ stores around it (the hole-fill path
// writes positions and slot maps between row moves).
__device__ __forceinline__ uint4 ld_cg16(const void* p) {
  uint4 r;
  asm volatile("ld.global.cg.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p)
               : "memory");
  return r;
}

// Asynchronous 16-byte global -> shared copy (LDGSTS), bypassing L1 and the
// register file; completion is tracked per thread with commit/wait groups.
__device__ __forceinline__ void cp_async16(uint32_t smem, const void* gptr) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem), "l"(gptr) : "memory");
}

__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}

template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

__device__ __forceinline__ uint4 ld_shared16(uint32_t addr) {
  uint4 r;
  asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "r"(addr)
               : "memory");
  return r;
}

// 8-byte shared-memory load into a packed fp32 pair.  volatile: issued at
// each use (a loop-invariant value the compiler would otherwise keep in
// registers); the data is written before the block barrier that precedes
// every use, so no memory clobber is needed.
__device__ __forceinline__ unsigned long long ld_shared_b64(uint32_t addr) {
  unsigned long long r;
  asm volatile("ld.shared.b64 %0, [%1];" : "=l"(r) : "r"(addr));
  return r;
}

__device__ __forceinline__ void st_shared16(uint32_t addr, const uint4& v) {
  asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};" ::"r"(addr), "r"(v.x), "r"(v.y), "r"(v.z),
               "r"(v.w)
               : "memory");
}

__device__ __forceinline__ float ld_shared_f32(uint32_t addr) {
  float r;
  asm volatile("ld.shared.f32 %0, [%1];" : "=f"(r) : "r"(addr) : "memory");
  return r;
}

__device__ __forceinline__ double ld_shared_f64(uint32_t addr) {
  double r;
  asm volatile("ld.shared.f64 %0, [%1];" : "=d"(r) : "r"(addr) : "memory");
  return r;
}

__device__ __forceinline__ void st_cluster_u16(uint32_t addr, uint16_t v) {
  asm volatile("st.shared::cluster.u16 [%0], %1;" ::"r"(addr), "h"(v) : "memory");
}

__device__ __forceinline__ void st16(void* p, const uint4& v) {
  asm volatile("st.global.v4.u32 [%0], {%1,%2,%3,%4};" ::"l"(p), "r"(v.x), "r"(v.y), "r"(v.z),
               "r"(v.w)
               : "memory");
}

// ---------------------------------------------------------------------------
// Programmatic dependent launch.  A kernel launched with programmatic stream
// serialization may start before the previous kernel on its stream has
// finished; griddepcontrol.wait blocks until that kernel has completed and
// its memory is visible (a no-op for a normal launch), so it must come before
// the first access to memory.  launch_dependents lets the next kernel on the
// stream, if it was launched the same way, be scheduled once every CTA of
// this grid has issued it (it then waits in its own griddepcontrol.wait).
// ---------------------------------------------------------------------------
__device__ __forceinline__ void grid_dependency_wait() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}

__device__ __forceinline__ void grid_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// ---------------------------------------------------------------------------
// Bulk copies: one thread moves a contiguous block of global memory into this
// CTA's own shared memory (cp.async.bulk, no multicast; both addresses and the
// size multiples of 16 bytes), and the copy's completion is counted on an
// mbarrier in shared memory (expect_tx bytes, complete_tx by the copy).
// ---------------------------------------------------------------------------
__device__ __forceinline__ void mbar_init(uint32_t bar, unsigned count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

// Makes barrier initialisations visible to the copy engine (and the cluster).
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

// Orders this thread's earlier shared-memory accesses before later bulk-copy
// writes into the same memory.
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes,
                                         uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
      ::"r"(dst), "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}

// Waits until the barrier's phase with the given parity has completed, for
// at most `limit` polls.  Returns false (and records kStTimeout) if it gave
// up: the caller then goes on with whatever the buffer holds, so that the
// kernel still ends and every barrier of the CTA or cluster is still reached.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, unsigned* status,
                                          unsigned limit = 1u << 22) {
  for (unsigned i = 0; i < limit; ++i) {
    uint32_t done;
    asm volatile(
        "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; "
        "selp.u32 %0, 1, 0, p; }"
        : "=r"(done)
        : "r"(bar), "r"(parity)
        : "memory");
    if (done) return true;
  }
  record_status(status, kStTimeout);
  return false;
}

// ---------------------------------------------------------------------------
// Double-float (hi + lo) sums in fp32 arithmetic.  Each element enters with
// Knuth's TwoSum, whose rounding error is exact and collected in lo, so a sum
// over thousands of bf16 rows keeps ~2^-44 relative accuracy without fp64 in
// the inner loop (fp64 throughput on GB300 is a small fraction of fp32).
// ---------------------------------------------------------------------------
struct ff {
  float hi, lo;
};

__device__ __forceinline__ void ff_accumulate(float& hi, float& lo, float x) {
  const float s = hi + x;
  const float bb = s - hi;
  lo += (hi - (s - bb)) + (x - bb);
  hi = s;
}

// ff_accumulate on two columns at once: the same seven roundings per element
// in the same order, on packed fp32 pairs (bit-identical results, half the
// instructions).
__device__ __forceinline__ void ff2_accumulate(unsigned long long& hi, unsigned long long& lo,
                                               unsigned long long x) {
  const unsigned long long s = f2_add(hi, x);
  const unsigned long long bb = f2_sub(s, hi);
  lo = f2_add(lo, f2_add(f2_sub(hi, f2_sub(s, bb)), f2_sub(x, bb)));
  hi = s;
}

__device__ __forceinline__ ff ff_add(ff a, ff b) {
  const float s = a.hi + b.hi;
  const float v = s - a.hi;
  float e = (a.hi - (s - v)) + (b.hi - v);
  e += a.lo + b.lo;
  const float hi = s + e;
  return {hi, e - (hi - s)};
}

__device__ __forceinline__ ff ff_shfl_xor(ff a, int off) {
  return {__shfl_xor_sync(kFull, a.hi, off), __shfl_xor_sync(kFull, a.lo, off)};
}

// ---------------------------------------------------------------------------
// Thread-block clusters: all CTAs of one (sequence, layer, head) unit form one
// cluster.  Shared memory of a peer CTA is addressed through `mapa`; the
// hardware cluster barrier (release/acquire) orders those accesses.
// ---------------------------------------------------------------------------
__device__ __forceinline__ unsigned cluster_ctarank() {
  unsigned r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

__device__ __forceinline__ unsigned cluster_id_x() {
  unsigned r;
  asm volatile("mov.u32 %0, %%clusterid.x;" : "=r"(r));
  return r;
}

// Not the .aligned forms: an .aligned barrier must be executed by all threads
// of a warp together, and several call sites follow code in which a warp's
// threads diverged (a loop with a per-thread trip count, a tid == 0 branch).
// The compiler gives an inline-asm barrier no reconvergence point, so with
// .aligned, whether a warp arrives converged would depend on code layout.
__device__ __forceinline__ void cluster_arrive() {
  asm volatile("barrier.cluster.arrive.release;" ::: "memory");
}

__device__ __forceinline__ void cluster_wait() {
  asm volatile("barrier.cluster.wait.acquire;" ::: "memory");
}

__device__ __forceinline__ void cluster_sync() {
  cluster_arrive();
  cluster_wait();
}

__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint32_t mapa(uint32_t addr, unsigned rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}

__device__ __forceinline__ void st_cluster_u32(uint32_t addr, uint32_t v) {
  asm volatile("st.shared::cluster.u32 [%0], %1;" ::"r"(addr), "r"(v) : "memory");
}

__device__ __forceinline__ uint32_t ld_cluster_u32(uint32_t addr) {
  uint32_t v;
  asm volatile("ld.shared::cluster.u32 %0, [%1];" : "=r"(v) : "r"(addr) : "memory");
  return v;
}

__device__ __forceinline__ uint64_t ld_cluster_u64(uint32_t addr) {
  uint64_t v;
  asm volatile("ld.shared::cluster.u64 %0, [%1];" : "=l"(v) : "r"(addr) : "memory");
  return v;
}

__device__ __forceinline__ float ld_cluster_f32(uint32_t addr) {
  return __uint_as_float(ld_cluster_u32(addr));
}

// ---------------------------------------------------------------------------
// Block-wide helpers for a kThreads-thread CTA.  `sh` is kWarps ints of shared
// scratch; every helper ends with a barrier so `sh` can be reused at once.
// ---------------------------------------------------------------------------
__device__ __forceinline__ int block_exclusive_scan(int v, int* sh, int& total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int y = __shfl_up_sync(kFull, x, off);
    if (lane >= off) x += y;
  }
  if (lane == 31) sh[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int t = lane < kWarps ? sh[lane] : 0;
#pragma unroll
    for (int off = 1; off < kWarps; off <<= 1) {
      const int y = __shfl_up_sync(kFull, t, off);
      if (lane >= off) t += y;
    }
    if (lane < kWarps) sh[lane] = t;
  }
  __syncthreads();
  const int res = (warp ? sh[warp - 1] : 0) + x - v;
  total = sh[kWarps - 1];
  __syncthreads();
  return res;
}

__device__ __forceinline__ uint64_t warp_min_u64(uint64_t v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const uint64_t o = __shfl_xor_sync(kFull, v, off);
    v = o < v ? o : v;
  }
  return v;
}

// Deterministic (fixed-order) block sum of one float per thread.
__device__ __forceinline__ float block_sum_f32(float v, float* sh) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(kFull, v, off);
  if (lane == 0) sh[warp] = v;
  __syncthreads();
  float t = 0.f;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) t += sh[w];
  __syncthreads();
  return t;
}

}  // namespace vd
