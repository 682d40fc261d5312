// vd_evict_norm.cu -- instantiates the fused eviction kernel and the short-cache
// kernel for one scoring rule (compiled separately so the translation units
// build in parallel).
#include "vd_evict.cuh"
#include "vd_small.cuh"

namespace vd {
const void* evict_kernel_norm(bool decode, bool holefill, bool fused) {
  const void* k[2][2][2] = {
      {{reinterpret_cast<const void*>(&evict_kernel<2, false, false, false>),
        reinterpret_cast<const void*>(&evict_kernel<2, false, false, true>)},
       {reinterpret_cast<const void*>(&evict_kernel<2, false, true, false>),
        reinterpret_cast<const void*>(&evict_kernel<2, false, true, true>)}},
      {{reinterpret_cast<const void*>(&evict_kernel<2, true, false, false>),
        reinterpret_cast<const void*>(&evict_kernel<2, true, false, true>)},
       {reinterpret_cast<const void*>(&evict_kernel<2, true, true, false>),
        reinterpret_cast<const void*>(&evict_kernel<2, true, true, true>)}}};
  return k[decode][holefill][fused];
}

const void* small_kernel_norm(bool decode, bool fused) {
  const void* k[2][2] = {
      {reinterpret_cast<const void*>(&small_evict_kernel<2, false, false>),
       reinterpret_cast<const void*>(&small_evict_kernel<2, false, true>)},
      {reinterpret_cast<const void*>(&small_evict_kernel<2, true, false>),
       reinterpret_cast<const void*>(&small_evict_kernel<2, true, true>)}};
  return k[decode][fused];
}

const void* score_kernel_norm() {
  return reinterpret_cast<const void*>(&evict_kernel<2, true, false, false, true>);
}
}  // namespace vd
