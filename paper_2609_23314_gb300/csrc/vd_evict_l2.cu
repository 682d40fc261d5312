// vd_evict_l2.cu -- instantiates the fused eviction kernel and the short-cache
// kernel for one scoring rule (compiled separately so the translation units
// build in parallel).
#include "vd_evict.cuh"
#include "vd_small.cuh"

namespace vd {
const void* evict_kernel_l2(bool decode, bool holefill, bool fused) {
  const void* k[2][2][2] = {
      {{reinterpret_cast<const void*>(&evict_kernel<0, false, false, false>),
        reinterpret_cast<const void*>(&evict_kernel<0, false, false, true>)},
       {reinterpret_cast<const void*>(&evict_kernel<0, false, true, false>),
        reinterpret_cast<const void*>(&evict_kernel<0, false, true, true>)}},
      {{reinterpret_cast<const void*>(&evict_kernel<0, true, false, false>),
        reinterpret_cast<const void*>(&evict_kernel<0, true, false, true>)},
       {reinterpret_cast<const void*>(&evict_kernel<0, true, true, false>),
        reinterpret_cast<const void*>(&evict_kernel<0, true, true, true>)}}};
  return k[decode][holefill][fused];
}

const void* small_kernel_l2(bool decode, bool fused) {
  const void* k[2][2] = {
      {reinterpret_cast<const void*>(&small_evict_kernel<0, false, false>),
       reinterpret_cast<const void*>(&small_evict_kernel<0, false, true>)},
      {reinterpret_cast<const void*>(&small_evict_kernel<0, true, false>),
       reinterpret_cast<const void*>(&small_evict_kernel<0, true, true>)}};
  return k[decode][fused];
}

const void* score_kernel_l2() {
  return reinterpret_cast<const void*>(&evict_kernel<0, true, false, false, true>);
}
}  // namespace vd
