// vd_evict_dir.cu -- instantiates the fused eviction kernel and the short-cache
// kernel for one scoring rule (compiled separately so the translation units
// build in parallel).
#include "vd_evict.cuh"
#include "vd_small.cuh"

namespace vd {
const void* evict_kernel_dir(bool decode, bool holefill, bool fused) {
  const void* k[2][2][2] = {
      {{reinterpret_cast<const void*>(&evict_kernel<1, false, false, false>),
        reinterpret_cast<const void*>(&evict_kernel<1, false, false, true>)},
       {reinterpret_cast<const void*>(&evict_kernel<1, false, true, false>),
        reinterpret_cast<const void*>(&evict_kernel<1, false, true, true>)}},
      {{reinterpret_cast<const void*>(&evict_kernel<1, true, false, false>),
        reinterpret_cast<const void*>(&evict_kernel<1, true, false, true>)},
       {reinterpret_cast<const void*>(&evict_kernel<1, true, true, false>),
        reinterpret_cast<const void*>(&evict_kernel<1, true, true, true>)}}};
  return k[decode][holefill][fused];
}

const void* small_kernel_dir(bool decode, bool fused) {
  const void* k[2][2] = {
      {reinterpret_cast<const void*>(&small_evict_kernel<1, false, false>),
       reinterpret_cast<const void*>(&small_evict_kernel<1, false, true>)},
      {reinterpret_cast<const void*>(&small_evict_kernel<1, true, false>),
       reinterpret_cast<const void*>(&small_evict_kernel<1, true, true>)}};
  return k[decode][fused];
}

const void* score_kernel_dir() {
  return reinterpret_cast<const void*>(&evict_kernel<1, true, false, false, true>);
}
}  // namespace vd
