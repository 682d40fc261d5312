// vd_evict_l2.cu -- instantiates the fused eviction kernel for one scoring
// rule (compiled separately so the translation units build in parallel).
#include "vd_evict.cuh"

namespace vd {
const void* evict_kernel_l2(bool decode, bool holefill) {
  if (holefill)
    return decode ? reinterpret_cast<const void*>(&evict_kernel<0, true, true>)
                  : reinterpret_cast<const void*>(&evict_kernel<0, false, true>);
  return decode ? reinterpret_cast<const void*>(&evict_kernel<0, true, false>)
                : reinterpret_cast<const void*>(&evict_kernel<0, false, false>);
}
}  // namespace vd
