// vd_evict_l2.cu -- instantiates the fused eviction kernel for one scoring
// rule (compiled separately so the translation units build in parallel).
#include "vd_evict.cuh"

namespace vd {
const void* evict_kernel_l2(bool decode) {
  return decode ? reinterpret_cast<const void*>(&evict_kernel<0, true>)
                : reinterpret_cast<const void*>(&evict_kernel<0, false>);
}
}  // namespace vd
