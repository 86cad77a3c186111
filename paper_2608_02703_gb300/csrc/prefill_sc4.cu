// Prefill kernel instances of the paper's packed format (SC4), compiled apart
// from the INT8 ones.
#include "prefill_kernel.cuh"

namespace archead {

template cudaError_t launch_prefill_fmt<true>(const archead_pack *, const void *, int, const uint16_t *, void *, int,
                                              bool, const int32_t *, int, float2 *, float *, cudaStream_t);

}  // namespace archead
