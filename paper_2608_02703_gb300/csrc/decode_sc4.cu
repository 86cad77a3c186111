// Decode kernel instances of the paper's packed format (SC4: 4-bit group-scale
// codes times a row scale), compiled apart from the INT8 ones.
#include "decode_kernel.cuh"

namespace archead {

template cudaError_t launch_decode_fmt<true>(const DecodeParams &, int, cudaStream_t, bool);

}  // namespace archead
