// Host entry points of the prefill kernel (prefill_kernel.cuh); the INT8
// format's instances compile here, the SC4 format's in prefill_sc4.cu.
#include "prefill_kernel.cuh"

namespace archead {

int prefill_parts_per_vt() { return 4; }

extern template cudaError_t launch_prefill_fmt<true>(const archead_pack *, const void *, int, const uint16_t *, void *,
                                                     int, bool, const int32_t *, int, float2 *, float *, cudaStream_t);
template cudaError_t launch_prefill_fmt<false>(const archead_pack *, const void *, int, const uint16_t *, void *, int,
                                               bool, const int32_t *, int, float2 *, float *, cudaStream_t);

cudaError_t launch_prefill(const archead_pack *pk, const void *x, int M, const uint16_t *T, void *out, int out_fp32,
                           bool argmax, const int32_t *targets, int row0, float2 *ce_part, float *ce_tlogit,
                           cudaStream_t s) {
  return pk->sc4 ? launch_prefill_fmt<true>(pk, x, M, T, out, out_fp32, argmax, targets, row0, ce_part, ce_tlogit, s)
                 : launch_prefill_fmt<false>(pk, x, M, T, out, out_fp32, argmax, targets, row0, ce_part, ce_tlogit,
                                             s);
}

}  // namespace archead
