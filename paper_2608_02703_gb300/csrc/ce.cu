// Second pass of the fused cross-entropy epilogue (paper, Section 4: CE over
// held-out tokens, PPL = exp(CE)).  The forward kernels leave, per token and
// per slice of the vocabulary, the running maximum and the sum of
// exp(y - max) of the fp32 logits, plus the target's logit.  This kernel
// merges the slices in a fixed order and returns
//
//   ce[m] = max + log(sum) - y[m, t_m].
//
// One warp per token; lanes stride over the slices and the partial results
// are merged by a fixed butterfly, so the result is deterministic.
#include "device.cuh"
#include "internal.h"

namespace archead {

__global__ void ce_finalize_kernel(const float2 *__restrict__ part, int num_parts, const float *__restrict__ tlogit,
                                   const int32_t *__restrict__ targets, int64_t V, int M, float *__restrict__ ce,
                                   int *err) {
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= M) return;
  LsePair acc{-INFINITY, 0.f};
  for (int i = lane; i < num_parts; i += 32) {
    const float2 v = part[(int64_t)i * M + warp];
    acc = lse_merge(acc, LsePair{v.x, v.y});
  }
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    LsePair o{__shfl_xor_sync(0xffffffffu, acc.m, off), __shfl_xor_sync(0xffffffffu, acc.s, off)};
    acc = lse_merge(acc, o);
  }
  if (lane == 0) {
    const int32_t t = targets[warp];
    if (t < 0 || (int64_t)t >= V) {
      ce[warp] = __int_as_float(0x7fc00000);
      atomicOr(err, kErrTargetRange);
    } else {
      ce[warp] = acc.m + logf(acc.s) - tlogit[warp];
    }
  }
}

cudaError_t launch_ce_finalize(const float2 *part, int num_parts, const float *tlogit, const int32_t *targets,
                               int64_t V, int M, float *ce, int *err, cudaStream_t s) {
  const int blocks = (M + 7) / 8;
  ce_finalize_kernel<<<blocks, 256, 0, s>>>(part, num_parts, tlogit, targets, V, M, ce, err);
  return cudaGetLastError();
}

}  // namespace archead
