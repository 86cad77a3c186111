// Second pass of the fused cross-entropy epilogue (paper, Section 4: CE over
// held-out tokens, PPL = exp(CE)).  The forward kernels leave, per token and
// per slice of the vocabulary, the running maximum and the sum of
// exp(y - max) of the fp32 logits, plus the target's logit.  This kernel
// merges the slices in a fixed order and returns
//
//   ce[m] = max + log(sum) - y[m, t_m].
//
// Few tokens: one warp per token; lanes stride over the slices and the
// partial results are merged by a fixed butterfly.  Many tokens: a block per
// 32 tokens (lane = token, so the slice reads are coalesced); its 32 warps
// stride over the slices, eight loads in flight per lane, and are merged in
// warp order.  Both orders are
// fixed, so the result is deterministic.
#include "device.cuh"
#include "internal.h"

namespace archead {

__device__ __forceinline__ void ce_store(const LsePair &acc, int m, const float *__restrict__ tlogit,
                                         const int32_t *__restrict__ targets, int64_t V, float *__restrict__ ce,
                                         int *err) {
  const int32_t t = targets[m];
  if (t < 0 || (int64_t)t >= V) {
    ce[m] = __int_as_float(0x7fc00000);
    atomicOr(err, kErrTargetRange);
  } else {
    ce[m] = acc.m + logf(acc.s) - tlogit[m];
  }
}

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
  if (lane == 0) ce_store(acc, warp, tlogit, targets, V, ce, err);
}

constexpr int kCeWarps = 32;

__global__ void __launch_bounds__(kCeWarps * 32) ce_finalize_wide_kernel(const float2 *__restrict__ part, int num_parts,
                                                               const float *__restrict__ tlogit,
                                                               const int32_t *__restrict__ targets, int64_t V, int M,
                                                               float *__restrict__ ce, int *err) {
  __shared__ float2 red[kCeWarps][32];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int m = blockIdx.x * 32 + lane;
  LsePair acc{-INFINITY, 0.f};
  if (m < M) {
    int i = warp;
    for (; i + 7 * kCeWarps < num_parts; i += 8 * kCeWarps) {
      float2 v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) v[u] = part[(int64_t)(i + u * kCeWarps) * M + m];
#pragma unroll
      for (int u = 0; u < 8; ++u) acc = lse_merge(acc, LsePair{v[u].x, v[u].y});
    }
    for (; i < num_parts; i += kCeWarps) {
      const float2 v = part[(int64_t)i * M + m];
      acc = lse_merge(acc, LsePair{v.x, v.y});
    }
  }
  red[warp][lane] = make_float2(acc.m, acc.s);
  __syncthreads();
  if (warp != 0 || m >= M) return;
  for (int w = 1; w < kCeWarps; ++w) acc = lse_merge(acc, LsePair{red[w][lane].x, red[w][lane].y});
  ce_store(acc, m, tlogit, targets, V, ce, err);
}

// Greedy decoding: merge the per-slice (value, row) partials of each token in
// a fixed order (lanes over slices, then a fixed butterfly); ties keep the
// lowest row, so the result is the first maximum as in argmax.
__global__ void argmax_finalize_kernel(const float2 *__restrict__ part, int num_parts, int M,
                                       int32_t *__restrict__ index, float *__restrict__ value) {
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= M) return;
  float bv = -INFINITY;
  int bi = 0x7fffffff;
  for (int i = lane; i < num_parts; i += 32) {
    const float2 v = part[(int64_t)i * M + warp];
    const int vi = __float_as_int(v.y);
    if (v.x > bv || (v.x == bv && vi < bi)) {
      bv = v.x;
      bi = vi;
    }
  }
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, bv, off);
    const int oi = __shfl_xor_sync(0xffffffffu, bi, off);
    if (ov > bv || (ov == bv && oi < bi)) {
      bv = ov;
      bi = oi;
    }
  }
  if (lane == 0) {
    index[warp] = bi;
    if (value) value[warp] = bv;
  }
}

cudaError_t launch_argmax_finalize(const float2 *part, int num_parts, int M, int32_t *index, float *value,
                                   cudaStream_t s) {
  argmax_finalize_kernel<<<(M + 7) / 8, 256, 0, s>>>(part, num_parts, M, index, value);
  return cudaGetLastError();
}

cudaError_t launch_ce_finalize(const float2 *part, int num_parts, const float *tlogit, const int32_t *targets,
                               int64_t V, int M, float *ce, int *err, cudaStream_t s) {
  if (M >= 32) {
    ce_finalize_wide_kernel<<<(M + 31) / 32, kCeWarps * 32, 0, s>>>(part, num_parts, tlogit, targets, V, M, ce, err);
  } else {
    ce_finalize_kernel<<<(M + 7) / 8, 256, 0, s>>>(part, num_parts, tlogit, targets, V, M, ce, err);
  }
  return cudaGetLastError();
}

}  // namespace archead
