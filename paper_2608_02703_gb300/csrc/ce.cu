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

// Where the merged (max, sum) of a token goes.  Whole head (row0 < 0):
// ce[m]; a target outside [0, V) gives NaN and latches kErrTargetRange.
// Vocabulary shard (row0 >= 0): out[3m .. 3m+2] = (max, sum, target logit),
// the target logit -inf when the target is not one of the shard's rows
// [row0, row0 + V) (another shard owns it; the combine checks the range).
__device__ __forceinline__ void ce_store(const LsePair &acc, int m, const float *__restrict__ tlogit,
                                         const int32_t *__restrict__ targets, int64_t row0, int64_t V,
                                         float *__restrict__ out, int *err) {
  const int64_t t = (int64_t)targets[m] - (row0 < 0 ? 0 : row0);
  const bool mine = t >= 0 && t < V;
  if (row0 >= 0) {
    out[3 * (int64_t)m] = acc.m;
    out[3 * (int64_t)m + 1] = acc.s;
    out[3 * (int64_t)m + 2] = mine ? tlogit[m] : -INFINITY;
  } else if (!mine) {
    out[m] = __int_as_float(0x7fc00000);
    atomicOr(err, kErrTargetRange);
  } else {
    out[m] = acc.m + logf(acc.s) - tlogit[m];
  }
}

__global__ void ce_finalize_kernel(const float2 *__restrict__ part, int num_parts, const float *__restrict__ tlogit,
                                   const int32_t *__restrict__ targets, int64_t row0, int64_t V, int M,
                                   float *__restrict__ ce, int *err) {
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
  if (lane == 0) ce_store(acc, warp, tlogit, targets, row0, V, ce, err);
}

constexpr int kCeWarps = 32;

__global__ void __launch_bounds__(kCeWarps * 32) ce_finalize_wide_kernel(const float2 *__restrict__ part, int num_parts,
                                                               const float *__restrict__ tlogit,
                                                               const int32_t *__restrict__ targets, int64_t row0,
                                                               int64_t V, int M, float *__restrict__ ce, int *err) {
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
  ce_store(acc, m, tlogit, targets, row0, V, ce, err);
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

static cudaError_t launch_finalize(const float2 *part, int num_parts, const float *tlogit, const int32_t *targets,
                                   int64_t row0, int64_t V, int M, float *out, int *err, cudaStream_t s) {
  if (M >= 32) {
    ce_finalize_wide_kernel<<<(M + 31) / 32, kCeWarps * 32, 0, s>>>(part, num_parts, tlogit, targets, row0, V, M, out,
                                                                    err);
  } else {
    ce_finalize_kernel<<<(M + 7) / 8, 256, 0, s>>>(part, num_parts, tlogit, targets, row0, V, M, out, err);
  }
  return cudaGetLastError();
}

cudaError_t launch_ce_finalize(const float2 *part, int num_parts, const float *tlogit, const int32_t *targets,
                               int64_t V, int M, float *ce, int *err, cudaStream_t s) {
  return launch_finalize(part, num_parts, tlogit, targets, -1, V, M, ce, err, s);
}

cudaError_t launch_lse_partial_finalize(const float2 *part, int num_parts, const float *tlogit,
                                        const int32_t *targets, int64_t row0, int64_t V, int M, float *parts3,
                                        cudaStream_t s) {
  return launch_finalize(part, num_parts, tlogit, targets, row0, V, M, parts3, nullptr, s);
}

// Combine of vocabulary shards (the paper's forward is row-separable, Eq. 7:
// each shard holds a contiguous block of rows).  Per token, the shards'
// (max, sum) pairs are merged in shard order and the target logit is taken
// from the one shard that owns the target:
//   ce[m] = max + log(sum) - y[m, t_m];
// NaN if no shard, or more than one, reports the target.
__global__ void lse_combine_kernel(const float *__restrict__ parts3, int num_shards, int M, float *__restrict__ ce) {
  const int m = blockIdx.x * blockDim.x + threadIdx.x;
  if (m >= M) return;
  LsePair acc{-INFINITY, 0.f};
  float t = 0.f;
  int owners = 0;
  for (int p = 0; p < num_shards; ++p) {
    const float *q = parts3 + ((int64_t)p * M + m) * 3;
    acc = lse_merge(acc, LsePair{q[0], q[1]});
    if (q[2] != -INFINITY) {
      t = q[2];
      ++owners;
    }
  }
  ce[m] = owners == 1 ? acc.m + logf(acc.s) - t : __int_as_float(0x7fc00000);
}

// Greedy output of vocabulary shards: the largest (value, global row) over
// the shards, lowest row on ties (global row = shard-local index + row0 of
// its shard).
__global__ void argmax_combine_kernel(const float *__restrict__ values, const int32_t *__restrict__ indices,
                                      const int32_t *__restrict__ row0, int num_shards, int M,
                                      int32_t *__restrict__ index, float *__restrict__ value) {
  const int m = blockIdx.x * blockDim.x + threadIdx.x;
  if (m >= M) return;
  float bv = -INFINITY;
  int bi = 0x7fffffff;
  for (int p = 0; p < num_shards; ++p) {
    const float v = values[(int64_t)p * M + m];
    const int i = indices[(int64_t)p * M + m] + row0[p];
    if (v > bv || (v == bv && i < bi)) {
      bv = v;
      bi = i;
    }
  }
  index[m] = bi;
  if (value) value[m] = bv;
}

cudaError_t launch_lse_combine(const float *parts3, int num_shards, int M, float *ce, cudaStream_t s) {
  lse_combine_kernel<<<(M + 255) / 256, 256, 0, s>>>(parts3, num_shards, M, ce);
  return cudaGetLastError();
}

cudaError_t launch_argmax_combine(const float *values, const int32_t *indices, const int32_t *row0, int num_shards,
                                  int M, int32_t *index, float *value, cudaStream_t s) {
  argmax_combine_kernel<<<(M + 255) / 256, 256, 0, s>>>(values, indices, row0, num_shards, M, index, value);
  return cudaGetLastError();
}

}  // namespace archead
