// Rank-r pre-pass (paper, Section 3.2, Eq. 7: the correction is evaluated as
// (H B_w^T) A_w^T, i.e. the d-side product first).  For every token m and
// extended rank column kk it computes, in fp32 from exact products,
//
//   core:        t[m,kk] = su[kk] sv[kk] sum_k x[m,k] qv[k,kk]          (kk < r_c)
//   correction:  t[m,kk] = sum_groups sb[grp,j] sum_{k in grp} x[m,k] qb[k,j]
//                                                       (kk = RCP + j, j < r_r)
//
// then splits t into bf16 hi + lo (hi = bf16(t), lo = bf16(t - hi)) so the
// tensor-core kernels can apply the rank-r branches with exact int8 codes of
// A_c and A_w as the other operand.  It also lays out the bf16 hidden states
// as m16n8k16 B-fragments for the decode kernel.
#include "device.cuh"
#include "internal.h"

namespace archead {

constexpr int kPreTok = 16;   // tokens per block
constexpr int kPreCols = 32;  // extended rank columns per block

// grid: (ceil(M/16), LR/32, d/256); 256 threads = 16 tokens x 16 column pairs.
__global__ void __launch_bounds__(256) prepass_partial_kernel(PrepassParams p) {
  __shared__ float xs[kPreTok][kPrepassKSplit + 1];
  __shared__ int8_t qs[kPrepassKSplit][kPreCols];
  const int m0 = blockIdx.x * kPreTok;
  const int c0 = blockIdx.y * kPreCols;
  const int k0 = blockIdx.z * kPrepassKSplit;
  const bool core = c0 < p.rcp;  // a 32-column block never straddles the core/correction boundary
  const int kn = min(kPrepassKSplit, p.d - k0);  // d is a multiple of 64, not necessarily of 256
  for (int e = threadIdx.x; e < kPreTok * kPrepassKSplit; e += blockDim.x) {
    const int m = e / kPrepassKSplit, k = e % kPrepassKSplit;
    float v = 0.f;
    if (m0 + m < p.M && k < kn) v = bf16_lo(p.x[(int64_t)(m0 + m) * p.d + k0 + k]);
    xs[m][k] = v;
  }
  for (int e = threadIdx.x; e < kPrepassKSplit * kPreCols; e += blockDim.x) {
    const int k = e / kPreCols, c = e % kPreCols;
    int8_t q = 0;
    if (k >= kn) {
    } else if (core) {
      const int j = c0 + c;
      if (j < p.rc) q = p.q_v[(int64_t)(k0 + k) * p.rc + j];
    } else {
      const int j = c0 + c - p.rcp;
      if (j < p.rr) q = p.q_b[(int64_t)(k0 + k) * p.rr + j];
    }
    qs[k][c] = q;
  }
  __syncthreads();
  const int m = threadIdx.x / 16;
  const int cp = (threadIdx.x % 16) * 2;
  float tot0 = 0.f, tot1 = 0.f, part0 = 0.f, part1 = 0.f;
  const int jb = c0 + cp - p.rcp;  // correction column of cp (when !core)
  for (int k = 0; k < kn; ++k) {
    const float xv = xs[m][k];
    part0 = fmaf(xv, (float)qs[k][cp], part0);
    part1 = fmaf(xv, (float)qs[k][cp + 1], part1);
    if (((k0 + k + 1) % p.g) == 0) {
      if (core) {
        tot0 += part0;
        tot1 += part1;
      } else {
        const int grp = (k0 + k) / p.g;
        const float s0 = jb < p.rr ? fp16_bits_to_f32(p.s_b[grp * p.rr + jb]) : 0.f;
        const float s1 = jb + 1 < p.rr ? fp16_bits_to_f32(p.s_b[grp * p.rr + jb + 1]) : 0.f;
        tot0 = fmaf(s0, part0, tot0);
        tot1 = fmaf(s1, part1, tot1);
      }
      part0 = part1 = 0.f;
    }
  }
  if (core) {  // groups may be wider than the 256-wide split
    tot0 += part0;
    tot1 += part1;
  }  // correction groups never straddle a split: 256 is a multiple of g and d of g
  if (m0 + m < p.M) {
    float *dst = p.partial + ((int64_t)blockIdx.z * p.M + m0 + m) * p.lr + c0 + cp;
    dst[0] = tot0;
    dst[1] = tot1;
  }
}

__device__ __forceinline__ uint16_t f32_to_bf16_bits(float v) {
  return __bfloat16_as_ushort(__float2bfloat16_rn(v));
}

// One thread per (token, extended column): sum the d-splits in a fixed order,
// apply the core scales, split into bf16 hi/lo and scatter to both layouts.
__global__ void prepass_finalize_kernel(PrepassParams p, int nsplit) {
  const int64_t total = (int64_t)p.M * p.lr;
  const int nls = p.lr / 16;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
    const int m = (int)(e / p.lr);
    const int kk = (int)(e % p.lr);
    float t = 0.f;
    for (int s = 0; s < nsplit; ++s) t += p.partial[((int64_t)s * p.M + m) * p.lr + kk];
    if (kk < p.rcp) {
      t = kk < p.rc ? t * fp16_bits_to_f32(p.s_v[kk]) * fp16_bits_to_f32(p.s_u[kk]) : 0.f;
    } else if (kk - p.rcp >= p.rr) {
      t = 0.f;
    }
    const uint16_t hi = f32_to_bf16_bits(t);
    const uint16_t lo = f32_to_bf16_bits(t - bf16_lo(hi));
    if (p.T) {
      uint16_t *row = p.T + (int64_t)m * (2 * p.lr);
      if (kk < p.rcp) {
        row[kk] = hi;
        row[p.rcp + kk] = lo;
      } else {
        const int j = kk - p.rcp;
        row[2 * p.rcp + j] = hi;
        row[2 * p.rcp + p.rrp + j] = lo;
      }
    }
    if (p.ts) {
      // B-fragment of step ls: register (k16 >= 8), lane = 4*(token%8) + (k16%8)/2.
      const int chunk = m / kDecodeMaxTokens, nl = m % kDecodeMaxTokens;
      const int nt = nl >> 3, gq = nl & 7;
      const int ls = kk >> 4, k16 = kk & 15;
      const int reg = k16 >> 3, cq = (k16 & 7) >> 1, h = k16 & 1;
      const int lane = gq * 4 + cq;
      uint16_t *ts16 = reinterpret_cast<uint16_t *>(p.ts);
      const int64_t base = ((((int64_t)chunk * nls + ls) * 2) * 2 + nt) * 32 + lane;  // hl = 0
      const int64_t hl_stride = 2 * 32;                                                // (nt, lane)
      ts16[(base) * 4 + reg * 2 + h] = hi;
      ts16[(base + hl_stride) * 4 + reg * 2 + h] = lo;
    }
  }
}

// Decode x-fragments: xs[chunk][nt][p][lane][4 words]; word w4 of step pair p
// is register (w4 & 1) of k16-step 2p + (w4 >> 1) for token 16*chunk + 8*nt + lane/4.
__global__ void build_xs_kernel(const uint16_t *__restrict__ x, uint32_t *__restrict__ xs, int M, int d) {
  const int nchunks = (M + kDecodeMaxTokens - 1) / kDecodeMaxTokens;
  const int64_t per_chunk = (int64_t)2 * (d / 32) * 32 * 4;
  const int64_t total = nchunks * per_chunk;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
    const int w4 = (int)(e & 3);
    const int lane = (int)((e >> 2) & 31);
    const int64_t rest = e >> 7;
    const int pp = (int)(rest % (d / 32));
    const int nt = (int)((rest / (d / 32)) % 2);
    const int chunk = (int)(rest / (2 * (d / 32)));
    const int s = 2 * pp + (w4 >> 1), reg = w4 & 1;
    const int n = chunk * kDecodeMaxTokens + nt * 8 + (lane >> 2);
    const int k = 16 * s + 2 * (lane & 3) + 8 * reg;
    uint32_t v = 0;
    if (n < M) v = *reinterpret_cast<const uint32_t *>(x + (int64_t)n * d + k);
    xs[e] = v;
  }
}

cudaError_t launch_prepass(const PrepassParams &pp, cudaStream_t s, archead_pack *pk) {
  const int nsplit = (pp.d + kPrepassKSplit - 1) / kPrepassKSplit;
  cudaEvent_t ev = nullptr;
  if (pp.lr > 0) {
    timer_begin(pk, "prepass_partial", s, &ev);
    dim3 grid((pp.M + kPreTok - 1) / kPreTok, pp.lr / kPreCols, nsplit);
    prepass_partial_kernel<<<grid, 256, 0, s>>>(pp);
    timer_end(pk, "prepass_partial", s, ev);
    if (pp.ts) {
      const int nchunks = (pp.M + kDecodeMaxTokens - 1) / kDecodeMaxTokens;
      cudaError_t e = cudaMemsetAsync(pp.ts, 0, (size_t)nchunks * (pp.lr / 16) * 1024, s);
      if (e != cudaSuccess) return e;
    }
    timer_begin(pk, "prepass_finalize", s, &ev);
    const int64_t total = (int64_t)pp.M * pp.lr;
    int64_t blocks = (total + 255) / 256;
    if (blocks > 4096) blocks = 4096;
    prepass_finalize_kernel<<<(unsigned)blocks, 256, 0, s>>>(pp, nsplit);
    timer_end(pk, "prepass_finalize", s, ev);
  }
  if (pp.xs) {
    timer_begin(pk, "build_xs", s, &ev);
    const int nchunks = (pp.M + kDecodeMaxTokens - 1) / kDecodeMaxTokens;
    const int64_t total = (int64_t)nchunks * 2 * pp.d * 4;
    int64_t blocks = (total + 255) / 256;
    if (blocks > 4096) blocks = 4096;
    build_xs_kernel<<<(unsigned)blocks, 256, 0, s>>>(pp.x, pp.xs, pp.M, pp.d);
    timer_end(pk, "build_xs", s, ev);
  }
  return cudaGetLastError();
}

}  // namespace archead
