// Rank-r pre-pass (paper, Section 3.2, Eq. 7: the correction is evaluated as
// (H B_w^T) A_w^T, i.e. the d-side product first).  For every token m and
// extended rank column kk it computes, in fp32 from exact products,
//
//   core:        t[m,kk] = su[kk] sv[kk] sum_k x[m,k] qv[k,kk]          (kk < r_c)
//   correction:  t[m,kk] = sum_k sb[k/g,j] x[m,k] qb[k,j]   (kk = RCP + j, j < r_r)
//
// then splits t into bf16 hi + lo (hi = bf16(t), lo = bf16(t - hi)) so the
// tensor-core kernels can apply the rank-r branches with exact int8 codes of
// A_c and A_w as the other operand.  Outputs: the decode kernel's B-fragment
// layout of (hi, lo) per 16-token chunk, and/or the prefill kernel's row-major
// extended operand T = [hi_core | lo_core | hi_corr | lo_corr].
//
// Grid: (32 extended columns, 16 tokens, 256-wide split of d).  In a block,
// warp w takes the 32-wide slice w of its split (a slice never straddles a
// quantisation group, g >= 32), lane = column (core or correction: RCP is a
// multiple of 16, so a block may hold both); a slice's partial sums are
// scaled by their group scale.  The eight warps' sums are added in a fixed
// order and written per split; the last block of a (columns, tokens) pair to
// finish adds the splits in split order and finalises (deterministic).
#include "device.cuh"
#include "internal.h"

namespace archead {

constexpr int kPreTok = 16;    // tokens per block
constexpr int kPreCols = 32;   // extended columns per block
constexpr int kPreChunk = 256; // d per staged chunk of x

__device__ __forceinline__ uint16_t f32_to_bf16_bits(float v) {
  return __bfloat16_as_ushort(__float2bfloat16_rn(v));
}

// Shared memory of one block for mt tokens: the staged x chunk [256][mt+1]
// (floats, token fastest) and, after it is consumed, the per-warp sums
// [8][mt][32] in the same space.
__host__ __device__ __forceinline__ size_t prepass_smem_bytes(int mt) {
  const size_t xs = (size_t)kPreChunk * (mt + 1) * 4;
  const size_t red = (size_t)8 * mt * kPreCols * 4;
  return xs > red ? xs : red;
}

__global__ void __launch_bounds__(256) prepass_kernel(PrepassParams p) {
  // Let the dependent forward kernel start streaming while this one runs; it
  // waits for this grid's results before it reads them.
  asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
  extern __shared__ float pre_smem[];
  __shared__ int last_block;
  const int c0 = blockIdx.x * kPreCols;
  const int m0 = blockIdx.y * kPreTok;
  const int k0 = blockIdx.z * kPreChunk;
  const int nsplit = gridDim.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const bool core = c0 + lane < p.rcp;  // a block may hold core and correction columns
  const int j = core ? c0 + lane : c0 + lane - p.rcp;
  const bool valid = core ? j < p.rc : j < p.rr;
  const int8_t *q = core ? p.q_v : p.q_b;
  const int ldq = core ? p.rc : p.rr;
  const int mt = min(kPreTok, p.M - m0);
  const int ms = mt + 1;  // row stride of the staged x
  const int kn = min(kPreChunk, p.d - k0);  // d is a multiple of 64
  float *xs = pre_smem;

  for (int e = threadIdx.x; e < kPreChunk * mt; e += blockDim.x) {
    const int m = e / kPreChunk, k = e % kPreChunk;
    xs[k * ms + m] = k < kn ? bf16_lo(p.x[(int64_t)(m0 + m) * p.d + k0 + k]) : 0.f;
  }
  __syncthreads();
  float tot[kPreTok];
#pragma unroll
  for (int m = 0; m < kPreTok; ++m) tot[m] = 0.f;
  const int sl = warp * 32;
  if (sl < kn) {
    float qv[32];  // the slice's codes of this column, loaded before use
#pragma unroll
    for (int kk = 0; kk < 32; ++kk) qv[kk] = valid ? (float)q[(int64_t)(k0 + sl + kk) * ldq + j] : 0.f;
#pragma unroll
    for (int kk = 0; kk < 32; ++kk) {
#pragma unroll
      for (int m = 0; m < kPreTok; ++m)
        if (m < mt) tot[m] = fmaf(xs[(sl + kk) * ms + m], qv[kk], tot[m]);
    }
    const float sc = (core || !valid) ? 1.f : fp16_bits_to_f32(p.s_b[((k0 + sl) / p.g) * p.rr + j]);
#pragma unroll
    for (int m = 0; m < kPreTok; ++m) tot[m] *= sc;
  }
  __syncthreads();  // x consumed: the space now holds the per-warp sums
  float *red = pre_smem;
#pragma unroll
  for (int m = 0; m < kPreTok; ++m)
    if (m < mt) red[(warp * mt + m) * kPreCols + lane] = tot[m];
  __syncthreads();
  const int64_t pair = (int64_t)blockIdx.y * gridDim.x + blockIdx.x;
  float *mine = p.partial + ((int64_t)blockIdx.z * gridDim.y * gridDim.x + pair) * (kPreTok * kPreCols);
  for (int e = threadIdx.x; e < kPreTok * kPreCols; e += blockDim.x) {
    const int m = e / kPreCols, c = e % kPreCols;
    float t = 0.f;
    if (m < mt) {
#pragma unroll
      for (int w = 0; w < 8; ++w) t += red[(w * mt + m) * kPreCols + c];
    }
    mine[e] = t;
  }
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) {
    const int done = atomicAdd(&p.counters[pair], 1);
    last_block = done == nsplit - 1;
  }
  __syncthreads();
  if (!last_block) return;
  __threadfence();

  for (int e = threadIdx.x; e < kPreTok * kPreCols; e += blockDim.x) {
    const int m = e / kPreCols, c = e % kPreCols;
    // Tokens past M in this 16-token chunk get zero fragments.
    if (m >= mt && !p.ts) continue;
    float t = 0.f;
    if (m < mt) {
      // Eight loads in flight, added in split order.
      const float *src = p.partial + (int64_t)pair * (kPreTok * kPreCols) + e;
      const int64_t step = (int64_t)gridDim.y * gridDim.x * (kPreTok * kPreCols);
      int sp = 0;
      for (; sp + 8 <= nsplit; sp += 8) {
        float v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) v[u] = __ldcg(src + (sp + u) * step);
#pragma unroll
        for (int u = 0; u < 8; ++u) t += v[u];
      }
      for (; sp < nsplit; ++sp) t += __ldcg(src + sp * step);
    }
    const int kk = c0 + c;
    if (kk < p.rcp) {
      t = kk < p.rc ? t * fp16_bits_to_f32(p.s_v[kk]) * fp16_bits_to_f32(p.s_u[kk]) : 0.f;
    } else if (kk - p.rcp >= p.rr) {
      t = 0.f;
    }
    const uint16_t hi = f32_to_bf16_bits(t);
    const uint16_t lo = f32_to_bf16_bits(t - bf16_lo(hi));
    const int mg = m0 + m;
    if (p.T && m < mt) {
      uint16_t *row = p.T + (int64_t)mg * (2 * p.lr);
      if (kk < p.rcp) {
        row[kk] = hi;
        row[p.rcp + kk] = lo;
      } else {
        const int jj = kk - p.rcp;
        row[2 * p.rcp + jj] = hi;
        row[2 * p.rcp + p.rrp + jj] = lo;
      }
    }
    // Column of the decode layout: the same as kk, or with core and
    // correction back to back (core columns as they are, correction ones
    // after the r_c core ones, and the core's padding columns, whose t is
    // zero, moved past the correction to zero the rest of the last step).
    const int pos = !p.ts_compact ? kk : kk < p.rc ? kk : kk < p.rcp ? kk + p.rr : p.ts_core + (kk - p.rcp);
    if (p.ts && pos < 16 * p.ts_nls) {
      // B-fragment of step ls: register (k16 >= 8), lane = 4*(token%8) + (k16%8)/2.
      const int chunk = mg / kDecodeMaxTokens, nl = mg % kDecodeMaxTokens;
      const int nt = nl >> 3, gq = nl & 7;
      const int ls = pos >> 4, k16 = pos & 15;
      const int reg = k16 >> 3, cq = (k16 & 7) >> 1, h = k16 & 1;
      const int ln = gq * 4 + cq;
      uint16_t *ts16 = reinterpret_cast<uint16_t *>(p.ts);
      const int64_t base = ((((int64_t)chunk * p.ts_nls + ls) * 2) * 2 + nt) * 32 + ln;  // hl = 0
      ts16[base * 4 + reg * 2 + h] = hi;
      ts16[(base + 2 * 32) * 4 + reg * 2 + h] = lo;  // hl = 1
    }
  }
  if (threadIdx.x == 0) p.counters[pair] = 0;  // ready for the next call
}

// ---------------------------------------------------------------------------
// Tensor-core pre-pass for many tokens (prefill).  Same t as above, written
// only to the row-major operand T.  Block: 64 tokens x 32 extended columns,
// the whole of d (no split, so no partial sums and no counters); warp w takes
// tokens 16w..16w+15 with mma.sync m16n8k16 (bf16 in, fp32 accumulate) over
// 128-wide chunks of d staged in shared memory by cp.async (double buffer;
// at 52 KB a block, four blocks share an SM and a 4096-token call is one wave).
// A = x rows, B = lr_t rows (the extended column's int8 codes as bf16).  In
// a correction block the accumulators are scaled by s_b at the end of every
// quantisation group and added to running sums; a core block scales once by
// s_u s_v at the end.
// ---------------------------------------------------------------------------
constexpr int kPtTok = 64;
constexpr int kPtCols = 32;
constexpr int kPtK = 128;
constexpr int kPtStride = kPtK + 8;  // bf16 per staged row: conflict-free fragment loads
constexpr int kPtStages = 2;
constexpr int kPtSmem = kPtStages * (kPtTok + kPtCols) * kPtStride * 2;

__device__ __forceinline__ void cp_async16(void *dst, const void *src, bool valid) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(smem_u32(dst)), "l"(src),
               "r"(valid ? 16 : 0)
               : "memory");
}

__global__ void __launch_bounds__(128) prepass_t_kernel(PrepassParams p, const uint16_t *__restrict__ lr_t,
                                                        int d_pad) {
  extern __shared__ __align__(16) uint16_t pt_smem[];
  uint16_t *xs = pt_smem;                                    // [stages][64][kPtStride]
  uint16_t *bs = pt_smem + kPtStages * kPtTok * kPtStride;   // [stages][32][kPtStride]
  const int c0 = blockIdx.x * kPtCols;
  const int m0 = blockIdx.y * kPtTok;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gq = lane >> 2, cq = lane & 3;
  // Eight-column slice n of the block is core (< RCP, a multiple of 16) or correction.
  auto core_n = [&](int n) { return c0 + n * 8 < p.rcp; };
  const int nchunks = d_pad / kPtK;

  auto stage = [&](int kc, int buf) {
    const int k0 = kc * kPtK;
    // x: 64 rows x 16 pieces of 16 bytes; tokens past M and k past d read as zero.
    for (int i = threadIdx.x; i < kPtTok * 16; i += blockDim.x) {
      const int r = i >> 4, c = i & 15;
      const int m = m0 + r, k = k0 + c * 8;
      const bool ok = m < p.M && k < p.d;
      cp_async16(xs + (buf * kPtTok + r) * kPtStride + c * 8, ok ? p.x + (int64_t)m * p.d + k : p.x, ok);
    }
    for (int i = threadIdx.x; i < kPtCols * 16; i += blockDim.x) {
      const int r = i >> 4, c = i & 15;
      cp_async16(bs + (buf * kPtCols + r) * kPtStride + c * 8, lr_t + (int64_t)(c0 + r) * d_pad + k0 + c * 8, true);
    }
    asm volatile("cp.async.commit_group;\n" ::: "memory");
  };

  float acc[4][4], run[4][4];
#pragma unroll
  for (int n = 0; n < 4; ++n)
#pragma unroll
    for (int i = 0; i < 4; ++i) acc[n][i] = run[n][i] = 0.f;

  // Chunk c is cp.async group c: kPtStages-1 are committed up front and one
  // (maybe empty) per iteration, after the wait, so when iteration kc waits
  // the newest kPtStages-2 groups are later chunks and waiting for all but
  // those completes chunk kc.  The barrier after the wait also guarantees
  // that every warp is done with chunk kc-1, whose buffer is restaged next.
  for (int kc = 0; kc < kPtStages - 1; ++kc) {
    if (kc < nchunks) stage(kc, kc);
    else asm volatile("cp.async.commit_group;\n" ::: "memory");
  }
  for (int kc = 0; kc < nchunks; ++kc) {
    const int buf = kc % kPtStages;
    asm volatile("cp.async.wait_group %0;\n" ::"n"(kPtStages - 2) : "memory");
    __syncthreads();
    if (kc + kPtStages - 1 < nchunks) stage(kc + kPtStages - 1, (kc + kPtStages - 1) % kPtStages);
    else asm volatile("cp.async.commit_group;\n" ::: "memory");
    const uint16_t *xa = xs + (buf * kPtTok + warp * 16) * kPtStride;
    const uint16_t *xb = bs + buf * kPtCols * kPtStride;
#pragma unroll
    for (int ks = 0; ks < kPtK / 16; ++ks) {
      const int kb = ks * 16 + 2 * cq;
      uint32_t a[4];
      a[0] = *reinterpret_cast<const uint32_t *>(xa + gq * kPtStride + kb);
      a[1] = *reinterpret_cast<const uint32_t *>(xa + (gq + 8) * kPtStride + kb);
      a[2] = *reinterpret_cast<const uint32_t *>(xa + gq * kPtStride + kb + 8);
      a[3] = *reinterpret_cast<const uint32_t *>(xa + (gq + 8) * kPtStride + kb + 8);
#pragma unroll
      for (int n = 0; n < 4; ++n) {
        const uint16_t *br = xb + (n * 8 + gq) * kPtStride + kb;
        mma_bf16_16816(acc[n], a, *reinterpret_cast<const uint32_t *>(br), *reinterpret_cast<const uint32_t *>(br + 8));
      }
      // End of a quantisation group of the correction factor: apply s_b to
      // the correction slices (core slices keep accumulating).
      const int kend = kc * kPtK + ks * 16 + 16;
      if (kend % p.g == 0) {
        const int grp = kend / p.g - 1;
#pragma unroll
        for (int n = 0; n < 4; ++n) {
          if (core_n(n)) continue;
          if (grp < p.d / p.g) {
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              const int j = c0 - p.rcp + n * 8 + 2 * cq + h;
              const float sb = j < p.rr ? fp16_bits_to_f32(p.s_b[(int64_t)grp * p.rr + j]) : 0.f;
              run[n][h] = fmaf(sb, acc[n][h], run[n][h]);
              run[n][2 + h] = fmaf(sb, acc[n][2 + h], run[n][2 + h]);
            }
          }
#pragma unroll
          for (int i = 0; i < 4; ++i) acc[n][i] = 0.f;
        }
      }
    }
  }

  // t for (token, column) pairs of this lane, then the bf16 hi/lo split.
#pragma unroll
  for (int n = 0; n < 4; ++n) {
    const bool core = core_n(n);
#pragma unroll
    for (int rh = 0; rh < 2; ++rh) {
      const int m = m0 + warp * 16 + gq + 8 * rh;
      if (m >= p.M) continue;
      uint32_t hi2 = 0, lo2 = 0;
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int kk = c0 + n * 8 + 2 * cq + h;
        float t;
        if (core) {
          t = kk < p.rc ? acc[n][2 * rh + h] * fp16_bits_to_f32(p.s_v[kk]) * fp16_bits_to_f32(p.s_u[kk]) : 0.f;
        } else {
          t = kk - p.rcp < p.rr ? run[n][2 * rh + h] : 0.f;
        }
        const uint16_t hi = f32_to_bf16_bits(t);
        const uint16_t lo = f32_to_bf16_bits(t - bf16_lo(hi));
        hi2 |= (uint32_t)hi << (16 * h);
        lo2 |= (uint32_t)lo << (16 * h);
      }
      const int kk = c0 + n * 8 + 2 * cq;
      uint16_t *row = p.T + (int64_t)m * (2 * p.lr);
      const int hi_col = core ? kk : p.rcp + kk;                 // = 2 rcp + j for the correction
      const int lo_col = core ? p.rcp + kk : p.rcp + p.rrp + kk;  // = 2 rcp + rrp + j
      *reinterpret_cast<uint32_t *>(row + hi_col) = hi2;
      *reinterpret_cast<uint32_t *>(row + lo_col) = lo2;
    }
  }
}

cudaError_t launch_prepass_t(const PrepassParams &pp, const uint16_t *lr_t, int d_pad, cudaStream_t s,
                             archead_pack *pk) {
  if (pp.lr == 0) return cudaSuccess;
  cudaEvent_t ev = nullptr;
  timer_begin(pk, "prepass", s, &ev);
  cudaError_t e = opt_in_smem(reinterpret_cast<const void *>(prepass_t_kernel), kPtSmem);
  if (e != cudaSuccess) return e;
  dim3 grid(pp.lr / kPtCols, (pp.M + kPtTok - 1) / kPtTok);
  prepass_t_kernel<<<grid, 128, kPtSmem, s>>>(pp, lr_t, d_pad);
  timer_end(pk, "prepass", s, ev);
  return cudaGetLastError();
}

int prepass_pairs(int M, int lr) { return (lr / kPreCols) * ((M + kPreTok - 1) / kPreTok); }

size_t prepass_partial_bytes(int M, int lr, int d) {
  return (size_t)prepass_pairs(M, lr) * ((d + kPreChunk - 1) / kPreChunk) * kPreTok * kPreCols * sizeof(float);
}

size_t prepass_smem(int M) { return prepass_smem_bytes(M < kPreTok ? M : kPreTok); }

cudaError_t launch_prepass(const PrepassParams &pp, cudaStream_t s, archead_pack *pk) {
  if (pp.lr == 0) return cudaSuccess;
  cudaEvent_t ev = nullptr;
  timer_begin(pk, "prepass", s, &ev);
  dim3 grid(pp.lr / kPreCols, (pp.M + kPreTok - 1) / kPreTok, (pp.d + kPreChunk - 1) / kPreChunk);
  const size_t smem = prepass_smem(pp.M);
  if (smem > 48 * 1024) {
    cudaError_t e = opt_in_smem(reinterpret_cast<const void *>(prepass_kernel), (int)smem);
    if (e != cudaSuccess) return e;
  }
  prepass_kernel<<<grid, 256, smem, s>>>(pp);
  timer_end(pk, "prepass", s, ev);
  return cudaGetLastError();
}

}  // namespace archead
