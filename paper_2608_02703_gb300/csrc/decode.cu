// Memory-bound decode kernel (M <= 16 tokens) of the packed LM-head forward
// (paper, Section 3.2, Eq. 7; Appendix B "At inference ... core path and
// correction path separately").
//
// Persistent grid, one block per SM.  A unit of work is 256 vocabulary rows
// (two 128-row tiles).  One producer warp streams each unit's INT4 codes,
// group scales and low-rank codes with 1-D bulk TMA copies into a ring of
// shared-memory stages (mbarrier full/empty pairs).  Eight consumer warps each
// own two 16-row m-tiles.  Per 16-wide k step a consumer converts one 32-bit
// word of offset-binary nibbles into the four bf16 A-fragment registers of an
// m16n8k16 MMA (exact small integers) and multiplies them with the bf16
// hidden states (B fragments, tokens on the 8-wide side) held in shared
// memory, accumulating in fp32.  At the end of every quantisation group the
// partial sums are promoted by that row's group scale in fp32.  The rank-r
// branches follow as extra k steps: int8 codes of A_c (core) or A_w
// (correction) times the bf16 hi/lo split of t = x V (pre-pass), the
// correction promoted by the row scale of A_w.
#include "device.cuh"
#include "internal.h"

namespace archead {

constexpr int kDecConsumerWarps = 8;
constexpr int kDecThreads = (kDecConsumerWarps + 1) * 32;
constexpr int kDecStageCodeBytes = 2 * 2 * kChunkBytes;  // 2 tiles x 2 chunks (128 of d)
constexpr int kDecStageScaleBytes = 2 * 4 * kTileRows * 2;  // 2 tiles x up to 4 groups
constexpr int kDecStageBytes = kDecStageCodeBytes + kDecStageScaleBytes;
constexpr int kDecLrStepsPerStage = 4;
constexpr int kSmemLimit = 227 * 1024;

struct DecodeSmemPlan {
  int stages;
  size_t xs_off, ts_off, bar_off, total;
};

static DecodeSmemPlan decode_plan(int d, int nls, int NT) {
  DecodeSmemPlan pl{};
  const size_t xs_bytes = (size_t)NT * 16 * d;
  const size_t ts_bytes = (size_t)nls * 1024;
  const size_t fixed = xs_bytes + ts_bytes + 256;
  int st = 4;
  while (st >= 2 && fixed + (size_t)st * kDecStageBytes > (size_t)kSmemLimit) --st;
  pl.stages = st;
  pl.xs_off = (size_t)st * kDecStageBytes;
  pl.ts_off = pl.xs_off + xs_bytes;
  pl.bar_off = pl.ts_off + ts_bytes;
  pl.total = pl.bar_off + 256;
  return pl;
}

template <int NT>
__global__ void __launch_bounds__(kDecThreads, 1) decode_kernel(DecodeParams p, int stages, int xs_off, int ts_off,
                                                                int bar_off) {
  extern __shared__ __align__(1024) uint8_t smem[];
  uint8_t *stage_base = smem;
  const uint32_t *xs_s = reinterpret_cast<const uint32_t *>(smem + xs_off);
  const uint32_t *ts_s = reinterpret_cast<const uint32_t *>(smem + ts_off);
  uint64_t *full = reinterpret_cast<uint64_t *>(smem + bar_off);
  uint64_t *empty = full + 4;
  uint64_t *xbar = full + 8;
  volatile int *abort_flag = reinterpret_cast<volatile int *>(full + 9);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int KC = p.d / kChunkK;
  const int res_stages = (KC + 1) / 2;
  const int lr_stages = (p.nls + kDecLrStepsPerStage - 1) / kDecLrStepsPerStage;
  const int num_units = (p.num_tiles + 1) / 2;

  if (threadIdx.x == 0) {
    for (int i = 0; i < stages; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], kDecConsumerWarps);
    }
    mbar_init(xbar, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();

  if (warp == kDecConsumerWarps) {
    // ---------------- producer warp ----------------
    if (lane != 0) return;
    const uint32_t xs_bytes = (uint32_t)(NT * 16 * p.d);
    const uint32_t ts_bytes = (uint32_t)(p.nls * 1024);
    mbar_arrive_expect_tx(xbar, xs_bytes + ts_bytes);
    bulk_g2s(smem + xs_off, p.xs, xs_bytes, xbar);
    if (ts_bytes) bulk_g2s(smem + ts_off, p.ts, ts_bytes, xbar);
    int it = 0;
    for (int unit = blockIdx.x; unit < num_units; unit += gridDim.x) {
      const int ntile = min(2, p.num_tiles - 2 * unit);
      for (int s = 0; s < res_stages + lr_stages; ++s, ++it) {
        const int st = it % stages;
        const uint32_t ph = (it / stages) & 1;
        if (!mbar_wait(&empty[st], ph ^ 1, p.wait_budget, abort_flag, p.err)) goto producer_abort;
        uint8_t *buf = stage_base + (size_t)st * kDecStageBytes;
        if (s < res_stages) {
          const int kc0 = 2 * s;
          const int nkc = min(2, KC - kc0);
          const int g0 = (kc0 * kChunkK) / p.g;
          const int g1 = ((kc0 + nkc) * kChunkK - 1) / p.g;
          const int ng = g1 - g0 + 1;
          mbar_arrive_expect_tx(&full[st], (uint32_t)(ntile * (nkc * kChunkBytes + ng * kTileRows * 2)));
          for (int t = 0; t < ntile; ++t) {
            const int64_t vt = 2 * (int64_t)unit + t;
            bulk_g2s(buf + t * 2 * kChunkBytes, p.codes + (vt * KC + kc0) * kChunkBytes, nkc * kChunkBytes,
                     &full[st]);
            bulk_g2s(buf + kDecStageCodeBytes + t * 4 * kTileRows * 2, p.scales + (vt * p.G + g0) * kTileRows,
                     ng * kTileRows * 2, &full[st]);
          }
        } else {
          const int ls0 = (s - res_stages) * kDecLrStepsPerStage;
          const int nl = min(kDecLrStepsPerStage, p.nls - ls0);
          const bool last = (s == res_stages + lr_stages - 1);
          mbar_arrive_expect_tx(&full[st], (uint32_t)(ntile * (nl * kLrStepBytes + (last ? kTileRows * 2 : 0))));
          for (int t = 0; t < ntile; ++t) {
            const int64_t vt = 2 * (int64_t)unit + t;
            bulk_g2s(buf + t * kDecLrStepsPerStage * kLrStepBytes, p.lr_codes + (vt * p.nls + ls0) * kLrStepBytes,
                     nl * kLrStepBytes, &full[st]);
            if (last)
              bulk_g2s(buf + kDecStageCodeBytes + t * kTileRows * 2, p.s_a + vt * kTileRows, kTileRows * 2,
                       &full[st]);
          }
        }
      }
    }
    return;
  producer_abort:
    // Let copies already issued land before the block exits.
    for (int k = 1; k <= stages && it - k >= 0; ++k) {
      const int j = it - k;
      mbar_wait(&full[j % stages], (j / stages) & 1, p.wait_budget, nullptr, p.err);
    }
    return;
  }

  // ---------------- consumer warps ----------------
  const int tsel = warp >> 2;            // which tile of the unit
  const int mi0 = 2 * (warp & 3);        // first of two m-tiles in that tile
  const int gq = lane >> 2, cq = lane & 3;
  if (!mbar_wait(xbar, 0, p.wait_budget, abort_flag, p.err)) return;

  int it = 0;
  for (int unit = blockIdx.x; unit < num_units; unit += gridDim.x) {
    const int ntile = min(2, p.num_tiles - 2 * unit);
    const bool active = tsel < ntile;
    float acc[2][NT][4];
    float part[2][NT][4];
#pragma unroll
    for (int a = 0; a < 2; ++a)
#pragma unroll
      for (int b = 0; b < NT; ++b)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[a][b][c] = part[a][b][c] = 0.f;

    // Residual: INT4 codes, promoted per group.
    for (int s = 0; s < res_stages; ++s, ++it) {
      const int st = it % stages;
      if (!mbar_wait(&full[st], (it / stages) & 1, p.wait_budget, abort_flag, p.err)) return;
      const uint8_t *buf = stage_base + (size_t)st * kDecStageBytes;
      const int kc0 = 2 * s;
      const int nkc = min(2, KC - kc0);
      const int g0 = (kc0 * kChunkK) / p.g;
      if (active) {
        const uint16_t *sc = reinterpret_cast<const uint16_t *>(buf + kDecStageCodeBytes + tsel * 4 * kTileRows * 2);
        for (int c = 0; c < nkc; ++c) {
          uint4 w[2];
#pragma unroll
          for (int mt = 0; mt < 2; ++mt)
            w[mt] = *reinterpret_cast<const uint4 *>(buf + ((tsel * 2 + c) * 8 + mi0 + mt) * 512 + lane * 16);
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const int s16 = (kc0 + c) * 4 + j;
            uint32_t b[NT][2];
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
              const uint2 bb = *reinterpret_cast<const uint2 *>(
                  xs_s + (((size_t)nt * (p.d / 32) + (s16 >> 1)) * 32 + lane) * 4 + (s16 & 1) * 2);
              b[nt][0] = bb.x;
              b[nt][1] = bb.y;
            }
#pragma unroll
            for (int mt = 0; mt < 2; ++mt) {
              const uint32_t word = j == 0 ? w[mt].x : j == 1 ? w[mt].y : j == 2 ? w[mt].z : w[mt].w;
              uint32_t a[4];
              unpack_int4x8(word, a);
#pragma unroll
              for (int nt = 0; nt < NT; ++nt) mma_bf16_16816(part[mt][nt], a, b[nt][0], b[nt][1]);
            }
            if (((s16 + 1) & ((1 << p.g_shift) - 1)) == 0) {
              const int grp = (s16 >> p.g_shift) - g0;
#pragma unroll
              for (int mt = 0; mt < 2; ++mt) {
                const int r = (mi0 + mt) * 16 + gq;
                const float s_lo = fp16_bits_to_f32(sc[grp * kTileRows + r]);
                const float s_hi = fp16_bits_to_f32(sc[grp * kTileRows + r + 8]);
#pragma unroll
                for (int nt = 0; nt < NT; ++nt) {
                  acc[mt][nt][0] = fmaf(s_lo, part[mt][nt][0], acc[mt][nt][0]);
                  acc[mt][nt][1] = fmaf(s_lo, part[mt][nt][1], acc[mt][nt][1]);
                  acc[mt][nt][2] = fmaf(s_hi, part[mt][nt][2], acc[mt][nt][2]);
                  acc[mt][nt][3] = fmaf(s_hi, part[mt][nt][3], acc[mt][nt][3]);
#pragma unroll
                  for (int c2 = 0; c2 < 4; ++c2) part[mt][nt][c2] = 0.f;
                }
              }
            }
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[st]);
    }

    // Rank-r branches as extra k steps (core: factor 1; correction: row scale of A_w).
    for (int s = 0; s < lr_stages; ++s, ++it) {
      const int st = it % stages;
      if (!mbar_wait(&full[st], (it / stages) & 1, p.wait_budget, abort_flag, p.err)) return;
      const uint8_t *buf = stage_base + (size_t)st * kDecStageBytes;
      const int ls0 = s * kDecLrStepsPerStage;
      const int nl = min(kDecLrStepsPerStage, p.nls - ls0);
      if (active) {
        for (int l = 0; l < nl; ++l) {
          const int ls = ls0 + l;
          uint32_t bh[NT][2], bl[NT][2];
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            const uint2 h2 = *reinterpret_cast<const uint2 *>(ts_s + ((((size_t)ls * 2 + 0) * 2 + nt) * 32 + lane) * 2);
            const uint2 l2 = *reinterpret_cast<const uint2 *>(ts_s + ((((size_t)ls * 2 + 1) * 2 + nt) * 32 + lane) * 2);
            bh[nt][0] = h2.x;
            bh[nt][1] = h2.y;
            bl[nt][0] = l2.x;
            bl[nt][1] = l2.y;
          }
#pragma unroll
          for (int mt = 0; mt < 2; ++mt) {
            const uint2 w2 = *reinterpret_cast<const uint2 *>(
                buf + (((size_t)tsel * kDecLrStepsPerStage + l) * 8 + mi0 + mt) * 256 + lane * 8);
            uint32_t a[4];
            unpack_int8x8(w2.x, w2.y, a);
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
              mma_bf16_16816(part[mt][nt], a, bh[nt][0], bh[nt][1]);
              mma_bf16_16816(part[mt][nt], a, bl[nt][0], bl[nt][1]);
            }
          }
          if (ls + 1 == p.nls_core || ls + 1 == p.nls) {
            const bool corr = ls + 1 == p.nls && p.nls > p.nls_core;
            const uint16_t *sa = reinterpret_cast<const uint16_t *>(buf + kDecStageCodeBytes + tsel * kTileRows * 2);
#pragma unroll
            for (int mt = 0; mt < 2; ++mt) {
              const int r = (mi0 + mt) * 16 + gq;
              const float f_lo = corr ? fp16_bits_to_f32(sa[r]) : 1.f;
              const float f_hi = corr ? fp16_bits_to_f32(sa[r + 8]) : 1.f;
#pragma unroll
              for (int nt = 0; nt < NT; ++nt) {
                acc[mt][nt][0] = fmaf(f_lo, part[mt][nt][0], acc[mt][nt][0]);
                acc[mt][nt][1] = fmaf(f_lo, part[mt][nt][1], acc[mt][nt][1]);
                acc[mt][nt][2] = fmaf(f_hi, part[mt][nt][2], acc[mt][nt][2]);
                acc[mt][nt][3] = fmaf(f_hi, part[mt][nt][3], acc[mt][nt][3]);
#pragma unroll
                for (int c2 = 0; c2 < 4; ++c2) part[mt][nt][c2] = 0.f;
              }
            }
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[st]);
    }

    // Epilogue.  acc[mt][nt][i]: row 16*(mi0+mt) + gq + 8*(i/2), token 8*nt + 2*cq + i%2.
    const int64_t row_base = (2 * (int64_t)unit + tsel) * kTileRows;
    if (p.out) {
      if (active) {
#pragma unroll
        for (int mt = 0; mt < 2; ++mt)
#pragma unroll
          for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              const int64_t row = row_base + (mi0 + mt) * 16 + gq + 8 * (i >> 1);
              const int tok = nt * 8 + 2 * cq + (i & 1);
              if (row < p.V && tok < p.M) {
                const int64_t o = (int64_t)(p.m0 + tok) * p.V + row;
                if (p.out_fp32)
                  reinterpret_cast<float *>(p.out)[o] = acc[mt][nt][i];
                else
                  reinterpret_cast<__nv_bfloat16 *>(p.out)[o] = __float2bfloat16_rn(acc[mt][nt][i]);
              }
            }
      }
    } else {
      // Cross-entropy partials: per (warp, token) running max and sum of exp.
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int tl = 0; tl < 2; ++tl) {
          const int tok = nt * 8 + 2 * cq + tl;
          const int tgt = tok < p.M ? p.targets[p.m0 + tok] : -1;
          float vals[4];
          float mx = -INFINITY;
#pragma unroll
          for (int mt = 0; mt < 2; ++mt)
#pragma unroll
            for (int ih = 0; ih < 2; ++ih) {
              const int64_t row = row_base + (mi0 + mt) * 16 + gq + 8 * ih;
              const float v = (active && row < p.V) ? acc[mt][nt][ih * 2 + tl] : -INFINITY;
              vals[mt * 2 + ih] = v;
              mx = fmaxf(mx, v);
              if (active && row < p.V && row == tgt) p.ce_tlogit[p.m0 + tok] = v;
            }
          float sum = 0.f;
#pragma unroll
          for (int q = 0; q < 4; ++q) sum += (vals[q] == -INFINITY) ? 0.f : __expf(vals[q] - mx);
          LsePair lp{mx, sum};
#pragma unroll
          for (int off = 4; off < 32; off <<= 1) {
            LsePair o{__shfl_xor_sync(0xffffffffu, lp.m, off), __shfl_xor_sync(0xffffffffu, lp.s, off)};
            lp = lse_merge(lp, o);
          }
          if (gq == 0 && tok < p.M)
            p.ce_part[((int64_t)unit * kDecConsumerWarps + warp) * p.M_total + p.m0 + tok] = make_float2(lp.m, lp.s);
        }
    }
  }
}

int decode_num_units(const archead_pack *p) { return (p->num_tiles + 1) / 2; }

int decode_parts_per_unit() { return kDecConsumerWarps; }

bool decode_supported(int d, int nls) { return decode_plan(d, nls, 2).stages >= 2; }

cudaError_t launch_decode(const DecodeParams &dp, int grid, cudaStream_t s) {
  const DecodeSmemPlan pl = decode_plan(dp.d, dp.nls, dp.NT);
  if (pl.stages < 2) return cudaErrorInvalidValue;
  cudaError_t e;
  if (dp.NT == 1) {
    e = cudaFuncSetAttribute(decode_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)pl.total);
    if (e != cudaSuccess) return e;
    decode_kernel<1><<<grid, kDecThreads, pl.total, s>>>(dp, pl.stages, (int)pl.xs_off, (int)pl.ts_off,
                                                         (int)pl.bar_off);
  } else {
    e = cudaFuncSetAttribute(decode_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)pl.total);
    if (e != cudaSuccess) return e;
    decode_kernel<2><<<grid, kDecThreads, pl.total, s>>>(dp, pl.stages, (int)pl.xs_off, (int)pl.ts_off,
                                                         (int)pl.bar_off);
  }
  return cudaGetLastError();
}

}  // namespace archead
