// Memory-bound decode kernel (M <= 16 tokens) of the packed LM-head forward
// (paper, Section 3.2, Eq. 7; Appendix B: the core and correction paths are
// evaluated separately and no dense head is formed).
//
// Persistent grid, one block per SM; a unit of work is 256 vocabulary rows
// (two 128-row tiles).  The tokens are the N = 16 side of tcgen05.mma
// (kind::f16, M = 128 rows, K = 16), with the A operand in tensor memory:
//
//   - warp 0 streams, per ring stage, 128 columns of both tiles' INT4 codes
//     (1-D bulk copies) and the matching two 64-wide chunks of x for the 16
//     tokens (2-D tensor copies, 128-byte swizzle: the MMA's B operand);
//     the rank-r stages carry 64 extended columns of INT8 codes and of the
//     pre-pass operand T = [hi_c | lo_c | hi_r | lo_r] instead;
//   - eight converter warps, one thread per row, turn a row's codes into
//     packed bf16 pairs (INT4: 136 + code, exact; INT8: the code) and store
//     them into tensor memory with tcgen05.st;
//   - one elected thread issues the MMAs into a tile's 16-column fp32
//     accumulator; every quantisation group (and each rank-r branch) ends in
//     its own accumulator (two alternate);
//   - four promotion warps read each finished accumulator with tcgen05.ld and
//     add s[row, group] * (D - 136 * sum of x over the group) in fp32 (the
//     core branch with factor 1, the correction with the row scale of A_w),
//     then write the logits or the cross-entropy partials.
//
// At M <= 16 the tensor core is nearly idle; what this layout saves is the
// per-element work of the warp-level MMA path (fragment loads, one mma.sync
// per 256 weights and its dependency stalls): a converter thread spends about
// one unpack instruction per 8 weights and one tcgen05.st per 64.
#include "device.cuh"
#include "internal.h"

namespace archead {

constexpr int kDecTiles = 2;                                 // 128-row tiles per unit
constexpr int kDecN = 16;                                    // MMA N: tokens (padded)
constexpr int kDecResK = 128;                                // columns of d per residual stage
constexpr int kDecCodeBytes = kDecTiles * 2 * kChunkBytes;   // 16 KB; also 4 rank-r steps x 2 tiles
constexpr int kDecXOff = kDecCodeBytes;                      // x / T chunks, 1 KB aligned
constexpr int kXChunkBytes = kDecN * kChunkK * 2;            // 16 tokens x 64 columns bf16
constexpr int kDecStageBytes = kDecCodeBytes + 2 * kXChunkBytes;  // 20 KB
constexpr int kDecMaxStages = 10;
constexpr int kDecNA = 3;                                    // tensor-memory A buffers
constexpr int kDecAcols = kDecTiles * (kDecResK / 2);        // 128 columns per A buffer
constexpr int kDecDcol = kDecNA * kDecAcols;                 // 384: the two accumulator sets
constexpr int kDecTmemCols = 512;
constexpr int kDecThreads = 512;                             // 16 warps
constexpr int kDecConvWarp0 = 4, kDecPromWarp0 = 12;
constexpr int kSmemLimit = 227 * 1024;

struct DecodePlan {
  int stages;
  size_t xsum_off, bar_off, total;
};

// Shared memory: the stage ring, then [G_PAD][16] -136 * (sum of x over a
// group) and the barriers.  The ring leaves room for one pre-pass block on the
// same SM (the two grids overlap under programmatic dependent launch).
static DecodePlan decode_plan(int d_pad, int g) {
  DecodePlan pl{};
  const size_t xsum_bytes = (size_t)(d_pad / g) * kDecodeMaxTokens * 4;
  const size_t fixed = xsum_bytes + 512;
  const size_t cap = (size_t)kSmemLimit - prepass_smem(kDecodeMaxTokens) - 2048;
  int st = kDecMaxStages;
  while (st >= 2 && fixed + (size_t)st * kDecStageBytes > cap) --st;
  pl.stages = st;
  pl.xsum_off = (size_t)st * kDecStageBytes;
  pl.bar_off = pl.xsum_off + xsum_bytes;
  pl.total = pl.bar_off + 512;
  return pl;
}

__global__ void __launch_bounds__(kDecThreads, 1) decode_kernel(const __grid_constant__ DecodeParams p, int stages,
                                                                int xsum_off, int bar_off) {
  // The kernel has no static shared memory, so the dynamic window starts on a
  // 1 KB boundary, which the 128-byte-swizzled boxes rely on (checked).
  extern __shared__ __align__(1024) uint8_t smem[];
  if ((smem_u32(smem) & 1023u) != 0) {
    if (threadIdx.x == 0) atomicOr(p.err, kErrLayout);
    return;
  }
  float *xsum_s = reinterpret_cast<float *>(smem + xsum_off);  // [group][16]
  uint64_t *full = reinterpret_cast<uint64_t *>(smem + bar_off);
  uint64_t *empty = full + kDecMaxStages;
  uint64_t *a_full = empty + kDecMaxStages;
  uint64_t *a_empty = a_full + kDecNA;
  uint64_t *acc_full = a_empty + kDecNA;
  uint64_t *acc_empty = acc_full + 2;
  uint64_t *drain = acc_empty + 2;
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(drain + 1);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int KC = p.d_pad / kChunkK;
  const int RS = p.d_pad / kDecResK;          // residual stages per unit
  const int LS = (p.rcp + p.rrp) / 32;         // rank-r stages per unit (64 extended columns each)
  const int num_units = (p.num_tiles + kDecTiles - 1) / kDecTiles;
  const int GS = p.g / 16;                     // k steps per quantisation group
  const int ng = p.d_pad / p.g;

  if (threadIdx.x == 0) {
    for (int i = 0; i < stages; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    for (int i = 0; i < kDecNA; ++i) {
      mbar_init(&a_full[i], 8);
      mbar_init(&a_empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], 4);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) tmem_alloc(tmem_slot, kDecTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  bool mma_leader = false;

  if (warp == 0) {
    // ------------------------------ producer ------------------------------
    const bool leader = elect_one();
    bool t_ready = false;
    int it = 0;
    for (int unit = blockIdx.x; unit < num_units; unit += gridDim.x) {
      const int ntile = min(kDecTiles, p.num_tiles - kDecTiles * unit);
      for (int s = 0; s < RS + LS; ++s, ++it) {
        const int st = it % stages;
        if (s == RS && !t_ready) {
          asm volatile("griddepcontrol.wait;\n" ::: "memory");  // T comes from the pre-pass grid
          t_ready = true;
        }
        if (!mbar_wait_warp(&empty[st], ((it / stages) & 1) ^ 1, p.wait_budget, abort_flag, p.err)) goto done;
        uint8_t *buf = smem + (size_t)st * kDecStageBytes;
        if (leader) {
          if (s < RS) {
            mbar_arrive_expect_tx(&full[st], (uint32_t)(ntile * 2 * kChunkBytes + 2 * kXChunkBytes));
            for (int t = 0; t < ntile; ++t) {
              const int64_t vt = (int64_t)kDecTiles * unit + t;
              bulk_g2s(buf + t * 2 * kChunkBytes, p.codes + (vt * KC + 2 * s) * kChunkBytes, 2 * kChunkBytes,
                       &full[st]);
            }
            for (int c = 0; c < 2; ++c)
              tma_load_2d(buf + kDecXOff + c * kXChunkBytes, &p.tmap_x, (2 * s + c) * kChunkK, p.m0, &full[st]);
          } else {
            const int xe = s - RS;
            mbar_arrive_expect_tx(&full[st], (uint32_t)(ntile * 4 * kLrStepBytes + kXChunkBytes));
            for (int t = 0; t < ntile; ++t) {
              const int64_t vt = (int64_t)kDecTiles * unit + t;
              for (int q = 0; q < 4; ++q) {
                const int kk = xe * 64 + q * 16;  // column of the extended operand
                const int ls = kk < 2 * p.rcp ? (kk % p.rcp) / 16 : p.nls_core + ((kk - 2 * p.rcp) % p.rrp) / 16;
                bulk_g2s(buf + t * 2 * kChunkBytes + q * kLrStepBytes,
                         p.lr_codes + (vt * p.nls + ls) * kLrStepBytes, kLrStepBytes, &full[st]);
              }
            }
            tma_load_2d(buf + kDecXOff, &p.tmap_t, xe * kChunkK, p.m0, &full[st]);
          }
        }
        __syncwarp();
      }
    }
  } else if (warp == 1) {
    // ------------------------------ MMA issuer ------------------------------
    const bool leader = elect_one();
    mma_leader = leader;
    constexpr uint32_t idesc = idesc_bf16(128, kDecN);
    const uint64_t xdesc0 = smem_desc_sw128(smem_u32(smem) + kDecXOff);
    constexpr uint32_t kStageDesc = kDecStageBytes >> 4;
    constexpr uint32_t kXChunkDesc = kXChunkBytes >> 4;
    int it = 0, bcount = 0;
    for (int unit = blockIdx.x; unit < num_units; unit += gridDim.x) {
      const int ntile = min(kDecTiles, p.num_tiles - kDecTiles * unit);
      // Blocks: ng residual groups of GS steps, then the core (2 RCP / 16
      // steps) and correction (2 RRP / 16 steps) branches.
      int blk = 0, in_blk = 0, blk_len = GS;
      for (int s = 0; s < RS + LS; ++s, ++it) {
        const int st = it % stages, ab = it % kDecNA;
        if (!mbar_wait_warp(&full[st], (it / stages) & 1, p.wait_budget, abort_flag, p.err)) goto done;
        if (!mbar_wait_warp(&a_full[ab], (it / kDecNA) & 1, p.wait_budget, abort_flag, p.err)) goto done;
        tc_fence_after();
        const uint64_t xd = xdesc0 + (uint64_t)(st * kStageDesc);
        const int nks = s < RS ? 8 : 4;
        for (int kk = 0; kk < nks; ++kk) {
          const int db = bcount & 1;
          if (in_blk == 0) {
            if (!mbar_wait_warp(&acc_empty[db], ((bcount >> 1) & 1) ^ 1, p.wait_budget, abort_flag, p.err))
              goto done;
            tc_fence_after();
          }
          // +2 per 16-wide k step inside a 64-column chunk (32 bytes in 16-byte units).
          const uint64_t bd = xd + (uint64_t)((kk >> 2) * kXChunkDesc + 2 * (kk & 3));
          for (int t = 0; t < ntile; ++t)
            if (leader)
              tc_mma_ts(tmem_base + kDecDcol + db * (kDecTiles * kDecN) + t * kDecN,
                        tmem_base + ab * kDecAcols + t * (kDecResK / 2) + kk * 8, bd, idesc, in_blk > 0);
          if (++in_blk == blk_len) {
            if (leader) tc_commit(&acc_full[db]);
            ++bcount;
            ++blk;
            in_blk = 0;
            blk_len = blk < ng ? GS : (blk == ng && p.rcp > 0 ? 2 * p.rcp / 16 : 2 * p.rrp / 16);
          }
        }
        if (leader) {
          tc_commit(&empty[st]);    // codes were read by the converters, x / T by these MMAs
          tc_commit(&a_empty[ab]);
        }
        __syncwarp();
      }
    }
  } else if (warp >= kDecConvWarp0 && warp < kDecPromWarp0) {
    // ------------------------------ converters ------------------------------
    const int tt = (warp - kDecConvWarp0) >> 2;  // tile of the unit
    const int q = warp & 3;                      // tensor-memory lane quarter
    const int r = q * 32 + lane;                 // row within the tile
    int it = 0;
    for (int unit = blockIdx.x; unit < num_units; unit += gridDim.x) {
      const bool active = tt < min(kDecTiles, p.num_tiles - kDecTiles * unit);
      for (int s = 0; s < RS + LS; ++s, ++it) {
        const int st = it % stages, ab = it % kDecNA;
        if (!mbar_wait_warp(&full[st], (it / stages) & 1, p.wait_budget, abort_flag, p.err)) goto done;
        if (!mbar_wait_warp(&a_empty[ab], ((it / kDecNA) & 1) ^ 1, p.wait_budget, abort_flag, p.err)) goto done;
        tc_fence_after();
        const uint8_t *cb = smem + (size_t)st * kDecStageBytes + tt * 2 * kChunkBytes;
        const uint32_t ta = tmem_base + ((uint32_t)(q * 32) << 16) + ab * kDecAcols + tt * (kDecResK / 2);
        if (active) {
          if (s < RS) {
#pragma unroll
            for (int c = 0; c < 2; ++c) {
              const uint4 w0 = *reinterpret_cast<const uint4 *>(cb + c * kChunkBytes + r * 32);
              const uint4 w1 = *reinterpret_cast<const uint4 *>(cb + c * kChunkBytes + r * 32 + 16);
              const uint32_t ws[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
              uint32_t a[32];
#pragma unroll
              for (int w = 0; w < 8; ++w) {
                uint32_t u[4];
                unpack_int4x8_biased(ws[w], u);
#pragma unroll
                for (int i = 0; i < 4; ++i) a[4 * w + i] = u[i];
              }
              tmem_st32(ta + c * 32, a);
            }
          } else {
            uint32_t a[32];
#pragma unroll
            for (int l = 0; l < 4; ++l) {
              uint32_t u[8];
              unpack_int8x16(*reinterpret_cast<const uint4 *>(cb + l * kLrStepBytes + r * 16), u);
#pragma unroll
              for (int i = 0; i < 8; ++i) a[8 * l + i] = u[i];
            }
            tmem_st32(ta, a);
          }
          tmem_wait_st();
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&a_full[ab]);
      }
    }
  } else if (warp >= kDecPromWarp0) {
    // ------------------------------ promotion + epilogue ------------------------------
    const int q = warp & 3;
    const int r = q * 32 + lane;
    const int pt = threadIdx.x - kDecPromWarp0 * 32;  // 0..127
    // -136 * (sum of x over each group) for the 16 tokens of this chunk.
    for (int e = pt; e < ng * kDecodeMaxTokens; e += 128) {
      const int grp = e / kDecodeMaxTokens, m = e % kDecodeMaxTokens;
      float sum = 0.f;
      if (m < p.M && grp * p.g < p.d) {
        const uint4 *src = reinterpret_cast<const uint4 *>(p.x + (int64_t)(p.m0 + m) * p.d + (int64_t)grp * p.g);
        for (int k = 0; k < p.g / 8; ++k) {
          const uint4 v = src[k];
          sum += bf16_lo(v.x) + bf16_hi(v.x) + bf16_lo(v.y) + bf16_hi(v.y);
          sum += bf16_lo(v.z) + bf16_hi(v.z) + bf16_lo(v.w) + bf16_hi(v.w);
        }
      }
      xsum_s[e] = -kInt4Bias * sum;
    }
    asm volatile("bar.sync 1, 128;\n" ::: "memory");  // the four promotion warps
    int tg[kDecodeMaxTokens];
#pragma unroll
    for (int n = 0; n < kDecodeMaxTokens; ++n) tg[n] = (!p.out && n < p.M) ? p.targets[p.m0 + n] : -1;
    int bcount = 0;
    for (int unit = blockIdx.x; unit < num_units; unit += gridDim.x) {
      const int ntile = min(kDecTiles, p.num_tiles - kDecTiles * unit);
      int64_t row[kDecTiles];
#pragma unroll
      for (int t = 0; t < kDecTiles; ++t) row[t] = ((int64_t)kDecTiles * unit + t) * kTileRows + r;
      float acc[kDecTiles][kDecN];
#pragma unroll
      for (int t = 0; t < kDecTiles; ++t)
#pragma unroll
        for (int n = 0; n < kDecN; ++n) acc[t][n] = 0.f;
      const int nb = ng + (p.rcp > 0) + (p.rrp > 0);
      // Group scales one block ahead (global loads; the promotion has slack).
      float f_next[kDecTiles];
#pragma unroll
      for (int t = 0; t < kDecTiles; ++t)
        f_next[t] = t < ntile ? fp16_bits_to_f32(p.scales[(row[t] / kTileRows * p.G_pad) * kTileRows + r]) : 0.f;
      for (int b = 0; b < nb; ++b) {
        float f[kDecTiles];
#pragma unroll
        for (int t = 0; t < kDecTiles; ++t) {
          if (b < ng) f[t] = f_next[t];
          else if (b == ng && p.rcp > 0) f[t] = 1.f;
          else f[t] = t < ntile ? fp16_bits_to_f32(p.s_a[row[t]]) : 0.f;
        }
        if (b + 1 < ng) {
#pragma unroll
          for (int t = 0; t < kDecTiles; ++t)
            if (t < ntile)
              f_next[t] = fp16_bits_to_f32(p.scales[((row[t] / kTileRows) * p.G_pad + b + 1) * kTileRows + r]);
        }
        const int db = bcount & 1;
        if (!mbar_wait_warp(&acc_full[db], (bcount >> 1) & 1, p.wait_budget, abort_flag, p.err)) goto done;
        tc_fence_after();
#pragma unroll
        for (int t = 0; t < kDecTiles; ++t) {
          if (t < ntile) {
            float v[kDecN];
            tmem_ld16(tmem_base + ((uint32_t)(q * 32) << 16) + kDecDcol + db * (kDecTiles * kDecN) + t * kDecN, v);
            if (b < ng) {
#pragma unroll
              for (int n = 0; n < kDecN; ++n)
                acc[t][n] = fmaf(f[t], v[n] + xsum_s[b * kDecodeMaxTokens + n], acc[t][n]);
            } else {
#pragma unroll
              for (int n = 0; n < kDecN; ++n) acc[t][n] = fmaf(f[t], v[n], acc[t][n]);
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&acc_empty[db]);
        ++bcount;
      }

      if (p.out) {
        // Logits: row-contiguous stores (32 rows per warp and token).
#pragma unroll
        for (int t = 0; t < kDecTiles; ++t) {
          if (t < ntile && row[t] < p.V) {
#pragma unroll
            for (int n = 0; n < kDecN; ++n) {
              if (n < p.M) {
                const int64_t o = (int64_t)(p.m0 + n) * p.V + row[t];
                if (p.out_fp32)
                  reinterpret_cast<float *>(p.out)[o] = acc[t][n];
                else
                  reinterpret_cast<__nv_bfloat16 *>(p.out)[o] = __float2bfloat16_rn(acc[t][n]);
              }
            }
          }
        }
      } else {
        // Cross entropy: target logits, then (max, sum exp) per token over the
        // warp's 32 rows of both tiles.  In-lane merge of the two rows, then a
        // butterfly that halves the token set per step (offsets 16, 8, 4, 2)
        // and a last plain merge (offset 1): lanes 2n and 2n+1 end with token n.
        float mv[kDecN], sv[kDecN];
#pragma unroll
        for (int n = 0; n < kDecN; ++n) {
          float m = -INFINITY, sm = 0.f;
#pragma unroll
          for (int t = 0; t < kDecTiles; ++t) {
            const bool ok = t < ntile && row[t] < p.V;
            if (ok && tg[n] == row[t]) p.ce_tlogit[p.m0 + n] = acc[t][n];
            lse_pair_merge(m, sm, ok ? acc[t][n] : -INFINITY, ok ? 1.f : 0.f, m, sm);
          }
          mv[n] = m;
          sv[n] = sm;
        }
#pragma unroll
        for (int h = 8, o = 16; h >= 1; h >>= 1, o >>= 1) {
          const bool up = lane & o;
#pragma unroll
          for (int j = 0; j < h; ++j) {
            const float km = up ? mv[j + h] : mv[j], ks = up ? sv[j + h] : sv[j];
            const float gm = up ? mv[j] : mv[j + h], gs = up ? sv[j] : sv[j + h];
            const float rm = __shfl_xor_sync(0xffffffffu, gm, o), rs = __shfl_xor_sync(0xffffffffu, gs, o);
            lse_pair_merge(km, ks, rm, rs, mv[j], sv[j]);
          }
        }
        {
          const float rm = __shfl_xor_sync(0xffffffffu, mv[0], 1), rs = __shfl_xor_sync(0xffffffffu, sv[0], 1);
          lse_pair_merge(mv[0], sv[0], rm, rs, mv[0], sv[0]);
        }
        const int n = lane >> 1;
        if ((lane & 1) == 0 && n < p.M)
          p.ce_part[((int64_t)unit * 4 + q) * p.M_total + p.m0 + n] = make_float2(mv[0], sv[0]);
      }
    }
  }
done:
  if (warp == 1 && mma_leader) {
    // Every MMA this thread issued has completed before tensor memory is released.
    tc_commit(drain);
    mbar_wait(drain, 0, p.wait_budget, nullptr, p.err);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kDecTmemCols);
  }
}

int decode_num_units(const archead_pack *p) { return (p->num_tiles + kDecTiles - 1) / kDecTiles; }

int decode_parts_per_unit() { return 4; }

bool decode_supported(int d_pad, int nls, int g) {
  (void)nls;
  return decode_plan(d_pad, g).stages >= 2;
}

cudaError_t launch_decode(const DecodeParams &dp, const uint16_t *T, int grid, cudaStream_t s, bool pdl) {
  const DecodePlan pl = decode_plan(dp.d_pad, dp.g);
  if (pl.stages < 2 || dp.M < 1 || dp.M > kDecodeMaxTokens) return cudaErrorInvalidValue;
  DecodeParams k = dp;
  if (!make_tma_map_bf16(&k.tmap_x, dp.x, dp.M_total, dp.d, kDecN)) return cudaErrorInvalidValue;
  const int lr = dp.rcp + dp.rrp;
  if (lr > 0) {
    if (!T || !make_tma_map_bf16(&k.tmap_t, T, dp.M_total, 2 * lr, kDecN)) return cudaErrorInvalidValue;
  }
  static int smem_set = 0;
  if ((int)pl.total > smem_set) {
    cudaError_t e = cudaFuncSetAttribute(decode_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)pl.total);
    if (e != cudaSuccess) return e;
    smem_set = (int)pl.total;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kDecThreads);
  cfg.dynamicSmemBytes = pl.total;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, decode_kernel, k, pl.stages, (int)pl.xsum_off, (int)pl.bar_off);
}

}  // namespace archead
