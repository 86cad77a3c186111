// Tensor-core prefill kernel (large M) of the packed LM-head forward (paper,
// Section 3.2, Eq. 7; no dense W_hat is formed, the residual is dequantised
// tile by tile inside the kernel as Appendix B allows).
//
// Tile: 128 vocabulary rows x 256 tokens.  The vocabulary rows are the MMA's
// M side (one TMEM lane each), the tokens the N side.  Per 64-wide k step:
//   - a producer warp loads the x tile (256 tokens x 64, bf16, 128-byte
//     swizzle) with two 2-D TMA copies and the tile's INT4 code chunk with a
//     1-D bulk copy;
//   - four converter warps turn the codes into exact bf16 integers and store
//     them as the K-major, 128-byte-swizzled A operand in shared memory;
//   - one thread issues four tcgen05.mma (kind::f16, 128x256x16, fp32
//     accumulate) into one of two TMEM accumulators; a quantisation group
//     (g of d) always ends in its own accumulator;
//   - eight promotion warps read each finished group with tcgen05.ld and add
//     s[row, group] * partial to fp32 registers (group-wise scales cannot be
//     folded into exact bf16 operands).
// The rank-r branches are further k steps: A = int8 codes of A_c (factor 1)
// or A_w (factor = row scale of A_w), B = the pre-pass's bf16 hi/lo split of
// x V_c and x B_w^T, read through a second tensor map.
//
// In the paper's packed format (SC4) a group scale is s_row * (q + 1) with a
// 4-bit code q.  The converters fold q + 1 into the operand (code * (q + 1)
// stays an exact bf16 integer, |.| <= 128), so the whole residual is one
// accumulator block promoted once by s_row: no per-group hand-back.
//
// Epilogues: logits (each promotion thread stores one row of its 128 tokens),
// greedy partials (largest logit and its row per token over each warp's 32
// rows) and cross-entropy partials (max and sum of exp per token over each
// warp's 32 rows, plus the target's logit).  The cross-entropy and greedy
// instances read TMEM in the 16x256b shape, so that a thread holds 4 rows
// of 32 tokens and most of the reduction over rows is thread-local.
#pragma once

#include <cfloat>
#include <cuda.h>

#include "device.cuh"
#include "internal.h"

namespace archead {

constexpr int kPfN = 256;                         // tokens per tile
constexpr int kPfStages = 4;
constexpr int kPfABytes = kTileRows * 64 * 2;     // 16 KB
constexpr int kPfBBytes = kPfN * 64 * 2;          // 32 KB
constexpr int kPfCodeBytes = 4 * kLrStepBytes;    // 8 KB (4 KB of INT4 or 4 low-rank steps)
constexpr int kPfStageBytes = kPfABytes + kPfBBytes + kPfCodeBytes;
constexpr int kPfThreads = 512;
constexpr int kPfTmemCols = 512;                  // two 256-column accumulators
constexpr int kPfSmem = 1024 + kPfStages * kPfStageBytes + 256;
constexpr float kLog2e = 1.4426950408889634f;  // log2(e)
constexpr float kLn2 = 0.6931471805599453f;    // ln(2)

struct PrefillParams {
  CUtensorMap tmap_x;   // bf16 [M][d], box 64 x 128, 128B swizzle
  CUtensorMap tmap_t;   // bf16 [M][2*LR], box 64 x 128, 128B swizzle
  const uint8_t *codes;
  const uint16_t *scales;  // fp16 group scales (INT8 format)
  const uint8_t *scodes;   // 4-bit group-scale codes (SC4 format)
  const uint16_t *s_row;   // residual row scales (SC4 format)
  const uint8_t *lr_codes;
  const uint16_t *s_a;
  int64_t V;
  int M, num_vt, num_mt, d_pad, G_pad, g, nls, nls_core, rcp, rrp;
  int sc4, G_pad2;
  void *out;
  int out_fp32;
  const int32_t *targets;  // global vocabulary rows
  int row0;                // global row of this pack's first row (vocabulary shards; 0 otherwise)
  float2 *ce_part;   // [num_vt * 4][M]
  float *ce_tlogit;  // [M]
  int *err;
  int64_t wait_budget;
};

// ------------------------------------------------------------------------
// tcgen05 / TMA wrappers (inline PTX).
// ------------------------------------------------------------------------
__device__ __forceinline__ void tmem_alloc(uint32_t *slot, uint32_t cols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(smem_u32(slot)), "r"(cols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t cols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(taddr), "r"(cols) : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory"); }

__device__ __forceinline__ void tc_commit(uint64_t *bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(smem_u32(bar))
               : "memory");
}

__device__ __forceinline__ void tc_mma(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                       uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// 32 lanes x 32 consecutive 32-bit columns starting at taddr (one value per column per thread).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
        "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// 16 lanes x 32 columns starting at taddr (lane field = first lane) in the
// 16x256b shape, 4 repetitions of 8 columns: in repetition c thread t holds
// v[4c + j] = (lane t/4 + 8 (j >> 1), column 8c + 2 (t % 4) + (j & 1)).
__device__ __forceinline__ void tmem_ld16x256b_x4(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.16x256b.x4.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// 2^x by the special-function unit (ex2.approx, flushes denormal results).
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;\n" : "=f"(y) : "f"(x));
  return y;
}

// d0 += a * b0 and d1 += a * b1 as one packed fp32x2 FMA (round to nearest).
__device__ __forceinline__ void fma2(float &d0, float &d1, float a, float b0, float b1) {
  asm("{\n .reg .b64 ra, rb, rd;\n mov.b64 ra, {%2, %2};\n mov.b64 rb, {%3, %4};\n mov.b64 rd, {%0, %1};\n"
      " fma.rn.f32x2 rd, ra, rb, rd;\n mov.b64 {%0, %1}, rd;\n}\n"
      : "+f"(d0), "+f"(d1)
      : "f"(a), "f"(b0), "f"(b1));
}

// One step of the base-2 log-sum-exp merge: (m, s) of two disjoint sets, s
// the sum of 2^(y - m), -> (m, s) of their union.  Maxima are finite: rows
// past the vocabulary enter as -FLT_MAX, whose difference with itself is 0
// and with any logit rounds to +-FLT_MAX or +-inf (weight 0).
__device__ __forceinline__ void lse2_merge(float am, float as, float bm, float bs, float &m, float &s) {
  const float d = am - bm;
  const float e = ex2_approx(-fabsf(d));
  s = d >= 0.f ? fmaf(bs, e, as) : fmaf(as, e, bs);
  m = fmaxf(am, bm);
}

// Shared-memory matrix descriptor: K-major operand in the 128-byte swizzle
// layout (8-row groups of 128-byte rows, 1024 bytes apart).
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t saddr) {
  uint64_t desc = 0;
  desc |= (uint64_t)((saddr >> 4) & 0x3FFF);        // start address
  desc |= (uint64_t)1 << 16;                        // leading byte offset (unused for this layout)
  desc |= (uint64_t)(1024 >> 4) << 32;              // stride byte offset: 8 rows x 128 B
  desc |= (uint64_t)1 << 46;                        // descriptor version (tcgen05)
  desc |= (uint64_t)2 << 61;                        // 128-byte swizzle
  return desc;
}

// Instruction descriptor: kind::f16, A = B = bf16, D = f32, K-major A and B.
__host__ __device__ constexpr uint32_t idesc_bf16(int m, int n) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(m >> 4) << 24);
}

// Byte offset of bf16 element (row, k) in a 128-row x 64 K-major tile with the
// 128-byte swizzle: 16-byte chunk k/8 of row r is stored at chunk (k/8) ^ (r%8).
__device__ __forceinline__ uint32_t sw128_off(int row, int k) {
  return (uint32_t)(row * 128 + ((((k >> 3) ^ (row & 7)) & 7) << 4) + (k & 7) * 2);
}

// ------------------------------------------------------------------------
// Promotion blocks of a tile: residual groups, then the core and the
// correction branches of the extended rank axis.
// ------------------------------------------------------------------------
struct BlockPlan {
  int nres, res_sub;       // residual blocks (groups; one for SC4), 16-wide sub-steps per block
  int core_sub, corr_sub;  // sub-steps of the core (2*RCP/16) and correction (2*RRP/16) blocks
  __device__ int nblocks() const { return nres + (core_sub > 0) + (corr_sub > 0); }
};

// bf16x2 fused multiply-add a * b + c (round to nearest even).
__device__ __forceinline__ uint32_t bf16x2_fma(uint32_t a, uint32_t b, uint32_t c) {
  uint32_t d;
  asm("fma.rn.bf16x2 %0, %1, %2, %3;\n" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  return d;
}

// For a 4-bit scale code q: bf16x2 (q+1, q+1) and (-136 (q+1), -136 (q+1)),
// so that fma(136 + code, m, -136 m) = code * (q + 1) exactly.
__device__ __forceinline__ void sc4_mult(uint32_t byte, int sh, uint32_t &m2, uint32_t &nb2) {
  const float m = (float)(((byte >> sh) & 15u) + 1u);
  m2 = pack_bf16x2(m, m);
  nb2 = pack_bf16x2(-kInt4Bias * m, -kInt4Bias * m);
}

// kMode 0: logits, 1: cross-entropy partials, 2: greedy (largest logit, row)
// partials; kSC4: the paper's packed format (group-scale codes times row scales).
template <int kMode, bool kSC4>
__global__ void __launch_bounds__(kPfThreads, 1) prefill_kernel(const __grid_constant__ PrefillParams p) {
  extern __shared__ uint8_t pf_smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(pf_smem_raw) + 1023) & ~(uintptr_t)1023);
  uint64_t *full = reinterpret_cast<uint64_t *>(smem + kPfStages * kPfStageBytes);
  uint64_t *a_full = full + kPfStages;
  uint64_t *empty = a_full + kPfStages;
  uint64_t *acc_full = empty + kPfStages;
  uint64_t *acc_empty = acc_full + 2;
  uint64_t *drain = acc_empty + 2;
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(drain + 1);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int KC = p.d_pad / 64;                 // residual k steps
  const int KE = (2 * (p.rcp + p.rrp)) / 64;   // extended (rank) k steps
  const int KS = KC + KE;
  const int num_tiles = p.num_vt * p.num_mt;
  BlockPlan bp{kSC4 ? 1 : p.G_pad, kSC4 ? p.d_pad / 16 : p.g / 16, 2 * p.rcp / 16, 2 * p.rrp / 16};

  if (threadIdx.x == 0) {
    for (int i = 0; i < kPfStages; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&a_full[i], 4);
      mbar_init(&empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], 8);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) tmem_alloc(tmem_slot, kPfTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  bool mma_leader = false;  // the lane of warp 1 that issues the MMAs

  // Registers are rebalanced between warpgroups (launch: 512 x 128): the
  // converters keep 88, the producer/MMA warpgroup 88 (logits) or 56 (cross
  // entropy, greedy), the two promotion warpgroups get the rest, 168 or 184
  // (128 fp32 accumulators per thread; the 4-row epilogues need more): 4*32*(88 + 88) + 8*32*168 = 4*32*(56 + 88) + 8*32*184 = 65536.
  // Each role's code follows its own setmaxnreg so that the compiler
  // allocates within that budget; these splits compile without spills.
  if (warp < 4) {
    if constexpr (kMode != 0)
      asm volatile("setmaxnreg.dec.sync.aligned.u32 56;\n" ::: "memory");
    else
      asm volatile("setmaxnreg.dec.sync.aligned.u32 88;\n" ::: "memory");
  if (warp == 0) {
    // ------------------------------ producer ------------------------------
    // The whole warp runs the loop (uniform waits); one elected lane issues.
    {
      const bool leader = elect_one();
      int s = 0;
      uint32_t ph = 0;
      for (int t = blockIdx.x; t < num_tiles; t += gridDim.x) {
        const int vt = t / p.num_mt, mt = t % p.num_mt;
        const int m0 = mt * kPfN;
        for (int e = 0; e < KS; ++e) {
          if (!mbar_wait_warp(&empty[s], ph ^ 1, p.wait_budget, abort_flag, p.err)) goto done;
          uint8_t *st = smem + s * kPfStageBytes;
          uint8_t *bdst = st + kPfABytes;
          uint8_t *cdst = bdst + kPfBBytes;
          if (!leader) {
          } else if (e < KC) {
            mbar_arrive_expect_tx(&full[s], kPfBBytes + kChunkBytes + (kSC4 ? kTileRows : 0));
            tma_load_2d(bdst, &p.tmap_x, e * 64, m0, &full[s]);
            tma_load_2d(bdst + kPfBBytes / 2, &p.tmap_x, e * 64, m0 + 128, &full[s]);
            bulk_g2s(cdst, p.codes + ((int64_t)vt * KC + e) * kChunkBytes, kChunkBytes, &full[s]);
            if constexpr (kSC4)  // the byte row of scale codes holding this k step's groups
              bulk_g2s(cdst + kChunkBytes, p.scodes + ((int64_t)vt * p.G_pad2 + ((e * 64) >> (__ffs(p.g) - 1) >> 1)) * kTileRows,
                       kTileRows, &full[s]);
          } else {
            const int xe = e - KC;
            mbar_arrive_expect_tx(&full[s], kPfBBytes + 4 * kLrStepBytes);
            tma_load_2d(bdst, &p.tmap_t, xe * 64, m0, &full[s]);
            tma_load_2d(bdst + kPfBBytes / 2, &p.tmap_t, xe * 64, m0 + 128, &full[s]);
            for (int q = 0; q < 4; ++q) {
              const int kk = xe * 64 + q * 16;  // column of the extended operand
              int ls;
              if (kk < 2 * p.rcp) ls = (kk % p.rcp) / 16;
              else ls = p.nls_core + ((kk - 2 * p.rcp) % p.rrp) / 16;
              bulk_g2s(cdst + q * kLrStepBytes, p.lr_codes + ((int64_t)vt * p.nls + ls) * kLrStepBytes, kLrStepBytes,
                       &full[s]);
            }
          }
          if (++s == kPfStages) s = 0, ph ^= 1;
          __syncwarp();
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------ MMA issuer ------------------------------
    // As for the producer: the warp runs the loop, one elected lane issues.
    // Keeping the loop warp-uniform (votes on every wait, elect.sync for the
    // issuing lane) is what lets the MMAs issue back to back.
    {
      const bool leader = elect_one();
      mma_leader = leader;
      constexpr uint32_t idesc = idesc_bf16(128, kPfN);
      const uint64_t desc0 = smem_desc_sw128(smem_u32(smem));
      constexpr uint32_t kStageDesc = kPfStageBytes >> 4;  // descriptor address step of one stage
      constexpr uint32_t kBDesc = kPfABytes >> 4;           // A -> B within a stage
      int s = 0;
      uint32_t ph = 0;
      int bcount = 0;  // accumulator blocks started so far
      for (int t = blockIdx.x; t < num_tiles; t += gridDim.x) {
        int blk = 0, in_blk = 0;
        int blk_len = bp.nres > 0 ? bp.res_sub : (bp.core_sub > 0 ? bp.core_sub : bp.corr_sub);
        for (int e = 0; e < KS; ++e) {
          // The converters arrive on a_full only after the stage's TMA bytes landed.
          if (!mbar_wait_warp(&a_full[s], ph, p.wait_budget, abort_flag, p.err)) goto done;
          tc_fence_after();
          const uint64_t ad = desc0 + (uint64_t)(s * kStageDesc);
          const uint64_t bd = ad + kBDesc;
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const int buf = bcount & 1;
            if (in_blk == 0) {
              if (!mbar_wait_warp(&acc_empty[buf], ((bcount >> 1) & 1) ^ 1, p.wait_budget, abort_flag, p.err))
                goto done;
              tc_fence_after();
            }
            // +2 per 16-wide k step: 32 bytes in the descriptor's 16-byte address units.
            if (leader) tc_mma(tmem_base + buf * kPfN, ad + 2 * q, bd + 2 * q, idesc, in_blk > 0);
            if (++in_blk == blk_len) {
              if (leader) tc_commit(&acc_full[buf]);
              ++bcount;
              ++blk;
              in_blk = 0;
              blk_len = blk < bp.nres ? bp.res_sub : (blk == bp.nres && bp.core_sub > 0 ? bp.core_sub : bp.corr_sub);
            }
          }
          if (leader) tc_commit(&empty[s]);
          if (++s == kPfStages) s = 0, ph ^= 1;
          __syncwarp();
        }
      }
    }
  }
  } else if (warp < 8) {
    // ------------------------------ converters ------------------------------
    asm volatile("setmaxnreg.dec.sync.aligned.u32 88;\n" ::: "memory");
    const int cw = warp - 4;
    const int gq = lane >> 2, cq = lane & 3;
    const int lg = __ffs(p.g) - 1;  // log2 g
    int s = 0;
    uint32_t ph = 0;
    for (int t = blockIdx.x; t < num_tiles; t += gridDim.x) {
      for (int e = 0; e < KS; ++e) {
        if (!mbar_wait_warp(&full[s], ph, p.wait_budget, abort_flag, p.err)) goto done;
        uint8_t *a_tile = smem + s * kPfStageBytes;
        const uint8_t *codes = a_tile + kPfABytes + kPfBBytes;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int mi = cw * 2 + h;
          if (e < KC) {
            const uint4 w4 = *reinterpret_cast<const uint4 *>(codes + (mi * 32 + lane) * 16);
            const uint32_t ws[4] = {w4.x, w4.y, w4.z, w4.w};
            // SC4: scale-code bytes of rows gq and gq + 8; the multipliers q + 1
            // are set for each 32-wide half of the k step (the halves' groups
            // differ only when g = 32).
            uint32_t b_lo = 0, b_hi = 0, m_lo = 0, nb_lo = 0, m_hi = 0, nb_hi = 0;
            if constexpr (kSC4) {
              b_lo = codes[kChunkBytes + mi * 16 + gq];
              b_hi = codes[kChunkBytes + mi * 16 + gq + 8];
            }
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              uint32_t a[4];
              if constexpr (kSC4) {
                if (j % 2 == 0) {
                  const int sh = 4 * (((e * 64 + 16 * j) >> lg) & 1);  // nibble of the half's group
                  sc4_mult(b_lo, sh, m_lo, nb_lo);
                  sc4_mult(b_hi, sh, m_hi, nb_hi);
                }
                unpack_int4x8_biased(ws[j], a);
                a[0] = bf16x2_fma(a[0], m_lo, nb_lo);
                a[1] = bf16x2_fma(a[1], m_hi, nb_hi);
                a[2] = bf16x2_fma(a[2], m_lo, nb_lo);
                a[3] = bf16x2_fma(a[3], m_hi, nb_hi);
              } else {
                unpack_int4x8(ws[j], a);
              }
#pragma unroll
              for (int i = 0; i < 4; ++i) {
                const int row = mi * 16 + gq + 8 * (i & 1);
                const int k = j * 16 + 2 * cq + 8 * (i >> 1);
                *reinterpret_cast<uint32_t *>(a_tile + sw128_off(row, k)) = a[i];
              }
            }
          } else {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              const uint2 w2 = *reinterpret_cast<const uint2 *>(codes + q * kLrStepBytes + (mi * 32 + lane) * 8);
              uint32_t a[4];
              unpack_int8x8(w2.x, w2.y, a);
#pragma unroll
              for (int i = 0; i < 4; ++i) {
                const int row = mi * 16 + gq + 8 * (i & 1);
                const int k = q * 16 + 2 * cq + 8 * (i >> 1);
                *reinterpret_cast<uint32_t *>(a_tile + sw128_off(row, k)) = a[i];
              }
            }
          }
        }
        fence_proxy_async_smem();  // make the generic-proxy stores visible to the tensor core
        __syncwarp();
        if (lane == 0) mbar_arrive(&a_full[s]);
        if (++s == kPfStages) s = 0, ph ^= 1;
      }
    }
  } else {
    // ------------------------------ promotion + epilogue ------------------------------
    if constexpr (kMode != 0)
      asm volatile("setmaxnreg.inc.sync.aligned.u32 184;\n" ::: "memory");
    else
      asm volatile("setmaxnreg.inc.sync.aligned.u32 168;\n" ::: "memory");
    const int pw = warp - 8;
    const int lg = pw & 3;            // TMEM lane group (rows 32*lg .. 32*lg+31)
    const int ch = pw >> 2;           // column half (tokens 128*ch .. 128*ch+127)
    const int r_in_tile = lg * 32 + lane;
    // Cross entropy and greedy read TMEM in the 16x256b shape (4 rows x 32
    // tokens per thread; cross entropy accumulates in base 2, its factors
    // times log2 e); logits read 32x32b (one row x 128 tokens per thread).
    constexpr bool kQuad = kMode != 0;
    int bcount = 0;
    for (int t = blockIdx.x; t < num_tiles; t += gridDim.x) {
      const int vt = t / p.num_mt, mt = t % p.num_mt;
      const int m0 = mt * kPfN + ch * 128;
      const int64_t row = (int64_t)vt * kTileRows + r_in_tile;
      float acc[128];
#pragma unroll
      for (int i = 0; i < 128; ++i) acc[i] = 0.f;
      const int nb = bp.nblocks();
      for (int b = 0; b < nb; ++b) {
        // Promotion factor of block b for the thread's row(s) of the tile.
        float f[kQuad ? 4 : 1];
        if constexpr (kQuad) {
          // Rows lane / 4 + 8k of the warp's 32: one base pointer, offsets 8k.
          const int rt0 = lg * 32 + (lane >> 2);
          const uint16_t *fs = nullptr;
          if (b < bp.nres)
            fs = kSC4 ? p.s_row + (int64_t)vt * kTileRows + rt0
                      : p.scales + ((int64_t)vt * p.G_pad + b) * kTileRows + rt0;
          else if (!(b == bp.nres && bp.core_sub > 0)) fs = p.s_a + (int64_t)vt * kTileRows + rt0;
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            f[k] = fs ? fp16_bits_to_f32(fs[8 * k]) : 1.f;
            if (kMode == 1) f[k] *= kLog2e;
          }
        } else {
          if (b < bp.nres)
            f[0] = kSC4 ? fp16_bits_to_f32(p.s_row[row])
                        : fp16_bits_to_f32(p.scales[((int64_t)vt * p.G_pad + b) * kTileRows + r_in_tile]);
          else if (b == bp.nres && bp.core_sub > 0) f[0] = 1.f;
          else f[0] = fp16_bits_to_f32(p.s_a[row]);
        }
        const int buf = bcount & 1;
        if (!mbar_wait_warp(&acc_full[buf], (bcount >> 1) & 1, p.wait_budget, abort_flag, p.err)) goto done;
        tc_fence_after();
        const uint32_t taddr = tmem_base + ((uint32_t)(lg * 32) << 16) + buf * kPfN + ch * 128;
        if constexpr (kQuad) {
          // acc[64h + 4kk + j] = row 8 (2h + (j >> 1)) + lane / 4 of the warp's
          // 32, token column 8kk + 2 (lane % 4) + (j & 1), kk = 0..15.
#pragma unroll
          for (int h = 0; h < 2; ++h) {
#pragma unroll
            for (int cc = 0; cc < 4; ++cc) {
              float v[16];
              tmem_ld16x256b_x4(taddr + ((uint32_t)(16 * h) << 16) + cc * 32, v);
              float *a = acc + 64 * h + 16 * cc;
#pragma unroll
              for (int c = 0; c < 4; ++c) {
                fma2(a[4 * c], a[4 * c + 1], f[2 * h], v[4 * c], v[4 * c + 1]);
                fma2(a[4 * c + 2], a[4 * c + 3], f[2 * h + 1], v[4 * c + 2], v[4 * c + 3]);
              }
            }
          }
        } else {
#pragma unroll
          for (int c = 0; c < 4; ++c) {
            float v[32];
            tmem_ld32(taddr + c * 32, v);
#pragma unroll
            for (int i = 0; i < 32; i += 2) fma2(acc[c * 32 + i], acc[c * 32 + i + 1], f[0], v[i], v[i + 1]);
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&acc_empty[buf]);
        ++bcount;
      }
      // Epilogue: columns are tokens m0 + i, this thread's row is `row`.
      if (kMode == 0) {
        if (row < p.V) {
          const int mcount = p.M - m0 < 128 ? p.M - m0 : 128;  // tokens of this column half inside M
          if (p.out_fp32) {
            float *o = reinterpret_cast<float *>(p.out) + (int64_t)m0 * p.V + row;
#pragma unroll
            for (int i = 0; i < 128; ++i, o += p.V)
              if (i < mcount) *o = acc[i];
          } else {
            __nv_bfloat16 *o = reinterpret_cast<__nv_bfloat16 *>(p.out) + (int64_t)m0 * p.V + row;
#pragma unroll
            for (int i = 0; i < 128; ++i, o += p.V)
              if (i < mcount) *o = __float2bfloat16_rn(acc[i]);
          }
        }
      } else if (kMode == 2) {
        // Greedy partials: the largest logit of each token over the warp's 32
        // rows and its row (the lowest on ties).  Layout as for the cross
        // entropy below: rows rbase + ru + 8 kr of the 32 token columns
        // col(k) = 8 (k >> 1) + 2 cq + (k & 1); first over the thread's 4
        // rows (ascending, so the first maximum wins), then a butterfly over
        // lane bits 4, 3, 2 that halves the column set per step.
        const int rbase = vt * kTileRows + lg * 32;
        const int ru = lane >> 2, cq = lane & 3;
        if (rbase + 32 > p.V) {
#pragma unroll
          for (int i = 0; i < 128; ++i) {
            const int kr = 2 * (i >> 6) + ((i >> 1) & 1);
            if (rbase + ru + 8 * kr >= p.V) acc[i] = -INFINITY;
          }
        }
        float bv[32];
        int bi[32];
#pragma unroll
        for (int k = 0; k < 32; ++k) {
          const int i0 = 4 * (k >> 1) + (k & 1);
          const int r = rbase + ru;
          float v = acc[i0];
          int ix = r;
          if (acc[i0 + 2] > v) v = acc[i0 + 2], ix = r + 8;
          if (acc[i0 + 64] > v) v = acc[i0 + 64], ix = r + 16;
          if (acc[i0 + 66] > v) v = acc[i0 + 66], ix = r + 24;
          bv[k] = v;
          bi[k] = ix;
        }
#pragma unroll
        for (int n = 32, o = 16; n > 4; n >>= 1, o >>= 1) {
          const bool up = lane & o;
#pragma unroll
          for (int j = 0; j < n / 2; ++j) {
            const float kv = up ? bv[j + n / 2] : bv[j];
            const int ki = up ? bi[j + n / 2] : bi[j];
            const float gv = up ? bv[j] : bv[j + n / 2];
            const int gi = up ? bi[j] : bi[j + n / 2];
            const float rv = __shfl_xor_sync(0xffffffffu, gv, o);
            const int ri = __shfl_xor_sync(0xffffffffu, gi, o);
            const bool take = rv > kv || (rv == kv && ri < ki);
            bv[j] = take ? rv : kv;
            bi[j] = take ? ri : ki;
          }
        }
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const int m = m0 + 16 * ru + 8 * (j >> 1) + 2 * cq + (j & 1);
          if (m < p.M) p.ce_part[((int64_t)vt * 4 + lg) * p.M + m] = make_float2(bv[j], __int_as_float(bi[j]));
        }
      } else {
        // Layout (see the promotion): this thread holds rows rbase + ru + 8 kr
        // (kr = 0..3) of 32 token columns col(k) = 8 (k >> 1) + 2 cq + (k & 1),
        // k = 0..31, row kr of column k at acc[i0(k) + {0, 2, 64, 66}[kr]].
        const int64_t rbase = (int64_t)vt * kTileRows + lg * 32;
        const int ru = lane >> 2, cq = lane & 3;
        // Target logits first: a token whose target is one of this warp's 32
        // rows takes its value from the thread holding it (rare: about one
        // token in 37 per warp and tile, so the slow path is a warp-uniform
        // branch).  Lane (ru, cq) reads the targets of the columns it ends
        // with: 16 ru + 8 (j >> 1) + 2 cq + (j & 1), j = 0..3.
        int tg[4];
        bool hit = false;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const int m = m0 + 16 * ru + 8 * (j >> 1) + 2 * cq + (j & 1);
          const int64_t t64 = m < p.M ? (int64_t)p.targets[m] - p.row0 - rbase : -1;  // row within the warp's 32
          tg[j] = t64 >= 0 && t64 < 32 ? (int)t64 : -1;
          hit |= tg[j] >= 0;
        }
        if (__any_sync(0xffffffffu, hit)) {
#pragma unroll
          for (int col = 0; col < 128; ++col) {
            const int j = 2 * ((col >> 3) & 1) + (col & 1);
            const int owner = 4 * (col >> 4) + ((col >> 1) & 3);  // lane that read this column's target
            const int r = __shfl_sync(0xffffffffu, tg[j], owner);
            if (r >= 0) {  // warp-uniform
              const int i0 = 4 * (col >> 3) + (col & 1);
              const float mine = r & 16 ? (r & 8 ? acc[i0 + 66] : acc[i0 + 64]) : (r & 8 ? acc[i0 + 2] : acc[i0]);
              const float v = __shfl_sync(0xffffffffu, mine, 4 * (r & 7) + ((col >> 1) & 3));
              if (lane == owner) p.ce_tlogit[m0 + col] = v * kLn2;
            }
          }
        }
        // Rows past V (last tile only) enter as -FLT_MAX: weight 0 against any
        // logit, and a finite (max, count) when the warp holds no real row.
        if (rbase + 32 > p.V) {
#pragma unroll
          for (int i = 0; i < 128; ++i) {
            const int kr = 2 * (i >> 6) + ((i >> 1) & 1);
            if (rbase + ru + 8 * kr >= p.V) acc[i] = -FLT_MAX;
          }
        }
        // (max, sum of 2^(y - max)) of each column over the thread's 4 rows...
        float mx[32], sm[32];
#pragma unroll
        for (int k = 0; k < 32; ++k) {
          const int i0 = 4 * (k >> 1) + (k & 1);
          const float v0 = acc[i0], v1 = acc[i0 + 2], v2 = acc[i0 + 64], v3 = acc[i0 + 66];
          const float mk = fmaxf(fmaxf(v0, v1), fmaxf(v2, v3));
          mx[k] = mk;
          sm[k] = (ex2_approx(v0 - mk) + ex2_approx(v1 - mk)) + (ex2_approx(v2 - mk) + ex2_approx(v3 - mk));
        }
        // ...then over the 8 lanes with the same lane % 4 (lane bits 4, 3, 2)
        // by a butterfly that halves the column set per step: the lane with
        // bit o set keeps the upper half and merges the partner's copy of it.
        // Lane (ru, cq) ends with k = 4 ru + j, j = 0..3.
#pragma unroll
        for (int n = 32, o = 16; n > 4; n >>= 1, o >>= 1) {
          const bool up = lane & o;
#pragma unroll
          for (int j = 0; j < n / 2; ++j) {
            const float km = up ? mx[j + n / 2] : mx[j], ks = up ? sm[j + n / 2] : sm[j];
            const float gm = up ? mx[j] : mx[j + n / 2], gs = up ? sm[j] : sm[j + n / 2];
            const float rm = __shfl_xor_sync(0xffffffffu, gm, o), rs = __shfl_xor_sync(0xffffffffu, gs, o);
            lse2_merge(km, ks, rm, rs, mx[j], sm[j]);
          }
        }
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const int m = m0 + 16 * ru + 8 * (j >> 1) + 2 * cq + (j & 1);
          if (m < p.M) p.ce_part[((int64_t)vt * 4 + lg) * p.M + m] = make_float2(mx[j] * kLn2, sm[j]);
        }
      }
    }
  }
done:
  if (warp == 1 && mma_leader) {
    // Every MMA this thread issued has completed before TMEM is released.
    tc_commit(drain);
    mbar_wait(drain, 0, p.wait_budget, nullptr, p.err);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kPfTmemCols);
  }
}

// ------------------------------------------------------------------------
// Host side: tensor maps and launch.
// ------------------------------------------------------------------------
// One packed format's kernel instances (INT8 in prefill.cu, SC4 in prefill_sc4.cu).
template <bool kSC4>
cudaError_t launch_prefill_fmt(const archead_pack *pk, const void *x, int M, const uint16_t *T, void *out,
                               int out_fp32, bool argmax, const int32_t *targets, int row0, float2 *ce_part,
                               float *ce_tlogit, cudaStream_t s) {
  PrefillParams p{};
  if (!make_tma_map_bf16(&p.tmap_x, x, M, pk->d, 128)) return cudaErrorInvalidValue;
  const int kt = 2 * (pk->rcp + pk->rrp);
  if (kt > 0) {
    if (!make_tma_map_bf16(&p.tmap_t, T, M, kt, 128)) return cudaErrorInvalidValue;
  }
  p.codes = pk->codes;
  p.scales = pk->scales;
  p.scodes = pk->scodes;
  p.s_row = pk->s_row;
  p.sc4 = pk->sc4;
  p.G_pad2 = pk->G_pad2;
  p.lr_codes = pk->lr_codes;
  p.s_a = pk->s_a;
  p.V = pk->V;
  p.M = M;
  p.num_vt = pk->num_tiles;
  p.num_mt = (M + kPfN - 1) / kPfN;
  p.d_pad = pk->d_pad;
  p.G_pad = pk->G_pad;
  p.g = pk->g;
  p.nls = pk->nls;
  p.nls_core = pk->nls_core;
  p.rcp = pk->rcp;
  p.rrp = pk->rrp;
  p.out = out;
  p.out_fp32 = out_fp32;
  p.targets = targets;
  p.row0 = row0;
  p.ce_part = ce_part;
  p.ce_tlogit = ce_tlogit;
  p.err = pk->err;
  p.wait_budget = pk->wait_budget;
  const int tiles = p.num_vt * p.num_mt;
  const int grid = tiles < pk->sm_count ? tiles : pk->sm_count;
  if (out) {
    cudaError_t e = opt_in_smem(reinterpret_cast<const void *>(prefill_kernel<0, kSC4>), kPfSmem);
    if (e != cudaSuccess) return e;
    prefill_kernel<0, kSC4><<<grid, kPfThreads, kPfSmem, s>>>(p);
  } else if (argmax) {
    cudaError_t e = opt_in_smem(reinterpret_cast<const void *>(prefill_kernel<2, kSC4>), kPfSmem);
    if (e != cudaSuccess) return e;
    prefill_kernel<2, kSC4><<<grid, kPfThreads, kPfSmem, s>>>(p);
  } else {
    cudaError_t e = opt_in_smem(reinterpret_cast<const void *>(prefill_kernel<1, kSC4>), kPfSmem);
    if (e != cudaSuccess) return e;
    prefill_kernel<1, kSC4><<<grid, kPfThreads, kPfSmem, s>>>(p);
  }
  return cudaGetLastError();
}


}  // namespace archead
