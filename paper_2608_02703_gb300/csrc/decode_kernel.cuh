// Memory-bound decode kernel (up to 64 tokens per launch) of the packed
// LM-head forward (paper, Section 3.2, Eq. 7; Appendix B: the core and
// correction paths are evaluated separately and no dense head is formed).
//
// Persistent grid, one block per SM.  A unit of work is one to four 128-row
// vocabulary tiles (by kernel instance, below).  One producer warp streams
// each unit's INT4 codes, group scales and low-rank codes with 1-D bulk TMA
// copies into a ring of shared-memory stages (mbarrier full/empty pairs).
// Consumer warps each own 16-row m-tiles of the unit and 8-token n-tiles.
// For up to 8 tokens the hidden states are staged once per block by TMA and
// converted in place to fp16, each token scaled by a power of two that keeps
// it in fp16 range (exact for bf16 inputs in the normal range); wider
// instances stream x through the ring as bf16.  Per 16-wide k step a
// consumer turns one 32-bit word of offset-binary nibbles into the four
// A-fragment registers of an m16n8k16 MMA (exact biased integers, see
// unpack_int4x8_f16 / unpack_int4x8_biased) and multiplies them with the
// hidden states (B fragments, tokens on the 8-wide side), accumulating in
// fp32.  Each quantisation group starts from its bias term and is promoted
// by the row's group scale at its end (part sums added into acc); the
// 64-token instance, with no registers for part sums, keeps its
// accumulators in units of the current group's scale instead (each group
// multiplies them by the ratio of the previous scale to its own, and the last
// scale multiplies the finished residual once).  The rank-r branches follow
// as extra k steps: int8 codes of A_c (core) or A_w (correction) times the
// bf16 hi/lo split of t = x V from the pre-pass, the correction promoted by
// the row scale of A_w.  The pre-pass runs as the preceding grid; this
// kernel starts streaming under programmatic dependent launch and waits for
// the pre-pass only before the first rank-r stage.
//
// In the paper's packed format (SC4) a group scale is s_row * (q + 1) with a
// 4-bit code q: the group promotion multiplies by q + 1 (read from the
// stage's code bytes) and the row scale s_row, which the first rank-r stage
// carries, multiplies the finished residual once per row.
#pragma once

#include "device.cuh"
#include "internal.h"

namespace archead {

constexpr int kSmemLimit = 227 * 1024;

// Kernel instances ("variants"), chosen per launch from the token count and
// the head's width:
//  - kDecResident1: up to 8 tokens (one 8-token n-tile), hidden states staged
//    once in shared memory as fp16; kDecResidentH the same in units of two
//    tiles with four 64-wide chunks per stage (eight warps of two m-tiles in
//    the paper's format, sixteen of one in the INT8 format), for the paper's
//    format and for heads whose four-tile units leave the last round of
//    blocks poorly filled;
//  - kDecStreamed2: 9..16 tokens (two n-tiles), and up to 8 tokens of heads
//    so wide that x of 8 tokens does not fit next to a working ring.  The
//    hidden states are not kept in shared memory (16 rows of d would take
//    most of it, leaving too shallow a ring to stream at full bandwidth):
//    each residual stage also carries the matching 64-wide chunks of x for
//    16 tokens, loaded by a 2-D TMA copy, and the operands stay bf16 (no fp16
//    staging).  Its warps read codes and x from the stage as they compute and
//    release it afterwards (the registers to copy a stage out first are not
//    there with two n-tiles).  Sixteen consumer warps of two m-tiles each
//    (92.1 us at M = 16 against 94.2 with eight warps of four; for M <= 8 the
//    resident instance keeps eight warps: 67.7 against 73.8 us with sixteen).
//    kDecStreamedH the same in units of two tiles (sixteen warps of one
//    m-tile, four 64-wide chunks per stage), where d is whole stages of four
//    chunks: 89.5 against 92.1 us at M = 16 on the Qwen3-8B-shaped head,
//    100.5 against 110.7 on the Gemma-shaped one.  (The 32-token instance
//    with four-chunk stages was slower: 174 against 154 us.)
// Measured alternatives that were slower on the Qwen3-8B-shaped head (and not
// kept): 16 tokens of x resident as fp16 with a 2-chunk ring (98.4 us at
// M = 16 against 94.8) or a 1-chunk ring with the next stage prefetched into
// registers (114 us); 1-chunk stages for M <= 8 (98 us at M = 1 against 65).
//  - kDecWide4, kDecWide8: 17..32 and 33..64 tokens (four and eight n-tiles)
//    with x streamed as above; the head is streamed once per 32 resp. 64
//    tokens, in units of two tiles.  kDecWide4 runs sixteen consumer warps of
//    one m-tile each (registers for a group's part sums at 96 a thread).
//    kDecWide8 runs eight warps of two m-tiles each, so that every B
//    fragment read from shared memory feeds two MMAs: with one m-tile a warp
//    the ldmatrix traffic held it at 277 us for 64 tokens on the
//    Qwen3-8B-shaped head, against 247 us.  Its 64 accumulators leave no
//    registers for part sums: it keeps them in units of the group scale.
//    Measured and not kept: kDecWide4 with eight warps of four m-tiles in
//    group-scale units (145-152 us for 17-32 tokens, no better; 207 us with
//    the paper's format, which spilled), and kDecWide8 with sixteen warps of
//    two m-tiles and four n-tiles each (265-278 us).
enum DecodeVariant {
  kDecResident1 = 0, kDecStreamed2 = 1, kDecWide4 = 2, kDecWide8 = 3, kDecResidentH = 4, kDecStreamedH = 5
};

__host__ __device__ constexpr int variant_nt(int v) {  // 8-token n-tiles
  return v == kDecResident1 || v == kDecResidentH ? 1 : v == kDecStreamed2 || v == kDecStreamedH ? 2 : v == kDecWide4 ? 4 : 8;
}
// Consumer warps and m-tiles per warp; kDecResidentH runs sixteen warps of
// one m-tile for the INT8 format (Gemma-shaped head: 77.4 against 79.3 us at
// M = 1) and eight of two for the paper's format (64.1 against 68.0 us).
__host__ __device__ constexpr int variant_cw(int v, bool sc4 = false) {
  return v == kDecStreamed2 || v == kDecStreamedH || v == kDecWide4 || (v == kDecResidentH && !sc4) ? 16 : 8;
}
__host__ __device__ constexpr int variant_mt(int v, bool sc4 = false) {  // 16-row m-tiles per consumer warp
  return v == kDecResident1 ? 4 : v == kDecWide4 || v == kDecStreamedH || (v == kDecResidentH && !sc4) ? 1 : 2;
}
// 128-row tiles per unit: the consumer warps cover them, MT m-tiles each.
__host__ __device__ constexpr int variant_tiles(int v) { return variant_cw(v) * variant_mt(v) / 8; }
__host__ __device__ constexpr int variant_threads(int v, bool sc4) { return (variant_cw(v, sc4) + 1) * 32; }  // + producer
__host__ __device__ constexpr int variant_tokens(int v) { return 8 * variant_nt(v); }  // largest M of one launch
__host__ __device__ constexpr bool streams_x(int v) { return v != kDecResident1 && v != kDecResidentH; }
// Token stride of the per-group sums of x (at least 16: the smallest instances' layout).
__host__ __device__ constexpr int xsum_tokens(int v) { return variant_tokens(v) < 16 ? 16 : variant_tokens(v); }
// 64-wide chunks of d per ring stage.  The shared-memory plan and the kernel
// instance launched both take it from here.
__host__ __device__ constexpr int stage_chunks(int v) { return v == kDecResidentH || v == kDecStreamedH ? 4 : 2; }
// One chunk of x in a stage: the instance's tokens x 64 of d, bf16, 128-byte swizzle.
__host__ __device__ constexpr int x_chunk_bytes(int v) { return variant_tokens(v) < 16 ? 16 * kChunkK * 2 : variant_tokens(v) * kChunkK * 2; }

// Stage geometry for SC chunks (64 of d each) per stage, TL tiles per unit
// and XB bytes of x per chunk (0: x not streamed).
template <int SC, int TL, int XB>
struct StageGeom {
  static constexpr int kCodeBytes = TL * SC * kChunkBytes;  // also holds 2*SC low-rank steps per tile
  static constexpr int kScaleBytesPerTile = (SC * kChunkK / 32) * kTileRows * 2;  // up to SC*64/g groups (g >= 32)
  static constexpr int kXOff = (kCodeBytes + TL * kScaleBytesPerTile + 1023) / 1024 * 1024;  // 1 KB aligned
  static constexpr int kBytes = kXOff + SC * XB;
  static constexpr int kLrSteps = 2 * SC;  // 16-wide low-rank steps per stage (2 KB per tile each)
};
template <int V>
using GeomOf = StageGeom<stage_chunks(V), variant_tiles(V), streams_x(V) ? x_chunk_bytes(V) : 0>;

struct DecodePlan {
  int stages, sc;
  size_t xs_off, ts_off, xsum_off, bar_off, total;
};

__host__ __device__ __forceinline__ int xs_row_elems(int d_pad) { return d_pad + 8; }  // +16 B: rows on distinct banks

// Shared memory: the stage ring, M rows of hidden states, the rank-r
// fragments, the per-group sums of x, and the barriers.  The total leaves
// room for one pre-pass block on the same SM (programmatic dependent launch
// overlaps the two grids) whenever the stage ring still holds 96 KB.
static DecodePlan decode_plan(int d_pad, int nls, int g, int M, int variant) {
  DecodePlan pl{};
  const bool xs = streams_x(variant);
  pl.sc = stage_chunks(variant);
  const size_t stage_bytes = variant == kDecResident1   ? GeomOf<kDecResident1>::kBytes
                             : variant == kDecStreamed2 ? GeomOf<kDecStreamed2>::kBytes
                             : variant == kDecWide4     ? GeomOf<kDecWide4>::kBytes
                             : variant == kDecWide8     ? GeomOf<kDecWide8>::kBytes
                             : variant == kDecResidentH ? GeomOf<kDecResidentH>::kBytes
                                                        : GeomOf<kDecStreamedH>::kBytes;
  const size_t xs_bytes = xs ? 0 : (size_t)M * xs_row_elems(d_pad) * 2;
  // rank-r fragments of the 16-token chunks the launch covers
  const size_t ts_bytes = (size_t)((variant_tokens(variant) + kDecodeMaxTokens - 1) / kDecodeMaxTokens) * nls * 1024;
  const size_t xsum_bytes = ((size_t)2 * (d_pad / g) * xsum_tokens(variant) + xsum_tokens(variant)) * 4;
  const size_t fixed = xs_bytes + ts_bytes + xsum_bytes + 256;
  const size_t shared_cap = (size_t)kSmemLimit - prepass_smem(M) - 2048;
  int st = 8;
  while (st >= 2 && fixed + (size_t)st * stage_bytes > shared_cap) --st;
  if (st < 2 || (size_t)st * stage_bytes < 96 * 1024) {  // too shallow a ring: give up co-residency
    st = 8;
    while (st >= 2 && fixed + (size_t)st * stage_bytes > (size_t)kSmemLimit) --st;
  }
  pl.stages = st;
  pl.xs_off = (size_t)st * stage_bytes;
  pl.ts_off = pl.xs_off + xs_bytes;
  pl.xsum_off = pl.ts_off + ts_bytes;
  pl.bar_off = pl.xsum_off + xsum_bytes;
  pl.total = pl.bar_off + 256;
  return pl;
}

// ldmatrix: four (two) 8x8 b16 matrices; lane L gives the address of row
// L % 8 of matrix L / 8.  Thread t receives row t / 4, elements 2 (t % 4) and
// 2 (t % 4) + 1 of each: the m16n8k16 B fragment when the rows are tokens
// and the 8 elements k values.
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2, uint32_t &r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x2(uint32_t addr, uint32_t &r0, uint32_t &r1) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0, %1}, [%2];\n" : "=r"(r0), "=r"(r1) : "r"(addr));
}

// acc += f_lo * part (rows gq) and f_hi * part (rows gq + 8).
template <int NT>
__device__ __forceinline__ void promote(float (&acc)[NT][4], const float (&part)[NT][4], float f_lo, float f_hi) {
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
    acc[nt][0] = fmaf(f_lo, part[nt][0], acc[nt][0]);
    acc[nt][1] = fmaf(f_lo, part[nt][1], acc[nt][1]);
    acc[nt][2] = fmaf(f_hi, part[nt][2], acc[nt][2]);
    acc[nt][3] = fmaf(f_hi, part[nt][3], acc[nt][3]);
  }
}

// q + 1 as a float for the 4-bit code at bit offset sh of byte b: 2^23 + q
// from the bit pattern, minus 2^23 - 1.
__device__ __forceinline__ float scale_mult(uint32_t b, int sh) {
  return __uint_as_float(0x4B000000u | ((b >> sh) & 15u)) - 8388607.0f;
}

// (q + 1) / 16 the same way: the code as the low mantissa bits of 2^19
// (unit 1/16), minus 2^19 - 1/16 (exact).
__device__ __forceinline__ float scale_mult_16th(uint32_t b, int sh) {
  return __uint_as_float(0x49000000u | ((b >> sh) & 15u)) - 524287.9375f;
}

// VAR: DecodeVariant (n-tiles of 8 tokens, resident or streamed x); SC:
// 64-wide chunks per stage; GS: 16-wide k steps per group.
template <int VAR, int SC, int GS, bool kSC4>
__global__ void __launch_bounds__(variant_threads(VAR, kSC4), 1) decode_kernel(const __grid_constant__ DecodeParams p, int stages,
                                                                int xs_off, int ts_off, int xsum_off, int bar_off) {
  constexpr int kDecWarps = variant_cw(VAR, kSC4);  // consumer warps
  constexpr int NT = variant_nt(VAR);          // n-tiles per warp
  constexpr bool kStreamX = streams_x(VAR);
  constexpr bool kF16 = !kStreamX;  // fp16 operands with x staged in shared memory
  constexpr int MT = variant_mt(VAR, kSC4);  // m-tiles per consumer warp
  static_assert(variant_cw(VAR, kSC4) * variant_mt(VAR, kSC4) == variant_cw(VAR) * variant_mt(VAR),
                "the unit size must not depend on the format");
  constexpr int TL = variant_tiles(VAR);     // 128-row tiles per unit
  constexpr int XT = xsum_tokens(VAR);       // token stride of the per-group sums
  constexpr int XCB = x_chunk_bytes(VAR);    // one chunk of streamed x
  using Geom = GeomOf<VAR>;
  constexpr int SS = 4 * SC;  // 16-wide k steps per stage
  constexpr bool kRatio = MT * NT > 8;  // accumulators in units of the group scale (no part sums)
  // The kernel has no static shared memory, so the dynamic window starts on a
  // 1 KB boundary, which the 128-byte-swizzled x boxes rely on (checked
  // below).  Offsets from this base stay compile-time friendly; a rounded-up
  // runtime base made the inner loops measurably slower.
  extern __shared__ __align__(1024) uint8_t smem[];
  if (kStreamX && (smem_u32(smem) & 1023u) != 0) {
    if (threadIdx.x == 0) atomicOr(p.err, kErrLayout);
    return;
  }
  uint16_t *xs_s = reinterpret_cast<uint16_t *>(smem + xs_off);
  const uint32_t *ts_s = reinterpret_cast<const uint32_t *>(smem + ts_off);
  // [group][16 tokens] -1032 * sum of x, then the same with -1152, then the
  // 16 tokens' scale factors (powers of two) that undo the fp16 staging scale.
  float *xsum_s = reinterpret_cast<float *>(smem + xsum_off);
  uint64_t *full = reinterpret_cast<uint64_t *>(smem + bar_off);
  uint64_t *empty = full + 8;
  uint64_t *xbar = full + 16;
  uint64_t *tbar = full + 17;
  volatile int *abort_flag = reinterpret_cast<volatile int *>(full + 18);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int KC = p.d_pad / kChunkK;
  const int res_stages = KC / SC;
  const int lr_stages = (p.nls + Geom::kLrSteps - 1) / Geom::kLrSteps;
  const int num_units = (p.num_tiles + TL - 1) / TL;
  const int xrow = xs_row_elems(p.d_pad);

  // Columns [d, d_pad) of the hidden states meet zero codes; zero them so
  // that no stale pattern (a NaN) reaches the accumulators.
  if (!kStreamX && p.d < p.d_pad) {
    const int per_row = (p.d_pad - p.d) / 8;  // uint4 per row
    for (int e = threadIdx.x; e < p.M * per_row; e += blockDim.x) {
      uint4 *dst = reinterpret_cast<uint4 *>(smem + xs_off + (size_t)(e / per_row) * xrow * 2 + (size_t)p.d * 2);
      dst[e % per_row] = make_uint4(0, 0, 0, 0);
    }
  }
  if (threadIdx.x == 0) {
    for (int i = 0; i < stages; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], kDecWarps);
    }
    mbar_init(xbar, 1);
    mbar_init(tbar, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();

  if (warp == kDecWarps) {
    // ---------------- producer warp ----------------
    // The whole warp runs the loop (voted waits keep it warp-uniform) and one
    // elected lane issues the copies: a single-lane loop issues bulk copies
    // several times more slowly.
    const bool leader = elect_one();
    // The head is read once per forward: keep it from evicting the small
    // data the pre-pass grid reads at the same time.
    const uint64_t stream_policy = make_evict_first_policy();
    if (!kStreamX && leader) {
      mbar_arrive_expect_tx(xbar, (uint32_t)(p.M * p.d * 2));
      for (int m = 0; m < p.M; ++m)
        bulk_g2s(smem + xs_off + (size_t)m * xrow * 2, p.x + (size_t)(p.m0 + m) * p.d, (uint32_t)(p.d * 2), xbar);
    }
    bool t_loaded = false;
    int it = 0;
    for (int unit = blockIdx.x; unit < num_units; unit += gridDim.x) {
      const int ntile = min(TL, p.num_tiles - TL * unit);
      for (int s = 0; s < res_stages + lr_stages; ++s, ++it) {
        const int st = it % stages;
        if (s == res_stages && !t_loaded) {
          // The rank-r fragments come from the pre-pass grid.
          asm volatile("griddepcontrol.wait;\n" ::: "memory");
          if (leader) {  // the t fragments of the 16-token chunks this launch holds
            const uint32_t tb = (uint32_t)(((p.M + kDecodeMaxTokens - 1) / kDecodeMaxTokens) * p.nls * 1024);
            mbar_arrive_expect_tx(tbar, tb);
            bulk_g2s(smem + ts_off, p.ts, tb, tbar);
          }
          t_loaded = true;
        }
        if (!mbar_wait_warp(&empty[st], ((it / stages) & 1) ^ 1, p.wait_budget, abort_flag, p.err))
          goto producer_abort;
        uint8_t *buf = smem + (size_t)st * Geom::kBytes;
        if (!leader) {
        } else if (s < res_stages) {
          const int kc0 = s * SC;
          const int g0 = (kc0 * kChunkK) / p.g;
          const int g1 = ((kc0 + SC) * kChunkK - 1) / p.g;
          const int ng = g1 - g0 + 1;
          // SC4: byte rows g0/2 .. g1/2 of the tile's scale codes instead of fp16 scales.
          const int nbr = (g1 >> 1) - (g0 >> 1) + 1;
          const int sbytes = kSC4 ? nbr * kTileRows : ng * kTileRows * 2;
          mbar_arrive_expect_tx(&full[st],
                                (uint32_t)(ntile * (SC * kChunkBytes + sbytes) + (kStreamX ? SC * XCB : 0)));
          if (kStreamX) {
            for (int c = 0; c < SC; ++c)
              tma_load_2d(buf + Geom::kXOff + c * XCB, &p.tmap_x, (kc0 + c) * kChunkK, p.m0, &full[st]);
          }
          for (int t = 0; t < ntile; ++t) {
            const int64_t vt = (int64_t)TL * unit + t;
            bulk_g2s_hint(buf + t * SC * kChunkBytes, p.codes + (vt * KC + kc0) * kChunkBytes, SC * kChunkBytes,
                          &full[st], stream_policy);
            if constexpr (kSC4)
              bulk_g2s_hint(buf + Geom::kCodeBytes + t * Geom::kScaleBytesPerTile,
                            p.scodes + (vt * p.G_pad2 + (g0 >> 1)) * kTileRows, sbytes, &full[st], stream_policy);
            else
              bulk_g2s_hint(buf + Geom::kCodeBytes + t * Geom::kScaleBytesPerTile,
                            p.scales + (vt * p.G_pad + g0) * kTileRows, sbytes, &full[st], stream_policy);
          }
        } else {
          const int ls0 = (s - res_stages) * Geom::kLrSteps;
          const int nl = min(Geom::kLrSteps, p.nls - ls0);
          // Narrow instances read the correction's row scales from the last
          // rank-r stage; SC4 row scales ride on the first.
          const bool last = !kRatio && s == res_stages + lr_stages - 1;
          const bool first_sc4 = kSC4 && s == res_stages;
          mbar_arrive_expect_tx(&full[st], (uint32_t)(ntile * (nl * kLrStepBytes + (last ? kTileRows * 2 : 0) +
                                                                (first_sc4 ? kTileRows * 2 : 0))));
          for (int t = 0; t < ntile; ++t) {
            const int64_t vt = (int64_t)TL * unit + t;
            bulk_g2s_hint(buf + t * Geom::kLrSteps * kLrStepBytes, p.lr_codes + (vt * p.nls + ls0) * kLrStepBytes,
                          nl * kLrStepBytes, &full[st], stream_policy);
            if (last)
              bulk_g2s(buf + Geom::kCodeBytes + t * Geom::kScaleBytesPerTile, p.s_a + vt * kTileRows, kTileRows * 2,
                       &full[st]);
            if (first_sc4)
              bulk_g2s(buf + Geom::kCodeBytes + t * Geom::kScaleBytesPerTile + kTileRows * 2, p.s_row + vt * kTileRows,
                       kTileRows * 2, &full[st]);
          }
        }
        __syncwarp();
      }
    }
    return;
  producer_abort:
    // Let copies already issued land before the block exits.
    for (int k = 1; k <= stages && it - k >= 0; ++k) {
      const int j = it - k;
      mbar_wait_warp(&full[j % stages], (j / stages) & 1, p.wait_budget, nullptr, p.err);
    }
    if (!kStreamX) mbar_wait_warp(xbar, 0, p.wait_budget, nullptr, p.err);
    if (t_loaded) mbar_wait_warp(tbar, 0, p.wait_budget, nullptr, p.err);
    return;
  }

  // ---------------- consumer warps ----------------
  const int tsel = warp / (8 / MT);          // tile of the unit
  const int mi0 = (warp % (8 / MT)) * MT;    // first of the warp's m-tiles in that tile
  const int gq = lane >> 2, cq = lane & 3;
  const int ng = p.d_pad / p.g;
  float *tscale = xsum_s + 2 * ng * XT;
  if (kStreamX) {
    // Per-group sums of x for removing the bf16 operand bias (136), read
    // straight from global memory; no staging scale.
    for (int e = threadIdx.x; e < ng * XT; e += kDecWarps * 32) {
      const int grp = e / XT, m = e % XT;
      float sum = 0.f;
      if (m < p.M && grp * p.g < p.d) {
        const uint4 *src = reinterpret_cast<const uint4 *>(p.x + (int64_t)(p.m0 + m) * p.d + (int64_t)grp * p.g);
        for (int q = 0; q < p.g / 8; ++q) {
          const uint4 v = src[q];
          sum += bf16_lo(v.x) + bf16_hi(v.x) + bf16_lo(v.y) + bf16_hi(v.y);
          sum += bf16_lo(v.z) + bf16_hi(v.z) + bf16_lo(v.w) + bf16_hi(v.w);
        }
      }
      xsum_s[e] = -kInt4Bias * sum;
      xsum_s[ng * XT + e] = -kInt4Bias * sum;
    }
    if (threadIdx.x < XT) tscale[threadIdx.x] = 1.f;
    asm volatile("bar.sync 1, %0;\n" ::"r"(kDecWarps * 32) : "memory");  // consumer warps only
  } else {
    const bool ok = mbar_wait_warp(xbar, 0, p.wait_budget, abort_flag, p.err);
    if (ok) {
      // Per-token power of two 2^-e that brings max |x| into [2^14, 2^15)
      // (fp16 range, and small tokens away from fp16 subnormals); tscale[m]
      // = 2^e undoes it after the residual.
      for (int m = warp; m < XT; m += kDecWarps) {
        uint32_t mx = 0;
        if (m < p.M) {
          const uint32_t *row = reinterpret_cast<const uint32_t *>(xs_s + m * xrow);
          for (int k = lane; k < p.d_pad / 2; k += 32) {
            const uint32_t v = row[k];
            mx = max(mx, max(v & 0x7FFFu, (v >> 16) & 0x7FFFu));
          }
        }
        mx = __reduce_max_sync(0xffffffffu, mx);
        const int ex = (int)(mx >> 7);             // biased bf16 exponent of the largest |x|
        const int e = max(ex - 141, -126);       // max |x| < 2^(ex-126); 2^-e of it lies below 2^15
        if (lane == 0) tscale[m] = __uint_as_float((uint32_t)(127 + e) << 23);
      }
      asm volatile("bar.sync 1, %0;\n" ::"r"(kDecWarps * 32) : "memory");
      // Convert each token's row to fp16 in place, group by group, and sum
      // the values the MMAs will see (for removing the operand bias).
      for (int e = threadIdx.x; e < ng * XT; e += kDecWarps * 32) {
        const int grp = e / XT, m = e % XT;
        float sum = 0.f;
        if (m < p.M) {
          const float inv = 1.f / tscale[m];  // exact: a power of two
          uint32_t *row = reinterpret_cast<uint32_t *>(xs_s + m * xrow + grp * p.g);
          for (int k = 0; k < p.g / 2; ++k) {
            const uint32_t v = row[k];
            const __half2 h = __floats2half2_rn(bf16_lo(v) * inv, bf16_hi(v) * inv);
            row[k] = *reinterpret_cast<const uint32_t *>(&h);
            sum += __low2float(h);
            sum += __high2float(h);
          }
        }
        xsum_s[e] = -kF16BiasLo * sum;
        xsum_s[ng * XT + e] = -kF16BiasHi * sum;
      }
    }
    asm volatile("bar.sync 1, %0;\n" ::"r"(kDecWarps * 32) : "memory");  // consumer warps only
    if (!ok) return;
  }
  // Factors that undo the staging scale for this lane's two token columns.
  float2 unscale[NT];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt)
    unscale[nt] = make_float2(tscale[8 * nt + 2 * cq], tscale[8 * nt + 2 * cq + 1]);
  // B-fragment bases: token 8*nt + gq (clamped to the M rows held; the extra
  // columns are never stored), column 2*cq (+ 16 per k step, + 8 for b1).
  const uint16_t *xb[NT];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) xb[nt] = kStreamX ? nullptr : xs_s + min(8 * nt + gq, p.M - 1) * xrow + 2 * cq;
  // ldmatrix row address of this lane (one token tile): token L % 8 (clamped
  // to the M rows held), k offset 8 (L / 8) % 2.
  const uint16_t *xl = kStreamX || !kSC4 ? nullptr : xs_s + min(lane & 7, p.M - 1) * xrow + 8 * ((lane >> 3) & 1);
  bool t_ready = false;

  int st = 0;     // ring slot
  uint32_t ph = 0;  // its phase parity
  for (int unit = blockIdx.x; unit < num_units; unit += gridDim.x) {
    const int ntile = min(TL, p.num_tiles - TL * unit);
    const bool active = tsel < ntile;
    // Narrow instances (MT * NT <= 8) sum each quantisation group in part,
    // starting from the group's bias term, and promote it into acc by the
    // group scale at the group's end.  Wide instances have no registers for
    // a second set: their accumulators hold the running sum in units of the
    // current group's scale (each group starts by multiplying them by
    // previous scale / this scale and adding the bias term, and the last
    // group's scale multiplies the finished residual once).  There a zero
    // group scale counts as 1: the pack stores zero codes for such groups.
    float acc[MT][NT][4];
    float part[kRatio ? 1 : MT][kRatio ? 1 : NT][4];
    float sp_lo[MT], sp_hi[MT];  // wide: the previous group's scale (rows gq, gq + 8)
#pragma unroll
    for (int a = 0; a < MT; ++a) {
      sp_lo[a] = sp_hi[a] = 0.f;
#pragma unroll
      for (int b = 0; b < NT; ++b)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[a][b][c] = 0.f;
    }
#pragma unroll
    for (int a = 0; a < (kRatio ? 1 : MT); ++a)
#pragma unroll
      for (int b = 0; b < (kRatio ? 1 : NT); ++b)
#pragma unroll
        for (int c = 0; c < 4; ++c) part[a][b][c] = 0.f;
    // Row scales of the correction branch (A_w).  Wide instances read them
    // here and run the correction's k steps on acc / s_a, multiplying back by
    // s_a at the end (a zero scale counts as 1; the pack stores zero codes
    // for such rows).  Narrow instances take them from the last rank-r stage.
    float a_lo[MT], a_hi[MT];
#pragma unroll
    for (int mt = 0; mt < MT; ++mt) a_lo[mt] = a_hi[mt] = 1.f;
    if (kRatio && active && p.has_corr) {
      const int64_t rb = ((int64_t)TL * unit + tsel) * kTileRows + mi0 * 16 + gq;
#pragma unroll
      for (int mt = 0; mt < MT; ++mt) {
        a_lo[mt] = fp16_bits_to_f32(p.s_a[rb + mt * 16]);
        a_hi[mt] = fp16_bits_to_f32(p.s_a[rb + mt * 16 + 8]);
        a_lo[mt] = a_lo[mt] == 0.f ? 1.f : a_lo[mt];
        a_hi[mt] = a_hi[mt] == 0.f ? 1.f : a_hi[mt];
      }
    }

    // Residual: INT4 codes, one scale per row and group.  With x resident,
    // each warp copies its share of a stage (codes and group scales) to
    // registers and releases the slot at once, so the producer can refill it
    // while the warp computes; with x streamed, it releases the slot after its
    // k steps.
    constexpr int NGS = GS <= SS ? SS / GS : 1;  // groups whose scales a stage carries
    for (int s = 0; s < res_stages; ++s) {
      if (!mbar_wait_warp(&full[st], ph, p.wait_budget, abort_flag, p.err)) return;
      uint4 w[kStreamX ? 1 : SC][MT];
      float s_lo[NGS][MT], s_hi[NGS][MT];
      const uint8_t *sbuf = smem + (size_t)st * Geom::kBytes;
      const uint8_t *cb = sbuf + tsel * SC * kChunkBytes + mi0 * 512 + lane * 16;
      if (active) {
        const uint8_t *sarea = sbuf + Geom::kCodeBytes + tsel * Geom::kScaleBytesPerTile;
        const uint16_t *sc = reinterpret_cast<const uint16_t *>(sarea) + mi0 * 16 + gq;
        if (!kStreamX) {
#pragma unroll
          for (int c = 0; c < (kStreamX ? 1 : SC); ++c)
#pragma unroll
            for (int mt = 0; mt < MT; ++mt)
              w[c][mt] = *reinterpret_cast<const uint4 *>(cb + c * kChunkBytes + mt * 512);
        }
        if constexpr (kSC4) {
          // Group ggl's code: byte row ggl/2 - gfirst/2 of the stage, nibble ggl % 2.
          const int gfirst = GS <= SS ? s * (SS / GS) : s / (GS / SS);
          const uint8_t *sc8 = sarea + mi0 * 16 + gq;
#pragma unroll
          for (int gi = 0; gi < NGS; ++gi) {
            const int ggl = gfirst + gi;
            const int br = (ggl >> 1) - (gfirst >> 1), sh = 4 * (ggl & 1);
#pragma unroll
            for (int mt = 0; mt < MT; ++mt) {
              s_lo[gi][mt] = scale_mult(sc8[br * kTileRows + mt * 16], sh);
              const uint32_t bh = sc8[br * kTileRows + mt * 16 + 8];
              s_hi[gi][mt] = kF16 ? scale_mult_16th(bh, sh) : scale_mult(bh, sh);  // fp16 operands: x16 rows
            }
          }
        } else {
#pragma unroll
          for (int gi = 0; gi < NGS; ++gi)
#pragma unroll
            for (int mt = 0; mt < MT; ++mt) {
              const float lo = fp16_bits_to_f32(sc[gi * kTileRows + mt * 16]);
              const float hi = fp16_bits_to_f32(sc[gi * kTileRows + mt * 16 + 8]);
              s_lo[gi][mt] = kRatio && lo == 0.f ? 1.f : lo;
              s_hi[gi][mt] = (kRatio && hi == 0.f ? 1.f : hi) * (kF16 ? 0.0625f : 1.f);  // fp16: x16
            }
        }
        // Wide: from here s_lo/s_hi hold the ratios to the previous group's scale.
#pragma unroll
        for (int gi = 0; gi < (kRatio ? NGS : 0); ++gi)
#pragma unroll
          for (int mt = 0; mt < MT; ++mt) {
            const float lo = s_lo[gi][mt], hi = s_hi[gi][mt];
            s_lo[gi][mt] = __fdividef(sp_lo[mt], lo);
            s_hi[gi][mt] = __fdividef(sp_hi[mt], hi);
            sp_lo[mt] = lo;
            sp_hi[mt] = hi;
          }
      }
      const int st_done = st;
      if (!kStreamX || !active) {
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty[st]);
      }
      if (++st == stages) st = 0, ph ^= 1;
      if (!active) continue;
      const int kbase = s * SS * 16;
#pragma unroll
      for (int c = 0; c < SC; ++c) {
        if (kStreamX) {
#pragma unroll
          for (int mt = 0; mt < MT; ++mt)
            w[0][mt] = *reinterpret_cast<const uint4 *>(cb + c * kChunkBytes + mt * 512);
        }
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const int ks = c * 4 + j;  // k step within the stage
          uint32_t b[NT][2];
          if constexpr (kStreamX && NT >= 2) {
            // Per 16 tokens q: matrices (tokens 16q + 0-7 | 8-15) x (k 0-7 |
            // 8-15) of the k step: lane L addresses token 16q + 8 (L / 16) +
            // L % 8 at 16-byte chunk 2j + (L / 8) % 2 of its 128-byte row
            // (chunk index XOR token % 8).
#pragma unroll
            for (int q = 0; q < NT / 2; ++q) {
              const int tok = 16 * q + 8 * (lane >> 4) + (lane & 7);
              ldsm_x4(smem_u32(sbuf + Geom::kXOff + c * XCB + tok * 128 +
                               (((2 * j + ((lane >> 3) & 1)) ^ (tok & 7)) << 4)),
                      b[2 * q][0], b[2 * q][1], b[2 * q + 1][0], b[2 * q + 1][1]);
            }
          } else if constexpr (!kStreamX && NT == 1 && kSC4) {
            // Tokens 0-7 (clamped to M) x (k 0-7 | 8-15) of the k step.  (The
            // INT8 format's resident instance keeps its two 32-bit loads: its
            // whole forward measured 0.4 us slower with ldmatrix here, the SC4
            // instance's 1.2 us faster.)
            ldsm_x2(smem_u32(xl + kbase + ks * 16), b[0][0], b[0][1]);
          } else {
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
              if (kStreamX) {
                const uint8_t *xr = sbuf + Geom::kXOff + c * XCB + (8 * nt + gq) * 128 + 4 * cq;
                b[nt][0] = *reinterpret_cast<const uint32_t *>(xr + (((2 * j) ^ gq) << 4));
                b[nt][1] = *reinterpret_cast<const uint32_t *>(xr + (((2 * j + 1) ^ gq) << 4));
              } else {
                const uint16_t *q = xb[nt] + kbase + ks * 16;
                b[nt][0] = *reinterpret_cast<const uint32_t *>(q);
                b[nt][1] = *reinterpret_cast<const uint32_t *>(q + 8);
              }
            }
          }
          // First k step of a group (compile-time when groups fit in a stage).
          // Its MMAs start from the group's bias term nb = -(operand bias) *
          // sum of x over the group, per token, for rows gq (bias 1032, or 136
          // for bf16) and gq + 8 (1152 or 136), so that the group adds its
          // exact-code dot product: narrow, part = nb (the MMA's C operand);
          // wide, acc = acc * (previous scale / this scale) + nb.
          const bool first = GS <= SS ? (ks % GS == 0) : (ks == 0 && (s % (GS / SS)) == 0);
          float2 nb_lo[kRatio ? 1 : NT], nb_hi[kRatio ? 1 : NT];
          if (first && !kRatio) {
            const int ggl = GS <= SS ? s * (SS / GS) + ks / GS : s / (GS / SS);
#pragma unroll
            for (int nt = 0; nt < (kRatio ? 1 : NT); ++nt) {
              const int o = ggl * XT + 8 * nt + 2 * cq;
              nb_lo[nt] = *reinterpret_cast<const float2 *>(xsum_s + o);
              nb_hi[nt] = kStreamX ? nb_lo[nt] : *reinterpret_cast<const float2 *>(xsum_s + ng * XT + o);
            }
          }
          if (first && kRatio) {
            const int ggl = GS <= SS ? s * (SS / GS) + ks / GS : s / (GS / SS);  // group index along d
            const int gi = GS <= SS ? ks / GS : 0;                                // group within the stage
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
              const int o = ggl * XT + 8 * nt + 2 * cq;
              const float2 nb_lo = *reinterpret_cast<const float2 *>(xsum_s + o);
              // bf16 operands carry one bias (136) on both row halves
              const float2 nb_hi = kStreamX ? nb_lo : *reinterpret_cast<const float2 *>(xsum_s + ng * XT + o);
#pragma unroll
              for (int mt = 0; mt < MT; ++mt) {
                acc[mt][nt][0] = fmaf(acc[mt][nt][0], s_lo[gi][mt], nb_lo.x);
                acc[mt][nt][1] = fmaf(acc[mt][nt][1], s_lo[gi][mt], nb_lo.y);
                acc[mt][nt][2] = fmaf(acc[mt][nt][2], s_hi[gi][mt], nb_hi.x);
                acc[mt][nt][3] = fmaf(acc[mt][nt][3], s_hi[gi][mt], nb_hi.y);
              }
            }
          }
#pragma unroll
          for (int mt = 0; mt < MT; ++mt) {
            const uint4 wv = w[kStreamX ? 0 : c][mt];
            const uint32_t word = j == 0 ? wv.x : j == 1 ? wv.y : j == 2 ? wv.z : wv.w;
            uint32_t a[4];
            if (kF16)
              unpack_int4x8_f16(word, a);
            else
              unpack_int4x8_biased(word, a);
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
              if constexpr (kRatio) {
                if (kF16)
                  mma_f16_16816(acc[mt][nt], a, b[nt][0], b[nt][1]);
                else
                  mma_bf16_16816(acc[mt][nt], a, b[nt][0], b[nt][1]);
              } else {
                float (&pt)[4] = part[kRatio ? 0 : mt][kRatio ? 0 : nt];
                if (kF16) {
                  if (first)
                    mma_f16_16816_c(pt, a, b[nt][0], b[nt][1], nb_lo[kRatio ? 0 : nt], nb_hi[kRatio ? 0 : nt]);
                  else
                    mma_f16_16816(pt, a, b[nt][0], b[nt][1]);
                } else {
                  if (first)
                    mma_bf16_16816_c(pt, a, b[nt][0], b[nt][1], nb_lo[kRatio ? 0 : nt], nb_hi[kRatio ? 0 : nt]);
                  else
                    mma_bf16_16816(pt, a, b[nt][0], b[nt][1]);
                }
              }
            }
          }
          // Narrow: group boundary (compile-time inside a stage when GS <= SS;
          // every GS/SS stages otherwise): promote part by the group scale.
          if constexpr (!kRatio) {
            const bool boundary = GS <= SS ? ((ks + 1) % GS == 0) : (ks == SS - 1 && ((s + 1) % (GS / SS)) == 0);
            if (boundary) {
              const int gi = GS <= SS ? ks / GS : 0;  // group within the stage
#pragma unroll
              for (int mt = 0; mt < MT; ++mt) promote<NT>(acc[mt], part[mt], s_lo[gi][mt], s_hi[gi][mt]);
            }
          }
        }
      }
      if (kStreamX) {
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty[st_done]);
      }
    }

    // The last group's scale, and back to the hidden states' own scale
    // (exact: powers of two).
#pragma unroll
    for (int a = 0; a < MT; ++a)
#pragma unroll
      for (int b = 0; b < NT; ++b) {
        const float ux = kF16 ? unscale[b].x : 1.f, uy = kF16 ? unscale[b].y : 1.f;
        const float fl = kRatio ? sp_lo[a] : 1.f, fh = kRatio ? sp_hi[a] : 1.f;
        acc[a][b][0] *= fl * ux;
        acc[a][b][1] *= fl * uy;
        acc[a][b][2] *= fh * ux;
        acc[a][b][3] *= fh * uy;
      }
    // SC4 without rank-r branches: no stage carries the row scales; read them here.
    if (kSC4 && lr_stages == 0 && active) {
      const int64_t rb = ((int64_t)TL * unit + tsel) * kTileRows + mi0 * 16 + gq;
#pragma unroll
      for (int mt = 0; mt < MT; ++mt) {
        const float r_lo = fp16_bits_to_f32(p.s_row[rb + mt * 16]), r_hi = fp16_bits_to_f32(p.s_row[rb + mt * 16 + 8]);
#pragma unroll
        for (int b = 0; b < NT; ++b) {
          acc[mt][b][0] *= r_lo;
          acc[mt][b][1] *= r_lo;
          acc[mt][b][2] *= r_hi;
          acc[mt][b][3] *= r_hi;
        }
      }
    }

    // Rank-r branches as extra k steps, with the same copy-then-release of
    // each stage.  Columns k < core_cols of the steps are the core's, the
    // rest the correction's (row scale of A_w).  INT8 format: each step is
    // one branch's.  SC4 format: the branches lie back to back (the paper's
    // r_c = 10, r_r = 6 share one step), so a step may hold both: its A
    // operand is split by masks, the core part goes straight into acc
    // (factor 1), the correction's into part (narrow, promoted once at the
    // end) or into acc scaled by 1 / s_a before its first column (wide).
#pragma unroll
    for (int a = 0; a < (kRatio ? 1 : MT); ++a)
#pragma unroll
      for (int b = 0; b < (kRatio ? 1 : NT); ++b)
#pragma unroll
        for (int c = 0; c < 4; ++c) part[a][b][c] = 0.f;
    for (int s = 0; s < lr_stages; ++s) {
      if (!t_ready) {
        if (!mbar_wait_warp(tbar, 0, p.wait_budget, abort_flag, p.err)) return;
        t_ready = true;
      }
      if (!mbar_wait_warp(&full[st], ph, p.wait_budget, abort_flag, p.err)) return;
      const int ls0 = s * Geom::kLrSteps;
      const int nl = min(Geom::kLrSteps, p.nls - ls0);
      uint2 lw[Geom::kLrSteps][MT];
      if (active) {
        const uint8_t *buf = smem + (size_t)st * Geom::kBytes;
#pragma unroll
        for (int l = 0; l < Geom::kLrSteps; ++l)
#pragma unroll
          for (int mt = 0; mt < MT; ++mt)
            if (l < nl)
              lw[l][mt] = *reinterpret_cast<const uint2 *>(
                  buf + ((size_t)(tsel * Geom::kLrSteps + l) * 8 + mi0 + mt) * 256 + lane * 8);
        const uint16_t *sa = reinterpret_cast<const uint16_t *>(buf + Geom::kCodeBytes + tsel * Geom::kScaleBytesPerTile);
        if (!kRatio && s == lr_stages - 1) {
#pragma unroll
          for (int mt = 0; mt < MT; ++mt) {
            const int r = (mi0 + mt) * 16 + gq;
            a_lo[mt] = fp16_bits_to_f32(sa[r]);
            a_hi[mt] = fp16_bits_to_f32(sa[r + 8]);
          }
        }
        if (kSC4 && s == 0) {
          // The residual's row scales (SC4), before any rank-r term is added.
#pragma unroll
          for (int mt = 0; mt < MT; ++mt) {
            const int r = (mi0 + mt) * 16 + gq;
            const float r_lo = fp16_bits_to_f32(sa[kTileRows + r]), r_hi = fp16_bits_to_f32(sa[kTileRows + r + 8]);
#pragma unroll
            for (int b = 0; b < NT; ++b) {
              acc[mt][b][0] *= r_lo;
              acc[mt][b][1] *= r_lo;
              acc[mt][b][2] *= r_hi;
              acc[mt][b][3] *= r_hi;
            }
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[st]);
      if (++st == stages) st = 0, ph ^= 1;
      if (!active) continue;
#pragma unroll
      for (int l = 0; l < Geom::kLrSteps; ++l) {
        if (l >= nl) break;
        const int ls = ls0 + l;
        const int kb = min(max(p.core_cols - 16 * ls, 0), 16);  // k < kb: core columns of this step
        // Core halves of this lane's k pairs (2cq, 2cq+1) and (2cq+8, 2cq+9).
        const uint32_t m0 = (2 * cq < kb ? 0x0000FFFFu : 0u) | (2 * cq + 1 < kb ? 0xFFFF0000u : 0u);
        const uint32_t m1 = (2 * cq + 8 < kb ? 0x0000FFFFu : 0u) | (2 * cq + 9 < kb ? 0xFFFF0000u : 0u);
        const bool first_corr = kb < 16 && 16 * ls <= p.core_cols;  // the correction starts in this step
        uint32_t bh[NT][2], bl[NT][2];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
          // t fragments of the 16-token chunk holding n-tile nt
          const uint32_t *tc = ts_s + (size_t)(nt >> 1) * p.nls * 256;
          const uint2 h2 = *reinterpret_cast<const uint2 *>(tc + ((((size_t)ls * 2 + 0) * 2 + (nt & 1)) * 32 + lane) * 2);
          const uint2 l2 = *reinterpret_cast<const uint2 *>(tc + ((((size_t)ls * 2 + 1) * 2 + (nt & 1)) * 32 + lane) * 2);
          bh[nt][0] = h2.x;
          bh[nt][1] = h2.y;
          bl[nt][0] = l2.x;
          bl[nt][1] = l2.y;
        }
        if constexpr (!kSC4) {
          // INT8 format: every step belongs to one branch (core_cols = the
          // core's padded columns); part sums promoted at each branch's end.
          const int nls_core = p.core_cols >> 4;
          if (kRatio && ls == nls_core) {  // first correction step: continue in units of s_a
#pragma unroll
            for (int mt = 0; mt < MT; ++mt) {
              const float il = __fdividef(1.f, a_lo[mt]), ih = __fdividef(1.f, a_hi[mt]);
#pragma unroll
              for (int nt = 0; nt < NT; ++nt) {
                acc[mt][nt][0] *= il;
                acc[mt][nt][1] *= il;
                acc[mt][nt][2] *= ih;
                acc[mt][nt][3] *= ih;
              }
            }
          }
#pragma unroll
          for (int mt = 0; mt < MT; ++mt) {
            uint32_t a[4];
            unpack_int8x8(lw[l][mt].x, lw[l][mt].y, a);
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
              float (&pt)[4] = kRatio ? acc[mt][nt] : part[kRatio ? 0 : mt][kRatio ? 0 : nt];
              mma_bf16_16816(pt, a, bh[nt][0], bh[nt][1]);
              mma_bf16_16816(pt, a, bl[nt][0], bl[nt][1]);
            }
          }
          if constexpr (!kRatio) {
            if (ls + 1 == nls_core || ls + 1 == p.nls) {
              const bool corr = ls + 1 == p.nls && p.has_corr;  // the correction ends with the last stage
#pragma unroll
              for (int mt = 0; mt < MT; ++mt) {
                promote<NT>(acc[mt], part[mt], corr ? a_lo[mt] : 1.f, corr ? a_hi[mt] : 1.f);
#pragma unroll
                for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                  for (int c = 0; c < 4; ++c) part[mt][nt][c] = 0.f;
              }
            }
          }
        } else {
#pragma unroll
          for (int mt = 0; mt < MT; ++mt) {
            uint32_t a[4];
            unpack_int8x8(lw[l][mt].x, lw[l][mt].y, a);
            if (kb > 0) {  // core columns
              uint32_t ac[4] = {a[0], a[1], a[2], a[3]};
              if (kb < 16) {
                ac[0] &= m0;
                ac[1] &= m0;
                ac[2] &= m1;
                ac[3] &= m1;
              }
#pragma unroll
              for (int nt = 0; nt < NT; ++nt) {
                mma_bf16_16816(acc[mt][nt], ac, bh[nt][0], bh[nt][1]);
                mma_bf16_16816(acc[mt][nt], ac, bl[nt][0], bl[nt][1]);
              }
            }
            if (kb < 16) {  // correction columns
              if (kb > 0) {
                a[0] &= ~m0;
                a[1] &= ~m0;
                a[2] &= ~m1;
                a[3] &= ~m1;
              }
              if (kRatio && first_corr) {  // continue in units of s_a
                const float il = __fdividef(1.f, a_lo[mt]), ih = __fdividef(1.f, a_hi[mt]);
#pragma unroll
                for (int nt = 0; nt < NT; ++nt) {
                  acc[mt][nt][0] *= il;
                  acc[mt][nt][1] *= il;
                  acc[mt][nt][2] *= ih;
                  acc[mt][nt][3] *= ih;
                }
              }
#pragma unroll
              for (int nt = 0; nt < NT; ++nt) {
                float (&pt)[4] = kRatio ? acc[mt][nt] : part[kRatio ? 0 : mt][kRatio ? 0 : nt];
                mma_bf16_16816(pt, a, bh[nt][0], bh[nt][1]);
                mma_bf16_16816(pt, a, bl[nt][0], bl[nt][1]);
              }
            }
          }
        }
      }
    }
    if constexpr (!kRatio && kSC4) {  // the correction's row scale
      if (active && p.has_corr) {
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) promote<NT>(acc[mt], part[mt], a_lo[mt], a_hi[mt]);
      }
    }
    if (kRatio && active && p.has_corr) {  // the correction's row scale
#pragma unroll
      for (int mt = 0; mt < MT; ++mt)
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
          acc[mt][nt][0] *= a_lo[mt];
          acc[mt][nt][1] *= a_lo[mt];
          acc[mt][nt][2] *= a_hi[mt];
          acc[mt][nt][3] *= a_hi[mt];
        }
    }

    // Epilogue.  acc[mt][nt][i]: row 16*(mi0+mt) + gq + 8*(i/2), token 8*nt + 2*cq + i%2.
    const int64_t row_base = ((int64_t)TL * unit + tsel) * kTileRows;
    if (p.out) {
      if (active) {
#pragma unroll
        for (int mt = 0; mt < MT; ++mt)
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
    } else if (p.argmax) {
      // Greedy partials: per (unit, warp, token) the largest logit and its
      // row (the lowest row on ties), as (value, row bits).
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int tl = 0; tl < 2; ++tl) {
          const int tok = nt * 8 + 2 * cq + tl;
          float bv = -INFINITY;
          int bi = 0x7fffffff;
#pragma unroll
          for (int mt = 0; mt < MT; ++mt)
#pragma unroll
            for (int ih = 0; ih < 2; ++ih) {
              const int64_t row = row_base + (mi0 + mt) * 16 + gq + 8 * ih;
              const float v = acc[mt][nt][ih * 2 + tl];
              if (active && row < p.V && (v > bv || (v == bv && (int)row < bi))) {
                bv = v;
                bi = (int)row;
              }
            }
#pragma unroll
          for (int off = 4; off < 32; off <<= 1) {
            const float ov = __shfl_xor_sync(0xffffffffu, bv, off);
            const int oi = __shfl_xor_sync(0xffffffffu, bi, off);
            if (ov > bv || (ov == bv && oi < bi)) {
              bv = ov;
              bi = oi;
            }
          }
          if (gq == 0 && tok < p.M)
            p.ce_part[((int64_t)unit * kDecWarps + warp) * p.M_total + p.m0 + tok] = make_float2(bv, __int_as_float(bi));
        }
    } else {
      // Cross-entropy partials: per (unit, warp, token) running max and sum of exp.
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int tl = 0; tl < 2; ++tl) {
          const int tok = nt * 8 + 2 * cq + tl;
          const int tgt = tok < p.M ? p.targets[p.m0 + tok] - p.row0 : -1;  // this pack's row numbering
          float vals[2 * MT];
          float mx = -INFINITY;
#pragma unroll
          for (int mt = 0; mt < MT; ++mt)
#pragma unroll
            for (int ih = 0; ih < 2; ++ih) {
              const int64_t row = row_base + (mi0 + mt) * 16 + gq + 8 * ih;
              const bool ok = active && row < p.V;
              const float v = ok ? acc[mt][nt][ih * 2 + tl] : -INFINITY;
              vals[mt * 2 + ih] = v;
              mx = fmaxf(mx, v);
              if (ok && row == tgt) p.ce_tlogit[p.m0 + tok] = v;
            }
          float sum = 0.f;
#pragma unroll
          for (int q = 0; q < 2 * MT; ++q) sum += (vals[q] == -INFINITY) ? 0.f : __expf(vals[q] - mx);
          LsePair lp{mx, sum};
#pragma unroll
          for (int off = 4; off < 32; off <<= 1) {
            LsePair o{__shfl_xor_sync(0xffffffffu, lp.m, off), __shfl_xor_sync(0xffffffffu, lp.s, off)};
            lp = lse_merge(lp, o);
          }
          if (gq == 0 && tok < p.M)
            p.ce_part[((int64_t)unit * kDecWarps + warp) * p.M_total + p.m0 + tok] = make_float2(lp.m, lp.s);
        }
    }
  }
}

template <int VAR, int SC, int GS, bool kSC4>
static cudaError_t launch_t(const DecodeParams &dp, int grid, cudaStream_t s, const DecodePlan &pl, bool pdl) {
  auto kern = decode_kernel<VAR, SC, GS, kSC4>;
  cudaError_t e = opt_in_smem(reinterpret_cast<const void *>(kern), (int)pl.total);
  if (e != cudaSuccess || grid == 0) return e;  // grid 0: opt-in only (prepare_decode)
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(variant_threads(VAR, kSC4));
  cfg.dynamicSmemBytes = pl.total;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kern, dp, pl.stages, (int)pl.xs_off, (int)pl.ts_off, (int)pl.xsum_off,
                            (int)pl.bar_off);
}

template <int VAR, bool kSC4>
static cudaError_t launch_g(const DecodeParams &dp, int grid, cudaStream_t s, const DecodePlan &pl, bool pdl) {
  constexpr int SC = stage_chunks(VAR);
  switch (dp.g) {
    case 32: return launch_t<VAR, SC, 2, kSC4>(dp, grid, s, pl, pdl);
    case 64: return launch_t<VAR, SC, 4, kSC4>(dp, grid, s, pl, pdl);
    case 128: return launch_t<VAR, SC, 8, kSC4>(dp, grid, s, pl, pdl);
    case 256: return launch_t<VAR, SC, 16, kSC4>(dp, grid, s, pl, pdl);
  }
  return cudaErrorInvalidValue;
}

// One packed format's kernel instances (INT8 in decode.cu, SC4 in decode_sc4.cu,
// so that the two sets compile in parallel).  grid == 0 only opts the
// instance into its shared memory (no launch).
template <bool kSC4>
cudaError_t launch_decode_fmt(const DecodeParams &dp, int grid, cudaStream_t s, bool pdl) {
  const DecodePlan pl = decode_plan(dp.d_pad, dp.nls, dp.g, dp.M, dp.variant);
  if (pl.stages < 2 || pl.sc != stage_chunks(dp.variant)) return cudaErrorInvalidValue;
  if (dp.d_pad % (pl.sc * kChunkK) != 0) return cudaErrorInvalidValue;  // the residual in whole stages
  if (dp.M < 1 || dp.M > variant_tokens(dp.variant)) return cudaErrorInvalidValue;
  if (dp.variant == kDecResident1) return launch_g<kDecResident1, kSC4>(dp, grid, s, pl, pdl);
  if (dp.variant == kDecResidentH) return launch_g<kDecResidentH, kSC4>(dp, grid, s, pl, pdl);
  if (dp.variant != kDecStreamed2 && dp.variant != kDecStreamedH && dp.variant != kDecWide4 && dp.variant != kDecWide8)
    return cudaErrorInvalidValue;
  DecodeParams dx = dp;
  if (grid > 0 && !make_tma_map_bf16(&dx.tmap_x, dp.x, dp.M_total, dp.d, variant_tokens(dp.variant)))
    return cudaErrorInvalidValue;
  if (dp.variant == kDecStreamed2) return launch_g<kDecStreamed2, kSC4>(dx, grid, s, pl, pdl);
  if (dp.variant == kDecStreamedH) return launch_g<kDecStreamedH, kSC4>(dx, grid, s, pl, pdl);
  if (dp.variant == kDecWide4) return launch_g<kDecWide4, kSC4>(dx, grid, s, pl, pdl);
  return launch_g<kDecWide8, kSC4>(dx, grid, s, pl, pdl);
}


}  // namespace archead
