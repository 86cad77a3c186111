// Host entry points of the decode kernel (decode_kernel.cuh); the INT8
// format's instances compile here, the SC4 format's in decode_sc4.cu.
#include <algorithm>

#include "decode_kernel.cuh"

namespace archead {

int decode_num_units(const archead_pack *p, int variant) {
  return (p->num_tiles + variant_tiles(variant) - 1) / variant_tiles(variant);
}

int decode_variant_tokens(int variant) { return variant_tokens(variant); }

int decode_parts_per_unit(int variant, bool sc4) { return variant_cw(variant, sc4); }

bool decode_supported(int d_pad, int nls, int g) {
  return decode_plan(d_pad, nls, g, kDecodeMaxTokens, kDecStreamed2).stages >= 2;
}

// Up to 8 tokens: x resident in shared memory (fp16) while that leaves a ring
// of at least 96 KB; otherwise, and for 9..16 tokens, the instance that
// streams x through the ring (very wide heads: 8 tokens of d = 16384 would
// take 256 KB).
// 17..32 and 33..64 tokens take the wide instances (one launch streams the
// head once for all of them) while their ring keeps at least four stages,
// else 16-token chunks of kDecStreamed2.  More than 64 tokens run in chunks
// of 64 (kDecWide8 for every chunk, the last one included).
static bool wide_fits(int d_pad, int nls, int g, int variant) {
  return decode_plan(d_pad, nls, g, variant_tokens(variant), variant).stages >= 4;
}

// Resident x in units of two tiles: for the paper's format (measured faster
// there: 63.8 against 65.7 us at M = 1 on the Qwen3-8B head), and for INT8
// heads whose four-tile units fill the last round of blocks at least 5 %
// worse than two-tile units would (Gemma-shaped head: 77.4 against 79.3 us
// with sixteen warps of one m-tile; on the Qwen3-8B head, where both fill it
// alike, two-tile units are 2.7 % slower).
static bool half_units(const archead_pack *p) {
  if (p->d_pad % (stage_chunks(kDecResidentH) * kChunkK) != 0) return false;  // whole stages of four chunks
  if (p->sc4) return true;
  const auto fill = [&](int tiles_per_unit) {
    const int units = (p->num_tiles + tiles_per_unit - 1) / tiles_per_unit;
    const int rounds = (units + p->sm_count - 1) / p->sm_count;
    return (double)units / ((double)rounds * p->sm_count);
  };
  return fill(2) > fill(4) + 0.05;
}

int decode_variant(const archead_pack *p, int M) {
  const int d_pad = p->d_pad, nls = p->nls_dec, g = p->g;
  if (M > 32 && wide_fits(d_pad, nls, g, kDecWide8)) return kDecWide8;
  if (M > 16 && wide_fits(d_pad, nls, g, kDecWide4)) return kDecWide4;
  // Streamed x, two n-tiles: in two-tile units where d is whole four-chunk
  // stages and that ring keeps at least four stages.
  const int streamed =
      d_pad % (stage_chunks(kDecStreamedH) * kChunkK) == 0 && wide_fits(d_pad, nls, g, kDecStreamedH)
          ? kDecStreamedH
          : kDecStreamed2;
  if (M > 8) return streamed;
  const int resident = half_units(p) ? kDecResidentH : kDecResident1;
  const DecodePlan pl = decode_plan(d_pad, nls, g, M, resident);
  return pl.stages >= 2 && pl.xs_off >= (size_t)96 * 1024 ? resident : streamed;
}

extern template cudaError_t launch_decode_fmt<true>(const DecodeParams &, int, cudaStream_t, bool);
template cudaError_t launch_decode_fmt<false>(const DecodeParams &, int, cudaStream_t, bool);

cudaError_t launch_decode(const DecodeParams &dp, int grid, cudaStream_t s, bool pdl) {
  return dp.sc4 ? launch_decode_fmt<true>(dp, grid, s, pdl) : launch_decode_fmt<false>(dp, grid, s, pdl);
}

// Opt in every instance the pack can launch: the largest token count of
// each variant needs the most shared memory.
cudaError_t prepare_decode(const archead_pack *p) {
  if (!decode_supported(p->d_pad, p->nls_dec, p->g)) return cudaSuccess;
  // For every instance some M <= 64 selects, the M that needs it most shared
  // memory (the instance can change with M on heads too wide for x of every
  // token count to stay resident).
  constexpr int kVariants = 6;
  static_assert(kDecStreamedH + 1 == kVariants, "one entry per decode instance");
  int best_m[kVariants] = {0, 0, 0, 0, 0, 0};
  size_t best_bytes[kVariants] = {0, 0, 0, 0, 0, 0};
  for (int M = 1; M <= kDecodeWideTokens; ++M) {
    const int v = decode_variant(p, M);
    const int m = std::min(M, variant_tokens(v));
    const size_t bytes = decode_plan(p->d_pad, p->nls_dec, p->g, m, v).total;
    if (v >= 0 && v < kVariants && bytes >= best_bytes[v]) best_bytes[v] = bytes, best_m[v] = m;
  }
  DecodeParams dp = decode_params(p, nullptr, kDecodeWideTokens);
  for (int v = 0; v < kVariants; ++v) {
    if (best_m[v] == 0) continue;
    dp.variant = v;
    dp.M = best_m[v];
    const cudaError_t e = launch_decode(dp, 0, nullptr, false);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace archead
