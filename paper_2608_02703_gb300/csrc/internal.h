// Internal definitions shared by the host API and the kernels of libarchead.
//
// Device layouts (all built by archead_pack_create from the canonical layout):
//
//  Residual codes, "fragment-native" tiling.  The vocabulary is cut into
//  tiles of 128 rows (V padded with zero rows), d (padded with zero codes to
//  D_PAD, a multiple of 128) into chunks of 64.  Chunk
//  (vt, kc) is 4 KB: [mi 0..7][lane 0..31][word j 0..3] of 32-bit words.
//  Word j of lane (gq = lane/4, cq = lane%4) in m-tile mi holds the 8 codes an
//  m16n8k16 A-fragment needs for k16-step 4*kc + j: nibble p (pair i = p%4,
//  half h = p/4) is row 16*mi + gq + 8*(i%2), column 16*(4*kc+j) + 2*cq +
//  8*(i/2) + h.  Codes are stored offset-binary (code + 8).
//    byte offset = ((((vt*KC + kc)*8 + mi)*32 + lane)*4 + j)*4,   KC = D_PAD/64
//
//  Residual scales: [vt][G_PAD][128] fp16 bits (row within tile fastest),
//  G_PAD = D_PAD/g; scales of padding groups and rows are zero.
//
//  The paper's packed format (ARCHEAD_FORMAT_SC4) replaces them by 4-bit
//  group-scale codes and one fp16 scale per row: codes [vt][G_PAD2][128]
//  bytes, G_PAD2 = ceil(G_PAD/2), byte j of a row holding groups 2j (low
//  nibble) and 2j+1; row scales [V_pad] fp16 (zero on padding rows).  The
//  group scale is s_row * (q + 1).  Its 5-bit core left codes are widened
//  into the low-rank codes below at pack time.
//
//  Low-rank codes: the extended rank axis kk in [0, LR) with LR = RCP + RRP,
//  RCP = r_c and RRP = r_r rounded up to 16, one of them raised by 16 when
//  the sum is not a multiple of 32 (RRP if r_r > 0): kk < RCP is
//  core_u[:, kk], kk >= RCP is corr_a[:, kk - RCP] (zero beyond the rank).
//  Step ls (16 wide) of tile vt: [mi][lane][8 bytes], bytes 2i, 2i+1 = pair i
//  (same row/column rule as above with 16*ls in place of the k16 offset),
//  stored offset-binary (code + 128).
//    byte offset = (((vt*NLS + ls)*8 + mi)*32 + lane)*8,          NLS = LR/16
//
//  Correction row scales: [V_pad] fp16 bits (zero on padding rows).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>
#include <vector>

#include "archead.h"

namespace archead {

constexpr int kTileRows = 128;     // vocabulary rows per tile
constexpr int kChunkK = 64;        // d per code chunk
constexpr int kChunkBytes = 4096;  // 128 rows x 64 codes / 2
constexpr int kLrStepBytes = 2048; // 128 rows x 16 codes
constexpr int kDecodeMaxTokens = 16;   // tokens per chunk of the rank-r fragments (and of noalloc calls)
constexpr int kDecodeWideTokens = 64;  // tokens of the widest decode launch
constexpr int kPrepassKSplit = 256;  // d per pre-pass block
constexpr int64_t kDefaultWaitBudget = 2000000000LL;  // cycles, about one second

struct DecodeParams {
  CUtensorMap tmap_x;   // x [M_total][d] bf16, box 64 x (the instance's tokens) rows (instances that stream x)
  const uint8_t *codes;
  const uint16_t *scales;   // fp16 group scales (INT8 format)
  const uint8_t *scodes;    // 4-bit group-scale codes (SC4 format)
  const uint16_t *s_row;    // residual row scales (SC4 format)
  const uint8_t *lr_codes;
  const uint16_t *s_a;
  const uint16_t *x;    // hidden states [M_total][d] bf16 (this chunk starts at row m0)
  const uint32_t *ts;   // t hi/lo fragments for this token chunk
  int64_t V;
  int num_tiles, d, d_pad, G_pad, g;
  int nls;              // 16-wide rank-r steps of lr_codes (decode layout)
  int core_cols;        // rank-r columns before the correction's: k < core_cols of the steps are A_c
  int has_corr;         // r_r > 0
  int sc4, G_pad2;      // SC4 format flag; byte rows of scale codes per tile
  int M;                // tokens in this chunk (1..16)
  int m0;               // index of the chunk's first token
  int variant;          // kernel instance (decode_variant)
  void *out;            // logits [M_total][V] (NULL in CE mode)
  int out_fp32;
  // CE mode (out == NULL, argmax == 0) or greedy mode (out == NULL, argmax != 0)
  int argmax;
  const int32_t *targets;  // [M_total], global vocabulary rows
  int row0;                // global row of this pack's first row (vocabulary shards; 0 otherwise)
  float2 *ce_part;         // [num_units][M_total] (max, sum exp)
  float *ce_tlogit;        // [M_total]
  int M_total;
  int *err;
  int64_t wait_budget;
};

struct PrepassParams {
  const uint16_t *x;       // [M][d] bf16
  const int8_t *q_v;       // [d][r_c]
  const int8_t *q_b;       // [d][r_r]
  const uint16_t *s_b;     // [G][r_r]
  const uint16_t *s_u, *s_v;
  int M, d, g, rc, rr, rcp, rrp, lr;
  float *partial;          // per-split partial sums (workspace)
  int *counters;           // one per (columns, tokens) block pair, zero between calls
  uint32_t *ts;            // decode t fragments, per 16-token chunk
  int ts_nls, ts_core;     // their steps and core columns (the decode layout of the rank-r codes)
  int ts_compact;          // decode layout packs core and correction back to back
  uint16_t *T;             // prefill extended-K operand [M][2*LR] bf16 (may be NULL)
};

struct KernelTimer {
  const char *name;
  int64_t launches = 0;
  double total_ms = 0.0;
  std::vector<std::pair<cudaEvent_t, cudaEvent_t>> pending;
};

}  // namespace archead

struct archead_pack {
  int device = 0;
  int sm_count = 0;
  int64_t V = 0, V_pad = 0;
  int d = 0, rc = 0, rr = 0, g = 0, G = 0, rcp = 0, rrp = 0, lr = 0, nls = 0, nls_core = 0;
  // Decode layout of the rank-r codes: core and correction columns back to
  // back, padded once to 16 (lr_codes_dec; the same buffer as lr_codes when
  // that saves no step, with core_cols = rcp).
  int nls_dec = 0, core_cols = 0;
  uint8_t *lr_codes_dec = nullptr;
  int d_pad = 0, G_pad = 0;  // d rounded up to 128, and its group count
  int num_tiles = 0;
  int sc4 = 0;               // ARCHEAD_FORMAT_SC4
  int G_pad2 = 0;            // ceil(G_pad / 2): bytes of scale codes per row (SC4)
  // device buffers owned by the pack
  uint8_t *codes = nullptr;
  uint16_t *scales = nullptr;  // INT8 format
  uint8_t *scodes = nullptr;   // SC4 format
  uint16_t *s_row = nullptr;   // SC4 format
  uint8_t *lr_codes = nullptr;
  uint16_t *s_a = nullptr;
  int8_t *q_v = nullptr, *q_b = nullptr;
  uint16_t *lr_t = nullptr;  // [lr][d_pad] bf16: extended column kk of [q_v | q_b] (zero padded), k fastest
  uint16_t *s_u = nullptr, *s_v = nullptr, *s_b = nullptr;
  int *err = nullptr;
  int64_t owned_bytes = 0;
  // workspace (grown on demand) and the pre-pass block counters (kept zero)
  void *ws = nullptr;
  size_t ws_bytes = 0;
  int *counters = nullptr;
  int counters_len = 0;
  // host staging for archead_forward_host
  void *xh_dev = nullptr, *yh_dev = nullptr;
  size_t xh_bytes = 0, yh_bytes = 0;
  int64_t wait_budget = archead::kDefaultWaitBudget;
  bool profiling = false;
  std::vector<archead::KernelTimer> timers;
};

namespace archead {

// Kernel parameters filled from the pack (the call-specific fields -- outputs,
// token chunk, workspace pointers -- are left for the caller).
PrepassParams prepass_params(const archead_pack *p, const void *x, int64_t M);
DecodeParams decode_params(const archead_pack *p, const void *x, int64_t M_total);

// Kernel launchers (each returns the launch's cudaError_t).
// res_scales and core_u are the canonical arrays of the pack's format (SC4:
// 4-bit scale codes and 5-bit core codes; row_scale its residual row scales).
cudaError_t launch_build_layouts(archead_pack *p, const uint8_t *res_codes, const void *res_scales,
                                 const uint16_t *row_scale, const void *core_u, const int8_t *corr_a,
                                 const uint16_t *corr_a_scale, cudaStream_t s);
cudaError_t launch_debug_dequant(const archead_pack *p, int comp, int64_t row0, int64_t nrows, float *out,
                                 cudaStream_t s);
cudaError_t launch_prepass(const PrepassParams &pp, cudaStream_t s, archead_pack *p);
int prepass_pairs(int M, int lr);
// Tensor-core pre-pass for many tokens: writes the prefill operand T only.
cudaError_t launch_prepass_t(const PrepassParams &pp, const uint16_t *lr_t, int d_pad, cudaStream_t s,
                             archead_pack *pk);
size_t prepass_smem(int M);  // dynamic shared memory of one pre-pass block
size_t prepass_partial_bytes(int M, int lr, int d);
// pdl: launch as a programmatic dependent of the immediately preceding pre-pass grid.
cudaError_t launch_decode(const DecodeParams &dp, int grid, cudaStream_t s, bool pdl);
// Shared-memory opt-in (and so module loading) of every decode kernel
// instance this pack can launch, done ahead of any launch.
cudaError_t prepare_decode(const archead_pack *p);
// Tensor map of a bf16 [rows][cols] row-major matrix: box 64 columns x
// box_rows rows, 128-byte swizzle, zero fill out of bounds.  False if the
// driver entry point is missing or the encoder rejects the layout (base or
// row pitch not 16-byte aligned).
bool make_tma_map_bf16(CUtensorMap *map, const void *base, int64_t rows, int64_t cols, int box_rows);
int decode_num_units(const archead_pack *p, int variant);  // units (and ce partial blocks) of a variant
int decode_variant_tokens(int variant);                    // tokens one launch of a variant takes
int decode_parts_per_unit(int variant, bool sc4);  // cross-entropy partial blocks per unit and token
bool decode_supported(int d_pad, int nls, int g);
// Kernel instance for a launch of M tokens (M > 64: the instance every
// 64-token chunk runs): 0 (4: units of two tiles) one 8-token n-tile, x
// resident; 1 (5: units of two tiles), 2, 3 two, four and eight n-tiles, x
// streamed.
int decode_variant(const archead_pack *p, int M);
cudaError_t launch_prefill(const archead_pack *pk, const void *x, int M, const uint16_t *T, void *out, int out_fp32,
                           bool argmax, const int32_t *targets, int row0, float2 *ce_part, float *ce_tlogit,
                           cudaStream_t s);
int prefill_parts_per_vt();
// Greedy second pass: per token the largest (value, row) over the partials,
// lowest row on ties.
cudaError_t launch_argmax_finalize(const float2 *part, int num_parts, int M, int32_t *index, float *value,
                                   cudaStream_t s);
cudaError_t launch_ce_finalize(const float2 *part, int num_parts, const float *tlogit, const int32_t *targets,
                               int64_t V, int M, float *ce, int *err, cudaStream_t s);
// Vocabulary shards: per token (max, sum of exp(y - max), target logit or
// -inf when the target is not one of this shard's rows [row0, row0 + V)).
cudaError_t launch_lse_partial_finalize(const float2 *part, int num_parts, const float *tlogit,
                                        const int32_t *targets, int64_t row0, int64_t V, int M, float *parts3,
                                        cudaStream_t s);
cudaError_t launch_lse_combine(const float *parts3, int num_shards, int M, float *ce, cudaStream_t s);
cudaError_t launch_argmax_combine(const float *values, const int32_t *indices, const int32_t *row0, int num_shards,
                                  int M, int32_t *index, float *value, cudaStream_t s);
cudaError_t launch_wait_timeout_probe(int *err, int64_t budget, cudaStream_t s);

// Opt `func` into `bytes` of dynamic shared memory on the current device:
// once per kernel, device and size (the attribute is per device); thread-safe.
cudaError_t opt_in_smem(const void *func, int bytes);

// Message returned by archead_last_error() for this thread.
void set_last_error_message(const char *msg);

// Profiling hooks (no-ops unless profiling is enabled on the pack).
void timer_begin(archead_pack *p, const char *name, cudaStream_t s, cudaEvent_t *ev0);
void timer_end(archead_pack *p, const char *name, cudaStream_t s, cudaEvent_t ev0);

}  // namespace archead
