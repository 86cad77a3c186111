// Host side of the C ABI declared in include/archead.h: argument checks, pack
// construction, workspace management, kernel sequencing and error reporting.
#include <cuda_runtime.h>

#include <algorithm>
#include <cstddef>
#include <cstring>
#include <map>
#include <mutex>
#include <string>
#include <utility>

#include "device.cuh"
#include "internal.h"

using namespace archead;

namespace {

thread_local std::string g_last_error;

archead_status cuda_status(cudaError_t e) {
  g_last_error = cudaGetErrorString(e);
  return e == cudaErrorMemoryAllocation ? ARCHEAD_ERR_OOM : ARCHEAD_ERR_CUDA;
}

#define AH_CUDA(call)                                  \
  do {                                                 \
    cudaError_t e_ = (call);                           \
    if (e_ != cudaSuccess) return cuda_status(e_);     \
  } while (0)

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

int64_t round_up(int64_t v, int64_t m) { return (v + m - 1) / m * m; }

template <typename T>
cudaError_t dev_alloc(archead_pack *p, T **ptr, size_t bytes) {
  *ptr = nullptr;
  if (bytes == 0) return cudaSuccess;
  cudaError_t e = cudaMalloc(reinterpret_cast<void **>(ptr), bytes);
  if (e == cudaSuccess) p->owned_bytes += (int64_t)bytes;
  return e;
}

void free_pack(archead_pack *p) {
  if (!p) return;
  if (p->lr_codes_dec == p->lr_codes) p->lr_codes_dec = nullptr;  // the same buffer
  void *bufs[] = {p->codes, p->scales, p->scodes, p->s_row,  p->lr_codes, p->lr_codes_dec, p->s_a,    p->q_v,
                  p->q_b,   p->lr_t,   p->s_u,    p->s_v,    p->s_b,      p->err,    p->ws,
                  p->xh_dev, p->yh_dev, p->counters};
  for (void *b : bufs)
    if (b) cudaFree(b);
  for (auto &t : p->timers)
    for (auto &pr : t.pending) {
      cudaEventDestroy(pr.first);
      cudaEventDestroy(pr.second);
    }
  delete p;
}

// Workspace carve-out: consecutive 256-byte aligned regions.
struct Carve {
  size_t off = 0;
  size_t take(size_t bytes) {
    size_t o = off;
    off += (bytes + 255) / 256 * 256;
    return o;
  }
};

// Growing a buffer synchronises the device, not only the caller's stream:
// a call made earlier on another stream may still be using the old one.
cudaError_t ensure_workspace(archead_pack *p, size_t bytes, cudaStream_t s) {
  (void)s;
  if (bytes <= p->ws_bytes) return cudaSuccess;
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return e;
  if (p->ws) {
    cudaFree(p->ws);
    p->owned_bytes -= (int64_t)p->ws_bytes;
    p->ws = nullptr;
    p->ws_bytes = 0;
  }
  size_t want = std::max(bytes, (size_t)1 << 20);
  e = cudaMalloc(&p->ws, want);
  if (e != cudaSuccess) return e;
  p->ws_bytes = want;
  p->owned_bytes += (int64_t)want;
  return cudaSuccess;
}

// Block counters of the pre-pass: zeroed once when (re)allocated; every
// pre-pass call leaves them zero again.
cudaError_t ensure_counters(archead_pack *p, int n, cudaStream_t s) {
  (void)s;
  if (n <= p->counters_len) return cudaSuccess;
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return e;
  if (p->counters) {
    cudaFree(p->counters);
    p->owned_bytes -= (int64_t)p->counters_len * 4;
    p->counters = nullptr;
    p->counters_len = 0;
  }
  const int len = std::max(n, 1024);
  e = cudaMalloc(&p->counters, (size_t)len * 4);
  if (e != cudaSuccess) return e;
  e = cudaMemset(p->counters, 0, (size_t)len * 4);
  if (e != cudaSuccess) return e;
  p->counters_len = len;
  p->owned_bytes += (int64_t)len * 4;
  return cudaSuccess;
}

struct ForwardPlan {
  size_t partial_off = 0, ts_off = 0, ce_part_off = 0, tlogit_off = 0, total = 0;
  int variant = 0, chunk_tokens = 0, nchunks = 0;
};

// Lay out the workspace of one forward over M tokens on the decode path: one
// kernel instance for every launch (so that the cross-entropy partial blocks
// have one layout), chunks of as many tokens as it takes.
ForwardPlan plan_decode(archead_pack *p, int64_t M, bool ce) {
  ForwardPlan f;
  Carve c;
  f.variant = decode_variant(p, (int)std::min<int64_t>(M, kDecodeWideTokens));
  f.chunk_tokens = decode_variant_tokens(f.variant);
  f.nchunks = (int)((M + f.chunk_tokens - 1) / f.chunk_tokens);
  f.partial_off = c.take(prepass_partial_bytes((int)M, p->lr, p->d));
  // rank-r fragments, in 16-token chunks
  f.ts_off = c.take((size_t)((M + kDecodeMaxTokens - 1) / kDecodeMaxTokens) * std::max(p->nls_dec, 1) * 1024);
  if (ce) {
    f.ce_part_off = c.take((size_t)decode_num_units(p, f.variant) * decode_parts_per_unit(f.variant, p->sc4) * M * sizeof(float2));
    f.tlogit_off = c.take((size_t)M * sizeof(float));
  }
  f.total = c.off;
  return f;
}

template <typename T>
T *at(void *base, size_t off) {
  return reinterpret_cast<T *>(static_cast<char *>(base) + off);
}

archead_status check_forward_args(archead_pack *p, const void *x, int64_t M, const void *out) {
  if (!p || M < 0) return ARCHEAD_ERR_INVALID_ARG;
  if (M == 0) return ARCHEAD_OK;
  if (!x || !out || !aligned16(x) || !aligned16(out)) return ARCHEAD_ERR_INVALID_ARG;
  if (M > (int64_t)1 << 30) return ARCHEAD_ERR_UNSUPPORTED;
  return ARCHEAD_OK;
}

// Decode path over M tokens, 16 at a time.  out == nullptr selects CE mode,
// or greedy mode when amax_idx is given.
archead_status run_decode(archead_pack *p, const void *x, int64_t M, void *out, int out_fp32,
                          const int32_t *targets, float *ce, int32_t *amax_idx, float *amax_val, int row0,
                          float *parts3, cudaStream_t s) {
  if (!decode_supported(p->d_pad, p->nls_dec, p->g)) return ARCHEAD_ERR_UNSUPPORTED;
  const bool ce_mode = out == nullptr;
  const bool greedy = amax_idx != nullptr;
  ForwardPlan f = plan_decode(p, M, ce_mode);
  AH_CUDA(ensure_workspace(p, f.total, s));
  AH_CUDA(ensure_counters(p, prepass_pairs((int)M, p->lr), s));
  PrepassParams pp = prepass_params(p, x, M);
  pp.partial = at<float>(p->ws, f.partial_off);
  pp.counters = p->counters;
  pp.ts = at<uint32_t>(p->ws, f.ts_off);
  pp.T = nullptr;
  AH_CUDA(launch_prepass(pp, s, p));

  DecodeParams dp = decode_params(p, x, M);
  dp.out = out;
  dp.out_fp32 = out_fp32;
  dp.targets = targets;
  dp.row0 = row0;
  dp.argmax = greedy;
  dp.ce_part = ce_mode ? at<float2>(p->ws, f.ce_part_off) : nullptr;
  dp.ce_tlogit = ce_mode ? at<float>(p->ws, f.tlogit_off) : nullptr;
  const int units = decode_num_units(p, f.variant);
  const int grid = std::min(units, p->sm_count);
  dp.variant = f.variant;
  for (int c = 0; c < f.nchunks; ++c) {
    dp.m0 = c * f.chunk_tokens;
    dp.M = (int)std::min<int64_t>(f.chunk_tokens, M - dp.m0);
    dp.ts = pp.ts + (size_t)(dp.m0 / kDecodeMaxTokens) * p->nls_dec * 256;
    cudaEvent_t ev = nullptr;
    timer_begin(p, "decode", s, &ev);
    // The first chunk overlaps the pre-pass grid (programmatic dependent launch).
    const bool pdl = c == 0 && p->lr > 0 && !p->profiling;
    cudaError_t e = launch_decode(dp, grid, s, pdl);
    timer_end(p, "decode", s, ev);
    if (e != cudaSuccess) return cuda_status(e);
  }
  if (ce_mode) {
    cudaEvent_t ev = nullptr;
    timer_begin(p, "ce_finalize", s, &ev);
    const int parts = units * decode_parts_per_unit(f.variant, p->sc4);
    cudaError_t e =
        greedy   ? launch_argmax_finalize(dp.ce_part, parts, (int)M, amax_idx, amax_val, s)
        : parts3 ? launch_lse_partial_finalize(dp.ce_part, parts, dp.ce_tlogit, targets, row0, p->V, (int)M, parts3, s)
                 : launch_ce_finalize(dp.ce_part, parts, dp.ce_tlogit, targets, p->V, (int)M, ce, p->err, s);
    timer_end(p, "ce_finalize", s, ev);
    if (e != cudaSuccess) return cuda_status(e);
  }
  return ARCHEAD_OK;
}

// Prefill path: rank-r pre-pass into the extended operand T, then the
// tensor-core kernel.  out == nullptr selects CE mode, or greedy mode when
// amax_idx is given.
archead_status run_prefill(archead_pack *p, const void *x, int64_t M, void *out, int out_fp32,
                           const int32_t *targets, float *ce, int32_t *amax_idx, float *amax_val, int row0,
                           float *parts3, cudaStream_t s) {
  const bool ce_mode = out == nullptr;
  const bool greedy = amax_idx != nullptr;
  Carve c;
  const size_t t_off = c.take((size_t)M * std::max(2 * p->lr, 64) * 2);
  size_t ce_part_off = 0, tlogit_off = 0;
  if (ce_mode) {
    ce_part_off = c.take((size_t)p->num_tiles * prefill_parts_per_vt() * M * sizeof(float2));
    tlogit_off = c.take((size_t)M * sizeof(float));
  }
  AH_CUDA(ensure_workspace(p, c.off, s));
  PrepassParams pp = prepass_params(p, x, M);
  pp.ts = nullptr;
  pp.T = at<uint16_t>(p->ws, t_off);
  AH_CUDA(launch_prepass_t(pp, p->lr_t, p->d_pad, s, p));
  float2 *ce_part = ce_mode ? at<float2>(p->ws, ce_part_off) : nullptr;
  float *tlogit = ce_mode ? at<float>(p->ws, tlogit_off) : nullptr;
  cudaEvent_t ev = nullptr;
  timer_begin(p, "prefill", s, &ev);
  cudaError_t e = launch_prefill(p, x, (int)M, pp.T, out, out_fp32, greedy, targets, row0, ce_part, tlogit, s);
  timer_end(p, "prefill", s, ev);
  if (e != cudaSuccess) return cuda_status(e);
  if (ce_mode) {
    timer_begin(p, "ce_finalize", s, &ev);
    const int parts = p->num_tiles * prefill_parts_per_vt();
    e = greedy   ? launch_argmax_finalize(ce_part, parts, (int)M, amax_idx, amax_val, s)
        : parts3 ? launch_lse_partial_finalize(ce_part, parts, tlogit, targets, row0, p->V, (int)M, parts3, s)
                 : launch_ce_finalize(ce_part, parts, tlogit, targets, p->V, (int)M, ce, p->err, s);
    timer_end(p, "ce_finalize", s, ev);
    if (e != cudaSuccess) return cuda_status(e);
  }
  return ARCHEAD_OK;
}

archead_status run_forward(archead_pack *p, const void *x, int64_t M, void *out, int out_fp32,
                           const int32_t *targets, float *ce, archead_path path, cudaStream_t s,
                           int32_t *amax_idx = nullptr, float *amax_val = nullptr, int row0 = 0,
                           float *parts3 = nullptr) {
  if (path != ARCHEAD_PATH_AUTO && path != ARCHEAD_PATH_DECODE && path != ARCHEAD_PATH_PREFILL)
    return ARCHEAD_ERR_INVALID_ARG;
  AH_CUDA(cudaSetDevice(p->device));
  // AUTO: one decode launch streams the head once for up to 64 tokens (16,
  // 32 or 64 per instance); a prefill launch computes full 256-token tiles
  // and costs about as much as one 64-token decode launch plus a fifth
  // (Qwen3-8B shape: ~350 us against ~150 us at 32 tokens and ~280 us at 64),
  // so AUTO decodes up to 64 tokens when that takes at most three launches
  // (heads too wide for the wide instances' ring run 16-token chunks).
  // Heads too wide for the decode kernel's shared memory plan (per-group
  // sums of x for 16 tokens, e.g. d = 2^20 at g = 32) take the prefill
  // kernel under AUTO.
  bool decode = path == ARCHEAD_PATH_DECODE;
  if (path == ARCHEAD_PATH_AUTO && M <= kDecodeWideTokens && decode_supported(p->d_pad, p->nls_dec, p->g)) {
    const int tok = decode_variant_tokens(decode_variant(p, (int)M));
    decode = (M + tok - 1) / tok <= 3;
  }
  if (decode) return run_decode(p, x, M, out, out_fp32, targets, ce, amax_idx, amax_val, row0, parts3, s);
  return run_prefill(p, x, M, out, out_fp32, targets, ce, amax_idx, amax_val, row0, parts3, s);
}

}  // namespace

namespace archead {

void set_last_error_message(const char *msg) { g_last_error = msg ? msg : ""; }

PrepassParams prepass_params(const archead_pack *p, const void *x, int64_t M) {
  PrepassParams pp{};
  pp.x = static_cast<const uint16_t *>(x);
  pp.q_v = p->q_v;
  pp.q_b = p->q_b;
  pp.s_b = p->s_b;
  pp.s_u = p->s_u;
  pp.s_v = p->s_v;
  pp.M = (int)M;
  pp.d = p->d;
  pp.g = p->g;
  pp.rc = p->rc;
  pp.rr = p->rr;
  pp.rcp = p->rcp;
  pp.rrp = p->rrp;
  pp.lr = p->lr;
  pp.ts_nls = p->nls_dec;
  pp.ts_core = p->core_cols;
  pp.ts_compact = p->nls_dec < p->nls;
  return pp;
}

DecodeParams decode_params(const archead_pack *p, const void *x, int64_t M_total) {
  DecodeParams dp{};
  dp.codes = p->codes;
  dp.scales = p->scales;
  dp.scodes = p->scodes;
  dp.s_row = p->s_row;
  dp.sc4 = p->sc4;
  dp.G_pad2 = p->G_pad2;
  dp.lr_codes = p->lr_codes_dec;
  dp.s_a = p->s_a;
  dp.x = static_cast<const uint16_t *>(x);
  dp.V = p->V;
  dp.num_tiles = p->num_tiles;
  dp.d = p->d;
  dp.d_pad = p->d_pad;
  dp.G_pad = p->G_pad;
  dp.g = p->g;
  dp.nls = p->nls_dec;
  dp.core_cols = p->core_cols;
  dp.has_corr = p->rr > 0;
  dp.M_total = (int)M_total;
  dp.err = p->err;
  dp.wait_budget = p->wait_budget;
  return dp;
}

cudaError_t opt_in_smem(const void *func, int bytes) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  static std::mutex mu;
  static std::map<std::pair<const void *, int>, int> opted;  // (kernel, device) -> bytes
  std::lock_guard<std::mutex> lock(mu);
  int &have = opted[{func, dev}];
  if (have >= bytes) return cudaSuccess;
  e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess) have = bytes;
  return e;
}

void timer_begin(archead_pack *p, const char *name, cudaStream_t s, cudaEvent_t *ev0) {
  *ev0 = nullptr;
  if (!p || !p->profiling) return;
  if (cudaEventCreate(ev0) != cudaSuccess) {
    *ev0 = nullptr;
    return;
  }
  cudaEventRecord(*ev0, s);
}

void timer_end(archead_pack *p, const char *name, cudaStream_t s, cudaEvent_t ev0) {
  if (!p || !p->profiling || !ev0) return;
  cudaEvent_t ev1;
  if (cudaEventCreate(&ev1) != cudaSuccess) {
    cudaEventDestroy(ev0);
    return;
  }
  cudaEventRecord(ev1, s);
  for (auto &t : p->timers)
    if (std::strcmp(t.name, name) == 0) {
      t.pending.emplace_back(ev0, ev1);
      return;
    }
  KernelTimer kt;
  kt.name = name;
  kt.pending.emplace_back(ev0, ev1);
  p->timers.push_back(kt);
}

}  // namespace archead

extern "C" {

int archead_abi_version(void) { return ARCHEAD_ABI_VERSION; }

archead_status archead_pack_create_ex(const archead_desc *desc, size_t desc_size, void *stream, archead_pack **out) {
  if (!out) return ARCHEAD_ERR_INVALID_ARG;
  *out = nullptr;
  if (!desc || desc_size < offsetof(archead_desc, res_row_scale)) return ARCHEAD_ERR_INVALID_ARG;
  // Fields past the caller's struct read as zero (absent).
  archead_desc d{};
  std::memcpy(&d, desc, std::min(desc_size, sizeof(archead_desc)));
  return archead_pack_create(&d, stream, out);
}

archead_status archead_pack_create(const archead_desc *desc, void *stream, archead_pack **out) {
  if (!out) return ARCHEAD_ERR_INVALID_ARG;
  *out = nullptr;
  if (!desc) return ARCHEAD_ERR_INVALID_ARG;
  const int64_t V = desc->vocab, d = desc->hidden;
  const int rc = desc->core_rank, rr = desc->corr_rank, g = desc->group_size;
  const int fmt = desc->format;
  if (fmt != ARCHEAD_FORMAT_INT8 && fmt != ARCHEAD_FORMAT_SC4) return ARCHEAD_ERR_INVALID_ARG;
  const bool sc4 = fmt == ARCHEAD_FORMAT_SC4;
  if (V < 1 || d < 64 || d % 64 != 0) return ARCHEAD_ERR_INVALID_ARG;
  if (!(g == 32 || g == 64 || g == 128 || g == 256) || d % g != 0) return ARCHEAD_ERR_INVALID_ARG;
  if (rc < 0 || rr < 0 || rc > 256 || rr > 256) return ARCHEAD_ERR_INVALID_ARG;
  if (d > (1 << 20) || V > ((int64_t)1 << 31) - 256) return ARCHEAD_ERR_UNSUPPORTED;
  if (!desc->res_codes || !desc->res_scales) return ARCHEAD_ERR_INVALID_ARG;
  if (sc4 && !desc->res_row_scale) return ARCHEAD_ERR_INVALID_ARG;
  if (rc > 0 && (!desc->core_u || !desc->core_u_scale || !desc->core_v || !desc->core_v_scale))
    return ARCHEAD_ERR_INVALID_ARG;
  if (rr > 0 && (!desc->corr_a || !desc->corr_a_scale || !desc->corr_b || !desc->corr_b_scale))
    return ARCHEAD_ERR_INVALID_ARG;

  cudaStream_t s = static_cast<cudaStream_t>(stream);
  archead_pack *p = new (std::nothrow) archead_pack();
  if (!p) return ARCHEAD_ERR_OOM;
  auto fail = [&](cudaError_t e) {
    archead_status st = cuda_status(e);
    free_pack(p);
    return st;
  };
  cudaError_t e = cudaGetDevice(&p->device);
  if (e != cudaSuccess) return fail(e);
  e = cudaDeviceGetAttribute(&p->sm_count, cudaDevAttrMultiProcessorCount, p->device);
  if (e != cudaSuccess) return fail(e);
  p->V = V;
  p->d = (int)d;
  p->rc = rc;
  p->rr = rr;
  p->g = g;
  p->G = (int)(d / g);
  p->d_pad = (int)round_up(d, 128);
  p->G_pad = p->d_pad / g;
  p->sc4 = sc4 ? 1 : 0;
  p->G_pad2 = (p->G_pad + 1) / 2;
  p->num_tiles = (int)((V + kTileRows - 1) / kTileRows);
  p->V_pad = (int64_t)p->num_tiles * kTileRows;
  // Extended rank axis: each branch padded to 16 columns (one k16 step), the
  // sum to 32 (whole 64-wide k steps of the prefill's hi/lo operand).
  p->rcp = (int)round_up(rc, 16);
  p->rrp = (int)round_up(rr, 16);
  if ((p->rcp + p->rrp) % 32 != 0) {
    if (rr > 0) p->rrp += 16;
    else p->rcp += 16;
  }
  p->lr = p->rcp + p->rrp;
  p->nls = p->lr / 16;
  p->nls_core = p->rcp / 16;
  // The decode kernel's rank-r steps in the paper's format: both branches
  // back to back, padded once (its r_c = 10, r_r = 6 fit one 16-wide step
  // instead of two).  The INT8 format keeps each branch padded to 16.
  if (sc4 && (rc + rr + 15) / 16 < p->nls) {
    p->nls_dec = (rc + rr + 15) / 16;
    p->core_cols = rc;
  } else {
    p->nls_dec = p->nls;
    p->core_cols = p->rcp;
  }

  const size_t G = p->G;
  if ((e = dev_alloc(p, &p->codes, (size_t)p->V_pad * p->d_pad / 2)) != cudaSuccess) return fail(e);
  if (sc4) {
    if ((e = dev_alloc(p, &p->scodes, (size_t)p->V_pad * p->G_pad2)) != cudaSuccess) return fail(e);
    if ((e = dev_alloc(p, &p->s_row, (size_t)p->V_pad * 2)) != cudaSuccess) return fail(e);
  } else {
    if ((e = dev_alloc(p, &p->scales, (size_t)p->V_pad * p->G_pad * 2)) != cudaSuccess) return fail(e);
  }
  if ((e = dev_alloc(p, &p->lr_codes, (size_t)p->num_tiles * p->nls * kLrStepBytes)) != cudaSuccess) return fail(e);
  if (p->nls_dec < p->nls) {
    if ((e = dev_alloc(p, &p->lr_codes_dec, (size_t)p->num_tiles * p->nls_dec * kLrStepBytes)) != cudaSuccess)
      return fail(e);
  } else {
    p->lr_codes_dec = p->lr_codes;
  }
  if ((e = dev_alloc(p, &p->s_a, (size_t)p->V_pad * 2)) != cudaSuccess) return fail(e);
  if ((e = dev_alloc(p, &p->q_v, (size_t)d * rc)) != cudaSuccess) return fail(e);
  if ((e = dev_alloc(p, &p->q_b, (size_t)d * rr)) != cudaSuccess) return fail(e);
  if ((e = dev_alloc(p, &p->lr_t, (size_t)p->lr * p->d_pad * 2)) != cudaSuccess) return fail(e);
  if ((e = dev_alloc(p, &p->s_u, (size_t)rc * 2)) != cudaSuccess) return fail(e);
  if ((e = dev_alloc(p, &p->s_v, (size_t)rc * 2)) != cudaSuccess) return fail(e);
  if ((e = dev_alloc(p, &p->s_b, G * rr * 2)) != cudaSuccess) return fail(e);
  if ((e = dev_alloc(p, &p->err, 16)) != cudaSuccess) return fail(e);
  if ((e = cudaMemsetAsync(p->err, 0, 16, s)) != cudaSuccess) return fail(e);

  // Canonical components: the V-indexed ones pass through temporaries on the
  // device and are re-tiled; the d-indexed ones are copied as they are.
  uint8_t *t_codes = nullptr, *t_scales = nullptr, *t_u = nullptr, *t_a = nullptr, *t_sa = nullptr,
          *t_srow = nullptr;
  auto free_tmp = [&]() {
    for (void *b : {(void *)t_codes, (void *)t_scales, (void *)t_u, (void *)t_a, (void *)t_sa, (void *)t_srow})
      if (b) cudaFree(b);
  };
  auto tmp_copy = [&](uint8_t **dst, const void *src, size_t bytes) -> cudaError_t {
    if (bytes == 0) return cudaSuccess;
    cudaError_t e2 = cudaMalloc(reinterpret_cast<void **>(dst), bytes);
    if (e2 != cudaSuccess) return e2;
    return cudaMemcpyAsync(*dst, src, bytes, cudaMemcpyDefault, s);
  };
  e = tmp_copy(&t_codes, desc->res_codes, (size_t)V * d / 2);
  // SC4: 4-bit scale codes (ceil(G/2) bytes a row), fp16 row scales, 5-bit core codes (ceil(5 r_c/8) bytes a row).
  if (e == cudaSuccess) e = tmp_copy(&t_scales, desc->res_scales, sc4 ? (size_t)V * ((G + 1) / 2) : (size_t)V * G * 2);
  if (e == cudaSuccess && sc4) e = tmp_copy(&t_srow, desc->res_row_scale, (size_t)V * 2);
  if (e == cudaSuccess && rc > 0) e = tmp_copy(&t_u, desc->core_u, sc4 ? (size_t)V * ((5 * rc + 7) / 8) : (size_t)V * rc);
  if (e == cudaSuccess && rr > 0) e = tmp_copy(&t_a, desc->corr_a, (size_t)V * rr);
  if (e == cudaSuccess && rr > 0) e = tmp_copy(&t_sa, desc->corr_a_scale, (size_t)V * 2);
  if (e == cudaSuccess && rc > 0) e = cudaMemcpyAsync(p->q_v, desc->core_v, (size_t)d * rc, cudaMemcpyDefault, s);
  if (e == cudaSuccess && rc > 0) e = cudaMemcpyAsync(p->s_u, desc->core_u_scale, (size_t)rc * 2, cudaMemcpyDefault, s);
  if (e == cudaSuccess && rc > 0) e = cudaMemcpyAsync(p->s_v, desc->core_v_scale, (size_t)rc * 2, cudaMemcpyDefault, s);
  if (e == cudaSuccess && rr > 0) e = cudaMemcpyAsync(p->q_b, desc->corr_b, (size_t)d * rr, cudaMemcpyDefault, s);
  if (e == cudaSuccess && rr > 0) e = cudaMemcpyAsync(p->s_b, desc->corr_b_scale, G * rr * 2, cudaMemcpyDefault, s);
  if (e == cudaSuccess)
    e = launch_build_layouts(p, t_codes, t_scales, reinterpret_cast<uint16_t *>(t_srow), t_u,
                             reinterpret_cast<int8_t *>(t_a), reinterpret_cast<uint16_t *>(t_sa), s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  free_tmp();
  if (e != cudaSuccess) return fail(e);
  *out = p;
  return ARCHEAD_OK;
}

void archead_destroy(archead_pack *pack) {
  if (!pack) return;
  cudaSetDevice(pack->device);
  cudaDeviceSynchronize();
  free_pack(pack);
}

archead_status archead_forward_path(archead_pack *pack, const void *x, int64_t M, void *logits,
                                    archead_out_dtype out_dtype, archead_path path, void *stream) {
  archead_status st = check_forward_args(pack, x, M, logits);
  if (st != ARCHEAD_OK || M == 0) return st;
  if (out_dtype != ARCHEAD_OUT_BF16 && out_dtype != ARCHEAD_OUT_FP32) return ARCHEAD_ERR_INVALID_ARG;
  return run_forward(pack, x, M, logits, out_dtype == ARCHEAD_OUT_FP32, nullptr, nullptr, path,
                     static_cast<cudaStream_t>(stream));
}

archead_status archead_forward(archead_pack *pack, const void *x, int64_t M, void *logits,
                               archead_out_dtype out_dtype, void *stream) {
  return archead_forward_path(pack, x, M, logits, out_dtype, ARCHEAD_PATH_AUTO, stream);
}

archead_status archead_forward_ce_path(archead_pack *pack, const void *x, int64_t M, const int32_t *targets,
                                       float *ce, archead_path path, void *stream) {
  archead_status st = check_forward_args(pack, x, M, ce);
  if (st != ARCHEAD_OK || M == 0) return st;
  if (!targets || !aligned16(targets)) return ARCHEAD_ERR_INVALID_ARG;
  return run_forward(pack, x, M, nullptr, 0, targets, ce, path, static_cast<cudaStream_t>(stream));
}

archead_status archead_forward_ce(archead_pack *pack, const void *x, int64_t M, const int32_t *targets, float *ce,
                                  void *stream) {
  return archead_forward_ce_path(pack, x, M, targets, ce, ARCHEAD_PATH_AUTO, stream);
}

archead_status archead_forward_argmax_path(archead_pack *pack, const void *x, int64_t M, int32_t *index,
                                           float *value, archead_path path, void *stream) {
  archead_status st = check_forward_args(pack, x, M, index);
  if (st != ARCHEAD_OK || M == 0) return st;
  if (value && !aligned16(value)) return ARCHEAD_ERR_INVALID_ARG;
  return run_forward(pack, x, M, nullptr, 0, nullptr, nullptr, path, static_cast<cudaStream_t>(stream), index, value);
}

archead_status archead_forward_argmax(archead_pack *pack, const void *x, int64_t M, int32_t *index, float *value,
                                      void *stream) {
  return archead_forward_argmax_path(pack, x, M, index, value, ARCHEAD_PATH_AUTO, stream);
}

archead_status archead_forward_lse_partial(archead_pack *pack, const void *x, int64_t M, const int32_t *targets,
                                          int64_t row0, float *parts, archead_path path, void *stream) {
  archead_status st = check_forward_args(pack, x, M, parts);
  if (st != ARCHEAD_OK || M == 0) return st;
  if (!targets || !aligned16(targets)) return ARCHEAD_ERR_INVALID_ARG;
  if (row0 < 0 || row0 + pack->V > ((int64_t)1 << 31) - 1) return ARCHEAD_ERR_INVALID_ARG;
  return run_forward(pack, x, M, nullptr, 0, targets, nullptr, path, static_cast<cudaStream_t>(stream), nullptr,
                     nullptr, (int)row0, parts);
}

archead_status archead_lse_combine(const float *parts, int num_shards, int64_t M, float *ce, void *stream) {
  if (M < 0 || num_shards < 1) return ARCHEAD_ERR_INVALID_ARG;
  if (M == 0) return ARCHEAD_OK;
  if (!parts || !ce || !aligned16(parts) || !aligned16(ce)) return ARCHEAD_ERR_INVALID_ARG;
  if (M > (int64_t)1 << 30) return ARCHEAD_ERR_UNSUPPORTED;
  AH_CUDA(launch_lse_combine(parts, num_shards, (int)M, ce, static_cast<cudaStream_t>(stream)));
  return ARCHEAD_OK;
}

archead_status archead_argmax_combine(const float *values, const int32_t *indices, const int32_t *row0,
                                      int num_shards, int64_t M, int32_t *index, float *value, void *stream) {
  if (M < 0 || num_shards < 1) return ARCHEAD_ERR_INVALID_ARG;
  if (M == 0) return ARCHEAD_OK;
  if (!values || !indices || !row0 || !index) return ARCHEAD_ERR_INVALID_ARG;
  if (!aligned16(values) || !aligned16(indices) || !aligned16(row0) || !aligned16(index) ||
      (value && !aligned16(value)))
    return ARCHEAD_ERR_INVALID_ARG;
  if (M > (int64_t)1 << 30) return ARCHEAD_ERR_UNSUPPORTED;
  AH_CUDA(launch_argmax_combine(values, indices, row0, num_shards, (int)M, index, value,
                                static_cast<cudaStream_t>(stream)));
  return ARCHEAD_OK;
}

archead_status archead_forward_host(archead_pack *pack, const void *x_host, int64_t M, void *logits_host,
                                    archead_out_dtype out_dtype, void *stream) {
  if (!pack || M < 0 || !x_host || !logits_host) return ARCHEAD_ERR_INVALID_ARG;
  if (out_dtype != ARCHEAD_OUT_BF16 && out_dtype != ARCHEAD_OUT_FP32) return ARCHEAD_ERR_INVALID_ARG;
  if (M == 0) return ARCHEAD_OK;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  AH_CUDA(cudaSetDevice(pack->device));
  const size_t xb = (size_t)M * pack->d * 2;
  const size_t yb = (size_t)M * pack->V * (out_dtype == ARCHEAD_OUT_FP32 ? 4 : 2);
  // A pinned, device-mapped output buffer (cudaHostAlloc / cudaMallocHost
  // under unified addressing) is written by the kernels directly, with no
  // staging copy; pageable memory goes through a device buffer.
  void *y_direct = nullptr;
  cudaPointerAttributes attr{};
  if (cudaPointerGetAttributes(&attr, logits_host) == cudaSuccess && attr.type == cudaMemoryTypeHost &&
      attr.devicePointer != nullptr && aligned16(attr.devicePointer))
    y_direct = attr.devicePointer;
  cudaGetLastError();  // a pointer the runtime does not know is not an error here
  const size_t need_y = y_direct ? 0 : yb;
  if (xb > pack->xh_bytes || need_y > pack->yh_bytes) {
    AH_CUDA(cudaDeviceSynchronize());  // earlier calls on any stream are done with the old buffers
    if (xb > pack->xh_bytes) {
      if (pack->xh_dev) cudaFree(pack->xh_dev), pack->owned_bytes -= (int64_t)pack->xh_bytes;
      pack->xh_dev = nullptr;
      pack->xh_bytes = 0;
      AH_CUDA(cudaMalloc(&pack->xh_dev, xb));
      pack->xh_bytes = xb;
      pack->owned_bytes += (int64_t)xb;
    }
    if (need_y > pack->yh_bytes) {
      if (pack->yh_dev) cudaFree(pack->yh_dev), pack->owned_bytes -= (int64_t)pack->yh_bytes;
      pack->yh_dev = nullptr;
      pack->yh_bytes = 0;
      AH_CUDA(cudaMalloc(&pack->yh_dev, need_y));
      pack->yh_bytes = need_y;
      pack->owned_bytes += (int64_t)need_y;
    }
  }
  AH_CUDA(cudaMemcpyAsync(pack->xh_dev, x_host, xb, cudaMemcpyHostToDevice, s));
  archead_status st = archead_forward(pack, pack->xh_dev, M, y_direct ? y_direct : pack->yh_dev, out_dtype, stream);
  if (st != ARCHEAD_OK) return st;
  if (!y_direct) AH_CUDA(cudaMemcpyAsync(logits_host, pack->yh_dev, yb, cudaMemcpyDeviceToHost, s));
  AH_CUDA(cudaStreamSynchronize(s));
  return ARCHEAD_OK;
}

int64_t archead_pack_bytes(const archead_pack *p) {
  if (!p) return -1;
  const int64_t V = p->V, d = p->d, rc = p->rc, rr = p->rr, G = p->G;
  int64_t b = V * d / 2;                      // INT4 residual
  if (p->sc4) {
    b += V * ((G + 1) / 2) + V * 2;           // 4-bit group-scale codes + row scales
    b += V * ((5 * rc + 7) / 8);              // 5-bit core left codes
  } else {
    b += V * G * 2 + V * rc;                  // fp16 group scales + INT8 core left codes
  }
  b += rc * 2 + d * rc + rc * 2;              // core scales + right codes
  b += V * rr + (rr > 0 ? V * 2 : 0);         // correction left + row scales
  b += d * rr + G * rr * 2;                   // correction right + group scales
  return b;
}

int64_t archead_device_bytes(const archead_pack *p) { return p ? p->owned_bytes : -1; }

archead_status archead_debug_dequant(const archead_pack *pack, int component, int64_t row0, int64_t nrows,
                                     float *out, void *stream) {
  if (!pack || !out || row0 < 0 || nrows < 0 || component < 0 || component > 4) return ARCHEAD_ERR_INVALID_ARG;
  const int64_t limit = (component == 2 || component == 4) ? pack->d : pack->V;
  if (row0 + nrows > limit) return ARCHEAD_ERR_INVALID_ARG;
  if ((component == 1 || component == 2) && pack->rc == 0) return ARCHEAD_ERR_INVALID_ARG;
  if ((component == 3 || component == 4) && pack->rr == 0) return ARCHEAD_ERR_INVALID_ARG;
  AH_CUDA(cudaSetDevice(pack->device));
  AH_CUDA(launch_debug_dequant(pack, component, row0, nrows, out, static_cast<cudaStream_t>(stream)));
  return ARCHEAD_OK;
}

archead_status archead_sync_status(archead_pack *pack, void *stream) {
  if (!pack) return ARCHEAD_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  AH_CUDA(cudaSetDevice(pack->device));
  AH_CUDA(cudaStreamSynchronize(s));
  int word = 0;
  AH_CUDA(cudaMemcpy(&word, pack->err, sizeof(int), cudaMemcpyDeviceToHost));
  AH_CUDA(cudaMemset(pack->err, 0, sizeof(int)));
  if (word & kErrWaitTimeout) return ARCHEAD_ERR_DEVICE_TIMEOUT;
  if (word & kErrTargetRange) return ARCHEAD_ERR_TARGET_RANGE;
  if (word & kErrLayout) {
    set_last_error_message("a kernel found its shared-memory window misaligned for its TMA layout and skipped its work");
    return ARCHEAD_ERR_UNSUPPORTED;
  }
  return ARCHEAD_OK;
}

archead_status archead_set_wait_budget(archead_pack *pack, int64_t cycles) {
  if (!pack || cycles <= 0) return ARCHEAD_ERR_INVALID_ARG;
  pack->wait_budget = cycles;
  return ARCHEAD_OK;
}

archead_status archead_debug_wait_timeout(archead_pack *pack, void *stream) {
  if (!pack) return ARCHEAD_ERR_INVALID_ARG;
  AH_CUDA(cudaSetDevice(pack->device));
  AH_CUDA(launch_wait_timeout_probe(pack->err, pack->wait_budget, static_cast<cudaStream_t>(stream)));
  return ARCHEAD_OK;
}

archead_status archead_profile_enable(archead_pack *pack, int enable) {
  if (!pack) return ARCHEAD_ERR_INVALID_ARG;
  pack->profiling = enable != 0;
  return ARCHEAD_OK;
}

int archead_profile_read(archead_pack *pack, archead_kernel_stat *out, int max_entries) {
  if (!pack || (!out && max_entries > 0)) return -1;
  for (auto &t : pack->timers) {
    for (auto &pr : t.pending) {
      float ms = 0.f;
      if (cudaEventSynchronize(pr.second) == cudaSuccess && cudaEventElapsedTime(&ms, pr.first, pr.second) == cudaSuccess) {
        t.total_ms += ms;
        t.launches += 1;
      }
      cudaEventDestroy(pr.first);
      cudaEventDestroy(pr.second);
    }
    t.pending.clear();
  }
  int n = 0;
  for (auto &t : pack->timers) {
    if (n >= max_entries) break;
    out[n].name = t.name;
    out[n].launches = t.launches;
    out[n].total_ms = t.total_ms;
    ++n;
  }
  return n;
}

const char *archead_status_string(archead_status st) {
  switch (st) {
    case ARCHEAD_OK: return "ARCHEAD_OK";
    case ARCHEAD_ERR_INVALID_ARG: return "ARCHEAD_ERR_INVALID_ARG";
    case ARCHEAD_ERR_UNSUPPORTED: return "ARCHEAD_ERR_UNSUPPORTED";
    case ARCHEAD_ERR_OOM: return "ARCHEAD_ERR_OOM";
    case ARCHEAD_ERR_CUDA: return "ARCHEAD_ERR_CUDA";
    case ARCHEAD_ERR_DEVICE_TIMEOUT: return "ARCHEAD_ERR_DEVICE_TIMEOUT";
    case ARCHEAD_ERR_TARGET_RANGE: return "ARCHEAD_ERR_TARGET_RANGE";
  }
  return "ARCHEAD_ERR_UNKNOWN";
}

const char *archead_last_error(void) { return g_last_error.c_str(); }

}  // extern "C"
