// Allocation-free decode forward (archead_forward_decode_noalloc).
//
// Who needs it: callers that must not allocate device memory while they run
// the head -- a serving loop that reserved all device memory up front for its
// KV cache and weights, code that runs while a CUDA graph is being captured on
// a stream whose pool forbids new allocations, or a latency-critical loop that
// cannot afford cudaMalloc / cudaFree (both take allocator locks and cudaFree
// synchronises the device).  archead_forward grows a per-pack workspace with
// cudaMalloc the first time it sees a larger M; this entry point never does.
//
// It runs the same pre-pass and decode kernels as archead_forward for
// M <= 16, but takes every scratch buffer (the pre-pass's per-split partial
// sums, its block counters and the rank-r B fragments) from one fixed array
// compiled into the library, g_noalloc_scratch, of kNoallocScratchBytes.
// Every device that loads the library holds this array until the process
// exits.  All calls on a device share it and it keeps the previous call's
// contents; the counters that must start at zero are cleared on the stream at
// the start of each call, everything else is fully rewritten before it is
// read.  Two calls whose work overlaps on the GPU (different streams, or
// different packs on the same device at the same time) race on the array.
#include <cuda_runtime.h>

#include <mutex>

#include "device.cuh"
#include "internal.h"

namespace archead {

constexpr size_t kNoallocScratchBytes = (size_t)512 << 10;  // 512 KiB
constexpr size_t kNoallocCounterBytes = 4096;              // 1024 block counters
constexpr int kNoallocMaxDevices = 64;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoallocScratchBytes];

// Device address of g_noalloc_scratch, resolved once per device with that
// device current.  In host code the symbol is only a host-side stand-in: a
// kernel handed &g_noalloc_scratch would fault (or silently touch host memory
// where the device can reach it), so kernels only ever get this address.
// The address is cached for the life of the process: calls after a
// cudaDeviceReset of that device are not supported (its module, and so the
// array, may be loaded elsewhere afterwards).
static void *g_scratch_dev[kNoallocMaxDevices];
static std::mutex g_scratch_mu;

static cudaError_t scratch_address(int device, void **out) {
  if (device < 0 || device >= kNoallocMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (!g_scratch_dev[device]) {
    void *ptr = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_dev[device] = ptr;
  }
  *out = g_scratch_dev[device];
  return cudaSuccess;
}

}  // namespace archead

using namespace archead;

extern "C" ARCHEAD_API archead_status archead_forward_decode_noalloc(archead_pack *pack, const void *x, int64_t M,
                                                                     void *logits, archead_out_dtype out_dtype,
                                                                     void *stream) {
  if (!pack || M < 0) return ARCHEAD_ERR_INVALID_ARG;
  if (M == 0) return ARCHEAD_OK;
  if (!x || !logits || (reinterpret_cast<uintptr_t>(x) & 15) || (reinterpret_cast<uintptr_t>(logits) & 15))
    return ARCHEAD_ERR_INVALID_ARG;
  if (out_dtype != ARCHEAD_OUT_BF16 && out_dtype != ARCHEAD_OUT_FP32) return ARCHEAD_ERR_INVALID_ARG;
  if (M > kDecodeMaxTokens) {
    set_last_error_message("archead_forward_decode_noalloc: M must be at most 16");
    return ARCHEAD_ERR_UNSUPPORTED;
  }
  if (!decode_supported(pack->d_pad, pack->nls_dec, pack->g)) {
    set_last_error_message("archead_forward_decode_noalloc: the decode kernel does not support this head shape");
    return ARCHEAD_ERR_UNSUPPORTED;
  }
  // Scratch: [block counters | pre-pass partial sums | rank-r fragments of one 16-token chunk].
  const int pairs = prepass_pairs((int)M, pack->lr);
  const size_t partial_bytes = (prepass_partial_bytes((int)M, pack->lr, pack->d) + 255) / 256 * 256;
  const size_t ts_bytes = (size_t)(pack->nls_dec > 0 ? pack->nls_dec : 1) * 1024;
  const size_t need = kNoallocCounterBytes + partial_bytes + ts_bytes;
  if (need > kNoallocScratchBytes || (size_t)pairs * sizeof(int) > kNoallocCounterBytes) {
    set_last_error_message(
        "archead_forward_decode_noalloc: this head needs more scratch than the fixed 512 KiB array holds");
    return ARCHEAD_ERR_UNSUPPORTED;
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e = cudaSetDevice(pack->device);
  void *base = nullptr;
  if (e == cudaSuccess) e = scratch_address(pack->device, &base);
  if (e != cudaSuccess) {
    set_last_error_message(cudaGetErrorString(e));
    return ARCHEAD_ERR_CUDA;
  }
  char *scratch = static_cast<char *>(base);
  int *counters = reinterpret_cast<int *>(scratch);
  float *partial = reinterpret_cast<float *>(scratch + kNoallocCounterBytes);
  uint32_t *ts = reinterpret_cast<uint32_t *>(scratch + kNoallocCounterBytes + partial_bytes);

  // The counters are the only state that must start at zero.
  e = cudaMemsetAsync(counters, 0, (size_t)pairs * sizeof(int), s);
  // Every decode instance this pack can use (the wide ones included) is
  // opted into its shared memory here, so that a first call at any M leaves
  // nothing for a later call at another M to set up (inside a capture, say).
  if (e == cudaSuccess) e = prepare_decode(pack);

  PrepassParams pp = prepass_params(pack, x, M);
  pp.partial = partial;
  pp.counters = counters;
  pp.ts = ts;
  pp.T = nullptr;
  if (e == cudaSuccess) e = launch_prepass(pp, s, nullptr);  // no profiling events on this path

  DecodeParams dp = decode_params(pack, x, M);
  dp.ts = ts;
  dp.M = (int)M;
  dp.m0 = 0;
  dp.variant = decode_variant(pack, (int)M);
  dp.out = logits;
  dp.out_fp32 = out_dtype == ARCHEAD_OUT_FP32;
  const int units = decode_num_units(pack, dp.variant);
  if (e == cudaSuccess) e = launch_decode(dp, units < pack->sm_count ? units : pack->sm_count, s, pack->lr > 0);
  if (e != cudaSuccess) {
    set_last_error_message(cudaGetErrorString(e));
    return ARCHEAD_ERR_CUDA;
  }
  return ARCHEAD_OK;
}
