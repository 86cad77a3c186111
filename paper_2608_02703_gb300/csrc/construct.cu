// Quantisation and packing steps of the offline construction of a packed
// head (paper, Section 3.4, Algorithm 1; Appendix B steps 3-7): symmetric
// group-wise quantisers for the core factors (Q_8, Q_5), the group-wise INT4
// residual (one fp16 scale per group, or the paper's 4-bit scale codes times
// a row scale), the row-wise and group-wise INT8 correction factors, the
// packing of the codes into the canonical byte layouts, and the
// dequantisation of what was stored (the realized core W_d whose error the
// correction fits).  The dense linear algebra of the construction (the
// covariance product, the eigendecomposition, the randomized SVDs) is left to
// library routines; these kernels take the integer decisions.
//
// Quantiser (every variant): scale = fp16(max|x| / qmax) over the scale's
// group (fp32 division, round to nearest even), code = clamp(rint(x / scale),
// -qmax, qmax) with the division and the rounding (ties to even) in fp32, and
// code 0 where the scale is 0.
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "internal.h"

namespace archead {

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// One warp per scale group of gr x gc elements of x [rows][cols].
__global__ void quantize_symmetric_kernel(const float *__restrict__ x, int64_t rows, int64_t cols, int64_t gr,
                                          int64_t gc, int qmax, int8_t *__restrict__ codes,
                                          uint16_t *__restrict__ scales) {
  const int lane = threadIdx.x & 31;
  const int64_t ngc = cols / gc;
  const int64_t ngroups = (rows / gr) * ngc;
  const int64_t gsize = gr * gc;
  for (int64_t grp = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5; grp < ngroups;
       grp += ((int64_t)gridDim.x * blockDim.x) >> 5) {
    const int64_t r0 = (grp / ngc) * gr, c0 = (grp % ngc) * gc;
    float mx = 0.f;
    for (int64_t i = lane; i < gsize; i += 32) mx = fmaxf(mx, fabsf(x[(r0 + i / gc) * cols + c0 + i % gc]));
    mx = warp_max(mx);
    const __half s16 = __float2half_rn(__fdiv_rn(mx, (float)qmax));
    const float s = __half2float(s16);
    if (lane == 0) scales[grp] = __half_as_ushort(s16);
    for (int64_t i = lane; i < gsize; i += 32) {
      const int64_t idx = (r0 + i / gc) * cols + c0 + i % gc;
      float q = 0.f;
      if (s > 0.f) q = fminf(fmaxf(rintf(__fdiv_rn(x[idx], s)), (float)-qmax), (float)qmax);
      codes[idx] = (int8_t)q;
    }
  }
}

// The paper's format: one warp per row.  Group maxima, s_row = fp16(max /
// (7 * 16)), q = clamp(ceil(max_g / (7 s_row)) - 1, 0, 15), codes against
// s_row (q + 1) (exact in fp32).  gmax: per-warp scratch of G floats in
// shared memory.
__global__ void quantize_residual_sc4_kernel(const float *__restrict__ r, int64_t rows, int64_t cols, int g,
                                             int8_t *__restrict__ codes, uint8_t *__restrict__ qcodes,
                                             uint16_t *__restrict__ row_scale) {
  extern __shared__ float sc4_smem[];
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  const int G = (int)(cols / g);
  float *gmax = sc4_smem + (size_t)wib * G;
  for (int64_t row = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5; row < rows;
       row += ((int64_t)gridDim.x * blockDim.x) >> 5) {
    const float *rr = r + row * cols;
    float rmax = 0.f;
    for (int grp = 0; grp < G; ++grp) {
      float mx = 0.f;
      for (int i = lane; i < g; i += 32) mx = fmaxf(mx, fabsf(rr[(int64_t)grp * g + i]));
      mx = warp_max(mx);
      if (lane == 0) gmax[grp] = mx;
      rmax = fmaxf(rmax, mx);
    }
    __syncwarp();
    const __half sr16 = __float2half_rn(__fdiv_rn(rmax, 112.f));
    const float sr = __half2float(sr16);
    if (lane == 0) row_scale[row] = __half_as_ushort(sr16);
    for (int grp = 0; grp < G; ++grp) {
      int q = 0;
      if (sr > 0.f) q = min(max((int)ceilf(__fdiv_rn(gmax[grp], 7.f * sr)) - 1, 0), 15);
      if (lane == 0) qcodes[row * G + grp] = (uint8_t)q;
      const float s = sr * (float)(q + 1);
      for (int i = lane; i < g; i += 32) {
        const int64_t idx = row * cols + (int64_t)grp * g + i;
        float c = 0.f;
        if (s > 0.f) c = fminf(fmaxf(rintf(__fdiv_rn(r[idx], s)), -7.f), 7.f);
        codes[idx] = (int8_t)c;
      }
    }
    __syncwarp();
  }
}

// bits 4: two's complement (or unsigned 0..15) nibbles, byte j of a row =
// columns 2j (low) and 2j+1 (high), a missing last column packed as 0.
// bits 5: code j of a row in bits 5j..5j+4 of the row's little-endian bit
// string, ceil(5 cols / 8) bytes per row, unused top bits 0.
__global__ void pack_codes_kernel(const int8_t *__restrict__ codes, int64_t rows, int64_t cols, int bits,
                                  uint8_t *__restrict__ packed, int64_t row_bytes) {
  const int64_t total = rows * row_bytes;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t row = e / row_bytes, b = e % row_bytes;
    const int8_t *cr = codes + row * cols;
    uint32_t v = 0;
    if (bits == 4) {
      const uint32_t lo = (uint32_t)cr[2 * b] & 15u;
      const uint32_t hi = 2 * b + 1 < cols ? (uint32_t)cr[2 * b + 1] & 15u : 0u;
      v = lo | (hi << 4);
    } else {
      for (int k = 0; k < 8; ++k) {
        const int64_t bit = 8 * b + k, j = bit / 5;
        if (j < cols && ((((uint32_t)cr[j] & 31u) >> (bit % 5)) & 1u)) v |= 1u << k;
      }
    }
    packed[e] = (uint8_t)v;
  }
}

// out = code * scale for scales over gr x gc groups (fp32; exact).
__global__ void dequant_symmetric_kernel(const int8_t *__restrict__ codes, const uint16_t *__restrict__ scales,
                                         int64_t rows, int64_t cols, int64_t gr, int64_t gc, float *__restrict__ out) {
  const int64_t total = rows * cols, ngc = cols / gc;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = e / cols, c = e % cols;
    out[e] = (float)codes[e] * __half2float(__ushort_as_half(scales[(r / gr) * ngc + c / gc]));
  }
}

// The paper's format: out = code * s_row * (q + 1).
__global__ void dequant_residual_sc4_kernel(const int8_t *__restrict__ codes, const uint8_t *__restrict__ qcodes,
                                            const uint16_t *__restrict__ row_scale, int64_t rows, int64_t cols, int g,
                                            float *__restrict__ out) {
  const int64_t total = rows * cols, G = cols / g;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = e / cols, c = e % cols;
    const float s = __half2float(__ushort_as_half(row_scale[r])) * (float)(qcodes[r * G + c / g] + 1);
    out[e] = (float)codes[e] * s;
  }
}

static unsigned grid_for(int64_t threads) {
  int64_t b = (threads + 255) / 256;
  return (unsigned)(b < 1 ? 1 : (b > 65535 * 8 ? 65535 * 8 : b));
}

}  // namespace archead

using namespace archead;

namespace {

archead_status fail_cuda(cudaError_t e) {
  set_last_error_message(cudaGetErrorString(e));
  return e == cudaErrorMemoryAllocation ? ARCHEAD_ERR_OOM : ARCHEAD_ERR_CUDA;
}

int qmax_of(int bits) { return bits == 8 ? 127 : bits == 5 ? 15 : bits == 4 ? 7 : 0; }

}  // namespace

extern "C" {

ARCHEAD_API archead_status archead_quantize_symmetric(const float *x, int64_t rows, int64_t cols, int64_t group_rows,
                                                      int64_t group_cols, int bits, int8_t *codes, uint16_t *scales,
                                                      void *stream) {
  if (rows < 0 || cols < 0 || group_rows < 1 || group_cols < 1) return ARCHEAD_ERR_INVALID_ARG;
  if (rows % group_rows || cols % group_cols || qmax_of(bits) == 0) return ARCHEAD_ERR_INVALID_ARG;
  if (rows == 0 || cols == 0) return ARCHEAD_OK;
  if (!x || !codes || !scales) return ARCHEAD_ERR_INVALID_ARG;
  const int64_t ngroups = (rows / group_rows) * (cols / group_cols);
  quantize_symmetric_kernel<<<grid_for(ngroups * 32), 256, 0, static_cast<cudaStream_t>(stream)>>>(
      x, rows, cols, group_rows, group_cols, qmax_of(bits), codes, scales);
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? ARCHEAD_OK : fail_cuda(e);
}

ARCHEAD_API archead_status archead_quantize_residual_sc4(const float *r, int64_t rows, int64_t cols, int group_size,
                                                         int8_t *codes, uint8_t *scale_codes, uint16_t *row_scale,
                                                         void *stream) {
  if (rows < 0 || cols < 0 || group_size < 1 || cols % group_size) return ARCHEAD_ERR_INVALID_ARG;
  if (rows == 0 || cols == 0) return ARCHEAD_OK;
  if (!r || !codes || !scale_codes || !row_scale) return ARCHEAD_ERR_INVALID_ARG;
  const int64_t G = cols / group_size;
  if (G > 1024) return ARCHEAD_ERR_UNSUPPORTED;  // per-warp group maxima in shared memory
  const size_t smem = (size_t)8 * G * sizeof(float);
  quantize_residual_sc4_kernel<<<grid_for(rows * 32), 256, smem, static_cast<cudaStream_t>(stream)>>>(
      r, rows, cols, group_size, codes, scale_codes, row_scale);
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? ARCHEAD_OK : fail_cuda(e);
}

ARCHEAD_API archead_status archead_pack_codes(const int8_t *codes, int64_t rows, int64_t cols, int bits,
                                              uint8_t *packed, void *stream) {
  if (rows < 0 || cols < 0 || (bits != 4 && bits != 5)) return ARCHEAD_ERR_INVALID_ARG;
  if (rows == 0 || cols == 0) return ARCHEAD_OK;
  if (!codes || !packed) return ARCHEAD_ERR_INVALID_ARG;
  const int64_t row_bytes = bits == 4 ? (cols + 1) / 2 : (5 * cols + 7) / 8;
  pack_codes_kernel<<<grid_for(rows * row_bytes), 256, 0, static_cast<cudaStream_t>(stream)>>>(codes, rows, cols,
                                                                                               bits, packed, row_bytes);
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? ARCHEAD_OK : fail_cuda(e);
}

ARCHEAD_API archead_status archead_dequant_symmetric(const int8_t *codes, const uint16_t *scales, int64_t rows,
                                                     int64_t cols, int64_t group_rows, int64_t group_cols, float *out,
                                                     void *stream) {
  if (rows < 0 || cols < 0 || group_rows < 1 || group_cols < 1 || rows % group_rows || cols % group_cols)
    return ARCHEAD_ERR_INVALID_ARG;
  if (rows == 0 || cols == 0) return ARCHEAD_OK;
  if (!codes || !scales || !out) return ARCHEAD_ERR_INVALID_ARG;
  dequant_symmetric_kernel<<<grid_for(rows * cols), 256, 0, static_cast<cudaStream_t>(stream)>>>(
      codes, scales, rows, cols, group_rows, group_cols, out);
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? ARCHEAD_OK : fail_cuda(e);
}

ARCHEAD_API archead_status archead_dequant_residual_sc4(const int8_t *codes, const uint8_t *scale_codes,
                                                        const uint16_t *row_scale, int64_t rows, int64_t cols,
                                                        int group_size, float *out, void *stream) {
  if (rows < 0 || cols < 0 || group_size < 1 || cols % group_size) return ARCHEAD_ERR_INVALID_ARG;
  if (rows == 0 || cols == 0) return ARCHEAD_OK;
  if (!codes || !scale_codes || !row_scale || !out) return ARCHEAD_ERR_INVALID_ARG;
  dequant_residual_sc4_kernel<<<grid_for(rows * cols), 256, 0, static_cast<cudaStream_t>(stream)>>>(
      codes, scale_codes, row_scale, rows, cols, group_size, out);
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? ARCHEAD_OK : fail_cuda(e);
}

}  // extern "C"
