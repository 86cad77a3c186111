// Re-tiling of the canonical packed head into the kernels' device layouts
// (see internal.h), and the debug dequantiser that reads those layouts back
// through the kernels' own unpacking functions.
#include "device.cuh"
#include "internal.h"

namespace archead {

// One thread per (row, 32-bit word) of a chunk: gather the word's 8 nibbles
// from the canonical layout (byte j of a row = columns 2j (low nibble) and
// 2j+1 (high nibble), two's complement).
__global__ void build_res_codes_kernel(const uint8_t *__restrict__ src, uint8_t *__restrict__ dst, int64_t V, int d,
                                       int d_pad) {
  const int KC = d_pad / kChunkK;
  const int64_t total = (int64_t)((V + kTileRows - 1) / kTileRows) * KC * kTileRows * 8;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
    const int q = (int)(e & 7);
    const int r = (int)((e >> 3) % kTileRows);
    const int64_t chunk = (e >> 3) / kTileRows;  // vt * KC + kc
    const int kc = (int)(chunk % KC);
    const int64_t vt = chunk / KC;
    const int64_t row = vt * kTileRows + r;
    uint32_t word = 0;
    for (int p = 0; p < 8; ++p) {
      const int k = kc * kChunkK + 8 * q + (p < 4 ? 2 * p : 2 * (p - 4) + 1);
      uint32_t nib = 0;  // padding rows and columns (k >= d) hold code 0
      if (row < V && k < d) {
        const uint8_t byte = src[row * (d / 2) + k / 2];
        nib = (k & 1) ? (byte >> 4) : (byte & 0xF);
      }
      word |= (nib ^ 0x8u) << (4 * p);  // two's complement -> offset binary
    }
    reinterpret_cast<uint32_t *>(dst)[e] = word;
  }
}

__global__ void build_res_scales_kernel(const uint16_t *__restrict__ src, uint16_t *__restrict__ dst, int64_t V,
                                        int64_t V_pad, int G, int G_pad) {
  const int64_t total = V_pad * G_pad;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = i % kTileRows;
    const int64_t grp = (i / kTileRows) % G_pad;
    const int64_t vt = i / ((int64_t)kTileRows * G_pad);
    const int64_t row = vt * kTileRows + r;
    dst[i] = (row < V && grp < G) ? src[row * G + grp] : (uint16_t)0;
  }
}

// One thread per byte of a (tile, 16-wide step) block.
__global__ void build_lr_codes_kernel(const int8_t *__restrict__ core_u, const int8_t *__restrict__ corr_a,
                                      uint8_t *__restrict__ dst, int64_t V, int rc, int rr, int rcp, int nls) {
  const int64_t total = (int64_t)((V + kTileRows - 1) / kTileRows) * nls * kLrStepBytes;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
    const int j = (int)(e & 15);
    const int r = (int)((e >> 4) % kTileRows);
    const int64_t blk = (e >> 4) / kTileRows;  // vt * nls + ls
    const int ls = (int)(blk % nls);
    const int64_t row = (blk / nls) * kTileRows + r;
    const int kk = ls * 16 + j;
    int code = 0;
    if (row < V) {
      if (kk < rcp) {
        if (kk < rc) code = core_u[row * rc + kk];
      } else if (kk - rcp < rr) {
        code = corr_a[row * rr + (kk - rcp)];
      }
    }
    dst[e] = (uint8_t)(code + 128);
  }
}

__global__ void build_row_scales_kernel(const uint16_t *__restrict__ src, uint16_t *__restrict__ dst, int64_t V,
                                        int64_t V_pad) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < V_pad; i += (int64_t)gridDim.x * blockDim.x)
    dst[i] = (src != nullptr && i < V) ? src[i] : (uint16_t)0;
}

// The pre-pass operand of the prefill path, transposed to [extended column][k]
// and widened to bf16 (the int8 codes are exact in bf16).
__global__ void build_lr_t_kernel(const int8_t *__restrict__ q_v, const int8_t *__restrict__ q_b,
                                  uint16_t *__restrict__ dst, int d, int d_pad, int rc, int rr, int rcp, int lr) {
  const int64_t total = (int64_t)lr * d_pad;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const int kk = (int)(i / d_pad), k = (int)(i % d_pad);
    int code = 0;
    if (k < d) {
      if (kk < rcp) {
        if (kk < rc) code = q_v[(int64_t)k * rc + kk];
      } else if (kk - rcp < rr) {
        code = q_b[(int64_t)k * rr + (kk - rcp)];
      }
    }
    dst[i] = __bfloat16_as_ushort(__int2bfloat16_rn(code));
  }
}

cudaError_t launch_build_layouts(archead_pack *p, const uint8_t *res_codes, const uint16_t *res_scales,
                                 const int8_t *core_u, const int8_t *corr_a, const uint16_t *corr_a_scale,
                                 cudaStream_t s) {
  build_res_codes_kernel<<<2048, 256, 0, s>>>(res_codes, p->codes, p->V, p->d, p->d_pad);
  build_res_scales_kernel<<<1024, 256, 0, s>>>(res_scales, p->scales, p->V, p->V_pad, p->G, p->G_pad);
  if (p->nls > 0)
    build_lr_codes_kernel<<<1024, 256, 0, s>>>(core_u, corr_a, p->lr_codes, p->V, p->rc, p->rr, p->rcp, p->nls);
  build_row_scales_kernel<<<256, 256, 0, s>>>(p->rr > 0 ? corr_a_scale : nullptr, p->s_a, p->V, p->V_pad);
  if (p->lr > 0)
    build_lr_t_kernel<<<256, 256, 0, s>>>(p->q_v, p->q_b, p->lr_t, p->d, p->d_pad, p->rc, p->rr, p->rcp, p->lr);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Debug dequantisation through the kernels' unpack functions.
// ---------------------------------------------------------------------------
struct DequantArgs {
  const uint8_t *codes;
  const uint16_t *scales;
  const uint8_t *lr_codes;
  const uint16_t *s_a, *s_u, *s_v, *s_b;
  const int8_t *q_v, *q_b;
  int d, d_pad, G_pad, g, rc, rr, rcp, nls;
};

__global__ void debug_dequant_kernel(DequantArgs a, int comp, int64_t row0, int64_t nrows, float *out) {
  const int cols = comp == 0 ? a.d : ((comp == 1 || comp == 2) ? a.rc : a.rr);
  const int64_t total = nrows * cols;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t row = row0 + e / cols;
    const int col = (int)(e % cols);
    float v = 0.f;
    if (comp == 0 || comp == 1 || comp == 3) {
      const int64_t vt = row / kTileRows;
      const int r = (int)(row % kTileRows);
      if (comp == 0) {
        // The word holding the column, unpacked as the prefill converter does.
        const int kc = col / kChunkK, kl = col % kChunkK;
        const int KC = a.d_pad / kChunkK;
        const uint32_t w =
            reinterpret_cast<const uint32_t *>(a.codes)[(((int64_t)vt * KC + kc) * kTileRows + r) * 8 + kl / 8];
        uint32_t q[4];
        unpack_int4x8(w, q);  // exact codes, pair i = columns (8q + 2i, 8q + 2i + 1)
        const int grp = col / a.g;
        const uint32_t pr = q[(kl & 7) >> 1];
        v = ((kl & 1) ? bf16_hi(pr) : bf16_lo(pr)) *
            fp16_bits_to_f32(a.scales[((int64_t)vt * a.G_pad + grp) * kTileRows + r]);
      } else {
        const int kk = comp == 1 ? col : a.rcp + col;
        const int ls = kk >> 4, j = kk & 15;
        const uint4 w4 = *reinterpret_cast<const uint4 *>(a.lr_codes + (((int64_t)vt * a.nls + ls) * kTileRows + r) * 16);
        uint32_t q[8];
        unpack_int8x16(w4, q);
        const uint32_t pr = q[j >> 1];
        const float sc = comp == 1 ? fp16_bits_to_f32(a.s_u[col]) : fp16_bits_to_f32(a.s_a[row]);
        v = ((j & 1) ? bf16_hi(pr) : bf16_lo(pr)) * sc;
      }
    } else if (comp == 2) {
      v = (float)a.q_v[row * a.rc + col] * fp16_bits_to_f32(a.s_v[col]);
    } else {
      v = (float)a.q_b[row * a.rr + col] * fp16_bits_to_f32(a.s_b[(row / a.g) * a.rr + col]);
    }
    out[e] = v;
  }
}

cudaError_t launch_debug_dequant(const archead_pack *p, int comp, int64_t row0, int64_t nrows, float *out,
                                 cudaStream_t s) {
  DequantArgs a{p->codes, p->scales, p->lr_codes, p->s_a, p->s_u, p->s_v, p->s_b, p->q_v, p->q_b,
                p->d,     p->d_pad,  p->G_pad,    p->g,   p->rc,  p->rr,  p->rcp, p->nls};
  const int cols = comp == 0 ? p->d : ((comp == 1 || comp == 2) ? p->rc : p->rr);
  const int64_t total = nrows * cols;
  if (total == 0) return cudaSuccess;
  int64_t blocks = (total + 255) / 256;
  if (blocks > 65535) blocks = 65535;
  debug_dequant_kernel<<<(unsigned)blocks, 256, 0, s>>>(a, comp, row0, nrows, out);
  return cudaGetLastError();
}

// A single block waits on an mbarrier that nothing completes; the bounded
// wait gives up after `budget` cycles and latches the timeout bit.
__global__ void wait_timeout_probe_kernel(int *err, int64_t budget) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) mbar_wait(&bar, 0, budget, &abort_flag, err);
}

cudaError_t launch_wait_timeout_probe(int *err, int64_t budget, cudaStream_t s) {
  wait_timeout_probe_kernel<<<1, 32, 0, s>>>(err, budget);
  return cudaGetLastError();
}

}  // namespace archead
