// Re-tiling of the canonical packed head into the kernels' device layouts
// (see internal.h), and the debug dequantiser that reads those layouts back
// through the kernels' own unpacking functions.
#include "device.cuh"
#include "internal.h"

namespace archead {

// One block per (vocabulary tile, 64-wide chunk of d): stage the canonical
// 128 x 32 bytes in shared memory, then emit the 1024 fragment words.  With
// fp16 group scales given (INT8 format), the codes of a group whose scale is
// zero are stored as zero: the weights are zero either way, and the decode
// kernel relies on it (it runs such a group at scale 1).
__global__ void build_res_codes_kernel(const uint8_t *__restrict__ src, const uint16_t *__restrict__ scales,
                                       uint8_t *__restrict__ dst, int64_t V, int d, int d_pad, int G, int g) {
  __shared__ uint8_t tile[kTileRows][kChunkK / 2];
  const int KC = d_pad / kChunkK;
  const int vt = blockIdx.x / KC;
  const int kc = blockIdx.x % KC;
  for (int i = threadIdx.x; i < kTileRows * (kChunkK / 2); i += blockDim.x) {
    int r = i / (kChunkK / 2), b = i % (kChunkK / 2);
    int64_t row = (int64_t)vt * kTileRows + r;
    // Padding rows and padding columns (k >= d; d is a multiple of 64) hold code 0.
    const int k = kc * kChunkK + 2 * b;
    const bool zero_scale = scales != nullptr && row < V && k < d && (scales[row * G + k / g] & 0x7FFFu) == 0;
    tile[r][b] = (row < V && k < d && !zero_scale) ? src[row * (d / 2) + (int64_t)kc * (kChunkK / 2) + b] : (uint8_t)0;
  }
  __syncthreads();
  uint32_t *out = reinterpret_cast<uint32_t *>(dst) + ((int64_t)vt * KC + kc) * 1024;
  for (int w = threadIdx.x; w < 1024; w += blockDim.x) {
    const int j = w & 3, lane = (w >> 2) & 31, mi = w >> 7;
    const int gq = lane >> 2, cq = lane & 3;
    uint32_t word = 0;
    for (int p = 0; p < 8; ++p) {
      const int i = p & 3, h = p >> 2;
      const int r = mi * 16 + gq + 8 * (i & 1);
      const int kl = j * 16 + 2 * cq + 8 * (i >> 1) + h;
      const uint8_t byte = tile[r][kl >> 1];
      const uint32_t nib = (kl & 1) ? (byte >> 4) : (byte & 0xF);
      word |= (nib ^ 0x8u) << (4 * p);  // two's complement -> offset binary
    }
    out[w] = word;
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

// SC4 group-scale codes: canonical [V][ceil(G/2)] bytes -> [vt][G_pad2][128].
// Nibbles of groups past G (padding groups) are cleared.
__global__ void build_scale_codes_kernel(const uint8_t *__restrict__ src, uint8_t *__restrict__ dst, int64_t V,
                                         int64_t V_pad, int G, int G_pad2) {
  const int nbc = (G + 1) / 2;
  const int64_t total = V_pad * G_pad2;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = i % kTileRows;
    const int j = (int)((i / kTileRows) % G_pad2);
    const int64_t row = (i / ((int64_t)kTileRows * G_pad2)) * kTileRows + r;
    uint8_t b = (row < V && j < nbc) ? src[row * nbc + j] : (uint8_t)0;
    if (2 * j + 1 >= G) b &= 0x0F;
    dst[i] = b;
  }
}

// Signed 5-bit code j of a row of ceil(5 r_c / 8) bytes (bits 5j..5j+4, LSB first).
__device__ __forceinline__ int int5_code(const uint8_t *row, int j) {
  const int bit = 5 * j, b = bit >> 3, sh = bit & 7;
  uint32_t v = (uint32_t)row[b] >> sh;
  if (sh > 3) v |= (uint32_t)row[b + 1] << (8 - sh);
  v &= 31u;
  return v >= 16 ? (int)v - 32 : (int)v;
}

// One block per (tile, 16-wide step of the extended rank axis).  core_u is
// int8 [V][r_c], or with u5 != 0 the SC4 5-bit codes [V][ceil(5 r_c / 8)].
// A correction row whose scale is zero is stored as zero codes (its weights
// are zero either way; the decode kernel runs it at scale 1).
__global__ void build_lr_codes_kernel(const void *__restrict__ core_u, const int8_t *__restrict__ corr_a,
                                      const uint16_t *__restrict__ corr_a_scale, uint8_t *__restrict__ dst, int64_t V,
                                      int rc, int rr, int rcp, int nls, int u5) {
  const int vt = blockIdx.x / nls;
  const int ls = blockIdx.x % nls;
  uint8_t *out = dst + ((int64_t)vt * nls + ls) * kLrStepBytes;
  for (int e = threadIdx.x; e < kLrStepBytes; e += blockDim.x) {
    const int b = e & 7, lane = (e >> 3) & 31, mi = e >> 8;
    const int gq = lane >> 2, cq = lane & 3;
    const int i = b >> 1, h = b & 1;
    const int64_t row = (int64_t)vt * kTileRows + mi * 16 + gq + 8 * (i & 1);
    const int kk = ls * 16 + 2 * cq + 8 * (i >> 1) + h;
    int code = 0;
    if (row < V) {
      if (kk < rcp) {
        if (kk < rc)
          code = u5 ? int5_code(static_cast<const uint8_t *>(core_u) + row * ((5 * rc + 7) / 8), kk)
                    : static_cast<const int8_t *>(core_u)[row * rc + kk];
      } else if (kk - rcp < rr && (corr_a_scale[row] & 0x7FFFu) != 0) {
        code = corr_a[row * rr + (kk - rcp)];
      }
    }
    out[e] = (uint8_t)(code + 128);
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

cudaError_t launch_build_layouts(archead_pack *p, const uint8_t *res_codes, const void *res_scales,
                                 const uint16_t *row_scale, const void *core_u, const int8_t *corr_a,
                                 const uint16_t *corr_a_scale, cudaStream_t s) {
  const int KC = p->d_pad / kChunkK;
  build_res_codes_kernel<<<p->num_tiles * KC, 256, 0, s>>>(
      res_codes, p->sc4 ? nullptr : static_cast<const uint16_t *>(res_scales), p->codes, p->V, p->d, p->d_pad, p->G, p->g);
  if (p->sc4) {
    build_scale_codes_kernel<<<1024, 256, 0, s>>>(static_cast<const uint8_t *>(res_scales), p->scodes, p->V, p->V_pad,
                                                  p->G, p->G_pad2);
    build_row_scales_kernel<<<256, 256, 0, s>>>(row_scale, p->s_row, p->V, p->V_pad);
  } else {
    build_res_scales_kernel<<<1024, 256, 0, s>>>(static_cast<const uint16_t *>(res_scales), p->scales, p->V, p->V_pad,
                                                 p->G, p->G_pad);
  }
  if (p->nls > 0)
    build_lr_codes_kernel<<<p->num_tiles * p->nls, 256, 0, s>>>(core_u, corr_a, corr_a_scale, p->lr_codes, p->V, p->rc,
                                                                 p->rr, p->rcp, p->nls, p->sc4);
  // The decode layout, when it differs: the same codes with the core's
  // columns unpadded (rcp taken as r_c) and nls_dec steps.
  if (p->nls_dec > 0 && p->lr_codes_dec != p->lr_codes)
    build_lr_codes_kernel<<<p->num_tiles * p->nls_dec, 256, 0, s>>>(core_u, corr_a, corr_a_scale, p->lr_codes_dec, p->V,
                                                                     p->rc, p->rr, p->rc, p->nls_dec, p->sc4);
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
  const uint8_t *scodes;
  const uint16_t *s_row;
  int sc4, G_pad2;
  const uint8_t *lr_codes;
  const uint16_t *s_a, *s_u, *s_v, *s_b;
  const int8_t *q_v, *q_b;
  int d, d_pad, G_pad, g, rc, rr, rcp, nls;
};

// Position of (row-in-tile, column-in-16-step) inside a fragment: returns the
// lane and sets pair index i and half h.
__device__ __forceinline__ int frag_pos(int r, int k16, int &i, int &h) {
  const int mrow = r & 15;
  const int gq = mrow & 7;
  const int ihi = k16 >> 3;
  const int kp = k16 & 7;
  i = (mrow >> 3) + 2 * ihi;
  h = kp & 1;
  return gq * 4 + (kp >> 1);
}

__device__ __forceinline__ float pair_half(uint32_t v, int h) { return h ? bf16_hi(v) : bf16_lo(v); }

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
      const int mi = r >> 4;
      int i, h;
      if (comp == 0) {
        const int kc = col / kChunkK, kl = col % kChunkK;
        const int j = kl >> 4;
        const int lane = frag_pos(r, kl & 15, i, h);
        const int KC = a.d_pad / kChunkK;
        const uint32_t w = reinterpret_cast<const uint32_t *>(
            a.codes)[((((int64_t)vt * KC + kc) * 8 + mi) * 32 + lane) * 4 + j];
        uint32_t q[4];
        unpack_int4x8_biased(w, q);  // the decode kernel's operands: 136 + code
        const int grp = col / a.g;
        float sc;
        if (a.sc4) {
          const uint8_t b = a.scodes[((int64_t)vt * a.G_pad2 + (grp >> 1)) * kTileRows + r];
          sc = fp16_bits_to_f32(a.s_row[row]) * (float)(((b >> (4 * (grp & 1))) & 15) + 1);
        } else {
          sc = fp16_bits_to_f32(a.scales[((int64_t)vt * a.G_pad + grp) * kTileRows + r]);
        }
        v = (pair_half(q[i], h) - kInt4Bias) * sc;
      } else {
        const int kk = comp == 1 ? col : a.rcp + col;
        const int ls = kk >> 4;
        const int lane = frag_pos(r, kk & 15, i, h);
        const uint2 w2 = *reinterpret_cast<const uint2 *>(
            a.lr_codes + ((((int64_t)vt * a.nls + ls) * 8 + mi) * 32 + lane) * 8);
        uint32_t q[4];
        unpack_int8x8(w2.x, w2.y, q);
        const float sc = comp == 1 ? fp16_bits_to_f32(a.s_u[col]) : fp16_bits_to_f32(a.s_a[row]);
        v = pair_half(q[i], h) * sc;
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
  DequantArgs a{p->codes, p->scales, p->scodes, p->s_row, p->sc4,  p->G_pad2, p->lr_codes, p->s_a,
                p->s_u,   p->s_v,    p->s_b,    p->q_v,   p->q_b,  p->d,      p->d_pad,    p->G_pad,
                p->g,     p->rc,     p->rr,     p->rcp,   p->nls};
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
