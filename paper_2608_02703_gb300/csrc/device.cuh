// Device helpers shared by the sm_103a kernels: code unpacking, mbarrier and
// bulk-copy wrappers (inline PTX), the warp-level mma.sync bf16 MMA used by the decode
// kernel, and the bounded-wait error protocol.
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <stdint.h>

namespace archead {

// Bits of the per-pack device error word.
constexpr int kErrWaitTimeout = 1;
constexpr int kErrTargetRange = 2;
constexpr int kErrLayout = 4;  // a kernel found its shared memory misaligned and did nothing

// ---------------------------------------------------------------------------
// INT4 / INT8 code unpacking to exact bf16 operands.
//
// Residual codes are stored offset-binary (code + 8, 0..15) in the tiled
// layout.  Nibbles i and i+4 of a 32-bit word form bf16 pair i: OR-ing the
// nibble into the mantissa of bf16 128.0 gives 128 + (code + 8) exactly.  The
// two halves of each output register are the (lower, higher) k of one pair.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t bf16x2_sub(uint32_t a, uint32_t b) {
  __nv_bfloat162 r = __hsub2(*reinterpret_cast<__nv_bfloat162 *>(&a), *reinterpret_cast<__nv_bfloat162 *>(&b));
  return *reinterpret_cast<uint32_t *>(&r);
}

// (a & b) | c in one LOP3.  Written out because the compiler splits the
// expression into two logic operations when b and c are both immediates.
__device__ __forceinline__ uint32_t lop3_and_or(uint32_t a, uint32_t b, uint32_t c) {
  uint32_t d;
  asm("lop3.b32 %0, %1, %2, %3, 0xEA;\n" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  return d;
}

// Biased operands: each half is 136 + code (128..143, exact in bf16).  The
// decode kernel multiplies these directly; the MMAs of each quantisation
// group start from -136 * sum(x) over the group, which removes the bias.
__device__ __forceinline__ void unpack_int4x8_biased(uint32_t w, uint32_t (&a)[4]) {
  const uint32_t kMask = 0x000F000Fu;
  const uint32_t kMagic = 0x43004300u;  // bf16 128.0 | 128.0
  a[0] = lop3_and_or(w, kMask, kMagic);
  a[1] = lop3_and_or(w >> 4, kMask, kMagic);
  a[2] = lop3_and_or(w >> 8, kMask, kMagic);
  a[3] = lop3_and_or(w >> 12, kMask, kMagic);
}

constexpr float kInt4Bias = 136.0f;

// fp16 operands for the decode kernel: OR-ing a nibble into the mantissa of
// fp16 1024.0 is exact at bits 0-3 (1024 + n) and at bits 4-7 (1024 + 16 n),
// so a word's eight nibbles need one shift and four LOP3s.  Registers a[0],
// a[2] (rows gq of the m16n8k16 A fragment) hold 1024 + n = 1032 + code;
// a[1], a[3] (rows gq + 8) hold 1024 + 16 n = 1152 + 16 code.  The kernel
// starts each group's MMAs from -1032 * sum(x) resp. -1152 * sum(x) and
// scales rows gq + 8 by 1/16 at promotion.
constexpr float kF16BiasLo = 1032.0f;
constexpr float kF16BiasHi = 1152.0f;

__device__ __forceinline__ void unpack_int4x8_f16(uint32_t w, uint32_t (&a)[4]) {
  const uint32_t kMagic = 0x64006400u;  // fp16 1024.0 | 1024.0
  const uint32_t t = w >> 8;
  a[0] = lop3_and_or(w, 0x000F000Fu, kMagic);
  a[1] = lop3_and_or(w, 0x00F000F0u, kMagic);
  a[2] = lop3_and_or(t, 0x000F000Fu, kMagic);
  a[3] = lop3_and_or(t, 0x00F000F0u, kMagic);
}

// Exact codes: the biased operands minus 136.0 (exact in bf16).
__device__ __forceinline__ void unpack_int4x8(uint32_t w, uint32_t (&a)[4]) {
  constexpr uint32_t kBias = 0x43084308u;  // bf16 136.0 | 136.0
  unpack_int4x8_biased(w, a);
#pragma unroll
  for (int i = 0; i < 4; ++i) a[i] = bf16x2_sub(a[i], kBias);
}

// INT8 codes are stored offset-binary (code + 128).  Placing byte u in the
// low mantissa bits of fp32 2^23 gives 2^23 + u exactly; subtracting
// 2^23 + 128 leaves the code, which bf16 represents exactly (|code| <= 128).
__device__ __forceinline__ float int8_ob_to_f32(uint32_t word, int byte) {
  uint32_t bits = __byte_perm(word, 0x4B000000u, 0x7650u | (uint32_t)byte);
  return __uint_as_float(bits) - 8388736.0f;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 r = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t *>(&r);
}

// Two words = eight offset-binary INT8 codes; bytes 2i, 2i+1 form pair i.
__device__ __forceinline__ void unpack_int8x8(uint32_t w0, uint32_t w1, uint32_t (&a)[4]) {
  a[0] = pack_bf16x2(int8_ob_to_f32(w0, 0), int8_ob_to_f32(w0, 1));
  a[1] = pack_bf16x2(int8_ob_to_f32(w0, 2), int8_ob_to_f32(w0, 3));
  a[2] = pack_bf16x2(int8_ob_to_f32(w1, 0), int8_ob_to_f32(w1, 1));
  a[3] = pack_bf16x2(int8_ob_to_f32(w1, 2), int8_ob_to_f32(w1, 3));
}

__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xFFFF0000u); }

__device__ __forceinline__ float fp16_bits_to_f32(uint16_t h) {
  return __half2float(__ushort_as_half(h));
}

// ---------------------------------------------------------------------------
// Warp-level bf16 MMA, m16n8k16, fp32 accumulate (used by the decode kernel,
// where the vocabulary rows are the 16-row side and tokens the 8-column side).
// ---------------------------------------------------------------------------
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Same with a zero accumulator input (the first k step of a group).
__device__ __forceinline__ void mma_bf16_16816_zero(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%10,%10,%10,%10};\n"
      : "=f"(d[0]), "=f"(d[1]), "=f"(d[2]), "=f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1), "f"(0.f));
}

// Same with the accumulator input taken from (c_lo.x, c_lo.y, c_hi.x, c_hi.y)
// (the first k step of a group, started from the group's bias term).
__device__ __forceinline__ void mma_bf16_16816_c(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1,
                                                 float2 c_lo, float2 c_hi) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%10,%11,%12,%13};\n"
      : "=f"(d[0]), "=f"(d[1]), "=f"(d[2]), "=f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1), "f"(c_lo.x), "f"(c_lo.y), "f"(c_hi.x),
        "f"(c_hi.y));
}

// fp16 x fp16 -> fp32 variants (the decode kernel's residual operands).
__device__ __forceinline__ void mma_f16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ void mma_f16_16816_zero(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%10,%10,%10,%10};\n"
      : "=f"(d[0]), "=f"(d[1]), "=f"(d[2]), "=f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1), "f"(0.f));
}

__device__ __forceinline__ void mma_f16_16816_c(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1,
                                                float2 c_lo, float2 c_hi) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%10,%11,%12,%13};\n"
      : "=f"(d[0]), "=f"(d[1]), "=f"(d[2]), "=f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1), "f"(c_lo.x), "f"(c_lo.y), "f"(c_hi.x),
        "f"(c_hi.y));
}

// ---------------------------------------------------------------------------
// mbarrier + bulk async copy (TMA, 1-D) wrappers.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void *p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;\n" ::"r"(smem_u32(bar)), "r"(count));
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
}

__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
  asm volatile("{\n .reg .b64 st;\n mbarrier.arrive.shared::cta.b64 st, [%0];\n}\n" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes) {
  asm volatile("{\n .reg .b64 st;\n mbarrier.arrive.expect_tx.shared::cta.b64 st, [%0], %1;\n}\n" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

// One probe of the phase with the given parity.  A thread whose phase is not
// complete yet may be suspended by the hardware for a system-dependent time
// (no explicit hint: a 1 ms hint measured 1-3 % slower in the prefill kernel,
// whose pipeline hand-offs are latency-critical).
__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait: spins until the phase with the given parity completed, the
// block-wide abort flag (if any) is raised, or `budget` clock cycles pass.  On
// timeout it latches kErrWaitTimeout in *err and raises the abort flag.
// Returns false when the caller must stop.
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity, int64_t budget, volatile int *abort_flag,
                                          int *err) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (abort_flag != nullptr && *abort_flag) return false;
    if (clock64() - t0 > budget) {
      atomicOr(err, kErrWaitTimeout);
      if (abort_flag != nullptr) *abort_flag = 1;
      return false;
    }
  }
}

// True in exactly one lane of a converged warp (elect.sync).  Guarding the
// single-thread issue of tcgen05 / TMA instructions with it, instead of a
// test on the lane index, keeps the issuing code warp-uniform.
__device__ __forceinline__ bool elect_one() {
  uint32_t pred = 0;
  asm volatile(
      "{\n .reg .b32 r;\n .reg .pred p;\n elect.sync r|p, 0xffffffff;\n selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(pred));
  return pred != 0;
}

// mbar_wait for a whole converged warp: every lane calls it and every lane
// gets the same answer (the decisions are warp votes), so the code after a
// wait stays warp-uniform.  Same bound and error reporting as mbar_wait.
__device__ __forceinline__ bool mbar_wait_warp(uint64_t *bar, uint32_t parity, int64_t budget,
                                               volatile int *abort_flag, int *err) {
  if (__all_sync(0xffffffffu, mbar_try_wait(bar, parity))) return true;
  const long long t0 = clock64();
  while (true) {
    if (__all_sync(0xffffffffu, mbar_try_wait(bar, parity))) return true;
    if (__any_sync(0xffffffffu, abort_flag != nullptr && *abort_flag)) return false;
    if (__any_sync(0xffffffffu, clock64() - t0 > budget)) {
      if (elect_one()) {
        atomicOr(err, kErrWaitTimeout);
        if (abort_flag != nullptr) *abort_flag = 1;
      }
      return false;
    }
  }
}

// 2-D tensor copy (TMA) of one box at (c0 = column, c1 = row) into shared
// memory, completing on an mbarrier.  c0 * element size must be a multiple
// of 16 bytes.
__device__ __forceinline__ void tma_load_2d(void *dst, const void *map, int c0, int c1, uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];\n" ::"r"(
          smem_u32(dst)),
      "l"(map), "r"(c0), "r"(c1), "r"(smem_u32(bar))
      : "memory");
}

// Global -> shared bulk copy completing on an mbarrier (size multiple of 16,
// both addresses 16-byte aligned).
__device__ __forceinline__ void bulk_g2s(void *dst_smem, const void *src_gmem, uint32_t bytes, uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];\n" ::"r"(
          smem_u32(dst_smem)),
      "l"(src_gmem), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

// Same, tagged with an L2 eviction policy (from make_evict_first_policy):
// data read once should not push out small hot data such as the rank-r
// factors that another warp reads while the stream runs.
__device__ __forceinline__ void bulk_g2s_hint(void *dst_smem, const void *src_gmem, uint32_t bytes, uint64_t *bar,
                                              uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;\n" ::"r"(
          smem_u32(dst_smem)),
      "l"(src_gmem), "r"(bytes), "r"(smem_u32(bar)), "l"(policy)
      : "memory");
}

__device__ __forceinline__ uint64_t make_evict_first_policy() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;\n" : "=l"(pol));
  return pol;
}

__device__ __forceinline__ int lane_id() { return threadIdx.x & 31; }

// Online log-sum-exp pair (running max, sum of exp(y - max)).
struct LsePair {
  float m, s;
};

__device__ __forceinline__ LsePair lse_merge(LsePair a, LsePair b) {
  if (a.m == -INFINITY) return b;
  if (b.m == -INFINITY) return a;
  float m = fmaxf(a.m, b.m);
  return {m, a.s * __expf(a.m - m) + b.s * __expf(b.m - m)};
}

}  // namespace archead
