// sq_device.cuh -- device-side helpers shared by the sm_103a kernels.
//
// Inline PTX used here: griddepcontrol (programmatic dependent launch),
// non-allocating 128-bit global loads, L2 bulk prefetch, mixed-precision
// fp16 x fp16 + fp32 fused multiply-add, E4M3 pair conversion.
#pragma once

#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace sq {

// Wait until the kernels this grid depends on (the previous launch on the
// stream) have completed and their writes are visible.  Without a
// programmatic dependency it returns at once.
__device__ __forceinline__ void griddep_wait() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}

// Allow the next kernel on the stream to start launching.  Its own
// griddep_wait() still waits for this grid to complete.
__device__ __forceinline__ void griddep_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// 16-byte load that streams through L1 without allocating (weights are
// read exactly once per launch).
__device__ __forceinline__ uint4 ld_stream16(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

// Asynchronous prefetch of [p, p + bytes) into L2.  p and bytes must be
// multiples of 16.
__device__ __forceinline__ void prefetch_l2_bulk(const void* p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes)
               : "memory");
}

// d = a * b + c with a, b fp16 and c, d fp32: the product of two fp16
// values is exact in fp32, so the only rounding is the fp32 sum.
__device__ __forceinline__ float fma_h(uint16_t a, uint16_t b, float c) {
  float d;
  asm("fma.rn.f32.f16 %0, %1, %2, %3;" : "=f"(d) : "h"(a), "h"(b), "f"(c));
  return d;
}

__device__ __forceinline__ uint16_t lo16(uint32_t v) { return (uint16_t)(v & 0xffffu); }
__device__ __forceinline__ uint16_t hi16(uint32_t v) { return (uint16_t)(v >> 16); }

// ss + x0^2 + x1^2 + ... + x7^2 (fp32 fused multiply-adds in element order)
// for eight fp16 values packed low half first: the RMSNorm sum of squares
// takes each 8-value chunk of a row in this order.
__device__ __forceinline__ float sumsq8(const uint4 q, float ss) {
  const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const float lo = __half2float(__ushort_as_half(lo16(w[e])));
    const float hi = __half2float(__ushort_as_half(hi16(w[e])));
    ss = fmaf(lo, lo, ss);
    ss = fmaf(hi, hi, ss);
  }
  return ss;
}

// Two E4M3 codes (low byte -> low half) to two fp16 values (exact: every
// E4M3 value is an fp16 value).
__device__ __forceinline__ uint32_t e4m3x2_to_f16x2(uint16_t codes) {
  uint32_t r;
  asm("cvt.rn.f16x2.e4m3x2 %0, %1;" : "=r"(r) : "h"(codes));
  return r;
}

// Two fp32 values to two E4M3 codes, nearest-even, saturating to +-448:
// `lo` goes to the low byte.
__device__ __forceinline__ uint16_t f32x2_to_e4m3x2(float lo, float hi) {
  uint16_t r;
  asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(r) : "f"(hi), "f"(lo));
  return r;
}

// Eight INT4 codes of one 32-bit word (nibble j = code for k = j, stored as
// c + 8) to four fp16x2 pairs holding the exact integers c:
//   out[0] = (k0, k4), out[1] = (k1, k5), out[2] = (k2, k6), out[3] = (k3, k7).
// 0x6400 is fp16 1024: OR-ing a nibble into the low mantissa bits gives
// 1024 + n exactly; a nibble in bits 4..7 gives 1024 + 16 n, which the
// multiply by 1/16 maps to 64 + n.  Subtracting (1024 + 8) or (64 + 8)
// leaves c = n - 8, exact in fp16.
__device__ __forceinline__ void int4x8_to_f16x2(uint32_t w, uint32_t out[4]) {
  const uint32_t MAGIC = 0x64006400u;
  const uint32_t LO = 0x000f000fu, HI = 0x00f000f0u;
  uint32_t a, b, c, d;
  const uint32_t w8 = w >> 8;
  asm("lop3.b32 %0, %1, %2, %3, 0xea;" : "=r"(a) : "r"(w), "r"(LO), "r"(MAGIC));
  asm("lop3.b32 %0, %1, %2, %3, 0xea;" : "=r"(b) : "r"(w), "r"(HI), "r"(MAGIC));
  asm("lop3.b32 %0, %1, %2, %3, 0xea;" : "=r"(c) : "r"(w8), "r"(LO), "r"(MAGIC));
  asm("lop3.b32 %0, %1, %2, %3, 0xea;" : "=r"(d) : "r"(w8), "r"(HI), "r"(MAGIC));
  const uint32_t SUB_LO = 0x64086408u;   // (1024 + 8, 1024 + 8)
  const uint32_t SIXTEENTH = 0x2c002c00u; // (1/16, 1/16)
  const uint32_t SUB_HI = 0xd480d480u;   // (-(64 + 8), -(64 + 8))
  asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(out[0]) : "r"(a), "r"(SUB_LO));
  asm("fma.rn.f16x2 %0, %1, %2, %3;" : "=r"(out[1]) : "r"(b), "r"(SIXTEENTH), "r"(SUB_HI));
  asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(out[2]) : "r"(c), "r"(SUB_LO));
  asm("fma.rn.f16x2 %0, %1, %2, %3;" : "=r"(out[3]) : "r"(d), "r"(SIXTEENTH), "r"(SUB_HI));
}

// The same eight codes as the raw fp16 values OR-ed onto 1024 (no bias
// removal): out[0] = (1024 + n0, 1024 + n4), out[1] = (1024 + 16 n1,
// 1024 + 16 n5), out[2] = (1024 + n2, 1024 + n6), out[3] = (1024 + 16 n3,
// 1024 + 16 n7), n_j = c_j + 8 the stored nibble.  Even k carry 1024 + n,
// odd k 1024 + 16 n; the linear kernel removes the offsets per 32-weight
// piece with precomputed activation sums.
__device__ __forceinline__ void int4x8_to_magic(uint32_t w, uint32_t out[4]) {
  const uint32_t MAGIC = 0x64006400u;
  const uint32_t LO = 0x000f000fu, HI = 0x00f000f0u;
  const uint32_t w8 = w >> 8;
  asm("lop3.b32 %0, %1, %2, %3, 0xea;" : "=r"(out[0]) : "r"(w), "r"(LO), "r"(MAGIC));
  asm("lop3.b32 %0, %1, %2, %3, 0xea;" : "=r"(out[1]) : "r"(w), "r"(HI), "r"(MAGIC));
  asm("lop3.b32 %0, %1, %2, %3, 0xea;" : "=r"(out[2]) : "r"(w8), "r"(LO), "r"(MAGIC));
  asm("lop3.b32 %0, %1, %2, %3, 0xea;" : "=r"(out[3]) : "r"(w8), "r"(HI), "r"(MAGIC));
}

// ---- packed fp32 pairs (f32x2) ------------------------------------------
// Accumulators and operands of fma.rn.f32x2 live in 64-bit registers holding
// (low = first, high = second) fp32 values.

__device__ __forceinline__ unsigned long long f2pack(float lo, float hi) {
  unsigned long long r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}

__device__ __forceinline__ float2 f2unpack(unsigned long long v) {
  float2 f;
  asm("mov.b64 {%0, %1}, %2;" : "=f"(f.x), "=f"(f.y) : "l"(v));
  return f;
}

// Two fp16 values (low half first) to an fp32 pair, exactly.
__device__ __forceinline__ unsigned long long h2_to_f2(uint32_t h2) {
  float lo, hi;
  asm("{\n"
      ".reg .b16 l, h;\n"
      "mov.b32 {l, h}, %2;\n"
      "cvt.f32.f16 %0, l;\n"
      "cvt.f32.f16 %1, h;\n"
      "}\n"
      : "=f"(lo), "=f"(hi)
      : "r"(h2));
  return f2pack(lo, hi);
}

// acc = a * b + acc on both lanes of the pairs (one instruction, two fp32
// fused multiply-adds rounded to nearest).
__device__ __forceinline__ void ffma2(unsigned long long& acc, unsigned long long a,
                                      unsigned long long b) {
  asm("fma.rn.f32x2 %0, %1, %2, %0;" : "+l"(acc) : "l"(a), "l"(b));
}

// ---- mbarrier and 1-D bulk copies (TMA engine, no tensor map) -------------

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

// Makes barrier initialisation visible to the async proxy (bulk copies).
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n"
      ".reg .pred p;\n"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      "selp.u32 %0, 1, 0, p;\n"
      "}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait for the phase with the given parity to complete.  Returns
// false after `limit` polls (each try_wait may itself suspend briefly); the
// caller then records a timeout instead of spinning forever.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity,
                                                  uint32_t limit = (1u << 26)) {
  for (uint32_t i = 0; i < limit; ++i)
    if (mbar_try_wait(bar, parity)) return true;
  return false;
}

// Bulk copy of `bytes` (multiple of 16, both addresses 16-byte aligned)
// from global memory into this CTA's shared memory, completing on `bar`.
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

// Named barrier over `count` threads (multiple of 32) of the CTA.
__device__ __forceinline__ void named_bar_sync(uint32_t id, uint32_t count) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

}  // namespace sq
