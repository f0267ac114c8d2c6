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
