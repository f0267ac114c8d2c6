// sq_quantize.cu -- derive the draft variants from the FP16 parent.
//
// Sec. III-A.1: Q4 = f(W16, 4).  Sec. III-A.2: Q8 = f(W16, 8).  The paper
// names no scheme; the one implemented (and documented in specquant.h):
//   INT4: per 128-wide group along K, s = fp16(fp32(amax / 7)) (2^-24 if
//         that rounds to zero for amax > 0), c = clamp(rint(w / s), -8, 7).
//   FP8:  per output row, s = fp32(amax / 448), code = E4M3_satfinite(w / s).
// Every division is the IEEE fp32 divide (__fdiv_rn) and every rounding is
// to nearest even, so codes and scales are bit-identical to the definition.
// These kernels never let the next kernel start early: linear kernels read
// their weights before waiting on the previous kernel, and the weights may
// be what this kernel writes.
// Both kernels are HBM-bound streaming passes: 2 B read per weight, 0.516 B
// (INT4) or 1 B (FP8) written.
#include "sq_internal.h"

namespace sq {

__device__ unsigned int g_quant_status;

// One warp per (row, group): lane l holds k = 4l .. 4l+3 of the group.
__global__ void __launch_bounds__(256) quant_int4_kernel(const __half* __restrict__ w, int64_t N,
                                                         int64_t K, uint8_t* __restrict__ codes,
                                                         __half* __restrict__ scales) {
  griddep_wait();  // no early trigger: a linear call may read these outputs at once
  const int lane = threadIdx.x & 31;
  const int64_t G = K / 128;
  const int64_t total = N * G;
  const int64_t nwarps = (int64_t)gridDim.x * (blockDim.x >> 5);
  for (int64_t gid = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); gid < total;
       gid += nwarps) {
    const int64_t n = gid / G, g = gid - n * G;
    const __half* src = w + n * K + g * 128 + lane * 4;
    const uint2 raw = *reinterpret_cast<const uint2*>(src);
    float v[4];
    v[0] = __half2float(__ushort_as_half(lo16(raw.x)));
    v[1] = __half2float(__ushort_as_half(hi16(raw.x)));
    v[2] = __half2float(__ushort_as_half(lo16(raw.y)));
    v[3] = __half2float(__ushort_as_half(hi16(raw.y)));
    float a = 0.0f;
    bool bad = false;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      bad |= !isfinite(v[i]);
      a = fmaxf(a, fabsf(v[i]));
    }
    if (__any_sync(0xffffffffu, bad) && lane == 0) atomicOr(&g_quant_status, SQ_DEV_NONFINITE_WEIGHT);
    const float amax = warp_max(a);
    __half sh = __float2half_rn(__fdiv_rn(amax, 7.0f));
    if (amax > 0.0f && __half_as_ushort(sh) == 0) sh = __ushort_as_half(1);
    const float s = __half2float(sh);
    uint32_t packed = 0;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      int c = 0;
      if (s != 0.0f) {
        float t = rintf(__fdiv_rn(v[i], s));
        t = fminf(fmaxf(t, -8.0f), 7.0f);
        c = (int)t;
      }
      packed |= (uint32_t)(c + 8) << (4 * i);
    }
    *reinterpret_cast<uint16_t*>(codes + n * (K / 2) + g * 64 + lane * 2) = (uint16_t)packed;
    if (lane == 0) scales[n * G + g] = sh;
  }
}

// One CTA per row (grid-stride): pass 1 finds amax, pass 2 (re-reading the
// row from L1/L2) encodes 8 weights per thread-iteration.
__global__ void __launch_bounds__(256) quant_fp8_kernel(const __half* __restrict__ w, int64_t N,
                                                        int64_t K, uint8_t* __restrict__ codes,
                                                        float* __restrict__ scales) {
  griddep_wait();  // no early trigger: a linear call may read these outputs at once
  __shared__ float red[8];
  __shared__ int red_bad[8];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t chunks = K / 8;
  for (int64_t n = blockIdx.x; n < N; n += gridDim.x) {
    const uint4* row = reinterpret_cast<const uint4*>(w + n * K);
    float a = 0.0f;
    int bad = 0;
    for (int64_t c = threadIdx.x; c < chunks; c += blockDim.x) {
      const uint4 r = row[c];
      const uint32_t u[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float x0 = __half2float(__ushort_as_half(lo16(u[i])));
        const float x1 = __half2float(__ushort_as_half(hi16(u[i])));
        bad |= !isfinite(x0) | !isfinite(x1);
        a = fmaxf(a, fmaxf(fabsf(x0), fabsf(x1)));
      }
    }
    a = warp_max(a);
    bad = __any_sync(0xffffffffu, bad);
    if (lane == 0) {
      red[warp] = a;
      red_bad[warp] = bad;
    }
    __syncthreads();
    float amax = 0.0f;
    int any_bad = 0;
    for (int i = 0; i < (int)(blockDim.x >> 5); ++i) {
      amax = fmaxf(amax, red[i]);
      any_bad |= red_bad[i];
    }
    __syncthreads();
    if (any_bad && threadIdx.x == 0) atomicOr(&g_quant_status, SQ_DEV_NONFINITE_WEIGHT);
    const float s = __fdiv_rn(amax, 448.0f);
    if (threadIdx.x == 0) scales[n] = s;
    uint2* out = reinterpret_cast<uint2*>(codes + n * K);
    for (int64_t c = threadIdx.x; c < chunks; c += blockDim.x) {
      const uint4 r = row[c];
      const uint32_t u[4] = {r.x, r.y, r.z, r.w};
      uint32_t o[2] = {0u, 0u};
      if (s != 0.0f) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const float x0 = __fdiv_rn(__half2float(__ushort_as_half(lo16(u[i]))), s);
          const float x1 = __fdiv_rn(__half2float(__ushort_as_half(hi16(u[i]))), s);
          o[i >> 1] |= (uint32_t)f32x2_to_e4m3x2(x0, x1) << (16 * (i & 1));
        }
      }
      out[c] = make_uint2(o[0], o[1]);
    }
  }
}

cudaError_t launch_quant_int4(const void* w, int64_t N, int64_t K, void* codes, void* scales,
                              cudaStream_t st) {
  const int64_t total = N * (K / 128);
  if (total == 0) return cudaSuccess;
  const int64_t want = (total + 7) / 8;
  const int grid = (int)(want < 152 * 16 ? want : 152 * 16);
  return launch_pdl(quant_int4_kernel, dim3(grid), dim3(256), 0, st,
                    reinterpret_cast<const __half*>(w), N, K, reinterpret_cast<uint8_t*>(codes),
                    reinterpret_cast<__half*>(scales));
}

cudaError_t launch_quant_fp8(const void* w, int64_t N, int64_t K, void* codes, void* scales,
                             cudaStream_t st) {
  if (N == 0) return cudaSuccess;
  const int grid = (int)(N < 152 * 8 ? N : 152 * 8);
  return launch_pdl(quant_fp8_kernel, dim3(grid), dim3(256), 0, st,
                    reinterpret_cast<const __half*>(w), N, K, reinterpret_cast<uint8_t*>(codes),
                    reinterpret_cast<float*>(scales));
}

cudaError_t take_quant_status(uint32_t* bits) {
  uint32_t v = 0, zero = 0;
  cudaError_t e = cudaMemcpyFromSymbol(&v, g_quant_status, sizeof(v));
  if (e != cudaSuccess) return e;
  if (v) e = cudaMemcpyToSymbol(g_quant_status, &zero, sizeof(zero));
  *bits |= v;
  return e;
}

}  // namespace sq
