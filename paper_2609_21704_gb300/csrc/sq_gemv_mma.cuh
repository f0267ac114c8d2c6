// sq_gemv_mma.cuh -- INT4 linear layer for ONE activation row (the draft pass
// at batch 1, Sec. III-D.2) with the multiply-adds on the tensor cores'
// register-operand path (mma.sync m16n8k16, fp16 inputs, fp32 accumulate).
//
// Why: at one activation row the CUDA-core GEMV spends most of its issue
// slots on products (one fp16 x fp16 -> fp32 multiply-add per weight plus
// the half-word moves around it), so the work left after its weights arrive
// is long.  Here a warp owns a tile of 16 output rows and a share of the
// 128-weight groups along K; per group each lane loads one 16-byte piece of
// row g and of row g + 8 (g = lane / 4: 32 codes each), turns them into the
// exact integers c = n - 8 as fp16 pairs in registers (int4x8_to_f16x2), and
// feeds them as the A operand of eight m16n8k16 steps.  The B operand is x:
// every lane supplies the same activations for its k slots, so all eight
// columns of the product equal the 16 dot products (no lane is wasted on
// selecting a column).  The k order inside a step is the order the nibble
// conversion produces; x is staged in shared memory in that order (chunk c
// of 8 values keeps its index, its values permuted).  Each group's 128
// products are summed by the MMA in fp32 from zero, then scaled by the
// group's fp16 scale into an fp32 accumulator (one fused multiply-add per
// row and group), exactly the streaming kernel's order of operations up to
// summation order.  Splitting K over S warps of a CTA keeps enough warps
// busy when there are few tiles; the S partial sums are added in warp order
// through shared memory (deterministic).  The fused RMSNorm of
// sq_linear_norm is applied while x is staged.
//
// Not tcgen05: its operands must sit in shared memory, and converting INT4
// codes into fp16 tiles there is what bounds the tile path's INT4 kernel; at
// one activation row the tensor cores only need to take over the products,
// which the register-operand MMA does with the converted codes still in
// registers.
#pragma once

#include "sq_gemv.cuh"

namespace sq {

constexpr int kMmaThreads = 256;
constexpr int kMmaWarps = kMmaThreads / 32;

// d = A * B + c for one m16n8k16 step (A row-major 16 x 16 fp16 in four
// fp16x2 registers, B column-major 16 x 8 fp16 in two, C and D fp32).
__device__ __forceinline__ void mma_16816(float d[4], const uint32_t a0, const uint32_t a1,
                                          const uint32_t a2, const uint32_t a3, const uint32_t b0,
                                          const uint32_t b1) {
  asm("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Eight activations (x0, x1), (x2, x3), (x4, x5), (x6, x7) reordered to the
// pairs the INT4 conversion yields: (x0, x4), (x2, x6), (x1, x5), (x3, x7).
__device__ __forceinline__ uint4 mma_x_order(const uint4 v) {
  return make_uint4(__byte_perm(v.x, v.z, 0x5410), __byte_perm(v.y, v.w, 0x5410),
                    __byte_perm(v.x, v.z, 0x7632), __byte_perm(v.y, v.w, 0x7632));
}

// RMSNorm of two fp16 values (low half first): fp16(x * r * gamma), each
// product rounded in fp32, as the standalone RMSNorm kernel computes it.
__device__ __forceinline__ uint32_t norm_f16x2(uint32_t xw, uint32_t gw, float r) {
  const float lo = __fmul_rn(__fmul_rn(__half2float(__ushort_as_half(lo16(xw))), r),
                             __half2float(__ushort_as_half(lo16(gw))));
  const float hi = __fmul_rn(__fmul_rn(__half2float(__ushort_as_half(hi16(xw))), r),
                             __half2float(__ushort_as_half(hi16(gw))));
  return (uint32_t)__half_as_ushort(__float2half_rn(lo)) |
         ((uint32_t)__half_as_ushort(__float2half_rn(hi)) << 16);
}

// SILU: gate rows [0, N) and up rows [N, 2N) of the weight, tile by tile;
// S: warps sharing one tile's K range.
// PIPE: two register batches alternate (the next batch's loads are issued
// before the current batch's products); 80 registers, three CTAs per SM.
// Without it, one batch at a time at 64 registers and four CTAs per SM.
template <bool SILU, int S, bool PIPE>
__global__ void __launch_bounds__(kMmaThreads, PIPE ? 3 : 4) gemv_mma_int4_kernel(const GemvArgs a) {
  constexpr int WR = SILU ? 2 : 1;     // weight tiles per output tile (gate, up)
  constexpr int TPC = kMmaWarps / S;   // output tiles a CTA works on at once
  constexpr int U = SILU ? 1 : 2;      // groups per load batch
  extern __shared__ uint4 xm[];        // x in MMA order (K / 8 chunks), then partial sums
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int g = lane >> 2, t = lane & 3;
  const int64_t G = a.K / 128;
  const int64_t ntiles = (a.N + 15) / 16;
  const int64_t nsets = (ntiles + TPC - 1) / TPC;
  const int part = warp % S;  // this warp's share of the groups: [j0, j1)
  const int64_t j0 = part * G / S, j1 = (part + 1) * G / S;
  float* red = reinterpret_cast<float*>(xm + a.K / 8);  // [warp][WR][16]
  const __half* gscale = reinterpret_cast<const __half*>(a.scales);

  // One batch: groups jb .. jb + U - 1 of rows g and g + 8 of the tile (and
  // of its up tile): this lane's 16-byte piece t of each group, and the
  // group scales.
  uint4 wv[U][WR][2];
  __half2 sv[U][WR];  // (row g, row g + 8)
  auto load = [&](int64_t tile, int64_t jb) {
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int64_t j = jb + u;
#pragma unroll
      for (int h = 0; h < WR; ++h) {
        __half s2[2];
#pragma unroll
        for (int rr = 0; rr < 2; ++rr) {
          const int64_t n = tile * 16 + g + 8 * rr;
          const bool ok = j < j1 && tile < ntiles && n < a.N;
          const int64_t row = (h ? a.N : 0) + (ok ? n : 0);
          wv[u][h][rr] = ok ? ld_stream16(a.w + row * a.row_bytes + j * 64 + t * 16)
                            : make_uint4(0u, 0u, 0u, 0u);
          s2[rr] = ok ? gscale[row * G + j] : __ushort_as_half(0);
        }
        sv[u][h] = __halves2half2(s2[0], s2[1]);
      }
    }
  };

  // the weights never depend on the previous kernel: first batch before the wait
  const int64_t first_tile = (int64_t)blockIdx.x * TPC + warp / S;
  if ((int64_t)blockIdx.x < nsets) load(first_tile, j0);

  griddep_wait();
  griddep_launch_dependents();

  // ---- stage x in MMA order.  With a.gamma (fused RMSNorm) the sum of
  // squares follows the standalone RMSNorm kernel's order (thread t takes the
  // 8-value chunks t, t + 256, ... in element order, then warp sums, then the
  // eight warp sums in order) and x * r * gamma is applied elementwise, so
  // the staged rows equal its output bit for bit.
  float ss = 0.0f;
  for (int64_t c = threadIdx.x; c < a.K / 8; c += kMmaThreads) {
    const uint4 v = reinterpret_cast<const uint4*>(a.x)[c];
    if (a.gamma != nullptr) ss = sumsq8(v, ss);
    xm[c] = mma_x_order(v);
  }
  if (a.gamma != nullptr) {
    __shared__ float nred[kMmaWarps];
    __shared__ float rinv;
    ss = warp_sum(ss);
    if (lane == 0) nred[warp] = ss;
    __syncthreads();
    if (threadIdx.x == 0) {
      float tot = 0.0f;
      for (int w = 0; w < kMmaWarps; ++w) tot += nred[w];
      rinv = 1.0f / sqrtf(tot / (float)a.K + a.eps);
    }
    __syncthreads();
    const float r = rinv;
    for (int64_t c = threadIdx.x; c < a.K / 8; c += kMmaThreads) {
      const uint4 q = xm[c];
      const uint4 gm = mma_x_order(reinterpret_cast<const uint4*>(a.gamma)[c]);
      xm[c] = make_uint4(norm_f16x2(q.x, gm.x, r), norm_f16x2(q.y, gm.y, r), norm_f16x2(q.z, gm.z, r),
                         norm_f16x2(q.w, gm.w, r));
    }
  }
  __syncthreads();

  // PIPE: two register batches alternate, so a warp always has a batch in
  // flight (the first batch of the CTA's first set was issued before the
  // wait on the previous kernel).
  uint4 wb[PIPE ? U : 1][WR][2];
  __half2 sb[PIPE ? U : 1][WR];
  auto load_into = [&](uint4 (&dw)[PIPE ? U : 1][WR][2], __half2 (&ds)[PIPE ? U : 1][WR], int64_t tile,
                       int64_t jb) {
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int64_t j = jb + u;
#pragma unroll
      for (int h = 0; h < WR; ++h) {
        __half s2[2];
#pragma unroll
        for (int rr = 0; rr < 2; ++rr) {
          const int64_t n = tile * 16 + g + 8 * rr;
          const bool ok = j < j1 && tile < ntiles && n < a.N;
          const int64_t row = (h ? a.N : 0) + (ok ? n : 0);
          dw[u][h][rr] = ok ? ld_stream16(a.w + row * a.row_bytes + j * 64 + t * 16)
                            : make_uint4(0u, 0u, 0u, 0u);
          s2[rr] = ok ? gscale[row * G + j] : __ushort_as_half(0);
        }
        ds[u][h] = __halves2half2(s2[0], s2[1]);
      }
    }
  };
  // products of one batch (groups jb .. jb + U - 1) into acc
  auto compute = [&](const uint4 (&cw)[U][WR][2], const __half2 (&cs)[U][WR], int64_t jb, float (&acc)[WR][2]) {
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int64_t j = jb + u;
      if (j >= j1) break;  // warp-uniform
      float d[WR][4];
#pragma unroll
      for (int h = 0; h < WR; ++h) d[h][0] = d[h][1] = d[h][2] = d[h][3] = 0.0f;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const uint4 xq = xm[j * 16 + t * 4 + q];
#pragma unroll
        for (int h = 0; h < WR; ++h) {
          uint32_t p0[4], p1[4];  // rows g and g + 8: (k0,k4) (k1,k5) (k2,k6) (k3,k7)
          const uint4 w0 = cw[u][h][0], w1 = cw[u][h][1];
          int4x8_to_f16x2(q == 0 ? w0.x : q == 1 ? w0.y : q == 2 ? w0.z : w0.w, p0);
          int4x8_to_f16x2(q == 0 ? w1.x : q == 1 ? w1.y : q == 2 ? w1.z : w1.w, p1);
          mma_16816(d[h], p0[0], p1[0], p0[2], p1[2], xq.x, xq.y);
          mma_16816(d[h], p0[1], p1[1], p0[3], p1[3], xq.z, xq.w);
        }
      }
#pragma unroll
      for (int h = 0; h < WR; ++h) {
        const float2 sc = __half22float2(cs[u][h]);
        acc[h][0] = fmaf(sc.x, d[h][0], acc[h][0]);  // row g, column 2t
        acc[h][1] = fmaf(sc.y, d[h][2], acc[h][1]);  // row g + 8
      }
    }
  };

  for (int64_t set = blockIdx.x; set < nsets; set += gridDim.x) {
    const int64_t tile = set * TPC + warp / S;
    float acc[WR][2];  // rows g and g + 8 of each weight tile
#pragma unroll
    for (int h = 0; h < WR; ++h) acc[h][0] = acc[h][1] = 0.0f;
    if constexpr (PIPE) {
      if (set != (int64_t)blockIdx.x) load(tile, j0);
      for (int64_t jb = j0; jb < j1; jb += 2 * U) {
        if (jb + U < j1) load_into(wb, sb, tile, jb + U);
        compute(wv, sv, jb, acc);
        if (jb + U < j1) {
          if (jb + 2 * U < j1) load_into(wv, sv, tile, jb + 2 * U);
          compute(wb, sb, jb + U, acc);
        }
      }
    } else {
      for (int64_t jb = j0; jb < j1; jb += U) {
        if (set != (int64_t)blockIdx.x || jb != j0) load(tile, jb);
        compute(wv, sv, jb, acc);
      }
    }
    // ---- the S shares of K in warp order, then the epilogue (lane t == 0
    // of each row pair writes rows g and g + 8)
    if constexpr (S == 1) {
      if (t == 0 && tile < ntiles)
#pragma unroll
        for (int rr = 0; rr < 2; ++rr) {
          const int64_t n = tile * 16 + g + 8 * rr;
          if (n < a.N) gemv_store<WK_INT4, SILU>(a, n, 0, acc[0][rr], acc[WR - 1][rr]);
        }
    } else {
      if (t == 0)
#pragma unroll
        for (int h = 0; h < WR; ++h)
#pragma unroll
          for (int rr = 0; rr < 2; ++rr) red[(warp * WR + h) * 16 + g + 8 * rr] = acc[h][rr];
      __syncthreads();
      if (part == 0 && t == 0 && tile < ntiles) {
#pragma unroll
        for (int rr = 0; rr < 2; ++rr) {
          const int64_t n = tile * 16 + g + 8 * rr;
          float v[WR];
#pragma unroll
          for (int h = 0; h < WR; ++h) {
            v[h] = 0.0f;
            for (int s = 0; s < S; ++s) v[h] += red[((warp + s) * WR + h) * 16 + g + 8 * rr];
          }
          if (n < a.N) gemv_store<WK_INT4, SILU>(a, n, 0, v[0], v[WR - 1]);
        }
      }
      __syncthreads();  // red is reused by the next set
    }
  }
}

// Shared memory of one CTA: x in MMA order, then the partial sums.
inline size_t gemv_mma_smem_bytes(int64_t K) { return (size_t)K * 2 + (size_t)kMmaWarps * 2 * 16 * 4; }

template <bool SILU, int S, bool PIPE>
cudaError_t launch_mma_inst(const GemvArgs& a, size_t smem, cudaStream_t st) {
  auto k = gemv_mma_int4_kernel<SILU, S, PIPE>;
  static int occ_cache[64] = {0};  // per device: resident CTAs per SM
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (smem > 48 * 1024) {
    e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  if (occ_cache[dev] == 0) {
    int occ = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, k, kMmaThreads, smem);
    if (e != cudaSuccess) return e;
    occ_cache[dev] = occ > 0 ? occ : 1;
  }
  constexpr int TPC = kMmaWarps / S;
  const int64_t nsets = ((a.N + 15) / 16 + TPC - 1) / TPC;
  const int64_t cap = (int64_t)device_sm_count() * occ_cache[dev];
  const int grid = (int)(nsets < cap ? nsets : cap);
  return launch_pdl(k, dim3(grid > 0 ? grid : 1), dim3(kMmaThreads), smem, st, a);
}

// S from the tile count: the smallest split that gives every SM a full
// complement of warps, at most one warp per 128-weight group.
inline int gemv_mma_split(int64_t N, int64_t K) {
  const int64_t tiles = (N + 15) / 16, G = K / 128;
  int S = 1;
  while (S < 8 && S * 2 <= G && tiles * S < (int64_t)device_sm_count() * 32) S *= 2;
  return S;
}

// The pipelined form when the whole grid is one wave at three CTAs per SM
// (measured on the 14B shapes, us per launch: q/k/v 7.71 -> 7.12, o 7.31 ->
// 6.83, down 15.54 -> 12.82; larger grids lose more to the lower occupancy
// than they gain: lm_head 82.3 -> 90.2, the 1.5B fused gate/up 5.0 -> 6.5).
inline bool gemv_mma_pipelined(int64_t N, int S) {
  const int64_t tiles = (N + 15) / 16;
  const int64_t nsets = (tiles + kMmaWarps / S - 1) / (kMmaWarps / S);
  return nsets <= 3 * (int64_t)device_sm_count();
}

inline cudaError_t launch_gemv_mma_int4_impl(const GemvArgs& a, bool silu, cudaStream_t st) {
  const size_t smem = gemv_mma_smem_bytes(a.K);
  const int S = gemv_mma_split(a.N, a.K);
  const bool pipe = gemv_mma_pipelined(a.N, S);
#define SQ_MMA_CASE(S_)                                                                           \
  if (S == S_) {                                                                                  \
    if (pipe) return silu ? launch_mma_inst<true, S_, true>(a, smem, st)                           \
                          : launch_mma_inst<false, S_, true>(a, smem, st);                          \
    return silu ? launch_mma_inst<true, S_, false>(a, smem, st) : launch_mma_inst<false, S_, false>(a, smem, st); \
  }
  SQ_MMA_CASE(1)
  SQ_MMA_CASE(2)
  SQ_MMA_CASE(4)
  SQ_MMA_CASE(8)
#undef SQ_MMA_CASE
  return cudaErrorInvalidValue;
}

}  // namespace sq
