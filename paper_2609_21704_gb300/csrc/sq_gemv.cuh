// sq_gemv.cuh -- skinny linear layer y = x W'^T for 1..16 activation rows
// on CUDA cores (Sec. III-D.2 draft pass at M = batch, Sec. III-D.3 verify
// pass at M = batch * (K+1) while that stays below a tensor-core tile).
//
// The work is HBM-bound: every weight byte is read once; x (M x K fp16) and
// y are small.  Mapping:
//   * a warp owns R weight rows (2R for the fused SiLU gate) and sweeps the
//     whole row, each lane taking one 16-byte piece of each row per step
//     (32 INT4, 16 FP8 or 8 FP16 weights) with a non-allocating 128-bit
//     load: 512 contiguous bytes per row per warp-step, fully coalesced;
//   * x is staged once per CTA into shared memory, permuted so that the
//     16-byte x chunk lane l needs at sub-step i sits at slot
//     (step * SUB + i) * 32 + l: 32 lanes read 512 consecutive bytes, no
//     bank conflicts, and each x chunk serves R rows from registers;
//   * products are fp16 x fp16 -> fp32 (exact) with fp32 accumulation
//     (fma.rn.f32.f16); INT4 codes become exact fp16 integers with two
//     logic ops and one packed fp16 op per pair, and the group scale is
//     applied once per 32-weight piece; the FP8 row scale once per output;
//   * the per-lane partial sums are reduced with warp shuffles in a fixed
//     order, so results are reproducible run to run.
// Each CTA owns a contiguous slice of row tiles and each warp the tiles
// w, w + 8, ... of it.  A lane keeps U 16-byte pieces of each of its rows in
// flight per batch (U x 512 B per row per warp), and every warp keeps the
// bytes of its next kPrefetchTiles tiles requested into L2 with bulk
// prefetches (cp.async.bulk.prefetch.L2).  The first batch and the first
// prefetches are issued before waiting on the kernel that produces x:
// weights never depend on it, so with programmatic dependent launch the
// weight fetch overlaps that kernel's tail.  The grid holds as many CTAs as
// can be resident at once (occupancy calculator): many warps per SM are
// what keeps the issue slots busy.
#pragma once

#include "sq_internal.h"

namespace sq {

enum { WK_FP16 = 0, WK_INT4 = 1, WK_FP8 = 2 };

template <int WK>
struct WTraits;
template <>
struct WTraits<WK_INT4> {
  static constexpr int kWeightsPerPiece = 32;
  static constexpr int kSub = 4;  // 8-weight x chunks per piece
};
template <>
struct WTraits<WK_FP8> {
  static constexpr int kWeightsPerPiece = 16;
  static constexpr int kSub = 2;
};
template <>
struct WTraits<WK_FP16> {
  static constexpr int kWeightsPerPiece = 8;
  static constexpr int kSub = 1;
};

constexpr int kGemvThreads = 256;
constexpr int kGemvWarps = kGemvThreads / 32;
constexpr int kPrefetchTiles = 2;  // tiles of its own a warp keeps requested into L2

// Status word of the GEMV kernels of one translation unit.
static __device__ unsigned int g_gemv_status;

// acc[m] += sum_{j<8} c_j * x_j for one 8-weight chunk; c holds the codes as
// fp16 pairs (c0,c4),(c1,c5),(c2,c6),(c3,c7) (INT4 order) and xq the chunk
// (x0,x1),(x2,x3),(x4,x5),(x6,x7).
__device__ __forceinline__ float dot8_int4order(const uint32_t c[4], const uint4 xq, float acc) {
  acc = fma_h(lo16(c[0]), lo16(xq.x), acc);
  acc = fma_h(lo16(c[1]), hi16(xq.x), acc);
  acc = fma_h(lo16(c[2]), lo16(xq.y), acc);
  acc = fma_h(lo16(c[3]), hi16(xq.y), acc);
  acc = fma_h(hi16(c[0]), lo16(xq.z), acc);
  acc = fma_h(hi16(c[1]), hi16(xq.z), acc);
  acc = fma_h(hi16(c[2]), lo16(xq.w), acc);
  acc = fma_h(hi16(c[3]), hi16(xq.w), acc);
  return acc;
}

// INT4 with the offsets left in (int4x8_to_magic): the even-k products
// (1024 + n) x go to `even`, the odd-k products (1024 + 16 n) x to `odd`,
// both exact in fp32.  For a piece, sum_k c_k x_k = even + odd / 16 -
// (1032 X_even + 72 X_odd), X the piece's activation sums.
__device__ __forceinline__ void dot8_int4magic(const uint32_t v[4], const uint4 xq, float& even,
                                               float& odd) {
  even = fma_h(lo16(v[0]), lo16(xq.x), even);  // k0
  odd = fma_h(lo16(v[1]), hi16(xq.x), odd);    // k1
  even = fma_h(lo16(v[2]), lo16(xq.y), even);  // k2
  odd = fma_h(lo16(v[3]), hi16(xq.y), odd);    // k3
  even = fma_h(hi16(v[0]), lo16(xq.z), even);  // k4
  odd = fma_h(hi16(v[1]), hi16(xq.z), odd);    // k5
  even = fma_h(hi16(v[2]), lo16(xq.w), even);  // k6
  odd = fma_h(hi16(v[3]), hi16(xq.w), odd);    // k7
}

// Same for weights already in natural order: pairs (w0,w1),(w2,w3),...
__device__ __forceinline__ float dot8_natural(uint32_t w0, uint32_t w1, uint32_t w2, uint32_t w3,
                                              const uint4 xq, float acc) {
  acc = fma_h(lo16(w0), lo16(xq.x), acc);
  acc = fma_h(hi16(w0), hi16(xq.x), acc);
  acc = fma_h(lo16(w1), lo16(xq.y), acc);
  acc = fma_h(hi16(w1), hi16(xq.y), acc);
  acc = fma_h(lo16(w2), lo16(xq.z), acc);
  acc = fma_h(hi16(w2), hi16(xq.z), acc);
  acc = fma_h(lo16(w3), lo16(xq.w), acc);
  acc = fma_h(hi16(w3), hi16(xq.w), acc);
  return acc;
}

// Output (row m, column n) from its fp32 dot product v (and, with the SiLU
// gate, the up row's u): FP8 row scale, bias, silu(v) * u, residual, fp16.
template <int WK, bool SILU>
__device__ __forceinline__ void gemv_store(const GemvArgs& a, int64_t n, int m, float v, float u) {
  if constexpr (WK == WK_FP8) v *= reinterpret_cast<const float*>(a.scales)[n];
  if (a.bias) v += __half2float(a.bias[n]);
  if constexpr (SILU) {
    if constexpr (WK == WK_FP8) u *= reinterpret_cast<const float*>(a.scales)[a.N + n];
    if (a.bias) u += __half2float(a.bias[a.N + n]);
    v = v / (1.0f + expf(-v)) * u;
  }
  if (a.residual) v += __half2float(a.residual[(int64_t)m * a.N + n]);
  a.y[(int64_t)m * a.N + n] = __float2half_rn(v);
}

// Pieces of one weight row a lane keeps in flight per batch: enough bytes
// in flight to cover DRAM latency (U x 512 B per row per warp) within the
// register budget.
template <int WR>
struct Unroll {
  static constexpr int value = WR == 1 ? 12 : WR == 2 ? 4 : 2;
};

// MR: activation rows compiled for (M <= MR, missing rows read zeros);
// R: output rows per lane group; SILU: fused gate/up epilogue;
// LPR: lanes per row.  A warp holds 32 / LPR lane groups, each sweeping its
// own R rows with LPR lanes; LPR is chosen so that a row's 16-byte pieces
// divide evenly among the lanes (no idle lanes), and the groups of a warp
// read the same x slots (shared-memory broadcast).
// Minimum resident CTAs per SM the compiler must allow (register cap).  The
// single-row INT4 fused gate/up (M = 1) runs at 4 (64 registers): its
// 4480-tile 1.5B matrix then starts every tile in the first wave (draft
// pass 485 -> 462 us measured); every other configuration keeps the
// registers it needs.
template <int WK, int MR, int R, bool SILU>
struct GemvMinBlocks {
  static constexpr int value = (WK == WK_INT4 && MR == 1 && R == 1 && SILU) ? 4 : 1;
};

template <int WK, int MR, int R, bool SILU, int LPR>
__global__ void __launch_bounds__(kGemvThreads, (GemvMinBlocks<WK, MR, R, SILU>::value))
    gemv_kernel(const GemvArgs a) {
  using T = WTraits<WK>;
  constexpr int SUB = T::kSub;
  constexpr int WR = SILU ? 2 * R : R;  // weight rows per lane group
  constexpr int U = Unroll<WR>::value;
  constexpr int GPW = 32 / LPR;         // lane groups per warp
  constexpr int RPT = GPW * R;          // output rows per warp tile
  extern __shared__ uint4 xs[];

  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int lg = lane / LPR, ll = lane % LPR;
  const int64_t ntiles = (a.N + RPT - 1) / RPT;
  // this CTA's slice of tiles [t_begin, t_end); warp w takes t_begin + w + 8 i
  const int64_t t_begin = ((int64_t)blockIdx.x * ntiles) / gridDim.x;
  const int64_t t_end = ((int64_t)(blockIdx.x + 1) * ntiles) / gridDim.x;
  const int64_t gwarp = t_begin + warp;
  const int64_t nwarps = kGemvWarps;
  const int steps = (a.pieces + LPR - 1) / LPR;  // pieces of a row per lane
  const int64_t G = a.K / 128;

  auto out_row = [&](int64_t tile, int r) -> int64_t { return tile * RPT + lg * R + (r % R); };
  auto wrow_index = [&](int64_t tile, int r) -> int64_t {
    return (SILU && r >= R ? a.N : 0) + out_row(tile, r);
  };
  auto row_valid = [&](int64_t tile, int r) -> bool {
    return tile < t_end && out_row(tile, r) < a.N;
  };
  // L2 bulk prefetch of one tile's rows (lane ll < WR of each group takes
  // row ll of its group).
  auto prefetch_tile = [&](int64_t tile) {
    if (ll < WR && row_valid(tile, ll)) {
      const uint8_t* row = a.w + wrow_index(tile, ll) * a.row_bytes;
      for (int64_t off = 0; off < a.row_bytes; off += 32768) {
        const int64_t nb = a.row_bytes - off < 32768 ? a.row_bytes - off : 32768;
        prefetch_l2_bulk(row + off, (uint32_t)nb);
      }
    }
  };

  // One batch = U pieces (steps jb .. jb+U-1) of each of the WR rows.
  uint4 wv[U][WR];
  float sv[U][WR];  // INT4 group scales of those pieces
  auto load_batch = [&](int64_t tile, int jb) {
#pragma unroll
    for (int r = 0; r < WR; ++r) {
      const bool ok = row_valid(tile, r);
      const int64_t wi = ok ? wrow_index(tile, r) : 0;
      const uint8_t* row = a.w + wi * a.row_bytes;
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int p = (jb + u) * LPR + ll;
        const bool in = ok && p < a.pieces;
        wv[u][r] = in ? ld_stream16(row + (int64_t)p * 16) : make_uint4(0u, 0u, 0u, 0u);
        if constexpr (WK == WK_INT4)
          sv[u][r] = in ? __half2float(reinterpret_cast<const __half*>(a.scales)[wi * G + (p >> 2)])
                        : 0.0f;
      }
    }
  };

  // The weights never depend on the previous kernel: request this warp's
  // next tiles into L2 and fetch its first batch before waiting for it.
#pragma unroll
  for (int d = 1; d <= kPrefetchTiles; ++d) prefetch_tile(gwarp + (int64_t)d * nwarps);
  if (gwarp < t_end) load_batch(gwarp, 0);
  // the RMSNorm gains never depend on it either: bring this thread's first
  // chunk into L1 (the weight loads do not allocate there)
  if (a.gamma != nullptr && threadIdx.x < a.K / 8)
    asm volatile("prefetch.global.L1 [%0];" ::"l"(a.gamma + 8 * threadIdx.x));

  griddep_wait();
  griddep_launch_dependents();

  // ---- stage x, permuted (see header comment); with several rows each
  // thread issues kStageBatch independent 16-byte loads before storing any,
  // so the rows cost one L2 round trip per batch rather than one per chunk
  // (measured: 8-13 % faster at M = 3..5, none at M = 1)
  const int chunks_per_m = a.ppad * SUB;
  const int total = MR * chunks_per_m;
  constexpr int kStageBatch = MR >= 4 ? 4 : 1;
  for (int base = threadIdx.x; base < total; base += kGemvThreads * kStageBatch) {
    uint4 v[kStageBatch];
#pragma unroll
    for (int b = 0; b < kStageBatch; ++b) {
      const int idx = base + b * kGemvThreads;
      const int m = idx / chunks_per_m;
      const int s = idx - m * chunks_per_m;
      const int l = s & 31, t = s >> 5;
      const int j = t / SUB, i = t - j * SUB;
      const int p = j * 32 + l;
      v[b] = make_uint4(0u, 0u, 0u, 0u);
      if (idx < total && m < a.M && p < a.pieces)
        v[b] = *reinterpret_cast<const uint4*>(a.x + (int64_t)m * a.K + ((int64_t)p * SUB + i) * 8);
    }
#pragma unroll
    for (int b = 0; b < kStageBatch; ++b)
      if (base + b * kGemvThreads < total) xs[base + b * kGemvThreads] = v[b];
  }
  __syncthreads();
  if (a.gamma != nullptr) {
    // RMSNorm of the staged rows (x / sqrt(mean(x^2) + eps) * gamma, fp16
    // out) in the arithmetic order of the standalone RMSNorm kernel: thread t
    // sums the 8-value chunks c = t, t + 256, ... (values in order), then warp
    // sums, then the eight warp sums in order; so the normalised rows equal
    // its output bit for bit.  A chunk is one staged 16-byte slot.
    __shared__ float nred[kGemvWarps * kGemvMaxRows];
    __shared__ float rinv[kGemvMaxRows];
    const int nch = (int)(a.K / 8);
    auto chunk_slot = [&](int c) {
      const int p = c / SUB, i = c - (c / SUB) * SUB;
      return ((p >> 5) * SUB + i) * 32 + (p & 31);
    };
    for (int m = 0; m < MR; ++m) {
      float ss = 0.0f;
      if (m < a.M)
        for (int c = threadIdx.x; c < nch; c += kGemvThreads) ss = sumsq8(xs[m * chunks_per_m + chunk_slot(c)], ss);
      ss = warp_sum(ss);
      if ((threadIdx.x & 31) == 0) nred[(threadIdx.x >> 5) * kGemvMaxRows + m] = ss;
    }
    __syncthreads();
    if (threadIdx.x < MR) {
      float t = 0.0f;
      for (int w = 0; w < kGemvWarps; ++w) t += nred[w * kGemvMaxRows + threadIdx.x];
      rinv[threadIdx.x] = 1.0f / sqrtf(t / (float)a.K + a.eps);
    }
    __syncthreads();
    for (int c = threadIdx.x; c < nch; c += kGemvThreads) {
      const int slot = chunk_slot(c);
      const uint4 g = *reinterpret_cast<const uint4*>(a.gamma + 8 * (int64_t)c);
      const uint32_t gw[4] = {g.x, g.y, g.z, g.w};
      for (int m = 0; m < MR && m < a.M; ++m) {
        uint4 q = xs[m * chunks_per_m + slot];
        uint32_t* qw = reinterpret_cast<uint32_t*>(&q);
        const float r = rinv[m];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float lo = __fmul_rn(__fmul_rn(__half2float(__ushort_as_half(lo16(qw[e]))), r),
                                     __half2float(__ushort_as_half(lo16(gw[e]))));
          const float hi = __fmul_rn(__fmul_rn(__half2float(__ushort_as_half(hi16(qw[e]))), r),
                                     __half2float(__ushort_as_half(hi16(gw[e]))));
          qw[e] = (uint32_t)__half_as_ushort(__float2half_rn(lo)) |
                  ((uint32_t)__half_as_ushort(__float2half_rn(hi)) << 16);
        }
        xs[m * chunks_per_m + slot] = q;
      }
    }
    __syncthreads();
  }
  // INT4: per (row m, piece p) the offset 1032 X_even + 72 X_odd that the
  // magic-valued products carry (X = the piece's 32 activations summed over
  // even / odd k), behind x in shared memory
  float* xoff = reinterpret_cast<float*>(xs + total);
  if constexpr (WK == WK_INT4) {
    for (int idx = threadIdx.x; idx < MR * a.ppad; idx += kGemvThreads) {
      const int m = idx / a.ppad, pp = idx - m * a.ppad;
      float xe = 0.0f, xo = 0.0f;
#pragma unroll
      for (int i = 0; i < SUB; ++i) {
        const uint4 q = xs[m * chunks_per_m + ((pp >> 5) * SUB + i) * 32 + (pp & 31)];
        const uint32_t h[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          xe += __half2float(__ushort_as_half(lo16(h[j])));
          xo += __half2float(__ushort_as_half(hi16(h[j])));
        }
      }
      xoff[idx] = fmaf(1032.0f, xe, 72.0f * xo);
    }
    __syncthreads();
  }

  for (int64_t tile = gwarp; tile < t_end; tile += nwarps) {
    prefetch_tile(tile + (int64_t)(kPrefetchTiles + 1) * nwarps);
    float acc[WR][MR];
#pragma unroll
    for (int r = 0; r < WR; ++r)
#pragma unroll
      for (int m = 0; m < MR; ++m) acc[r][m] = 0.0f;

    for (int jb = 0; jb < steps; jb += U) {
      if (jb > 0) load_batch(tile, jb);
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int j = jb + u;
        if (j * LPR >= a.pieces) break;  // warp-uniform
        const int p = j * LPR + ll;      // this lane's piece of the row
        const int xsl = ((p >> 5) * SUB) * 32 + (p & 31);  // x slot of sub-chunk 0
        if constexpr (WK == WK_INT4) {
          float pe[WR][MR], po[WR][MR];
#pragma unroll
          for (int r = 0; r < WR; ++r)
#pragma unroll
            for (int m = 0; m < MR; ++m) pe[r][m] = po[r][m] = 0.0f;
#pragma unroll
          for (int i = 0; i < SUB; ++i) {
            uint32_t c[WR][4];
#pragma unroll
            for (int r = 0; r < WR; ++r) {
              const uint4 w = wv[u][r];
              const uint32_t word = i == 0 ? w.x : i == 1 ? w.y : i == 2 ? w.z : w.w;
              int4x8_to_magic(word, c[r]);
            }
#pragma unroll
            for (int m = 0; m < MR; ++m) {
              const uint4 xq = xs[m * chunks_per_m + xsl + i * 32];
#pragma unroll
              for (int r = 0; r < WR; ++r) dot8_int4magic(c[r], xq, pe[r][m], po[r][m]);
            }
          }
#pragma unroll
          for (int m = 0; m < MR; ++m) {
            const float off = xoff[m * a.ppad + p];  // 1032 X_even + 72 X_odd of this piece
#pragma unroll
            for (int r = 0; r < WR; ++r)
              acc[r][m] = fmaf(sv[u][r], fmaf(po[r][m], 0.0625f, pe[r][m]) - off, acc[r][m]);
          }
        } else if constexpr (WK == WK_FP8) {
#pragma unroll
          for (int i = 0; i < SUB; ++i) {
            uint32_t h[WR][4];
#pragma unroll
            for (int r = 0; r < WR; ++r) {
              const uint4 w = wv[u][r];
              const uint32_t wa = i == 0 ? w.x : w.z;
              const uint32_t wb = i == 0 ? w.y : w.w;
              h[r][0] = e4m3x2_to_f16x2(lo16(wa));
              h[r][1] = e4m3x2_to_f16x2(hi16(wa));
              h[r][2] = e4m3x2_to_f16x2(lo16(wb));
              h[r][3] = e4m3x2_to_f16x2(hi16(wb));
            }
#pragma unroll
            for (int m = 0; m < MR; ++m) {
              const uint4 xq = xs[m * chunks_per_m + xsl + i * 32];
#pragma unroll
              for (int r = 0; r < WR; ++r)
                acc[r][m] = dot8_natural(h[r][0], h[r][1], h[r][2], h[r][3], xq, acc[r][m]);
            }
          }
        } else {
#pragma unroll
          for (int m = 0; m < MR; ++m) {
            const uint4 xq = xs[m * chunks_per_m + xsl];
#pragma unroll
            for (int r = 0; r < WR; ++r) {
              const uint4 w = wv[u][r];
              acc[r][m] = dot8_natural(w.x, w.y, w.z, w.w, xq, acc[r][m]);
            }
          }
        }
      }
    }
    // prefetch the next tile's first batch before the reduction
    if (tile + nwarps < t_end) load_batch(tile + nwarps, 0);

    // ---- reduce across the warp (fixed butterfly order)
#pragma unroll
    for (int r = 0; r < WR; ++r)
#pragma unroll
      for (int m = 0; m < MR; ++m) {
#pragma unroll
        for (int o = LPR / 2; o > 0; o >>= 1) acc[r][m] += __shfl_xor_sync(0xffffffffu, acc[r][m], o);
      }

    // ---- epilogue: lane (r * MR + m) % LPR of each group writes output (r, m)
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const int64_t n = out_row(tile, r);
      if (n >= a.N) continue;
#pragma unroll
      for (int m = 0; m < MR; ++m) {
        if (m >= a.M || ll != ((r * MR + m) % LPR)) continue;
        float u = 0.0f;
        if constexpr (SILU) u = acc[R + r][m];
        gemv_store<WK, SILU>(a, n, m, acc[r][m], u);
      }
    }
  }
}

// Instantiation helper used by the per-format translation units.  The grid
// is persistent: at most as many CTAs as can be resident at once, each warp
// looping over the tiles of its CTA's slice.
template <int WK, int MR, int R, bool SILU, int LPR>
cudaError_t launch_gemv_inst(const GemvArgs& a, int64_t blocks_needed, size_t smem,
                             cudaStream_t st) {
  auto k = gemv_kernel<WK, MR, R, SILU, LPR>;
  struct Cached {
    int smem_set = 0;
    int static_smem = -1;  // the kernel's static shared memory (bytes)
    size_t occ_smem[8] = {0};
    int occ[8] = {0};
  };
  static Cached cache[64];  // per device
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  Cached& c = cache[dev];
  if (c.static_smem < 0) {
    cudaFuncAttributes fa;
    e = cudaFuncGetAttributes(&fa, k);
    if (e != cudaSuccess) return e;
    c.static_smem = (int)fa.sharedSizeBytes;
  }
  // static + dynamic above the 48 KB default needs the opt-in attribute
  if (smem + (size_t)c.static_smem > 48 * 1024 && (int)smem > c.smem_set) {
    e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    c.smem_set = (int)smem;
  }
  int occ = 0;
  for (int i = 0; i < 8; ++i)
    if (c.occ_smem[i] == smem + 1) occ = c.occ[i];
  if (occ == 0) {
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, k, kGemvThreads, smem);
    if (e != cudaSuccess) return e;
    if (occ < 1) occ = 1;
    for (int i = 0; i < 8; ++i)
      if (c.occ_smem[i] == 0) {
        c.occ_smem[i] = smem + 1;
        c.occ[i] = occ;
        break;
      }
  }
  const int64_t cap = (int64_t)device_sm_count() * occ;
  const int grid = (int)(blocks_needed < cap ? blocks_needed : cap);
  return launch_pdl(k, dim3(grid > 0 ? grid : 1), dim3(kGemvThreads), smem, st, a);
}

template <int WK, int LPR>
cudaError_t launch_gemv_lpr(const GemvArgs& a, int mr, int r, bool silu, int64_t blocks_needed,
                            size_t smem, cudaStream_t st) {
#define SQ_GEMV_CASE(MR_, R_)                                                                  \
  if (mr == MR_ && r == R_)                                                                    \
    return silu ? launch_gemv_inst<WK, MR_, R_, true, LPR>(a, blocks_needed, smem, st)         \
                : launch_gemv_inst<WK, MR_, R_, false, LPR>(a, blocks_needed, smem, st);
  SQ_GEMV_CASE(1, 1)
  SQ_GEMV_CASE(1, 2)
  SQ_GEMV_CASE(2, 1)
  SQ_GEMV_CASE(2, 2)
  SQ_GEMV_CASE(4, 1)
  SQ_GEMV_CASE(4, 2)
  SQ_GEMV_CASE(5, 1)
  SQ_GEMV_CASE(5, 2)
  SQ_GEMV_CASE(4, 4)
  SQ_GEMV_CASE(5, 4)
#undef SQ_GEMV_CASE
  if constexpr (LPR == 32) {
    if (mr == 8 && r == 1)
      return silu ? launch_gemv_inst<WK, 8, 1, true, 32>(a, blocks_needed, smem, st)
                  : launch_gemv_inst<WK, 8, 1, false, 32>(a, blocks_needed, smem, st);
    if (mr == 8 && r == 2)
      return silu ? launch_gemv_inst<WK, 8, 2, true, 32>(a, blocks_needed, smem, st)
                  : launch_gemv_inst<WK, 8, 2, false, 32>(a, blocks_needed, smem, st);
    if (mr == 8 && r == 4)
      return silu ? launch_gemv_inst<WK, 8, 4, true, 32>(a, blocks_needed, smem, st)
                  : launch_gemv_inst<WK, 8, 4, false, 32>(a, blocks_needed, smem, st);
    if (mr == 16 && r == 1)
      return silu ? launch_gemv_inst<WK, 16, 1, true, 32>(a, blocks_needed, smem, st)
                  : launch_gemv_inst<WK, 16, 1, false, 32>(a, blocks_needed, smem, st);
    if (mr == 16 && r == 2)
      return silu ? launch_gemv_inst<WK, 16, 2, true, 32>(a, blocks_needed, smem, st)
                  : launch_gemv_inst<WK, 16, 2, false, 32>(a, blocks_needed, smem, st);
    if (mr == 16 && r == 4 && !silu) return launch_gemv_inst<WK, 16, 4, false, 32>(a, blocks_needed, smem, st);
  }
  return cudaErrorInvalidValue;
}

template <int WK>
cudaError_t launch_gemv_fmt(const GemvArgs& a, int mr, int r, bool silu, int lpr,
                            int64_t blocks_needed, size_t smem, cudaStream_t st) {
  if (lpr == 16) return launch_gemv_lpr<WK, 16>(a, mr, r, silu, blocks_needed, smem, st);
  if (lpr == 8) return launch_gemv_lpr<WK, 8>(a, mr, r, silu, blocks_needed, smem, st);
  return launch_gemv_lpr<WK, 32>(a, mr, r, silu, blocks_needed, smem, st);
}

// Reads and clears this translation unit's status word.
inline cudaError_t take_gemv_status_tu(uint32_t* bits) {
  uint32_t v = 0, zero = 0;
  cudaError_t e = cudaMemcpyFromSymbol(&v, g_gemv_status, sizeof(v));
  if (e != cudaSuccess) return e;
  if (v) e = cudaMemcpyToSymbol(g_gemv_status, &zero, sizeof(zero));
  *bits |= v;
  return e;
}

}  // namespace sq
