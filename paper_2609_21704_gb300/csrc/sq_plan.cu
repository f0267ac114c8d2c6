// sq_plan.cu -- how a linear call runs: device properties, the choice of
// engine (CUDA-core GEMV or tcgen05 tensor cores) and, for the GEMV, the
// activation-row chunking and the rows-per-group / lanes-per-row
// configuration.  Host code only; the kernels live in sq_gemv*.cu and
// sq_tc.cu, argument checking in sq_capi.cu.
#include <stdlib.h>

#include "sq_internal.h"

namespace sq {

int device_sm_count() {
  static int cache[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return kNumSMs;
  if (cache[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
      n = kNumSMs;
    cache[dev] = n;
  }
  return cache[dev];
}

bool pdl_enabled() {
  static const bool on = [] {
    const char* e = getenv("SQ_PDL");
    return !(e && e[0] == '0');
  }();
  return on;
}

int device_max_smem() {
  static int cache[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 227 * 1024;
  if (cache[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess ||
        n <= 0)
      n = 227 * 1024;
    cache[dev] = n;
  }
  return cache[dev];
}

// ---------------------------------------------------------------- GEMV plan

static int sub_of(int wk) { return wk == SQ_W_INT4 ? 4 : wk == SQ_W_FP8 ? 2 : 1; }
int64_t weights_per_piece(int wk) { return wk == SQ_W_INT4 ? 32 : wk == SQ_W_FP8 ? 16 : 8; }
int64_t row_bytes_of(int wk, int64_t K) {
  return wk == SQ_W_INT4 ? K / 2 : wk == SQ_W_FP8 ? K : 2 * K;
}

size_t gemv_smem_bytes(int wk, int mr, int64_t K) {
  const int64_t pieces = K / weights_per_piece(wk);
  const int64_t ppad = (pieces + 31) / 32 * 32;
  // staged x, plus one fp32 offset per (row, piece) for INT4
  return (size_t)mr * (size_t)ppad * ((size_t)sub_of(wk) * 16u + (wk == SQ_W_INT4 ? 4u : 0u));
}

// Compiled activation-row counts (sq_gemv.cuh instantiations).
static const int kMRs[] = {1, 2, 4, 5, 8, 16};

int gemv_pick_mr(int M) {
  for (int mr : kMRs)
    if (M <= mr) return mr;
  return 16;
}

// Largest compiled MR whose staged x fits in shared memory.
int gemv_cap_mr(int wk, int64_t K) {
  const size_t limit = (size_t)device_max_smem() - 1024;
  int best = 0;
  for (int mr : kMRs)
    if (gemv_smem_bytes(wk, mr, K) <= limit) best = mr;
  return best;
}

// Tensor cores or CUDA cores.  From 16 rows on a CUDA-core GEMV is issue
// bound (16 fused multiply-adds per weight); below that the choice follows
// timings of both paths on the 1.5B/7B/14B projection shapes:
//   * 8..15 rows: tensor cores for FP16 and FP8 weights (1.5-3x faster on
//     every shape), and for INT4 weights from 8 Mi weights on (the INT4
//     GEMV keeps small matrices, where its 8 x dequant reuse still pays);
//   * 3..7 rows, FP16 weights: tensor cores for long rows (K >= 8192), the
//     fused gate/up from 16 Mi weights, and wide outputs (N >= 65536) with
//     K >= 2048; the GEMV for the rest (its many warps fill the GPU better
//     than 128-row tiles do when N is small);
//   * fewer rows, or FP8/INT4 below 8 rows: the GEMV.
bool use_tensor_cores(int wk, int M, int64_t N, int64_t K, int epi) {
  const bool silu = epi == SQ_EPI_SILU_GATE;
  const int64_t weights = (silu ? 2 * N : N) * K;
  if (M >= 16) return true;
  if (M >= 8) return wk != SQ_W_INT4 || weights >= ((int64_t)8 << 20);
  if (wk == SQ_W_FP16 && M >= 3)
    return K >= 8192 || (silu && weights >= ((int64_t)16 << 20)) || (N >= 65536 && K >= 2048);
  return false;
}

cudaError_t launch_gemv(int wk, const GemvArgs& a0, cudaStream_t st) {
  // one INT4 row over many 16-row tiles: products on the tensor cores
  if (gemv_uses_mma(wk, a0.M, a0.N))
    return launch_gemv_mma_int4(a0, a0.epi == SQ_EPI_SILU_GATE, st);
  GemvArgs a = a0;
  const int cap = gemv_cap_mr(wk, a.K);
  if (cap == 0) return cudaErrorInvalidValue;
  // Rows of x are processed in chunks of at most `cap` (each chunk reads the
  // weights once); M <= 16 with K up to ~19k fits in one or two chunks.
  for (int m0 = 0; m0 < a0.M;) {
    const int rem = a0.M - m0;
    int mr = gemv_pick_mr(rem < cap ? rem : cap);
    if (mr > cap) {
      mr = 0;
      for (int c : kMRs)
        if (c <= cap) mr = c;
    }
    const int m_here = rem < mr ? rem : mr;
    a.M = m_here;
    a.x = a0.x + (int64_t)m0 * a0.K;
    a.y = a0.y + (int64_t)m0 * a0.N;
    a.residual = a0.residual ? a0.residual + (int64_t)m0 * a0.N : nullptr;
    const bool silu = a.epi == SQ_EPI_SILU_GATE;
    // rows per lane group and lanes per row, fitted to timings of every
    // projection shape of the 1.5B/7B/14B stacks (within 1 % of the best
    // of the nine (R, LPR) choices overall): two rows per group once there
    // are enough rows to keep every warp busy; SiLU already doubles the
    // rows a group holds
    int r = 1;
    if (mr <= 5) r = (a.N >= 4096 && !silu) ? 2 : 1;
    else r = (mr == 16 && silu) ? 1 : 2;
    // lanes per row: 32 for long rows (>= 256 pieces, several batches per
    // row anyway) and for MR >= 8 (compiled for 32 only); otherwise the
    // largest of 32/16/8 that divides the row's 16-byte pieces (no idle
    // lanes), unless that leaves too few tiles to spread over the warps
    int lpr = 32;
    if (mr <= 5 && a.pieces < 256) {
      for (int cand : {32, 16, 8}) {
        if (a.pieces % cand) continue;
        const int64_t per_tile = (int64_t)(32 / cand) * r;
        const int64_t tiles = (a.N + per_tile - 1) / per_tile;
        if (cand == 32 || tiles >= (int64_t)device_sm_count() * 4) lpr = cand;
        break;
      }
    }
    const int64_t rows_per_tile = (int64_t)(32 / lpr) * r;
    const int64_t ntiles = (a.N + rows_per_tile - 1) / rows_per_tile;
    const int64_t blocks = (ntiles + 7) / 8;
    const size_t smem = gemv_smem_bytes(wk, mr, a.K);
    cudaError_t e;
    if (wk == SQ_W_INT4) e = launch_gemv_int4(a, mr, r, silu, lpr, blocks, smem, st);
    else if (wk == SQ_W_FP8) e = launch_gemv_fp8(a, mr, r, silu, lpr, blocks, smem, st);
    else e = launch_gemv_fp16(a, mr, r, silu, lpr, blocks, smem, st);
    if (e != cudaSuccess) return e;
    m0 += m_here;
  }
  return cudaSuccess;
}

// The shared-memory ring engine (sq_ring.cu), one activation row, where it
// measured faster than the GEMV family (GB300, graphs of whole-stack launch
// sequences; us per launch, ring vs previous engine):
//   INT4 fused gate/up of >= 64 Mi weights (7B, 14B): 14B 19.5 vs 25.8;
//     the 1.5B one (27.5 Mi) stays on the register-operand path (6.9 vs 5.0);
//   FP16 fused gate/up of >= 16 Mi weights: 14B 49.5 vs 54.0, 1.5B 10.0 vs
//     11.3; FP16 lm_head (N >= 65536): 14B 228 vs 375, 1.5B 74.6 vs 79.5;
//   FP8 lm_head of >= 400 Mi weights: 14B 124 vs 164 (1.5B: 46.0 vs 41.1).
// q/k/v, o and down (96..448 tiles of 16 rows) stay on the GEMV family: at
// 2-3 tiles per SM the ring's whole-tile work split leaves SMs idle.
bool use_ring(int wkind, int M, int64_t N, int64_t K, int epi) {
  if (!ring_supported(wkind, M, K)) return false;
  // two to eight rows cost the products of one on the ring: INT4 and FP8
  // take it there, ahead of the tcgen05 tiles too (14B 8-layer passes, us:
  // INT4 at 4 rows 1197 -> 655, at 8 rows 1099 -> 880; FP8 at 4 rows
  // 1067 -> 872, at 8 rows 1271 -> 946); FP16 stays on the GEMV and the
  // tiles (ring 1228 -> 1264 at 4 rows, 1229 -> 1283 at 8)
  if (M > 1) return wkind != SQ_W_FP16;
  const bool silu = epi == SQ_EPI_SILU_GATE;
  const int64_t weights = (silu ? 2 * N : N) * K;
  const int64_t Mi = (int64_t)1 << 20;
  switch (wkind) {
    case SQ_W_INT4: return silu && weights >= 64 * Mi;
    case SQ_W_FP16: return (silu && weights >= 16 * Mi) || (!silu && N >= 65536);
    case SQ_W_FP8: return !silu && weights >= 400 * Mi;
  }
  return false;
}

}  // namespace sq
