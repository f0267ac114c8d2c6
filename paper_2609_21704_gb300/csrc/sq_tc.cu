// sq_tc.cu -- tensor-core (tcgen05 / TMEM) linear layer (skinny GEMM, M rows
// padded to a multiple of 16 on the MMA's N side).
//
// Sec. III-D.3: the verify pass scores B * (K+1) rows at once (the draft
// pass B rows).  sq_linear_ex sends a call here from 16 rows on, and from 3
// to 15 rows for the formats and shapes where this path measured faster
// than the CUDA-core GEMV (rows past M are zero-filled by the TMA load).  Swap-AB: the weight tile is the MMA's A
// operand (M_mma = 128 weight rows), the activations are B (N_mma = NB, the
// activation rows padded to a multiple of 16), D = 128 x NB fp32 in TMEM:
//     D[n, m] = sum_k W[n, k] * x[m, k]   ->   y[m, n]
// Both operands are K-major fp16 tiles of 64 k (128 bytes per row) loaded by
// 2-D TMA with 128-byte swizzle into a ring of shared-memory stages; warp 0
// lane 0 issues the TMA copies, warp 1 lane 0 issues tcgen05.mma (4 x K16
// per stage) and commits each stage back to the producer; warps 2..5 read
// the accumulator with tcgen05.ld (each warp its 32-lane TMEM sub-partition)
// and run the epilogue.  With the fused SiLU gate the CTA also loads the up
// rows' tile and accumulates a second NB-column block of TMEM.
//
// FP8 and INT4 weights: TMA brings the code tiles instead, and the four
// epilogue warps (idle until the accumulator is final) dequantise each stage
// into the swizzled fp16 A tile (generic stores, fence.proxy.async, then an
// mbarrier arrive that releases the stage to the MMA thread).  FP8: exact
// E4M3 -> fp16, the per-row scale applied in the epilogue (exact).  INT4:
// c * s rounded once to fp16 (c exact, s the fp16 group scale), a relative
// rounding of at most 2^-11 per weight, far inside the linear layers' 1e-3
// relative-L2 tolerance (the per-(row, group) scale cannot be factored out
// of an MMA that accumulates over several groups).
//
// Split-K: the S CTAs of a cluster take consecutive K ranges of the same
// weight tile; each writes its fp32 partial tile to its own shared memory,
// and after a cluster barrier CTA r sums its share of the 128 rows (about
// 128/S consecutive rows) over the S partials in rank order through
// distributed shared memory, so the result does not depend on timing.  Every mbarrier wait is bounded (a wait
// that gives up sets SQ_DEV_TIMEOUT and is skipped from then on), so every
// thread always reaches the cluster barriers.  After a wait gives up, the
// TMA producer requests nothing more and waits (bounded) for the copies it
// still has in flight, the MMA issuer issues nothing more, and the epilogue
// waits (bounded) on the commit that tracks every MMA issued before it
// reads TMEM and the allocation is released; the tile's results are then
// invalid and the status bit says so.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "sq_internal.h"

namespace sq {

static __device__ unsigned int g_tc_status;

constexpr int kTcBM = 128;      // weight rows per tile (MMA M)
constexpr int kTcBK = 64;       // k per stage: 64 fp16 = one 128-byte swizzle row
// Warp roles: warp 0 TMA, warp 1 MMA + TMEM, warps 2..5 epilogue (one TMEM
// sub-partition each).  Quantised weights add converter warps: warps 2..
// 2 + warps - 1 dequantise each stage (two per SM sub-partition, so that
// one's dependent chain hides behind the other's).
template <int WK>
struct TcConv {
  static constexpr int warps = WK == 0 ? 4 : 8;
  static constexpr int threads = 64 + 32 * warps;
};
constexpr int kTcStageA = kTcBM * kTcBK * 2;  // 16 KB
// CTAs per cluster along K: up to 16 (non-portable cluster size, allowed at
// launch); the INT4 search keeps to the portable 8 it was measured at.
constexpr int kTcMaxSplit = 16;
constexpr int kTcMaxSplitInt4 = 8;

// ---------------------------------------------------------------- PTX

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int c0, int c1,
                                            uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(smem_u32(bar))
      : "memory");
}

// Shared-memory matrix descriptor of a K-major tile with 128-byte swizzle:
// start address >> 4, leading byte offset 16 (unused by this layout), stride
// byte offset 1024 (one 8-row swizzle atom), descriptor version 1, swizzle
// mode 2 (128 B).
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)1 << 16;
  d |= (uint64_t)(1024 >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

__device__ __forceinline__ void tc_mma_f16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                           uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n"
      ".reg .pred p;\n"
      "setp.ne.u32 p, %4, 0;\n"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n"
      "}\n" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void tc_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// 16 consecutive fp32 columns of this thread's TMEM lane.
__device__ __forceinline__ void tc_ld16(uint32_t taddr, float v[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, "
      "%12, %13, %14, %15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;" ::
                   : "memory");
}
__device__ __forceinline__ float ld_dsmem_f32(const float* local, uint32_t rank) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(local)), "r"(rank));
  float v;
  asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(remote) : "memory");
  return v;
}
// Four consecutive floats (16-byte aligned) of CTA `rank`'s shared memory.
__device__ __forceinline__ float4 ld_dsmem_f32x4(const float* local, uint32_t rank) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(local)), "r"(rank));
  float4 v;
  asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(remote)
               : "memory");
  return v;
}

// ---------------------------------------------------------------- kernel

struct TcArgs {
  const void* scales;  // FP8: fp32 [rows]; INT4: fp16 [rows, K/128]; FP16: unused
  int M;            // activation rows present
  int NB;           // MMA N: M rounded up to 16
  int64_t N;        // output columns (weight rows, or gate rows with SILU)
  int64_t K;
  int epi;
  int ksteps;       // ceil(K / 64)
  int splits;       // CTAs per cluster along K
  int nstages;
  int tmem_cols;
  uint32_t idesc;
  int stage_bytes;  // A (+ A_up) + B, multiple of 1024
  int b_off;        // offset of B inside a stage
  int c_off;        // offset of the code tiles inside a stage (FP8 / INT4)
  int c_bytes;      // bytes of one code tile
  int part_stride;  // floats between columns of the partial tile
  int sc_off;       // INT4: byte offset of the CTA's group-scale block
  int sc_ng;        // INT4: groups per row held in the block (>= any CTA's need)
  int max_split;    // largest split-K factor whose partial tile fits in the stages
  int two_per_sm;   // stages sized so that two CTAs share an SM
  int int4_large;   // INT4 weights of 20 MB and more at few rows: power-of-two split rule
  const __half* bias;
  const __half* residual;
  __half* y;
};

// WK: 0 fp16 weights, 1 INT4 codes, 2 FP8 codes (the GEMV family's numbering).
template <int WK, bool SILU>
__global__ void __launch_bounds__(TcConv<WK>::threads, 1)
    tc_linear_kernel(const __grid_constant__ CUtensorMap tw, const __grid_constant__ CUtensorMap tx,
                     const TcArgs a) {
  constexpr bool QUANT = WK != 0;
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte alignment for the swizzle atoms
  const uint32_t raw = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + (((raw + 1023u) & ~1023u) - raw);
  // a ring of stages [A (gate, up) | B | codes (gate, up; quantised only)]:
  // TMA brings B and either the fp16 A tiles or the code tiles, which the
  // converter warps dequantise into the stage's A tiles
  uint8_t* stages = smem;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + (size_t)a.nstages * a.stage_bytes);
  uint64_t* full = bars;                       // stage landed (TMA)
  uint64_t* empty = bars + a.nstages;          // stage free again (MMA commit)
  uint64_t* accf = bars + 2 * a.nstages;       // accumulator final
  uint64_t* conv = bars + 2 * a.nstages + 1;   // A tiles converted (quantised)
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 3 * a.nstages + 1);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int S = a.splits;
  const uint32_t rank = S > 1 ? cluster_rank() : 0u;
  const int64_t tile = blockIdx.y;
  const int k_begin = (int)(((int64_t)rank * a.ksteps) / S);
  const int k_end = (int)(((int64_t)(rank + 1) * a.ksteps) / S);
  const int nk = k_end - k_begin;

  if (tid == 0) {
    for (int s = 0; s < a.nstages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
      mbar_init(&conv[s], TcConv<WK>::warps);
    }
    mbar_init(accf, 1);
    fence_mbar_init();
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_slot)),
                 "r"(a.tmem_cols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  griddep_launch_dependents();

  bool timed_out = false;
  if (warp == 0) {
    if (lane == 0) {
      // --------------------------------------------------------- producer
      const uint32_t bytes =
          (uint32_t)((QUANT ? a.c_bytes : kTcStageA) * (SILU ? 2 : 1) + a.NB * 128);
      // weight tiles land in A (fp16) or in the stage's code area (quantised)
      const int wdst = QUANT ? a.c_off : 0;
      const int wdst_up = QUANT ? a.c_off + a.c_bytes : kTcStageA;
      // TMA x coordinate of a weight tile: k (fp16, FP8 bytes) or k / 2 (INT4 bytes)
      auto wx = [&](int k0) { return WK == 1 ? k0 / 2 : k0; };
      const int pre = nk < a.nstages ? nk : a.nstages;
      // weights never depend on the previous kernel: start them first
      for (int it = 0; it < pre; ++it) {
        uint8_t* st = stages + (size_t)it * a.stage_bytes;
        const int k0 = (k_begin + it) * kTcBK;
        mbar_arrive_expect_tx(&full[it], bytes);
        tma_load_2d(st + wdst, &tw, wx(k0), (int)(tile * kTcBM), &full[it]);
        if (SILU) tma_load_2d(st + wdst_up, &tw, wx(k0), (int)(a.N + tile * kTcBM), &full[it]);
      }
      griddep_wait();
      for (int it = 0; it < pre; ++it)
        tma_load_2d(stages + (size_t)it * a.stage_bytes + a.b_off, &tx, (k_begin + it) * kTcBK, 0,
                    &full[it]);
      int issued = pre;  // iterations whose copies were requested
      for (int it = pre; it < nk; ++it) {
        const int s = it % a.nstages;
        const uint32_t ph = (uint32_t)(it / a.nstages) & 1u;
        if (!mbar_wait_bounded(&empty[s], ph ^ 1u)) {
          // the stage was never released: request nothing more
          timed_out = true;
          atomicOr(&g_tc_status, SQ_DEV_TIMEOUT);
          break;
        }
        uint8_t* st = stages + (size_t)s * a.stage_bytes;
        const int k0 = (k_begin + it) * kTcBK;
        mbar_arrive_expect_tx(&full[s], bytes);
        tma_load_2d(st + wdst, &tw, wx(k0), (int)(tile * kTcBM), &full[s]);
        if (SILU) tma_load_2d(st + wdst_up, &tw, wx(k0), (int)(a.N + tile * kTcBM), &full[s]);
        tma_load_2d(st + a.b_off, &tx, k0, 0, &full[s]);
        issued = it + 1;
      }
      if (timed_out) {
        // each stage has at most one request outstanding (its last): wait for
        // it (bounded) so that no copy lands after the CTA has left
        for (int s = 0; s < a.nstages && s < issued; ++s) {
          const int last = s + ((issued - 1 - s) / a.nstages) * a.nstages;
          mbar_wait_bounded(&full[s], (uint32_t)(last / a.nstages) & 1u, 1u << 20);
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // --------------------------------------------------------- MMA issuer
      for (int it = 0; it < nk; ++it) {
        const int s = it % a.nstages;
        const uint32_t ph = (uint32_t)(it / a.nstages) & 1u;
        if (!mbar_wait_bounded(QUANT ? &conv[s] : &full[s], ph)) {
          // the stage never arrived: issue no MMA on it or after it (the
          // commit below still tracks every MMA issued so far)
          timed_out = true;
          atomicOr(&g_tc_status, SQ_DEV_TIMEOUT);
          break;
        }
        tc_fence_after();
        const uint32_t st = smem_u32(stages + (size_t)s * a.stage_bytes);
        const uint64_t ad = sw128_desc(st);
        const uint64_t au = sw128_desc(st + kTcStageA);
        const uint64_t bd = sw128_desc(st + a.b_off);
#pragma unroll
        for (int kk = 0; kk < kTcBK / 16; ++kk) {
          const uint32_t acc = (it > 0 || kk > 0) ? 1u : 0u;
          // advancing 16 fp16 along K inside the swizzled row = +32 bytes
          tc_mma_f16(tmem, ad + 2 * kk, bd + 2 * kk, a.idesc, acc);
          if (SILU) tc_mma_f16(tmem + a.NB, au + 2 * kk, bd + 2 * kk, a.idesc, acc);
        }
        tc_commit(&empty[s]);
      }
      tc_commit(accf);
    }
  } else {
    // ------------------------------------- converters (quantised), epilogue
    if constexpr (QUANT) {
      if constexpr (WK == 1) {
        // INT4: this CTA's group scales (128 rows x the groups its K range
        // touches, gate and up) into shared memory once, before waiting on
        // the previous kernel: scales never depend on it, and the per-stage
        // conversion then never waits on a global load
        const int ct = tid - 64;
        const int64_t G = a.K / 128;
        const int64_t wrows = SILU ? 2 * a.N : a.N;
        const int g_lo = (k_begin * kTcBK) >> 7;
        const int ng = nk > 0 ? (((k_end * kTcBK) - 1) >> 7) + 1 - g_lo : 0;
        __half* sblk = reinterpret_cast<__half*>(smem + a.sc_off);
        for (int r = ct; r < (SILU ? 2 : 1) * kTcBM; r += 32 * TcConv<WK>::warps) {
          const int h = r / kTcBM, rr = r - h * kTcBM;
          const int64_t wrow = (h ? a.N : 0) + tile * kTcBM + rr;
          const __half* src = reinterpret_cast<const __half*>(a.scales) + wrow * G + g_lo;
          __half* dst = sblk + (size_t)r * a.sc_ng;
          for (int gi = 0; gi < ng; ++gi) dst[gi] = wrow < wrows ? __ldg(src + gi) : __ushort_as_half(0);
        }
        named_bar_sync(1, 32 * TcConv<WK>::warps);  // the converter warps
      }
    }
    griddep_wait();
    if constexpr (QUANT) {
      const int ct = tid - 64;  // 0 .. 32 * converter warps - 1
      const int g_lo = (k_begin * kTcBK) >> 7;
      const __half* sblk = reinterpret_cast<const __half*>(smem + a.sc_off);
      for (int it = 0; it < nk; ++it) {
        const int s = it % a.nstages;
        const uint32_t ph = (uint32_t)(it / a.nstages) & 1u;
        const int gi = (((k_begin + it) * kTcBK) >> 7) - g_lo;  // this stage's group
        if (!timed_out && !mbar_wait_bounded(&full[s], ph)) {
          timed_out = true;
          if (lane == 0) atomicOr(&g_tc_status, SQ_DEV_TIMEOUT);
        }
        uint8_t* st = stages + (size_t)s * a.stage_bytes;
#pragma unroll
        for (int h = 0; h < (SILU ? 2 : 1); ++h) {
          const uint8_t* codes = st + a.c_off + h * a.c_bytes;
          uint8_t* at = st + h * kTcStageA;
          // one job = 16 code bytes of one row: 32 INT4 / 16 FP8 weights,
          // i.e. 4 / 2 of the row's eight 16-byte fp16 chunks.  Per warp the
          // code loads cover 512 contiguous bytes and each quarter-warp's
          // chunk stores hit 8 distinct 16-byte bank groups (swizzle), so
          // neither conflicts.
          constexpr int kJobsPerRow = WK == 1 ? 2 : 4;
          constexpr int kChunksPerJob = 8 / kJobsPerRow;
#pragma unroll
          for (int job = ct; job < kTcBM * kJobsPerRow; job += 32 * TcConv<WK>::warps) {
            const int row = job / kJobsPerRow, jp = job % kJobsPerRow;
            const uint4 cw = *reinterpret_cast<const uint4*>(codes + row * (kTcBK * (WK == 1 ? 1 : 2) / 2) +
                                                             jp * 16);
            uint8_t* arow = at + row * 128;
            if constexpr (WK == 2) {
              const uint32_t wv[4] = {cw.x, cw.y, cw.z, cw.w};
#pragma unroll
              for (int q = 0; q < 2; ++q) {
                uint4 out;
                out.x = e4m3x2_to_f16x2(lo16(wv[2 * q]));
                out.y = e4m3x2_to_f16x2(hi16(wv[2 * q]));
                out.z = e4m3x2_to_f16x2(lo16(wv[2 * q + 1]));
                out.w = e4m3x2_to_f16x2(hi16(wv[2 * q + 1]));
                const int c = jp * kChunksPerJob + q;
                *reinterpret_cast<uint4*>(arow + ((c ^ (row & 7)) << 4)) = out;
              }
            } else {
              const __half2 s2 = __half2half2(sblk[(size_t)(h * kTcBM + row) * a.sc_ng + gi]);
              auto mul = [&](uint32_t v) {
                const __half2 r = __hmul2(*reinterpret_cast<const __half2*>(&v), s2);
                return *reinterpret_cast<const uint32_t*>(&r);
              };
              const uint32_t wv[4] = {cw.x, cw.y, cw.z, cw.w};
#pragma unroll
              for (int q = 0; q < 4; ++q) {
                uint32_t v[4];
                int4x8_to_f16x2(wv[q], v);  // (k0,k4),(k1,k5),(k2,k6),(k3,k7)
                uint4 out;
                out.x = mul(__byte_perm(v[0], v[1], 0x5410));  // (k0, k1)
                out.y = mul(__byte_perm(v[2], v[3], 0x5410));  // (k2, k3)
                out.z = mul(__byte_perm(v[0], v[1], 0x7632));  // (k4, k5)
                out.w = mul(__byte_perm(v[2], v[3], 0x7632));  // (k6, k7)
                const int c = jp * kChunksPerJob + q;
                *reinterpret_cast<uint4*>(arow + ((c ^ (row & 7)) << 4)) = out;
              }
            }
          }
        }
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncwarp();
        if (lane == 0) mbar_arrive(&conv[s]);
      }
    }
  }
  if (warp >= 2 && warp < 6) {
    // --------------------------------------------------------- epilogue
    if (!mbar_wait_bounded(accf, 0u)) {
      timed_out = true;
      if (lane == 0) atomicOr(&g_tc_status, SQ_DEV_TIMEOUT);
    }
    tc_fence_after();
    const int q = warp & 3;  // TMEM sub-partition this warp may read
    const int row = q * 32 + lane;
    const uint32_t taddr = tmem + ((uint32_t)(q * 32) << 16);
    const int64_t n = tile * kTcBM + row;
    if (S == 1) {
      for (int c0 = 0; c0 < a.NB; c0 += 16) {
        float g[16], u[16];
        tc_ld16(taddr + (uint32_t)c0, g);
        if (SILU) tc_ld16(taddr + (uint32_t)(a.NB + c0), u);
        if (n < a.N) {
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const int m = c0 + j;
            if (m >= a.M) break;
            float v = g[j];
            if constexpr (WK == 2) v *= reinterpret_cast<const float*>(a.scales)[n];
            if (a.bias) v += __half2float(a.bias[n]);
            if (SILU) {
              float uu = u[j];
              if constexpr (WK == 2) uu *= reinterpret_cast<const float*>(a.scales)[a.N + n];
              if (a.bias) uu += __half2float(a.bias[a.N + n]);
              v = v / (1.0f + expf(-v)) * uu;
            }
            if (a.residual) v += __half2float(a.residual[(int64_t)m * a.N + n]);
            a.y[(int64_t)m * a.N + n] = __float2half_rn(v);
          }
        }
      }
    } else {
      // partial tile -> this CTA's shared memory, [column][row] (stages are
      // free: every MMA has completed)
      float* part = reinterpret_cast<float*>(stages);
      const int cols = a.NB * (SILU ? 2 : 1);
      for (int c0 = 0; c0 < cols; c0 += 16) {
        float v[16];
        tc_ld16(taddr + (uint32_t)c0, v);
#pragma unroll
        for (int j = 0; j < 16; ++j) part[(size_t)(c0 + j) * a.part_stride + row] = v[j];
      }
    }
  }

  tc_fence_before();
  if (S > 1) {
    cluster_sync();  // every partial tile is written
    if (warp >= 2) {
      const int et = tid - 64;  // 0 .. blockDim.x - 65
      // this rank's rows [r0, r0 + nr).  Small splits over many columns:
      // four consecutive rows per 16-byte load of each partial and four such
      // items in flight per thread, the shares rounded up to four rows so
      // that every rank starts on a 16-byte boundary (14B FP16 at 144 rows,
      // S = 2-3: qkv 42 -> 30 us, down 65 -> 53 us; the element loop there
      // waited one cluster-load latency per element).  Otherwise one element
      // per thread, with all S loads of an element in flight, and shares as
      // even as possible (7B FP16 at 48 rows, S = 7-10: the four-row form,
      // which waits one latency per rank, measured 1123 us against 1045 us
      // per pass; INT4 at 16 rows, S = 8).  The decision depends only on S,
      // M and the block, so every rank takes the same.  The partials are
      // added in rank order either way.
      const int nthr = (int)blockDim.x - 64;
      const int rows1 = (kTcBM + S - 1) / S;
      const int rows4 = (rows1 + 3) & ~3;
      const bool vec = S <= 4 && (rows4 >> 2) * a.M >= nthr;
      const int rows = vec ? rows4 : rows1;
      const int r0 = (int)rank * rows;
      const int nr = max(0, min(rows, kTcBM - r0));
      const float* part = reinterpret_cast<const float*>(stages);
      // output (column m, row) from the summed partials g (and u, the up row's)
      auto emit = [&](int m, int row, float g, float u) {
        const int64_t n = tile * kTcBM + row;
        if (n >= a.N) return;
        float v = g;
        if constexpr (WK == 2) v *= reinterpret_cast<const float*>(a.scales)[n];
        if (a.bias) v += __half2float(a.bias[n]);
        if (SILU) {
          if constexpr (WK == 2) u *= reinterpret_cast<const float*>(a.scales)[a.N + n];
          if (a.bias) u += __half2float(a.bias[a.N + n]);
          v = v / (1.0f + expf(-v)) * u;
        }
        if (a.residual) v += __half2float(a.residual[(int64_t)m * a.N + n]);
        a.y[(int64_t)m * a.N + n] = __float2half_rn(v);
      };
      if (vec) {
        constexpr int kIt = 4;
        const int nq = nr >> 2;
        const int items = nq * a.M;
        for (int i0 = et; i0 < items; i0 += kIt * nthr) {
          float4 g[kIt], u[kIt];
#pragma unroll
          for (int j = 0; j < kIt; ++j) g[j] = u[j] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
          for (int qq = 0; qq < S; ++qq) {
#pragma unroll
            for (int j = 0; j < kIt; ++j) {
              const int i = i0 + j * nthr;
              if (i < items) {
                const int m = i / nq, r = r0 + 4 * (i - m * nq);
                const float4 v = ld_dsmem_f32x4(part + (size_t)m * a.part_stride + r, (uint32_t)qq);
                g[j].x += v.x;
                g[j].y += v.y;
                g[j].z += v.z;
                g[j].w += v.w;
                if (SILU) {
                  const float4 w = ld_dsmem_f32x4(part + (size_t)(a.NB + m) * a.part_stride + r, (uint32_t)qq);
                  u[j].x += w.x;
                  u[j].y += w.y;
                  u[j].z += w.z;
                  u[j].w += w.w;
                }
              }
            }
          }
#pragma unroll
          for (int j = 0; j < kIt; ++j) {
            const int i = i0 + j * nthr;
            if (i < items) {
              const int m = i / nq, r = r0 + 4 * (i - m * nq);
              emit(m, r, g[j].x, u[j].x);
              emit(m, r + 1, g[j].y, u[j].y);
              emit(m, r + 2, g[j].z, u[j].z);
              emit(m, r + 3, g[j].w, u[j].w);
            }
          }
        }
      } else {
        for (int idx = et; idx < nr * a.M; idx += nthr) {
          const int m = idx / nr, row = r0 + (idx - m * nr);
          float g = 0.0f, u = 0.0f;
          for (int qq = 0; qq < S; ++qq) {
            g += ld_dsmem_f32(part + (size_t)m * a.part_stride + row, (uint32_t)qq);
            if (SILU) u += ld_dsmem_f32(part + (size_t)(a.NB + m) * a.part_stride + row, (uint32_t)qq);
          }
          emit(m, row, g, u);
        }
      }
    }
    cluster_sync();  // no CTA leaves while another still reads its partial
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                 "r"(a.tmem_cols)
                 : "memory");
  }
}

// ---------------------------------------------------------------- host side

static PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// [rows, inner] row-major -> 2-D tensor map with box (box_inner, box_rows);
// zero fill outside the tensor.
static bool make_map(CUtensorMap* m, const void* base, CUtensorMapDataType dt, int elem_bytes,
                     int64_t rows, int64_t inner, int box_inner, int box_rows,
                     CUtensorMapSwizzle swz) {
  auto enc = tensor_map_encoder();
  if (!enc) return false;
  cuuint64_t dims[2] = {(cuuint64_t)inner, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)inner * (cuuint64_t)elem_bytes};
  cuuint32_t box[2] = {(cuuint32_t)box_inner, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  return enc(m, dt, 2, const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
             swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// instruction descriptor, kind::f16: D fp32, A and B fp16, both K-major,
// N = nb, M = 128
static uint32_t make_idesc(int nb) {
  uint32_t d = 0;
  d |= 1u << 4;                       // D format fp32
  d |= (uint32_t)(nb >> 3) << 17;     // N / 8
  d |= (uint32_t)(kTcBM >> 4) << 24;  // M / 16
  return d;
}

bool tc_supported(int M, int64_t K, int epi) {
  (void)epi;
  return M >= 1 && M <= 256 && K % 8 == 0 && tensor_map_encoder() != nullptr;
}

// Raises the kernel's dynamic shared-memory limit to `smem` (once per size
// and device) and allows cluster sizes above 8.
template <int WK, bool SILU>
static cudaError_t tc_prepare(size_t smem) {
  auto k = tc_linear_kernel<WK, SILU>;
  static int smem_set[64] = {0};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if ((int)smem > smem_set[dev]) {
    e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(k, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
    smem_set[dev] = (int)smem;
  }
  return cudaSuccess;
}

// Clusters of S CTAs (with `smem` bytes each) that can be resident at once,
// from the occupancy calculator; cached per device, S and size.
template <int WK, bool SILU>
static int tc_max_clusters(int S, size_t smem) {
  struct Entry {
    size_t smem;
    int n;
  };
  static Entry cache[64][kTcMaxSplit + 1][4] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64 || S < 1 || S > kTcMaxSplit) return 0;
  for (Entry& en : cache[dev][S])
    if (en.smem == smem + 1) return en.n;
  if (tc_prepare<WK, SILU>(smem) != cudaSuccess) return 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)S, 1, 1);
  cfg.blockDim = dim3(TcConv<WK>::threads);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)S;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, tc_linear_kernel<WK, SILU>, &cfg) != cudaSuccess) {
    (void)cudaGetLastError();
    n = 0;
  }
  for (Entry& en : cache[dev][S])
    if (en.smem == 0) {
      en.smem = smem + 1;
      en.n = n;
      break;
    }
  return n;
}

// Split-K factor.  FP16 and FP8 weights (HBM-bound): double S while the
// split tiles still fill at most half the SMs, so that the next kernel's
// CTAs find free SMs and start their weight loads early (programmatic
// dependent launch) -- filling every SM measured slower on the 7B shapes.
// INT4 weights (bound by the in-CTA dequantisation): the S in
// 1..kTcMaxSplit that minimises (waves of resident clusters) x (k-steps per
// CTA + 2 for the split reduction), at least 2 k-steps per CTA; ties keep
// the smaller S.
template <int WK, bool SILU>
static int tc_pick_split(int64_t tiles, int ksteps, size_t smem, int max_split, bool two_per_sm,
                         bool int4_large = false, bool many_rows = false) {
  if (WK == 1 && int4_large) {
    // two CTAs per SM: the largest power-of-two split with at most 2.2 CTAs
    // per SM in all and at least 12 k-steps per CTA (odd splits of 3 and 7
    // measured 20-50 % slower than their neighbours)
    const int sms = device_sm_count();
    int S = 1;
    for (int s = 2; s <= max_split && s <= kTcMaxSplitInt4; s <<= 1)
      if (tiles * s * 10 <= 22 * (int64_t)sms && ksteps >= 12 * s) S = s;
    return S;
  }
  if (WK != 1) {
    const int sms = device_sm_count();
    int S = 1;
    if (two_per_sm) {
      // two CTAs per SM: the largest S (up to 16, a cluster on 8 SMs) that
      // still fits one wave (1.5B down projection, M = 5: 10.4 -> 8.7 us
      // from S = 8 to 16)
      while (S < max_split && tiles * (S + 1) <= 2 * sms && ksteps >= 4 * (S + 1)) ++S;
      return S;
    }
    // one CTA per SM: clusters of at most the portable 8 SMs
    if (many_rows) {
      // many activation rows (NB > 64: every k-step also streams a large
      // activation tile and runs a long MMA): the largest S that still fits
      // one wave
      while (S + 1 <= max_split && S + 1 <= 8 && tiles * (S + 1) <= sms && ksteps >= 4 * (S + 1)) ++S;
      return S;
    }
    while (2 * S <= max_split && 2 * S <= 8 && tiles * S * 2 <= sms && ksteps >= 4 * S * 2) S <<= 1;
    return S;
  }
  int best_s = 1;
  int64_t best = INT64_MAX;
  for (int S = 1; S <= max_split && S <= kTcMaxSplitInt4 && ksteps >= 2 * S; ++S) {
    const int nc = tc_max_clusters<WK, SILU>(S, smem);
    if (nc <= 0) continue;
    const int64_t waves = (tiles + nc - 1) / nc;
    const int64_t cost = waves * ((ksteps + S - 1) / S + (S > 1 ? 2 : 0));
    if (cost < best) {
      best = cost;
      best_s = S;
    }
  }
  return best_s;
}

template <int WK, bool SILU>
static cudaError_t tc_launch_inst(const CUtensorMap& tw, const CUtensorMap& tx, TcArgs a,
                                  int64_t tiles, size_t smem, cudaStream_t st) {
  auto k = tc_linear_kernel<WK, SILU>;
  cudaError_t e = tc_prepare<WK, SILU>(smem);
  if (e != cudaSuccess) return e;
  const int S = tc_pick_split<WK, SILU>(tiles, a.ksteps, smem, a.max_split, a.two_per_sm != 0,
                                       a.int4_large != 0, a.NB > 64);
  a.splits = S;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)S, (unsigned)tiles, 1);
  cfg.blockDim = dim3(TcConv<WK>::threads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  int na = 0;
  attr[na].id = cudaLaunchAttributeClusterDimension;
  attr[na].val.clusterDim.x = (unsigned)S;
  attr[na].val.clusterDim.y = 1;
  attr[na].val.clusterDim.z = 1;
  ++na;
  const bool legacy = (st == nullptr || st == cudaStreamLegacy || st == cudaStreamPerThread);
  if (!legacy && pdl_enabled()) {
    attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[na].val.programmaticStreamSerializationAllowed = 1;
    ++na;
  }
  cfg.attrs = attr;
  cfg.numAttrs = na;
  return cudaLaunchKernelEx(&cfg, k, tw, tx, a);
}

cudaError_t launch_tc(int wk, const __half* x, const void* w, const void* scales, const __half* bias,
                      const __half* residual, __half* y, int M, int64_t N, int64_t K, int epi,
                      cudaStream_t st) {
  const bool silu = epi == SQ_EPI_SILU_GATE;
  const int nb = (M + 15) / 16 * 16;
  const int64_t wrows = silu ? 2 * N : N;
  CUtensorMap tw, tx;
  bool ok;
  int c_bytes = 0;
  if (wk == SQ_W_FP16) {
    ok = make_map(&tw, w, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, wrows, K, kTcBK, kTcBM,
                  CU_TENSOR_MAP_SWIZZLE_128B);
  } else if (wk == SQ_W_FP8) {
    c_bytes = kTcBM * kTcBK;  // 64 codes per row
    ok = make_map(&tw, w, CU_TENSOR_MAP_DATA_TYPE_UINT8, 1, wrows, K, kTcBK, kTcBM,
                  CU_TENSOR_MAP_SWIZZLE_NONE);
  } else {
    c_bytes = kTcBM * kTcBK / 2;  // 64 nibbles = 32 bytes per row
    ok = make_map(&tw, w, CU_TENSOR_MAP_DATA_TYPE_UINT8, 1, wrows, K / 2, kTcBK / 2, kTcBM,
                  CU_TENSOR_MAP_SWIZZLE_NONE);
  }
  ok = ok && make_map(&tx, x, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, M, K, kTcBK, nb,
                      CU_TENSOR_MAP_SWIZZLE_128B);
  if (!ok) return cudaErrorInvalidValue;
  TcArgs a = {};
  a.scales = scales;
  a.M = M;
  a.NB = nb;
  a.N = N;
  a.K = K;
  a.epi = epi;
  a.ksteps = (int)((K + kTcBK - 1) / kTcBK);
  a.bias = bias;
  a.residual = residual;
  a.y = y;
  a.idesc = make_idesc(nb);
  const int S2 = silu ? 2 : 1;
  const int cols = nb * S2;
  int tc = 32;
  while (tc < cols) tc <<= 1;
  a.tmem_cols = tc;
  const int a_bytes = kTcStageA * S2;
  const int b_bytes = (nb * 128 + 1023) / 1024 * 1024;
  a.b_off = a_bytes;
  a.c_off = a_bytes + b_bytes;
  a.c_bytes = c_bytes;
  a.stage_bytes = a.c_off + (c_bytes * S2 + 1023) / 1024 * 1024;
  // the split of K over a cluster is chosen per kernel instance (occupancy)
  const int64_t tiles = (N + kTcBM - 1) / kTcBM;
  a.part_stride = kTcBM + 4;
  const size_t part_bytes = (size_t)cols * a.part_stride * 4;
  // INT4: room for a CTA's group scales, sized for an unsplit K range
  // (a range of n stages touches at most (n - 1) / 2 + 2 groups)
  a.sc_ng = 0;
  size_t sc_bytes = 0;
  if (wk == SQ_W_INT4) {
    const int64_t G = K / 128;
    const int64_t need = (a.ksteps - 1) / 2 + 2;
    a.sc_ng = (int)(need < G ? need : G);
    sc_bytes = (size_t)S2 * kTcBM * (size_t)a.sc_ng * 2;
  }
  // Few activation rows (NB <= 64) and few row tiles: stages for two CTAs
  // per SM (100 KB each) and a deeper split, so every SM streams and one
  // CTA's prologue and epilogue overlap the other's loads (measured 8-28 %
  // faster on the 1.5B/7B down, qkv and o shapes); otherwise one CTA per SM
  // with 200 KB of stages.
  // INT4 weights of 20 MB and more at NB <= 64 (the draft pass at 8 or 16
  // rows: 7B/14B gate/up, down and lm_head) take two CTAs per SM too, with a
  // power-of-two split: measured 20-40 % faster than one CTA per SM with the
  // occupancy cost model (14B lm_head at M = 16: 332 -> 203 us; gate/up 57
  // -> 45 us; down 45 -> 36 us).
  const int sms = device_sm_count();
  const double wbytes = (double)wrows * (double)(K / 2) + (double)wrows * (double)(K / 128) * 2.0;
  a.int4_large = (wk == SQ_W_INT4 && nb <= 64 && wbytes >= 20e6) ? 1 : 0;
  a.two_per_sm = (a.int4_large || (nb <= 64 && tiles * 2 <= sms)) ? 1 : 0;
  const int budget = (a.two_per_sm ? 100 : 200) * 1024;
  int ns = (int)((budget - (int64_t)sc_bytes) / a.stage_bytes);
  if (ns > 8) ns = 8;
  if (ns < 2) ns = 2;
  a.nstages = ns;
  // split-K keeps its fp32 partial tile in the (then idle) stage memory;
  // where that does not fit (very large M), K is not split
  a.max_split = (size_t)ns * a.stage_bytes >= part_bytes ? kTcMaxSplit : 1;
  const size_t fixed = (size_t)ns * a.stage_bytes + (3 * (size_t)ns + 2) * 8 + 16;
  a.sc_off = (int)((fixed + 15) / 16 * 16);
  const size_t smem = 1024 + (size_t)a.sc_off + sc_bytes;
  if (smem > 227 * 1024) return cudaErrorInvalidValue;
#define SQ_TC_CASE(WK_)                                                                \
  if (wk == WK_) return silu ? tc_launch_inst<WK_, true>(tw, tx, a, tiles, smem, st)  \
                             : tc_launch_inst<WK_, false>(tw, tx, a, tiles, smem, st);
  SQ_TC_CASE(SQ_W_FP16)
  SQ_TC_CASE(SQ_W_INT4)
  SQ_TC_CASE(SQ_W_FP8)
#undef SQ_TC_CASE
  return cudaErrorInvalidValue;
}

// Failure-path self-test: one thread waits, with the tile kernel's bounded
// poll loop, on an mbarrier that nothing arrives at; after `polls` polls it
// gives up and sets SQ_DEV_TIMEOUT, exactly as a tile kernel's wait would.
// Nothing is in flight (no bulk copy, no MMA), so giving up is clean.
__global__ void wait_selftest_poll_kernel(uint32_t polls) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x != 0) return;
  mbar_init(&bar, 1);
  fence_mbar_init();
  if (!mbar_wait_bounded(&bar, 0, polls)) atomicOr(&g_tc_status, SQ_DEV_TIMEOUT);
}

cudaError_t launch_wait_selftest_poll(uint32_t polls, cudaStream_t st) {
  wait_selftest_poll_kernel<<<1, 32, 0, st>>>(polls);
  return cudaGetLastError();
}

cudaError_t take_tc_status(uint32_t* bits) {
  uint32_t v = 0, zero = 0;
  cudaError_t e = cudaMemcpyFromSymbol(&v, g_tc_status, sizeof(v));
  if (e != cudaSuccess) return e;
  if (v) e = cudaMemcpyToSymbol(g_tc_status, &zero, sizeof(zero));
  *bits |= v;
  return e;
}

}  // namespace sq
