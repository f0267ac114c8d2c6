// sq_tc.cu -- tensor-core (tcgen05 / TMEM) linear layer for M >= 16 rows.
//
// Sec. III-D.3: the verify pass scores B * (K+1) rows at once; from 16 rows
// up this is a real dense tile.  Swap-AB: the weight tile is the MMA's A
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
// Split-K: the S CTAs of a cluster take consecutive K ranges of the same
// weight tile; each writes its fp32 partial tile to its own shared memory,
// and after a cluster barrier CTA r sums rows [r*128/S, (r+1)*128/S) over
// the S partials in rank order through distributed shared memory, so the
// result does not depend on timing.  Every mbarrier wait is bounded (a wait
// that gives up sets SQ_DEV_TIMEOUT and is skipped from then on), so every
// thread always reaches the cluster barriers.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "sq_internal.h"

namespace sq {

static __device__ unsigned int g_tc_status;

constexpr int kTcBM = 128;      // weight rows per tile (MMA M)
constexpr int kTcBK = 64;       // k per stage: 64 fp16 = one 128-byte swizzle row
constexpr int kTcThreads = 192;  // warp 0 TMA, warp 1 MMA + TMEM, warps 2..5 epilogue
constexpr int kTcStageA = kTcBM * kTcBK * 2;  // 16 KB

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

// ---------------------------------------------------------------- kernel

struct TcArgs {
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
  int part_stride;  // floats between columns of the partial tile
  const __half* bias;
  const __half* residual;
  __half* y;
};

template <bool SILU>
__global__ void __launch_bounds__(kTcThreads, 1)
    tc_linear_kernel(const __grid_constant__ CUtensorMap tw, const __grid_constant__ CUtensorMap tx,
                     const TcArgs a) {
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte alignment for the swizzle atoms
  const uint32_t raw = smem_u32(smem_raw);
  uint8_t* smem = smem_raw + (((raw + 1023u) & ~1023u) - raw);
  uint8_t* stages = smem;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + (size_t)a.nstages * a.stage_bytes);
  uint64_t* full = bars;
  uint64_t* empty = bars + a.nstages;
  uint64_t* accf = bars + 2 * a.nstages;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * a.nstages + 1);

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
      const uint32_t bytes = (uint32_t)(kTcStageA * (SILU ? 2 : 1) + a.NB * 128);
      const int pre = nk < a.nstages ? nk : a.nstages;
      // weights never depend on the previous kernel: start them first
      for (int it = 0; it < pre; ++it) {
        uint8_t* st = stages + (size_t)it * a.stage_bytes;
        const int k0 = (k_begin + it) * kTcBK;
        mbar_arrive_expect_tx(&full[it], bytes);
        tma_load_2d(st, &tw, k0, (int)(tile * kTcBM), &full[it]);
        if (SILU) tma_load_2d(st + kTcStageA, &tw, k0, (int)(a.N + tile * kTcBM), &full[it]);
      }
      griddep_wait();
      for (int it = 0; it < pre; ++it)
        tma_load_2d(stages + (size_t)it * a.stage_bytes + a.b_off, &tx, (k_begin + it) * kTcBK, 0,
                    &full[it]);
      for (int it = pre; it < nk; ++it) {
        const int s = it % a.nstages;
        const uint32_t ph = (uint32_t)(it / a.nstages) & 1u;
        if (!timed_out && !mbar_wait_bounded(&empty[s], ph ^ 1u)) {
          timed_out = true;
          atomicOr(&g_tc_status, SQ_DEV_TIMEOUT);
        }
        uint8_t* st = stages + (size_t)s * a.stage_bytes;
        const int k0 = (k_begin + it) * kTcBK;
        mbar_arrive_expect_tx(&full[s], bytes);
        tma_load_2d(st, &tw, k0, (int)(tile * kTcBM), &full[s]);
        if (SILU) tma_load_2d(st + kTcStageA, &tw, k0, (int)(a.N + tile * kTcBM), &full[s]);
        tma_load_2d(st + a.b_off, &tx, k0, 0, &full[s]);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // --------------------------------------------------------- MMA issuer
      for (int it = 0; it < nk; ++it) {
        const int s = it % a.nstages;
        const uint32_t ph = (uint32_t)(it / a.nstages) & 1u;
        if (!timed_out && !mbar_wait_bounded(&full[s], ph)) {
          timed_out = true;
          atomicOr(&g_tc_status, SQ_DEV_TIMEOUT);
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
    // ----------------------------------------------------------- epilogue
    griddep_wait();
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
            if (a.bias) v += __half2float(a.bias[n]);
            if (SILU) {
              float uu = u[j];
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
      const int et = tid - 64;  // 0..127
      const int rows = kTcBM / S;
      const int r0 = (int)rank * rows;
      const float* part = reinterpret_cast<const float*>(stages);
      for (int idx = et; idx < rows * a.M; idx += 128) {
        const int m = idx / rows, row = r0 + (idx - m * rows);
        const int64_t n = tile * kTcBM + row;
        float g = 0.0f, u = 0.0f;
        for (int qq = 0; qq < S; ++qq) {
          g += ld_dsmem_f32(part + (size_t)m * a.part_stride + row, (uint32_t)qq);
          if (SILU) u += ld_dsmem_f32(part + (size_t)(a.NB + m) * a.part_stride + row, (uint32_t)qq);
        }
        if (n < a.N) {
          float v = g;
          if (a.bias) v += __half2float(a.bias[n]);
          if (SILU) {
            if (a.bias) u += __half2float(a.bias[a.N + n]);
            v = v / (1.0f + expf(-v)) * u;
          }
          if (a.residual) v += __half2float(a.residual[(int64_t)m * a.N + n]);
          a.y[(int64_t)m * a.N + n] = __float2half_rn(v);
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

// fp16 [rows, K] row-major -> 2-D tensor map, box (64 k, box_rows), 128-byte
// swizzle, zero fill outside the tensor.
static bool make_map(CUtensorMap* m, const void* base, int64_t rows, int64_t K, int box_rows) {
  auto enc = tensor_map_encoder();
  if (!enc) return false;
  cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)K * 2};
  cuuint32_t box[2] = {(cuuint32_t)kTcBK, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// instruction descriptor, kind::f16: D fp32, A and B fp16, both K-major,
// N = nb, M = 128
static uint32_t make_idesc(int nb) {
  uint32_t d = 0;
  d |= 1u << 4;                  // D format fp32
  d |= (uint32_t)(nb >> 3) << 17;  // N / 8
  d |= (uint32_t)(kTcBM >> 4) << 24;  // M / 16
  return d;
}

bool tc_supported(int M, int64_t K, int epi) {
  (void)epi;
  return M >= 16 && M <= 256 && K % 8 == 0 && tensor_map_encoder() != nullptr;
}

cudaError_t launch_tc_fp16(const __half* x, const __half* w, const __half* bias, const __half* residual,
                           __half* y, int M, int64_t N, int64_t K, int epi, cudaStream_t st) {
  const bool silu = epi == SQ_EPI_SILU_GATE;
  const int nb = (M + 15) / 16 * 16;
  const int64_t wrows = silu ? 2 * N : N;
  CUtensorMap tw, tx;
  if (!make_map(&tw, w, wrows, K, kTcBM) || !make_map(&tx, x, M, K, nb)) return cudaErrorInvalidValue;
  TcArgs a = {};
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
  const int cols = nb * (silu ? 2 : 1);
  int tc = 32;
  while (tc < cols) tc <<= 1;
  a.tmem_cols = tc;
  const int a_bytes = kTcStageA * (silu ? 2 : 1);
  const int b_bytes = (nb * 128 + 1023) / 1024 * 1024;
  a.b_off = a_bytes;
  a.stage_bytes = a_bytes + b_bytes;
  // split K over a cluster until the tiles cover the SMs
  const int64_t tiles = (N + kTcBM - 1) / kTcBM;
  const int sms = device_sm_count();
  int S = 1;
  while (S < 8 && tiles * S * 2 <= sms && a.ksteps >= 4 * S * 2) S <<= 1;
  a.splits = S;
  a.part_stride = kTcBM + 4;
  const size_t part_bytes = (size_t)cols * a.part_stride * 4;
  int ns = (int)((200 * 1024) / a.stage_bytes);
  if (ns > 8) ns = 8;
  if (ns < 2) ns = 2;
  while ((size_t)ns * a.stage_bytes < part_bytes) ++ns;
  a.nstages = ns;
  const size_t smem = 1024 + (size_t)ns * a.stage_bytes + (2 * ns + 2) * 8 + 16;
  auto k = silu ? tc_linear_kernel<true> : tc_linear_kernel<false>;
  static int smem_set[2][64] = {{0}};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if ((int)smem > smem_set[silu][dev]) {
    e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    if (S > 1) {
      e = cudaFuncSetAttribute(k, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
      if (e != cudaSuccess) return e;
    }
    smem_set[silu][dev] = (int)smem;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)S, (unsigned)tiles, 1);
  cfg.blockDim = dim3(kTcThreads);
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

cudaError_t take_tc_status(uint32_t* bits) {
  uint32_t v = 0, zero = 0;
  cudaError_t e = cudaMemcpyFromSymbol(&v, g_tc_status, sizeof(v));
  if (e != cudaSuccess) return e;
  if (v) e = cudaMemcpyToSymbol(g_tc_status, &zero, sizeof(zero));
  *bits |= v;
  return e;
}

}  // namespace sq
