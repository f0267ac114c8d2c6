// sq_internal.h -- declarations shared by the library's translation units.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/specquant.h"
#include "sq_device.cuh"

namespace sq {

constexpr int kNumSMs = 152;  // GB300: 2 dies x 76 SMs (queried at run time too)

// sq_plan.cu: device properties and the choice of engine and configuration
int device_sm_count();
int device_max_smem();  // opt-in shared memory per block
bool pdl_enabled();     // SQ_PDL environment knob, read once
int64_t weights_per_piece(int wkind);         // weights in one 16-byte piece of a row
int64_t row_bytes_of(int wkind, int64_t K);   // bytes of one weight row
int gemv_cap_mr(int wkind, int64_t K);        // largest activation-row chunk whose x fits
bool use_tensor_cores(int wkind, int M, int64_t N, int64_t K, int epi);

// Launch with programmatic dependent launch allowed: the kernel may begin
// while the previous kernel on the stream drains; it must call
// griddep_wait() before touching data that kernel produced or consumes.
// The legacy default stream gets a plain launch.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t st, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  const bool legacy = (st == nullptr || st == cudaStreamLegacy || st == cudaStreamPerThread);
  const bool pdl = !legacy && pdl_enabled();
  cfg.attrs = pdl ? attr : nullptr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// sq_quantize.cu
cudaError_t launch_quant_int4(const void* w, int64_t N, int64_t K, void* codes, void* scales,
                              cudaStream_t st);
cudaError_t launch_quant_fp8(const void* w, int64_t N, int64_t K, void* codes, void* scales,
                             cudaStream_t st);
cudaError_t take_quant_status(uint32_t* bits);

// GEMV family (sq_gemv_*.cu): M <= 16 rows of activations on CUDA cores.
struct GemvArgs {
  const __half* x;         // [M, K]
  const uint8_t* w;        // weight rows (codes or fp16 bytes)
  const void* scales;      // INT4: fp16 [rows, K/128]; FP8: fp32 [rows]; FP16: unused
  const __half* bias;      // [rows] or null
  const __half* residual;  // [M, N] or null
  __half* y;               // [M, N]
  int M;                   // activation rows present (<= template MR)
  int epi;                 // sq_epilogue
  int64_t N;               // output columns
  int64_t K;
  int64_t row_bytes;       // bytes of one weight row
  int pieces;              // 16-byte pieces per weight row
  int ppad;                // pieces rounded up to a multiple of 32
  const __half* gamma;     // [K] RMSNorm gains: x is normalised while staged; null = x as is
  float eps;
};
constexpr int kGemvMaxRows = 16;
size_t gemv_smem_bytes(int wkind, int mr, int64_t K);
int gemv_pick_mr(int M);
cudaError_t launch_gemv(int wkind, const GemvArgs& a, cudaStream_t st);
// blocks_needed: CTAs that would give every warp one tile; the launcher
// caps it at the number of CTAs that can be resident at once.
cudaError_t launch_gemv_int4(const GemvArgs& a, int mr, int r, bool silu, int lpr, int64_t blocks_needed,
                             size_t smem, cudaStream_t st);
cudaError_t launch_gemv_fp8(const GemvArgs& a, int mr, int r, bool silu, int lpr, int64_t blocks_needed,
                            size_t smem, cudaStream_t st);
cudaError_t launch_gemv_fp16(const GemvArgs& a, int mr, int r, bool silu, int lpr, int64_t blocks_needed,
                             size_t smem, cudaStream_t st);
// INT4 weights, one activation row, products on the tensor cores' register
// path (sq_gemv_mma.cuh); used from kMmaMinTiles 16-row output tiles on (every
// projection of the 7B and 14B stacks the ring engine does not take, the
// 1.5B fused gate/up and lm_head).  Measured: 1.5B draft pass with its
// q/k/v, o and down (96-128 tiles) on it too 170 us against 150 per 8
// layers (too few warps per SM to keep the loads in flight); the 7B ones
// (224-288 tiles) gain, 433 -> 403 us per 8 layers.
constexpr int64_t kMmaMinTiles = 192;
cudaError_t launch_gemv_mma_int4(const GemvArgs& a, bool silu, cudaStream_t st);
inline bool gemv_uses_mma(int wkind, int M, int64_t N) {
  return wkind == SQ_W_INT4 && M == 1 && (N + 15) / 16 >= kMmaMinTiles;
}
cudaError_t take_gemv_status_int4(uint32_t* bits);
cudaError_t take_gemv_status_fp8(uint32_t* bits);
cudaError_t take_gemv_status_fp16(uint32_t* bits);

// sq_tc.cu: tcgen05 tensor-core path (fp16, FP8 or INT4 weights), any M <= 256
bool tc_supported(int M, int64_t K, int epi);
cudaError_t launch_tc(int wkind, const __half* x, const void* w, const void* scales, const __half* bias,
                      const __half* residual, __half* y, int M, int64_t N, int64_t K, int epi,
                      cudaStream_t st);
cudaError_t take_tc_status(uint32_t* bits);

// sq_ring.cu: one to eight activation rows streamed through a shared-memory
// ring, products on the register-operand tensor path (mma.sync).
bool ring_supported(int wkind, int M, int64_t K);
bool use_ring(int wkind, int M, int64_t N, int64_t K, int epi);
cudaError_t launch_ring(int wkind, const __half* x, const void* w, const void* scales, const __half* bias,
                        const __half* residual, __half* y, int M, int64_t N, int64_t K, int epi,
                        cudaStream_t st);
cudaError_t take_ring_status(uint32_t* bits);
// Failure-path self-tests (sq_selftest_wait): a bounded wait that must run out.
cudaError_t launch_wait_selftest_poll(uint32_t polls, cudaStream_t st);      // sq_tc.cu
cudaError_t launch_wait_selftest_time(uint64_t limit_ns, cudaStream_t st);   // sq_ring.cu

// sq_accept.cu
struct AcceptArgs {
  const float* p;
  const float* q;
  const int32_t* draft;
  const float* u;
  int B, K;
  int64_t V;
  int mode;
  int32_t* n_out;
  int32_t* tok_out;
  unsigned long long* part;  // [B][C][slots]
  unsigned int* counter;     // [B]
  int C;                     // chunks per sequence
  int chunk;                 // vocabulary entries per chunk
  int slots;                 // partial slots per chunk
};
constexpr int kAcceptChunk = 2048;
size_t accept_workspace_bytes(int B, int K, int64_t V);
// Size of the static scratch behind sq_accept_noalloc (1 MiB).
constexpr size_t kAcceptNoallocScratchBytes = (size_t)1 << 20;
cudaError_t accept_noalloc_scratch(void** ptr);
cudaError_t launch_accept(const AcceptArgs& a, cudaStream_t st);

// Softmax statistics of the logit rows of one accept-from-logits call:
// target rows zp [rp = B (K+1), V], then draft rows zq [K B, V].
constexpr int kSoftmaxChunk = 2048;
struct SoftmaxArgs {
  const __half* zp;
  const __half* zq;
  int64_t rp;                // target rows
  int64_t rows;              // target + draft rows
  int64_t V;
  float invT;                // 1 / temperature (fp32)
  int C;                     // chunks per row
  float* m;                  // [rows] row maxima
  float* s;                  // [rows] normalisers
  float* pmax;               // [rows * C]
  unsigned long long* psum;  // [rows * C]
  unsigned int* counter;     // [rows], zero on entry, left zero
};
size_t softmax_rows_workspace_bytes(int64_t rows, int64_t V);
size_t softmax_workspace_bytes(int B, int K, int64_t V);
// Points sa's counter / m / s / partial arrays into ws (sa.rows, sa.V set).
void softmax_layout(SoftmaxArgs& sa, void* ws);
cudaError_t launch_accept_logits(const AcceptArgs& a, const SoftmaxArgs& sa, cudaStream_t st);
cudaError_t launch_softmax(const SoftmaxArgs& sa, float* p, cudaStream_t st);
cudaError_t take_accept_status(uint32_t* bits);

}  // namespace sq
