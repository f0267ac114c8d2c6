// sq_capi.cu -- the C ABI (include/specquant.h): argument validation, status
// reporting and dispatch to the kernels.  Nothing here computes any part of
// the hot path; it only checks arguments and launches.
#include <stdarg.h>
#include <stdio.h>
#include <stdlib.h>

#include <nvtx3/nvToolsExt.h>

#include <cmath>
#include <string>

#include "sq_decoder.h"
#include "sq_internal.h"

namespace sq {

static thread_local std::string g_last_error;

static sq_status fail(sq_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return s;
}

static sq_status cuda_fail(cudaError_t e, const char* where) {
  return fail(SQ_ERR_CUDA, "%s: %s (%s)", where, cudaGetErrorName(e), cudaGetErrorString(e));
}

static bool aligned(const void* p, uintptr_t a) { return ((uintptr_t)p % a) == 0; }

// One NVTX range per entry point that launches or waits on device work,
// named after it, so that a timeline attributes every kernel to the call
// that issued it.  Host-only, no allocation; with no profiler attached a push
// and a pop cost a few nanoseconds.
struct CallRange {
  explicit CallRange(const char* name) { nvtxRangePushA(name); }
  ~CallRange() { nvtxRangePop(); }
  CallRange(const CallRange&) = delete;
  CallRange& operator=(const CallRange&) = delete;
};
#define SQ_RANGE() ::sq::CallRange sq_call_range_(__func__)

}  // namespace sq

using namespace sq;

extern "C" {

const char* sq_last_error(void) { return g_last_error.c_str(); }

const char* sq_status_string(sq_status s) {
  switch (s) {
    case SQ_OK: return "SQ_OK";
    case SQ_ERR_INVALID_ARG: return "SQ_ERR_INVALID_ARG";
    case SQ_ERR_SHAPE: return "SQ_ERR_SHAPE";
    case SQ_ERR_ALIGN: return "SQ_ERR_ALIGN";
    case SQ_ERR_UNSUPPORTED: return "SQ_ERR_UNSUPPORTED";
    case SQ_ERR_WORKSPACE: return "SQ_ERR_WORKSPACE";
    case SQ_ERR_CUDA: return "SQ_ERR_CUDA";
    case SQ_ERR_DEVICE: return "SQ_ERR_DEVICE";
  }
  return "SQ_STATUS_UNKNOWN";
}

int sq_version(void) { return 100; }

sq_status sq_check(sq_stream_t stream, uint32_t* device_bits) {
  SQ_RANGE();
  cudaError_t e = cudaStreamSynchronize((cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "sq_check: stream synchronize");
  uint32_t bits = 0;
  if ((e = take_quant_status(&bits)) != cudaSuccess) return cuda_fail(e, "sq_check: quantize status");
  if ((e = take_accept_status(&bits)) != cudaSuccess) return cuda_fail(e, "sq_check: accept status");
  if ((e = take_gemv_status_int4(&bits)) != cudaSuccess ||
      (e = take_gemv_status_fp8(&bits)) != cudaSuccess ||
      (e = take_gemv_status_fp16(&bits)) != cudaSuccess || (e = take_tc_status(&bits)) != cudaSuccess ||
      (e = take_attn_status(&bits)) != cudaSuccess || (e = take_ring_status(&bits)) != cudaSuccess)
    return cuda_fail(e, "sq_check: linear status");
  if (device_bits) *device_bits = bits;
  if (bits) return fail(SQ_ERR_DEVICE, "sq_check: device status bits 0x%x", bits);
  return SQ_OK;
}

size_t sq_quantized_bytes(sq_qkind kind, int64_t N, int64_t K, size_t* scale_bytes) {
  if (scale_bytes) *scale_bytes = 0;
  if (N < 0 || K <= 0) return 0;
  if (kind == SQ_INT4_G128) {
    if (K % 128) return 0;
    if (scale_bytes) *scale_bytes = (size_t)N * (size_t)(K / 128) * 2u;
    return (size_t)N * (size_t)(K / 2);
  }
  if (kind == SQ_FP8_E4M3_ROW) {
    if (K % 16) return 0;
    if (scale_bytes) *scale_bytes = (size_t)N * 4u;
    return (size_t)N * (size_t)K;
  }
  return 0;
}

sq_status sq_quantize(const void* w16, int64_t N, int64_t K, sq_qkind kind, void* codes,
                      void* scales, sq_stream_t stream) {
  SQ_RANGE();
  if (kind != SQ_INT4_G128 && kind != SQ_FP8_E4M3_ROW)
    return fail(SQ_ERR_INVALID_ARG, "sq_quantize: unknown kind %d", (int)kind);
  if (N < 0 || K <= 0) return fail(SQ_ERR_SHAPE, "sq_quantize: N=%lld K=%lld", (long long)N, (long long)K);
  if (kind == SQ_INT4_G128 && K % 128)
    return fail(SQ_ERR_SHAPE, "sq_quantize: INT4 needs K %% 128 == 0 (K=%lld)", (long long)K);
  if (kind == SQ_FP8_E4M3_ROW && K % 16)
    return fail(SQ_ERR_SHAPE, "sq_quantize: FP8 needs K %% 16 == 0 (K=%lld)", (long long)K);
  if (N == 0) return SQ_OK;
  if (!w16 || !codes || !scales) return fail(SQ_ERR_INVALID_ARG, "sq_quantize: NULL pointer");
  if (!aligned(w16, 16) || !aligned(codes, 16))
    return fail(SQ_ERR_ALIGN, "sq_quantize: w16 and codes must be 16-byte aligned");
  if (!aligned(scales, kind == SQ_INT4_G128 ? 2 : 4))
    return fail(SQ_ERR_ALIGN, "sq_quantize: scales misaligned");
  cudaError_t e = kind == SQ_INT4_G128 ? launch_quant_int4(w16, N, K, codes, scales, (cudaStream_t)stream)
                                       : launch_quant_fp8(w16, N, K, codes, scales, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "sq_quantize: launch");
  return SQ_OK;
}

// Kind and size rules of sq_linear_ex (shared with sq_linear_path).
static sq_status check_linear_sizes(sq_wkind wkind, int M, int64_t N, int64_t K, sq_epilogue epi) {
  if (wkind != SQ_W_FP16 && wkind != SQ_W_INT4 && wkind != SQ_W_FP8)
    return fail(SQ_ERR_INVALID_ARG, "sq_linear: unknown weight kind %d", (int)wkind);
  if (epi != SQ_EPI_NONE && epi != SQ_EPI_SILU_GATE && epi != SQ_EPI_RESIDUAL)
    return fail(SQ_ERR_INVALID_ARG, "sq_linear: unknown epilogue %d", (int)epi);
  if (M < 1 || M > 256 || N < 1 || K < 1)
    return fail(SQ_ERR_SHAPE, "sq_linear: need 1 <= M <= 256, N >= 1, K >= 1 (M=%d N=%lld K=%lld)", M,
                (long long)N, (long long)K);
  if (wkind == SQ_W_INT4 && K % 128)
    return fail(SQ_ERR_SHAPE, "sq_linear_w4a16: K %% 128 != 0 (K=%lld)", (long long)K);
  if (wkind == SQ_W_FP8 && K % 16)
    return fail(SQ_ERR_SHAPE, "sq_linear_fp8: K %% 16 != 0 (K=%lld)", (long long)K);
  if (wkind == SQ_W_FP16 && K % 8)
    return fail(SQ_ERR_SHAPE, "sq_verify: K %% 8 != 0 (K=%lld)", (long long)K);
  if (N > (int64_t)1 << 30 || K > (int64_t)1 << 20)
    return fail(SQ_ERR_SHAPE, "sq_linear: N or K too large");
  if (gemv_cap_mr(wkind, K) == 0)
    return fail(SQ_ERR_SHAPE, "sq_linear: K=%lld too large for the staged activations", (long long)K);
  return SQ_OK;
}

// Pointer and alignment rules of one linear call.
static sq_status check_linear_ptrs(const sq_linear_op& op) {
  if (!op.x || !op.w || !op.y) return fail(SQ_ERR_INVALID_ARG, "sq_linear: NULL x, weight or y");
  if (op.wkind != SQ_W_FP16 && !op.scales) return fail(SQ_ERR_INVALID_ARG, "sq_linear: NULL scales");
  if (op.epi == SQ_EPI_RESIDUAL && !op.residual)
    return fail(SQ_ERR_INVALID_ARG, "sq_linear: SQ_EPI_RESIDUAL needs a residual");
  if (!aligned(op.x, 16) || !aligned(op.w, 16) || !aligned(op.y, 2))
    return fail(SQ_ERR_ALIGN, "sq_linear: x and weights must be 16-byte aligned, y 2-byte aligned");
  if (op.scales && !aligned(op.scales, op.wkind == SQ_W_FP8 ? 4 : 2))
    return fail(SQ_ERR_ALIGN, "sq_linear: scales misaligned");
  if ((op.bias && !aligned(op.bias, 2)) || (op.residual && !aligned(op.residual, 2)))
    return fail(SQ_ERR_ALIGN, "sq_linear: bias/residual misaligned");
  return SQ_OK;
}

static sq_status check_linear(const sq_linear_op& op) {
  if (op.reserved != 0) return fail(SQ_ERR_INVALID_ARG, "sq_linear_chain: reserved field must be 0");
  sq_status st = check_linear_sizes(op.wkind, op.M, op.N, op.K, op.epi);
  if (st != SQ_OK) return st;
  return check_linear_ptrs(op);
}

// Launches one checked call.
// gamma != null: y = linear(rmsnorm(x) * gamma).  The GEMV kernels normalise
// the rows they stage; the tensor-core tile path writes the normalised rows to
// xn first.
static sq_status run_linear(const sq_linear_op& op, cudaStream_t stream, const __half* gamma = nullptr,
                            float eps = 0.0f, __half* xn = nullptr) {
  GemvArgs a = {};
  a.x = reinterpret_cast<const __half*>(op.x);
  a.gamma = gamma;
  a.eps = eps;
  a.w = reinterpret_cast<const uint8_t*>(op.w);
  a.scales = op.scales;
  a.bias = reinterpret_cast<const __half*>(op.bias);
  a.residual = op.epi == SQ_EPI_RESIDUAL ? reinterpret_cast<const __half*>(op.residual) : nullptr;
  a.y = reinterpret_cast<__half*>(op.y);
  a.M = op.M;
  a.epi = op.epi;
  a.N = op.N;
  a.K = op.K;
  a.row_bytes = row_bytes_of(op.wkind, op.K);
  a.pieces = (int)(op.K / weights_per_piece(op.wkind));
  a.ppad = (a.pieces + 31) / 32 * 32;
  cudaError_t e;
  // the ring engine where the planner sends it, else the tcgen05 tile path,
  // else the GEMV family (sq_plan.cu)
  const bool ring = use_ring(op.wkind, op.M, op.N, op.K, op.epi);
  const bool tc = !ring && use_tensor_cores(op.wkind, op.M, op.N, op.K, op.epi) &&
                  tc_supported(op.M, op.K, op.epi);
  if (gamma && (tc || ring)) {
    // the tensor-core tile path and the ring engine stage x by copies: the
    // standalone RMSNorm first
    e = launch_rmsnorm(a.x, gamma, op.M, op.K, eps, xn, stream);
    if (e != cudaSuccess) return cuda_fail(e, "sq_linear_norm: rmsnorm launch");
    a.x = xn;
    a.gamma = nullptr;
  }
  if (ring) {
    // one to eight rows through the shared-memory ring, register-operand tensor cores
    e = launch_ring(op.wkind, a.x, op.w, op.scales, a.bias, a.residual, a.y, op.M, op.N, op.K, op.epi,
                    stream);
    if (e != cudaSuccess) return cuda_fail(e, "sq_linear: ring launch");
    return SQ_OK;
  }
  if (tc) {
    // tcgen05 tensor cores, weights on the MMA's M side
    e = launch_tc(op.wkind, a.x, op.w, op.scales, a.bias, a.residual, a.y, op.M, op.N, op.K, op.epi,
                  stream);
    if (e != cudaSuccess) return cuda_fail(e, "sq_linear: tensor-core launch");
    return SQ_OK;
  }
  e = launch_gemv(op.wkind, a, stream);
  if (e != cudaSuccess) return cuda_fail(e, "sq_linear: launch");
  return SQ_OK;
}

sq_status sq_linear_norm(sq_wkind wkind, const void* x, const void* gamma, float eps, void* xn, const void* w,
                         const void* scales, const void* bias, const void* residual, sq_epilogue epi, void* y,
                         int M, int64_t N, int64_t K, sq_stream_t stream) {
  SQ_RANGE();
  sq_linear_op op = {};
  op.wkind = wkind;
  op.epi = epi;
  op.M = M;
  op.N = N;
  op.K = K;
  op.x = x;
  op.w = w;
  op.scales = scales;
  op.bias = bias;
  op.residual = residual;
  op.y = y;
  sq_status st = check_linear(op);
  if (st != SQ_OK) return st;
  if (M == 0 || N == 0) return SQ_OK;
  if (!gamma || !xn) return fail(SQ_ERR_INVALID_ARG, "sq_linear_norm: NULL gamma or xn");
  if (!aligned(gamma, 16) || !aligned(xn, 16))
    return fail(SQ_ERR_ALIGN, "sq_linear_norm: gamma and xn must be 16-byte aligned");
  if (!(eps >= 0.0f) || !std::isfinite(eps)) return fail(SQ_ERR_INVALID_ARG, "sq_linear_norm: bad eps");
  if (xn == y || xn == x || (residual && xn == residual))
    return fail(SQ_ERR_INVALID_ARG, "sq_linear_norm: xn must not alias x, y or the residual");
  return run_linear(op, (cudaStream_t)stream, reinterpret_cast<const __half*>(gamma), eps,
                    reinterpret_cast<__half*>(xn));
}

sq_status sq_linear_ex(sq_wkind wkind, const void* x, const void* w, const void* scales,
                       const void* bias, const void* residual, sq_epilogue epi, void* y, int M,
                       int64_t N, int64_t K, sq_stream_t stream) {
  SQ_RANGE();
  sq_linear_op op = {};
  op.wkind = wkind;
  op.epi = epi;
  op.M = M;
  op.N = N;
  op.K = K;
  op.x = x;
  op.w = w;
  op.scales = scales;
  op.bias = bias;
  op.residual = residual;
  op.y = y;
  sq_status st = check_linear(op);
  if (st != SQ_OK) return st;
  return run_linear(op, (cudaStream_t)stream);
}

sq_status sq_linear_chain(const sq_linear_op* ops, int count, sq_stream_t stream) {
  SQ_RANGE();
  if (count < 0 || (count > 0 && !ops))
    return fail(SQ_ERR_INVALID_ARG, "sq_linear_chain: need ops and count >= 0");
  for (int i = 0; i < count; ++i) {
    sq_status st = check_linear(ops[i]);
    if (st != SQ_OK) return fail(st, "sq_linear_chain: op %d: %s", i, g_last_error.c_str());
  }
  for (int i = 0; i < count; ++i) {
    sq_status st = run_linear(ops[i], (cudaStream_t)stream);
    if (st != SQ_OK) return fail(st, "sq_linear_chain: op %d: %s", i, g_last_error.c_str());
  }
  return SQ_OK;
}

sq_status sq_selftest_wait(int which, uint64_t limit, sq_stream_t stream) {
  SQ_RANGE();
  if (which != 0 && which != 1) return fail(SQ_ERR_INVALID_ARG, "sq_selftest_wait: which must be 0 or 1");
  if (which == 0 && (limit < 1 || limit > ((uint64_t)1 << 24)))
    return fail(SQ_ERR_INVALID_ARG, "sq_selftest_wait: polls must be in [1, 2^24]");
  if (which == 1 && (limit < 1 || limit > 1000000000ull))
    return fail(SQ_ERR_INVALID_ARG, "sq_selftest_wait: limit must be in [1 ns, 1 s]");
  cudaError_t e = which == 0 ? launch_wait_selftest_poll((uint32_t)limit, (cudaStream_t)stream)
                             : launch_wait_selftest_time(limit, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "sq_selftest_wait: launch");
  return SQ_OK;
}

int sq_linear_path(sq_wkind wkind, int M, int64_t N, int64_t K, sq_epilogue epi) {
  if (check_linear_sizes(wkind, M, N, K, epi) != SQ_OK) return -1;
  if (use_ring(wkind, M, N, K, epi)) return 3;
  if (use_tensor_cores(wkind, M, N, K, epi) && tc_supported(M, K, epi)) return 1;
  return gemv_uses_mma(wkind, M, N) ? 2 : 0;
}

sq_status sq_linear_w4a16(const void* x, const void* codes, const void* scales, const void* bias,
                          void* y, int M, int64_t N, int64_t K, sq_stream_t stream) {
  SQ_RANGE();
  return sq_linear_ex(SQ_W_INT4, x, codes, scales, bias, nullptr, SQ_EPI_NONE, y, M, N, K, stream);
}

sq_status sq_linear_fp8(const void* x, const void* codes, const float* scales, const void* bias,
                        void* y, int M, int64_t N, int64_t K, sq_stream_t stream) {
  SQ_RANGE();
  return sq_linear_ex(SQ_W_FP8, x, codes, scales, bias, nullptr, SQ_EPI_NONE, y, M, N, K, stream);
}

sq_status sq_verify(const void* x, const void* w16, const void* bias, void* y, int M, int64_t N,
                    int64_t K, sq_stream_t stream) {
  SQ_RANGE();
  return sq_linear_ex(SQ_W_FP16, x, w16, nullptr, bias, nullptr, SQ_EPI_NONE, y, M, N, K, stream);
}

size_t sq_accept_workspace_bytes(int B, int K, int64_t V) {
  if (B < 0 || K < 0 || K > 16 || V < 1 || V >= ((int64_t)1 << 20)) return 0;
  return accept_workspace_bytes(B, K, V);
}

// clear_counters: zero the ticket counters at the head of the workspace first
// (the static scratch of sq_accept_noalloc), once every argument is valid.
static sq_status accept_common(const char* who, const float* p, const float* q, const int32_t* draft,
                               const float* u, int B, int K, int64_t V, int mode, int32_t* n_accepted,
                               int32_t* tokens, void* workspace, size_t ws_bytes,
                               sq_stream_t stream, bool clear_counters = false) {
  if (mode != SQ_ACCEPT_SAMPLE && mode != SQ_ACCEPT_GREEDY)
    return fail(SQ_ERR_INVALID_ARG, "%s: unknown mode %d", who, mode);
  if (B < 0 || K < 0 || K > 16 || V < 1 || V >= ((int64_t)1 << 20))
    return fail(SQ_ERR_SHAPE, "%s: need B >= 0, 0 <= K <= 16, 1 <= V < 2^20 (B=%d K=%d V=%lld)", who, B,
                K, (long long)V);
  if (B == 0) return SQ_OK;
  if (!p || !u || !tokens || (K > 0 && !draft))
    return fail(SQ_ERR_INVALID_ARG, "%s: NULL p, u, draft or tokens", who);
  if (K > 0 && mode == SQ_ACCEPT_SAMPLE && !q)
    return fail(SQ_ERR_INVALID_ARG, "%s: sampling mode with K > 0 needs q", who);
  if (!aligned(p, 4) || (q && !aligned(q, 4)) || !aligned(u, 4) || (draft && !aligned(draft, 4)) ||
      !aligned(tokens, 4) || (n_accepted && !aligned(n_accepted, 4)))
    return fail(SQ_ERR_ALIGN, "%s: pointers must be 4-byte aligned", who);
  const size_t need = accept_workspace_bytes(B, K, V);
  if (!workspace || ws_bytes < need)
    return fail(SQ_ERR_WORKSPACE, "%s: workspace %zu bytes < %zu required", who, ws_bytes, need);
  if (!aligned(workspace, 16)) return fail(SQ_ERR_ALIGN, "%s: workspace must be 16-byte aligned", who);
  AcceptArgs a = {};
  a.p = p;
  a.q = K > 0 ? q : nullptr;
  a.draft = draft;
  a.u = u;
  a.B = B;
  a.K = K;
  a.V = V;
  a.mode = mode;
  a.n_out = n_accepted;
  a.tok_out = tokens;
  const size_t ctr = (((size_t)B * 4u) + 15u) & ~(size_t)15u;
  a.counter = reinterpret_cast<unsigned int*>(workspace);
  a.part = reinterpret_cast<unsigned long long*>(reinterpret_cast<char*>(workspace) + ctr);
  a.C = (int)((V + kAcceptChunk - 1) / kAcceptChunk);
  a.chunk = kAcceptChunk;
  a.slots = K + 1 > 2 ? K + 1 : 2;
  cudaError_t e;
  if (clear_counters) {
    e = cudaMemsetAsync(workspace, 0, ctr, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, "sq_accept: clearing the ticket counters");
  }
  e = launch_accept(a, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "sq_accept: launch");
  return SQ_OK;
}

sq_status sq_accept(const float* p, const float* q, const int32_t* draft, const float* u, int B, int K,
                    int64_t V, sq_accept_mode mode, int32_t* n_accepted, int32_t* tokens,
                    void* workspace, size_t ws_bytes, sq_stream_t stream) {
  SQ_RANGE();
  if (!n_accepted && B > 0) return fail(SQ_ERR_INVALID_ARG, "sq_accept: NULL n_accepted");
  return accept_common("sq_accept", p, q, draft, u, B, K, V, (int)mode, n_accepted, tokens, workspace,
                       ws_bytes, stream);
}

sq_status sq_sample(const float* probs, const float* u, int B, int64_t V, int32_t* tokens,
                    void* workspace, size_t ws_bytes, sq_stream_t stream) {
  SQ_RANGE();
  return accept_common("sq_sample", probs, nullptr, nullptr, u, B, 0, V, SQ_ACCEPT_SAMPLE, nullptr,
                       tokens, workspace, ws_bytes, stream);
}

size_t sq_accept_logits_workspace_bytes(int B, int K, int64_t V) {
  const size_t acc = accept_workspace_bytes(B, K, V);
  const size_t sm = softmax_workspace_bytes(B, K, V);
  if (acc == 0 || sm == 0) return 0;
  return ((acc + 15u) & ~(size_t)15u) + sm;
}

static sq_status accept_logits_common(const char* who, const void* zp, const void* zq,
                                      const int32_t* draft, const float* u, int B, int K, int64_t V,
                                      float temperature, int mode, int32_t* n_accepted,
                                      int32_t* tokens, void* workspace, size_t ws_bytes,
                                      sq_stream_t stream) {
  if (mode != SQ_ACCEPT_SAMPLE && mode != SQ_ACCEPT_GREEDY)
    return fail(SQ_ERR_INVALID_ARG, "%s: unknown mode %d", who, mode);
  if (B < 0 || K < 0 || K > 16 || V < 1 || V >= ((int64_t)1 << 20))
    return fail(SQ_ERR_SHAPE, "%s: need B >= 0, 0 <= K <= 16, 1 <= V < 2^20 (B=%d K=%d V=%lld)", who, B,
                K, (long long)V);
  if (!(temperature > 0.0f) || !std::isfinite(temperature))
    return fail(SQ_ERR_INVALID_ARG, "%s: temperature must be positive and finite", who);
  if (B == 0) return SQ_OK;
  if (!zp || !u || !tokens || (K > 0 && (!draft || !zq)))
    return fail(SQ_ERR_INVALID_ARG, "%s: NULL logits, u, draft or tokens", who);
  if (!aligned(zp, 2) || (zq && !aligned(zq, 2)) || !aligned(u, 4) || (draft && !aligned(draft, 4)) ||
      !aligned(tokens, 4) || (n_accepted && !aligned(n_accepted, 4)))
    return fail(SQ_ERR_ALIGN, "%s: logits must be 2-byte, other pointers 4-byte aligned", who);
  const size_t need = sq_accept_logits_workspace_bytes(B, K, V);
  if (!workspace || ws_bytes < need)
    return fail(SQ_ERR_WORKSPACE, "%s: workspace %zu bytes < %zu required", who, ws_bytes, need);
  if (!aligned(workspace, 16)) return fail(SQ_ERR_ALIGN, "%s: workspace must be 16-byte aligned", who);
  auto up16 = [](size_t x) { return (x + 15u) & ~(size_t)15u; };
  char* ws = reinterpret_cast<char*>(workspace);
  AcceptArgs a = {};
  a.draft = draft;
  a.u = u;
  a.B = B;
  a.K = K;
  a.V = V;
  a.mode = mode;
  a.n_out = n_accepted;
  a.tok_out = tokens;
  const size_t ctr = up16((size_t)B * 4u);
  a.counter = reinterpret_cast<unsigned int*>(ws);
  a.part = reinterpret_cast<unsigned long long*>(ws + ctr);
  a.C = (int)((V + kAcceptChunk - 1) / kAcceptChunk);
  a.chunk = kAcceptChunk;
  a.slots = K + 1 > 2 ? K + 1 : 2;
  // softmax statistics after the accept workspace
  SoftmaxArgs sa = {};
  sa.zp = reinterpret_cast<const __half*>(zp);
  sa.zq = K > 0 ? reinterpret_cast<const __half*>(zq) : nullptr;
  sa.rp = (int64_t)B * (K + 1);
  sa.rows = sa.rp + (int64_t)B * K;
  sa.V = V;
  sa.invT = 1.0f / temperature;
  softmax_layout(sa, ws + up16(accept_workspace_bytes(B, K, V)));
  cudaError_t e = launch_accept_logits(a, sa, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "sq_accept_logits: launch");
  return SQ_OK;
}

sq_status sq_accept_logits(const void* zp, const void* zq, const int32_t* draft, const float* u, int B,
                           int K, int64_t V, float temperature, sq_accept_mode mode,
                           int32_t* n_accepted, int32_t* tokens, void* workspace, size_t ws_bytes,
                           sq_stream_t stream) {
  SQ_RANGE();
  if (!n_accepted && B > 0) return fail(SQ_ERR_INVALID_ARG, "sq_accept_logits: NULL n_accepted");
  return accept_logits_common("sq_accept_logits", zp, zq, draft, u, B, K, V, temperature, (int)mode,
                              n_accepted, tokens, workspace, ws_bytes, stream);
}

sq_status sq_sample_logits(const void* z, const float* u, int B, int64_t V, float temperature,
                           int32_t* tokens, void* workspace, size_t ws_bytes, sq_stream_t stream) {
  SQ_RANGE();
  return accept_logits_common("sq_sample_logits", z, nullptr, nullptr, u, B, 0, V, temperature,
                              SQ_ACCEPT_SAMPLE, nullptr, tokens, workspace, ws_bytes, stream);
}

size_t sq_softmax_workspace_bytes(int64_t R, int64_t V) { return softmax_rows_workspace_bytes(R, V); }

sq_status sq_softmax(const void* z, int64_t R, int64_t V, float temperature, float* p, void* workspace,
                     size_t ws_bytes, sq_stream_t stream) {
  SQ_RANGE();
  if (R < 0 || V < 1 || V >= ((int64_t)1 << 20))
    return fail(SQ_ERR_SHAPE, "sq_softmax: need R >= 0, 1 <= V < 2^20 (R=%lld V=%lld)", (long long)R,
                (long long)V);
  if (!(temperature > 0.0f) || !std::isfinite(temperature))
    return fail(SQ_ERR_INVALID_ARG, "sq_softmax: temperature must be positive and finite");
  if (R == 0) return SQ_OK;
  if (!z || !p) return fail(SQ_ERR_INVALID_ARG, "sq_softmax: NULL z or p");
  if (!aligned(z, 2) || !aligned(p, 4))
    return fail(SQ_ERR_ALIGN, "sq_softmax: z must be 2-byte, p 4-byte aligned");
  const size_t need = softmax_rows_workspace_bytes(R, V);
  if (!workspace || ws_bytes < need)
    return fail(SQ_ERR_WORKSPACE, "sq_softmax: workspace %zu bytes < %zu required", ws_bytes, need);
  if (!aligned(workspace, 16)) return fail(SQ_ERR_ALIGN, "sq_softmax: workspace must be 16-byte aligned");
  SoftmaxArgs sa = {};
  sa.zp = reinterpret_cast<const __half*>(z);
  sa.zq = nullptr;
  sa.rp = R;
  sa.rows = R;
  sa.V = V;
  sa.invT = 1.0f / temperature;
  softmax_layout(sa, workspace);
  cudaError_t e = launch_softmax(sa, p, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "sq_softmax: launch");
  return SQ_OK;
}

// ---- decoder pieces

sq_status sq_rmsnorm(const void* x, const void* gamma, int M, int64_t H, float eps, void* y,
                     sq_stream_t stream) {
  SQ_RANGE();
  if (M < 0 || H < 1) return fail(SQ_ERR_SHAPE, "sq_rmsnorm: need M >= 0, H >= 1");
  if (!(eps >= 0.0f) || !std::isfinite(eps)) return fail(SQ_ERR_INVALID_ARG, "sq_rmsnorm: bad eps");
  if (M == 0) return SQ_OK;
  if (!x || !gamma || !y) return fail(SQ_ERR_INVALID_ARG, "sq_rmsnorm: NULL pointer");
  if (!aligned(x, 2) || !aligned(gamma, 2) || !aligned(y, 2))
    return fail(SQ_ERR_ALIGN, "sq_rmsnorm: pointers must be 2-byte aligned");
  cudaError_t e = launch_rmsnorm(reinterpret_cast<const __half*>(x), reinterpret_cast<const __half*>(gamma),
                                 M, H, eps, reinterpret_cast<__half*>(y), (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "sq_rmsnorm: launch");
  return SQ_OK;
}

static sq_status check_attn(const char* who, const void* qkv, int B, int T, int Hq, int Hkv, int D,
                            const int32_t* pos0, float theta, const void* kc, const void* vc,
                            int64_t max_ctx) {
  if (B < 0 || T < 0 || Hq < 1 || Hkv < 1 || Hq % Hkv || max_ctx < 1)
    return fail(SQ_ERR_SHAPE, "%s: need B, T >= 0, Hq a positive multiple of Hkv, max_ctx >= 1", who);
  if (D != 128) return fail(SQ_ERR_UNSUPPORTED, "%s: head dimension %d (only 128 is built)", who, D);
  if ((Hq / Hkv) * T > 200 || T > attention_max_tokens())
    return fail(SQ_ERR_SHAPE, "%s: need (Hq / Hkv) * T <= 200 and T <= %d", who, attention_max_tokens());
  if (!(theta > 1.0f) || !std::isfinite(theta)) return fail(SQ_ERR_INVALID_ARG, "%s: theta must be > 1", who);
  if (B > 0 && T > 0 && (!qkv || !pos0 || !kc || !vc))
    return fail(SQ_ERR_INVALID_ARG, "%s: NULL pointer", who);
  if (!aligned(qkv, 2) || !aligned(pos0, 4) || !aligned(kc, 16) || !aligned(vc, 16))
    return fail(SQ_ERR_ALIGN, "%s: misaligned pointer (caches need 16 bytes)", who);
  return SQ_OK;
}

sq_status sq_kv_append(const void* qkv, int B, int T, int Hq, int Hkv, int D, const int32_t* pos0,
                       float theta, void* k_cache, void* v_cache, int64_t max_ctx, sq_stream_t stream) {
  SQ_RANGE();
  sq_status st = check_attn("sq_kv_append", qkv, B, T, Hq, Hkv, D, pos0, theta, k_cache, v_cache, max_ctx);
  if (st != SQ_OK) return st;
  cudaError_t e = launch_kv_append(reinterpret_cast<const __half*>(qkv), B, T, Hq, Hkv, pos0, (double)theta,
                                   reinterpret_cast<__half*>(k_cache), reinterpret_cast<__half*>(v_cache),
                                   max_ctx, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "sq_kv_append: launch");
  return SQ_OK;
}

size_t sq_attention_workspace_bytes(int B, int T, int Hq, int Hkv, int D, int64_t max_ctx) {
  if (D != 128 || Hkv < 1 || Hq % Hkv) return 0;
  return attention_workspace_bytes(B, T, Hq, Hkv, max_ctx);
}

static sq_status attention_common(const char* who, const void* qkv, int B, int T, int Hq, int Hkv, int D,
                                  const int32_t* pos0, float theta, const void* k_cache, const void* v_cache,
                                  int64_t max_ctx, void* out, void* workspace, size_t ws_bytes, bool append,
                                  sq_stream_t stream) {
  sq_status st = check_attn(who, qkv, B, T, Hq, Hkv, D, pos0, theta, k_cache, v_cache, max_ctx);
  if (st != SQ_OK) return st;
  if (B == 0 || T == 0) return SQ_OK;
  if (!out || !aligned(out, 2)) return fail(SQ_ERR_ALIGN, "%s: out NULL or misaligned", who);
  const size_t need = attention_workspace_bytes(B, T, Hq, Hkv, max_ctx);
  if (!workspace || ws_bytes < need)
    return fail(SQ_ERR_WORKSPACE, "%s: workspace %zu bytes < %zu required", who, ws_bytes, need);
  if (!aligned(workspace, 16)) return fail(SQ_ERR_ALIGN, "%s: workspace must be 16-byte aligned", who);
  if (attention_smem_bytes((Hq / Hkv) * T) > (size_t)device_max_smem())
    return fail(SQ_ERR_SHAPE, "%s: query group too large for shared memory", who);
  if (max_ctx > ((int64_t)1 << 17)) return fail(SQ_ERR_SHAPE, "%s: max_ctx > 2^17", who);
  __half* kw = append ? reinterpret_cast<__half*>(const_cast<void*>(k_cache)) : nullptr;
  __half* vw = append ? reinterpret_cast<__half*>(const_cast<void*>(v_cache)) : nullptr;
  cudaError_t e = launch_attention(reinterpret_cast<const __half*>(qkv), B, T, Hq, Hkv, pos0, (double)theta,
                                   reinterpret_cast<const __half*>(k_cache),
                                   reinterpret_cast<const __half*>(v_cache), max_ctx,
                                   reinterpret_cast<__half*>(out), workspace, (cudaStream_t)stream, kw, vw);
  if (e != cudaSuccess) return cuda_fail(e, who);
  return SQ_OK;
}

sq_status sq_attention(const void* qkv, int B, int T, int Hq, int Hkv, int D, const int32_t* pos0,
                       float theta, const void* k_cache, const void* v_cache, int64_t max_ctx, void* out,
                       void* workspace, size_t ws_bytes, sq_stream_t stream) {
  SQ_RANGE();
  return attention_common("sq_attention", qkv, B, T, Hq, Hkv, D, pos0, theta, k_cache, v_cache, max_ctx, out,
                          workspace, ws_bytes, false, stream);
}

sq_status sq_attention_append(const void* qkv, int B, int T, int Hq, int Hkv, int D, const int32_t* pos0,
                              float theta, void* k_cache, void* v_cache, int64_t max_ctx, void* out,
                              void* workspace, size_t ws_bytes, sq_stream_t stream) {
  SQ_RANGE();
  return attention_common("sq_attention_append", qkv, B, T, Hq, Hkv, D, pos0, theta, k_cache, v_cache,
                          max_ctx, out, workspace, ws_bytes, true, stream);
}

sq_status sq_kv_rollback(const int32_t* base, const int32_t* n_accepted, int B, int limit, int32_t* len,
                         sq_stream_t stream) {
  SQ_RANGE();
  if (B < 0 || limit < 0) return fail(SQ_ERR_SHAPE, "sq_kv_rollback: need B >= 0, limit >= 0");
  if (B == 0) return SQ_OK;
  if (!base || !n_accepted || !len) return fail(SQ_ERR_INVALID_ARG, "sq_kv_rollback: NULL pointer");
  if (!aligned(base, 4) || !aligned(n_accepted, 4) || !aligned(len, 4))
    return fail(SQ_ERR_ALIGN, "sq_kv_rollback: pointers must be 4-byte aligned");
  cudaError_t e = launch_kv_rollback(base, n_accepted, B, limit, len, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "sq_kv_rollback: launch");
  return SQ_OK;
}

sq_status sq_embed(const int32_t* ids, int M, int64_t ids_stride, const void* table, int64_t V, int64_t H,
                   void* out, sq_stream_t stream) {
  SQ_RANGE();
  if (M < 0 || V < 1 || H < 1 || ids_stride < 1)
    return fail(SQ_ERR_SHAPE, "sq_embed: need M >= 0, V >= 1, H >= 1, ids_stride >= 1");
  if (M == 0) return SQ_OK;
  if (!ids || !table || !out) return fail(SQ_ERR_INVALID_ARG, "sq_embed: NULL pointer");
  if (!aligned(ids, 4) || !aligned(table, 2) || !aligned(out, 2))
    return fail(SQ_ERR_ALIGN, "sq_embed: misaligned pointer");
  cudaError_t e = launch_embed(ids, M, ids_stride, reinterpret_cast<const __half*>(table), V, H,
                               reinterpret_cast<__half*>(out), (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "sq_embed: launch");
  return SQ_OK;
}

sq_status sq_spec_commit(const int32_t* n_accepted, const int32_t* tokens, int ldt, int B, int K, int32_t* hist,
                         int cap, int32_t* len, int32_t* pos, int32_t* last2, sq_stream_t stream) {
  SQ_RANGE();
  if (B < 0 || K < 0 || ldt < 1 || cap < 1)
    return fail(SQ_ERR_SHAPE, "sq_spec_commit: need B >= 0, K >= 0, ldt >= 1, cap >= 1");
  if (B == 0) return SQ_OK;
  if (!tokens || !hist || !len || !pos || !last2) return fail(SQ_ERR_INVALID_ARG, "sq_spec_commit: NULL pointer");
  if (!aligned(n_accepted, 4) || !aligned(tokens, 4) || !aligned(hist, 4) || !aligned(len, 4) ||
      !aligned(pos, 4) || !aligned(last2, 4))
    return fail(SQ_ERR_ALIGN, "sq_spec_commit: pointers must be 4-byte aligned");
  cudaError_t e = launch_spec_commit(n_accepted, tokens, ldt, B, K, hist, cap, len, pos, last2,
                                     (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "sq_spec_commit: launch");
  return SQ_OK;
}

sq_status sq_spec_drafts(const int32_t* samples, const int32_t* last2, int B, int K, int32_t* verify_tokens,
                         int32_t* draft, sq_stream_t stream) {
  SQ_RANGE();
  if (B < 0 || K < 0) return fail(SQ_ERR_SHAPE, "sq_spec_drafts: need B >= 0, K >= 0");
  if (B == 0) return SQ_OK;
  if (!last2 || !verify_tokens || (K > 0 && (!samples || !draft)))
    return fail(SQ_ERR_INVALID_ARG, "sq_spec_drafts: NULL pointer");
  if (!aligned(samples, 4) || !aligned(last2, 4) || !aligned(verify_tokens, 4) || !aligned(draft, 4))
    return fail(SQ_ERR_ALIGN, "sq_spec_drafts: pointers must be 4-byte aligned");
  cudaError_t e = launch_spec_drafts(samples, last2, B, K, verify_tokens, draft, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "sq_spec_drafts: launch");
  return SQ_OK;
}

// Same step as sq_accept for callers that cannot allocate device memory:
// the scratch is the library's own static device array (see sq_accept.cu).
// The ticket counters in it are cleared on the stream before each launch;
// nothing here allocates.
sq_status sq_accept_noalloc(const float* p, const float* q, const int32_t* draft, const float* u,
                            int B, int K, int64_t V, sq_accept_mode mode, int32_t* n_accepted,
                            int32_t* tokens, sq_stream_t stream) {
  SQ_RANGE();
  if (B < 0 || K < 0 || K > 16 || V < 1 || V >= ((int64_t)1 << 20))
    return fail(SQ_ERR_SHAPE, "sq_accept_noalloc: need B >= 0, 0 <= K <= 16, 1 <= V < 2^20 (B=%d K=%d V=%lld)",
                B, K, (long long)V);
  if (B == 0) return SQ_OK;
  if (!n_accepted) return fail(SQ_ERR_INVALID_ARG, "sq_accept_noalloc: NULL n_accepted");
  const size_t need = accept_workspace_bytes(B, K, V);
  if (need > kAcceptNoallocScratchBytes)
    return fail(SQ_ERR_SHAPE,
                "sq_accept_noalloc: B=%d K=%d V=%lld needs %zu bytes of scratch but the static scratch "
                "holds %zu; use sq_accept with a workspace, or fewer sequences per call",
                B, K, (long long)V, need, kAcceptNoallocScratchBytes);
  void* scratch = nullptr;
  cudaError_t e = accept_noalloc_scratch(&scratch);
  if (e != cudaSuccess) return cuda_fail(e, "sq_accept_noalloc: scratch address");
  // the counters are cleared only after accept_common has accepted every
  // argument: a rejected call queues nothing
  return accept_common("sq_accept_noalloc", p, q, draft, u, B, K, V, (int)mode, n_accepted, tokens,
                       scratch, kAcceptNoallocScratchBytes, stream, true);
}

}  // extern "C"
