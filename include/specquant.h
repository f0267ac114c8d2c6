/*
 * specquant.h -- C ABI of the GB300 (sm_103a) SpecQuant draft/verify hot path.
 *
 * Paper: "SpecQuant -- Speculative Decoding with Multi-Parent Quantization
 * for Adaptive LLM Inference".  One FP16 parent W16 gives an INT4 variant
 * Q4 = f(W16, 4) (Sec. III-A.1) and an FP8 variant Q8 = f(W16, 8)
 * (Sec. III-A.2).  The variants draft tokens (Sec. III-D.2), the parent
 * verifies the draft block in one pass (Sec. III-D.3), and the accept step
 * keeps the agreeing prefix and supplies the correction (Sec. III-A.3 token
 * rule, Sec. III-D.4).
 *
 * Conventions shared by every call
 *  - Every tensor pointer is a DEVICE pointer owned by the caller; the
 *    library allocates nothing in these calls and keeps no reference after
 *    the call returns.  Row-major, densely packed, no strides.
 *  - Every call is asynchronous and ordered on `stream` (NULL = the legacy
 *    default stream).  Kernels are launched with programmatic dependent
 *    launch allowed, so a linear call may start fetching its weights while
 *    the previous kernel on the stream finishes; it reads activations and
 *    writes outputs only after that kernel completed.  Consequence: the
 *    weights and scales of a linear call must not be written by the call
 *    issued immediately before it on the same stream if that call is a
 *    linear or accept call of this library (those let the next kernel start
 *    early).  Writes by sq_quantize, by copies and by other libraries'
 *    kernels are always complete first.
 *  - Return value: SQ_OK, or an error code whose text sq_last_error()
 *    returns (per host thread).  Arguments are validated on the host before
 *    anything is launched; an invalid call launches nothing.  No call traps,
 *    aborts or throws.
 *  - Data-dependent problems found on the device (a non-finite weight, a
 *    draft token outside [0, V), a resampling row without mass) set bits of
 *    a per-device status word that sq_check() reads and clears.
 *  - fp16 means IEEE binary16; E4M3 means the OCP FP8 E4M3 format.
 *  - Environment: SQ_PDL=0 launches without programmatic dependent launch
 *    (default: allowed on every stream but the legacy default stream).
 */
#ifndef SPECQUANT_H
#define SPECQUANT_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__) || defined(__clang__)
#define SQ_API __attribute__((visibility("default")))
#else
#define SQ_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* A CUDA runtime stream (cudaStream_t); declared here so that callers need
 * no CUDA header. */
typedef struct CUstream_st* sq_stream_t;

typedef enum {
  SQ_OK = 0,
  SQ_ERR_INVALID_ARG = 1,  /* NULL pointer, negative size, unknown enum   */
  SQ_ERR_SHAPE = 2,        /* sizes outside the documented limits         */
  SQ_ERR_ALIGN = 3,        /* pointer not 16-byte aligned where required  */
  SQ_ERR_UNSUPPORTED = 4,  /* valid request this build does not implement */
  SQ_ERR_WORKSPACE = 5,    /* workspace NULL or smaller than required     */
  SQ_ERR_CUDA = 6,         /* a CUDA runtime call failed (message says)   */
  SQ_ERR_DEVICE = 7        /* sq_check: the device flagged invalid data   */
} sq_status;

typedef enum { SQ_INT4_G128 = 1, SQ_FP8_E4M3_ROW = 2 } sq_qkind;
typedef enum { SQ_ACCEPT_SAMPLE = 0, SQ_ACCEPT_GREEDY = 1 } sq_accept_mode;

/* Device status bits reported through sq_check(). */
#define SQ_DEV_NONFINITE_WEIGHT 0x1u  /* sq_quantize saw a NaN or infinity  */
#define SQ_DEV_BAD_DRAFT_TOKEN  0x2u  /* sq_accept: draft token not in [0,V) */
#define SQ_DEV_NO_MASS          0x4u  /* sq_accept/sq_sample: row w/o mass   */
#define SQ_DEV_BAD_UNIFORM      0x8u  /* resampling uniform not in [0,1)     */
#define SQ_DEV_TIMEOUT          0x10u /* a kernel gave up a bounded wait     */
#define SQ_DEV_NONFINITE_LOGIT  0x20u /* a logit row held inf or NaN         */
#define SQ_DEV_BAD_POSITION     0x40u /* a token position outside the cache  */
#define SQ_DEV_BAD_TOKEN_ID     0x80u /* an embedding id outside [0, V)      */

/* Thread-local text of the last error raised on this host thread. */
SQ_API const char* sq_last_error(void);
/* Fixed name of a status code. */
SQ_API const char* sq_status_string(sq_status s);
/* Library version, major * 10000 + minor * 100 + patch. */
SQ_API int sq_version(void);

/* Synchronises `stream`, then reads and clears the device status word of
 * the current device.  Returns SQ_OK, SQ_ERR_DEVICE (bits in *device_bits,
 * which may be NULL) or SQ_ERR_CUDA. */
SQ_API sq_status sq_check(sq_stream_t stream, uint32_t* device_bits);

/* ------------------------------------------------------------------------
 * Sec. III-A.1 / III-A.2: derive the draft variants from the FP16 parent.
 *
 * sq_quantized_bytes: bytes of the code and scale buffers of a variant of
 * an [N, K] weight (scale_bytes may be NULL); 0 for an invalid request.
 *
 * sq_quantize: w16 fp16 [N, K] -> codes + scales.
 *   SQ_INT4_G128 (the paper fixes no scheme; this is symmetric RTN INT4):
 *     per row n and 128-wide group g along K: amax = max|w|,
 *     s = fp16(fp32(amax / 7)), s = 2^-24 if amax > 0 rounded s to zero,
 *     c = clamp(rint(fp32(w / s)), -8, 7) (ties to even), c = 0 if s = 0.
 *     codes: uint8 [N, K/2], byte j of a row holds k = 2j in its low nibble
 *     and k = 2j+1 in its high nibble, each as c + 8.
 *     scales: fp16 [N, K/128].  Requires K % 128 == 0.
 *   SQ_FP8_E4M3_ROW: s_n = fp32(amax_n / 448) (fp32 [N]),
 *     code = E4M3(fp32(w / s_n)) rounded to nearest even, saturating to
 *     +-448; code +0 for a row with s_n = 0.  codes: uint8 [N, K].
 *     Requires K % 16 == 0.
 *   Codes and scales are bit-identical to the definition above.  Alignment:
 *   w16, codes 16 B.  A non-finite weight sets SQ_DEV_NONFINITE_WEIGHT.
 * ---------------------------------------------------------------------- */
SQ_API size_t sq_quantized_bytes(sq_qkind kind, int64_t N, int64_t K, size_t* scale_bytes);
SQ_API sq_status sq_quantize(const void* w16, int64_t N, int64_t K, sq_qkind kind,
                      void* codes, void* scales, sq_stream_t stream);

/* ------------------------------------------------------------------------
 * Sec. III-D.2 (draft pass) / III-D.3 (verify pass): linear layers.
 *
 *   y[m, n] = sum_k x[m, k] * w'[n, k] (+ bias[n]),  m < M, n < N,
 * with w' the dequantised weight: c * s (INT4), s_n * E4M3(c) (FP8) or the
 * fp16 parent weight (sq_verify).  x: fp16 [M, K]; y: fp16 [M, N]; bias:
 * fp16 [N] or NULL.  Products are exact and sums are fp32; y is rounded to
 * nearest fp16 once.  1 <= M <= 256; N >= 1; K as for sq_quantize (INT4:
 * K % 128 == 0, FP8: K % 16 == 0, FP16: K % 8 == 0).  x, codes, w16 and y
 * must be 16-byte aligned.  Each call runs on one of these engines, chosen
 * from (format, M, N, K, epilogue) alone (sq_linear_path reports which):
 * the CUDA-core GEMV family for few rows (for one INT4 row over many output
 * rows, with its products on the tensor cores' register-operand path), the
 * shared-memory ring engine for one to eight rows of large or quantised
 * weights, and the tcgen05 tensor-core tile path from 16 rows on and, below
 * that, for the formats and shapes where it is faster.  All give the same
 * fp32-accumulated result up to summation order.
 * y must not overlap x, the weights or the scales.
 * ---------------------------------------------------------------------- */
SQ_API sq_status sq_linear_w4a16(const void* x, const void* codes, const void* scales,
                          const void* bias, void* y, int M, int64_t N, int64_t K,
                          sq_stream_t stream);
SQ_API sq_status sq_linear_fp8(const void* x, const void* codes, const float* scales,
                        const void* bias, void* y, int M, int64_t N, int64_t K,
                        sq_stream_t stream);
SQ_API sq_status sq_verify(const void* x, const void* w16, const void* bias, void* y,
                    int M, int64_t N, int64_t K, sq_stream_t stream);

/* Fused epilogues of the same three linear layers (the transformer block's
 * MLP, not specified by the paper).
 *  SQ_EPI_SILU_GATE: the weight holds 2N rows, rows [0, N) the gate and
 *    rows [N, 2N) the up projection; y[m, n] = silu(g) * u with
 *    g = x . w'[n], u = x . w'[N + n], silu(g) = g / (1 + exp(-g)), in fp32.
 *    bias (if any) has 2N entries.
 *  SQ_EPI_RESIDUAL: y[m, n] = residual[m, n] + x . w'[n] (+ bias[n]);
 *    residual fp16 [M, N]; it may be the same buffer as y (in place). */
typedef enum { SQ_EPI_NONE = 0, SQ_EPI_SILU_GATE = 1, SQ_EPI_RESIDUAL = 2 } sq_epilogue;
typedef enum { SQ_W_FP16 = 0, SQ_W_INT4 = 1, SQ_W_FP8 = 2 } sq_wkind;

/* Generic form of the three linear calls: wkind selects the weight format
 * (w = w16 for SQ_W_FP16, codes otherwise; scales NULL for SQ_W_FP16),
 * epi the epilogue.  residual is read only for SQ_EPI_RESIDUAL. */
SQ_API sq_status sq_linear_ex(sq_wkind wkind, const void* x, const void* w, const void* scales,
                       const void* bias, const void* residual, sq_epilogue epi, void* y,
                       int M, int64_t N, int64_t K, sq_stream_t stream);

/* sq_linear_norm: y = epi((rmsnorm(x) * gamma) W'^T + bias) -- the decoder's
 * pre-norm projections (q/k/v, gate/up, lm_head) in one call.  rmsnorm is
 * sq_rmsnorm's (fp32 arithmetic, the normalised rows rounded to fp16) and
 * the result is bit-identical to sq_rmsnorm followed by sq_linear_ex.  The
 * CUDA-core GEMV normalises the activation rows as it stages them (no extra
 * launch); the tensor-core path and the shared-memory ring engine write them
 * to xn (fp16 [M, K], 16-byte aligned, not aliasing x, y or the residual)
 * first.  gamma fp16 [K], 16-byte
 * aligned; eps >= 0. */
SQ_API sq_status sq_linear_norm(sq_wkind wkind, const void* x, const void* gamma, float eps, void* xn,
                                const void* w, const void* scales, const void* bias, const void* residual,
                                sq_epilogue epi, void* y, int M, int64_t N, int64_t K, sq_stream_t stream);

/* Engine sq_linear_ex would use for these sizes: 1 = tcgen05 tensor cores,
 * 0 = CUDA-core GEMV, 2 = one INT4 activation row over at least 192 16-row
 * output tiles with the products on the tensor cores' register-operand path
 * (mma.sync), 3 = one to eight activation rows streamed through a
 * shared-memory ring of asynchronous copies, products on the same
 * register-operand path,
 * -1 = sizes or kinds sq_linear_ex rejects (pointers are not examined;
 * nothing runs on the device).  The paper has no counterpart: this is
 * introspection for tests and tuning. */
SQ_API int sq_linear_path(sq_wkind wkind, int M, int64_t N, int64_t K, sq_epilogue epi);

/* Failure-path self-test (the paper has no counterpart).  Every wait inside
 * the library's kernels is bounded; a wait that runs out sets SQ_DEV_TIMEOUT
 * and the kernel finishes, so the device stays usable.  sq_selftest_wait
 * makes one such wait run out on purpose: a one-thread kernel waits on an
 * mbarrier that nothing ever arrives at, with nothing else in flight.
 *   which = 0: the poll-bounded wait of the tcgen05 tile path, giving up
 *              after `limit` polls (1 .. 2^24);
 *   which = 1: the time-bounded wait of the shared-memory ring engine,
 *              giving up after `limit` nanoseconds (1 .. 10^9).
 * The next sq_check() reports SQ_ERR_DEVICE with SQ_DEV_TIMEOUT set (and
 * clears it); the stream and the device stay usable.  Invalid arguments:
 * SQ_ERR_INVALID_ARG, nothing launched. */
SQ_API sq_status sq_selftest_wait(int which, uint64_t limit, sq_stream_t stream);

/* Sec. III-D.2 / III-D.3: a draft or verify pass runs every projection of
 * every layer plus lm_head, one after another.  sq_linear_chain runs `count`
 * linear calls in order on `stream` with exactly the results of calling
 * sq_linear_ex on each (an op may read what an earlier op wrote): one host
 * call per pass.  Every op is checked before the first launch; on an error
 * nothing is launched and sq_last_error names the op.  `ops` is host memory
 * read during the call only.  Each op follows sq_linear_ex's rules;
 * `reserved` must be 0. */
typedef struct sq_linear_op {
  sq_wkind wkind;        /* weight format */
  sq_epilogue epi;       /* epilogue */
  int M;                 /* activation rows */
  int reserved;          /* must be 0 */
  int64_t N, K;          /* output columns, inner size */
  const void* x;         /* fp16 [M, K] */
  const void* w;         /* codes, or fp16 [N or 2N, K] */
  const void* scales;    /* NULL for SQ_W_FP16 */
  const void* bias;      /* or NULL */
  const void* residual;  /* read only for SQ_EPI_RESIDUAL */
  void* y;               /* fp16 [M, N] */
} sq_linear_op;
SQ_API sq_status sq_linear_chain(const sq_linear_op* ops, int count, sq_stream_t stream);


/* ------------------------------------------------------------------------
 * Sec. III-A.3 token rule and Sec. III-D.4 acceptance / correction, for a
 * batch of B independent sequences with K draft tokens each over a
 * vocabulary of V tokens.
 *
 *   p      fp32 [B, K+1, V]  target (parent) probabilities, positions 0..K
 *   q      fp32 [B, K, V]    draft probabilities (NULL allowed when K == 0
 *                            or mode == SQ_ACCEPT_GREEDY)
 *   draft  int32 [B, K]      draft tokens
 *   u      fp32 [B, K+1]     uniforms in [0, 1): u[b, i] for the test of
 *                            draft i, u[b, K] for the correction/bonus draw
 *   n_accepted int32 [B], tokens int32 [B, K+1] (outputs)
 *
 * SQ_ACCEPT_SAMPLE (the lossless speculative-sampling rule the paper says
 * it follows, Sec. I): draft i is kept iff u_i * q_i(x_i) < p_i(x_i),
 * evaluated exactly; n = number kept before the first rejection.  The
 * correction token is drawn from r = max(0, p_n - q_n) (fp32 subtraction)
 * if n < K, else from r = p_K; if n < K and r has no mass, from p_n.  The
 * draw is a fixed-point inverse CDF: R_v = floor(r_v * 2^44),
 * S = sum_v R_v, T = floor(u_K * S), token = min{v : R_0 + .. + R_v > T};
 * every integer sum is exact, so the result does not depend on reduction
 * order and is bit-identical to the definition.
 * SQ_ACCEPT_GREEDY (the token rule read literally): draft i is kept iff it
 * equals argmax p_i (lowest index on ties); the correction is argmax p_n.
 *
 * tokens[b] = draft[b, 0..n-1], correction, then -1 up to K+1 entries;
 * n_accepted[b] = n.  A sequence with a draft token outside [0, V), a
 * correction uniform outside [0, 1) or a correction row without mass gets
 * n_accepted = -1 and all tokens -1, and sets the matching device status bit.
 *
 * Limits: B >= 0, 0 <= K <= 16, 1 <= V < 2^20.  p, q in [0, 1], finite
 * (rows need not sum to exactly 1).  Pointers 4-byte aligned (16 B for p
 * and q when V % 4 == 0 lets the kernel use vector loads).
 *
 * workspace: device memory of at least sq_accept_workspace_bytes(B, K, V)
 * bytes, 16-byte aligned.  It must be zero-filled before its first use; each
 * call leaves it zero-filled when it completes.  Calls that share one
 * workspace must not run concurrently on the GPU.
 * ---------------------------------------------------------------------- */
SQ_API size_t sq_accept_workspace_bytes(int B, int K, int64_t V);
SQ_API sq_status sq_accept(const float* p, const float* q, const int32_t* draft, const float* u,
                    int B, int K, int64_t V, sq_accept_mode mode,
                    int32_t* n_accepted, int32_t* tokens,
                    void* workspace, size_t ws_bytes, sq_stream_t stream);

/* Draft-side sampling, token[b] ~ probs[b, :] with uniform u[b]: the K = 0
 * case of sq_accept in sampling mode (same fixed-point inverse CDF, same
 * workspace rules, workspace size sq_accept_workspace_bytes(B, 0, V)). */
SQ_API sq_status sq_sample(const float* probs, const float* u, int B, int64_t V, int32_t* tokens,
                    void* workspace, size_t ws_bytes, sq_stream_t stream);

/* ------------------------------------------------------------------------
 * Sec. III-D.4 from logits: the same accept / reject / resample step, with
 * the probabilities computed inside the library from the lm_head outputs
 * instead of read from memory (no [B, K+1, V] fp32 array is written).
 *
 *   zp  fp16 [B, K+1, V]  target logits (row b (K+1) + i: sequence b,
 *                         position i: the verify pass's lm_head output)
 *   zq  fp16 [K, B, V]    draft logits (block i: the lm_head output of draft
 *                         step i for all B sequences; NULL allowed when
 *                         K == 0)
 *   temperature T > 0 and finite.
 *
 * p_i = softmax(zp[b, i, :] / T), q_i = softmax(zq[i, b, :] / T), each row
 * computed exactly as
 *   m = max_v z_v,  invT = 1/T (fp32),  e_v = exp_neg((z_v - m) * invT),
 *   S = sum_v floor(e_v * 2^40) (64-bit integer),  s = (float)(S * 2^-40),
 *   p_v = e_v / s (fp32 division),
 * where exp_neg(x) (x <= 0) is a Cody-Waite reduction by ln 2 (16-bit head
 * plus tail) and a degree-7 Taylor polynomial evaluated with fused
 * multiply-adds, scaled by 2^n, and 0 for x <= -104; every step is an IEEE
 * fp32 operation rounded to nearest, so the probabilities are bit-identical
 * to this definition.  Everything after that is sq_accept on these rows
 * (both modes; greedy takes argmax p).  A sequence with a non-finite logit in
 * any of its 2K+1 rows gets n_accepted = -1 and all tokens -1, and sets
 * SQ_DEV_NONFINITE_LOGIT.  Pointers: zp, zq 2-byte aligned, the rest as for
 * sq_accept.  workspace: sq_accept_logits_workspace_bytes(B, K, V) bytes,
 * 16-byte aligned, zero-filled before first use (each call leaves it so);
 * calls sharing a workspace must not overlap on the GPU. */
SQ_API size_t sq_accept_logits_workspace_bytes(int B, int K, int64_t V);
SQ_API sq_status sq_accept_logits(const void* zp, const void* zq, const int32_t* draft,
                                  const float* u, int B, int K, int64_t V, float temperature,
                                  sq_accept_mode mode, int32_t* n_accepted, int32_t* tokens,
                                  void* workspace, size_t ws_bytes, sq_stream_t stream);
/* Draft-side sampling from logits: token[b] ~ softmax(z[b, :] / T) with
 * uniform u[b] (the K = 0 case of sq_accept_logits; z fp16 [B, V];
 * workspace sq_accept_logits_workspace_bytes(B, 0, V)). */
SQ_API sq_status sq_sample_logits(const void* z, const float* u, int B, int64_t V,
                                  float temperature, int32_t* tokens, void* workspace,
                                  size_t ws_bytes, sq_stream_t stream);

/* The probabilities of sq_accept_logits on their own: p[r, :] =
 * softmax(z[r, :] / T) for R rows of fp16 logits z [R, V] into fp32 p [R, V],
 * by the definition above (bit-identical to it); a row holding a non-finite
 * logit gives NaN and sets SQ_DEV_NONFINITE_LOGIT.  workspace:
 * sq_softmax_workspace_bytes(R, V) bytes, 16-byte aligned, zero-filled
 * before first use (each call leaves it so). */
SQ_API size_t sq_softmax_workspace_bytes(int64_t R, int64_t V);
SQ_API sq_status sq_softmax(const void* z, int64_t R, int64_t V, float temperature, float* p,
                            void* workspace, size_t ws_bytes, sq_stream_t stream);

/* ------------------------------------------------------------------------
 * The decoder around the linear stack.  Sec. III-D.2/3 run the whole model
 * for draft and verify; Sec. III-D.4 restarts from the first rejected
 * token, so each model's KV cache keeps only the accepted prefix.  The
 * paper gives no model internals; these follow the Qwen2.5 decoder:
 *
 * sq_rmsnorm: y[m, :] = x[m, :] / sqrt(mean(x[m, :]^2) + eps) * gamma, fp32
 *   arithmetic, fp16 x, gamma [H], y [M, H] (y may equal x).
 *
 * Attention layout: qkv fp16 [B*T, (Hq + 2 Hkv) * D], the fused q/k/v
 * projection's output for T new tokens of each of B sequences (row b*T + t:
 * q heads, then k heads, then v heads); D = 128; Hq a multiple of Hkv; token
 * t of sequence b is at position pos0[b] + t (pos0 int32 [B], device).
 * Caches k_cache, v_cache fp16 [B, Hkv, max_ctx, D], 16-byte aligned.  RoPE rotates pairs
 * (d, d + D/2) by pos * theta^(-2d/D) (angle computed in fp64).
 *
 * sq_kv_append: rotates the new keys and writes keys and values into the
 *   caches at their positions.  A position outside [0, max_ctx) writes
 *   nothing and sets SQ_DEV_BAD_POSITION.
 * sq_attention: out fp16 [B*T, Hq * D]: for query head h of token t,
 *   softmax_j(q . k_j / sqrt(D)) v_j over cache positions j <= pos0[b] + t
 *   of key/value head h / (Hq / Hkv), q rotated at its position; the keys
 *   of the current tokens must already be appended.  Accumulation in fp32.
 *   T <= 32, (Hq / Hkv) * T <= 200, max_ctx <= 2^17.  workspace: sq_attention_workspace_bytes(...)
 *   bytes, 16-byte aligned (no zero-fill needed).
 * sq_kv_rollback: len[b] = base[b] + min(n_accepted[b] + 1, limit), or
 *   base[b] when n_accepted[b] < 0 (the cache length to keep after
 *   acceptance: the verified prefix plus the accepted drafts); int32
 *   device arrays. */
SQ_API sq_status sq_rmsnorm(const void* x, const void* gamma, int M, int64_t H, float eps, void* y,
                            sq_stream_t stream);
SQ_API sq_status sq_kv_append(const void* qkv, int B, int T, int Hq, int Hkv, int D,
                              const int32_t* pos0, float theta, void* k_cache, void* v_cache,
                              int64_t max_ctx, sq_stream_t stream);
SQ_API size_t sq_attention_workspace_bytes(int B, int T, int Hq, int Hkv, int D, int64_t max_ctx);
SQ_API sq_status sq_attention(const void* qkv, int B, int T, int Hq, int Hkv, int D,
                              const int32_t* pos0, float theta, const void* k_cache,
                              const void* v_cache, int64_t max_ctx, void* out, void* workspace,
                              size_t ws_bytes, sq_stream_t stream);
/* sq_attention_append: sq_kv_append followed by sq_attention in one launch
 * (same arguments; the caches are written): the cache chunk that holds a
 * new token's position rotates its key from qkv, writes key and value, and
 * attends to them directly.  Caches and output are bit-identical to the two
 * calls.  A position outside [0, max_ctx) writes nothing, sets
 * SQ_DEV_BAD_POSITION and leaves the sequence's output rows zero. */
SQ_API sq_status sq_attention_append(const void* qkv, int B, int T, int Hq, int Hkv, int D,
                                     const int32_t* pos0, float theta, void* k_cache, void* v_cache,
                                     int64_t max_ctx, void* out, void* workspace, size_t ws_bytes,
                                     sq_stream_t stream);
SQ_API sq_status sq_kv_rollback(const int32_t* base, const int32_t* n_accepted, int B, int limit,
                                int32_t* len, sq_stream_t stream);
/* sq_embed: out[m, :] = table[ids[m * ids_stride], :] for M token ids
 * (int32, device), table fp16 [V, H], out fp16 [M, H]; an id outside [0, V)
 * gives a zero row and sets SQ_DEV_BAD_TOKEN_ID.  This is how accepted and
 * drafted tokens re-enter the model (the same call gathers rows of any
 * [rows, H] fp16 matrix).
 *
 * Speculative bookkeeping on the device, so that a whole draft / verify /
 * accept cycle runs without the host (Sec. III-D.4: the accepted prefix plus
 * the correction token is the context the next cycle starts from).  Per
 * sequence b: hist int32 [B, cap] holds the committed tokens, len[b] of them.
 *
 * sq_spec_commit: appends tokens[b, 0 .. n] (n = n_accepted[b], or 0 when
 *   n_accepted is NULL; row stride ldt; nothing when n < 0) to hist[b] and
 *   adds them to len[b]; then, with L the new length, writes the next
 *   cycle's positions pos int32 [K + 1, B]: pos[0, b] = L - 2 (the first
 *   draft step feeds the last two committed tokens, T = 2), pos[k, b] =
 *   L - 1 + k for draft steps k = 1 .. K-1 (T = 1), pos[K, b] = L - 1 (the
 *   verify pass, T = K + 1; with K = 0 this is direct decoding); and
 *   last2 int32 [B, 2] = (hist[b, L-2], hist[b, L-1]).  An overfull history,
 *   n >= ldt, a length outside [0, cap] or L < 2 sets SQ_DEV_BAD_POSITION
 *   (missing tokens read as -1).
 * sq_spec_drafts: verify_tokens int32 [B, K+1] = (last2[b, 1], samples[0,b],
 *   .., samples[K-1, b]) and draft int32 [B, K] = samples^T, from the K
 *   draft steps' tokens samples int32 [K, B]. */
SQ_API sq_status sq_embed(const int32_t* ids, int M, int64_t ids_stride, const void* table, int64_t V,
                          int64_t H, void* out, sq_stream_t stream);
SQ_API sq_status sq_spec_commit(const int32_t* n_accepted, const int32_t* tokens, int ldt, int B, int K,
                                int32_t* hist, int cap, int32_t* len, int32_t* pos, int32_t* last2,
                                sq_stream_t stream);
SQ_API sq_status sq_spec_drafts(const int32_t* samples, const int32_t* last2, int B, int K,
                                int32_t* verify_tokens, int32_t* draft, sq_stream_t stream);

/* ------------------------------------------------------------------------
 * sq_accept_noalloc: sq_accept without a caller workspace.  The paper has
 * no counterpart; it exists for callers that cannot allocate device memory
 * where they run the accept step -- code inside a host framework that owns
 * every device byte through its own pool and does not let components call
 * cudaMalloc, or a latency-critical loop where an allocation (which may
 * synchronise the device) is not acceptable.
 *
 * Same arguments, semantics, limits and results as sq_accept, minus the
 * workspace.  The scratch is a static device array inside the library of
 * SQ_ACCEPT_NOALLOC_SCRATCH_BYTES (1 MiB); every GPU that loads the library
 * holds it until the process exits.  A call whose
 * sq_accept_workspace_bytes(B, K, V) exceeds that size is rejected with
 * SQ_ERR_SHAPE (e.g. V = 152064 with K = 4 fits up to B = 349).  The call clears
 * the ticket counters in the scratch on `stream` before launching and never
 * calls cudaMalloc, cudaFree or any allocating routine.
 *
 * Every call on a device shares the one scratch array, which keeps the last
 * call's contents: calls that overlap on the GPU (two streams, two host
 * threads) race and give wrong results; serialise them.
 * The first call on a device looks up the scratch's device address (once per
 * device, with that device current); make that first call before any stream
 * capture begins.
 * ---------------------------------------------------------------------- */
#define SQ_ACCEPT_NOALLOC_SCRATCH_BYTES ((size_t)1 << 20)
SQ_API sq_status sq_accept_noalloc(const float* p, const float* q, const int32_t* draft,
                                   const float* u, int B, int K, int64_t V, sq_accept_mode mode,
                                   int32_t* n_accepted, int32_t* tokens, sq_stream_t stream);

#ifdef __cplusplus
}
#endif
#endif
