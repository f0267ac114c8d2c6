/*
 * sq_oracle.h -- CPU oracle for the SpecQuant draft/verify hot path.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test suite, the package's smoke check
 * and the benchmark's CPU-baseline leg may load this code.  The GPU product
 * path never calls it, links it or falls back to it.  It shares no header,
 * helper, table or constant with the CUDA library: every definition below is
 * written out from the paper and from the number-format standards it leans on.
 *
 * Paper: "SpecQuant -- Speculative Decoding with Multi-Parent Quantization
 * for Adaptive LLM Inference".  Section references are to that paper:
 *   Sec. III-A.1  low-precision parent  Q4  = f(W16, 4)
 *   Sec. III-A.2  medium-precision parent Q8 = f(W16, 8)
 *   Sec. III-A.3  full-precision parent Q16 = W16, and the token rule
 *                 y_t = y_t^draft if the parent agrees, else f(x_{1:t-1})
 *   Sec. III-D.2  draft generation, Sec. III-D.3 parent verification,
 *   Sec. III-D.4  token acceptance or correction
 *   Sec. I / II-A adherence to standard speculative decoding
 *
 * The paper fixes neither the quantisation scheme nor the sampling rule.
 * The readings implemented here (symmetric INT4 with group 128 along K and
 * fp16 scales, FP8-E4M3 with one fp32 scale per output row, the lossless
 * speculative-sampling accept rule with a 2^-44 fixed-point CDF) are listed
 * next to each function.
 *
 * Parity pins: every function here is checked by tests against something
 * other than itself (library casts, brute force, exact rational arithmetic,
 * exhaustive enumeration of the accept rule over the uniform grid).
 */
#ifndef SQ_ORACLE_H
#define SQ_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Status codes returned by the oracle (its own numbering). */
#define OQ_OK 0
#define OQ_BAD_ARG 1     /* shape not allowed, non-finite weight, ... */
#define OQ_BAD_SEQ 2     /* at least one sequence was invalid (see oq_accept) */

/* ---- number formats ------------------------------------------------------ */

/* IEEE 754 binary16: bits -> exact value. */
double oq_f16_decode(uint16_t h);
/* Nearest binary16 to x, ties to the even bit pattern, overflow to +-inf. */
uint16_t oq_f16_encode(double x);
/* OCP FP8 E4M3 (bias 7, no infinities, S.1111.111 = NaN): bits -> value. */
double oq_e4m3_decode(uint8_t c);
/* Nearest E4M3 to x, ties to even mantissa, finite overflow saturates to
 * +-448 ("satfinite"), sign of zero kept, NaN -> 0x7F. */
uint8_t oq_e4m3_encode(double x);

void oq_f16_decode_array(const uint16_t* h, int64_t n, double* out);
void oq_f16_encode_array(const double* x, int64_t n, uint16_t* out);
void oq_e4m3_encode_array(const float* x, int64_t n, uint8_t* out);

/* ---- Sec. III-A.1: Q4 = f(W16, 4) ---------------------------------------- */
/* w16 [N,K] fp16 row-major -> codes [N,K/2] (low nibble = even k, value
 * c+8), scales [N,K/128] fp16 bits.  K % 128 == 0. */
int oq_quantize_int4(const uint16_t* w16, int64_t N, int64_t K,
                     uint8_t* codes, uint16_t* scales);
/* codes/scales -> exact dequantised weights c*s as double [N,K]. */
int oq_dequant_int4(const uint8_t* codes, const uint16_t* scales,
                    int64_t N, int64_t K, double* w);

/* ---- Sec. III-A.2: Q8 = f(W16, 8) ---------------------------------------- */
/* w16 [N,K] -> codes [N,K] E4M3 bits, scales [N] fp32 (amax_n / 448). */
int oq_quantize_fp8(const uint16_t* w16, int64_t N, int64_t K,
                    uint8_t* codes, float* scales);
int oq_dequant_fp8(const uint8_t* codes, const float* scales,
                   int64_t N, int64_t K, double* w);

/* ---- Sec. III-D.2/3: the linear layers of draft and verify passes -------- */
/* y[M,N] = x[M,K] . w[N,K]^T (+ bias[N]), every product and sum in fp64. */
void oq_linear(const double* x, const double* w, const double* bias,
               int64_t M, int64_t N, int64_t K, double* y);
/* h = silu(g) * u elementwise, silu(g) = g / (1 + exp(-g)), fp64. */
void oq_silu_gate(const double* g, const double* u, int64_t n, double* h);

/* ---- Sec. III-A.3 token rule and Sec. III-D.4 acceptance ------------------ */
#define OQ_ACCEPT_SAMPLE 0
#define OQ_ACCEPT_GREEDY 1
/* floor(r * 2^44) for a finite r in [0, 1]. */
uint64_t oq_fix44(float r);
/* floor(u * S) for u in [0, 1), computed exactly. */
uint64_t oq_scale_floor(float u, uint64_t S);
/* p [B,K+1,V], q [B,K,V] (may be NULL when K == 0), draft [B,K],
 * u [B,K+1] -> n_accepted [B], tokens [B,K+1] (-1 padded).
 * A sequence whose draft token is outside [0,V), whose last uniform is
 * outside [0,1), or whose resampling row has zero fixed-point mass gets
 * n_accepted = -1 and all tokens -1; the call then returns OQ_BAD_SEQ. */
int oq_accept(const float* p, const float* q, const int32_t* draft,
              const float* u, int64_t B, int64_t K, int64_t V, int mode,
              int32_t* n_accepted, int32_t* tokens);
/* Draft-side sampling: token[b] ~ probs[b,:] by the same fixed-point
 * inverse CDF (the K = 0 case of oq_accept in sampling mode). */
int oq_sample(const float* probs, const float* u, int64_t B, int64_t V,
              int32_t* tokens);

/* ---- probabilities from logits (softmax with temperature) ------------------
 * The paper's parents emit next-token distributions (Sec. III-D.2/3); a
 * decoder's lm_head emits logits z, and p = softmax(z / T).  The paper fixes
 * no arithmetic for it; the definition implemented here is exactly
 * reproducible in IEEE fp32 on any machine:
 *   m    = max_v z_v (fp16 logits, exact in fp32)
 *   invT = 1 / T (fp32 division)
 *   e_v  = exp_neg((z_v - m) * invT)        (fp32 subtract, then multiply)
 *   S    = sum_v floor(e_v * 2^40)          (64-bit integer, order-free)
 *   s    = (float)((double)S * 2^-40)
 *   p_v  = e_v / s                          (fp32 division)
 * exp_neg(x) for x <= 0: Cody-Waite reduction x = n ln2 + r (ln 2 split in
 * a 16-bit head and a tail so n * head is exact), e^r by its degree-7
 * Taylor polynomial in Horner form with fused multiply-adds, then the
 * exact scaling by 2^n (through 2^(n+64) * 2^-64 below 2^-126); 0 for
 * x <= -104 (below the smallest subnormal). */
float oq_exp_neg(float x);
void oq_exp_neg_array(const float* x, int64_t n, float* out);
/* One row: z [V] fp16 bit patterns, T > 0 -> p [V].  OQ_BAD_ARG for V < 1,
 * T not a positive finite number, or a non-finite logit. */
int oq_softmax_row(const uint16_t* z, int64_t V, float T, float* p);
/* Sec. III-D.4 from logits: zp [B,K+1,V] (target, position-major per
 * sequence), zq [K,B,V] (draft, one [B,V] block per draft step); p and q
 * rows by oq_softmax_row, then exactly oq_accept. */
int oq_accept_logits(const uint16_t* zp, const uint16_t* zq, const int32_t* draft,
                     const float* u, int64_t B, int64_t K, int64_t V, float T,
                     int mode, int32_t* n_accepted, int32_t* tokens);
/* Draft-side sampling from logits: token[b] ~ softmax(z[b,:] / T). */
int oq_sample_logits(const uint16_t* z, const float* u, int64_t B, int64_t V,
                     float T, int32_t* tokens);

/* ---- the decoder around the linear stack (attention, KV cache) -----------
 * Sec. III-D.2/3 run the full model; Sec. III-D.4 rolls the parent's state
 * back to the first rejected token ("recommence ... starting with the first
 * token that was rejected").  The paper states no model internals; these
 * follow the Qwen2.5 decoder the workloads are shaped after, in fp64:
 *   RMSNorm   y = x / sqrt(mean(x^2) + eps) * gamma
 *   RoPE      for d < D/2, f_d = theta^(-2d/D), a = pos * f_d:
 *             (x_d, x_{d+D/2}) -> (x_d cos a - x_{d+D/2} sin a,
 *                                   x_{d+D/2} cos a + x_d sin a)
 *   attention out_h = softmax_j(q_h . k_j / sqrt(D)) v_j over the cache
 *             positions j <= pos of the query, key/value head h / (Hq/Hkv)
 *             (grouped-query attention). */
/* x, y [M, H] (x values), gamma [H]. */
void oq_rmsnorm(const double* x, const double* gamma, int64_t M, int64_t H, double eps, double* y);
/* In place on rows [M, nheads * D] at positions pos[M]. */
void oq_rope(double* x, const int64_t* pos, int64_t M, int64_t nheads, int64_t D, double theta);
/* q [T, Hq, D] already rotated, k and v [L, Hkv, D] (k rotated), query t at
 * position qpos[t] sees keys j <= qpos[t] (j < L) -> out [T, Hq, D]. */
void oq_attention(const double* q, const double* k, const double* v, const int64_t* qpos,
                  int64_t T, int64_t L, int64_t Hq, int64_t Hkv, int64_t D, double* out);

/* ---- exhaustive-enumeration harness (sq_enumerate.c) --------------------- */
/* Runs oq_accept on one sequence 2^grid_bits times, with the uniform at
 * position `pos` set to m * 2^-grid_bits for every m, the others taken from
 * u_fixed, and histograms the outcome: hist[n * V + token_at_n] counts,
 * hist[(K+1)*V] counts invalid outcomes. */
int oq_enum_sweep(const float* p, const float* q, const int32_t* draft,
                  const float* u_fixed, int64_t K, int64_t V, int mode,
                  int pos, int grid_bits, uint64_t* hist);

#ifdef __cplusplus
}
#endif
#endif
