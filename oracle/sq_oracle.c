/*
 * sq_oracle.c -- plain, slow, obviously correct CPU oracle.
 *
 * TEST INFRASTRUCTURE ONLY (tests, smoke check, CPU-baseline timing).
 * Built with -ffp-contract=off and without fast-math so that every float
 * operation is the single IEEE operation written, on x86-64 and AArch64.
 * All accumulation is fp64.  No blocking, fusion or reordering beyond the
 * definitions quoted at each function.
 */
#include "sq_oracle.h"

#include <math.h>
#include <stddef.h>
#include <stdlib.h>
#include <string.h>

/* ======================================================================== */
/* Number formats                                                            */
/* ======================================================================== */

/* IEEE 754 binary16: 1 sign bit, 5 exponent bits (bias 15), 10 fraction
 * bits.  Exponent field 0 holds zero and subnormals f * 2^-24. */
double oq_f16_decode(uint16_t h) {
  int sign = (h >> 15) & 1;
  int e = (h >> 10) & 0x1f;
  int f = h & 0x3ff;
  double v;
  if (e == 0) {
    v = ldexp((double)f, -24);
  } else if (e == 31) {
    v = f ? NAN : INFINITY;
  } else {
    v = ldexp((double)(1024 + f), e - 25);
  }
  return sign ? -v : v;
}

/* Round-to-nearest-even written as its definition: among the finite
 * non-negative patterns 0 .. last (whose values increase with the pattern),
 * find the largest pattern whose value does not exceed a, then pick the
 * nearer of it and the next one; on a tie pick the even pattern (the even
 * least significant mantissa bit).  `above_last` is the value one step
 * past the last finite pattern, used only to decide the final interval. */
typedef double (*oq_decode_fn)(uint32_t);

static double dec16(uint32_t h) { return oq_f16_decode((uint16_t)h); }

static uint32_t round_to_table(double a, uint32_t last, double above_last,
                               oq_decode_fn dec) {
  uint32_t lo = 0, hi = last; /* invariant: dec(lo) <= a */
  if (a >= dec(last)) {
    lo = last;
  } else {
    while (hi - lo > 1) {
      uint32_t mid = lo + (hi - lo) / 2;
      if (dec(mid) <= a) lo = mid; else hi = mid;
    }
  }
  double v0 = dec(lo);
  if (v0 == a) return lo;
  double v1 = (lo == last) ? above_last : dec(lo + 1);
  double d0 = a - v0, d1 = v1 - a; /* exact: all values are short dyadics */
  if (d0 < d1) return lo;
  if (d1 < d0) return lo + 1;
  return (lo & 1u) ? lo + 1 : lo;
}

uint16_t oq_f16_encode(double x) {
  if (isnan(x)) return 0x7e00;
  uint16_t sign = signbit(x) ? 0x8000 : 0;
  double a = fabs(x);
  /* 0x7bff = 65504 is the largest finite value; 65536 would be the next
   * step, so pattern 0x7c00 (infinity) is the "one past the last" result. */
  uint32_t r = round_to_table(a, 0x7bff, 65536.0, dec16);
  if (r > 0x7bff) r = 0x7c00;
  return (uint16_t)(sign | r);
}

/* OCP 8-bit floating point, E4M3: 1 sign bit, 4 exponent bits (bias 7),
 * 3 mantissa bits; exponent field 0 holds zero and subnormals m * 2^-9;
 * S.1111.111 is NaN; no infinities; largest finite 1.75 * 2^8 = 448. */
double oq_e4m3_decode(uint8_t c) {
  int sign = (c >> 7) & 1;
  int e = (c >> 3) & 0xf;
  int m = c & 7;
  double v;
  if (e == 15 && m == 7) return NAN;
  if (e == 0) v = ldexp((double)m, -9);
  else v = ldexp((double)(8 + m), e - 10);
  return sign ? -v : v;
}

static double dec8(uint32_t c) { return oq_e4m3_decode((uint8_t)c); }

uint8_t oq_e4m3_encode(double x) {
  if (isnan(x)) return 0x7f;
  uint8_t sign = signbit(x) ? 0x80 : 0;
  double a = fabs(x);
  /* satfinite: every magnitude at or above the largest finite value maps
   * to it (448 = pattern 0x7e). */
  if (a >= 448.0) return (uint8_t)(sign | 0x7e);
  uint32_t r = round_to_table(a, 0x7e, 480.0, dec8);
  if (r > 0x7e) r = 0x7e;
  return (uint8_t)(sign | r);
}

void oq_f16_decode_array(const uint16_t* h, int64_t n, double* out) {
  for (int64_t i = 0; i < n; ++i) out[i] = oq_f16_decode(h[i]);
}

void oq_f16_encode_array(const double* x, int64_t n, uint16_t* out) {
  for (int64_t i = 0; i < n; ++i) out[i] = oq_f16_encode(x[i]);
}

void oq_e4m3_encode_array(const float* x, int64_t n, uint8_t* out) {
  for (int64_t i = 0; i < n; ++i) out[i] = oq_e4m3_encode((double)x[i]);
}

/* ======================================================================== */
/* Sec. III-A.1: Q4 = f(W16, 4)                                             */
/* ======================================================================== */
/* Reading (the paper names no scheme): symmetric round-to-nearest INT4 with
 * one fp16 scale per 128 consecutive weights of a row.  Per row n and group
 * g:  amax = max |w|;  s = fp16(fp32(amax / 7));  if amax > 0 and s rounded
 * to zero, s = 2^-24;  c = clamp(rint(fp32(w / s)), -8, 7);  c = 0 when
 * s = 0.  Stored: nibble c + 8, even k in the low nibble. */
#define OQ_G 128

int oq_quantize_int4(const uint16_t* w16, int64_t N, int64_t K,
                     uint8_t* codes, uint16_t* scales) {
  if (N < 0 || K <= 0 || K % OQ_G != 0) return OQ_BAD_ARG;
  const int64_t G = K / OQ_G;
  for (int64_t i = 0; i < N * K; ++i)
    if (!isfinite(oq_f16_decode(w16[i]))) return OQ_BAD_ARG;
  for (int64_t n = 0; n < N; ++n) {
    for (int64_t g = 0; g < G; ++g) {
      const uint16_t* wg = w16 + n * K + g * OQ_G;
      float amax = 0.0f;
      for (int j = 0; j < OQ_G; ++j) {
        float a = (float)fabs(oq_f16_decode(wg[j]));
        if (a > amax) amax = a;
      }
      float s32 = amax / 7.0f;
      uint16_t sh = oq_f16_encode((double)s32);
      if (amax > 0.0f && sh == 0) sh = 0x0001;
      scales[n * G + g] = sh;
      float s = (float)oq_f16_decode(sh);
      for (int j = 0; j < OQ_G; ++j) {
        int c = 0;
        if (s != 0.0f) {
          float w = (float)oq_f16_decode(wg[j]);
          float t = rintf(w / s);
          if (t < -8.0f) t = -8.0f;
          if (t > 7.0f) t = 7.0f;
          c = (int)t;
        }
        int64_t k = g * OQ_G + j;
        uint8_t nib = (uint8_t)(c + 8);
        uint8_t* byte = codes + n * (K / 2) + k / 2;
        if ((k & 1) == 0) *byte = (uint8_t)((*byte & 0xf0) | nib);
        else *byte = (uint8_t)((*byte & 0x0f) | (nib << 4));
      }
    }
  }
  return OQ_OK;
}

int oq_dequant_int4(const uint8_t* codes, const uint16_t* scales,
                    int64_t N, int64_t K, double* w) {
  if (N < 0 || K <= 0 || K % OQ_G != 0) return OQ_BAD_ARG;
  const int64_t G = K / OQ_G;
  for (int64_t n = 0; n < N; ++n) {
    for (int64_t k = 0; k < K; ++k) {
      uint8_t byte = codes[n * (K / 2) + k / 2];
      int nib = (k & 1) ? (byte >> 4) : (byte & 0x0f);
      double s = oq_f16_decode(scales[n * G + k / OQ_G]);
      w[n * K + k] = (double)(nib - 8) * s;
    }
  }
  return OQ_OK;
}

/* ======================================================================== */
/* Sec. III-A.2: Q8 = f(W16, 8)                                             */
/* ======================================================================== */
/* Reading: FP8-E4M3 codes with one fp32 scale per output row.
 * s_n = fp32(amax_n / 448);  code = e4m3_satfinite(fp32(w / s_n));
 * code = +0 when s_n = 0. */
int oq_quantize_fp8(const uint16_t* w16, int64_t N, int64_t K,
                    uint8_t* codes, float* scales) {
  if (N < 0 || K <= 0) return OQ_BAD_ARG;
  for (int64_t i = 0; i < N * K; ++i)
    if (!isfinite(oq_f16_decode(w16[i]))) return OQ_BAD_ARG;
  for (int64_t n = 0; n < N; ++n) {
    const uint16_t* wr = w16 + n * K;
    float amax = 0.0f;
    for (int64_t k = 0; k < K; ++k) {
      float a = (float)fabs(oq_f16_decode(wr[k]));
      if (a > amax) amax = a;
    }
    float s = amax / 448.0f;
    scales[n] = s;
    for (int64_t k = 0; k < K; ++k) {
      uint8_t c = 0;
      if (s != 0.0f) {
        float w = (float)oq_f16_decode(wr[k]);
        c = oq_e4m3_encode((double)(w / s));
      }
      codes[n * K + k] = c;
    }
  }
  return OQ_OK;
}

int oq_dequant_fp8(const uint8_t* codes, const float* scales,
                   int64_t N, int64_t K, double* w) {
  if (N < 0 || K <= 0) return OQ_BAD_ARG;
  for (int64_t n = 0; n < N; ++n)
    for (int64_t k = 0; k < K; ++k)
      w[n * K + k] = (double)scales[n] * oq_e4m3_decode(codes[n * K + k]);
  return OQ_OK;
}

/* ======================================================================== */
/* Sec. III-D.2 / III-D.3: linear layers of the draft and verify passes      */
/* ======================================================================== */
/* y = x W^T (+ b): the textbook dot product, in fp64. */
void oq_linear(const double* x, const double* w, const double* bias,
               int64_t M, int64_t N, int64_t K, double* y) {
  for (int64_t m = 0; m < M; ++m) {
    for (int64_t n = 0; n < N; ++n) {
      double acc = 0.0;
      for (int64_t k = 0; k < K; ++k) acc += x[m * K + k] * w[n * K + k];
      if (bias) acc += bias[n];
      y[m * N + n] = acc;
    }
  }
}

/* SiLU-gated MLP input (the gate/up pair of a Qwen2.5 MLP block). */
void oq_silu_gate(const double* g, const double* u, int64_t n, double* h) {
  for (int64_t i = 0; i < n; ++i) h[i] = g[i] / (1.0 + exp(-g[i])) * u[i];
}

/* ======================================================================== */
/* Sec. III-A.3 token rule, Sec. III-D.4 acceptance / correction             */
/* ======================================================================== */
/* Sampling mode (the standard lossless speculative-sampling rule the paper
 * says it adheres to, Sec. I):
 *   draft i (0-based) is accepted iff  u_i * q_i(x_i) < p_i(x_i)  (exact in
 *   fp64); n = number accepted before the first rejection.
 *   Correction row r: max(0, p_n - q_n) (fp32 subtraction) when n < K,
 *   otherwise p_K (the bonus position).  If n < K and r has no fixed-point
 *   mass, r = p_n.
 *   Fixed-point inverse CDF: R_v = floor(r_v 2^44), S = sum R_v,
 *   T = floor(u_K * S), token = min { v : R_0 + ... + R_v > T }.
 * Greedy mode (the paper's rule read literally, "if parent agrees"):
 *   accept iff x_i = argmax p_i (lowest index on ties); correction token
 *   argmax p_n. */

uint64_t oq_fix44(float r) {
  /* r * 2^44 is exact in double (power-of-two scaling of a 24-bit
   * significand) and below 2^53, so floor is exact. */
  return (uint64_t)floor(ldexp((double)r, 44));
}

uint64_t oq_scale_floor(float u, uint64_t S) {
  if (u <= 0.0f || S == 0) return 0;
  int ex;
  double f = frexp((double)u, &ex);           /* u = f 2^ex, f in [0.5,1) */
  uint64_t mu = (uint64_t)ldexp(f, 24);       /* u = mu 2^(ex-24) exactly */
  int shift = 24 - ex;                        /* u = mu / 2^shift */
  unsigned __int128 prod = (unsigned __int128)mu * S;
  if (shift >= 128) return 0;
  if (shift <= 0) return (uint64_t)(prod << (-shift));
  return (uint64_t)(prod >> shift);
}

static int64_t argmax_lowest(const float* row, int64_t V) {
  int64_t best = 0;
  for (int64_t v = 1; v < V; ++v)
    if (row[v] > row[best]) best = v;
  return best;
}

/* Returns the sampled token, or -1 when the row has no mass. */
static int64_t inverse_cdf(const float* r, int64_t V, float u) {
  uint64_t S = 0;
  for (int64_t v = 0; v < V; ++v) S += oq_fix44(r[v]);
  if (S == 0) return -1;
  uint64_t T = oq_scale_floor(u, S);
  uint64_t c = 0;
  for (int64_t v = 0; v < V; ++v) {
    c += oq_fix44(r[v]);
    if (c > T) return v;
  }
  return -1;
}

static int accept_one(const float* p, const float* q, const int32_t* x,
                      const float* u, int64_t K, int64_t V, int mode,
                      float* scratch, int32_t* n_out, int32_t* tok) {
  for (int64_t i = 0; i <= K; ++i) tok[i] = -1;
  *n_out = -1;
  for (int64_t i = 0; i < K; ++i)
    if (x[i] < 0 || x[i] >= V) return OQ_BAD_SEQ;
  if (!(u[K] >= 0.0f && u[K] < 1.0f)) return OQ_BAD_SEQ;

  int64_t n = 0;
  for (int64_t i = 0; i < K; ++i) {
    const float* pi = p + i * V;
    int accept;
    if (mode == OQ_ACCEPT_GREEDY) {
      accept = (argmax_lowest(pi, V) == x[i]);
    } else {
      const float* qi = q + i * V;
      accept = (double)u[i] * (double)qi[x[i]] < (double)pi[x[i]];
    }
    if (!accept) break;
    ++n;
  }

  int64_t token;
  const float* pn = p + n * V;
  if (mode == OQ_ACCEPT_GREEDY) {
    token = argmax_lowest(pn, V);
  } else if (n < K) {
    const float* qn = q + n * V;
    for (int64_t v = 0; v < V; ++v) {
      float d = pn[v] - qn[v];
      scratch[v] = d > 0.0f ? d : 0.0f;
    }
    token = inverse_cdf(scratch, V, u[K]);
    if (token < 0) token = inverse_cdf(pn, V, u[K]);
  } else {
    token = inverse_cdf(pn, V, u[K]);
  }
  if (token < 0) return OQ_BAD_SEQ;

  for (int64_t i = 0; i < n; ++i) tok[i] = x[i];
  tok[n] = (int32_t)token;
  *n_out = (int32_t)n;
  return OQ_OK;
}

int oq_accept(const float* p, const float* q, const int32_t* draft,
              const float* u, int64_t B, int64_t K, int64_t V, int mode,
              int32_t* n_accepted, int32_t* tokens) {
  if (B < 0 || K < 0 || V <= 0) return OQ_BAD_ARG;
  if (K > 0 && mode != OQ_ACCEPT_GREEDY && q == NULL) return OQ_BAD_ARG;
  float small[64];
  float* scratch = V <= 64 ? small : (float*)malloc((size_t)V * sizeof(float));
  if (!scratch) return OQ_BAD_ARG;
  int status = OQ_OK;
  for (int64_t b = 0; b < B; ++b) {
    int st = accept_one(p + b * (K + 1) * V, q ? q + b * K * V : NULL,
                        draft + b * K, u + b * (K + 1), K, V, mode, scratch,
                        n_accepted + b, tokens + b * (K + 1));
    if (st != OQ_OK) status = OQ_BAD_SEQ;
  }
  if (scratch != small) free(scratch);
  return status;
}

int oq_sample(const float* probs, const float* u, int64_t B, int64_t V,
              int32_t* tokens) {
  if (B < 0 || V <= 0) return OQ_BAD_ARG;
  int status = OQ_OK;
  for (int64_t b = 0; b < B; ++b) {
    int64_t t = -1;
    if (u[b] >= 0.0f && u[b] < 1.0f) t = inverse_cdf(probs + b * V, V, u[b]);
    tokens[b] = (int32_t)t;
    if (t < 0) status = OQ_BAD_SEQ;
  }
  return status;
}

/* ---- probabilities from logits ------------------------------------------ */

float oq_exp_neg(float x) {
  /* fp32 constants (exact hexadecimal values):
   *   log2(e) rounded; ln 2 = LN2_HI + LN2_LO with LN2_HI holding 16
   *   significant bits (so n * LN2_HI is exact for |n| < 256); 1/k! rounded. */
  const float LOG2E = 0x1.715476p+0f;
  const float LN2_HI = 0x1.62e4p-1f;
  const float LN2_LO = 0x1.7f7d1cp-20f;
  const float C2 = 0x1p-1f, C3 = 0x1.555556p-3f, C4 = 0x1.555556p-5f;
  const float C5 = 0x1.111112p-7f, C6 = 0x1.6c16c2p-10f, C7 = 0x1.a01a02p-13f;
  if (!(x > -104.0f)) return 0.0f;
  const float n = rintf(x * LOG2E);
  float r = fmaf(-n, LN2_HI, x);
  r = fmaf(-n, LN2_LO, r);
  float p = C7;
  p = fmaf(p, r, C6);
  p = fmaf(p, r, C5);
  p = fmaf(p, r, C4);
  p = fmaf(p, r, C3);
  p = fmaf(p, r, C2);
  p = fmaf(p, r, 1.0f);
  p = fmaf(p, r, 1.0f);
  const int ni = (int)n;
  union { uint32_t u; float f; } sc;
  if (ni >= -126) {
    sc.u = (uint32_t)(ni + 127) << 23;
    return p * sc.f;
  }
  sc.u = (uint32_t)(ni + 127 + 64) << 23;   /* 2^(n+64), normal */
  const float t = p * sc.f;                 /* exact */
  return t * 0x1p-64f;                      /* one rounding into the subnormals */
}

void oq_exp_neg_array(const float* x, int64_t n, float* out) {
  for (int64_t i = 0; i < n; ++i) out[i] = oq_exp_neg(x[i]);
}

int oq_softmax_row(const uint16_t* z, int64_t V, float T, float* p) {
  if (V < 1 || !(T > 0.0f) || !isfinite(T)) return OQ_BAD_ARG;
  float m = -INFINITY;
  for (int64_t v = 0; v < V; ++v) {
    const float zv = (float)oq_f16_decode(z[v]);
    if (!isfinite(zv)) return OQ_BAD_ARG;
    if (zv > m) m = zv;
  }
  const float invT = 1.0f / T;
  uint64_t S = 0;
  for (int64_t v = 0; v < V; ++v) {
    const float e = oq_exp_neg(((float)oq_f16_decode(z[v]) - m) * invT);
    p[v] = e;                                      /* e_v for now */
    S += (uint64_t)floor(ldexp((double)e, 40));    /* exact: e <= 1 */
  }
  const float s = (float)ldexp((double)S, -40);
  for (int64_t v = 0; v < V; ++v) p[v] = p[v] / s;
  return OQ_OK;
}

int oq_accept_logits(const uint16_t* zp, const uint16_t* zq, const int32_t* draft,
                     const float* u, int64_t B, int64_t K, int64_t V, float T,
                     int mode, int32_t* n_accepted, int32_t* tokens) {
  if (B < 0 || K < 0 || V <= 0) return OQ_BAD_ARG;
  if (K > 0 && zq == NULL) return OQ_BAD_ARG;
  float* p = (float*)malloc((size_t)(B * (K + 1) * V + (K > 0 ? B * K * V : 0) + 1) * sizeof(float));
  if (!p) return OQ_BAD_ARG;
  float* q = p + B * (K + 1) * V;
  int st = OQ_OK;
  for (int64_t b = 0; b < B && st == OQ_OK; ++b) {
    for (int64_t i = 0; i <= K && st == OQ_OK; ++i)
      st = oq_softmax_row(zp + (b * (K + 1) + i) * V, V, T, p + (b * (K + 1) + i) * V);
    for (int64_t i = 0; i < K && st == OQ_OK; ++i)  /* zq row of step i, sequence b */
      st = oq_softmax_row(zq + (i * B + b) * V, V, T, q + (b * K + i) * V);
  }
  if (st == OQ_OK)
    st = oq_accept(p, K > 0 ? q : NULL, draft, u, B, K, V, mode, n_accepted, tokens);
  free(p);
  return st;
}

int oq_sample_logits(const uint16_t* z, const float* u, int64_t B, int64_t V,
                     float T, int32_t* tokens) {
  if (B < 0 || V <= 0) return OQ_BAD_ARG;
  float* p = (float*)malloc((size_t)(B * V + 1) * sizeof(float));
  if (!p) return OQ_BAD_ARG;
  int st = OQ_OK;
  for (int64_t b = 0; b < B && st == OQ_OK; ++b) st = oq_softmax_row(z + b * V, V, T, p + b * V);
  if (st == OQ_OK) st = oq_sample(p, u, B, V, tokens);
  free(p);
  return st;
}

/* ---- decoder: RMSNorm, RoPE, attention ----------------------------------- */

void oq_rmsnorm(const double* x, const double* gamma, int64_t M, int64_t H, double eps, double* y) {
  for (int64_t m = 0; m < M; ++m) {
    double ss = 0.0;
    for (int64_t h = 0; h < H; ++h) ss += x[m * H + h] * x[m * H + h];
    const double r = 1.0 / sqrt(ss / (double)H + eps);
    for (int64_t h = 0; h < H; ++h) y[m * H + h] = x[m * H + h] * r * gamma[h];
  }
}

void oq_rope(double* x, const int64_t* pos, int64_t M, int64_t nheads, int64_t D, double theta) {
  const int64_t half = D / 2;
  for (int64_t m = 0; m < M; ++m)
    for (int64_t h = 0; h < nheads; ++h) {
      double* r = x + (m * nheads + h) * D;
      for (int64_t d = 0; d < half; ++d) {
        const double f = pow(theta, -2.0 * (double)d / (double)D);
        const double a = (double)pos[m] * f;
        const double c = cos(a), s = sin(a);
        const double x1 = r[d], x2 = r[d + half];
        r[d] = x1 * c - x2 * s;
        r[d + half] = x2 * c + x1 * s;
      }
    }
}

void oq_attention(const double* q, const double* k, const double* v, const int64_t* qpos,
                  int64_t T, int64_t L, int64_t Hq, int64_t Hkv, int64_t D, double* out) {
  const int64_t G = Hq / Hkv;
  const double scale = 1.0 / sqrt((double)D);
  double* w = (double*)malloc((size_t)(L > 0 ? L : 1) * sizeof(double));
  for (int64_t t = 0; t < T; ++t)
    for (int64_t h = 0; h < Hq; ++h) {
      const int64_t kh = h / G;
      const double* qr = q + (t * Hq + h) * D;
      int64_t n = qpos[t] + 1 < L ? qpos[t] + 1 : L;  /* keys 0 .. qpos[t] */
      double mx = -INFINITY;
      for (int64_t j = 0; j < n; ++j) {
        double dot = 0.0;
        for (int64_t d = 0; d < D; ++d) dot += qr[d] * k[(j * Hkv + kh) * D + d];
        w[j] = dot * scale;
        if (w[j] > mx) mx = w[j];
      }
      double sum = 0.0;
      for (int64_t j = 0; j < n; ++j) {
        w[j] = exp(w[j] - mx);
        sum += w[j];
      }
      double* o = out + (t * Hq + h) * D;
      for (int64_t d = 0; d < D; ++d) o[d] = 0.0;
      for (int64_t j = 0; j < n; ++j)
        for (int64_t d = 0; d < D; ++d) o[d] += w[j] / sum * v[(j * Hkv + kh) * D + d];
    }
  free(w);
}
