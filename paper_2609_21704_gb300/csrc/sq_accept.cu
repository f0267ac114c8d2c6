// sq_accept.cu -- accept / reject / resample over the vocabulary.
//
// Sec. III-A.3 (token rule) and Sec. III-D.4 (token acceptance or
// correction); sampling mode is the lossless speculative-sampling rule the
// paper says it adheres to (Sec. I).  Semantics are stated in specquant.h.
//
// Layout of the work: one CTA per (sequence b, vocabulary chunk c) of 2048
// entries.  Every CTA evaluates the K accept tests of its sequence (K
// gathers), then reduces its chunk of the correction row to a 64-bit
// fixed-point partial sum (sampling) or a packed (value, index) maximum per
// position (greedy).  The partials go to the workspace; the last CTA of a
// sequence to arrive (atomic ticket) combines them, turns the uniform into
// an integer target T = floor(u * S), finds the chunk holding T and scans
// that chunk alone for the token.  All sums are integer, so the outcome is
// independent of the order in which CTAs arrive.
//
// Bytes per sequence: sampling 2 V fp32 (p_n and q_n) + 2K gathers;
// greedy (K+1) V fp32.
#include <mutex>

#include "sq_internal.h"

namespace sq {

__device__ unsigned int g_accept_status;

// Scratch of sq_accept_noalloc: ticket counters and per-chunk partials live
// here instead of in a caller-provided workspace.  Every device that loads
// the library keeps this array until the process exits, and every call of
// sq_accept_noalloc on a device reuses the same bytes.
static __device__ __align__(256) unsigned char g_accept_scratch[kAcceptNoallocScratchBytes];

// floor(r * 2^Q) from the fp32 bits of r in [0, 1] (exact integer shifts).
template <int Q>
__device__ __forceinline__ unsigned long long fixq(float r) {
  const uint32_t b = __float_as_uint(r);
  const uint32_t e = (b >> 23) & 0xffu;
  if ((b >> 31) || e == 0) return 0ull;  // zero, negative, or below 2^-126
  const unsigned long long mant = (unsigned long long)((b & 0x7fffffu) | 0x800000u);
  const int sh = (int)e - 150 + Q;       // r = mant * 2^(e-150)
  if (sh >= 0) return mant << sh;
  if (sh <= -64) return 0ull;
  return mant >> (-sh);
}
__device__ __forceinline__ unsigned long long fix44(float r) { return fixq<44>(r); }

// ---- probabilities from logits (softmax with temperature) -----------------
// e^x for x <= 0 in explicitly rounded fp32 operations: Cody-Waite reduction
// x = n ln2 + r (ln 2 split into a head of 16 significant bits, so that
// n * head is exact for |n| < 256, and a tail), e^r by its degree-7 Taylor
// polynomial in Horner form with fused multiply-adds, then the exact
// scaling by 2^n (through 2^(n+64) * 2^-64 below 2^-126: one rounding into
// the subnormals); 0 for x <= -104 (below the smallest subnormal).  Only
// _rn intrinsics are used, so nothing is contracted or reordered and the
// bits follow from the definition.
__device__ __forceinline__ float exp_neg(float x) {
  if (!(x > -104.0f)) return 0.0f;
  const float n = rintf(__fmul_rn(x, 0x1.715476p+0f));  // x log2(e), nearest integer
  float r = __fmaf_rn(-n, 0x1.62e4p-1f, x);              // x - n ln2 (head)
  r = __fmaf_rn(-n, 0x1.7f7d1cp-20f, r);                 // ... (tail)
  float p = 0x1.a01a02p-13f;                             // 1/7!
  p = __fmaf_rn(p, r, 0x1.6c16c2p-10f);                  // 1/6!
  p = __fmaf_rn(p, r, 0x1.111112p-7f);                   // 1/5!
  p = __fmaf_rn(p, r, 0x1.555556p-5f);                   // 1/4!
  p = __fmaf_rn(p, r, 0x1.555556p-3f);                   // 1/3!
  p = __fmaf_rn(p, r, 0.5f);
  p = __fmaf_rn(p, r, 1.0f);
  p = __fmaf_rn(p, r, 1.0f);
  const int ni = (int)n;
  if (ni >= -126) return __fmul_rn(p, __uint_as_float((uint32_t)(ni + 127) << 23));
  return __fmul_rn(__fmul_rn(p, __uint_as_float((uint32_t)(ni + 127 + 64) << 23)), 0x1p-64f);
}

// p_v = e_v / s with e_v = exp_neg((z_v - m) * invT) (fp32 subtract, multiply,
// divide, each rounded to nearest).
__device__ __forceinline__ float logit_prob(__half z, float m, float invT, float s) {
  return __fdiv_rn(exp_neg(__fmul_rn(__fsub_rn(__half2float(z), m), invT)), s);
}

// Probability sources of the accept kernel: rows of stored fp32
// probabilities, or rows of fp16 logits with their softmax statistics.
// Each row type reads one entry, or the 8 entries [v, v + 8) (those at or
// past vend read as 0) with vector loads where the addresses allow.
struct ProbRow {
  const float* p;
  __device__ __forceinline__ float operator()(int64_t v) const { return p[v]; }
  __device__ __forceinline__ void load8(int64_t v, int64_t vend, float out[8]) const {
    if (v + 8 <= vend && ((reinterpret_cast<uintptr_t>(p + v) & 15u) == 0)) {
      const float4 a = *reinterpret_cast<const float4*>(p + v);
      const float4 b = *reinterpret_cast<const float4*>(p + v + 4);
      out[0] = a.x; out[1] = a.y; out[2] = a.z; out[3] = a.w;
      out[4] = b.x; out[5] = b.y; out[6] = b.z; out[7] = b.w;
    } else {
#pragma unroll
      for (int j = 0; j < 8; ++j) out[j] = v + j < vend ? p[v + j] : 0.0f;
    }
  }
};
struct ProbSrc {
  const float* p;  // [B, K+1, V]
  const float* q;  // [B, K, V] or null
  int K;
  int64_t V;
  __device__ __forceinline__ ProbRow prow(int b, int i) const {
    return ProbRow{p + ((int64_t)b * (K + 1) + i) * V};
  }
  __device__ __forceinline__ ProbRow qrow(int b, int i) const {
    return ProbRow{q + ((int64_t)b * K + i) * V};
  }
  __device__ __forceinline__ bool has_q() const { return q != nullptr; }
  __device__ __forceinline__ bool rows_ok(int, int) const { return true; }
};
struct LogitRow {
  const __half* z;
  float m, invT, s;
  __device__ __forceinline__ float operator()(int64_t v) const { return logit_prob(z[v], m, invT, s); }
  __device__ __forceinline__ void load8(int64_t v, int64_t vend, float out[8]) const {
    if (v + 8 <= vend && ((reinterpret_cast<uintptr_t>(z + v) & 15u) == 0)) {
      const uint4 w = *reinterpret_cast<const uint4*>(z + v);
      const uint32_t h[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        out[2 * j] = logit_prob(__ushort_as_half(lo16(h[j])), m, invT, s);
        out[2 * j + 1] = logit_prob(__ushort_as_half(hi16(h[j])), m, invT, s);
      }
    } else {
#pragma unroll
      for (int j = 0; j < 8; ++j) out[j] = v + j < vend ? logit_prob(z[v + j], m, invT, s) : 0.0f;
    }
  }
};

// The 8 fp16 values [v, v + 8) of a row as fp32; entries at or past vend are
// reported invalid through `ok`.
__device__ __forceinline__ void load8_half(const __half* z, int64_t v, int64_t vend, float out[8],
                                           bool ok[8]) {
  if (v + 8 <= vend && ((reinterpret_cast<uintptr_t>(z + v) & 15u) == 0)) {
    const uint4 w = *reinterpret_cast<const uint4*>(z + v);
    const uint32_t h[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      out[2 * j] = __half2float(__ushort_as_half(lo16(h[j])));
      out[2 * j + 1] = __half2float(__ushort_as_half(hi16(h[j])));
      ok[2 * j] = ok[2 * j + 1] = true;
    }
  } else {
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      ok[j] = v + j < vend;
      out[j] = ok[j] ? __half2float(z[v + j]) : 0.0f;
    }
  }
}
struct LogitSrc {
  const __half* zp;  // [B, K+1, V]
  const __half* zq;  // [K, B, V]
  const float* m;    // row maxima: target rows b (K+1) + i, then draft rows B (K+1) + i B + b
  const float* s;    // row normalisers, same order
  float invT;
  int B, K;
  int64_t V;
  __device__ __forceinline__ LogitRow prow(int b, int i) const {
    const int64_t r = (int64_t)b * (K + 1) + i;
    return LogitRow{zp + r * V, m[r], invT, s[r]};
  }
  __device__ __forceinline__ LogitRow qrow(int b, int i) const {
    if (K == 0) return LogitRow{zp, 0.0f, 0.0f, 1.0f};  // no draft rows; never read
    const int64_t r = (int64_t)i * B + b;
    const int64_t rs = (int64_t)B * (K + 1) + r;
    return LogitRow{zq + r * V, m[rs], invT, s[rs]};
  }
  __device__ __forceinline__ bool has_q() const { return K > 0; }
  // row j of sequence b's 2K+1 rows has finite statistics (finite logits)
  __device__ __forceinline__ bool rows_ok(int b, int j) const {
    const int64_t r = j <= K ? (int64_t)b * (K + 1) + j : (int64_t)B * (K + 1) + (int64_t)(j - K - 1) * B + b;
    return isfinite(m[r]) && isfinite(s[r]);
  }
};

// floor(u * S) for u in [0, 1), exact (128-bit product of the 24-bit
// significand and S, then a right shift).
__device__ __forceinline__ unsigned long long scale_floor(float u, unsigned long long S) {
  const uint32_t b = __float_as_uint(u);
  const uint32_t e = (b >> 23) & 0xffu;
  if ((b >> 31) || e == 0 || S == 0) return 0ull;
  const unsigned long long mant = (unsigned long long)((b & 0x7fffffu) | 0x800000u);
  const int shift = 150 - (int)e;        // u = mant / 2^shift, shift >= 24
  const unsigned long long lo = mant * S;
  const unsigned long long hi = __umul64hi(mant, S);
  if (shift >= 128) return 0ull;
  if (shift >= 64) return hi >> (shift - 64);
  return (lo >> shift) | (hi << (64 - shift));
}

__device__ __forceinline__ unsigned long long warp_sum_u64(unsigned long long v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ unsigned long long warp_max_u64(unsigned long long v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const unsigned long long w = __shfl_xor_sync(0xffffffffu, v, o);
    v = w > v ? w : v;
  }
  return v;
}

// (value, index) -> key whose unsigned maximum is the largest value with
// the lowest index (values are non-negative, so their bits order like ints).
__device__ __forceinline__ unsigned long long argmax_key(float v, int64_t idx) {
  return ((unsigned long long)__float_as_uint(v) << 32) | (0xffffffffull - (unsigned long long)idx);
}

// Block-wide reductions over one value per thread (every thread of the
// block calls them; `blk` holds one slot per warp).  The results reach
// every thread.
template <int NT>
__device__ __forceinline__ unsigned long long block_sum_u64(unsigned long long v, unsigned long long* blk) {
  v = warp_sum_u64(v);
  __syncthreads();
  if ((threadIdx.x & 31) == 0) blk[threadIdx.x >> 5] = v;
  __syncthreads();
  unsigned long long t = 0;
#pragma unroll
  for (int w = 0; w < NT / 32; ++w) t += blk[w];
  return t;
}

template <int NT>
__device__ __forceinline__ unsigned long long block_max_u64(unsigned long long v, unsigned long long* blk) {
  v = warp_max_u64(v);
  __syncthreads();
  if ((threadIdx.x & 31) == 0) blk[threadIdx.x >> 5] = v;
  __syncthreads();
  unsigned long long t = 0;
#pragma unroll
  for (int w = 0; w < NT / 32; ++w) t = blk[w] > t ? blk[w] : t;
  return t;
}

// Exclusive prefix sum in thread order; `total` receives the block total.
template <int NT>
__device__ __forceinline__ unsigned long long block_excl_scan_u64(unsigned long long v, unsigned long long* blk,
                                                                 unsigned long long& total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  unsigned long long incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned long long t = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += t;
  }
  __syncthreads();
  if (lane == 31) blk[warp] = incl;
  __syncthreads();
  unsigned long long base = 0, tot = 0;
#pragma unroll
  for (int w = 0; w < NT / 32; ++w) {
    if (w < warp) base += blk[w];
    tot += blk[w];
  }
  total = tot;
  return base + incl - v;
}

constexpr int kAcceptThreads = 256;
static_assert(kAcceptChunk == 8 * kAcceptThreads, "a thread owns 8 consecutive entries of a chunk");
static_assert(kSoftmaxChunk == 8 * kAcceptThreads, "a thread owns 8 consecutive entries of a chunk");

template <class Src>
__global__ void __launch_bounds__(kAcceptThreads) accept_kernel(AcceptArgs a, Src src) {
  griddep_wait();
  griddep_launch_dependents();
  __shared__ unsigned long long red[kAcceptThreads / 32][17];
  __shared__ unsigned long long blk[kAcceptThreads / 32];
  __shared__ unsigned long long s_best[17];
  __shared__ int s_n, s_valid, s_last;
  __shared__ unsigned long long s_T;
  __shared__ int s_chunk, s_use_p, s_token;

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t bc = blockIdx.x;
  const int b = (int)(bc / a.C), c = (int)(bc - (int64_t)b * a.C);
  const int K = a.K;
  const int64_t V = a.V;
  const int32_t* xb = a.draft + (int64_t)b * K;
  const float* ub = a.u + (int64_t)b * (K + 1);
  const int64_t v0 = (int64_t)c * a.chunk;
  const int64_t v1 = v0 + a.chunk < V ? v0 + a.chunk : V;
  unsigned long long* part = a.part + ((int64_t)b * a.C + c) * a.slots;

  // ---- validity and (sampling) the accept tests, evaluated by warp 0
  if (warp == 0) {
    bool bad = false, acc = true;
    // finite statistics for the sequence's rows (logits only)
    bool rows_bad = false;
    for (int j = lane; j <= 2 * K; j += 32) rows_bad |= !src.rows_ok(b, j);
    const unsigned rows_mask = __ballot_sync(0xffffffffu, rows_bad);
    if (lane < K) {
      const int32_t x = xb[lane];
      bad = (x < 0 || (int64_t)x >= V);
      if (!bad && !rows_mask && a.mode == SQ_ACCEPT_SAMPLE)
        acc = (double)ub[lane] * (double)src.qrow(b, lane)(x) < (double)src.prow(b, lane)(x);
    }
    const float uk = ub[K];
    const bool bad_u = !(uk >= 0.0f && uk < 1.0f);
    const unsigned bad_mask = __ballot_sync(0xffffffffu, bad);
    const unsigned rej_mask = __ballot_sync(0xffffffffu, lane < K && !acc);
    if (lane == 0) {
      s_valid = (bad_mask == 0u) && !bad_u && !rows_mask;
      s_n = rej_mask ? (__ffs(rej_mask) - 1) : K;
      if (c == 0 && bad_mask) atomicOr(&g_accept_status, SQ_DEV_BAD_DRAFT_TOKEN);
      if (c == 0 && bad_u) atomicOr(&g_accept_status, SQ_DEV_BAD_UNIFORM);
    }
  }
  __syncthreads();
  const int n = s_n;

  // ---- chunk partials
  if (a.mode == SQ_ACCEPT_SAMPLE) {
    const auto pn = src.prow(b, n);
    const bool use_q = n < K;
    const auto qn = src.qrow(b, use_q ? n : 0);
    unsigned long long sr = 0, sp = 0;
    // thread t: the 8 entries [v0 + 8t, v0 + 8t + 8) of the chunk
    for (int64_t vb = v0 + 8 * (int64_t)tid; vb < v1; vb += 8 * kAcceptThreads) {
      float pv[8], qv[8];
      pn.load8(vb, v1, pv);
      if (use_q) qn.load8(vb, v1, qv);
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        if (use_q) {
          const float d = pv[j] - qv[j];
          sr += fix44(d > 0.0f ? d : 0.0f);
          sp += fix44(pv[j]);
        } else {
          sr += fix44(pv[j]);
        }
      }
    }
    sr = warp_sum_u64(sr);
    sp = warp_sum_u64(sp);
    if (lane == 0) {
      red[warp][0] = sr;
      red[warp][1] = sp;
    }
    __syncthreads();
    if (tid == 0) {
      unsigned long long tr = 0, tp = 0;
      for (int w = 0; w < kAcceptThreads / 32; ++w) {
        tr += red[w][0];
        tp += red[w][1];
      }
      part[0] = tr;
      part[1] = tp;
    }
  } else {
    // greedy: per position i, the maximum key over the chunk
    for (int i = 0; i <= K; ++i) {
      const auto pi = src.prow(b, i);
      unsigned long long best = 0;
      for (int64_t vb = v0 + 8 * (int64_t)tid; vb < v1; vb += 8 * kAcceptThreads) {
        float pv[8];
        pi.load8(vb, v1, pv);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          if (vb + j >= v1) break;
          const unsigned long long k = argmax_key(pv[j], vb + j);
          best = k > best ? k : best;
        }
      }
      best = warp_max_u64(best);
      if (lane == 0) red[warp][i] = best;
    }
    __syncthreads();
    if (tid <= K) {
      unsigned long long best = 0;
      for (int w = 0; w < kAcceptThreads / 32; ++w) best = red[w][tid] > best ? red[w][tid] : best;
      part[tid] = best;
    }
  }

  // ---- ticket: the last CTA of the sequence finishes it
  __syncthreads();
  if (tid == 0) {
    __threadfence();
    const unsigned ticket = atomicAdd(&a.counter[b], 1u);
    s_last = (ticket == (unsigned)(a.C - 1));
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  const unsigned long long* pall = a.part + (int64_t)b * a.C * a.slots;
  int32_t* tok = a.tok_out + (int64_t)b * (K + 1);

  // every thread takes the partials of chunks 2t and 2t + 1 (C <= 512)
  const int c0 = 2 * tid, c1 = 2 * tid + 1;
  auto partial = [&](int cc, int slot) -> unsigned long long {
    return cc < a.C ? __ldcg(pall + (int64_t)cc * a.slots + slot) : 0ull;
  };

  if (a.mode == SQ_ACCEPT_GREEDY) {
    for (int i = 0; i <= K; ++i) {
      const unsigned long long k0 = partial(c0, i), k1 = partial(c1, i);
      const unsigned long long best = block_max_u64<kAcceptThreads>(k0 > k1 ? k0 : k1, blk);
      if (tid == 0) s_best[i] = best;
    }
    __syncthreads();
    if (tid == 0) {
      int nn = K;
      int64_t am_n = -1;
      for (int i = 0; i <= K; ++i) {
        const int64_t am = (int64_t)(0xffffffffull - (s_best[i] & 0xffffffffull));
        if (i < nn && i < K && am != xb[i]) nn = i;
        if (i == nn) {
          am_n = am;
          break;
        }
      }
      const bool ok = s_valid != 0;
      if (a.n_out) a.n_out[b] = ok ? nn : -1;
      for (int i = 0; i <= K; ++i) tok[i] = ok ? (i < nn ? xb[i] : (i == nn ? (int32_t)am_n : -1)) : -1;
      a.counter[b] = 0u;
    }
    return;
  }

  // sampling: the row's total mass, the target T and the chunk holding it
  // (block-wide sum, then an exclusive scan of the chunk masses)
  const unsigned long long r0 = partial(c0, 0), r1 = partial(c1, 0);
  unsigned long long S = block_sum_u64<kAcceptThreads>(r0 + r1, blk);
  const int use_p = (S == 0 && n < K) ? 1 : 0;  // block-uniform
  unsigned long long m0 = r0, m1 = r1;
  if (use_p) {
    m0 = partial(c0, 1);
    m1 = partial(c1, 1);
    S = block_sum_u64<kAcceptThreads>(m0 + m1, blk);
  }
  const int ok = s_valid && S != 0;
  const unsigned long long T = ok ? scale_floor(ub[K], S) : 0ull;
  if (tid == 0) {
    if (s_valid && S == 0) atomicOr(&g_accept_status, SQ_DEV_NO_MASS);
    s_chunk = a.C - 1;
    s_T = 0;
    s_use_p = use_p;
    s_token = -1;
  }
  unsigned long long total;
  const unsigned long long excl = block_excl_scan_u64<kAcceptThreads>(m0 + m1, blk, total);
  if (ok && excl <= T && T < excl + m0 + m1) {  // exactly one thread
    if (T < excl + m0) {
      s_chunk = c0;
      s_T = T - excl;
    } else {
      s_chunk = c1;
      s_T = T - excl - m0;
    }
  }
  __syncthreads();
  if (tid == 0) s_valid = ok;
  __syncthreads();
  if (s_valid) {
    const auto pn = src.prow(b, n);
    const bool use_q = n < K && !s_use_p;
    const auto qn = src.qrow(b, use_q ? n : 0);
    const int64_t w0 = (int64_t)s_chunk * a.chunk;
    const int64_t w1 = w0 + a.chunk < V ? w0 + a.chunk : V;
    const unsigned long long T = s_T;
    // thread t holds the 8 entries [w0 + 8t, w0 + 8t + 8) (the chunk is
    // 8 x the block): local prefix sums, then one block-wide exclusive scan
    // of the thread totals; the thread whose range holds T finds the token
    const int64_t vb = w0 + 8 * (int64_t)tid;
    unsigned long long R[8];
    {
      float pv[8], qv[8];
      pn.load8(vb, w1, pv);
      if (use_q) qn.load8(vb, w1, qv);
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        if (use_q) {
          const float d = pv[j] - qv[j];
          R[j] = fix44(d > 0.0f ? d : 0.0f);
        } else {
          R[j] = fix44(pv[j]);
        }
      }
    }
    unsigned long long tot = 0;
#pragma unroll
    for (int j = 0; j < 8; ++j) tot += R[j];
    unsigned long long incl = tot;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const unsigned long long t = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += t;
    }
    if (lane == 31) red[warp][0] = incl;
    __syncthreads();
    unsigned long long wbase = 0;
    for (int w = 0; w < warp; ++w) wbase += red[w][0];
    const unsigned long long excl = incl - tot + wbase;
    if (excl <= T && T < excl + tot) {  // exactly one thread's range holds T
      unsigned long long c = excl;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        c += R[j];
        if (c > T) {
          s_token = (int)(vb + j);
          break;
        }
      }
    }
  }
  __syncthreads();
  if (tid == 0) {
    const bool ok = s_valid && s_token >= 0;
    if (a.n_out) a.n_out[b] = ok ? n : -1;
    for (int i = 0; i <= K; ++i) tok[i] = ok ? (i < n ? xb[i] : (i == n ? s_token : -1)) : -1;
    a.counter[b] = 0u;
  }
}

size_t accept_workspace_bytes(int B, int K, int64_t V) {
  if (B < 0 || K < 0 || V <= 0) return 0;
  const int64_t C = (V + kAcceptChunk - 1) / kAcceptChunk;
  const int64_t slots = K + 1 > 2 ? K + 1 : 2;
  const size_t part = (size_t)B * (size_t)C * (size_t)slots * 8u;
  const size_t ctr = (((size_t)B * 4u) + 15u) & ~(size_t)15u;
  return ctr + part + 16u;
}

cudaError_t launch_accept(const AcceptArgs& a, cudaStream_t st) {
  if (a.B == 0) return cudaSuccess;
  const int64_t blocks = (int64_t)a.B * a.C;
  ProbSrc src{a.p, a.q, a.K, a.V};
  return launch_pdl(accept_kernel<ProbSrc>, dim3((unsigned)blocks), dim3(kAcceptThreads), 0, st, a,
                    src);
}

// ---- softmax statistics of logit rows --------------------------------------
// One CTA per (row, chunk of kSoftmaxChunk entries).  Pass 1: the row
// maximum (a NaN marks a row holding a non-finite logit); pass 2: the
// fixed-point normaliser S = sum_v floor(e_v 2^40) and s = float(S 2^-40).
// The last CTA of a row (atomic ticket, counter left at zero) combines the
// chunk partials; max and integer sums do not depend on their order.
__device__ __forceinline__ const __half* softmax_row_ptr(const SoftmaxArgs& a, int64_t r) {
  return r < a.rp ? a.zp + r * a.V : a.zq + (r - a.rp) * a.V;
}

__global__ void __launch_bounds__(kAcceptThreads) softmax_max_kernel(SoftmaxArgs a) {
  griddep_wait();
  griddep_launch_dependents();
  __shared__ float red[kAcceptThreads / 32];
  __shared__ int red_bad[kAcceptThreads / 32];
  __shared__ int s_last;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t r = blockIdx.x / a.C;
  const int c = (int)(blockIdx.x - r * a.C);
  const __half* z = softmax_row_ptr(a, r);
  const int64_t v0 = (int64_t)c * kSoftmaxChunk;
  const int64_t v1 = v0 + kSoftmaxChunk < a.V ? v0 + kSoftmaxChunk : a.V;
  float mx = -INFINITY;
  int bad = 0;
  {
    float f[8];
    bool ok[8];
    load8_half(z, v0 + 8 * (int64_t)tid, v1, f, ok);
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if (ok[j]) {
        bad |= !isfinite(f[j]);
        mx = fmaxf(mx, f[j]);
      }
  }
  mx = warp_max(mx);
  bad = __any_sync(0xffffffffu, bad);
  if (lane == 0) {
    red[warp] = mx;
    red_bad[warp] = bad;
  }
  __syncthreads();
  if (tid == 0) {
    float m = -INFINITY;
    int any_bad = 0;
    for (int w = 0; w < kAcceptThreads / 32; ++w) {
      m = fmaxf(m, red[w]);
      any_bad |= red_bad[w];
    }
    a.pmax[r * a.C + c] = any_bad ? __int_as_float(0x7fc00000) : m;
    __threadfence();
    s_last = atomicAdd(&a.counter[r], 1u) == (unsigned)(a.C - 1);
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  // the last CTA of the row: every thread takes chunks t and t + 256
  float m = -INFINITY;
  int nan = 0;
  for (int cc = tid; cc < a.C; cc += kAcceptThreads) {
    const float pm = __ldcg(a.pmax + r * a.C + cc);
    nan |= isnan(pm);
    m = fmaxf(m, pm);
  }
  m = warp_max(m);
  nan = __any_sync(0xffffffffu, nan);
  __syncthreads();
  if (lane == 0) {
    red[warp] = m;
    red_bad[warp] = nan;
  }
  __syncthreads();
  if (tid == 0) {
    float mm = -INFINITY;
    int any_nan = 0;
    for (int w = 0; w < kAcceptThreads / 32; ++w) {
      mm = fmaxf(mm, red[w]);
      any_nan |= red_bad[w];
    }
    if (any_nan) {
      mm = __int_as_float(0x7fc00000);
      atomicOr(&g_accept_status, SQ_DEV_NONFINITE_LOGIT);
    }
    a.m[r] = mm;
    a.counter[r] = 0u;
  }
}

__global__ void __launch_bounds__(kAcceptThreads) softmax_sum_kernel(SoftmaxArgs a) {
  griddep_wait();
  griddep_launch_dependents();
  __shared__ unsigned long long red[kAcceptThreads / 32];
  __shared__ int s_last;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t r = blockIdx.x / a.C;
  const int c = (int)(blockIdx.x - r * a.C);
  const __half* z = softmax_row_ptr(a, r);
  const int64_t v0 = (int64_t)c * kSoftmaxChunk;
  const int64_t v1 = v0 + kSoftmaxChunk < a.V ? v0 + kSoftmaxChunk : a.V;
  const float m = a.m[r];
  unsigned long long acc = 0;
  if (isfinite(m)) {
    float f[8];
    bool ok[8];
    load8_half(z, v0 + 8 * (int64_t)tid, v1, f, ok);
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if (ok[j]) acc += fixq<40>(exp_neg(__fmul_rn(__fsub_rn(f[j], m), a.invT)));
  }
  acc = warp_sum_u64(acc);
  if (lane == 0) red[warp] = acc;
  __syncthreads();
  if (tid == 0) {
    unsigned long long t = 0;
    for (int w = 0; w < kAcceptThreads / 32; ++w) t += red[w];
    a.psum[r * a.C + c] = t;
    __threadfence();
    s_last = atomicAdd(&a.counter[r], 1u) == (unsigned)(a.C - 1);
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  unsigned long long part = 0;
  for (int cc = tid; cc < a.C; cc += kAcceptThreads) part += __ldcg(a.psum + r * a.C + cc);
  const unsigned long long S = block_sum_u64<kAcceptThreads>(part, red);
  if (tid == 0) {
    a.s[r] = isfinite(m) ? __double2float_rn(__ull2double_rn(S) * 0x1p-40)
                         : __int_as_float(0x7fc00000);
    a.counter[r] = 0u;
  }
}

cudaError_t launch_accept_logits(const AcceptArgs& a, const SoftmaxArgs& sa, cudaStream_t st) {
  if (a.B == 0) return cudaSuccess;
  const int64_t sblocks = sa.rows * sa.C;
  cudaError_t e = launch_pdl(softmax_max_kernel, dim3((unsigned)sblocks), dim3(kAcceptThreads), 0, st, sa);
  if (e != cudaSuccess) return e;
  e = launch_pdl(softmax_sum_kernel, dim3((unsigned)sblocks), dim3(kAcceptThreads), 0, st, sa);
  if (e != cudaSuccess) return e;
  LogitSrc src{sa.zp, sa.zq, sa.m, sa.s, sa.invT, a.B, a.K, a.V};
  const int64_t blocks = (int64_t)a.B * a.C;
  return launch_pdl(accept_kernel<LogitSrc>, dim3((unsigned)blocks), dim3(kAcceptThreads), 0, st, a,
                    src);
}

size_t softmax_rows_workspace_bytes(int64_t rows, int64_t V) {
  if (rows < 0 || V <= 0) return 0;
  const int64_t C = (V + kSoftmaxChunk - 1) / kSoftmaxChunk;
  auto up16 = [](size_t x) { return (x + 15u) & ~(size_t)15u; };
  return up16((size_t)rows * 4u) * 3u + up16((size_t)rows * (size_t)C * 4u) +
         up16((size_t)rows * (size_t)C * 8u);
}

size_t softmax_workspace_bytes(int B, int K, int64_t V) {
  if (B < 0 || K < 0) return 0;
  return softmax_rows_workspace_bytes((int64_t)B * (K + 1) + (int64_t)B * K, V);
}

void softmax_layout(SoftmaxArgs& sa, void* ws) {
  auto up16 = [](size_t x) { return (x + 15u) & ~(size_t)15u; };
  char* sw = reinterpret_cast<char*>(ws);
  sa.C = (int)((sa.V + kSoftmaxChunk - 1) / kSoftmaxChunk);
  const size_t rows4 = up16((size_t)sa.rows * 4u);
  sa.counter = reinterpret_cast<unsigned int*>(sw);
  sa.m = reinterpret_cast<float*>(sw + rows4);
  sa.s = reinterpret_cast<float*>(sw + 2 * rows4);
  sa.pmax = reinterpret_cast<float*>(sw + 3 * rows4);
  sa.psum = reinterpret_cast<unsigned long long*>(sw + 3 * rows4 + up16((size_t)sa.rows * sa.C * 4u));
}

// p[r, v] from the row statistics (the same expression the accept kernel
// evaluates); NaN for a row holding a non-finite logit.
__global__ void __launch_bounds__(kAcceptThreads) softmax_write_kernel(SoftmaxArgs a, float* p) {
  griddep_wait();
  griddep_launch_dependents();
  const int64_t r = blockIdx.x / a.C;
  const int c = (int)(blockIdx.x - r * a.C);
  const __half* z = softmax_row_ptr(a, r);
  const int64_t v0 = (int64_t)c * kSoftmaxChunk;
  const int64_t v1 = v0 + kSoftmaxChunk < a.V ? v0 + kSoftmaxChunk : a.V;
  const float m = a.m[r], sc = a.s[r];
  const bool ok = isfinite(m) && isfinite(sc);
  float* pr = p + r * a.V;
  const int64_t vb = v0 + 8 * (int64_t)threadIdx.x;
  float f[8];
  bool in[8];
  load8_half(z, vb, v1, f, in);
#pragma unroll
  for (int j = 0; j < 8; ++j)
    if (in[j])
      pr[vb + j] = ok ? __fdiv_rn(exp_neg(__fmul_rn(__fsub_rn(f[j], m), a.invT)), sc)
                      : __int_as_float(0x7fc00000);
}

cudaError_t launch_softmax(const SoftmaxArgs& sa, float* p, cudaStream_t st) {
  if (sa.rows == 0) return cudaSuccess;
  const int64_t sblocks = sa.rows * sa.C;
  cudaError_t e = launch_pdl(softmax_max_kernel, dim3((unsigned)sblocks), dim3(kAcceptThreads), 0, st, sa);
  if (e != cudaSuccess) return e;
  e = launch_pdl(softmax_sum_kernel, dim3((unsigned)sblocks), dim3(kAcceptThreads), 0, st, sa);
  if (e != cudaSuccess) return e;
  return launch_pdl(softmax_write_kernel, dim3((unsigned)sblocks), dim3(kAcceptThreads), 0, st, sa, p);
}

// Device address of g_accept_scratch for the current device.  In host code
// the array's name is only a host-side stand-in, so the address is asked of
// the runtime once per device (with that device current) and cached.
cudaError_t accept_noalloc_scratch(void** ptr) {
  static std::mutex mu;
  static void* addr[64] = {nullptr};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(mu);
  if (addr[dev] == nullptr) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_accept_scratch);
    if (e != cudaSuccess) return e;
    addr[dev] = p;
  }
  *ptr = addr[dev];
  return cudaSuccess;
}

cudaError_t take_accept_status(uint32_t* bits) {
  uint32_t v = 0, zero = 0;
  cudaError_t e = cudaMemcpyFromSymbol(&v, g_accept_status, sizeof(v));
  if (e != cudaSuccess) return e;
  if (v) e = cudaMemcpyToSymbol(g_accept_status, &zero, sizeof(zero));
  *bits |= v;
  return e;
}

}  // namespace sq
