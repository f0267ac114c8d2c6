// sq_attention.cu -- the decoder around the linear stack: RMSNorm, rotary
// embedding with the KV-cache append, grouped-query decode attention over
// the cache, and the rollback of cache lengths after acceptance.
//
// Sec. III-D.2/3 run the whole model for the draft and verify passes;
// Sec. III-D.4 restarts from the first rejected token, so each model's
// cache keeps only the accepted prefix.  Definitions (no model internals
// are given in the paper; these are the Qwen2.5 decoder's):
//   RMSNorm   y = x / sqrt(mean(x^2) + eps) * gamma       (fp32, fp16 out)
//   RoPE      pairs (d, d + D/2), angle pos * theta^(-2d/D) (fp64 angle)
//   attention softmax(q . k / sqrt(D)) v over cache positions <= the
//             query's position; query head h reads key/value head
//             h / (Hq / Hkv).
// Layouts: qkv rows [B*T, (Hq + 2 Hkv) D] (q heads, k heads, v heads, the
// fused projection's output); caches [B, Hkv, max_ctx, D] fp16; attention
// output rows [B*T, Hq D].  Token t of sequence b sits at position
// pos0[b] + t.
//
// Attention is split over 32-key chunks of the cache (one CTA per
// (sequence, key/value head, chunk)): all G * T queries of the group read
// the chunk once from shared memory, then a combine kernel merges the
// chunks' (max, sum, weighted value) partials.  Bound: the cache bytes
// (2 * pos * Hkv * D * 2 per sequence) and, for long query groups, CUDA-core
// arithmetic (G * T * 2 D flops per cached key).
#include <math.h>

#include "sq_decoder.h"

namespace sq {

__device__ unsigned int g_attn_status;

constexpr int kHeadDim = 128;
constexpr int kAttnChunk = 32;      // cache positions per CTA
constexpr int kAttnThreads = 256;
constexpr int kRowPad = kHeadDim + 4;  // fp32 row stride in shared memory (16-byte rows, fewer conflicts)
constexpr int kMaxT = 32;           // new tokens per sequence and call
// Per-query partial record in the workspace: (max, sum, 2 unused, o[D]):
// 132 floats = 528 bytes, so records and their o[] stay 16-byte aligned.
constexpr int kPartStride = kHeadDim + 4;
constexpr int kPartO = 4;

// ---- RMSNorm -----------------------------------------------------------------
__global__ void __launch_bounds__(256) rmsnorm_kernel(const __half* __restrict__ x,
                                                      const __half* __restrict__ gamma, int64_t H,
                                                      float eps, __half* __restrict__ y) {
  griddep_wait();
  griddep_launch_dependents();
  __shared__ float red[8];
  const int64_t m = blockIdx.x;
  const __half* xr = x + m * H;
  // sum of squares over 8-value chunks: thread t takes chunks c = t, t + 256,
  // ..., the values of a chunk in order (the order the projections that
  // normalise their own staged rows use, so both give the same bits)
  float ss = 0.0f;
  const int64_t nch = H / 8;
  const bool vec = (reinterpret_cast<uintptr_t>(xr) & 15) == 0;
  for (int64_t c = threadIdx.x; c < nch; c += blockDim.x) {
    if (vec) {
      ss = sumsq8(reinterpret_cast<const uint4*>(xr)[c], ss);
    } else {
      for (int e = 0; e < 8; ++e) {
        const float v = __half2float(xr[8 * c + e]);
        ss = fmaf(v, v, ss);
      }
    }
  }
  if (threadIdx.x == nch % blockDim.x)  // the ragged tail chunk (H % 8 values)
    for (int64_t h = 8 * nch; h < H; ++h) {
      const float v = __half2float(xr[h]);
      ss = fmaf(v, v, ss);
    }
  ss = warp_sum(ss);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  float t = 0.0f;
  for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t += red[w];
  const float r = 1.0f / sqrtf(t / (float)H + eps);
  for (int64_t h = threadIdx.x; h < H; h += blockDim.x)
    y[m * H + h] = __float2half_rn(__half2float(xr[h]) * r * __half2float(gamma[h]));
}

// ---- RoPE --------------------------------------------------------------------
// Inverse frequencies theta^(-2d/D), d < D/2, computed on the host in fp64.
struct RopeFreq {
  double f[kHeadDim / 2];
};

// cos and sin of pos * f: the angle and its reduction modulo 2 pi in fp64
// (positions up to 2^20 keep the reduced angle within ~1e-10), then fp32
// sincosf of the reduced angle.
__device__ __forceinline__ float2 rope_cs(int pos, double f) {
  const double a = (double)pos * f;
  const double k = rint(a * 0.15915494309189535);       // a / (2 pi)
  double r = fma(-k, 6.283185307179586, a);              // 2 pi, head
  r = fma(-k, 2.4492935982947064e-16, r);                 // 2 pi, tail
  float s, c;
  sincosf((float)r, &s, &c);
  return make_float2(c, s);
}

// The rotated pair (x1 c - x2 s, x2 c + x1 s), rounded to fp16 as the cache
// stores it; the products and differences are rounded one by one (no
// contraction), so the separate append and the fused attention write the
// same bits.
__device__ __forceinline__ void rope_rotate_f16(float x1, float x2, float2 cs, __half& y1, __half& y2) {
  y1 = __float2half_rn(__fsub_rn(__fmul_rn(x1, cs.x), __fmul_rn(x2, cs.y)));
  y2 = __float2half_rn(__fadd_rn(__fmul_rn(x2, cs.x), __fmul_rn(x1, cs.y)));
}

// One CTA per (token row, key/value head): rotate the new key, copy the
// value, both into the caches at the token's position.
__global__ void __launch_bounds__(64) kv_append_kernel(const __half* __restrict__ qkv, int T, int Hq,
                                                       int Hkv, const int32_t* __restrict__ pos0,
                                                       const RopeFreq rf, __half* __restrict__ kc,
                                                       __half* __restrict__ vc, int64_t max_ctx) {
  griddep_wait();
  griddep_launch_dependents();
  const int row = blockIdx.x, h = blockIdx.y;
  const int b = row / T, t = row - b * T;
  const int pos = pos0[b] + t;
  if (pos < 0 || (int64_t)pos >= max_ctx) {
    if (threadIdx.x == 0) atomicOr(&g_attn_status, SQ_DEV_BAD_POSITION);
    return;
  }
  const int64_t width = (int64_t)(Hq + 2 * Hkv) * kHeadDim;
  const __half* kr = qkv + row * width + (int64_t)(Hq + h) * kHeadDim;
  const __half* vr = qkv + row * width + (int64_t)(Hq + Hkv + h) * kHeadDim;
  const int64_t dst = (((int64_t)b * Hkv + h) * max_ctx + pos) * kHeadDim;
  const int d = threadIdx.x;  // pair (d, d + D/2)
  const float2 cs = rope_cs(pos, rf.f[d]);
  rope_rotate_f16(__half2float(kr[d]), __half2float(kr[d + kHeadDim / 2]), cs, kc[dst + d],
                  kc[dst + d + kHeadDim / 2]);
  vc[dst + d] = vr[d];
  vc[dst + d + kHeadDim / 2] = vr[d + kHeadDim / 2];
}

// ---- attention ----------------------------------------------------------------
__device__ __forceinline__ float h2f_lo(uint32_t w) { return __half2float(__ushort_as_half((uint16_t)(w & 0xffffu))); }
__device__ __forceinline__ float h2f_hi(uint32_t w) { return __half2float(__ushort_as_half((uint16_t)(w >> 16))); }

struct AttnArgs {
  const __half* qkv;
  const __half* kc;
  const __half* vc;
  __half* kcw;  // the same caches, written when append != 0
  __half* vcw;
  int append;   // the new tokens' keys/values are appended by the chunk that holds them
  const int32_t* pos0;
  __half* out;
  float* part;  // [(B*Hkv) * nsplit * Q * kPartStride]: per query (m, l, -, -, o[D])
  int B, T, Hq, Hkv, G, Q;
  int64_t max_ctx;
  int nsplit;
  float scale;  // 1 / sqrt(D)
  RopeFreq rf;
};

// Shared memory (fp32): cos/sin of the T positions [T][D/2], q [Q][kRowPad]
// (rotated, scaled), k [C][kRowPad], v [C][kRowPad], scores [Q][C].
// Queries q = g * T + t (head kvh * G + g, token t).
__global__ void __launch_bounds__(kAttnThreads) attention_partial_kernel(const AttnArgs a) {
  griddep_wait();
  griddep_launch_dependents();
  extern __shared__ __align__(16) float sm[];
  const int Q = a.Q, T = a.T;
  float2* cst = reinterpret_cast<float2*>(sm);                  // [T][D/2]
  float* qs = sm + 2 * kMaxT * (kHeadDim / 2);                  // [Q][kRowPad]
  float* ks = qs + Q * kRowPad;                                 // [C][kRowPad]
  float* vs = ks + kAttnChunk * kRowPad;                        // [C][kRowPad]
  float* sc = vs + kAttnChunk * kRowPad;                        // [Q][C]
  const int bh = blockIdx.x, split = blockIdx.y;
  const int b = bh / a.Hkv, kvh = bh - b * a.Hkv;
  const int tid = threadIdx.x;
  const int p0 = a.pos0[b];
  const int64_t len = (int64_t)p0 + T;  // cache entries after the append
  const int64_t j0 = (int64_t)split * kAttnChunk;
  float* part = a.part + ((int64_t)bh * a.nsplit + split) * Q * kPartStride;
  if (a.append && (p0 < 0 || len > a.max_ctx) && split == 0 && tid == 0)
    atomicOr(&g_attn_status, SQ_DEV_BAD_POSITION);
  if (j0 >= len || p0 < 0 || len > a.max_ctx) {  // empty chunk: neutral partials
    for (int q = tid; q < Q; q += kAttnThreads) {
      part[(int64_t)q * kPartStride] = -INFINITY;
      part[(int64_t)q * kPartStride + 1] = 0.0f;
    }
    return;
  }
  const int nk = (int)(len - j0 < kAttnChunk ? len - j0 : kAttnChunk);
  const int64_t width = (int64_t)(a.Hq + 2 * a.Hkv) * kHeadDim;
  const int64_t cbase = (((int64_t)b * a.Hkv + kvh) * a.max_ctx + j0) * kHeadDim;
  // positions p0 .. p0+T-1 are the new tokens: with append, this chunk's
  // share of them is rotated from qkv, written to the caches and used
  // directly (every position belongs to one chunk, so each is written once)
  const int j_new = a.append ? (int)((int64_t)p0 - j0) : kAttnChunk;  // first new key of the chunk
  const int n_old = j_new < nk ? (j_new > 0 ? j_new : 0) : nk;         // keys read from the caches
  // cached keys and values: 16-byte pieces (8 values), all of a thread's
  // loads issued before the RoPE table is computed
  constexpr int kPieces = kAttnChunk * kHeadDim / 8;
  constexpr int kPerThread = kPieces / kAttnThreads;
  static_assert(kPieces % kAttnThreads == 0, "whole pieces per thread");
  uint4 kraw[kPerThread], vraw[kPerThread];
#pragma unroll
  for (int r = 0; r < kPerThread; ++r) {
    const int pc = tid + r * kAttnThreads;
    const int j = pc / (kHeadDim / 8);
    const bool in = j < n_old;
    kraw[r] = in ? *reinterpret_cast<const uint4*>(a.kc + cbase + (int64_t)pc * 8) : make_uint4(0u, 0u, 0u, 0u);
    vraw[r] = in ? *reinterpret_cast<const uint4*>(a.vc + cbase + (int64_t)pc * 8) : make_uint4(0u, 0u, 0u, 0u);
  }
  for (int idx = tid; idx < T * (kHeadDim / 2); idx += kAttnThreads) {
    const int t = idx / (kHeadDim / 2), d = idx - t * (kHeadDim / 2);
    cst[idx] = rope_cs(p0 + t, a.rf.f[d]);
  }
#pragma unroll
  for (int r = 0; r < kPerThread; ++r) {
    const int pc = tid + r * kAttnThreads;
    const int j = pc / (kHeadDim / 8), d8 = pc - j * (kHeadDim / 8);
    if (j >= n_old && j < nk) continue;  // a new key: written below
    const uint32_t kw[4] = {kraw[r].x, kraw[r].y, kraw[r].z, kraw[r].w};
    const uint32_t vw[4] = {vraw[r].x, vraw[r].y, vraw[r].z, vraw[r].w};
    float4* kd = reinterpret_cast<float4*>(ks + j * kRowPad + d8 * 8);
    float4* vd = reinterpret_cast<float4*>(vs + j * kRowPad + d8 * 8);
    kd[0] = make_float4(h2f_lo(kw[0]), h2f_hi(kw[0]), h2f_lo(kw[1]), h2f_hi(kw[1]));
    kd[1] = make_float4(h2f_lo(kw[2]), h2f_hi(kw[2]), h2f_lo(kw[3]), h2f_hi(kw[3]));
    vd[0] = make_float4(h2f_lo(vw[0]), h2f_hi(vw[0]), h2f_lo(vw[1]), h2f_hi(vw[1]));
    vd[1] = make_float4(h2f_lo(vw[2]), h2f_hi(vw[2]), h2f_lo(vw[3]), h2f_hi(vw[3]));
  }
  if (n_old < nk) {  // new keys of this chunk (append): rotate from qkv
    __syncthreads();  // cst is read below
    for (int idx = n_old * kHeadDim + tid; idx < nk * kHeadDim; idx += kAttnThreads) {
      const int j = idx / kHeadDim, d = idx - j * kHeadDim;
      const int t = (int)(j0 + j - p0);
      const __half* row = a.qkv + ((int64_t)b * T + t) * width;
      const __half* kr = row + (int64_t)(a.Hq + kvh) * kHeadDim;
      const __half vh = row[(int64_t)(a.Hq + a.Hkv + kvh) * kHeadDim + d];
      const int pd = d & (kHeadDim / 2 - 1);
      __half y1, y2;
      rope_rotate_f16(__half2float(kr[pd]), __half2float(kr[pd + kHeadDim / 2]), cst[t * (kHeadDim / 2) + pd],
                      y1, y2);
      const __half kh = d < kHeadDim / 2 ? y1 : y2;
      a.kcw[cbase + idx] = kh;
      a.vcw[cbase + idx] = vh;
      ks[j * kRowPad + d] = __half2float(kh);
      vs[j * kRowPad + d] = __half2float(vh);
    }
  }
  __syncthreads();
  // queries: each thread rotates 8 pairs (d, d + D/2) read as two 16-byte
  // pieces (q rows are 16-byte aligned when qkv is: D = 128 halves)
  const bool qvec = (reinterpret_cast<uintptr_t>(a.qkv) & 15) == 0;
  for (int idx = tid; idx < Q * (kHeadDim / 16); idx += kAttnThreads) {
    const int q = idx / (kHeadDim / 16), d0 = (idx - q * (kHeadDim / 16)) * 8;
    const int g = q / T, t = q - g * T;
    const __half* qr = a.qkv + ((int64_t)b * T + t) * width + (int64_t)(kvh * a.G + g) * kHeadDim;
    float x1[8], x2[8];
    if (qvec) {
      const uint4 u1 = *reinterpret_cast<const uint4*>(qr + d0);
      const uint4 u2 = *reinterpret_cast<const uint4*>(qr + d0 + kHeadDim / 2);
      const uint32_t w1[4] = {u1.x, u1.y, u1.z, u1.w}, w2[4] = {u2.x, u2.y, u2.z, u2.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        x1[2 * e] = h2f_lo(w1[e]);
        x1[2 * e + 1] = h2f_hi(w1[e]);
        x2[2 * e] = h2f_lo(w2[e]);
        x2[2 * e + 1] = h2f_hi(w2[e]);
      }
    } else {
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        x1[e] = __half2float(qr[d0 + e]);
        x2[e] = __half2float(qr[d0 + e + kHeadDim / 2]);
      }
    }
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const float2 cs = cst[t * (kHeadDim / 2) + d0 + e];
      qs[q * kRowPad + d0 + e] = (x1[e] * cs.x - x2[e] * cs.y) * a.scale;
      qs[q * kRowPad + d0 + e + kHeadDim / 2] = (x2[e] * cs.x + x1[e] * cs.y) * a.scale;
    }
  }
  __syncthreads();
  // scores: each thread a 2-query x 4-key tile, 16-byte shared loads along D
  const int qpairs = (Q + 1) / 2;
  for (int tile = tid; tile < qpairs * (kAttnChunk / 4); tile += kAttnThreads) {
    const int qp = tile / (kAttnChunk / 4), kq = tile - qp * (kAttnChunk / 4);
    const int q0 = 2 * qp, q1 = q0 + 1 < Q ? q0 + 1 : q0;
    float acc[2][4] = {};
    const float4* qa = reinterpret_cast<const float4*>(qs + q0 * kRowPad);
    const float4* qb = reinterpret_cast<const float4*>(qs + q1 * kRowPad);
#pragma unroll 4
    for (int d4 = 0; d4 < kHeadDim / 4; ++d4) {
      const float4 x0 = qa[d4], x1 = qb[d4];
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        const float4 kv = reinterpret_cast<const float4*>(ks + (4 * kq + kk) * kRowPad)[d4];
        acc[0][kk] = fmaf(x0.x, kv.x, fmaf(x0.y, kv.y, fmaf(x0.z, kv.z, fmaf(x0.w, kv.w, acc[0][kk]))));
        acc[1][kk] = fmaf(x1.x, kv.x, fmaf(x1.y, kv.y, fmaf(x1.z, kv.z, fmaf(x1.w, kv.w, acc[1][kk]))));
      }
    }
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const int q = i ? q1 : q0;
      if (i && q1 == q0) break;
      const int t = q % T;
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        const int j = 4 * kq + kk;
        sc[q * kAttnChunk + j] = (j < nk && j0 + j <= (int64_t)p0 + t) ? acc[i][kk] : -INFINITY;
      }
    }
  }
  __syncthreads();
  // per query: chunk max, exp, sum (one warp per query, one key per lane)
  static_assert(kAttnChunk == 32, "one key per lane");
  const int warp = tid >> 5, lane = tid & 31;
  for (int q = warp; q < Q; q += kAttnThreads / 32) {
    const float v = sc[q * kAttnChunk + lane];
    const float mx = warp_max(v);
    const float e = mx == -INFINITY ? 0.0f : expf(v - mx);
    sc[q * kAttnChunk + lane] = e;
    const float l = warp_sum(e);
    if (lane == 0) {
      part[(int64_t)q * kPartStride] = mx;
      part[(int64_t)q * kPartStride + 1] = l;
    }
  }
  __syncthreads();
  // weighted values: each thread a 2-query x 4-dim tile
  for (int tile = tid; tile < qpairs * (kHeadDim / 4); tile += kAttnThreads) {
    const int qp = tile / (kHeadDim / 4), d4 = tile - qp * (kHeadDim / 4);
    const int q0 = 2 * qp, q1 = q0 + 1 < Q ? q0 + 1 : q0;
    float4 o0 = make_float4(0.f, 0.f, 0.f, 0.f), o1 = o0;
    for (int j = 0; j < nk; ++j) {
      const float e0 = sc[q0 * kAttnChunk + j], e1 = sc[q1 * kAttnChunk + j];
      const float4 vv = reinterpret_cast<const float4*>(vs + j * kRowPad)[d4];
      o0.x = fmaf(e0, vv.x, o0.x); o0.y = fmaf(e0, vv.y, o0.y);
      o0.z = fmaf(e0, vv.z, o0.z); o0.w = fmaf(e0, vv.w, o0.w);
      o1.x = fmaf(e1, vv.x, o1.x); o1.y = fmaf(e1, vv.y, o1.y);
      o1.z = fmaf(e1, vv.z, o1.z); o1.w = fmaf(e1, vv.w, o1.w);
    }
    *reinterpret_cast<float4*>(part + (int64_t)q0 * kPartStride + kPartO + 4 * d4) = o0;
    if (q1 != q0) *reinterpret_cast<float4*>(part + (int64_t)q1 * kPartStride + kPartO + 4 * d4) = o1;
  }
}

// One CTA per (sequence and key/value head, query): the chunk maxima and
// sums are read in parallel into shared memory, then each thread (one per
// head dimension) merges the chunks' weighted values.
__global__ void __launch_bounds__(kHeadDim) attention_combine_kernel(const AttnArgs a) {
  griddep_wait();
  griddep_launch_dependents();
  extern __shared__ float cm[];  // [2 * nsplit]: chunk max, chunk sum
  __shared__ float red[kHeadDim / 32];
  const int bh = blockIdx.x, q = blockIdx.y, d = threadIdx.x;
  const int b = bh / a.Hkv, kvh = bh - b * a.Hkv;
  const float* base = a.part + (int64_t)bh * a.nsplit * a.Q * kPartStride;
  float M = -INFINITY;
  for (int s = d; s < a.nsplit; s += kHeadDim) {
    const float* ps = base + ((int64_t)s * a.Q + q) * kPartStride;
    cm[s] = ps[0];
    cm[a.nsplit + s] = ps[1];
    M = fmaxf(M, ps[0]);
  }
  M = warp_max(M);
  if ((d & 31) == 0) red[d >> 5] = M;
  __syncthreads();
  M = -INFINITY;
#pragma unroll
  for (int w = 0; w < kHeadDim / 32; ++w) M = fmaxf(M, red[w]);
  float L = 0.0f, O = 0.0f;
  if (M != -INFINITY)
    for (int s0 = 0; s0 < a.nsplit; s0 += 8) {
      // the chunks' weighted values, eight loads in flight; then the same
      // sums, chunk by chunk in order
      float ov[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int s = s0 + u;
        ov[u] = (s < a.nsplit && cm[s] != -INFINITY) ? base[((int64_t)s * a.Q + q) * kPartStride + kPartO + d]
                                                      : 0.0f;
      }
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int s = s0 + u;
        if (s >= a.nsplit) break;
        const float ms = cm[s];
        if (ms == -INFINITY) continue;
        const float w = expf(ms - M);
        L = fmaf(w, cm[a.nsplit + s], L);
        O = fmaf(w, ov[u], O);
      }
    }
  const int g = q / a.T, t = q - g * a.T;
  const int64_t row = (int64_t)b * a.T + t;
  a.out[row * (int64_t)a.Hq * kHeadDim + (int64_t)(kvh * a.G + g) * kHeadDim + d] =
      __float2half_rn(L > 0.0f ? O / L : 0.0f);
}

// ---- embedding ---------------------------------------------------------------------
// out[m, :] = table[ids[m], :] (fp16 copy, 16-byte pieces when aligned); an id
// outside [0, V) gives a zero row and sets SQ_DEV_BAD_TOKEN_ID.
__global__ void __launch_bounds__(256) embed_kernel(const int32_t* __restrict__ ids, int64_t ids_stride,
                                                    const __half* __restrict__ table, int64_t V,
                                                    int64_t H, __half* __restrict__ out) {
  griddep_wait();
  griddep_launch_dependents();
  const int64_t m = blockIdx.x;
  const int32_t id = ids[m * ids_stride];
  const bool ok = id >= 0 && (int64_t)id < V;
  if (!ok && threadIdx.x == 0) atomicOr(&g_attn_status, SQ_DEV_BAD_TOKEN_ID);
  const __half* src = table + (ok ? (int64_t)id : 0) * H;
  __half* dst = out + m * H;
  if ((H & 7) == 0 && ((reinterpret_cast<uintptr_t>(table) | reinterpret_cast<uintptr_t>(out)) & 15) == 0) {
    for (int64_t i = threadIdx.x; i < H / 8; i += blockDim.x)
      reinterpret_cast<uint4*>(dst)[i] = ok ? reinterpret_cast<const uint4*>(src)[i] : make_uint4(0, 0, 0, 0);
  } else {
    for (int64_t i = threadIdx.x; i < H; i += blockDim.x) dst[i] = ok ? src[i] : __ushort_as_half(0);
  }
}

cudaError_t launch_embed(const int32_t* ids, int M, int64_t ids_stride, const __half* table, int64_t V,
                         int64_t H, __half* out, cudaStream_t st) {
  if (M == 0) return cudaSuccess;
  return launch_pdl(embed_kernel, dim3((unsigned)M), dim3(256), 0, st, ids, ids_stride, table, V, H, out);
}

// ---- speculative bookkeeping (Sec. III-D.4: the accepted prefix plus the
// correction becomes the context of the next cycle) ----------------------------------
// One thread per sequence.  Appends the n + 1 committed tokens to the history
// and derives the next cycle's inputs: the positions of the K draft steps and
// of the verify pass, and the last two committed tokens (the draft's first
// step re-reads the second-last one, whose key/value the draft may not have
// computed when every draft was accepted).
__global__ void spec_commit_kernel(const int32_t* __restrict__ n_acc, const int32_t* __restrict__ tokens,
                                   int ldt, int B, int K, int32_t* __restrict__ hist, int cap,
                                   int32_t* __restrict__ len, int32_t* __restrict__ pos,
                                   int32_t* __restrict__ last2) {
  griddep_wait();
  griddep_launch_dependents();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  int L = len[b];
  int32_t* h = hist + (int64_t)b * cap;
  bool bad = L < 0 || L > cap;
  if (!bad) {
    const int na = n_acc ? n_acc[b] : 0;
    if (na >= ldt) {
      bad = true;
    } else if (na >= 0) {
      const int cnt = na + 1 < cap - L ? na + 1 : cap - L;
      for (int i = 0; i < cnt; ++i) h[L + i] = tokens[(int64_t)b * ldt + i];
      if (cnt < na + 1) bad = true;
      L += cnt;
    }
  }
  if (bad || L < 2) {
    atomicOr(&g_attn_status, SQ_DEV_BAD_POSITION);
    if (L < 0 || L > cap) L = 0;
  }
  len[b] = L;
  last2[2 * b] = L >= 2 ? h[L - 2] : -1;
  last2[2 * b + 1] = L >= 1 ? h[L - 1] : -1;
  if (K >= 1) pos[b] = L - 2;
  for (int k = 1; k < K; ++k) pos[(int64_t)k * B + b] = L - 1 + k;
  pos[(int64_t)K * B + b] = L - 1;
}

// verify_tokens[b, :] = (last committed token, draft 1 .. K); draft[b, k] =
// samples[k, b] (the draft steps write one token per sequence).
__global__ void spec_drafts_kernel(const int32_t* __restrict__ samples, const int32_t* __restrict__ last2,
                                   int B, int K, int32_t* __restrict__ verify, int32_t* __restrict__ draft) {
  griddep_wait();
  griddep_launch_dependents();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  verify[(int64_t)b * (K + 1)] = last2[2 * b + 1];
  for (int k = 0; k < K; ++k) {
    const int32_t t = samples[(int64_t)k * B + b];
    verify[(int64_t)b * (K + 1) + 1 + k] = t;
    draft[(int64_t)b * K + k] = t;
  }
}

cudaError_t launch_spec_commit(const int32_t* n, const int32_t* tokens, int ldt, int B, int K, int32_t* hist,
                               int cap, int32_t* len, int32_t* pos, int32_t* last2, cudaStream_t st) {
  if (B == 0) return cudaSuccess;
  return launch_pdl(spec_commit_kernel, dim3((unsigned)((B + 127) / 128)), dim3(128), 0, st, n, tokens, ldt,
                    B, K, hist, cap, len, pos, last2);
}

cudaError_t launch_spec_drafts(const int32_t* samples, const int32_t* last2, int B, int K, int32_t* verify,
                               int32_t* draft, cudaStream_t st) {
  if (B == 0) return cudaSuccess;
  return launch_pdl(spec_drafts_kernel, dim3((unsigned)((B + 127) / 128)), dim3(128), 0, st, samples, last2,
                    B, K, verify, draft);
}

// ---- rollback -------------------------------------------------------------------
__global__ void kv_rollback_kernel(const int32_t* __restrict__ base, const int32_t* __restrict__ n,
                                   int B, int limit, int32_t* __restrict__ len) {
  griddep_wait();
  griddep_launch_dependents();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  const int na = n[b];
  len[b] = na < 0 ? base[b] : base[b] + (na + 1 < limit ? na + 1 : limit);
}

// ---- host side -------------------------------------------------------------------
cudaError_t launch_rmsnorm(const __half* x, const __half* gamma, int M, int64_t H, float eps, __half* y,
                           cudaStream_t st) {
  if (M == 0) return cudaSuccess;
  return launch_pdl(rmsnorm_kernel, dim3((unsigned)M), dim3(256), 0, st, x, gamma, H, eps, y);
}

static RopeFreq rope_freq(double theta) {
  RopeFreq rf;
  for (int d = 0; d < kHeadDim / 2; ++d) rf.f[d] = pow(theta, -2.0 * d / (double)kHeadDim);
  return rf;
}

cudaError_t launch_kv_append(const __half* qkv, int B, int T, int Hq, int Hkv, const int32_t* pos0,
                             double theta, __half* kc, __half* vc, int64_t max_ctx, cudaStream_t st) {
  if (B == 0 || T == 0) return cudaSuccess;
  return launch_pdl(kv_append_kernel, dim3((unsigned)(B * T), (unsigned)Hkv), dim3(kHeadDim / 2), 0, st,
                    qkv, T, Hq, Hkv, pos0, rope_freq(theta), kc, vc, max_ctx);
}

size_t attention_workspace_bytes(int B, int T, int Hq, int Hkv, int64_t max_ctx) {
  if (B < 0 || T < 0 || Hkv <= 0 || max_ctx <= 0) return 0;
  const int64_t nsplit = (max_ctx + kAttnChunk - 1) / kAttnChunk;
  const int64_t Q = (int64_t)(Hq / Hkv) * T;
  return (size_t)B * Hkv * nsplit * Q * kPartStride * sizeof(float);
}

size_t attention_smem_bytes(int Q) {
  return ((size_t)2 * kMaxT * (kHeadDim / 2) + (size_t)Q * kRowPad + (size_t)2 * kAttnChunk * kRowPad +
          (size_t)Q * kAttnChunk) * sizeof(float);
}

int attention_max_tokens() { return kMaxT; }

cudaError_t launch_attention(const __half* qkv, int B, int T, int Hq, int Hkv, const int32_t* pos0,
                             double theta, const __half* kc, const __half* vc, int64_t max_ctx,
                             __half* out, void* ws, cudaStream_t st, __half* kc_append,
                             __half* vc_append) {
  if (B == 0 || T == 0) return cudaSuccess;
  AttnArgs a = {};
  a.qkv = qkv;
  a.kc = kc;
  a.vc = vc;
  a.kcw = kc_append;
  a.vcw = vc_append;
  a.append = kc_append != nullptr && vc_append != nullptr;
  a.pos0 = pos0;
  a.out = out;
  a.part = reinterpret_cast<float*>(ws);
  a.B = B;
  a.T = T;
  a.Hq = Hq;
  a.Hkv = Hkv;
  a.G = Hq / Hkv;
  a.Q = a.G * T;
  a.max_ctx = max_ctx;
  a.nsplit = (int)((max_ctx + kAttnChunk - 1) / kAttnChunk);
  a.rf = rope_freq(theta);
  a.scale = 1.0f / sqrtf((float)kHeadDim);
  const size_t smem = attention_smem_bytes(a.Q);
  static int smem_set[64] = {0};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if ((int)smem > smem_set[dev]) {
    e = cudaFuncSetAttribute(attention_partial_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    smem_set[dev] = (int)smem;
  }
  e = launch_pdl(attention_partial_kernel, dim3((unsigned)(B * Hkv), (unsigned)a.nsplit),
                 dim3(kAttnThreads), smem, st, a);
  if (e != cudaSuccess) return e;
  return launch_pdl(attention_combine_kernel, dim3((unsigned)(B * Hkv), (unsigned)a.Q), dim3(kHeadDim),
                    (size_t)2 * a.nsplit * sizeof(float), st, a);
}

cudaError_t launch_kv_rollback(const int32_t* base, const int32_t* n, int B, int limit, int32_t* len,
                               cudaStream_t st) {
  if (B == 0) return cudaSuccess;
  return launch_pdl(kv_rollback_kernel, dim3((unsigned)((B + 127) / 128)), dim3(128), 0, st, base, n, B,
                    limit, len);
}

cudaError_t take_attn_status(uint32_t* bits) {
  uint32_t v = 0, zero = 0;
  cudaError_t e = cudaMemcpyFromSymbol(&v, g_attn_status, sizeof(v));
  if (e != cudaSuccess) return e;
  if (v) e = cudaMemcpyToSymbol(g_attn_status, &zero, sizeof(zero));
  *bits |= v;
  return e;
}

}  // namespace sq
