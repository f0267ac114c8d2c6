// sq_ring.cu -- linear layer for one to eight activation rows (the draft
// pass at small batch, Sec. III-D.2; the verify pass of one sequence, Sec.
// III-D.3) streamed through a shared-memory ring, products on the tensor
// cores' register-operand path.
//
// Used for the large single-row matrices (fused gate/up, lm_head) where it
// measured faster than the GEMV family; the engine rule is in sq_plan.cu.
//
// Design:
//   * one CTA per SM (12 or 16 warps for INT4, 8 for FP16 / FP8) takes a
//     contiguous share of the 16-row output tiles; each warp owns a private
//     ring of NS 4 KB slots and walks its jobs (one tile, one range of
//     64-byte row units; a tile's units are split over S warps when tiles
//     are few) as stages of 4 units of 16 rows (2 units of the 32 rows of the
//     fused gate/up);
//   * a stage is requested with 16-byte asynchronous copies (cp.async, one
//     warp instruction moves 512 contiguous bytes) that arrive on the slot's
//     mbarrier; the ring is filled BEFORE waiting on the kernel that produces
//     x (weights never depend on it);
//   * products: mma.sync m16n8k16, fp16 x fp16 -> fp32.  A = 16 weight rows
//     from the slot (INT4 nibbles and E4M3 codes turned into exact fp16
//     values in registers), B = up to eight activation rows, one per column
//     (lanes of columns past M read row M - 1; those columns are dropped),
//     so M <= 8 rows cost the instructions of one.  INT4 groups
//     are summed from zero in four (fused gate/up: two) independent
//     accumulators and scaled by the group's fp16 scale into an fp32 sum;
//     the scales travel with the stage (4-byte copies into a 128-byte scale
//     slot beside it, so INT4 rows need an even number of groups).  FP8 and FP16
//     accumulate in two alternating accumulator sets;
//   * S > 1: the warps' fp32 sums of a tile are added in warp order through
//     shared memory (deterministic).
// Slots hold rows 256 (128) bytes apart with the 16-byte pieces of odd rows
// swapped within each 128-byte line, so the two rows a group of eight lanes
// reads lie in different bank halves.  Every wait is bounded in time; a
// wait that runs out sets SQ_DEV_TIMEOUT, the warp stops requesting and
// waits (bounded) for the copies it still has in flight before it exits.
#include "sq_internal.h"

namespace sq {

namespace {

// Warps per CTA: 8 for FP16 / FP8 (memory-bound); for INT4 (bound by the
// nibble conversion: many warps hide its latency; 8 warps measured 1.3x
// slower at one row) 16 at one or two activation rows and 12 from three rows
// on, unless the staged activations leave no room for them.  Measured on the
// 14B draft pass: 12 warps (up to 168 registers a thread instead of 128)
// take 4 rows in 599 us against 654 us with 16 and 8 rows in 753 us against
// 864 us, but cost 2-10 us at one and two rows; 10 or 14 warps are no better.
constexpr int kWarpsHalf = 8;
constexpr int kWarpsMid = 12;
constexpr int kWarpsFull = 16;
constexpr int kStageBytes = 4096;          // weights of one ring slot
constexpr int kScaleBytes = 128;           // INT4 group scales of one slot
constexpr int kUnitBytes = 64;             // a unit: 64 bytes of one weight row
constexpr int kUps16 = 4;                  // units per stage of 16 rows
constexpr int kUps32 = 2;                  // units per stage of 32 rows (fused gate/up)
constexpr int kSmemFull = 227 * 1024;     // the whole opt-in shared memory of an SM
constexpr uint64_t kWaitNs = 2000000000ull;
constexpr uint64_t kDrainNs = 1000000ull;

struct RingArgs {
  const __half* x;         // [M, K]
  const uint8_t* w;        // weight rows
  const void* scales;      // INT4 fp16 [rows, K/128]; FP8 fp32 [rows]; FP16 unused
  const __half* bias;      // [rows] or null
  const __half* residual;  // [M, N] or null
  __half* y;               // [M, N]
  int64_t N;               // output columns
  int64_t row_bytes;
  int64_t T;               // 16-column output tiles
  int32_t U;               // 64-byte units per weight row (INT4: one unit = one group)
  int32_t S;               // warps sharing one tile's units
  int32_t silu;            // fused gate/up: rows [0, N) gate, [N, 2N) up
  int32_t ns;              // ring slots per warp
  int32_t x_bytes;         // shared bytes of the staged activations
  int32_t K;
  int32_t ugran;           // parts of a row start on multiples of this many units
  int32_t tmax;            // most tiles a CTA owns (ceil(T / grid))
  int32_t M;               // activation rows, 1 .. 8 (the MMA's N columns)
  int32_t x_stride;        // shared bytes between staged activation rows
};

static __device__ unsigned int g_ring_status;

__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ bool mbar_wait_ns(uint64_t* bar, uint32_t parity, uint64_t limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  while (!mbar_try_wait(bar, parity))
    if (global_ns() - t0 > limit_ns) return false;
  return true;
}

__device__ __forceinline__ uint4 lds16(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"(addr));
  return v;
}

__device__ __forceinline__ void mma16816(float d[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
  asm("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Eight activations (x0,x1)(x2,x3)(x4,x5)(x6,x7) to the pairs the INT4
// conversion yields: (x0,x4)(x2,x6)(x1,x5)(x3,x7).
__device__ __forceinline__ uint4 int4_x_order(const uint4 v) {
  return make_uint4(__byte_perm(v.x, v.z, 0x5410), __byte_perm(v.y, v.w, 0x5410),
                    __byte_perm(v.x, v.z, 0x7632), __byte_perm(v.y, v.w, 0x7632));
}

// Byte offset of 16-byte piece p of row r in a slot with rows of rb bytes:
// the pieces of odd rows are swapped with their partners four pieces away
// (64 bytes), so rows 2i and 2i + 1 read at the same column fall in different
// bank halves.
__device__ __forceinline__ uint32_t slot_off(int r, int p, int rb) {
  return (uint32_t)(r * rb + ((p ^ ((r & 1) << 2)) << 4));
}

// A warp's position: job j (tile ta + j / S, part j % S of its units), first
// unit u of the stage, end unit u1 of the job.  Warp w takes the jobs w,
// w + NW, w + 2 NW, ... of its CTA.
struct Cur {
  int j;
  int u, u1;
  int64_t tile;
  bool live;
};

__device__ __forceinline__ void cur_job(const RingArgs& a, int64_t ta, int64_t tb, Cur& c) {
  c.tile = ta + c.j / a.S;
  c.live = c.tile < tb;
  const int p = c.j % a.S;
  const int ug = a.ugran;  // INT4: parts start on even units (4-byte scale copies)
  c.u = ug * (p * (a.U / ug) / a.S);
  c.u1 = p + 1 == a.S ? a.U : ug * ((p + 1) * (a.U / ug) / a.S);
}

template <int NW, bool SILU>
__device__ __forceinline__ void cur_next(const RingArgs& a, int64_t ta, int64_t tb, Cur& c) {
  c.u += SILU ? kUps32 : kUps16;
  if (c.u < c.u1) return;
  c.j += NW;
  cur_job(a, ta, tb, c);
}

// Request the stage at c into slot `slot` with 16-byte asynchronous copies:
// 16 rows x 256 B (lane l copies piece l & 15 of rows 2i + l / 16) or, for
// the fused gate/up, 32 rows x 128 B (piece l & 7 of rows 4i + l / 8, gate
// rows first); one warp instruction moves 512 contiguous bytes.  INT4: every
// lane also copies 4 bytes of group scales (16 rows x 2 copies, or 32 rows
// x 1) into the scale slot.  Then every lane arms the slot's mbarrier to
// arrive when its copies have landed.  Rows past N are not copied.
template <int WK, bool SILU>
__device__ __forceinline__ void issue_stage(const RingArgs& a, const Cur& c, uint32_t slot, uint32_t sslot,
                                            uint64_t* bar, int lane) {
  constexpr int UPS = SILU ? kUps32 : kUps16;
  constexpr int LPR = UPS * 4;   // 16-byte pieces of a full stage row
  constexpr int RPI = 32 / LPR;  // rows per instruction
  constexpr int RB = UPS * kUnitBytes;
  const int nu = min(UPS, c.u1 - c.u);
  const int piece = lane % LPR;
  const int r0 = lane / LPR;
  const int64_t n0 = c.tile * 16;
  if (piece < nu * 4) {
    const uint8_t* src = a.w + (n0 + r0) * a.row_bytes + (int64_t)c.u * kUnitBytes + piece * 16;
    const int64_t step = (int64_t)RPI * a.row_bytes;
    const int64_t up = (a.N - 16) * a.row_bytes;  // gate row r -> up row r: + N rows
    const bool full = n0 + 16 <= a.N;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int r = i * RPI + r0;
      const uint8_t* p = src + i * step + ((SILU && r >= 16) ? up : 0);
      if (full || n0 + (r & 15) < a.N)
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(slot + slot_off(r, piece, RB)), "l"(p)
                     : "memory");
    }
  }
  if constexpr (WK == SQ_W_INT4) {
    const int r = SILU ? lane : lane >> 1;
    const int cpy = SILU ? 0 : lane & 1;
    const int64_t n = n0 + (r & 15);
    if (2 * cpy < nu && n < a.N) {
      const int64_t row = (SILU && r >= 16 ? a.N : 0) + n;
      const uint8_t* src = reinterpret_cast<const uint8_t*>(a.scales) + (row * a.U + c.u + 2 * cpy) * 2;
      asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(sslot + r * (UPS * 2) + cpy * 4), "l"(src)
                   : "memory");
    }
  }
  asm volatile("cp.async.mbarrier.arrive.noinc.shared::cta.b64 [%0];" ::"r"(smem_u32(bar)) : "memory");
}

// ---- one stage of products -----------------------------------------------
// acc[h][c][e]: tile h (gate / up), accumulator set c, MMA D register e
// (e = 0: row g, e = 2: row g + 8; all columns hold the same sums).

// Address of 16-byte piece (unit u, lane t) of row g (+ 8 rr) of tile h in a
// slot: rows of RB = UPS * 64 bytes, gate rows then up rows.
template <int WR>
__device__ __forceinline__ uint32_t chunk_addr(uint32_t slot, int h, int u, int r, int t) {
  constexpr int RB = (WR == 2 ? kUps32 : kUps16) * kUnitBytes;
  return slot + slot_off(h * 16 + r, u * 4 + t, RB);
}

template <int WR, bool FULL>
__device__ __forceinline__ void stage_int4(uint32_t slot, uint32_t sslot, int nu, int ug, uint32_t xs, int pr,
                                           int t, float (&acc)[2][2][4]) {
  constexpr int UPS = WR == 2 ? kUps32 : kUps16;
  // this lane's scales: rows pr and pr + 8 of each tile h, units
  // 0 .. UPS - 1, as fp16 pairs (units 2j, 2j + 1) per 32-bit word
  uint32_t sw[WR][2][UPS / 2];
#pragma unroll
  for (int h = 0; h < WR; ++h)
#pragma unroll
    for (int rr = 0; rr < 2; ++rr) {
      const uint32_t at = sslot + (uint32_t)((h * 16 + pr + 8 * rr) * (UPS * 2));
      if constexpr (UPS == 4) {
        asm volatile("ld.shared.v2.u32 {%0, %1}, [%2];" : "=r"(sw[h][rr][0]), "=r"(sw[h][rr][1]) : "r"(at));
      } else {
        asm volatile("ld.shared.u32 %0, [%1];" : "=r"(sw[h][rr][0]) : "r"(at));
      }
    }
#pragma unroll
  for (int u = 0; u < UPS; ++u) {
    if (FULL || u < nu) {
      uint4 wv[WR][2];
#pragma unroll
      for (int h = 0; h < WR; ++h)
#pragma unroll
        for (int rr = 0; rr < 2; ++rr) wv[h][rr] = lds16(chunk_addr<WR>(slot, h, u, pr + 8 * rr, t));
      constexpr int NC = WR == 2 ? 2 : 4;  // independent accumulator chains
      float d[WR][NC][4];
#pragma unroll
      for (int h = 0; h < WR; ++h)
#pragma unroll
        for (int q = 0; q < NC; ++q) d[h][q][0] = d[h][q][1] = d[h][q][2] = d[h][q][3] = 0.0f;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const uint4 xq = lds16(xs + (uint32_t)(((ug + u) * 16 + q * 4 + t) * 16));
#pragma unroll
        for (int h = 0; h < WR; ++h) {
          uint32_t p0[4], p1[4];
          const uint4 w0 = wv[h][0], w1 = wv[h][1];
          int4x8_to_f16x2(q == 0 ? w0.x : q == 1 ? w0.y : q == 2 ? w0.z : w0.w, p0);
          int4x8_to_f16x2(q == 0 ? w1.x : q == 1 ? w1.y : q == 2 ? w1.z : w1.w, p1);
          mma16816(d[h][q % NC], p0[0], p1[0], p0[2], p1[2], xq.x, xq.y);
          mma16816(d[h][q % NC], p0[1], p1[1], p0[3], p1[3], xq.z, xq.w);
        }
      }
#pragma unroll
      for (int h = 0; h < WR; ++h) {
        // (row pr, row pr + 8) scales of unit u
        const uint32_t spair = __byte_perm(sw[h][0][u >> 1], sw[h][1][u >> 1], (u & 1) ? 0x7632 : 0x5410);
        const float2 s = __half22float2(*reinterpret_cast<const __half2*>(&spair));
#pragma unroll
        for (int e = 0; e < 4; ++e) {  // (row pr | pr + 8) x (column 2t | 2t + 1)
          float r = d[h][0][e] + d[h][1][e];
          if constexpr (NC == 4) r += d[h][2][e] + d[h][3][e];
          acc[h][0][e] = fmaf(e < 2 ? s.x : s.y, r, acc[h][0][e]);
        }
      }
    }
  }
}

template <int WR, bool FULL>
__device__ __forceinline__ void stage_fp16(uint32_t slot, int nu, int ug, uint32_t xs, int pr, int t,
                                           float (&acc)[2][2][4]) {
  constexpr int UPS = WR == 2 ? kUps32 : kUps16;
#pragma unroll
  for (int u = 0; u < UPS; ++u) {
    if (FULL || u < nu) {
      const uint4 xq = lds16(xs + (uint32_t)(((ug + u) * 4 + t) * 16));
#pragma unroll
      for (int h = 0; h < WR; ++h) {
        const uint4 w0 = lds16(chunk_addr<WR>(slot, h, u, pr, t));
        const uint4 w1 = lds16(chunk_addr<WR>(slot, h, u, pr + 8, t));
        mma16816(acc[h][0], w0.x, w1.x, w0.y, w1.y, xq.x, xq.y);
        mma16816(acc[h][1], w0.z, w1.z, w0.w, w1.w, xq.z, xq.w);
      }
    }
  }
}

template <int WR, bool FULL>
__device__ __forceinline__ void stage_fp8(uint32_t slot, int nu, int ug, uint32_t xs, int pr, int t,
                                          float (&acc)[2][2][4]) {
  constexpr int UPS = WR == 2 ? kUps32 : kUps16;
#pragma unroll
  for (int u = 0; u < UPS; ++u) {
    if (FULL || u < nu) {
      const uint4 xa = lds16(xs + (uint32_t)(((ug + u) * 8 + 2 * t) * 16));
      const uint4 xb = lds16(xs + (uint32_t)(((ug + u) * 8 + 2 * t + 1) * 16));
      const uint32_t xv[8] = {xa.x, xa.y, xa.z, xa.w, xb.x, xb.y, xb.z, xb.w};
#pragma unroll
      for (int h = 0; h < WR; ++h) {
        const uint4 w0 = lds16(chunk_addr<WR>(slot, h, u, pr, t));
        const uint4 w1 = lds16(chunk_addr<WR>(slot, h, u, pr + 8, t));
        const uint32_t r0[4] = {w0.x, w0.y, w0.z, w0.w}, r1[4] = {w1.x, w1.y, w1.z, w1.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          // codes k = 16 t + 4 i .. 4 i + 3 of rows g and g + 8
          const uint32_t a0 = e4m3x2_to_f16x2(lo16(r0[i])), a2 = e4m3x2_to_f16x2(hi16(r0[i]));
          const uint32_t a1 = e4m3x2_to_f16x2(lo16(r1[i])), a3 = e4m3x2_to_f16x2(hi16(r1[i]));
          mma16816(acc[h][i & 1], a0, a1, a2, a3, xv[2 * i], xv[2 * i + 1]);
        }
      }
    }
  }
}

// y[n] from the fp32 dot product v (and the up row's u): FP8 row scale,
// bias, silu(v) * u, residual, fp16 -- the order of the GEMV kernels.
template <int WK, bool SILU>
__device__ __forceinline__ void ring_store(const RingArgs& a, int64_t n, int m, float v, float u) {
  if constexpr (WK == SQ_W_FP8) v *= reinterpret_cast<const float*>(a.scales)[n];
  if (a.bias) v += __half2float(a.bias[n]);
  if constexpr (SILU) {
    if constexpr (WK == SQ_W_FP8) u *= reinterpret_cast<const float*>(a.scales)[a.N + n];
    if (a.bias) u += __half2float(a.bias[a.N + n]);
    v = v / (1.0f + expf(-v)) * u;
  }
  if (a.residual) v += __half2float(a.residual[(int64_t)m * a.N + n]);
  a.y[(int64_t)m * a.N + n] = __float2half_rn(v);
}

template <int WK, bool SILU, int NW>
__global__ void __launch_bounds__(NW * 32, NW > 8 ? 1 : 2) ring_linear_kernel(const RingArgs a) {
  constexpr int UPS = SILU ? kUps32 : kUps16;
  extern __shared__ __align__(128) uint8_t smem[];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int g = lane >> 2, t = lane & 3;
  // [x][partials: tmax * S * 32 fp32][arrival counters: tmax][mbarriers][slots][scale slots]
  const int pb = 32 * a.M;  // floats of one job's partial sums: [tile h][row][column]
  const int red_floats = a.S > 1 ? a.tmax * a.S * pb : 0;
  const int ncnt = a.S > 1 ? a.tmax : 0;
  float* red = reinterpret_cast<float*>(smem + a.x_bytes);
  int* cnt = reinterpret_cast<int*>(red + red_floats);
  const int bar_off = a.x_bytes + red_floats * 4 + (ncnt * 4 + 15) / 16 * 16;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + bar_off);
  const uint32_t base = smem_u32(smem);
  const uint32_t slot0 = (base + bar_off + NW * a.ns * 8 + 127) / 128 * 128;
  uint64_t* mybar = bars + w * a.ns;
  // this lane's activation row: column g of B (columns past M repeat row M - 1)
  const uint32_t xs_addr = base + (uint32_t)((g < a.M ? g : a.M - 1) * a.x_stride);
  const uint32_t slot_addr = slot0 + (uint32_t)(w * a.ns * kStageBytes);
  const uint32_t sslot_addr = slot0 + (uint32_t)(NW * a.ns * kStageBytes + w * a.ns * kScaleBytes);
  const int pr = g;  // rows g and g + 8 of the tile

  const int64_t ta = (int64_t)blockIdx.x * a.T / gridDim.x;
  const int64_t tb = (int64_t)(blockIdx.x + 1) * a.T / gridDim.x;

  if (lane == 0) {
    for (int i = 0; i < a.ns; ++i) mbar_init(&mybar[i], 32);  // one arrival per lane's copies
    fence_mbar_init();
  }
  for (int i = threadIdx.x; i < ncnt; i += NW * 32) cnt[i] = 0;
  __syncwarp();

  // ---- before the producer of x finishes: fill the ring
  Cur ic;
  ic.j = w;
  cur_job(a, ta, tb, ic);
  uint32_t issued = 0;
  for (int i = 0; i < a.ns && ic.live; ++i) {
    issue_stage<WK, SILU>(a, ic, slot_addr + (uint32_t)i * kStageBytes, sslot_addr + (uint32_t)i * kScaleBytes,
                          &mybar[i], lane);
    cur_next<NW, SILU>(a, ta, tb, ic);
    ++issued;
  }
  Cur cc;
  cc.j = w;
  cur_job(a, ta, tb, cc);
  // The next kernel is not signalled early: measured on the 14B INT4 draft
  // pass (8 layers), signalling at entry 660 us, before the epilogue 549 us,
  // at completion 483 us; FP16 / FP8 passes unchanged either way.
  griddep_wait();

  // ---- stage x: INT4 in the conversion's pair order with unit j's chunk
  // (t, q) at slot j * 16 + q * 4 + t; FP8 and FP16 in natural order
  {
    const int nch = a.K / 8;  // 16-byte chunks of one row
    const int total = a.M * nch;
    constexpr int B = 4;
    for (int b0 = threadIdx.x; b0 < total; b0 += NW * 32 * B) {
      uint4 v[B];
#pragma unroll
      for (int b = 0; b < B; ++b) {
        const int i = b0 + b * NW * 32;
        v[b] = i < total ? reinterpret_cast<const uint4*>(a.x)[i] : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int b = 0; b < B; ++b) {
        const int i = b0 + b * NW * 32;
        if (i < total) {
          const int m = i / nch, c = i - m * nch;
          uint4* xs = reinterpret_cast<uint4*>(smem + m * a.x_stride);
          if constexpr (WK == SQ_W_INT4)
            xs[(c >> 4) * 16 + (c & 3) * 4 + ((c >> 2) & 3)] = int4_x_order(v[b]);
          else
            xs[c] = v[b];
        }
      }
    }
  }
  __syncthreads();

  uint32_t status = 0, consumed = 0, broken_at = 0;
  bool broken = false;
  while (cc.live) {
    const Cur job = cc;
    float acc[2][2][4];
#pragma unroll
    for (int h = 0; h < 2; ++h)
#pragma unroll
      for (int c = 0; c < 2; ++c) acc[h][c][0] = acc[h][c][1] = acc[h][c][2] = acc[h][c][3] = 0.0f;
    while (cc.live && cc.j == job.j) {
      const uint32_t k = consumed % (uint32_t)a.ns;
      const uint32_t parity = (consumed / (uint32_t)a.ns) & 1u;
      Cur nx = cc;
      cur_next<NW, SILU>(a, ta, tb, nx);
      const int nu = min(UPS, cc.u1 - cc.u);
      bool ok = false;
      if (!broken) {
        ok = __any_sync(0xffffffffu, mbar_wait_ns(&mybar[k], parity, kWaitNs));
        if (!ok) {
          broken = true;
          broken_at = consumed;
          status |= SQ_DEV_TIMEOUT;
        }
      }
      if (ok) {
        const uint32_t sa = slot_addr + k * kStageBytes, ss = sslot_addr + k * kScaleBytes;
        constexpr int WR = SILU ? 2 : 1;
        if (nu == UPS) {  // full stage: no per-unit predicate
          if constexpr (WK == SQ_W_INT4) stage_int4<WR, true>(sa, ss, UPS, cc.u, xs_addr, pr, t, acc);
          else if constexpr (WK == SQ_W_FP8) stage_fp8<WR, true>(sa, UPS, cc.u, xs_addr, pr, t, acc);
          else stage_fp16<WR, true>(sa, UPS, cc.u, xs_addr, pr, t, acc);
        } else {
          if constexpr (WK == SQ_W_INT4) stage_int4<WR, false>(sa, ss, nu, cc.u, xs_addr, pr, t, acc);
          else if constexpr (WK == SQ_W_FP8) stage_fp8<WR, false>(sa, nu, cc.u, xs_addr, pr, t, acc);
          else stage_fp16<WR, false>(sa, nu, cc.u, xs_addr, pr, t, acc);
        }
      }
      ++consumed;
      __syncwarp();
      if (!broken && ic.live) {
        issue_stage<WK, SILU>(a, ic, slot_addr + k * kStageBytes, sslot_addr + k * kScaleBytes, &mybar[k], lane);
        cur_next<NW, SILU>(a, ta, tb, ic);
        ++issued;
      }
      cc = nx;
    }
    // ---- epilogue of the job: D register e of tile h (gate / up) is row
    // pr + 8 (e >> 1), activation row (column) 2t + (e & 1)
    float v[2][4];
#pragma unroll
    for (int h = 0; h < 2; ++h)
#pragma unroll
      for (int e = 0; e < 4; ++e) v[h][e] = acc[h][0][e] + acc[h][1][e];
    if (a.S == 1) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int m = 2 * t + (e & 1);
        const int64_t n = job.tile * 16 + pr + 8 * (e >> 1);
        if (m < a.M && n < a.N) ring_store<WK, SILU>(a, n, m, v[0][e], v[1][e]);
      }
    } else {
      // the S parts of a tile meet in shared memory; the warp that completes
      // the tile adds them in part order and stores
      const int tl = (int)(job.tile - ta), part = job.j % a.S;
      float* rp = red + (tl * a.S + part) * pb;
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int m = 2 * t + (e & 1);
        const int row = pr + 8 * (e >> 1);
        if (m < a.M) {
          rp[row * a.M + m] = v[0][e];
          rp[(16 + row) * a.M + m] = v[1][e];
        }
      }
      __threadfence_block();
      __syncwarp();
      int last = 0;
      if (lane == 0) last = atomicAdd(&cnt[tl], 1) == a.S - 1;
      last = __shfl_sync(0xffffffffu, last, 0);
      if (last) {
        __threadfence_block();
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int m = 2 * t + (e & 1);
          const int row = pr + 8 * (e >> 1);
          const int64_t n = job.tile * 16 + row;
          if (m < a.M && n < a.N) {
            float sv = 0.0f, su = 0.0f;
            for (int q = 0; q < a.S; ++q) {
              sv += red[(tl * a.S + q) * pb + row * a.M + m];
              su += red[(tl * a.S + q) * pb + (16 + row) * a.M + m];
            }
            ring_store<WK, SILU>(a, n, m, sv, su);
          }
        }
      }
    }
  }
  if (broken) {
    // at most one copy per slot is still outstanding: wait for each (bounded)
    for (uint32_t q = broken_at; q < issued; ++q)
      mbar_wait_ns(&mybar[q % (uint32_t)a.ns], (q / (uint32_t)a.ns) & 1u, kDrainNs);
  }
  if (status) atomicOr(&g_ring_status, status);
}

// Shared memory of one CTA of nw warps with ns slots per warp, x_bytes of
// staged activations and red_floats fp32 partial sums with ncnt counters.
size_t ring_smem(int nw, int x_bytes, int ns, int red_floats = 0, int ncnt = 0) {
  // + 128: the slots are aligned up to 128 bytes at run time
  const int slot0 = x_bytes + red_floats * 4 + (ncnt * 4 + 15) / 16 * 16 + nw * ns * 8 + 128;
  return (size_t)slot0 + (size_t)nw * ns * (kStageBytes + kScaleBytes);
}

// Staged activation rows: K fp16 each, rows 64 bytes past a multiple of 128
// apart when there are several (lanes of columns 2i and 2i + 1 then read
// different bank halves).
int ring_x_stride(int M, int64_t K) {
  const int row = (int)((K * 2 + 127) / 128 * 128);
  return M > 1 ? row + 64 : row;
}
int ring_x_bytes(int M, int64_t K) { return (M * ring_x_stride(M, K) + 127) / 128 * 128; }

// Warps per CTA: 8 for FP16 / FP8; for INT4 16 (one or two rows) or 12
// (three or more) when two slots per warp fit beside the staged activations,
// else the next smaller count that fits.
int ring_warps(int wkind, int M, int64_t K) {
  if (wkind != SQ_W_INT4) return kWarpsHalf;
  const int xb = ring_x_bytes(M, K);
  if (M <= 2 && ring_smem(kWarpsFull, xb, 2, 4096, 128) <= (size_t)kSmemFull) return kWarpsFull;
  if (ring_smem(kWarpsMid, xb, 2, 4096, 128) <= (size_t)kSmemFull) return kWarpsMid;
  return kWarpsHalf;
}

template <int WK, bool SILU, int NW>
cudaError_t launch_inst(const RingArgs& a, size_t smem, int grid, cudaStream_t st) {
  auto k = ring_linear_kernel<WK, SILU, NW>;
  static bool attr_set[64] = {false};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (!attr_set[dev]) {
    e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemFull);
    if (e != cudaSuccess) return e;
    attr_set[dev] = true;
  }
  return launch_pdl(k, dim3(grid), dim3(NW * 32), smem, st, a);
}

template <int WK>
cudaError_t launch_wk(const RingArgs& a, int nw, size_t smem, int grid, cudaStream_t st) {
  const bool silu = a.silu != 0;
  if constexpr (WK == SQ_W_INT4) {
    if (nw == kWarpsFull)
      return silu ? launch_inst<WK, true, kWarpsFull>(a, smem, grid, st)
                  : launch_inst<WK, false, kWarpsFull>(a, smem, grid, st);
    if (nw == kWarpsMid)
      return silu ? launch_inst<WK, true, kWarpsMid>(a, smem, grid, st)
                  : launch_inst<WK, false, kWarpsMid>(a, smem, grid, st);
  }
  return silu ? launch_inst<WK, true, kWarpsHalf>(a, smem, grid, st)
              : launch_inst<WK, false, kWarpsHalf>(a, smem, grid, st);
}

}  // namespace

bool ring_supported(int wkind, int M, int64_t K) {
  if (M < 1 || M > 8 || K % 128 != 0) return false;
  // INT4: an even number of groups per row (the scales travel in 4-byte copies)
  if (wkind == SQ_W_INT4 && (K / 128) % 2 != 0) return false;
  // at least two slots per warp beside the staged activations (and up to 16 KB
  // of partial sums with their counters)
  return ring_smem(ring_warps(wkind, M, K), ring_x_bytes(M, K), 2, 4096, 128) <= (size_t)kSmemFull;
}

cudaError_t launch_ring(int wkind, const __half* x, const void* w, const void* scales, const __half* bias,
                        const __half* residual, __half* y, int M, int64_t N, int64_t K, int epi,
                        cudaStream_t st) {
  RingArgs a = {};
  a.x = x;
  a.w = reinterpret_cast<const uint8_t*>(w);
  a.scales = scales;
  a.bias = bias;
  a.residual = residual;
  a.y = y;
  a.M = M;
  a.N = N;
  a.K = (int32_t)K;
  a.row_bytes = row_bytes_of(wkind, K);
  a.U = (int32_t)(a.row_bytes / kUnitBytes);
  a.T = (N + 15) / 16;
  a.silu = epi == SQ_EPI_SILU_GATE;
  a.ugran = wkind == SQ_W_INT4 ? 2 : 1;
  const int C0 = device_sm_count();
  const int nw = ring_warps(wkind, M, K);
  const int grid = (int)(a.T < C0 ? a.T : C0);
  a.tmax = (int32_t)((a.T + grid - 1) / grid);
  // K split: each CTA owns whole tiles; its warps take (tile, part) jobs in
  // turn.  FP16 / FP8 (memory-bound): S minimises the busiest warp's work,
  // ceil(tmax S / nw) jobs of ceil(U / S) units plus about one unit of
  // overhead per job (epilogue, partial sums).  INT4 (the SM's conversion
  // throughput is the bound, not the busiest warp): the smallest S that gives
  // three quarters of the warps a job (14B fused gate/up: S = 2; the
  // balanced S = 8 measured 2.9 us slower per launch).  Within 16 KB of
  // partial sums.
  const int umax = a.U / a.ugran;
  int best_s = 1;
  int64_t best_cost = -1;
  for (int S = 1; S <= umax && S <= 64; S *= 2) {
    if (S > 1 && (int64_t)a.tmax * S * 32 * M * 4 > 16 * 1024) break;
    if (wkind == SQ_W_INT4) {
      best_s = S;
      if ((int64_t)a.tmax * S * 4 >= 3 * nw) break;
      continue;
    }
    const int64_t jobs = ((int64_t)a.tmax * S + nw - 1) / nw;
    const int64_t cost = jobs * ((a.U + S - 1) / S + 1);
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best_s = S;
    }
  }
  a.S = best_s;
  const int red_floats = a.S > 1 ? a.tmax * a.S * 32 * M : 0;
  const int ncnt = a.S > 1 ? a.tmax : 0;
  a.x_stride = ring_x_stride(M, K);
  a.x_bytes = ring_x_bytes(M, K);
  int ns = 4;
  while (ns > 2 && ring_smem(nw, a.x_bytes, ns, red_floats, ncnt) > (size_t)kSmemFull) --ns;
  a.ns = ns;
  const size_t smem = ring_smem(nw, a.x_bytes, ns, red_floats, ncnt);
  switch (wkind) {
    case SQ_W_INT4: return launch_wk<SQ_W_INT4>(a, nw, smem, grid, st);
    case SQ_W_FP8: return launch_wk<SQ_W_FP8>(a, nw, smem, grid, st);
    default: return launch_wk<SQ_W_FP16>(a, nw, smem, grid, st);
  }
}

// Failure-path self-test of the ring's timed wait: one thread waits on an
// mbarrier that nothing arrives at, gives up after limit_ns nanoseconds and
// sets SQ_DEV_TIMEOUT.  Nothing is in flight, so giving up is clean.
__global__ void wait_selftest_time_kernel(uint64_t limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x != 0) return;
  mbar_init(&bar, 1);
  fence_mbar_init();
  if (!mbar_wait_ns(&bar, 0, limit_ns)) atomicOr(&g_ring_status, SQ_DEV_TIMEOUT);
}

cudaError_t launch_wait_selftest_time(uint64_t limit_ns, cudaStream_t st) {
  wait_selftest_time_kernel<<<1, 32, 0, st>>>(limit_ns);
  return cudaGetLastError();
}

cudaError_t take_ring_status(uint32_t* bits) {
  unsigned int v = 0;
  cudaError_t e = cudaMemcpyFromSymbol(&v, g_ring_status, sizeof(v));
  if (e != cudaSuccess) return e;
  if (v) {
    const unsigned int z = 0;
    e = cudaMemcpyToSymbol(g_ring_status, &z, sizeof(z));
    if (e != cudaSuccess) return e;
  }
  *bits |= v;
  return cudaSuccess;
}

}  // namespace sq
