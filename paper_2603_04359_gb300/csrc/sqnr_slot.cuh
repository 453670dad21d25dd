// Cross-CTA reduction of the SQNR sums (Sec. 2, Eq. 1: 10 log10(sum y^2 / sum (y - y_hat)^2))
// without a launch that zeroes the output first.
//
// Each launch is handed one slot of device scratch on the host (round robin over kSqnrSlots).
// Every CTA writes its two partial sums to its own row of the slot and then bumps the slot's
// counter; the CTA that brings the counter to gridDim.x adds the rows in CTA order (the result does
// not depend on which CTA finishes first, so it is the same on every run), writes
// {sum y^2, sum e^2, dB} to the caller's out3 and sets the counter back to zero.  A slot is thus
// clean whenever a launch starts, graph replays included, as long as fewer than kSqnrSlots launches
// of one kernel family run concurrently.  Each translation unit that includes this header has its
// own scratch.
#pragma once
#include <atomic>
#include <math.h>
#include <stdint.h>

namespace cat {

constexpr int kSqnrSlots = 8;
constexpr int kSqnrMaxCtas = 2048;   // rows per slot: the largest grid a reducing kernel may use

// Partial sums are carried as unevaluated pairs of floats (hi + lo, |lo| <= ulp(hi) / 2, about
// 48 significant bits) and added with error-free transformations on the FP32 pipe: a float64 add
// has a latency of 100+ cycles on this GPU, and the reduction is a chain of adds at the end of
// every SQNR-forming kernel.
struct f32x2 {
  float hi, lo;
};

// Pair + pair: Knuth's two-sum of the high parts, the low parts folded in, then renormalized
// (Dekker's fast two-sum).  No products, so nothing is contracted into an FMA.  The result does
// not depend on the order of the operands.
__device__ __forceinline__ f32x2 f2_add(f32x2 a, f32x2 b) {
  const float s = a.hi + b.hi;
  if (!isfinite(s)) return {s, 0.f};   // an infinite or NaN sum stays what it is
  const float bv = s - a.hi;
  float e = (a.hi - (s - bv)) + (b.hi - bv);
  e += a.lo + b.lo;
  const float hi = s + e;
  return {hi, e - (hi - s)};
}
__device__ __forceinline__ f32x2 f2_add(f32x2 a, float b) { return f2_add(a, f32x2{b, 0.f}); }

__device__ __forceinline__ f32x2 f2_shfl_xor(f32x2 v, int off) {
  return {__shfl_xor_sync(0xFFFFFFFFu, v.hi, off), __shfl_xor_sync(0xFFFFFFFFu, v.lo, off)};
}
__device__ __forceinline__ f32x2 f2_shfl_down(f32x2 v, int off) {
  return {__shfl_down_sync(0xFFFFFFFFu, v.hi, off), __shfl_down_sync(0xFFFFFFFFu, v.lo, off)};
}

// Warp sum with a butterfly: every lane ends with the same, order-fixed total.
__device__ __forceinline__ f32x2 f2_warp_sum(f32x2 v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v = f2_add(v, f2_shfl_xor(v, off));
  return v;
}

static __device__ float4 g_sqnr_part[kSqnrSlots][kSqnrMaxCtas];   // {sig.hi, sig.lo, err.hi, err.lo}
static __device__ unsigned int g_sqnr_count[kSqnrSlots];

inline int next_sqnr_slot() {
  static std::atomic<unsigned> next{0};
  return (int)(next.fetch_add(1, std::memory_order_relaxed) % kSqnrSlots);
}

// 10 log10(sig / err) from the high parts, in FP32: the mantissa ratio and the exponent difference
// separately, so no ratio overflows (|error| ~1e-5 dB).
__device__ __forceinline__ double sqnr_db_of(float sig, float err) {
  if (!(err > 0.f)) return sig > 0.f ? HUGE_VAL : 0.0;
  int es, ee;
  const float ms = frexpf(sig, &es), me = frexpf(err, &ee);
  return (double)(10.f * (log10f(ms / me) + (float)(es - ee) * 0.30102999566398120f));
}

// Called by all 32 lanes of one warp per CTA, once, with the CTA's sums in every lane (only lane
// 0's are used).  Requires gridDim.x <= kSqnrMaxCtas (checked by the launchers).
__device__ __forceinline__ void sqnr_cta_done(int slot, f32x2 sig, f32x2 err, double* out3) {
  const int lane = threadIdx.x & 31;
  unsigned last = 0;
  if (lane == 0) {
    g_sqnr_part[slot][blockIdx.x] = make_float4(sig.hi, sig.lo, err.hi, err.lo);
    // one acquire-release increment instead of two GPU-scope fences: its release orders this CTA's row
    // before the count, and the last CTA's acquire (the counter's increments form one release
    // sequence) orders every row before its reads
    unsigned old;
    asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;" : "=r"(old) : "l"(&g_sqnr_count[slot]) : "memory");
    last = old == gridDim.x - 1;
  }
  last = __shfl_sync(0xFFFFFFFFu, last, 0);
  if (!last) return;
  __syncwarp();   // the other lanes' loads come after lane 0's acquire
  // every other CTA's row is visible (each released it with its counter increment); lane l
  // adds rows l, l + 32, ... with eight loads in flight at a time
  f32x2 a = {0.f, 0.f}, b = {0.f, 0.f};
  const unsigned rows = gridDim.x;
  for (unsigned c0 = 0; c0 < rows; c0 += 8 * 32) {
    float4 r[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const unsigned c = c0 + 32u * j + lane;
      r[j] = c < rows ? __ldcg(&g_sqnr_part[slot][c]) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      a = f2_add(a, f32x2{r[j].x, r[j].y});
      b = f2_add(b, f32x2{r[j].z, r[j].w});
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {   // a fixed pattern: lane 0's total is reproducible
    a = f2_add(a, f2_shfl_down(a, off));
    b = f2_add(b, f2_shfl_down(b, off));
  }
  if (lane == 0) {
    out3[0] = (double)a.hi + (double)a.lo;
    out3[1] = (double)b.hi + (double)b.lo;
    out3[2] = sqnr_db_of(a.hi, b.hi);
    g_sqnr_count[slot] = 0u;   // the slot is clean for the next launch handed it
  }
}

}  // namespace cat
