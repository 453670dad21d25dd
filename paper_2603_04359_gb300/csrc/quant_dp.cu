// Block transform + per-row b-bit quantization written as E4M3 digit planes (bit widths and the
// asymmetric activation quantizer of Sec. 6).
//
//   v'_{t,b} = A_b v_{t,b}                          (Sec. 3, Eq. 5: activations A_b = T_b; weight rows
//                                                     A_b = (T_b^{-1})^T, i.e. w' = w T^{-1})
//   symmetric  (Lemma 2 range 2 max|v|):  q = clamp(round(qmax v / a), -qmax, qmax),  a = c max|v|,
//              qmax = 2^(b-1) - 1, c = 1 or the row's L_2.4 clip ratio (Sec. 6, weights)
//   asymmetric (Lemma 2 range max - min): lo = min(min v, 0), hi = max(max v, 0), N = 2^b - 1,
//              z = round(N (-lo) / (hi - lo)),  q = clamp(round(N v / (hi - lo)) + z, 0, N)
// Rounding is half to even and every decision is exact: symmetric codes by qcode_exact (a
// two-product test at half-integers); asymmetric codes by a float32 estimate, redone in float64 as
// (N v) / (hi - lo) wherever the estimate lies within 2^-12 of a half-integer -- the float64
// quotient of two exact operands, which rounds like the exact quotient there.
//
// Digit planes: a code is written as D = 1 or 2 base-16 digits, q = d0 + 16 d1, each digit stored as
// the E4M3 byte (sign << 7 | |d|), which is exactly d * 2^-9 for |d| <= 16.  Symmetric: D = 1 for
// b <= 4 (d0 = q), else d0 = ((q + 8) mod 16) - 8 in [-8, 7] and d1 = (q - d0) / 16 in [-8, 8].
// Asymmetric: D = 1 for b <= 4 (d0 = q in [0, 15]), else d0 = q mod 16, d1 = q / 16.  Plane p of an
// [R][d] code matrix is the byte matrix at planes + p * R * d.
//
// The row statistics span every block of a row while a CTA holds one block, so the work runs in
// passes over the same tiles (64 rows x OC channels of one block, the block slab and the input rows
// staged transposed in shared memory, each thread 4 rows x 8 channels):
//   pass 0: per-row maximum |v'| (symmetric) or order-preserving keys of max v' and min v'
//           (asymmetric), folded into global buffers with integer atomics;
//   pass R (weights with the L_2.4 range only): per row and candidate range a_i = a (100 - i) / 100,
//           sum |w' - Q(w')|^2.4, added in float64; a select kernel keeps the first candidate with the
//           smallest sum (codes on a shrunk range are decided from exact operands, qcode_shrunk);
//   pass 1: the codes (and, optionally, each row's code sum), written as digit planes;
//   finalize: steps s (and zero points).
#include "common.cuh"

namespace cat {
namespace {

constexpr int kRows = 64;
constexpr int kL24Cands = 80;        // candidate ranges (1 - i/100) max|w|, i = 0 .. 79
constexpr float kL24Norm = 2.4f;

template <int K>
struct DpCfg {
  static constexpr int OC = K < 128 ? K : 128;
  static constexpr int THREADS = 2 * OC;
  static constexpr int AS_LD = OC + 4;
  static constexpr int XS_LD = kRows + 4;
  static constexpr size_t SMEM = (size_t)(K * AS_LD + K * XS_LD) * sizeof(float);
};

struct DpMode {
  int bits;      // 2..8
  int asym;      // 0: symmetric, 1: asymmetric
  int planes;    // digit planes D
  float qmax;    // symmetric: 2^(b-1) - 1; asymmetric: N = 2^b - 1
};

// Order-preserving key of a float (max of keys = key of the max), for signed min / max atomics.
__device__ __forceinline__ uint32_t fkey(float f) {
  const uint32_t b = __float_as_uint(f);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
__device__ __forceinline__ float fkey_inv(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k);
}

__device__ __forceinline__ uint32_t e4m3_digit(int d) { return (d < 0 ? 0x80u : 0u) | (uint32_t)(d < 0 ? -d : d); }

// The digits' E4M3 bytes of one code.
__device__ __forceinline__ void code_digits(int q, const DpMode& m, uint32_t* b0, uint32_t* b1) {
  if (m.planes == 1) {
    *b0 = e4m3_digit(q);
    *b1 = 0u;
  } else if (m.asym) {
    *b0 = (uint32_t)(q & 15);
    *b1 = (uint32_t)(q >> 4);
  } else {
    const int lo = ((q + 8) & 15) - 8;
    *b0 = e4m3_digit(lo);
    *b1 = e4m3_digit((q - lo) / 16);
  }
}

// Per-row asymmetric grid: float32 estimate inputs and the float64 operands of the exact route.
struct AsymRow {
  float inv;      // fl(N / fl(hi - lo)); 0 for a zero or non-finite row
  double lo, r;   // lo and hi - lo in float64
  int z;
};

__device__ __forceinline__ AsymRow asym_row(float hi, float lo, float N) {
  AsymRow a;
  a.lo = lo;
  a.r = (double)hi - (double)lo;
  a.inv = 0.f;
  a.z = 0;
  if (!(isfinite(hi) && isfinite(lo)) || !(a.r > 0.0)) return a;
  a.inv = __fdiv_rn(N, __fsub_rn(hi, lo));
  a.z = (int)rint(((double)N * -a.lo) / a.r);
  return a;
}

__device__ __forceinline__ int asym_code(float v, const AsymRow& a, float N) {
  if (a.inv == 0.f || !isfinite(v)) return a.inv == 0.f ? 0 : a.z;
  const float p = __fmul_rn(v, a.inv);
  float rq = rintf(p);
  if (fabsf(p - rq) > 0.5f - 0x1p-12f) rq = (float)rint(((double)N * (double)v) / a.r);  // exact route
  int q = (int)rq + a.z;
  const int top = (int)N;
  return q < 0 ? 0 : (q > top ? top : q);
}

// Symmetric code on a shrunk range a_i = a (100 - i) / 100 (the L_2.4 choice): the float32 estimate
// v * fl(qmax / fl(a_i)), redone as (100 qmax v) / (a (100 - i)) in float64 -- two exact operands,
// so ties stay exact -- wherever it lies within 2^-12 of a half-integer or is not finite.
__device__ __forceinline__ int qcode_shrunk(float v, float a, int keep, float inv, float qmax) {
  if (!(a > 0.f) || !isfinite(a) || !isfinite(v)) return 0;
  const float p = __fmul_rn(v, inv);
  float rq = rintf(p);
  if (!(fabsf(p - rq) <= 0.5f - 0x1p-12f))
    rq = (float)rint((100.0 * (double)qmax * (double)v) / ((double)a * (double)keep));
  const int q = (int)rq, top = (int)qmax;
  return q > top ? top : (q < -top ? -top : q);
}

template <typename Tin, int K>
__device__ __forceinline__ void stage_tile(const Tin* __restrict__ x, int64_t n, int64_t d, const float* __restrict__ A,
                                           int b, int c0, int64_t t0, float* As, float* xs) {
  using C = DpCfg<K>;
  const int tid = threadIdx.x;
  const float* Ab = A + (size_t)b * K * K;
  for (int e = tid; e < C::OC * K; e += C::THREADS) {
    const int i = e / K, j = e % K;
    As[j * C::AS_LD + i] = Ab[(size_t)(c0 + i) * K + j];
  }
  for (int e = tid; e < kRows * K; e += C::THREADS) {
    const int r = e / K, j = e % K;
    const int64_t t = t0 + r;
    xs[j * C::XS_LD + r] = (t < n) ? to_f32(x[t * d + (int64_t)b * K + j]) : 0.f;
  }
}

template <int K>
__device__ __forceinline__ void tile_product(const float* As, const float* xs, float (&acc)[4][8]) {
  using C = DpCfg<K>;
  const int tg = threadIdx.x & 15, cg = threadIdx.x >> 4;
#pragma unroll
  for (int r = 0; r < 4; ++r)
#pragma unroll
    for (int c = 0; c < 8; ++c) acc[r][c] = 0.f;
#pragma unroll 4
  for (int j = 0; j < K; ++j) {
    const float4 xv = *reinterpret_cast<const float4*>(&xs[j * C::XS_LD + 4 * tg]);
    const float4 a0 = *reinterpret_cast<const float4*>(&As[j * C::AS_LD + 8 * cg]);
    const float4 a1 = *reinterpret_cast<const float4*>(&As[j * C::AS_LD + 8 * cg + 4]);
    const float xr[4] = {xv.x, xv.y, xv.z, xv.w};
    const float ac[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
#pragma unroll
    for (int r = 0; r < 4; ++r)
#pragma unroll
      for (int c = 0; c < 8; ++c) acc[r][c] = fmaf(ac[c], xr[r], acc[r][c]);
  }
}

// PASS 0: row statistics.  PASS 1: codes.  PASS 2: L_2.4 scores of the candidate ranges.
//   key_hi: symmetric -> max|v'| float bits; asymmetric -> key of max v'.   key_lo: asymmetric key of min v'.
template <typename Tin, int K, int PASS>
__global__ void __launch_bounds__(DpCfg<K>::THREADS) transform_quant_dp_kernel(
    const Tin* __restrict__ x, int64_t n, int64_t d, const float* __restrict__ A, DpMode m,
    uint32_t* __restrict__ key_hi, uint32_t* __restrict__ key_lo, const float* __restrict__ row_a,
    const int32_t* __restrict__ shrink, double* __restrict__ l24, uint8_t* __restrict__ planes,
    int32_t* __restrict__ rowsum, uint32_t* __restrict__ status) {
  using C = DpCfg<K>;
  extern __shared__ __align__(16) float smem[];
  float* As = smem;
  float* xs = smem + K * C::AS_LD;
  __shared__ uint32_t red_hi[kRows], red_lo[kRows];
  __shared__ float red_l24[PASS == 2 ? kRows * kL24Cands : 1];

  const int slabs = K / C::OC;
  const int b = blockIdx.y / slabs;
  const int c0 = (blockIdx.y % slabs) * C::OC;
  const int64_t t0 = (int64_t)blockIdx.x * kRows;
  const int tid = threadIdx.x, tg = tid & 15, cg = tid >> 4;

  stage_tile<Tin, K>(x, n, d, A, b, c0, t0, As, xs);
  if (PASS == 0)
    for (int r = tid; r < kRows; r += C::THREADS) {
      red_hi[r] = 0u;
      red_lo[r] = 0xFFFFFFFFu;
    }
  if (PASS == 2)
    for (int e = tid; e < kRows * kL24Cands; e += C::THREADS) red_l24[e] = 0.f;
  __syncthreads();

  float acc[4][8];
  tile_product<K>(As, xs, acc);

  if (PASS == 0) {
    bool finite = true;
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      if (m.asym) {
        uint32_t hi = 0u, lo = 0xFFFFFFFFu;
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          finite &= isfinite(acc[r][c]);
          const uint32_t kv = fkey(acc[r][c]);
          hi = kv > hi ? kv : hi;
          lo = kv < lo ? kv : lo;
        }
        atomicMax(&red_hi[4 * tg + r], hi);
        atomicMin(&red_lo[4 * tg + r], lo);
      } else {
        float mx = 0.f;
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          finite &= isfinite(acc[r][c]);
          mx = fmaxf(mx, fabsf(acc[r][c]));
        }
        atomicMax(&red_hi[4 * tg + r], __float_as_uint(mx));
      }
    }
    if (!finite) report(status, kStatusNonFinite);
    __syncthreads();
    for (int r = tid; r < kRows; r += C::THREADS)
      if (t0 + r < n) {
        atomicMax(&key_hi[t0 + r], red_hi[r]);
        if (m.asym) atomicMin(&key_lo[t0 + r], red_lo[r]);
      }
  } else if (PASS == 2) {
    // L_2.4 score of every candidate range (symmetric weights): sum over the tile of |w' - s q|^2.4
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int64_t t = t0 + 4 * tg + r;
      const float a = t < n ? __uint_as_float(key_hi[t]) : 0.f;
      if (!(isfinite(a) && a > 0.f)) continue;
      for (int i = 0; i < kL24Cands; ++i) {
        const float ai = (float)((double)a * (double)(100 - i) / 100.0);
        const float s = (float)((double)a * (double)(100 - i) / 100.0 / (double)m.qmax);
        const float inv = __fdiv_rn(m.qmax, ai);
        float part = 0.f;
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          const float v = acc[r][c];
          const int q = qcode_shrunk(v, a, 100 - i, inv, m.qmax);
          const float e = fabsf(v - s * (float)q);
          part += e == 0.f ? 0.f : e * e * exp2f((kL24Norm - 2.f) * log2f(e));   // |e|^2.4
        }
        atomicAdd(&red_l24[(4 * tg + r) * kL24Cands + i], part);
      }
    }
    __syncthreads();
    for (int e = tid; e < kRows * kL24Cands; e += C::THREADS) {
      const int64_t t = t0 + e / kL24Cands;
      if (t < n) atomicAdd(&l24[t * kL24Cands + e % kL24Cands], (double)red_l24[e]);
    }
  } else {
    const int64_t col = (int64_t)b * K + c0 + 8 * cg;
    const int64_t plane_stride = n * d;
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int64_t t = t0 + 4 * tg + r;
      if (t >= n) continue;
      int q[8];
      if (m.asym) {
        const AsymRow ar = asym_row(fkey_inv(key_hi[t]), fkey_inv(key_lo[t]), m.qmax);
        // the range holds zero: keys start at the extremes and the row's max / min are clamped
#pragma unroll
        for (int c = 0; c < 8; ++c) q[c] = asym_code(acc[r][c], ar, m.qmax);
      } else if (shrink) {                           // the L_2.4 range
        const float a = __uint_as_float(key_hi[t]), ai = row_a[t];
        const int keep = 100 - shrink[t];
        const float inv = (ai > 0.f && isfinite(ai)) ? __fdiv_rn(m.qmax, ai) : 0.f;
#pragma unroll
        for (int c = 0; c < 8; ++c) q[c] = qcode_shrunk(acc[r][c], a, keep, inv, m.qmax);
      } else {
        const QRow qr = qrow_setup(__uint_as_float(key_hi[t]), m.qmax);
#pragma unroll
        for (int c = 0; c < 8; ++c) q[c] = qcode_exact(acc[r][c], qr, m.qmax);
      }
      uint32_t lo0 = 0u, lo1 = 0u, hi0 = 0u, hi1 = 0u;   // 8 bytes per plane
      int sum = 0;
#pragma unroll
      for (int c = 0; c < 8; ++c) {
        uint32_t d0, d1;
        code_digits(q[c], m, &d0, &d1);
        sum += q[c];
        if (c < 4) {
          lo0 |= d0 << (8 * c);
          hi0 |= d1 << (8 * c);
        } else {
          lo1 |= d0 << (8 * (c - 4));
          hi1 |= d1 << (8 * (c - 4));
        }
      }
      *reinterpret_cast<uint2*>(planes + t * d + col) = make_uint2(lo0, lo1);
      if (m.planes == 2) *reinterpret_cast<uint2*>(planes + plane_stride + t * d + col) = make_uint2(hi0, hi1);
      if (rowsum) atomicAdd(&rowsum[t], sum);
    }
  }
}

// Symmetric rows: keys hold max|v'| bits; asymmetric: keys of max and min, the range clamped to hold 0.
__global__ void dp_init_kernel(uint32_t* __restrict__ key_hi, uint32_t* __restrict__ key_lo, int32_t* __restrict__ rowsum,
                               int64_t n, int asym) {
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= n) return;
  key_hi[t] = asym ? fkey(0.f) : 0u;
  if (asym) key_lo[t] = fkey(0.f);
  if (rowsum) rowsum[t] = 0;
}

// L_2.4 selection: the first candidate with the smallest score; row_a = that candidate's range.
__global__ void dp_select_kernel(const uint32_t* __restrict__ key_hi, double* __restrict__ l24, float* __restrict__ row_a,
                                 int32_t* __restrict__ shrink, int64_t n) {
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= n) return;
  const float a = __uint_as_float(key_hi[t]);
  int best = 0;
  double bs = l24[t * kL24Cands];
  for (int i = 1; i < kL24Cands; ++i) {
    const double v = l24[t * kL24Cands + i];
    if (v < bs) {
      bs = v;
      best = i;
    }
  }
  for (int i = 0; i < kL24Cands; ++i) l24[t * kL24Cands + i] = 0.0;   // clean for the next use
  shrink[t] = best;
  row_a[t] = (float)((double)a * (double)(100 - best) / 100.0);
}

// Steps (and zero points): symmetric s = a / qmax (a = the row's range, clipped or not); asymmetric
// s = (hi - lo) / N and z.  Non-finite rows get s = 0 (their codes are 0 / z) and raise the status.
__global__ void dp_finalize_kernel(const uint32_t* __restrict__ key_hi, const uint32_t* __restrict__ key_lo,
                                   const int32_t* __restrict__ shrink, DpMode m, float* __restrict__ scale,
                                   int32_t* __restrict__ zero, int64_t n, uint32_t* __restrict__ status) {
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= n) return;
  if (m.asym) {
    const float hi = fkey_inv(key_hi[t]), lo = fkey_inv(key_lo[t]);
    const AsymRow ar = asym_row(hi, lo, m.qmax);
    if (!(isfinite(hi) && isfinite(lo))) report(status, kStatusNonFinite);
    scale[t] = ar.inv == 0.f ? 0.f : (float)(ar.r / (double)m.qmax);
    zero[t] = ar.z;
  } else {
    const float a = __uint_as_float(key_hi[t]);
    float s = 0.f;
    if (!isfinite(a))
      report(status, kStatusNonFinite);
    else if (shrink)   // (a (100 - i) / 100) / qmax, rounded once
      s = (float)((double)a * (double)(100 - shrink[t]) / 100.0 / (double)m.qmax);
    else
      s = __fdiv_rn(a, m.qmax);
    scale[t] = s;
  }
}

template <typename Tin, int K>
cudaError_t launch_dp_k(const Tin* x, int64_t n, int64_t d, const float* A, DpMode m, int l24, uint8_t* planes,
                        float* scale, int32_t* zero, int32_t* rowsum, void* work, uint32_t* status, cudaStream_t stream) {
  using C = DpCfg<K>;
  // The row keys live in the caller's outputs until the finalize kernel turns them into steps and
  // zero points in place: key_hi in scale, key_lo (asymmetric) in zero.  work (L_2.4 only): row_a
  // [n] f32, then the scores [n][80] f64 (zero on entry; the select kernel leaves them zero).
  uint32_t* key_hi = reinterpret_cast<uint32_t*>(scale);
  uint32_t* key_lo = reinterpret_cast<uint32_t*>(zero);
  float* row_a = reinterpret_cast<float*>(work);
  int32_t* shrink = reinterpret_cast<int32_t*>(row_a + n);
  double* scores = l24 ? reinterpret_cast<double*>(reinterpret_cast<uintptr_t>(shrink + n + 2) & ~uintptr_t(7)) : nullptr;
  auto k0 = transform_quant_dp_kernel<Tin, K, 0>;
  auto k1 = transform_quant_dp_kernel<Tin, K, 1>;
  auto k2 = transform_quant_dp_kernel<Tin, K, 2>;
  cudaError_t e;
  if ((e = cudaFuncSetAttribute(k0, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM)) != cudaSuccess) return e;
  if ((e = cudaFuncSetAttribute(k1, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM)) != cudaSuccess) return e;
  if ((e = cudaFuncSetAttribute(k2, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM)) != cudaSuccess) return e;
  const int64_t row_tiles = (n + kRows - 1) / kRows;
  if (row_tiles > 0x7FFFFFFF) return cudaErrorInvalidValue;
  const int64_t ny = (d / K) * (K / C::OC);
  if (ny > 65535) return cudaErrorInvalidValue;
  dim3 grid((unsigned)row_tiles, (unsigned)ny);
  const unsigned rb = (unsigned)((n + 255) / 256);
  note_launch();
  dp_init_kernel<<<rb, 256, 0, stream>>>(key_hi, key_lo, rowsum, n, m.asym);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  note_launch();
  k0<<<grid, C::THREADS, C::SMEM, stream>>>(x, n, d, A, m, key_hi, key_lo, nullptr, nullptr, nullptr, planes, rowsum,
                                            status);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  const float* ra = nullptr;
  const int32_t* sh = nullptr;
  if (l24) {
    note_launch();
    k2<<<grid, C::THREADS, C::SMEM, stream>>>(x, n, d, A, m, key_hi, key_lo, nullptr, nullptr, scores, planes, rowsum,
                                              status);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    note_launch();
    dp_select_kernel<<<rb, 256, 0, stream>>>(key_hi, scores, row_a, shrink, n);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    ra = row_a;
    sh = shrink;
  }
  note_launch();
  k1<<<grid, C::THREADS, C::SMEM, stream>>>(x, n, d, A, m, key_hi, key_lo, ra, sh, nullptr, planes, rowsum, status);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  note_launch();
  dp_finalize_kernel<<<rb, 256, 0, stream>>>(key_hi, key_lo, sh, m, scale, zero, n, status);
  return cudaGetLastError();
}

template <typename Tin>
cudaError_t launch_dp_t(const Tin* x, int64_t n, int64_t d, int k, const float* A, DpMode m, int l24, uint8_t* planes,
                        float* scale, int32_t* zero, int32_t* rowsum, void* work, uint32_t* status, cudaStream_t s) {
  switch (k) {
    case 16: return launch_dp_k<Tin, 16>(x, n, d, A, m, l24, planes, scale, zero, rowsum, work, status, s);
    case 32: return launch_dp_k<Tin, 32>(x, n, d, A, m, l24, planes, scale, zero, rowsum, work, status, s);
    case 64: return launch_dp_k<Tin, 64>(x, n, d, A, m, l24, planes, scale, zero, rowsum, work, status, s);
    case 128: return launch_dp_k<Tin, 128>(x, n, d, A, m, l24, planes, scale, zero, rowsum, work, status, s);
    case 256: return launch_dp_k<Tin, 256>(x, n, d, A, m, l24, planes, scale, zero, rowsum, work, status, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

int dp_planes(int bits, int asym) {
  (void)asym;   // symmetric codes up to 7 and asymmetric codes up to 15 are one digit
  return bits <= 4 ? 1 : 2;
}

// Workspace of the L_2.4 range search (weights): row ranges and the candidates' scores.
size_t dp_l24_work_bytes(int64_t n) { return (size_t)n * 8 + 16 + (size_t)n * kL24Cands * sizeof(double); }

// scale [n] and, for asymmetric rows, zero [n] hold the row keys until the last launch writes the
// steps and zero points there.  With l24 the workspace (dp_l24_work_bytes) must be zero on entry.
cudaError_t launch_transform_quantize_dp(const void* x, int dtype, int64_t n, int64_t d, int k, const float* A, int bits,
                                         int asym, int l24, uint8_t* planes, float* scale, int32_t* zero,
                                         int32_t* rowsum, void* work, uint32_t* status, cudaStream_t stream) {
  if (n == 0) return cudaSuccess;
  DpMode m;
  m.bits = bits;
  m.asym = asym;
  m.planes = dp_planes(bits, asym);
  m.qmax = asym ? (float)((1 << bits) - 1) : (float)((1 << (bits - 1)) - 1);
  if (dtype == 0) return launch_dp_t(static_cast<const float*>(x), n, d, k, A, m, l24, planes, scale, zero, rowsum, work,
                                     status, stream);
  return launch_dp_t(static_cast<const __nv_bfloat16*>(x), n, d, k, A, m, l24, planes, scale, zero, rowsum, work, status,
                     stream);
}

}  // namespace cat
