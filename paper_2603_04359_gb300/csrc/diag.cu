// Per-layer diagnostics (Sec. 2): the row statistics that the concentration C(v) = E||v||^2 / E r(v)^2
// (Lemmas 2 and 3, symmetric range r(v) = 2 max_i |v_i|) and the alignment
// A(x, W) = E||W x||^2 / (||W||_F^2 E||x||^2) are made of, for rows transformed block by block:
//   v'_b = M_b v_b          (activations, M = T: x' = T x)
//   v'_b = M_b^T v_b        (weight rows, M = T^{-1}: w' = w T^{-1})
// Off the timed path; a plain SIMT kernel.  A CTA takes 64 rows of one block: the rows' block
// slice and one 64-output slab of M_b at a time sit in shared memory, every thread accumulates a
// 4-row x (JT / 16)-output register tile in fp32, and each row's partial sum of squares and
// maximum go to per-row accumulators (float atomics; the maximum on the float bits, which order
// like the values for non-negative floats).  A second kernel adds the rows' sums of squares and
// squared ranges through the cross-CTA reduction of sqnr_slot.cuh, which also forms
// 10 log10(sum ||v'||^2 / sum r^2) = C in dB.
#include <cmath>
#include <cstring>
#include <mutex>

#include "common.cuh"
#include "sqnr_slot.cuh"

namespace cat {
namespace {

constexpr int kRows = 64;        // rows per CTA
constexpr int kThreads = 256;    // 16 row groups of 4 x 16 output groups

template <int K>
struct DiagCfg {
  static constexpr int JT = K < 64 ? K : 64;     // outputs per slab
  static constexpr int OJ = JT / 16;             // outputs per thread
  static constexpr size_t SMEM = (size_t)K * kRows * 4 + (size_t)K * JT * 4;
};

__device__ __forceinline__ float load_elem(const void* V, int dtype, size_t idx) {
  if (dtype == 0) return reinterpret_cast<const float*>(V)[idx];
  return __bfloat162float(reinterpret_cast<const __nv_bfloat16*>(V)[idx]);
}

template <int K>
__global__ void __launch_bounds__(kThreads)
    block_row_stats_kernel(const void* __restrict__ V, int dtype, int rows, int d, const float* __restrict__ M,
                           int transpose, float* __restrict__ row_sumsq, uint32_t* __restrict__ row_amax_bits,
                           float* __restrict__ Vt) {
  using C = DiagCfg<K>;
  extern __shared__ float sm[];
  float* vs = sm;                       // [K][kRows]: the rows' block slice, transposed
  float* ms = sm + K * kRows;           // [K][JT]: ms[i][j] is the weight of input i in output j of the slab
  const int tid = threadIdx.x, r0 = blockIdx.x * kRows, b = blockIdx.y;
  const float* Mb = M + (size_t)b * K * K;
  for (int e = tid; e < K * kRows; e += kThreads) {   // i fastest: coalesced along the row
    const int r = e / K, i = e % K;
    vs[i * kRows + r] = (r0 + r < rows) ? load_elem(V, dtype, (size_t)(r0 + r) * d + (size_t)b * K + i) : 0.f;
  }
  const int tr = tid >> 4, tj = tid & 15;
  float sumsq[4] = {0.f, 0.f, 0.f, 0.f}, amax[4] = {0.f, 0.f, 0.f, 0.f};
  for (int j0 = 0; j0 < K; j0 += C::JT) {
    __syncthreads();                                   // the previous slab is no longer read
    for (int e = tid; e < K * C::JT; e += kThreads) {
      if (transpose) {                                 // ms[i][j] = M_b[i][j0 + j]
        const int i = e / C::JT, j = e % C::JT;
        ms[i * C::JT + j] = Mb[(size_t)i * K + j0 + j];
      } else {                                         // ms[i][j] = M_b[j0 + j][i]
        const int j = e / K, i = e % K;
        ms[i * C::JT + j] = Mb[(size_t)(j0 + j) * K + i];
      }
    }
    __syncthreads();
    float acc[4][C::OJ];
#pragma unroll
    for (int rr = 0; rr < 4; ++rr)
#pragma unroll
      for (int oj = 0; oj < C::OJ; ++oj) acc[rr][oj] = 0.f;
#pragma unroll 4
    for (int i = 0; i < K; ++i) {
      const float4 v4 = *reinterpret_cast<const float4*>(&vs[i * kRows + 4 * tr]);
      const float vv[4] = {v4.x, v4.y, v4.z, v4.w};
#pragma unroll
      for (int oj = 0; oj < C::OJ; ++oj) {
        const float m = ms[i * C::JT + tj * C::OJ + oj];
#pragma unroll
        for (int rr = 0; rr < 4; ++rr) acc[rr][oj] = fmaf(vv[rr], m, acc[rr][oj]);
      }
    }
#pragma unroll
    for (int rr = 0; rr < 4; ++rr)
#pragma unroll
      for (int oj = 0; oj < C::OJ; ++oj) {
        sumsq[rr] = fmaf(acc[rr][oj], acc[rr][oj], sumsq[rr]);
        amax[rr] = fmaxf(amax[rr], fabsf(acc[rr][oj]));
      }
    if (Vt) {                                          // the transformed rows themselves
#pragma unroll
      for (int rr = 0; rr < 4; ++rr) {
        const int r = r0 + 4 * tr + rr;
        if (r < rows)
#pragma unroll
          for (int oj = 0; oj < C::OJ; ++oj) Vt[(size_t)r * d + (size_t)b * K + j0 + tj * C::OJ + oj] = acc[rr][oj];
      }
    }
  }
  if (!row_sumsq) return;
  // the 16 output groups of a row group are the 16 lanes that differ in bits 0..3 of the lane index
#pragma unroll
  for (int rr = 0; rr < 4; ++rr) {
#pragma unroll
    for (int off = 8; off > 0; off >>= 1) {
      sumsq[rr] += __shfl_xor_sync(0xFFFFFFFFu, sumsq[rr], off);
      amax[rr] = fmaxf(amax[rr], __shfl_xor_sync(0xFFFFFFFFu, amax[rr], off));
    }
    const int r = r0 + 4 * tr + rr;
    if (tj == 0 && r < rows) {
      atomicAdd(&row_sumsq[r], sumsq[rr]);
      atomicMax(&row_amax_bits[r], __float_as_uint(amax[rr]));
    }
  }
}

// sum_r ||v'_r||^2 and sum_r (2 max_i |v'_ri|)^2 over all rows, and 10 log10 of their ratio.
__global__ void __launch_bounds__(kThreads)
    row_stats_reduce_kernel(const float* __restrict__ row_sumsq, const float* __restrict__ row_amax, int rows,
                            double* __restrict__ out3, int slot) {
  f32x2 s = {0.f, 0.f}, r2 = {0.f, 0.f};
  for (int r = blockIdx.x * kThreads + threadIdx.x; r < rows; r += gridDim.x * kThreads) {
    const float a = 2.f * row_amax[r];
    s = f2_add(s, row_sumsq[r]);
    r2 = f2_add(r2, a * a);
  }
  s = f2_warp_sum(s);
  r2 = f2_warp_sum(r2);
  __shared__ f32x2 ws[kThreads / 32][2];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) {
    ws[warp][0] = s;
    ws[warp][1] = r2;
  }
  __syncthreads();
  if (warp == 0) {
    f32x2 a = {0.f, 0.f}, b = {0.f, 0.f};
    for (int w = 0; w < kThreads / 32; ++w) {
      a = f2_add(a, ws[w][0]);
      b = f2_add(b, ws[w][1]);
    }
    sqnr_cta_done(slot, a, b, out3);
  }
}

template <int K>
cudaError_t launch_k(const void* V, int dtype, int64_t rows, int64_t d, const float* M, int transpose,
                     float* row_sumsq, float* row_amax, float* Vt, cudaStream_t stream) {
  using C = DiagCfg<K>;
  static std::once_flag once;
  static cudaError_t attr = cudaSuccess;
  std::call_once(once, [] {
    attr = cudaFuncSetAttribute(block_row_stats_kernel<K>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM);
  });
  if (attr != cudaSuccess) return attr;
  dim3 grid((unsigned)((rows + kRows - 1) / kRows), (unsigned)(d / K), 1);
  note_launch();
  block_row_stats_kernel<K><<<grid, kThreads, C::SMEM, stream>>>(V, dtype, (int)rows, (int)d, M, transpose, row_sumsq,
                                                                 reinterpret_cast<uint32_t*>(row_amax), Vt);
  return cudaGetLastError();
}

}  // namespace

// row_sumsq and row_amax are zeroed here and accumulated by the block kernel; out3 is written by the
// reduction (no zeroing needed).
cudaError_t launch_block_row_stats(const void* V, int dtype, int64_t rows, int64_t d, int k, const float* M,
                                   int transpose, float* row_sumsq, float* row_amax, double* out3,
                                   cudaStream_t stream) {
  cudaError_t e = cudaMemsetAsync(row_sumsq, 0, (size_t)rows * sizeof(float), stream);
  if (e == cudaSuccess) e = cudaMemsetAsync(row_amax, 0, (size_t)rows * sizeof(float), stream);
  if (e != cudaSuccess) return e;
  switch (k) {
    case 16: e = launch_k<16>(V, dtype, rows, d, M, transpose, row_sumsq, row_amax, nullptr, stream); break;
    case 32: e = launch_k<32>(V, dtype, rows, d, M, transpose, row_sumsq, row_amax, nullptr, stream); break;
    case 64: e = launch_k<64>(V, dtype, rows, d, M, transpose, row_sumsq, row_amax, nullptr, stream); break;
    case 128: e = launch_k<128>(V, dtype, rows, d, M, transpose, row_sumsq, row_amax, nullptr, stream); break;
    case 256: e = launch_k<256>(V, dtype, rows, d, M, transpose, row_sumsq, row_amax, nullptr, stream); break;
    default: return cudaErrorInvalidValue;
  }
  if (e != cudaSuccess) return e;
  int64_t grid = (rows + 4 * kThreads - 1) / (4 * kThreads);
  if (grid < 1) grid = 1;
  if (grid > kSqnrMaxCtas) grid = kSqnrMaxCtas;
  note_launch();
  row_stats_reduce_kernel<<<(unsigned)grid, kThreads, 0, stream>>>(row_sumsq, row_amax, (int)rows, out3,
                                                                   next_sqnr_slot());
  return cudaGetLastError();
}

// v'_b = M_b v_b (or M_b^T v_b) for every row, written to Vt [rows][d] float32.
cudaError_t launch_block_transform(const void* V, int dtype, int64_t rows, int64_t d, int k, const float* M,
                                   int transpose, float* Vt, cudaStream_t stream) {
  switch (k) {
    case 16: return launch_k<16>(V, dtype, rows, d, M, transpose, nullptr, nullptr, Vt, stream);
    case 32: return launch_k<32>(V, dtype, rows, d, M, transpose, nullptr, nullptr, Vt, stream);
    case 64: return launch_k<64>(V, dtype, rows, d, M, transpose, nullptr, nullptr, Vt, stream);
    case 128: return launch_k<128>(V, dtype, rows, d, M, transpose, nullptr, nullptr, Vt, stream);
    case 256: return launch_k<256>(V, dtype, rows, d, M, transpose, nullptr, nullptr, Vt, stream);
    default: return cudaErrorInvalidValue;
  }
}

namespace {

// s_r * q from SM4x8 codes: one thread per packed word (8 codes).
__global__ void dequantize_sm4x8_kernel(const uint32_t* __restrict__ words, const float* __restrict__ scale, int64_t rows,
                                        int64_t d, float* __restrict__ out) {
  const int64_t wpr = d / 8;
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= rows * wpr) return;
  const int64_t r = idx / wpr;
  const uint32_t w = words[idx];
  const uint32_t lo = sm4_lo(w), hi = sm4_hi(w);
  const float s = scale[r];
  float v[8];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint32_t bl = (lo >> (8 * i)) & 0xFFu, bh = (hi >> (8 * i)) & 0xFFu;
    v[i] = (float)((bl & 0x80u) ? -(int)(bl & 7u) : (int)(bl & 7u)) * s;
    v[4 + i] = (float)((bh & 0x80u) ? -(int)(bh & 7u) : (int)(bh & 7u)) * s;
  }
  float4* o = reinterpret_cast<float4*>(out + idx * 8);
  o[0] = make_float4(v[0], v[1], v[2], v[3]);
  o[1] = make_float4(v[4], v[5], v[6], v[7]);
}

// C[m][n] = sum_k A[m][k] B[n][k] in float32: 128 x 128 tiles, 16-deep K slices staged transposed in
// shared memory, 256 threads with 8 x 8 outputs each.
constexpr int GT = 128, GK = 16;
__global__ void __launch_bounds__(256) gemm_f32_nt_kernel(const float* __restrict__ A, const float* __restrict__ B,
                                                          float* __restrict__ Cm, int M, int N, int K) {
  __shared__ __align__(16) float As[GK][GT + 4];
  __shared__ __align__(16) float Bs[GK][GT + 4];
  const int tid = threadIdx.x, tm = tid >> 4, tn = tid & 15;
  const int m0 = blockIdx.y * GT, n0 = blockIdx.x * GT;
  float acc[8][8];
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[i][j] = 0.f;
  for (int k0 = 0; k0 < K; k0 += GK) {
    for (int e = tid; e < GT * GK; e += 256) {            // k fastest: coalesced along the rows
      const int r = e / GK, kk = e % GK;
      const int ka = k0 + kk;
      As[kk][r] = (m0 + r < M && ka < K) ? A[(size_t)(m0 + r) * K + ka] : 0.f;
      Bs[kk][r] = (n0 + r < N && ka < K) ? B[(size_t)(n0 + r) * K + ka] : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < GK; ++kk) {
      float a[8], b[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) a[i] = As[kk][tm + 16 * i];
#pragma unroll
      for (int j = 0; j < 8; ++j) b[j] = Bs[kk][tn + 16 * j];
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int m = m0 + tm + 16 * i;
    if (m >= M) continue;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int n = n0 + tn + 16 * j;
      if (n < N) Cm[(size_t)m * N + n] = acc[i][j];
    }
  }
}

// In place, orthonormal: v <- H_d v / sqrt(d) for every row (Sylvester order), d = 2^m <= 32768.  One
// CTA per row, the row in shared memory, log2(d) butterfly stages.
__global__ void __launch_bounds__(512) fwht_rows_kernel(float* __restrict__ V, int64_t rows, int d, float scale) {
  extern __shared__ float buf[];
  const int64_t r = blockIdx.x;
  float* row = V + r * d;
  for (int i = threadIdx.x; i < d; i += blockDim.x) buf[i] = row[i];
  __syncthreads();
  for (int h = 1; h < d; h <<= 1) {
    for (int p = threadIdx.x; p < d / 2; p += blockDim.x) {
      const int i = (p / h) * 2 * h + (p % h), j = i + h;
      const float a = buf[i], b = buf[j];
      buf[i] = a + b;
      buf[j] = a - b;
    }
    __syncthreads();
  }
  for (int i = threadIdx.x; i < d; i += blockDim.x) row[i] = buf[i] * scale;
}

// C[i][j] = sum_t X[t][i] X[t][j] in float32 (the full Gram matrix of the rows of X [n][d]): the
// 128 x 128 tiles of the GEMM above, operands read down the columns of X (coalesced along i).
template <typename Tin>
__global__ void __launch_bounds__(256) gram_f32_kernel(const Tin* __restrict__ X, float* __restrict__ Cm, int n, int d) {
  __shared__ __align__(16) float As[GK][GT + 4];
  __shared__ __align__(16) float Bs[GK][GT + 4];
  const int tid = threadIdx.x, tm = tid >> 4, tn = tid & 15;
  const int m0 = blockIdx.y * GT, n0 = blockIdx.x * GT;
  float acc[8][8];
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[i][j] = 0.f;
  for (int k0 = 0; k0 < n; k0 += GK) {
    for (int e = tid; e < GT * GK; e += 256) {
      const int kk = e / GT, c = e % GT;
      const int t = k0 + kk;
      As[kk][c] = (t < n && m0 + c < d) ? to_f32(X[(size_t)t * d + m0 + c]) : 0.f;
      Bs[kk][c] = (t < n && n0 + c < d) ? to_f32(X[(size_t)t * d + n0 + c]) : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < GK; ++kk) {
      float a[8], b[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) a[i] = As[kk][tm + 16 * i];
#pragma unroll
      for (int j = 0; j < 8; ++j) b[j] = Bs[kk][tn + 16 * j];
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int m = m0 + tm + 16 * i;
    if (m >= d) continue;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int c = n0 + tn + 16 * j;
      if (c < d) Cm[(size_t)m * d + c] = acc[i][j];
    }
  }
}

}  // namespace

cudaError_t launch_fwht_rows(float* V, int64_t rows, int64_t d, cudaStream_t stream) {
  if (rows == 0) return cudaSuccess;
  const size_t smem = (size_t)d * sizeof(float);
  static std::once_flag once;
  static cudaError_t attr = cudaSuccess;
  std::call_once(once, [] {
    attr = cudaFuncSetAttribute(fwht_rows_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 32768 * 4);
  });
  if (attr != cudaSuccess) return attr;
  const int threads = d / 2 < 512 ? (int)(d / 2 < 32 ? 32 : d / 2) : 512;
  note_launch();
  fwht_rows_kernel<<<(unsigned)rows, threads, smem, stream>>>(V, rows, (int)d, (float)(1.0 / std::sqrt((double)d)));
  return cudaGetLastError();
}

cudaError_t launch_gram_f32(const void* X, int dtype, int64_t n, int64_t d, float* C, cudaStream_t stream) {
  const int64_t g = (d + GT - 1) / GT;
  if (g > 65535) return cudaErrorInvalidValue;
  note_launch();
  if (dtype == 0)
    gram_f32_kernel<float><<<dim3((unsigned)g, (unsigned)g), 256, 0, stream>>>(static_cast<const float*>(X), C, (int)n, (int)d);
  else
    gram_f32_kernel<__nv_bfloat16><<<dim3((unsigned)g, (unsigned)g), 256, 0, stream>>>(
        static_cast<const __nv_bfloat16*>(X), C, (int)n, (int)d);
  return cudaGetLastError();
}

cudaError_t launch_dequantize_sm4x8(const uint8_t* codes, const float* scale, int64_t rows, int64_t d, float* out,
                                    cudaStream_t stream) {
  const int64_t words = rows * (d / 8);
  if (words == 0) return cudaSuccess;
  note_launch();
  dequantize_sm4x8_kernel<<<(unsigned)((words + 255) / 256), 256, 0, stream>>>(reinterpret_cast<const uint32_t*>(codes),
                                                                              scale, rows, d, out);
  return cudaGetLastError();
}

cudaError_t launch_gemm_f32_nt(const float* A, const float* B, float* C, int64_t M, int64_t N, int64_t K,
                               cudaStream_t stream) {
  if (M == 0 || N == 0) return cudaSuccess;
  const int64_t gx = (N + GT - 1) / GT, gy = (M + GT - 1) / GT;
  if (gy > 65535 || gx > 0x7FFFFFFF) return cudaErrorInvalidValue;
  note_launch();
  gemm_f32_nt_kernel<<<dim3((unsigned)gx, (unsigned)gy), 256, 0, stream>>>(A, B, C, (int)M, (int)N, (int)K);
  return cudaGetLastError();
}

}  // namespace cat
