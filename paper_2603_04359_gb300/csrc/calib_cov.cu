// Calibration autocorrelation blocks (Sec. 4: Sigma_x = E[x x^T]; Eq. 10 needs only its k x k
// diagonal blocks):  sigma[b] (+)= sum_t x_{t,b} x_{t,b}^T.  This file holds the path for fp32 rows
// (and the entry point); bf16 rows take the tensor-core kernel in calib_cov_tc.cu.
//
// One CTA computes a TS x TS tile of one k x k block over a range of tokens, staging 32 tokens
// at a time in shared memory.  Each product of two bf16 values is exact in fp32 (fp32 inputs add
// the FMA-recovered product error); the running sum is a compensated pair (hi, lo): every
// addition is an error-free TwoSum whose rounding error goes into lo.  The pair is widened to
// float64 at the end, so the result agrees with a float64 accumulation to ~n * 2^-48.
#include "common.cuh"

namespace cat {
namespace {

constexpr int kTokChunk = 32;

// Error-free TwoSum; the _rn intrinsics keep the compiler from contracting or reassociating.
__device__ __forceinline__ void two_sum_acc(float& hi, float& lo, float p) {
  const float s = __fadd_rn(hi, p);
  const float bp = __fsub_rn(s, hi);
  const float e = __fadd_rn(__fsub_rn(hi, __fsub_rn(s, bp)), __fsub_rn(p, bp));
  hi = s;
  lo = __fadd_rn(lo, e);
}

template <typename Tin, int TS>
__global__ void __launch_bounds__(256) calib_cov_kernel(const Tin* __restrict__ x, int64_t n, int64_t d, int k,
                                                        int tiles_per_dim, int64_t tok_per_split,
                                                        double* __restrict__ sigma, int use_atomic) {
  constexpr int R = TS / 16;  // outputs per thread along each dimension
  __shared__ __align__(16) float xa[kTokChunk][TS];
  __shared__ __align__(16) float xb[kTokChunk][TS];
  const int b = blockIdx.x;
  const int ti0 = (blockIdx.y / tiles_per_dim) * TS;
  const int tj0 = (blockIdx.y % tiles_per_dim) * TS;
  const int64_t t_begin = (int64_t)blockIdx.z * tok_per_split;
  const int64_t t_end = min(n, t_begin + tok_per_split);
  const int tid = threadIdx.x, ty = tid >> 4, tx = tid & 15;
  const int64_t ca = (int64_t)b * k + ti0;
  const int64_t cb = (int64_t)b * k + tj0;

  float hi[R][R], lo[R][R];
#pragma unroll
  for (int i = 0; i < R; ++i)
#pragma unroll
    for (int j = 0; j < R; ++j) hi[i][j] = lo[i][j] = 0.f;

  for (int64_t t0 = t_begin; t0 < t_end; t0 += kTokChunk) {
    for (int e = tid; e < kTokChunk * TS; e += 256) {
      const int tt = e / TS, c = e % TS;
      const int64_t t = t0 + tt;
      float va = 0.f, vb = 0.f;
      if (t < t_end) {
        va = to_f32(x[t * d + ca + c]);
        vb = to_f32(x[t * d + cb + c]);
      }
      xa[tt][c] = va;
      xb[tt][c] = vb;
    }
    __syncthreads();
#pragma unroll 4
    for (int tt = 0; tt < kTokChunk; ++tt) {
      float a[R], bv[R];
#pragma unroll
      for (int r = 0; r < R; ++r) {
        a[r] = xa[tt][ty * R + r];
        bv[r] = xb[tt][tx * R + r];
      }
#pragma unroll
      for (int i = 0; i < R; ++i)
#pragma unroll
        for (int j = 0; j < R; ++j) {
          const float p = __fmul_rn(a[i], bv[j]);
          two_sum_acc(hi[i][j], lo[i][j], p);
          if (sizeof(Tin) == 4) lo[i][j] = __fadd_rn(lo[i][j], fmaf(a[i], bv[j], -p));  // fp32: product error
        }
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < R; ++i)
#pragma unroll
    for (int j = 0; j < R; ++j) {
      const double v = (double)hi[i][j] + (double)lo[i][j];
      const int64_t idx = ((int64_t)b * k + ti0 + ty * R + i) * k + tj0 + tx * R + j;
      if (use_atomic)
        atomicAdd(&sigma[idx], v);
      else
        sigma[idx] = v;
    }
}

template <typename Tin>
cudaError_t launch_typed(const Tin* x, int64_t n, int64_t d, int k, double* sigma, int accumulate,
                         cudaStream_t stream) {
  const int nb = (int)(d / k);
  const size_t bytes = (size_t)nb * k * k * sizeof(double);
  if (n == 0) return accumulate ? cudaSuccess : cudaMemsetAsync(sigma, 0, bytes, stream);
  const int TS = k >= 64 ? 64 : k;
  const int tiles_per_dim = k / TS;
  const int64_t units = (int64_t)nb * tiles_per_dim * tiles_per_dim;
  const int64_t chunks = (n + kTokChunk - 1) / kTokChunk;
  int64_t splits = (600 + units - 1) / units;  // aim for ~4 CTAs per SM
  if (splits > chunks) splits = chunks;
  if (splits < 1) splits = 1;
  if (splits > 65535) splits = 65535;
  const int64_t tok_per_split = ((chunks + splits - 1) / splits) * kTokChunk;
  splits = (n + tok_per_split - 1) / tok_per_split;
  const int use_atomic = (accumulate || splits > 1) ? 1 : 0;
  if (!accumulate && use_atomic) {
    cudaError_t e = cudaMemsetAsync(sigma, 0, bytes, stream);
    if (e != cudaSuccess) return e;
  }
  dim3 grid(nb, tiles_per_dim * tiles_per_dim, (unsigned)splits);
  switch (TS) {
    case 64:
      note_launch();
      calib_cov_kernel<Tin, 64><<<grid, 256, 0, stream>>>(x, n, d, k, tiles_per_dim, tok_per_split, sigma, use_atomic);
      break;
    case 32:
      note_launch();
      calib_cov_kernel<Tin, 32><<<grid, 256, 0, stream>>>(x, n, d, k, tiles_per_dim, tok_per_split, sigma, use_atomic);
      break;
    case 16:
      note_launch();
      calib_cov_kernel<Tin, 16><<<grid, 256, 0, stream>>>(x, n, d, k, tiles_per_dim, tok_per_split, sigma, use_atomic);
      break;
    default:
      return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace

bool calib_cov_tc_supported(int dtype, int k, int64_t n, int64_t d);
cudaError_t launch_calib_cov_tc(const void* x, int64_t n, int64_t d, int k, double* sigma, int accumulate,
                                uint32_t* status, cudaStream_t stream);

// bf16 rows: tensor-core SYRK (calib_cov_tc.cu); fp32 rows: the compensated SIMT kernel above.
cudaError_t launch_calib_cov(const void* x, int dtype, int64_t n, int64_t d, int k, double* sigma, int accumulate,
                             uint32_t* status, cudaStream_t stream) {
  if (dtype == 0) return launch_typed(static_cast<const float*>(x), n, d, k, sigma, accumulate, stream);
  if (calib_cov_tc_supported(dtype, k, n, d)) return launch_calib_cov_tc(x, n, d, k, sigma, accumulate, status, stream);
  return launch_typed(static_cast<const __nv_bfloat16*>(x), n, d, k, sigma, accumulate, stream);
}

}  // namespace cat
