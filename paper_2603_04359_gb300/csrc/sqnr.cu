// SQNR of the layer output (Sec. 2, Eq. 1):  10 log10( sum y^2 / sum (y - y_hat)^2 ).
//
// HBM-bound: 8 bytes read per element.  Each thread issues the loads of 4 float4 pairs at once
// (bytes in flight), sums squares in fp32 over runs of 16 elements (short runs keep the fp32
// rounding at ~1e-7 of a run) and adds the run sums to float-pair accumulators; warps reduce with
// shuffles, and each CTA hands its two partial sums to a slot of device scratch whose last arrival
// adds them in CTA order and forms the ratio (sqnr_slot.cuh), so the whole reduction is one launch
// and its result is the same on every run.
#include "common.cuh"
#include "sqnr_slot.cuh"

namespace cat {
namespace {

constexpr int kThreads = 256;

__global__ void __launch_bounds__(kThreads) sqnr_partial_kernel(const float* __restrict__ yr,
                                                                 const float* __restrict__ yh, int64_t numel,
                                                                 double* __restrict__ out3, int slot) {
  const int64_t n4 = numel / 4;
  const float4* r4 = reinterpret_cast<const float4*>(yr);
  const float4* h4 = reinterpret_cast<const float4*>(yh);
  f32x2 sig = {0.f, 0.f}, err = {0.f, 0.f};
  // CTA tiles of 4 x kThreads consecutive float4 (16 KiB of each input), tiles strided by the grid
  const float4 zero = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int64_t base = (int64_t)blockIdx.x * 4 * kThreads; base < n4; base += (int64_t)gridDim.x * 4 * kThreads) {
    float4 a[4], b[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {  // all 8 loads in flight before the first use
      const int64_t j = base + u * kThreads + threadIdx.x;
      a[u] = j < n4 ? __ldcs(r4 + j) : zero;
      b[u] = j < n4 ? __ldcs(h4 + j) : zero;
    }
    float s_run = 0.f, e_run = 0.f;
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const float ex = a[u].x - b[u].x, ey = a[u].y - b[u].y, ez = a[u].z - b[u].z, ew = a[u].w - b[u].w;
      s_run += a[u].x * a[u].x + a[u].y * a[u].y + a[u].z * a[u].z + a[u].w * a[u].w;
      e_run += ex * ex + ey * ey + ez * ez + ew * ew;
    }
    sig = f2_add(sig, s_run);
    err = f2_add(err, e_run);
  }
  if (blockIdx.x == 0) {  // scalar tail
    for (int64_t j = n4 * 4 + threadIdx.x; j < numel; j += kThreads) {
      const float a = yr[j], e = a - yh[j];
      sig = f2_add(sig, a * a);
      err = f2_add(err, e * e);
    }
  }
  __shared__ f32x2 ssig[kThreads / 32], serr[kThreads / 32];
  sig = f2_warp_sum(sig);
  err = f2_warp_sum(err);
  if ((threadIdx.x & 31) == 0) {
    ssig[threadIdx.x >> 5] = sig;
    serr[threadIdx.x >> 5] = err;
  }
  __syncthreads();
  if (threadIdx.x < 32) {
    f32x2 a = {0.f, 0.f}, b = {0.f, 0.f};
    for (int w = 0; w < kThreads / 32; ++w) {
      a = f2_add(a, ssig[w]);
      b = f2_add(b, serr[w]);
    }
    sqnr_cta_done(slot, a, b, out3);
  }
}

int num_sms() {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 148;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0) return 148;
  return sms;
}

}  // namespace

cudaError_t launch_sqnr(const float* y_ref, const float* y_hat, int64_t numel, double* out3, cudaStream_t stream) {
  // numel == 0: one CTA with nothing to read writes {0, 0, 0}
  const int64_t want = (numel / 4 + kThreads * 4 - 1) / (kThreads * 4);  // one 4-float4 tile per thread at least
  int64_t cap = (int64_t)num_sms() * 8;
  if (cap > kSqnrMaxCtas) cap = kSqnrMaxCtas;
  const unsigned grid = (unsigned)(want < 1 ? 1 : (want > cap ? cap : want));
  note_launch();
  sqnr_partial_kernel<<<grid, kThreads, 0, stream>>>(y_ref, y_hat, numel, out3, next_sqnr_slot());
  return cudaGetLastError();
}

}  // namespace cat
