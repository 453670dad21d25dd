// Block transform + per-row absmax + symmetric INT4 quantization + SM4x8 packing.
//
//   v'_{t,b} = A_b v_{t,b}             for every row t and k x k block b
//   s_t      = max_i |v'_{t,i}| / 7    (Lemma 2 symmetric range r = 2 max|v|; grid step r / 14)
//   q_{t,i}  = clamp(rint(v'_{t,i} * 7 / max|v'_t|), -7, 7)       (round half to even)
//
// Activations (Sec. 3, Eq. 5: x' = T x, quantized per token, Sec. 6) use A_b = T_b; weight rows
// (W' = W T^{-1}, quantized per output channel) use A_b = (T_b^{-1})^T.
//
// The row maximum spans every block of the row while a CTA holds one block, so the work runs in
// two passes over the same tiles: pass 0 folds per-row maxima into the scale buffer with integer
// atomicMax on the (non-negative) float bits; pass 1 recomputes the tile, quantizes and packs;
// a last pass turns the maxima into steps.  No scratch memory is used.
//
// Tile: 64 rows x OC output channels of one block (OC = min(k, 128)), the block slab A_b[c0:c0+OC, :]
// and the 64 input rows are staged transposed in shared memory; each thread owns 4 rows x 8
// consecutive channels (32 fp32 accumulators), which is exactly one packed word per row.
#include "common.cuh"

namespace cat {
namespace {

constexpr int kRows = 64;

template <int K>
struct ActCfg {
  static constexpr int OC = K < 128 ? K : 128;         // output channels per CTA
  static constexpr int THREADS = 2 * OC;               // 16 row groups x OC/8 channel groups
  static constexpr int AS_LD = OC + 4;                 // padded row of the transposed slab
  static constexpr int XS_LD = kRows + 4;              // padded row of the transposed inputs
  static constexpr size_t SMEM = (size_t)(K * AS_LD + K * XS_LD) * sizeof(float);
};

template <typename Tin, int K, int PASS>
__global__ void __launch_bounds__(ActCfg<K>::THREADS) transform_quant_kernel(
    const Tin* __restrict__ x, int64_t n, int64_t d, const float* __restrict__ A, uint32_t* __restrict__ amax_bits,
    uint32_t* __restrict__ codes, uint32_t* __restrict__ status) {
  using C = ActCfg<K>;
  extern __shared__ __align__(16) float smem[];
  float* As = smem;                    // [K][AS_LD]: As[j][i] = A_b[c0 + i][j]
  float* xs = smem + K * C::AS_LD;     // [K][XS_LD]: xs[j][r] = x[t0 + r][b*K + j]
  __shared__ uint32_t red[kRows];

  const int slabs = K / C::OC;
  const int b = blockIdx.y / slabs;
  const int c0 = (blockIdx.y % slabs) * C::OC;
  const int64_t t0 = (int64_t)blockIdx.x * kRows;
  const int tid = threadIdx.x;
  const int tg = tid & 15;   // rows 4*tg .. 4*tg+3
  const int cg = tid >> 4;   // channels c0 + 8*cg .. +7

  // Stage the slab transposed.
  const float* Ab = A + (size_t)b * K * K;
  for (int e = tid; e < C::OC * K; e += C::THREADS) {
    const int i = e / K, j = e % K;
    As[j * C::AS_LD + i] = Ab[(size_t)(c0 + i) * K + j];
  }
  // Stage the input rows transposed (rows past n read as zero).
  for (int e = tid; e < kRows * K; e += C::THREADS) {
    const int r = e / K, j = e % K;
    const int64_t t = t0 + r;
    xs[j * C::XS_LD + r] = (t < n) ? to_f32(x[t * d + (int64_t)b * K + j]) : 0.f;
  }
  if (PASS == 0)
    for (int r = tid; r < kRows; r += C::THREADS) red[r] = 0u;
  __syncthreads();

  float acc[4][8];
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

  if (PASS == 0) {
    bool finite = true;
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      float m = 0.f;
#pragma unroll
      for (int c = 0; c < 8; ++c) {
        finite &= isfinite(acc[r][c]);
        m = fmaxf(m, fabsf(acc[r][c]));
      }
      atomicMax(&red[4 * tg + r], __float_as_uint(m));
    }
    if (!finite) report(status, kStatusNonFinite);
    __syncthreads();
    for (int r = tid; r < kRows; r += C::THREADS)
      if (t0 + r < n) atomicMax(&amax_bits[t0 + r], red[r]);
  } else {
    const int64_t words_per_row = d / 8;
    const int64_t word = ((int64_t)b * K + c0 + 8 * cg) / 8;
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int64_t t = t0 + 4 * tg + r;
      if (t >= n) continue;
      const QRow qr = qrow_setup(__uint_as_float(amax_bits[t]), 7.0f);
      int q[8];
#pragma unroll
      for (int c = 0; c < 8; ++c) q[c] = qcode_exact(acc[r][c], qr, 7.0f);
      codes[t * words_per_row + word] = sm4_pack(q);
    }
  }
}

// scale[t] = max|v'_t| / 7 (in place).  Non-finite maxima become 0 and raise the status bit.
__global__ void finalize_scale_kernel(uint32_t* __restrict__ amax_bits, int64_t n, uint32_t* __restrict__ status) {
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= n) return;
  const float a = __uint_as_float(amax_bits[t]);
  float s = 0.f;
  if (isfinite(a))
    s = __fdiv_rn(a, 7.0f);
  else
    report(status, kStatusNonFinite);
  reinterpret_cast<float*>(amax_bits)[t] = s;
}

template <typename Tin, int K>
cudaError_t launch_k(const Tin* x, int64_t n, int64_t d, const float* A, uint8_t* codes, float* scale,
                     uint32_t* status, cudaStream_t stream) {
  using C = ActCfg<K>;
  cudaError_t e = cudaMemsetAsync(scale, 0, (size_t)n * sizeof(float), stream);
  if (e != cudaSuccess) return e;
  auto k0 = transform_quant_kernel<Tin, K, 0>;
  auto k1 = transform_quant_kernel<Tin, K, 1>;
  if ((e = cudaFuncSetAttribute(k0, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM)) != cudaSuccess) return e;
  if ((e = cudaFuncSetAttribute(k1, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM)) != cudaSuccess) return e;
  const int64_t row_tiles = (n + kRows - 1) / kRows;
  if (row_tiles > 0x7FFFFFFF) return cudaErrorInvalidValue;
  const int64_t ny = (d / K) * (K / C::OC);
  if (ny > 65535) return cudaErrorInvalidValue;
  dim3 grid((unsigned)row_tiles, (unsigned)ny);
  uint32_t* amax = reinterpret_cast<uint32_t*>(scale);
  uint32_t* words = reinterpret_cast<uint32_t*>(codes);
  note_launch();
  k0<<<grid, C::THREADS, C::SMEM, stream>>>(x, n, d, A, amax, words, status);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  note_launch();
  k1<<<grid, C::THREADS, C::SMEM, stream>>>(x, n, d, A, amax, words, status);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  note_launch();
  finalize_scale_kernel<<<(unsigned)((n + 255) / 256), 256, 0, stream>>>(amax, n, status);
  return cudaGetLastError();
}

template <typename Tin>
cudaError_t launch_t(const Tin* x, int64_t n, int64_t d, int k, const float* A, uint8_t* codes, float* scale,
                     uint32_t* status, cudaStream_t stream) {
  switch (k) {
    case 16: return launch_k<Tin, 16>(x, n, d, A, codes, scale, status, stream);
    case 32: return launch_k<Tin, 32>(x, n, d, A, codes, scale, status, stream);
    case 64: return launch_k<Tin, 64>(x, n, d, A, codes, scale, status, stream);
    case 128: return launch_k<Tin, 128>(x, n, d, A, codes, scale, status, stream);
    case 256: return launch_k<Tin, 256>(x, n, d, A, codes, scale, status, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

bool transform_quantize_tc_supported(int dtype, int k, int64_t n, int64_t d);
cudaError_t launch_transform_quantize_tc(const void* x, int64_t n, int64_t d, int k, const float* A,
                                         const uint8_t* planes, uint32_t* amax, uint32_t* words, float* scale,
                                         uint32_t* status, cudaStream_t stream);

cudaError_t launch_transform_quantize_tc_fused(const void* x, int64_t n, int64_t d, int k, const float* A,
                                               const uint8_t* planes, uint32_t* amax, uint32_t* words, int e8,
                                               uint32_t* status, cudaStream_t stream);

// planes (optional): T's pre-split bf16 planes (cat_split_transform), used by the tensor-core path.
cudaError_t launch_transform_quantize(const void* x, int dtype, int64_t n, int64_t d, int k, const float* A,
                                      uint8_t* codes, float* scale, uint32_t* status, cudaStream_t stream,
                                      const uint8_t* planes) {
  if (n == 0) return cudaSuccess;
  if (transform_quantize_tc_supported(dtype, k, n, d)) {  // bf16 rows: tensor-core path
    uint32_t* amax = reinterpret_cast<uint32_t*>(scale);
    const cudaError_t ef = launch_transform_quantize_tc_fused(x, n, d, k, A, planes, amax,
                                                              reinterpret_cast<uint32_t*>(codes), 0, status, stream);
    if (ef != cudaErrorNotSupported) return ef;  // done (or failed) in one launch
    if (k != 256) {                               // k = 256 has the fused kernel only
      // two passes with the maxima in device scratch: pass 1 writes the steps
      const cudaError_t es = launch_transform_quantize_tc(x, n, d, k, A, planes, nullptr,
                                                          reinterpret_cast<uint32_t*>(codes), scale, status, stream);
      if (es != cudaErrorNotSupported) return es;
      // more rows than the scratch holds: the maxima in the scale buffer, then a finalize launch
      cudaError_t e = cudaMemsetAsync(scale, 0, (size_t)n * sizeof(float), stream);
      if (e == cudaSuccess) e = launch_transform_quantize_tc(x, n, d, k, A, planes, amax,
                                                             reinterpret_cast<uint32_t*>(codes), nullptr, status, stream);
      if (e != cudaSuccess) return e;
      note_launch();
      finalize_scale_kernel<<<(unsigned)((n + 255) / 256), 256, 0, stream>>>(amax, n, status);
      return cudaGetLastError();
    }
    // k = 256 beyond the fused kernel (more 64-output groups than SMs, more rows than its scratch):
    // the SIMT kernel below
  }
  if (dtype == 0) return launch_t(static_cast<const float*>(x), n, d, k, A, codes, scale, status, stream);
  return launch_t(static_cast<const __nv_bfloat16*>(x), n, d, k, A, codes, scale, status, stream);
}

// The same codes as byte codes ([n][d], one E4M3 byte per code), written by the fused tensor-core
// kernel; cudaErrorNotSupported (nothing launched) where that kernel does not apply.
cudaError_t launch_transform_quantize_e8(const void* x, int dtype, int64_t n, int64_t d, int k, const float* A,
                                         uint8_t* codes8, float* scale, uint32_t* status, cudaStream_t stream,
                                         const uint8_t* planes) {
  if (n == 0) return cudaSuccess;
  if (!transform_quantize_tc_supported(dtype, k, n, d)) return cudaErrorNotSupported;
  return launch_transform_quantize_tc_fused(x, n, d, k, A, planes, reinterpret_cast<uint32_t*>(scale),
                                            reinterpret_cast<uint32_t*>(codes8), 1, status, stream);
}

}  // namespace cat
