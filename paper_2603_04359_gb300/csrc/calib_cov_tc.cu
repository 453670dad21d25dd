// Calibration autocorrelation blocks on tensor cores (bf16 rows; Sec. 4: Sigma_x = E[x x^T], Eq. 10
// keeps the k x k diagonal blocks):  sigma[b] (+)= sum_t x_{t,b} x_{t,b}^T.
//
// D = X_G^T X_G for a group of G = max(k, 128) consecutive channels is one MMA chain contracting
// over tokens: both operands are the same token-by-channel tile, read MN-major (channels
// contiguous) straight from the TMA-loaded layout, so nothing is transposed.  bf16 products are
// exact; tokens accumulate in fp32 in tensor memory.  The tensor cores' fp32 accumulation rounds
// more coarsely than round-to-nearest, with an error that grows with the number of MMA steps, so
// for k <= 128 the 16-token MMA steps go round-robin to NACC = 4 accumulators (512 TMEM columns),
// each summing a quarter of the tokens, and the epilogue adds them (fp32) before widening them to
// float64 with integer operations (the FP64 pipe of this GPU is ~60x slower than FP32).  The result is
// within ~1e-6 of a float64 sum, which moves the block transform by ~1e-6 (its square roots damp
// the calibration error) -- far below the INT4 step.  Only the diagonal k x k blocks are written.
//
// CTA = (channel group, token split).  Warps: 0 TMA producer + TMEM allocator, 1 MMA issuer,
// 2..5 epilogue (one TMEM lane quadrant each).  Tokens arrive in 64-row chunks of 64-channel,
// 128B-swizzled boxes through a 4-stage ring.
#include <cstring>
#include <mutex>

#include "common.cuh"

namespace cat {
namespace {

constexpr int kChunk = 64;      // tokens per stage
constexpr int kStages = 4;
constexpr int kThreads = 192;
constexpr uint32_t kBox = kChunk * 128;  // one 64-token x 64-channel bf16 box, 8 KiB

template <int G2>  // 128-channel tiles per dimension of a group (1: k <= 128, 2: k = 256)
struct CovCfg {
  static constexpr int G = 128 * G2;
  static constexpr int BOXES = G / 64;
  static constexpr uint32_t STAGE = BOXES * kBox;
  static constexpr uint32_t BAR_OFF = kStages * STAGE;
  static constexpr size_t SMEM = BAR_OFF + 256 + 1024;
  static constexpr int NACC = G2 == 1 ? 4 : 1;              // round-robin accumulators per tile
  static constexpr uint32_t TMEM_COLS = G2 * G2 * 128 * NACC;
  // kind::f16, D fp32, A = B = BF16, both MN-major (bits 15, 16), M = N = 128
  static constexpr uint32_t IDESC = (1u << 4) | (1u << 7) | (1u << 10) | (1u << 15) | (1u << 16) |
                                    ((uint32_t)(128 >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
};

struct CovBars {
  uint64_t full[kStages], empty[kStages], acc_full, mma_done;
  uint32_t tmem_addr;
  int abort;
};

// MN-major operand, 128-byte swizzle: 64 contiguous channels per 128-byte row, one row per token,
// 8-token groups 1 KiB apart (SBO), 64-channel atoms kBox bytes apart (LBO).
__device__ __forceinline__ uint64_t sdesc_mnmajor_sw128(uint32_t saddr, uint32_t lbo) {
  return (uint64_t)((saddr >> 4) & 0x3FFFu) | ((uint64_t)((lbo >> 4) & 0x3FFFu) << 16) | (64ull << 32) |
         (1ull << 46) | (2ull << 61);
}

// float -> double without the FP64 pipe: re-bias the exponent of a normal float (zero, subnormal,
// inf and nan take the regular conversion).
__device__ __forceinline__ double f32_to_f64_exact(float f) {
  const uint32_t u = __float_as_uint(f);
  const uint32_t e = (u >> 23) & 0xFFu;
  if (e == 0u || e == 0xFFu) return (double)f;
  const uint64_t bits = ((uint64_t)(u >> 31) << 63) | ((uint64_t)(e - 127u + 1023u) << 52) |
                        ((uint64_t)(u & 0x7FFFFFu) << 29);
  return __longlong_as_double((long long)bits);
}

__device__ __forceinline__ void mma_bf16_ss(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{ .reg .pred p; setp.ne.b32 p, %4, 0; "
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p; }" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

template <int G2>
__global__ void __launch_bounds__(kThreads, 1)
    calib_cov_tc_kernel(const __grid_constant__ CUtensorMap tmX, int n, int d, int k, int tok_per_split,
                        double* __restrict__ sigma, int mode /* 0 store, 1 add, 2 atomic add */,
                        uint32_t* __restrict__ status) {
  using C = CovCfg<G2>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  CovBars* bars = reinterpret_cast<CovBars*>(smem + C::BAR_OFF);
  volatile int* abort_flag = &bars->abort;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int c0 = blockIdx.x * C::G;
  const int t_begin = blockIdx.y * tok_per_split;
  const int t_end = min(n, t_begin + tok_per_split);
  const int chunks = (t_end - t_begin + kChunk - 1) / kChunk;
  const int total_steps = chunks * (kChunk / 16);

  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&bars->full[s], 1);
      mbar_init(&bars->empty[s], 1);
    }
    mbar_init(&bars->acc_full, 1);
    mbar_init(&bars->mma_done, 1);
    bars->abort = 0;
    fence_mbar_init();
  }
  __syncwarp();
  if (warp == 0) tmem_alloc(&bars->tmem_addr, C::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem_addr;

  if (warp == 0) {
    if (lane == 0) {
      prefetch_tensormap(&tmX);
      bool ok = true;
      int c = 0;
      for (; c < chunks && ok; ++c) {
        const uint32_t s = c % kStages;
        if (c >= kStages && !(ok = mbar_wait_bounded(&bars->empty[s], ((c / kStages) - 1) & 1, abort_flag))) break;
        mbar_arrive_expect_tx(&bars->full[s], C::STAGE);
        for (int bx = 0; bx < C::BOXES; ++bx)
          tma_load_2d(smem + s * C::STAGE + bx * kBox, &tmX, c0 + 64 * bx, t_begin + c * kChunk, &bars->full[s]);
      }
      const int first = c > kStages ? c - kStages : 0;
      volatile int no_abort = 0;
      for (int q = first; q < c; ++q) mbar_wait_bounded(&bars->full[q % kStages], (q / kStages) & 1, &no_abort);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      bool ok = true;
      for (int c = 0; c < chunks && ok; ++c) {
        const uint32_t s = c % kStages;
        if (!(ok = mbar_wait_bounded(&bars->full[s], (c / kStages) & 1, abort_flag))) break;
        tc_fence_after();
        const uint32_t base = smem_u32(smem + s * C::STAGE);
#pragma unroll
        for (int kk = 0; kk < kChunk / 16; ++kk) {  // 16 tokens per MMA: 16 rows of 128 B
          const int step = c * (kChunk / 16) + kk;
          const int acc = step % C::NACC;            // accumulator of this 16-token step
#pragma unroll
          for (int ih = 0; ih < G2; ++ih)
#pragma unroll
            for (int jh = 0; jh < G2; ++jh) {
              const uint64_t da = sdesc_mnmajor_sw128(base + 2 * ih * kBox + kk * 2048, kBox);
              const uint64_t db = sdesc_mnmajor_sw128(base + 2 * jh * kBox + kk * 2048, kBox);
              mma_bf16_ss(tmem + ((acc * G2 + ih) * G2 + jh) * 128, da, db, C::IDESC, step >= C::NACC);
            }
        }
        mma_commit(&bars->empty[s]);
      }
      if (ok && chunks > 0) mma_commit(&bars->acc_full);
      mma_commit(&bars->mma_done);
      volatile int no_abort = 0;
      mbar_wait_bounded(&bars->mma_done, 0, &no_abort);
    }
  } else if (chunks > 0) {
    // epilogue: thread = one channel row of the group; keep its diagonal-block columns
    const int quad = warp & 3;
    if (mbar_wait_bounded(&bars->acc_full, 0, abort_flag)) {
      __syncwarp();
      tc_fence_after();
#pragma unroll 1
      for (int ih = 0; ih < G2; ++ih) {
        const int r0 = ih * 128 + quad * 32;            // first row (within the group) of this warp
        const int row = r0 + lane;
        const int ch = c0 + row;                         // channel of this thread
        const int kw = k < 32 ? 32 : k;                  // columns a warp reads for its rows
        const int col0 = (r0 / kw) * kw;                 // first diagonal-block column (within the group)
#pragma unroll 1
        for (int cc = 0; cc < kw / 32; ++cc) {
          const int col = col0 + 32 * cc;
          const int jh = col / 128;
          float v32[32];  // the accumulators summed in fp32 (FP64 arithmetic is scarce on this GPU)
#pragma unroll
          for (int e = 0; e < 32; ++e) v32[e] = 0.f;
          const int used = total_steps < C::NACC ? total_steps : C::NACC;  // accumulators written
#pragma unroll 1
          for (int a = 0; a < used; ++a) {
            uint32_t r[32];
            __syncwarp();
            CAT_TMEM_LD32(tmem + ((uint32_t)(quad * 32) << 16) + ((a * G2 + ih) * G2 + jh) * 128 + (col % 128), r);
            tmem_ld_wait();
#pragma unroll
            for (int e = 0; e < 32; ++e) v32[e] += __uint_as_float(r[e]);
          }
          if (ch >= d) continue;
#pragma unroll
          for (int e = 0; e < 32; ++e) {
            const int jc = col + e;                      // column within the group
            if (k < 32 && (jc / k) != (row / k)) continue;  // k = 16: other half belongs to the neighbour
            double* dst = sigma + (int64_t)ch * k + (jc % k);
            const double v = f32_to_f64_exact(v32[e]);
            if (mode == 2)
              atomicAdd(dst, v);
            else
              *dst = (mode == 1 ? *dst : 0.0) + v;
          }
        }
      }
    }
  }

  __syncthreads();
  if (bars->abort && tid == 0) report(status, kStatusTimeout);
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

int num_sms() {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 148;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0) return 148;
  return sms;
}

template <int G2>
cudaError_t launch_g(const void* x, int64_t n, int64_t d, int k, double* sigma, int accumulate, uint32_t* status,
                     cudaStream_t stream) {
  using C = CovCfg<G2>;
  EncodeTiledFn fn = encode_fn();
  if (!fn) return cudaErrorNotSupported;
  CUtensorMap map;
  memset(&map, 0, sizeof(map));
  cuuint64_t dims[2] = {(cuuint64_t)d, (cuuint64_t)n};
  cuuint64_t strides[1] = {(cuuint64_t)d * 2};
  cuuint32_t box[2] = {64, kChunk};
  cuuint32_t estr[2] = {1, 1};
  if (fn(&map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(x), dims, strides, box, estr,
         CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  static std::once_flag once;
  static cudaError_t attr = cudaSuccess;
  std::call_once(once, [] {
    attr = cudaFuncSetAttribute(calib_cov_tc_kernel<G2>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM);
  });
  if (attr != cudaSuccess) return attr;
  const int64_t groups = (d + C::G - 1) / C::G;
  const int64_t chunks = (n + kChunk - 1) / kChunk;
  int64_t splits = (num_sms() + groups - 1) / groups;  // fill the GPU when there are few groups
  const int64_t min_chunks_per_split = 8;               // but keep >= 512 tokens per CTA
  if (splits > chunks / min_chunks_per_split) splits = chunks / min_chunks_per_split;
  if (splits < 1) splits = 1;
  const int64_t tps = ((chunks + splits - 1) / splits) * kChunk;
  splits = (n + tps - 1) / tps;
  int mode = accumulate ? 1 : 0;
  if (splits > 1) {
    mode = 2;
    if (!accumulate) {
      cudaError_t e = cudaMemsetAsync(sigma, 0, (size_t)d * k * sizeof(double), stream);
      if (e != cudaSuccess) return e;
    }
  }
  dim3 grid((unsigned)groups, (unsigned)splits);
  calib_cov_tc_kernel<G2><<<grid, kThreads, C::SMEM, stream>>>(map, (int)n, (int)d, k, (int)tps, sigma, mode, status);
  return cudaGetLastError();
}

}  // namespace

bool calib_cov_tc_supported(int dtype, int k, int64_t n, int64_t d) {
  return dtype == 1 && n > 0 && n <= 0x7FFFFFFF && d <= 0x7FFFFFFF && (k == 16 || k == 32 || k == 64 || k == 128 || k == 256);
}

cudaError_t launch_calib_cov_tc(const void* x, int64_t n, int64_t d, int k, double* sigma, int accumulate,
                                uint32_t* status, cudaStream_t stream) {
  if (k == 256) return launch_g<2>(x, n, d, k, sigma, accumulate, status, stream);
  return launch_g<1>(x, n, d, k, sigma, accumulate, status, stream);
}

}  // namespace cat
