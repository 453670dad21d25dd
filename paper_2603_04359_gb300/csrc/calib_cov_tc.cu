// Calibration autocorrelation blocks on tensor cores (bf16 rows; Sec. 4: Sigma_x = E[x x^T], Eq. 10
// keeps the k x k diagonal blocks):  sigma[b] (+)= sum_t x_{t,b} x_{t,b}^T.
//
// A group of G = max(k, 128) consecutive channels is contracted over tokens on tensor cores: both
// operands are slices of the same token-by-channel tile, read MN-major (channels contiguous) straight
// from the TMA-loaded layout, so nothing is transposed.  bf16 products are exact; tokens accumulate in
// fp32 in tensor memory.  The tensor cores' fp32 accumulation rounds more coarsely than
// round-to-nearest, with an error that grows with the number of MMA steps, so the 16-token MMA steps
// go round-robin to 4 accumulators (runs of up to 1024 tokens) or 8 (longer runs), and the epilogue
// adds them (fp32) before widening them to float64 with integer operations (the FP64 pipe of this GPU is
// ~60x slower than FP32).  The result is within ~1e-6 of a float64 sum, which moves the block
// transform by ~1e-6 (its square roots damp the calibration error) -- far below the INT4 step.
//
// CTA = (channel group, 128-row half of the group (k = 256), 64-column slice of the group, token
// split): D = X_rows^T X_cols over its tokens, M = 128, N = 64 (one 128-byte swizzle atom of
// channels).  No reduction between CTAs: the column slices of a group are separate CTAs, and only
// long calibration runs split the tokens (their CTAs add their results with float64 atomics).  Only
// the diagonal k x k blocks are written, and through the symmetry of X^T X: lane r of a warp holds
// row r of D and writes it as column r of the block, so a warp's stores of one D column are 32
// consecutive doubles (256 bytes) -- the written blocks are D^T, equal to D up to the rounding of
// the accumulation order.
// Warps: 0 TMA producer + TMEM allocator, 1 MMA issuer, 2..9 epilogue (a TMEM lane quadrant and a
// 32-column half of the slice each).  Tokens arrive in 64-row chunks of 64-channel, 128B-swizzled
// boxes; with up to kStages chunks in flight, the 512-token calibration split of the configurations
// is read in one go.
#include <cstring>
#include <mutex>

#include "common.cuh"

namespace cat {
namespace {

constexpr int kChunk = 64;      // tokens per stage
constexpr int kStages = 8;      // 512 tokens in flight at once
constexpr int kThreads = 320;         // producer, MMA issuer, 8 epilogue warps
constexpr uint32_t kBox = kChunk * 128;  // one 64-token x 64-channel bf16 box, 8 KiB
constexpr int NACC = 8;                  // round-robin accumulators: all 512 TMEM columns
constexpr int kSliceN = 64;              // columns of a CTA's tile: one 128-byte swizzle atom
constexpr uint32_t kTmemCols = NACC * kSliceN;

template <int G2>  // 128-row halves per group (1: k <= 128, 2: k = 256)
struct CovCfg {
  static constexpr int G = 128 * G2;
  static constexpr int SLICES = G / kSliceN;               // column slices per group
  static constexpr int CTAS = G2 * SLICES;                 // CTAs per group (per token split)
  // per stage: the two 64-channel boxes of the CTA's 128 rows (their first holds the column slice
  // when k <= 128), and at k = 256 the column slice's own box
  static constexpr int BOXES = G2 == 1 ? 2 : 3;
  static constexpr uint32_t STAGE = BOXES * kBox;
  static constexpr uint32_t BAR_OFF = kStages * STAGE;
  static constexpr size_t SMEM = BAR_OFF + 256 + 1024;
  // kind::f16, D fp32, A = B = BF16, both MN-major (bits 15, 16), M = 128, N = 64
  static constexpr uint32_t IDESC = (1u << 4) | (1u << 7) | (1u << 10) | (1u << 15) | (1u << 16) |
                                    ((uint32_t)(kSliceN >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
};
static_assert(CovCfg<2>::SMEM <= 227 * 1024, "shared memory budget");

struct CovBars {
  uint64_t full[kStages], empty[kStages], acc_full, mma_done;
  uint32_t tmem_addr;
  int abort;
};
static_assert(sizeof(CovBars) <= 256, "barrier room");

// MN-major operand, 128-byte swizzle: 64 contiguous channels per 128-byte row, one row per token,
// 8-token groups 1 KiB apart (SBO), 64-channel atoms kBox bytes apart (LBO).
__device__ __forceinline__ uint64_t sdesc_mnmajor_sw128(uint32_t saddr, uint32_t lbo) {
  return (uint64_t)((saddr >> 4) & 0x3FFFu) | ((uint64_t)((lbo >> 4) & 0x3FFFu) << 16) | (64ull << 32) |
         (1ull << 46) | (2ull << 61);
}

// float -> double without the FP64 pipe (the exact widening, done in integer registers): a normal
// float re-biases its exponent; a subnormal is normalized (its leading one becomes the implicit
// bit); zero keeps its sign; inf and nan keep their payload under the all-ones exponent.
__device__ __forceinline__ double f32_to_f64_exact(float f) {
  const uint32_t u = __float_as_uint(f);
  const uint32_t e = (u >> 23) & 0xFFu, m = u & 0x7FFFFFu;
  const uint64_t sign = (uint64_t)(u >> 31) << 63;
  uint64_t bits;
  if (e == 0xFFu) {
    bits = sign | (0x7FFull << 52) | ((uint64_t)m << 29);
  } else if (e != 0u) {
    bits = sign | ((uint64_t)(e - 127u + 1023u) << 52) | ((uint64_t)m << 29);
  } else if (m == 0u) {
    bits = sign;
  } else {                                   // m * 2^-149 with its leading one at bit p
    const int p = 31 - __clz(m);
    bits = sign | ((uint64_t)(p - 149 + 1023) << 52) | ((uint64_t)((m << (23 - p)) & 0x7FFFFFu) << 29);
  }
  return __longlong_as_double((long long)bits);
}


// The same widening on its common route: a normal float re-biases its exponent by 1023 - 127 = 896
// (exponent and mantissa shift right by 3 into the high word, the mantissa's low 3 bits go to the
// top of the low word) and a zero keeps its sign -- a few integer operations, no branch.  Subnormals,
// inf and nan (`rare`) must take the exact function above.
__device__ __forceinline__ bool f32_widen_rare(float f) {
  const uint32_t u = __float_as_uint(f), e = u & 0x7F800000u;
  return (u & 0x7FFFFFFFu) != 0u && (e == 0u || e == 0x7F800000u);
}
__device__ __forceinline__ double f32_to_f64_fast(float f) {
  const uint32_t u = __float_as_uint(f);
  const uint32_t mag = u & 0x7FFFFFFFu;
  const uint32_t hi = (u & 0x80000000u) | (mag == 0u ? 0u : (mag >> 3) + (896u << 20));
  return __hiloint2double((int)hi, (int)(u << 29));
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
  const int g = blockIdx.x / C::CTAS;                 // channel group
  const int ih = (blockIdx.x % C::CTAS) / C::SLICES;  // its 128-row half (k = 256)
  const int h = blockIdx.x % C::SLICES;               // its 64-column slice
  const int c0 = g * C::G;                            // first channel of the group
  const int t_begin = blockIdx.y * tok_per_split;
  const int t_end = min(n, t_begin + tok_per_split);
  const int chunks = (t_end - t_begin + kChunk - 1) / kChunk;
  const int total_steps = chunks * (kChunk / 16);
  // accumulators in use: 4 (16 MMA steps each at most) for short runs, 8 beyond -- fewer
  // accumulators are fewer tensor-memory reads in the epilogue, more keep each one's sum short
  const int nacc = total_steps > 4 * 16 ? NACC : NACC / 2;
  // the column slice's box within a stage: one of the row boxes, or its own (k = 256, other half)
  const int b_box = G2 == 1 ? h : ((h >> 1) == ih ? (h & 1) : 2);

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
  pdl_wait_then_release();                        // nothing global or in tensor memory before this
  if (warp == 0) tmem_alloc(&bars->tmem_addr, kTmemCols);
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
        if (c >= kStages && !(ok = mbar_wait_bounded(&bars->empty[s], ((c / kStages) - 1) & 1, abort_flag, __LINE__))) break;
        mbar_arrive_expect_tx(&bars->full[s], C::STAGE);
        const int t0 = t_begin + c * kChunk;
        for (int bx = 0; bx < 2; ++bx)            // the CTA's 128 rows
          tma_load_2d(smem + s * C::STAGE + bx * kBox, &tmX, c0 + ih * 128 + 64 * bx, t0, &bars->full[s]);
        if (G2 == 2)                              // the column slice's box
          tma_load_2d(smem + s * C::STAGE + 2 * kBox, &tmX, c0 + kSliceN * h, t0, &bars->full[s]);
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
        if (!(ok = mbar_wait_bounded(&bars->full[s], (c / kStages) & 1, abort_flag, __LINE__))) break;
        tc_fence_after();
        const uint32_t base = smem_u32(smem + s * C::STAGE);
#pragma unroll
        for (int kk = 0; kk < kChunk / 16; ++kk) {  // 16 tokens per MMA: 16 rows of 128 B
          const int step = c * (kChunk / 16) + kk;
          const uint64_t da = sdesc_mnmajor_sw128(base + kk * 2048, kBox);
          const uint64_t db = sdesc_mnmajor_sw128(base + b_box * kBox + kk * 2048, kBox);
          mma_bf16_ss(tmem + (step % nacc) * kSliceN, da, db, C::IDESC, step >= nacc);
        }
        mma_commit(&bars->empty[s]);
      }
      if (ok && chunks > 0) mma_commit(&bars->acc_full);
      mma_commit(&bars->mma_done);
      volatile int no_abort = 0;
      mbar_wait_bounded(&bars->mma_done, 0, &no_abort);
    }
  } else {
    // ---------------------------------------------------------------- epilogue: one tile row per lane
    const int quad = warp & 3;                        // the TMEM lane quadrant this warp may access
    const int lk = 31 - __clz(k);                     // k = 2^lk
    const int rg = ih * 128 + quad * 32 + lane;       // this lane's row within the group
    const bool live = chunks > 0 && mbar_wait_bounded(&bars->acc_full, 0, abort_flag, __LINE__);
    const int used = total_steps < nacc ? total_steps : nacc;   // accumulators written
    if (__all_sync(0xFFFFFFFFu, live)) {              // warp-uniform: TMEM loads need the whole warp
      tc_fence_after();
      {
        const int cc = (warp - 2) >> 2;               // this warp's 32-column chunk of the slice
        const int cg0 = kSliceN * h + 32 * cc;        // first column (within the group) of this chunk
        // the chunk's columns share a diagonal block with some lane's row
        const bool need = (rg / k) * k < cg0 + 32 && cg0 < (rg / k + 1) * k;
        if (__any_sync(0xFFFFFFFFu, need)) {
        float v[32];
#pragma unroll
        for (int e = 0; e < 32; ++e) v[e] = 0.f;
#pragma unroll 1
        for (int a = 0; a < used; a += 2) {           // two accumulators per tensor-memory round trip
          uint32_t rr[32], rq[32];
          __syncwarp();
          CAT_TMEM_LD32(tmem + ((uint32_t)(quad * 32) << 16) + a * kSliceN + 32 * cc, rr);
          if (a + 1 < used) CAT_TMEM_LD32(tmem + ((uint32_t)(quad * 32) << 16) + (a + 1) * kSliceN + 32 * cc, rq);
          tmem_ld_wait();
#pragma unroll
          for (int e = 0; e < 32; ++e) v[e] += __uint_as_float(rr[e]);
          if (a + 1 < used) {
#pragma unroll
            for (int e = 0; e < 32; ++e) v[e] += __uint_as_float(rq[e]);
          }
        }
        // D[rg][cg] = sigma entry (cg, rg) of their block (the symmetry): for each column the lanes
        // of a block write consecutive doubles.  k is a power of two (shifts, no divisions), and the
        // store mode is chosen once per chunk: inside the element loop the compiler would turn the
        // read-modify-write of `add` (an FP64 add and a global load per element) into work every
        // element pays for.
        const int row = c0 + rg;
        double* rowbase = sigma + ((int64_t)(row >> lk) << (2 * lk)) + (row & (k - 1));
        const int rblk = rg >> lk;
        uint32_t ok_mask = 0u;                        // columns of the chunk this lane writes
        bool rare = false;
        double w[32];
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          const int cg = cg0 + e;
          if ((cg >> lk) == rblk && row < d && c0 + cg < d) ok_mask |= 1u << e;
          rare |= f32_widen_rare(v[e]);
          w[e] = f32_to_f64_fast(v[e]);
        }
        if (__any_sync(0xFFFFFFFFu, rare)) {         // a subnormal, inf or nan in the warp's chunk
#pragma unroll
          for (int e = 0; e < 32; ++e) w[e] = f32_to_f64_exact(v[e]);
        }
        // entry (col % k, row % k) of the block sits (col % k) k doubles after its row's base
        const int cbase = (c0 + cg0) & (k - 1);
        if (mode == 0) {
#pragma unroll
          for (int e = 0; e < 32; ++e)
            if (ok_mask >> e & 1u) rowbase[(int64_t)((cbase + e) & (k - 1)) << lk] = w[e];
        } else if (mode == 1) {
#pragma unroll
          for (int e = 0; e < 32; ++e)
            if (ok_mask >> e & 1u) rowbase[(int64_t)((cbase + e) & (k - 1)) << lk] += w[e];
        } else {
#pragma unroll
          for (int e = 0; e < 32; ++e)
            if (ok_mask >> e & 1u) atomicAdd(rowbase + ((int64_t)((cbase + e) & (k - 1)) << lk), w[e]);
        }
        }
      }
    }
    tc_fence_before();
  }

  __syncthreads();
  if (bars->abort && tid == 0) report(status, timeout_bits(kWhereCalib, bars->abort));
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
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
  const int sms = num_sms();
  // token splits (their CTAs add with float64 atomics) only for long calibration runs: >= 2048 tokens
  // per CTA, within one wave
  int64_t ysplits = sms / (groups * C::CTAS);
  if (ysplits > chunks / 32) ysplits = chunks / 32;
  if (ysplits < 1) ysplits = 1;
  const int64_t tps = ((chunks + ysplits - 1) / ysplits) * kChunk;
  int mode = accumulate ? 1 : 0;
  if (ysplits > 1) {
    mode = 2;
    if (!accumulate) {
      cudaError_t e = cudaMemsetAsync(sigma, 0, (size_t)d * k * sizeof(double), stream);
      if (e != cudaSuccess) return e;
    }
  }
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = dim3((unsigned)(groups * C::CTAS), (unsigned)ysplits, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = C::SMEM;
  cfg.stream = stream;
  // not a programmatic dependent launch: measured, one gained ~0.4 us per c4 step and lost ~0.7 us per
  // c2 step (the kernel still releases its dependents early)
  note_launch();
  cudaError_t e = cudaLaunchKernelEx(&cfg, calib_cov_tc_kernel<G2>, map, (int)n, (int)d, k, (int)tps, sigma, mode,
                                     status);
  if (e != cudaSuccess) return e;
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
