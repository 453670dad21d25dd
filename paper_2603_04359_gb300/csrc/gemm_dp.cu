// Integer GEMM of b-bit codes held as E4M3 digit planes, on 5th-generation tensor cores (sm_103a).
//
//   acc[t, o] = sum_i (q_x[t, i] - z[t]) q_w[o, i],   y[t, o] = acc * s_x[t] * s_w[o]    (Sec. 3, Eq. 5)
//
// Codes of more than 4 bits do not fit one FP8 operand exactly, so each code is split into base-16
// digits, q = d0 + 16 d1 (|d| <= 16), one E4M3 byte per digit (d * 2^-9, exact).  With DX activation
// and DW weight digit planes the product splits by digit weight:
//   sum_i q_x q_w = sum_{g} 16^g P_g,   P_g = sum_{a + b = g} sum_i d_a(x) d_b(w),
// and every P_g is accumulated by tcgen05.mma kind::f8f6f4 in its own fp32 tensor-memory accumulator:
// its terms are products of digits (|d_x d_w| <= 16 * 8), so |P_g| * 2^18 stays below 2^24 and the
// accumulation is exact for d_in up to 2^16 (checked on the host).  The epilogue turns each P_g into
// an integer and adds them in int32; asymmetric activations then subtract z[t] times the weight row's
// code sum (the zero-point correction), and the product is scaled by the two steps in fp32.
//
// Tile: 128 tokens (MMA M) x 128 output channels (MMA N) per CTA, K steps of 128 codes (one 128-byte
// swizzle atom per row and plane).  One TMA producer thread loads, per K step, every digit plane of
// the token tile and of the weight tile through a ring of stages (full / empty mbarriers); one thread
// issues the MMAs (four of K = 32 per digit pair); four epilogue warps (thread = token row = TMEM
// lane) read the accumulators, combine, scale and store y.  Every wait is bounded.
#include <cstring>
#include <mutex>

#include "common.cuh"

namespace cat {
namespace {

constexpr int BM = 128, BN = 128, KB = 128;          // tokens, channels, codes (bytes) per K step
constexpr uint32_t kTile = BM * KB;                  // 16 KiB per plane and operand (BN == BM)
constexpr int kThreads = 192;                        // warp 0 TMA, warp 1 MMA, warps 2..5 epilogue
constexpr int kEpiWarp0 = 2;
constexpr size_t kSmemBudget = 200 * 1024;

template <int DX, int DW>
struct DpGemmCfg {
  static constexpr int G = DX + DW - 1;                                   // accumulators (digit weights)
  static constexpr uint32_t STAGE = (uint32_t)(DX + DW) * kTile;
  static constexpr int S = (int)(kSmemBudget / STAGE) < 8 ? (int)(kSmemBudget / STAGE) : 8;
  static constexpr uint32_t TMEM_COLS = G * BN <= 128 ? 128 : (G * BN <= 256 ? 256 : 512);
  static constexpr size_t SMEM = 1024 + (size_t)S * STAGE + 256;
  static_assert(S >= 2, "stages");
};

// Bound of the pipeline waits (ns); kWaitLimitNs unless a test shortens it (cat_set_wait_limit_ns).
__device__ uint64_t g_dp_wait_limit = kWaitLimitNs;

struct DpBars {
  uint64_t full[8], empty[8], acc_full, mma_done;
  uint32_t tmem_addr;
  int abort;
};

__device__ __forceinline__ void tma_load_3d(void* smem_dst, const CUtensorMap* map, int32_t x, int32_t y, int32_t z,
                                            uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(
          smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void mma_ss_f8(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{ .reg .pred p; setp.ne.b32 p, %4, 0; "
      "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p; }" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

template <int DX, int DW>
__global__ void __launch_bounds__(kThreads, 1)
    dp_gemm_kernel(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmW,
                   const float* __restrict__ sx, const int32_t* __restrict__ zx, const float* __restrict__ sw,
                   const int32_t* __restrict__ w_rowsum, int n, int d_in, int d_out, float* __restrict__ y,
                   int32_t* __restrict__ acc_out, uint32_t* __restrict__ status) {
  using C = DpGemmCfg<DX, DW>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  DpBars* bars = reinterpret_cast<DpBars*>(smem + (size_t)C::S * C::STAGE);
  volatile int* abort_flag = &bars->abort;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int o0 = blockIdx.x * BN, t0 = blockIdx.y * BM;
  const int num_k = (d_in + KB - 1) / KB;
  const uint64_t lim = g_dp_wait_limit;

  if (tid == 0) {
    for (int s = 0; s < C::S; ++s) {
      mbar_init(&bars->full[s], 1);
      mbar_init(&bars->empty[s], 1);
    }
    mbar_init(&bars->acc_full, 1);
    mbar_init(&bars->mma_done, 1);
    bars->abort = 0;
    fence_mbar_init();
  }
  pdl_wait_then_release();
  if (warp == 1) tmem_alloc(&bars->tmem_addr, C::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem_addr;

  if (warp == 0) {
    // ------------------------------------------------------------------ TMA producer
    if (lane == 0) {
      prefetch_tensormap(&tmX);
      prefetch_tensormap(&tmW);
      int kb = 0;
      for (; kb < num_k; ++kb) {
        const int s = kb % C::S;
        if (kb >= C::S && !mbar_wait_bounded(&bars->empty[s], ((kb / C::S) - 1) & 1, abort_flag, __LINE__, lim)) break;
        uint8_t* st = smem + (size_t)s * C::STAGE;
        mbar_arrive_expect_tx(&bars->full[s], C::STAGE);
#pragma unroll
        for (int p = 0; p < DX; ++p) tma_load_3d(st + p * kTile, &tmX, kb * KB, t0, p, &bars->full[s]);
#pragma unroll
        for (int p = 0; p < DW; ++p) tma_load_3d(st + (DX + p) * kTile, &tmW, kb * KB, o0, p, &bars->full[s]);
      }
      // loads in flight land before the CTA exits (their stages were never waited for by the MMA
      // thread if it gave up)
      volatile int no_abort = 0;
      for (int q = kb > C::S ? kb - C::S : 0; q < kb; ++q) mbar_wait_bounded(&bars->full[q % C::S], (q / C::S) & 1, &no_abort);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t kIdesc = idesc_e4m3_f32(BM, BN);
      bool started[C::G];
#pragma unroll
      for (int g = 0; g < C::G; ++g) started[g] = false;
      for (int kb = 0; kb < num_k; ++kb) {
        const int s = kb % C::S;
        if (!mbar_wait_bounded(&bars->full[s], (kb / C::S) & 1, abort_flag, __LINE__, lim)) break;
        tc_fence_after();
        const uint32_t base = smem_u32(smem + (size_t)s * C::STAGE);
#pragma unroll
        for (int a = 0; a < DX; ++a)
#pragma unroll
          for (int b = 0; b < DW; ++b) {
            const int g = a + b;
            const uint64_t da = sdesc_kmajor_sw128(base + a * kTile);
            const uint64_t db = sdesc_kmajor_sw128(base + (DX + b) * kTile);
#pragma unroll
            for (int kk = 0; kk < KB / 32; ++kk) {   // K = 32 bytes (E4M3) per MMA: +32 B in the atom
              mma_ss_f8(tmem + g * BN, da + 2 * kk, db + 2 * kk, kIdesc, started[g] ? 1u : 0u);
              started[g] = true;
            }
          }
        mma_commit(&bars->empty[s]);
      }
      mma_commit(&bars->acc_full);
      mma_commit(&bars->mma_done);
      volatile int no_abort = 0;
      mbar_wait_bounded(&bars->mma_done, 0, &no_abort);
    }
  } else {
    // ------------------------------------------------------------------ epilogue: token row = TMEM lane
    const int quad = warp & 3;
    const int t = t0 + quad * 32 + lane;
    const bool t_ok = t < n;
    const float sxt = t_ok ? sx[t] : 0.f;
    const int zt = (t_ok && zx) ? zx[t] : 0;
    if (mbar_wait_bounded(&bars->acc_full, 0, abort_flag, __LINE__, lim)) {
      __syncwarp();
      tc_fence_after();
#pragma unroll 1
      for (int c = 0; c < BN / 32; ++c) {
        int acc[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) acc[j] = 0;
#pragma unroll
        for (int g = 0; g < C::G; ++g) {
          uint32_t r[32];
          __syncwarp();
          CAT_TMEM_LD32(tmem + ((uint32_t)(quad * 32) << 16) + g * BN + c * 32, r);
          tmem_ld_wait();
#pragma unroll
          for (int j = 0; j < 32; ++j) acc[j] += __float2int_rn(__uint_as_float(r[j]) * kAccScale) * (1 << (4 * g));
        }
        if (!t_ok) continue;
        const int ob = o0 + c * 32;
        float* yrow = y + (int64_t)t * d_out;
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const int o = ob + j;
          if (o >= d_out) break;
          // the zero-point correction in 64 bits: both terms fit int32, their difference too
          const int a = (int)((long long)acc[j] - (zx ? (long long)zt * w_rowsum[o] : 0ll));
          yrow[o] = (float)a * sxt * sw[o];
          if (acc_out) acc_out[(int64_t)t * d_out + o] = a;
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (bars->abort && tid == 0) report(status, timeout_bits(kWhereGemmDp, bars->abort));
  if (warp == 1) {
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

// Tensor map of D digit planes [D][rows][d_in] bytes: box 128 codes x 128 rows x 1 plane, 128B swizzle;
// rows past the end read as zero.
bool plane_map(CUtensorMap* map, const uint8_t* planes, int64_t rows, int64_t d_in, int D) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  memset(map, 0, sizeof(*map));
  cuuint64_t dims[3] = {(cuuint64_t)d_in, (cuuint64_t)rows, (cuuint64_t)D};
  cuuint64_t strides[2] = {(cuuint64_t)d_in, (cuuint64_t)(rows * d_in)};
  cuuint32_t box[3] = {(cuuint32_t)KB, (cuuint32_t)BM, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 3, const_cast<uint8_t*>(planes), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int DX, int DW>
cudaError_t launch_dx_dw(const CUtensorMap& mx, const CUtensorMap& mw, const float* sx, const int32_t* zx,
                         const float* sw, const int32_t* rowsum, int64_t n, int64_t d_in, int64_t d_out, float* y,
                         int32_t* acc_out, uint32_t* status, cudaStream_t stream) {
  using C = DpGemmCfg<DX, DW>;
  static std::once_flag once;
  static cudaError_t attr = cudaSuccess;
  std::call_once(once, [] {
    attr = cudaFuncSetAttribute(dp_gemm_kernel<DX, DW>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM);
  });
  if (attr != cudaSuccess) return attr;
  const int64_t gx = (d_out + BN - 1) / BN, gy = (n + BM - 1) / BM;
  if (gx > 0x7FFFFFFF || gy > 65535) return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = dim3((unsigned)gx, (unsigned)gy, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = C::SMEM;
  cfg.stream = stream;
  cudaLaunchAttribute attrs[1] = {pdl_attr()};
  cfg.attrs = attrs;
  cfg.numAttrs = 1;
  note_launch();
  return cudaLaunchKernelEx(&cfg, dp_gemm_kernel<DX, DW>, mx, mw, sx, zx, sw, rowsum, (int)n, (int)d_in, (int)d_out, y,
                            acc_out, status);
}

}  // namespace

cudaError_t set_dp_wait_limit(uint64_t ns) { return cudaMemcpyToSymbol(g_dp_wait_limit, &ns, sizeof(ns)); }

// x_planes [DX][n][d_in], w_planes [DW][d_out][d_in] digit bytes; zx / w_rowsum both given for
// asymmetric activations (else both NULL).
cudaError_t launch_dp_gemm(const uint8_t* x_planes, int DX, const float* sx, const int32_t* zx, const uint8_t* w_planes,
                           int DW, const float* sw, const int32_t* w_rowsum, int64_t n, int64_t d_in, int64_t d_out,
                           float* y, int32_t* acc_out, uint32_t* status, cudaStream_t stream) {
  if (n == 0) return cudaSuccess;
  CUtensorMap mx, mw;
  if (!plane_map(&mx, x_planes, n, d_in, DX) || !plane_map(&mw, w_planes, d_out, d_in, DW)) return cudaErrorInvalidValue;
  if (DX == 1 && DW == 1) return launch_dx_dw<1, 1>(mx, mw, sx, zx, sw, w_rowsum, n, d_in, d_out, y, acc_out, status, stream);
  if (DX == 2 && DW == 1) return launch_dx_dw<2, 1>(mx, mw, sx, zx, sw, w_rowsum, n, d_in, d_out, y, acc_out, status, stream);
  if (DX == 1 && DW == 2) return launch_dx_dw<1, 2>(mx, mw, sx, zx, sw, w_rowsum, n, d_in, d_out, y, acc_out, status, stream);
  if (DX == 2 && DW == 2) return launch_dx_dw<2, 2>(mx, mw, sx, zx, sw, w_rowsum, n, d_in, d_out, y, acc_out, status, stream);
  return cudaErrorInvalidValue;
}

}  // namespace cat
