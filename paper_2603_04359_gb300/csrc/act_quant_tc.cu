// Block transform + per-row absmax + INT4 quantization on tensor cores (bf16 rows, k = 64 or 128).
//
//   v'_{t,b} = A_b v_{t,b}      (activations: A_b = T_b, Sec. 3 Eq. 5; weight rows: A_b = (T_b^{-1})^T)
//
// The row values are bf16, hence exact MMA operands.  Each fp32 block A_b is split into three bf16
// matrices A_b = H + M + L (24 significant bits: H = bf16(A), M = bf16(A - H), L = bf16(A - H - M)),
// so D = V H^T + V M^T + V L^T on kind::f16 tensor cores gives exact products and fp32 accumulation,
// the same accuracy as an fp32 FMA loop.  The 128-row tile of V arrives by TMA (128B swizzle); the
// three splits are written into 128B-swizzled shared memory once per block by converter warps.
//
// Work unit = (block b, 128-row tile); a persistent CTA walks a contiguous, block-major range of
// units, so it re-splits A_b only when b changes.  D is double-buffered in tensor memory.  The
// epilogue thread owns one row (TMEM lane), so its row maximum needs no reduction:
//   pass 0: atomicMax of the row maxima into the scale buffer (float bits, non-negative),
//   pass 1: recompute, q = clamp(rint(v' * (7 / max)), -7, 7), pack SM4x8, store.
// Warps: 0 TMA producer + TMEM allocator, 1 MMA issuer, 4..7 epilogue, 8..15 converters.
#include <cstring>
#include <mutex>

#include "common.cuh"

namespace cat {
namespace {

constexpr int TM = 128;                 // rows per tile
constexpr int kThreads = 512;
constexpr int kEpiWarp0 = 4, kCvtWarp0 = 8, kCvtWarps = 8;
constexpr int kXStages = 2;

template <int K>
struct TcCfg {
  static constexpr int ATOMS = K / 64;                       // 128-byte K atoms (64 bf16)
  static constexpr uint32_t X_STAGE = TM * K * 2;            // bf16 tile of 128 rows
  static constexpr uint32_t SPLIT = K * K * 2;               // one bf16 split of A_b
  static constexpr uint32_t X_OFF = 0;
  static constexpr uint32_t T_OFF = kXStages * X_STAGE;
  static constexpr uint32_t BAR_OFF = T_OFF + 3 * SPLIT;
  static constexpr size_t SMEM = BAR_OFF + 256 + 1024;
  static constexpr uint32_t TMEM_COLS = 2 * K;               // double-buffered accumulator
  // kind::f16: D fp32 (bit 4), A = B = BF16 (format 1 at bits 7 and 10), K-major, M = 128, N = K
  static constexpr uint32_t IDESC = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(K >> 3) << 17) |
                                    ((uint32_t)(TM >> 4) << 24);
};

struct TcBars {
  uint64_t x_full[kXStages], x_empty[kXStages], d_full[2], d_empty[2], t_full, t_empty, mma_done;
  uint32_t tmem_addr;
  int abort;
};

__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                         uint32_t accumulate) {
  asm volatile(
      "{ .reg .pred p; setp.ne.b32 p, %4, 0; "
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p; }" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ uint32_t bf16x2_bits(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

template <int K, int PASS>
__global__ void __launch_bounds__(kThreads, 1)
    transform_quant_tc_kernel(const __grid_constant__ CUtensorMap tmX, const float* __restrict__ A, int n, int d,
                              uint32_t* __restrict__ amax_bits, uint32_t* __restrict__ codes,
                              uint32_t* __restrict__ status) {
  using C = TcCfg<K>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* xs = smem + C::X_OFF;
  uint8_t* ts = smem + C::T_OFF;
  TcBars* bars = reinterpret_cast<TcBars*>(smem + C::BAR_OFF);
  volatile int* abort_flag = &bars->abort;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nb = d / K;
  const int num_tiles = (n + TM - 1) / TM;
  const int64_t units = (int64_t)nb * num_tiles;
  const int64_t u0 = units * blockIdx.x / gridDim.x;
  const int64_t u1 = units * (blockIdx.x + 1) / gridDim.x;

  if (tid == 0) {
    for (int s = 0; s < kXStages; ++s) {
      mbar_init(&bars->x_full[s], 1);
      mbar_init(&bars->x_empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&bars->d_full[s], 1);
      mbar_init(&bars->d_empty[s], 4);
    }
    mbar_init(&bars->t_full, kCvtWarps);
    mbar_init(&bars->t_empty, 1);
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
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      prefetch_tensormap(&tmX);
      bool ok = true;
      uint32_t j = 0;
      for (int64_t u = u0; u < u1 && ok; ++u, ++j) {
        const int b = (int)(u / num_tiles), tile = (int)(u % num_tiles);
        const uint32_t s = j % kXStages;
        if (j >= kXStages && !(ok = mbar_wait_bounded(&bars->x_empty[s], ((j / kXStages) - 1) & 1, abort_flag))) break;
        mbar_arrive_expect_tx(&bars->x_full[s], C::X_STAGE);
#pragma unroll
        for (int a = 0; a < C::ATOMS; ++a)
          tma_load_2d(xs + s * C::X_STAGE + a * (TM * 128), &tmX, b * K + 64 * a, tile * TM, &bars->x_full[s]);
      }
      const uint32_t issued = j, first = issued > kXStages ? issued - kXStages : 0;
      volatile int no_abort = 0;
      for (uint32_t q = first; q < issued; ++q)
        mbar_wait_bounded(&bars->x_full[q % kXStages], (q / kXStages) & 1, &no_abort);
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      bool ok = true;
      uint32_t j = 0, version = 0;
      int cur_b = -1;
      for (int64_t u = u0; u < u1 && ok; ++u, ++j) {
        const int b = (int)(u / num_tiles);
        if (b != cur_b) {
          if (!(ok = mbar_wait_bounded(&bars->t_full, version & 1, abort_flag))) break;
          ++version;
          cur_b = b;
        }
        const uint32_t s = j % kXStages, sd = j & 1;
        if (!(ok = mbar_wait_bounded(&bars->x_full[s], (j / kXStages) & 1, abort_flag))) break;
        if (j >= 2 && !(ok = mbar_wait_bounded(&bars->d_empty[sd], ((j >> 1) - 1) & 1, abort_flag))) break;
        tc_fence_after();
        const uint32_t dcol = tmem + sd * K;
        const uint32_t xbase = smem_u32(xs + s * C::X_STAGE);
        const uint32_t tbase = smem_u32(ts);
#pragma unroll
        for (int kk = 0; kk < K / 16; ++kk) {  // K = 16 bf16 = 32 bytes per MMA
          const uint32_t a_off = (kk >> 2) * (TM * 128) + (kk & 3) * 32;
          const uint32_t b_off = (kk >> 2) * (K * 128) + (kk & 3) * 32;
          const uint64_t da = sdesc_kmajor_sw128(xbase + a_off);
#pragma unroll
          for (int sp = 0; sp < 3; ++sp)
            mma_bf16(dcol, da, sdesc_kmajor_sw128(tbase + sp * C::SPLIT + b_off), C::IDESC, (kk | sp) != 0);
        }
        mma_commit(&bars->x_empty[s]);
        mma_commit(&bars->d_full[sd]);
        const bool last_of_block = (u + 1 >= u1) || ((int)((u + 1) / num_tiles) != b);
        if (last_of_block) mma_commit(&bars->t_empty);
      }
      mma_commit(&bars->mma_done);
      volatile int no_abort = 0;
      mbar_wait_bounded(&bars->mma_done, 0, &no_abort);
    }
  } else if (warp >= kCvtWarp0) {
    // ---------------------------------------------------------------- split A_b into bf16 H, M, L
    const int ct = tid - kCvtWarp0 * 32;
    bool ok = true;
    uint32_t version = 0;
    int cur_b = -1;
    for (int64_t u = u0; u < u1 && ok; ++u) {
      const int b = (int)(u / num_tiles);
      if (b == cur_b) continue;
      if (version > 0 && !(ok = mbar_wait_bounded(&bars->t_empty, (version - 1) & 1, abort_flag))) break;
      cur_b = b;
      const float* Ab = A + (size_t)b * K * K;
      for (int ch = ct; ch < K * K / 8; ch += kCvtWarps * 32) {  // 8 consecutive inputs of one output row
        const int i = ch / (K / 8), j0 = (ch % (K / 8)) * 8;
        const float4 p = *reinterpret_cast<const float4*>(Ab + (size_t)i * K + j0);
        const float4 q = *reinterpret_cast<const float4*>(Ab + (size_t)i * K + j0 + 4);
        const float v[8] = {p.x, p.y, p.z, p.w, q.x, q.y, q.z, q.w};
        uint32_t hw[4], mw[4], lw[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float a0 = v[2 * e], a1 = v[2 * e + 1];
          const float h0 = __bfloat162float(__float2bfloat16_rn(a0)), h1 = __bfloat162float(__float2bfloat16_rn(a1));
          const float r0 = a0 - h0, r1 = a1 - h1;  // exact
          const float m0 = __bfloat162float(__float2bfloat16_rn(r0)), m1 = __bfloat162float(__float2bfloat16_rn(r1));
          hw[e] = bf16x2_bits(h0, h1);
          mw[e] = bf16x2_bits(m0, m1);
          lw[e] = bf16x2_bits(r0 - m0, r1 - m1);
        }
        const int atom = j0 / 64, chunk = (j0 % 64) / 8;
        const uint32_t off = atom * (K * 128) + i * 128 + ((chunk ^ (i & 7)) << 4);
        *reinterpret_cast<uint4*>(ts + off) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
        *reinterpret_cast<uint4*>(ts + C::SPLIT + off) = make_uint4(mw[0], mw[1], mw[2], mw[3]);
        *reinterpret_cast<uint4*>(ts + 2 * C::SPLIT + off) = make_uint4(lw[0], lw[1], lw[2], lw[3]);
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars->t_full);
      ++version;
    }
  } else if (warp >= kEpiWarp0) {
    // ---------------------------------------------------------------- epilogue: one row per thread
    const int quad = warp & 3;
    const int64_t words_per_row = d / 8;
    bool ok = true, finite = true;
    uint32_t j = 0;
    for (int64_t u = u0; u < u1 && ok; ++u, ++j) {
      const int b = (int)(u / num_tiles), tile = (int)(u % num_tiles);
      const uint32_t sd = j & 1;
      const int t = tile * TM + quad * 32 + lane;
      float inv = 0.f;
      if (PASS == 1 && t < n) {
        const float a = __uint_as_float(amax_bits[t]);
        inv = (isfinite(a) && a > 0.f) ? __fdiv_rn(7.0f, a) : 0.f;
      }
      if (!(ok = mbar_wait_bounded(&bars->d_full[sd], (j >> 1) & 1, abort_flag))) break;
      __syncwarp();
      tc_fence_after();
      float m = 0.f;
#pragma unroll 1
      for (int c = 0; c < K / 32; ++c) {
        uint32_t r[32];
        __syncwarp();
        CAT_TMEM_LD32(tmem + ((uint32_t)(quad * 32) << 16) + sd * K + c * 32, r);
        tmem_ld_wait();
        if (PASS == 0) {
#pragma unroll
          for (int e = 0; e < 32; ++e) {
            const float v = __uint_as_float(r[e]);
            finite &= isfinite(v);
            m = fmaxf(m, fabsf(v));
          }
        } else if (t < n) {
          uint32_t w[4];
#pragma unroll
          for (int g = 0; g < 4; ++g) {
            int q[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              const float v = __uint_as_float(r[8 * g + e]) * inv;
              const int iv = isfinite(v) ? __float2int_rn(v) : 0;
              q[e] = iv > 7 ? 7 : (iv < -7 ? -7 : iv);
            }
            w[g] = sm4_pack(q);
          }
          *reinterpret_cast<uint4*>(codes + (int64_t)t * words_per_row + ((int64_t)b * K + c * 32) / 8) =
              make_uint4(w[0], w[1], w[2], w[3]);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars->d_empty[sd]);
      if (PASS == 0 && t < n) atomicMax(&amax_bits[t], __float_as_uint(m));
    }
    if (PASS == 0 && !finite) report(status, kStatusNonFinite);
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

template <int K>
cudaError_t launch_k(const __nv_bfloat16* x, int64_t n, int64_t d, const float* A, uint32_t* amax, uint32_t* words,
                     uint32_t* status, cudaStream_t stream) {
  using C = TcCfg<K>;
  EncodeTiledFn fn = encode_fn();
  if (!fn) return cudaErrorNotSupported;
  CUtensorMap map;
  memset(&map, 0, sizeof(map));
  cuuint64_t dims[2] = {(cuuint64_t)d, (cuuint64_t)n};
  cuuint64_t strides[1] = {(cuuint64_t)d * 2};
  cuuint32_t box[2] = {64, TM};
  cuuint32_t estr[2] = {1, 1};
  if (fn(&map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<__nv_bfloat16*>(x), dims, strides, box, estr,
         CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  auto k0 = transform_quant_tc_kernel<K, 0>;
  auto k1 = transform_quant_tc_kernel<K, 1>;
  static std::once_flag once;
  static cudaError_t attr = cudaSuccess;
  std::call_once(once, [&] {
    attr = cudaFuncSetAttribute(k0, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM);
    if (attr == cudaSuccess) attr = cudaFuncSetAttribute(k1, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM);
  });
  if (attr != cudaSuccess) return attr;
  const int64_t units = (d / K) * ((n + TM - 1) / TM);
  const int grid = (int)(units < num_sms() ? units : num_sms());
  k0<<<grid, kThreads, C::SMEM, stream>>>(map, A, (int)n, (int)d, amax, words, status);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  k1<<<grid, kThreads, C::SMEM, stream>>>(map, A, (int)n, (int)d, amax, words, status);
  return cudaGetLastError();
}

}  // namespace

bool transform_quantize_tc_supported(int dtype, int k, int64_t n, int64_t d) {
  return dtype == 1 && (k == 64 || k == 128) && n <= 0x7FFFFFFF && d <= 0x7FFFFFFF;
}

// Passes 0 and 1; the caller zeroes the scale buffer before and finalizes it after.
cudaError_t launch_transform_quantize_tc(const void* x, int64_t n, int64_t d, int k, const float* A, uint32_t* amax,
                                         uint32_t* words, uint32_t* status, cudaStream_t stream) {
  const __nv_bfloat16* xb = static_cast<const __nv_bfloat16*>(x);
  if (k == 64) return launch_k<64>(xb, n, d, A, amax, words, status, stream);
  if (k == 128) return launch_k<128>(xb, n, d, A, amax, words, status, stream);
  return cudaErrorInvalidValue;
}

}  // namespace cat
