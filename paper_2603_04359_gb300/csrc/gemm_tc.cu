// W4A4 GEMM with fused dequantization on 5th-generation tensor cores (sm_103a).
//
//   acc[t, o] = sum_i q_x[t, i] q_w[o, i]          (exact integers)
//   y[t, o]   = acc[t, o] * s_x[t] * s_w[o]        (Sec. 3, Eq. 5: y ~ Q(W T^{-1}) Q(T x))
//
// sm_103a has no integer tcgen05 MMA, so the INT4 codes run on the FP8 path: an SM4x8 word
// decodes with two masks into the E4M3 bytes q * 2^-9 (subnormals, exact), the MMA accumulates
// products q_x q_w 2^-18 in fp32 tensor memory (exact: |acc| <= 49 d_in < 2^24), and the epilogue
// multiplies by 2^18 s_x s_w.
//
// Persistent warp-specialized CTA (one per SM), output tile 128 tokens x 256 channels, K step 128:
//   warp 0      TMA producer: packed A (128 x 64 B) and B (256 x 64 B) tiles into a 4-stage ring
//   warp 1      TMEM allocator; lane 0 issues tcgen05.mma (4 x K=32 per K step) and commits
//   warps 2..5  decode packed stages into 128B-swizzled E4M3 operand stages (2-stage ring), then
//               run the epilogue: tcgen05.ld of their TMEM lane quadrant, scale, store y.
// Every mbarrier wait is bounded (common.cuh); a wait that gives up raises the device status
// word and every role drains and exits; TMEM is always released.
#include <mutex>

#include "common.cuh"

namespace cat {
namespace {

constexpr int BM = 128, BN = 256, BK = 128;
constexpr int BKP = BK / 2;   // packed bytes per row per K step
constexpr int SP = 4;         // packed stages
constexpr int SE = 2;         // decoded (E4M3) stages
constexpr uint32_t kPackedA = BM * BKP;               // 8 KiB
constexpr uint32_t kPackedB = BN * BKP;               // 16 KiB
constexpr uint32_t kPackedStage = kPackedA + kPackedB;
constexpr uint32_t kE4A = BM * BK;                    // 16 KiB
constexpr uint32_t kE4B = BN * BK;                    // 32 KiB
constexpr uint32_t kE4Stage = kE4A + kE4B;
constexpr int kThreads = 192;
constexpr int kConvThreads = 128;
constexpr uint32_t kTmemCols = 256;
constexpr uint32_t kIdesc = idesc_e4m3_f32(BM, BN);
constexpr uint32_t kBarOffset = SE * kE4Stage + SP * kPackedStage;
constexpr size_t kSmemBytes = kBarOffset + 256 + 1024;  // + barriers + alignment slack

struct Bars {
  uint64_t p_full[SP], p_empty[SP], e_full[SE], e_empty[SE], acc_full, mma_done;
  uint32_t tmem_addr;
  int abort;
};

__device__ __forceinline__ void decode_chunk(const uint8_t* src, uint8_t* dst_row, int j, int r) {
  // 16 packed bytes = codes 32j .. 32j+31 of one row -> 32 E4M3 bytes = 16-byte chunks 2j, 2j+1
  const uint4 w = *reinterpret_cast<const uint4*>(src);
  uint4 o0, o1;
  o0.x = sm4_lo(w.x); o0.y = sm4_hi(w.x); o0.z = sm4_lo(w.y); o0.w = sm4_hi(w.y);
  o1.x = sm4_lo(w.z); o1.y = sm4_hi(w.z); o1.z = sm4_lo(w.w); o1.w = sm4_hi(w.w);
  const int sw = r & 7;  // 128B swizzle: 16-byte chunk c of row r lives at chunk c ^ (r % 8)
  *reinterpret_cast<uint4*>(dst_row + (((2 * j) ^ sw) << 4)) = o0;
  *reinterpret_cast<uint4*>(dst_row + (((2 * j + 1) ^ sw) << 4)) = o1;
}

__global__ void __launch_bounds__(kThreads, 1)
    w4a4_gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                        const float* __restrict__ sx, const float* __restrict__ sw, int n, int d_in, int d_out,
                        float* __restrict__ y, int32_t* __restrict__ acc_out, uint32_t* __restrict__ status) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* e4 = smem;                          // SE x [A 128x128 | B 256x128], swizzled
  uint8_t* pk = smem + SE * kE4Stage;          // SP x [A 128x64 | B 256x64], dense
  Bars* bars = reinterpret_cast<Bars*>(smem + kBarOffset);
  volatile int* abort_flag = &bars->abort;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int num_m = (n + BM - 1) / BM;
  const int num_n = (d_out + BN - 1) / BN;
  const int num_k = (d_in + BK - 1) / BK;
  const int num_tiles = num_m * num_n;

  if (tid == 0) {
    for (int s = 0; s < SP; ++s) {
      mbar_init(&bars->p_full[s], 1);
      mbar_init(&bars->p_empty[s], kConvThreads / 32);
    }
    for (int s = 0; s < SE; ++s) {
      mbar_init(&bars->e_full[s], kConvThreads / 32);
      mbar_init(&bars->e_empty[s], 1);
    }
    mbar_init(&bars->acc_full, 1);
    mbar_init(&bars->mma_done, 1);
    bars->abort = 0;
    fence_mbar_init();
  }
  if (warp == 1) tmem_alloc(&bars->tmem_addr, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem_addr;

  if (warp == 0) {
    // ------------------------------------------------------------------ TMA producer
    if (lane == 0) {
      prefetch_tensormap(&tmA);
      prefetch_tensormap(&tmB);
      uint32_t it = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x) {
        const int m = tile % num_m, nn = tile / num_m;
        for (int ks = 0; ks < num_k; ++ks, ++it) {
          const uint32_t s = it % SP, use = it / SP;
          if (use > 0 && !(ok = mbar_wait_bounded(&bars->p_empty[s], (use - 1) & 1, abort_flag))) break;
          uint8_t* dst = pk + s * kPackedStage;
          mbar_arrive_expect_tx(&bars->p_full[s], kPackedStage);
          tma_load_2d(dst, &tmA, ks * BKP, m * BM, &bars->p_full[s]);
          tma_load_2d(dst + kPackedA, &tmB, ks * BKP, nn * BN, &bars->p_full[s]);
        }
      }
      // Drain: every issued copy must have landed before the CTA exits.
      const uint32_t issued = it;
      const uint32_t first = issued > SP ? issued - SP : 0;
      volatile int no_abort = 0;
      for (uint32_t j = first; j < issued; ++j) mbar_wait_bounded(&bars->p_full[j % SP], (j / SP) & 1, &no_abort);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      uint32_t it = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x) {
        for (int ks = 0; ks < num_k; ++ks, ++it) {
          const uint32_t s = it % SE;
          if (!(ok = mbar_wait_bounded(&bars->e_full[s], (it / SE) & 1, abort_flag))) break;
          tc_fence_after();
          const uint64_t da = sdesc_kmajor_sw128(smem_u32(e4 + s * kE4Stage));
          const uint64_t db = sdesc_kmajor_sw128(smem_u32(e4 + s * kE4Stage + kE4A));
#pragma unroll
          for (int kk = 0; kk < BK / 32; ++kk)  // K = 32 bytes per instruction: +2 in the 16-byte address field
            mma_f8f6f4(tmem, da + 2 * kk, db + 2 * kk, kIdesc, (ks | kk) != 0);
          mma_commit(&bars->e_empty[s]);
        }
        if (ok) mma_commit(&bars->acc_full);
      }
      // All MMAs must be complete before TMEM is released.
      mma_commit(&bars->mma_done);
      volatile int no_abort = 0;
      mbar_wait_bounded(&bars->mma_done, 0, &no_abort);
    }
  } else {
    // ------------------------------------------------------------------ decode + epilogue
    const int ct = tid - 64;          // 0..127
    const int quad = warp & 3;        // TMEM lane quadrant this warp may access
    uint32_t it = 0, tcount = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x, ++tcount) {
      const int m = tile % num_m, nn = tile / num_m;
      for (int ks = 0; ks < num_k; ++ks, ++it) {
        const uint32_t ps = it % SP, es = it % SE;
        if (!(ok = mbar_wait_bounded(&bars->p_full[ps], (it / SP) & 1, abort_flag))) break;
        if (it >= SE && !(ok = mbar_wait_bounded(&bars->e_empty[es], ((it / SE) - 1) & 1, abort_flag))) break;
        const uint8_t* src = pk + ps * kPackedStage;
        uint8_t* dst = e4 + es * kE4Stage;
#pragma unroll 4
        for (int c = ct; c < (BM + BN) * 4; c += kConvThreads) {
          const int r = c >> 2, j = c & 3;  // row of the A|B stack, 16-byte packed chunk within the row
          decode_chunk(src + r * BKP + j * 16, dst + r * 128, j, r);
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(&bars->p_empty[ps]);
          mbar_arrive(&bars->e_full[es]);
        }
      }
      if (!ok) break;
      // Epilogue for this tile.
      if (!(ok = mbar_wait_bounded(&bars->acc_full, tcount & 1, abort_flag))) break;
      __syncwarp();
      tc_fence_after();
      const int t = m * BM + quad * 32 + lane;
      const bool row_ok = t < n;
      const float sxt = row_ok ? sx[t] * kAccScale : 0.f;
      const bool vec = (d_out & 3) == 0;
#pragma unroll 1
      for (int cchunk = 0; cchunk < BN / 32; ++cchunk) {
        uint32_t r[32];
        __syncwarp();
        CAT_TMEM_LD32(tmem + ((uint32_t)(quad * 32) << 16) + cchunk * 32, r);
        tmem_ld_wait();
        const int o0 = nn * BN + cchunk * 32;
        if (!row_ok || o0 >= d_out) continue;
        float* yrow = y + (size_t)t * d_out;
        if (vec && o0 + 32 <= d_out) {
#pragma unroll
          for (int i = 0; i < 32; i += 4) {
            const float4 s4 = *reinterpret_cast<const float4*>(sw + o0 + i);
            float4 v;
            v.x = __uint_as_float(r[i + 0]) * sxt * s4.x;
            v.y = __uint_as_float(r[i + 1]) * sxt * s4.y;
            v.z = __uint_as_float(r[i + 2]) * sxt * s4.z;
            v.w = __uint_as_float(r[i + 3]) * sxt * s4.w;
            *reinterpret_cast<float4*>(yrow + o0 + i) = v;
          }
        } else {
#pragma unroll
          for (int i = 0; i < 32; ++i)
            if (o0 + i < d_out) yrow[o0 + i] = __uint_as_float(r[i]) * sxt * sw[o0 + i];
        }
        if (acc_out) {
          int32_t* arow = acc_out + (size_t)t * d_out;
#pragma unroll
          for (int i = 0; i < 32; ++i)
            if (o0 + i < d_out) arow[o0 + i] = __float2int_rn(__uint_as_float(r[i]) * kAccScale);
        }
      }
      tc_fence_before();
    }
  }

  __syncthreads();
  if (bars->abort && tid == 0) report(status, kStatusTimeout);
  if (warp == 1) {
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

// 2-D byte tensor [rows][row_bytes], box [box_rows][64 bytes], no swizzle, out-of-range reads zero.
bool make_packed_map(CUtensorMap* map, const uint8_t* base, int64_t rows, int64_t row_bytes, int box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {(cuuint64_t)row_bytes, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)row_bytes};
  cuuint32_t box[2] = {(cuuint32_t)BKP, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<uint8_t*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

int num_sms() {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 148;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0) return 148;
  return sms;
}

}  // namespace

cudaError_t launch_w4a4_gemm_tc(const uint8_t* xq, const float* sx, const uint8_t* wq, const float* sw, int64_t n,
                                int64_t d_in, int64_t d_out, float* y, int32_t* acc_out, uint32_t* status,
                                cudaStream_t stream) {
  CUtensorMap ta, tb;
  if (!make_packed_map(&ta, xq, n, d_in / 2, BM) || !make_packed_map(&tb, wq, d_out, d_in / 2, BN))
    return cudaErrorInvalidValue;
  static std::once_flag attr_once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(attr_once, [] {
    attr_err = cudaFuncSetAttribute(w4a4_gemm_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
  });
  if (attr_err != cudaSuccess) return attr_err;
  const int64_t tiles = ((n + BM - 1) / BM) * ((d_out + BN - 1) / BN);
  const int grid = (int)(tiles < num_sms() ? tiles : num_sms());
  w4a4_gemm_tc_kernel<<<grid, kThreads, kSmemBytes, stream>>>(ta, tb, sx, sw, (int)n, (int)d_in, (int)d_out, y,
                                                              acc_out, status);
  return cudaGetLastError();
}

}  // namespace cat
