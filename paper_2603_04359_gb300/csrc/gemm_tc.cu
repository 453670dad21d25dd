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
// Data path.  The tensor cores read their shared-memory operands on a path of their own (their
// rate does not change under concurrent LSU shared-memory traffic), an MMA with A in tensor memory
// runs at ~93% of peak, and shared-memory stores top out near 100 B/clk/SM.  So:
//   * packed A (128 x 64 B) and B (256 x 64 B) tiles arrive by TMA with a 64-byte swizzle, which
//     makes one-row-per-thread 16-byte shared loads conflict-free;
//   * A is decoded one row per thread and written to tensor memory (tcgen05.st), never to
//     shared memory; the MMA reads A from tensor memory;
//   * only B is decoded into 128B-swizzled shared memory (32 KiB of stores per K step).
//
// Persistent CTA (one per SM, 512 threads), output tile 128 tokens x 256 channels, K step 128:
//   warp 0       TMA producer (packed ring) and TMEM allocator
//   warp 1       lane 0 issues tcgen05.mma (4 x K=32 per K step) and commits
//   warps 4..7   epilogue: tcgen05.ld of their TMEM lane quadrant, scale, stage the rows in
//                128B-swizzled shared memory, TMA store (plain stores when the TMA rules don't hold)
//   warps 8..15  decode: B chunks (all 8 warps) and A rows (warps 8..11, one TMEM quadrant each)
// TMEM: accumulator columns [0, 256), A stages at 256 + 32 s.  Every mbarrier wait is bounded;
// a wait that gives up raises the device status word and all roles drain and exit.
#include <cstring>
#include <mutex>

#include "common.cuh"

namespace cat {
namespace {

constexpr int BM = 128, BN = 256, BK = 128;
constexpr int BKP = BK / 2;                 // packed bytes per row per K step
constexpr int SP = 3;                       // packed stages (TMA)
constexpr int SE = 3;                       // decoded stages (A in TMEM, B in shared memory)
constexpr uint32_t kPackedA = BM * BKP;     // 8 KiB
constexpr uint32_t kPackedB = BN * BKP;     // 16 KiB
constexpr uint32_t kPackedStage = kPackedA + kPackedB;
constexpr uint32_t kStageB = BN * BK;       // 32 KiB of E4M3 per stage
constexpr int kThreads = 512;
constexpr int kDecWarp0 = 8, kDecWarps = 8, kDecThreads = kDecWarps * 32;
constexpr int kEpiWarp0 = 4, kEpiWarps = 4;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kAccCols = 256;
constexpr uint32_t kIdesc = idesc_e4m3_f32(BM, BN);
constexpr uint32_t kEpiStage = 32 * 32 * 4;                 // 32 rows x 32 fp32 columns, 4 KiB
constexpr int kEpiBufs = 2;                                  // TMA-store staging buffers per epilogue warp
constexpr uint32_t kPkOffset = SE * kStageB;                 // after the decoded B stages
constexpr uint32_t kEpiOffset = kPkOffset + SP * kPackedStage;
constexpr uint32_t kScaleOffset = kEpiOffset + kEpiWarps * kEpiBufs * kEpiStage;
constexpr uint32_t kBarOffset = kScaleOffset + kEpiWarps * BN * 4;
constexpr size_t kSmemBytes = kBarOffset + 256 + 1024;      // + barriers + alignment slack

struct Bars {
  uint64_t p_full[SP], p_empty[SP], full[SE], empty[SE], acc_full, acc_empty, mma_done;
  uint32_t tmem_addr;
  int abort;
};

// ---- tensor-memory stores and the TMA store path -------------------------------------------
#define CAT_TMEM_ST32(taddr, v)                                                                                 \
  asm volatile("tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16," \
               "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),                   \
               "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]),      \
               "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15]), "r"(v[16]),          \
               "r"(v[17]), "r"(v[18]), "r"(v[19]), "r"(v[20]), "r"(v[21]), "r"(v[22]), "r"(v[23]), "r"(v[24]),         \
               "r"(v[25]), "r"(v[26]), "r"(v[27]), "r"(v[28]), "r"(v[29]), "r"(v[30]), "r"(v[31])                     \
               : "memory")

__device__ __forceinline__ void tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

__device__ __forceinline__ void mma_f8f6f4_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                              uint32_t accumulate) {
  asm volatile(
      "{ .reg .pred p; setp.ne.b32 p, %4, 0; "
      "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], [%1], %2, %3, p; }" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, const void* smem_src, int32_t x, int32_t y) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(x), "r"(y), "r"(smem_u32(smem_src))
               : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read_le1() { asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// 64-byte swizzle of the packed TMA tiles: 16-byte chunk j of 64-byte row r sits at chunk
// j ^ ((r >> 1) & 3), so 8 consecutive rows read at the same j touch 8 distinct bank groups.
__device__ __forceinline__ uint32_t sw64_off(int r, int j) { return r * 64 + ((j ^ ((r >> 1) & 3)) << 4); }

__global__ void __launch_bounds__(kThreads, 1)
    w4a4_gemm_tc_kernel(const __grid_constant__ CUtensorMap tmY, const __grid_constant__ CUtensorMap tmA,
                        const __grid_constant__ CUtensorMap tmB, const float* __restrict__ sx,
                        const float* __restrict__ sw, int n, int d_in, int d_out, float* __restrict__ y,
                        int32_t* __restrict__ acc_out, int use_tma_store, uint32_t* __restrict__ status) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* bst = smem;                         // SE x [256 rows x 128 B] E4M3, 128B-swizzled
  uint8_t* pk = smem + kPkOffset;              // SP x [A 128 x 64 B | B 256 x 64 B] packed, 64B-swizzled
  uint8_t* epi = smem + kEpiOffset;            // 4 warps x 2 x [32 rows x 128 B], 128B-swizzled
  float* scl = reinterpret_cast<float*>(smem + kScaleOffset);  // 4 warps x 256 output-channel steps
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
      mbar_init(&bars->p_empty[s], kDecWarps);
    }
    for (int s = 0; s < SE; ++s) {
      mbar_init(&bars->full[s], kDecWarps);
      mbar_init(&bars->empty[s], 1);
    }
    mbar_init(&bars->acc_full, 1);
    mbar_init(&bars->acc_empty, kEpiWarps);
    mbar_init(&bars->mma_done, 1);
    bars->abort = 0;
    fence_mbar_init();
  }
  __syncwarp();
  if (warp == 0) tmem_alloc(&bars->tmem_addr, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem_addr;

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
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
      const uint32_t issued = it, first = issued > SP ? issued - SP : 0;
      volatile int no_abort = 0;
      for (uint32_t j = first; j < issued; ++j) mbar_wait_bounded(&bars->p_full[j % SP], (j / SP) & 1, &no_abort);
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      uint32_t it = 0, tcount = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x, ++tcount) {
        // the epilogue must have drained the accumulator of the previous tile
        if (tcount > 0 && !(ok = mbar_wait_bounded(&bars->acc_empty, (tcount - 1) & 1, abort_flag))) break;
        tc_fence_after();
        for (int ks = 0; ks < num_k; ++ks, ++it) {
          const uint32_t s = it % SE;
          if (!(ok = mbar_wait_bounded(&bars->full[s], (it / SE) & 1, abort_flag))) break;
          tc_fence_after();
          const uint64_t db = sdesc_kmajor_sw128(smem_u32(bst + s * kStageB));
          const uint32_t ta = tmem + kAccCols + 32u * s;
#pragma unroll
          for (int kk = 0; kk < BK / 32; ++kk)  // K = 32 bytes per MMA: 8 TMEM columns of A, +2 in B's address field
            mma_f8f6f4_ts(tmem, ta + 8u * kk, db + 2 * kk, kIdesc, (ks | kk) != 0);
          mma_commit(&bars->empty[s]);
        }
        if (ok) mma_commit(&bars->acc_full);
      }
      mma_commit(&bars->mma_done);  // all MMAs complete before TMEM is released
      volatile int no_abort = 0;
      mbar_wait_bounded(&bars->mma_done, 0, &no_abort);
    }
  } else if (warp >= kEpiWarp0 && warp < kEpiWarp0 + kEpiWarps) {
    // ---------------------------------------------------------------- epilogue
    const int quad = warp & 3;
    uint8_t* stage0 = epi + (warp - kEpiWarp0) * kEpiBufs * kEpiStage;
    float* wsc = scl + (warp - kEpiWarp0) * BN;
    uint32_t tcount = 0, nstore = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x, ++tcount) {
      const int m = tile % num_m, nn = tile / num_m;
      const int row0 = m * BM + quad * 32;
      const int t = row0 + lane;
      const float sxt = (t < n) ? sx[t] * kAccScale : 0.f;
      __syncwarp();
#pragma unroll
      for (int i = 0; i < BN / 32; ++i) {  // this tile's output-channel steps, staged once per tile
        const int o = nn * BN + 32 * i + lane;
        wsc[32 * i + lane] = (o < d_out) ? sw[o] : 0.f;
      }
      __syncwarp();
      if (!(ok = mbar_wait_bounded(&bars->acc_full, tcount & 1, abort_flag))) break;
      __syncwarp();
      tc_fence_after();
#pragma unroll 1
      for (int c = 0; c < BN / 32; ++c) {
        uint32_t r[32];
        __syncwarp();
        CAT_TMEM_LD32(tmem + ((uint32_t)(quad * 32) << 16) + c * 32, r);
        tmem_ld_wait();
        if (c == BN / 32 - 1) {  // accumulator fully read: let the next tile's MMAs start
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&bars->acc_empty);
        }
        const int o0 = nn * BN + c * 32;
        if (o0 >= d_out || row0 >= n) continue;  // warp-uniform: nothing of this chunk is in range
        if (use_tma_store) {
          uint8_t* buf = stage0 + (nstore % kEpiBufs) * kEpiStage;
          if (lane == 0) bulk_wait_read_le1();  // the store issued two chunks ago has read this buffer
          __syncwarp();
#pragma unroll
          for (int q = 0; q < 8; ++q) {  // row `lane`, 16-byte chunk q at q ^ (lane % 8)
            const float4 s4 = *reinterpret_cast<const float4*>(wsc + c * 32 + 4 * q);
            *reinterpret_cast<float4*>(buf + lane * 128 + ((q ^ (lane & 7)) << 4)) =
                make_float4(__uint_as_float(r[4 * q]) * sxt * s4.x, __uint_as_float(r[4 * q + 1]) * sxt * s4.y,
                            __uint_as_float(r[4 * q + 2]) * sxt * s4.z, __uint_as_float(r[4 * q + 3]) * sxt * s4.w);
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            tma_store_2d(&tmY, buf, o0, row0);
            bulk_commit();
          }
          ++nstore;
        } else if (t < n) {
          float* yrow = y + (size_t)t * d_out;
#pragma unroll
          for (int i = 0; i < 32; ++i)
            if (o0 + i < d_out) yrow[o0 + i] = __uint_as_float(r[i]) * sxt * wsc[c * 32 + i];
        }
        if (acc_out && t < n) {
          int32_t* arow = acc_out + (size_t)t * d_out;
#pragma unroll
          for (int i = 0; i < 32; ++i)
            if (o0 + i < d_out) arow[o0 + i] = __float2int_rn(__uint_as_float(r[i]) * kAccScale);
        }
      }
    }
    if (lane == 0) bulk_wait_all();
    __syncwarp();
  } else if (warp >= kDecWarp0) {
    // ---------------------------------------------------------------- decode
    const int dt = tid - kDecWarp0 * 32;          // 0..255
    const bool a_warp = warp < kDecWarp0 + 4;     // warps 8..11 also decode A rows
    const int quad = warp & 3;
    const int a_row = quad * 32 + lane;           // this thread's A row = TMEM lane
    uint32_t it = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x) {
      for (int ks = 0; ks < num_k; ++ks, ++it) {
        const uint32_t ps = it % SP, s = it % SE;
        if (!(ok = mbar_wait_bounded(&bars->p_full[ps], (it / SP) & 1, abort_flag))) break;
        if (it >= SE && !(ok = mbar_wait_bounded(&bars->empty[s], ((it / SE) - 1) & 1, abort_flag))) break;
        tc_fence_after();
        const uint8_t* pa = pk + ps * kPackedStage;
        const uint8_t* pb = pa + kPackedA;
        if (a_warp) {  // A: one 64-byte row per thread -> 128 E4M3 bytes = 32 TMEM columns
          uint32_t av[32];
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const uint4 w = *reinterpret_cast<const uint4*>(pa + sw64_off(a_row, j));
            av[8 * j + 0] = sm4_lo(w.x); av[8 * j + 1] = sm4_hi(w.x);
            av[8 * j + 2] = sm4_lo(w.y); av[8 * j + 3] = sm4_hi(w.y);
            av[8 * j + 4] = sm4_lo(w.z); av[8 * j + 5] = sm4_hi(w.z);
            av[8 * j + 6] = sm4_lo(w.w); av[8 * j + 7] = sm4_hi(w.w);
          }
          __syncwarp();
          CAT_TMEM_ST32(tmem + ((uint32_t)(quad * 32) << 16) + kAccCols + 32u * s, av);
        }
        // B: 1024 chunks of 16 packed bytes (256 rows x 4), 4 per thread, consecutive per warp
        uint8_t* bs = bst + s * kStageB;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int id = dt + kDecThreads * i;
          const int row = id >> 2, j = id & 3, swz = row & 7;
          const uint4 w = *reinterpret_cast<const uint4*>(pb + sw64_off(row, j));
          uint8_t* dst = bs + row * 128;
          *reinterpret_cast<uint4*>(dst + (((2 * j) ^ swz) << 4)) =
              make_uint4(sm4_lo(w.x), sm4_hi(w.x), sm4_lo(w.y), sm4_hi(w.y));
          *reinterpret_cast<uint4*>(dst + (((2 * j + 1) ^ swz) << 4)) =
              make_uint4(sm4_lo(w.z), sm4_hi(w.z), sm4_lo(w.w), sm4_hi(w.w));
        }
        if (a_warp) tmem_st_wait();
        fence_proxy_async_smem();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(&bars->p_empty[ps]);
          mbar_arrive(&bars->full[s]);
        }
      }
    }
  }

  __syncthreads();
  if (bars->abort && tid == 0) report(status, kStatusTimeout);
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

// y [n][d_out] fp32, box 32 x 32, 128-byte swizzle (matches the epilogue staging layout).
bool make_output_map(CUtensorMap* map, float* y, int64_t n, int64_t d_out) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {(cuuint64_t)d_out, (cuuint64_t)n};
  cuuint64_t strides[1] = {(cuuint64_t)d_out * sizeof(float)};
  cuuint32_t box[2] = {32, 32};
  cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, y, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
            CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
         CUDA_SUCCESS;
}

// Packed codes [rows][row_bytes], box [box_rows][64 bytes], 64-byte swizzle, out-of-range reads zero.
bool make_packed_map(CUtensorMap* map, const uint8_t* base, int64_t rows, int64_t row_bytes, int box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {(cuuint64_t)row_bytes, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)row_bytes};
  cuuint32_t box[2] = {(cuuint32_t)BKP, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<uint8_t*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
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
  CUtensorMap ty, ta, tb;
  memset(&ty, 0, sizeof(ty));
  int use_tma = (d_out % 4 == 0) ? 1 : 0;
  if (use_tma && !make_output_map(&ty, y, n, d_out)) use_tma = 0;
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
  note_launch();
  w4a4_gemm_tc_kernel<<<grid, kThreads, kSmemBytes, stream>>>(ty, ta, tb, sx, sw, (int)n, (int)d_in, (int)d_out, y,
                                                              acc_out, use_tma, status);
  return cudaGetLastError();
}

}  // namespace cat
