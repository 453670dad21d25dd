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
// Shared-memory bandwidth is the budget that matters: decoding on the way into the tensor cores
// costs a write per operand byte.  So the token operand A never touches shared memory -- each
// decode thread owns one token row, loads its packed bytes straight from global memory, decodes
// them in registers and writes the E4M3 row into tensor memory (tcgen05.st), from where the MMA
// reads A -- and only the weight operand B is decoded into 128B-swizzled shared memory.
//
// Persistent CTA (one per SM, 512 threads), output tile 128 tokens x 256 channels, K step 128:
//   warp 0       TMEM allocator; lane 0 issues tcgen05.mma (4 x K=32 per K step) and commits
//   warps 4..7   epilogue: tcgen05.ld of their TMEM lane quadrant, scale, stage the rows in
//                128B-swizzled shared memory, TMA store (plain stores when the TMA rules don't hold)
//   warps 8..15  decode: prefetch packed A rows and B chunks two K steps ahead into registers
//                (three rotating buffers);
//                A -> TMEM stage, B -> shared-memory stage (4-stage ring)
// TMEM: accumulator columns [0, 256), A stages at 256 + 32 s.  Every mbarrier wait is bounded;
// a wait that gives up raises the device status word and all roles drain and exit.
#include <cstring>
#include <mutex>

#include "common.cuh"

namespace cat {
namespace {

constexpr int BM = 128, BN = 256, BK = 128;
constexpr int BKP = BK / 2;                 // packed bytes per row per K step
constexpr int SE = 4;                       // decoded stages (A in TMEM, B in shared memory)
constexpr uint32_t kStageB = BN * BK;       // 32 KiB of E4M3 per stage
constexpr int kThreads = 512;
constexpr int kDecWarp0 = 8, kDecWarps = 8, kDecThreads = kDecWarps * 32;
constexpr int kEpiWarp0 = 4, kEpiWarps = 4;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kAccCols = 256;
constexpr uint32_t kIdesc = idesc_e4m3_f32(BM, BN);
constexpr uint32_t kEpiStage = 32 * 32 * 4;                 // 32 rows x 32 fp32 columns, 4 KiB
constexpr int kEpiBufs = 4;                                  // TMA-store staging buffers per epilogue warp
constexpr uint32_t kEpiOffset = SE * kStageB;                // after the B stages
constexpr uint32_t kScaleOffset = kEpiOffset + kEpiWarps * kEpiBufs * kEpiStage;
constexpr uint32_t kBarOffset = kScaleOffset + kEpiWarps * BN * 4;
constexpr size_t kSmemBytes = kBarOffset + 256 + 1024;      // + barriers + alignment slack

struct Bars {
  uint64_t full[SE], empty[SE], acc_full, acc_empty, mma_done;
  uint32_t tmem_addr;
  int abort;
};

// ---- tensor-memory stores and the TMA store path -------------------------------------------
#define CAT_TMEM_ST16(taddr, v)                                                                              \
  asm volatile("tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15," \
               "%16};" ::"r"(taddr),                                                                         \
               "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]),   \
               "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15])                  \
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
__device__ __forceinline__ void bulk_wait_read_le3() { asm volatile("cp.async.bulk.wait_group.read 3;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// Predicated 128-bit load into a zeroed destination: nothing depends on the loaded value until
// it is consumed, so a prefetch issued here does not wait for its data.
__device__ __forceinline__ void ldg_nc_pred(uint4& v, const uint8_t* p, bool pred) {
  asm volatile(
      "{ .reg .pred q; setp.ne.b32 q, %4, 0; mov.b32 %0, 0; mov.b32 %1, 0; mov.b32 %2, 0; mov.b32 %3, 0;\n"
      "  @q ld.global.nc.v4.u32 {%0,%1,%2,%3}, [%5]; }"
      : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
      : "r"((int)pred), "l"(p));
}

// Packed inputs of one K step for one decode thread: its A row half (2 x 16 B) and 4 B chunks.
struct StepRegs {
  uint4 a[2];
  uint4 b[4];
};

struct DecodeCtx {
  const uint8_t* xq;
  const uint8_t* wq;
  int64_t row_bytes;
  int a_row;        // token row (global), this thread's TMEM lane
  int a_half;       // which 32-byte half of the K step's 64 packed bytes
  int n, d_out;
  int b_row[4];     // B rows (within the tile) of this thread's 4 chunks
  int b_chunk[4];   // 16-byte chunk (0..3) within the row's 64 bytes
};

__device__ __forceinline__ void load_step(const DecodeCtx& c, int m0, int n0, int ks, StepRegs& r) {
  const int64_t kb = (int64_t)ks * BKP;
  const int t = m0 + c.a_row;
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int64_t off = kb + c.a_half * 32 + h * 16;
    const bool in = t < c.n && off < c.row_bytes;
    ldg_nc_pred(r.a[h], c.xq + (in ? (int64_t)t * c.row_bytes + off : 0), in);
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int o = n0 + c.b_row[i];
    const int64_t off = kb + c.b_chunk[i] * 16;
    const bool in = o < c.d_out && off < c.row_bytes;
    ldg_nc_pred(r.b[i], c.wq + (in ? (int64_t)o * c.row_bytes + off : 0), in);
  }
}

__global__ void __launch_bounds__(kThreads, 1)
    w4a4_gemm_tc_kernel(const __grid_constant__ CUtensorMap tmY, const uint8_t* __restrict__ xq,
                        const uint8_t* __restrict__ wq, const float* __restrict__ sx, const float* __restrict__ sw,
                        int n, int d_in, int d_out, float* __restrict__ y, int32_t* __restrict__ acc_out,
                        int use_tma_store, uint32_t* __restrict__ status) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* bst = smem;                         // SE x [256 rows x 128 B], 128B-swizzled
  uint8_t* epi = smem + kEpiOffset;            // 4 warps x 4 x [32 rows x 128 B], 128B-swizzled
  float* scl = reinterpret_cast<float*>(smem + kScaleOffset);  // 4 warps x 256 output-channel steps
  Bars* bars = reinterpret_cast<Bars*>(smem + kBarOffset);
  volatile int* abort_flag = &bars->abort;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int num_m = (n + BM - 1) / BM;
  const int num_n = (d_out + BN - 1) / BN;
  const int num_k = (d_in + BK - 1) / BK;
  const int num_tiles = num_m * num_n;

  if (tid == 0) {
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
          if (lane == 0) bulk_wait_read_le3();  // the store issued kEpiBufs chunks ago has read this buffer
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
    const int quad = warp & 3;
    DecodeCtx c;
    c.xq = xq;
    c.wq = wq;
    c.row_bytes = d_in / 2;
    c.a_row = quad * 32 + lane;
    c.a_half = (warp - kDecWarp0) >> 2;           // warps 8..11 first half, 12..15 second half
    c.n = n;
    c.d_out = d_out;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int id = dt + kDecThreads * i;         // 1024 chunks = 256 rows x 4
      c.b_row[i] = id >> 2;
      c.b_chunk[i] = id & 3;
    }
    // The CTA's (tile, ks) sequence with register prefetch two steps ahead: three buffers, each
    // loaded and then consumed two steps later (no register copies of loads in flight).
    auto advance = [&](int& tl, int& k) {
      if (++k == num_k) {
        k = 0;
        tl += gridDim.x;
      }
    };
    auto load = [&](int tl, int k, StepRegs& r) {
      if (tl < num_tiles) load_step(c, (tl % num_m) * BM, (tl / num_m) * BN, k, r);
    };
    uint32_t it = 0;
    bool ok = true;
    auto process = [&](const StepRegs& r) {
      const uint32_t s = it % SE;
      if (it >= SE && !(ok = mbar_wait_bounded(&bars->empty[s], ((it / SE) - 1) & 1, abort_flag))) return;
      tc_fence_after();
      // A: this thread's token row, 32 packed bytes -> 64 E4M3 bytes = 16 TMEM columns
      uint32_t av[16];
      const uint32_t aw[8] = {r.a[0].x, r.a[0].y, r.a[0].z, r.a[0].w, r.a[1].x, r.a[1].y, r.a[1].z, r.a[1].w};
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        av[2 * u] = sm4_lo(aw[u]);
        av[2 * u + 1] = sm4_hi(aw[u]);
      }
      __syncwarp();
      CAT_TMEM_ST16(tmem + ((uint32_t)(quad * 32) << 16) + kAccCols + 32u * s + 16u * c.a_half, av);
      // B: 4 chunks of 16 packed bytes -> 2 x 16 E4M3 bytes each, 128B-swizzled rows
      uint8_t* bs = bst + s * kStageB;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const uint4 w = r.b[i];
        const int row = c.b_row[i], j = c.b_chunk[i], swz = row & 7;
        uint8_t* dst = bs + row * 128;
        *reinterpret_cast<uint4*>(dst + (((2 * j) ^ swz) << 4)) =
            make_uint4(sm4_lo(w.x), sm4_hi(w.x), sm4_lo(w.y), sm4_hi(w.y));
        *reinterpret_cast<uint4*>(dst + (((2 * j + 1) ^ swz) << 4)) =
            make_uint4(sm4_lo(w.z), sm4_hi(w.z), sm4_lo(w.w), sm4_hi(w.w));
      }
      tmem_st_wait();
      fence_proxy_async_smem();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars->full[s]);
      ++it;
    };
    StepRegs ra, rb, rc;
    int tA = blockIdx.x, kA = 0;
    int tB = tA, kB = kA;
    advance(tB, kB);
    int tC = tB, kC = kB;
    advance(tC, kC);
    load(tA, kA, ra);
    load(tB, kB, rb);
    while (ok) {
      if (tA >= num_tiles) break;
      load(tC, kC, rc);
      process(ra);
      tA = tC, kA = kC;
      advance(tA, kA);
      if (!ok || tB >= num_tiles) break;
      load(tA, kA, ra);
      process(rb);
      tB = tA, kB = kA;
      advance(tB, kB);
      if (!ok || tC >= num_tiles) break;
      load(tB, kB, rb);
      process(rc);
      tC = tB, kC = kB;
      advance(tC, kC);
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
  CUtensorMap ty;
  memset(&ty, 0, sizeof(ty));
  int use_tma = (d_out % 4 == 0) ? 1 : 0;
  if (use_tma && !make_output_map(&ty, y, n, d_out)) use_tma = 0;
  static std::once_flag attr_once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(attr_once, [] {
    attr_err = cudaFuncSetAttribute(w4a4_gemm_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
  });
  if (attr_err != cudaSuccess) return attr_err;
  const int64_t tiles = ((n + BM - 1) / BM) * ((d_out + BN - 1) / BN);
  const int grid = (int)(tiles < num_sms() ? tiles : num_sms());
  w4a4_gemm_tc_kernel<<<grid, kThreads, kSmemBytes, stream>>>(ty, xq, wq, sx, sw, (int)n, (int)d_in, (int)d_out, y,
                                                              acc_out, use_tma, status);
  return cudaGetLastError();
}

}  // namespace cat
