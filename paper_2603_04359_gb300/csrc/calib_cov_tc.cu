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
// CTA = (channel group, token split).  The token splits of a group form a thread-block cluster of
// S <= 4 CTAs: each CTA sums its accumulators into an fp32 tile in its own shared memory, and after
// a cluster barrier CTA r reduces rows [r 128/S, (r+1) 128/S) of the S tiles through distributed
// shared memory and writes them as coalesced float64 rows.  More splits than one cluster (large
// token counts) add their clusters' results with float64 atomics.  Since D = X^T X is symmetric,
// the staged tile is the transpose of the TMEM tile (thread = TMEM row writes one shared-memory
// column, so the stores are conflict-free) and the written blocks are D^T, equal to D up to the
// rounding of the accumulation order.
// Warps: 0 TMA producer + TMEM allocator, 1 MMA issuer, 2..5 epilogue (one TMEM lane quadrant
// each).  Tokens arrive in 64-row chunks of 64-channel, 128B-swizzled boxes through a 4-stage ring.
#include <cstring>
#include <mutex>

#include "common.cuh"

namespace cat {
namespace {

constexpr int kChunk = 64;      // tokens per stage
constexpr int kStages = 4;
constexpr int kThreads = 192;
constexpr uint32_t kBox = kChunk * 128;  // one 64-token x 64-channel bf16 box, 8 KiB
constexpr int kMaxCluster = 4;           // token splits reduced on chip
constexpr uint32_t kRedTile = 128 * 128 * 4;  // fp32 128 x 128 reduction tile (reuses the stage ring)
static_assert(kStages * 2 * kBox >= kRedTile, "the reduction tile must fit in the stage ring");

template <int G2>  // 128-channel tiles per dimension of a group (1: k <= 128, 2: k = 256)
struct CovCfg {
  static constexpr int G = 128 * G2;
  static constexpr int BOXES = G / 64;
  static constexpr uint32_t STAGE = BOXES * kBox;
  static constexpr uint32_t BAR_OFF = kStages * STAGE;
  // more than half of an SM's shared memory: one CTA per SM, so that a CTA waiting at a cluster
  // barrier never holds tensor memory that a CTA of another cluster on the same SM is waiting for
  static constexpr size_t SMEM = (BAR_OFF + 256 + 1024) > 120 * 1024 ? (BAR_OFF + 256 + 1024) : 120 * 1024;
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

__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_nctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(r));
  return r;
}
// all threads of all CTAs of the cluster; release / acquire orders the shared-memory tiles
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ uint32_t map_cluster(uint32_t saddr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
  return r;
}
__device__ __forceinline__ float4 ld_cluster_f32x4(uint32_t caddr) {
  float4 v;
  asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(caddr)
               : "memory");
  return v;
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
  pdl_wait_then_release();                        // nothing global or in tensor memory before this
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
        if (c >= kStages && !(ok = mbar_wait_bounded(&bars->empty[s], ((c / kStages) - 1) & 1, abort_flag, __LINE__))) break;
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
        if (!(ok = mbar_wait_bounded(&bars->full[s], (c / kStages) & 1, abort_flag, __LINE__))) break;
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
  }

  // ---- reduction over the cluster's token splits and the float64 store ---------------------
  __syncthreads();
  const bool epi = warp >= 2;
  const int ew = warp - 2;                            // epilogue warp 0..3
  const int quad = warp & 3;                          // the TMEM lane quadrant this warp may access
  const uint32_t S = cluster_nctarank();
  const uint32_t rank = cluster_ctarank();
  const bool have_acc = chunks > 0 && !bars->abort;
  if (epi && have_acc) {
    if (!mbar_wait_bounded(&bars->acc_full, 0, abort_flag, __LINE__)) {
      // gave up: the tile below is not written; the status word reports it
    }
    __syncwarp();
    tc_fence_after();
  }
  float* red = reinterpret_cast<float*>(smem);        // the stage ring is idle once acc_full fired
  const int used = total_steps < C::NACC ? total_steps : C::NACC;  // accumulators written
  const int kw = G2 == 2 ? 128 : k;                   // needed columns per row within a tile
#pragma unroll 1
  for (int ih = 0; ih < G2; ++ih)
#pragma unroll 1
    for (int jh = 0; jh < G2; ++jh) {
      if (epi) {
        // phase 1: this CTA's partial tile, summed over its accumulators, stored transposed
        const int r = quad * 32 + lane;               // TMEM lane = tile row
        const int cw = kw < 32 ? 32 : kw;             // columns a warp's 32 rows need
        const int col0 = G2 == 2 ? 0 : ((quad * 32) / cw) * cw;
        const bool live = have_acc && !__any_sync(0xFFFFFFFFu, *abort_flag);  // warp-uniform
#pragma unroll 1
        for (int cc = 0; cc < cw / 32; ++cc) {
          const int col = col0 + 32 * cc;
          float v32[32];
#pragma unroll
          for (int e = 0; e < 32; ++e) v32[e] = 0.f;
          if (live) {
#pragma unroll 1
            for (int a = 0; a < used; a += 2) {      // two accumulators per tensor-memory round trip
              uint32_t rr[32], rq[32];
              __syncwarp();
              CAT_TMEM_LD32(tmem + ((uint32_t)(quad * 32) << 16) + ((a * G2 + ih) * G2 + jh) * 128 + col, rr);
              if (a + 1 < used)
                CAT_TMEM_LD32(tmem + ((uint32_t)(quad * 32) << 16) + (((a + 1) * G2 + ih) * G2 + jh) * 128 + col, rq);
              tmem_ld_wait();
#pragma unroll
              for (int e = 0; e < 32; ++e) v32[e] += __uint_as_float(rr[e]);
              if (a + 1 < used) {
#pragma unroll
                for (int e = 0; e < 32; ++e) v32[e] += __uint_as_float(rq[e]);
              }
            }
          }
#pragma unroll
          for (int e = 0; e < 32; ++e) red[(col + e) * 128 + r] = v32[e];
        }
      }
      __syncwarp();
      tc_fence_before();
      cluster_sync_all();                             // every CTA's tile is written
      if (epi) {
        // phase 2: rows [rank 128/S, (rank+1) 128/S) of the S tiles; lanes_per_row lanes cover a
        // row's kw needed columns 4 at a time
        const int rows = 128 / (int)S;
        const int r_lo = (int)rank * rows;
        const int lpr = kw / 4 < 32 ? kw / 4 : 32;
        const int rpp = 32 / lpr;                     // rows per warp pass
        const int sub = lane / lpr, l4 = lane % lpr;
        const uint32_t red_addr = smem_u32(red);
        // kRowsInFlight rows per round: all their remote loads (S per row and 4-column group) are in
        // flight before the first sum (remote shared-memory loads are slow); the sums run in a fixed
        // source order, so they are deterministic
        constexpr int kRowsInFlight = 4;
#pragma unroll 1
        for (int R0 = r_lo + ew * rpp + sub; R0 < r_lo + rows; R0 += kRowsInFlight * 4 * rpp) {
#pragma unroll 1
          for (int C4i = 4 * l4; C4i < kw; C4i += 4 * lpr) {
            float4 part[kRowsInFlight][kMaxCluster];
#pragma unroll
            for (int q = 0; q < kRowsInFlight; ++q) {
              const int R = R0 + q * 4 * rpp;
              const int cb = G2 == 2 ? 0 : (R / k) * k;   // first column of R's diagonal block in the tile
              const uint32_t off = red_addr + (uint32_t)(R * 128 + cb + C4i) * 4u;
#pragma unroll
              for (int src = 0; src < kMaxCluster; ++src)
                part[q][src] = (R < r_lo + rows && (uint32_t)src < S) ? ld_cluster_f32x4(map_cluster(off, (uint32_t)src))
                                                                       : make_float4(0.f, 0.f, 0.f, 0.f);
            }
#pragma unroll
            for (int q = 0; q < kRowsInFlight; ++q) {
              const int R = R0 + q * 4 * rpp;
              if (R >= r_lo + rows) break;
              const int cb = G2 == 2 ? 0 : (R / k) * k;
              const int C4 = cb + C4i;
              float4 acc = part[q][0];
#pragma unroll
              for (int src = 1; src < kMaxCluster; ++src)
                if ((uint32_t)src < S) {
                  acc.x += part[q][src].x; acc.y += part[q][src].y; acc.z += part[q][src].z; acc.w += part[q][src].w;
                }
              // staged tile (ih, jh) is transposed: entry (R, C) belongs to group row jh*128 + R
              const int grow = c0 + jh * 128 + R;
              if (grow >= d) continue;
              double* dst = sigma + (int64_t)grow * k + ((ih * 128 + C4) % k);
              const double v[4] = {f32_to_f64_exact(acc.x), f32_to_f64_exact(acc.y), f32_to_f64_exact(acc.z),
                                   f32_to_f64_exact(acc.w)};
              if (mode == 2) {
#pragma unroll
                for (int e = 0; e < 4; ++e) atomicAdd(dst + e, v[e]);
              } else if (mode == 1) {
#pragma unroll
                for (int e = 0; e < 4; ++e) dst[e] += v[e];
              } else {
                reinterpret_cast<double2*>(dst)[0] = make_double2(v[0], v[1]);
                reinterpret_cast<double2*>(dst)[1] = make_double2(v[2], v[3]);
              }
            }
          }
        }
      }
      __syncwarp();
      cluster_sync_all();                             // the tiles may be overwritten / released
    }

  if (bars->abort && tid == 0) report(status, timeout_bits(kWhereCalib, bars->abort));
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
  const int sms = num_sms();
  // S token splits per group reduced on chip (a cluster), while the grid stays within one wave
  int S = 1;
  while (S < kMaxCluster && groups * S * 2 <= sms && chunks >= S * 2) S *= 2;
  // more clusters per group (float64 atomics) only for long calibration runs: >= 2048 tokens per CTA
  const int64_t per_cta = (chunks + S - 1) / S;
  int64_t ysplits = (sms + groups * S - 1) / (groups * S);
  if (ysplits > per_cta / 32) ysplits = per_cta / 32;
  if (ysplits < 1) ysplits = 1;
  const int64_t tps = ((chunks + S * ysplits - 1) / (S * ysplits)) * kChunk;
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
  cfg.gridDim = dim3((unsigned)groups, (unsigned)(S * ysplits), 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = C::SMEM;
  cfg.stream = stream;
  // not a programmatic dependent launch: measured, one gained ~0.4 us per c4 step and lost ~0.7 us per
  // c2 step (the kernel still releases its dependents early)
  cudaLaunchAttribute attr_cluster[1];
  attr_cluster[0].id = cudaLaunchAttributeClusterDimension;
  attr_cluster[0].val.clusterDim.x = 1;
  attr_cluster[0].val.clusterDim.y = (unsigned)S;
  attr_cluster[0].val.clusterDim.z = 1;
  cfg.attrs = attr_cluster;
  cfg.numAttrs = 1;
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
