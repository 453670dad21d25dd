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
//   pass 1: recompute, q = clamp(round_half_even(7 v' / max), -7, 7) decided exactly, pack SM4x8, store.
// Warps: 0 TMA producer + TMEM allocator, 1 MMA issuer, 4..7 epilogue, 8..15 converters.
#include <algorithm>
#include <atomic>
#include <cstring>
#include <mutex>

#include "common.cuh"

namespace cat {
namespace {

constexpr int TM = 128;                 // rows per tile
constexpr int kThreads = 512;
constexpr int kEpiWarp0 = 4, kCvtWarp0 = 8, kCvtWarps = 8;
constexpr int kXStages = 4;                    // every unit of a CTA in flight at once (<= 4 units at k = 128)
static_assert((64 * 64 / 8) % (kCvtWarps * 32) == 0, "converter items must divide evenly");

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

// Shared-memory layout of the fused kernel.  A unit is (group of N output channels, 128-row tile);
// the group's block has KD input channels (N = KD = 128 or 64; N = 64, KD = 256 for 256-blocks, whose
// three bf16 planes would not fit whole: a group is a quarter of the block's outputs).  An x stage
// holds 128 rows x min(KD, 128) channels; a unit takes XH = KD / 128 stages (1 below 256).  U units'
// x' tiles are resident in tensor memory at once (their slots, N columns each); with WAVES a CTA has
// more units than slots and reuses a slot once the unit in it is quantized.  A slot's final row
// maxima (128 floats): in a single wave at N = KD = 128 (at most kXStages units) in the unit's x
// stage, free once its MMAs are done; otherwise in their own room, with one x stage fewer at 128 in
// waves, and three at KD = 256, to make room.
template <int N, int KD, bool WAVES>
struct FusedCfg {
  static constexpr int U = 512 / N;
  static constexpr int XH = KD > 128 ? KD / 128 : 1;
  static constexpr int XW = KD > 128 ? 128 : KD;
  static constexpr int XATOMS = XW / 64;                     // 128-byte channel atoms of an x stage
  static constexpr uint32_t X_STAGE = TM * XW * 2;
  static constexpr int XS = KD > 128 ? 3 : ((WAVES && N == 128) ? kXStages - 1 : kXStages);
  static constexpr uint32_t SPLIT = N * KD * 2;              // one bf16 plane of a group
  static constexpr uint32_t X_OFF = 0;
  static constexpr uint32_t T_OFF = XS * X_STAGE;
  static constexpr uint32_t BAR_OFF = T_OFF + 3 * SPLIT;
  static constexpr uint32_t BAR_BYTES = 512;
  static constexpr bool AMAX_IN_X = !WAVES && N == 128 && KD == 128;
  static constexpr uint32_t AMAX_OFF = BAR_OFF + BAR_BYTES;
  static constexpr size_t SMEM = AMAX_OFF + (AMAX_IN_X ? 0 : U * TM * 4) + 1024;
  // kind::f16: D fp32 (bit 4), A = B = BF16 (format 1 at bits 7 and 10), K-major, M = 128, N
  static constexpr uint32_t IDESC = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) |
                                    ((uint32_t)(TM >> 4) << 24);
  __device__ static float* amax_slot(uint8_t* smem, int slot) {
    return reinterpret_cast<float*>(AMAX_IN_X ? smem + X_OFF + slot * X_STAGE : smem + AMAX_OFF + slot * TM * 4);
  }
};
static_assert(FusedCfg<128, 128, false>::SMEM <= 227 * 1024 && FusedCfg<128, 128, true>::SMEM <= 227 * 1024 &&
                  FusedCfg<64, 256, true>::SMEM <= 227 * 1024,
              "shared memory");

struct TcBars {
  uint64_t x_full[kXStages], x_empty[kXStages], d_full[2], d_empty[2], t_full, t_empty, mma_done;
  uint64_t t_first;                              // fused kernel: the CTA's first T_b split is in shared memory
  uint32_t tmem_addr;
  int abort;
};
// the barrier block fits the 256 bytes reserved for it (the fused kernel reserves FusedCfg::BAR_BYTES)
static_assert(sizeof(TcBars) <= 256, "barrier room");

__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                         uint32_t accumulate) {
  asm volatile(
      "{ .reg .pred p; setp.ne.b32 p, %4, 0; "
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p; }" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Units (block b, 128-row tile) of CTA c, block-major.  With at least as many CTAs as blocks, every
// CTA works inside one block (its split of T_b is made once) and the CTAs of a block share its tiles
// evenly; otherwise CTAs take contiguous ranges of units.
__host__ __device__ inline void unit_range(int c, int grid, int nb, int tiles, int64_t* u0, int64_t* u1) {
  if (grid >= nb) {
    const int b = (int)((int64_t)c * nb / grid);
    const int c_lo = (int)(((int64_t)b * grid + nb - 1) / nb);
    const int c_hi = (int)(((int64_t)(b + 1) * grid + nb - 1) / nb);
    const int m = c_hi - c_lo, i = c - c_lo;
    *u0 = (int64_t)b * tiles + (int64_t)tiles * i / m;
    *u1 = (int64_t)b * tiles + (int64_t)tiles * (i + 1) / m;
  } else {
    const int64_t units = (int64_t)nb * tiles;
    *u0 = units * c / grid;
    *u1 = units * (c + 1) / grid;
  }
}

// The fused kernel's units of CTA c.  With at least as many CTAs as blocks, the m CTAs of block b
// take its row tiles round robin (the i-th of them: tiles i, i + m, i + 2m, ...), so that tile t sits
// at position t / m in its CTA in every block, and the tiles' row maxima become final in ascending
// tile order across the grid; otherwise contiguous block-major ranges as unit_range.
struct FusedUnits {
  int64_t u0;        // contiguous ranges: the first unit (block-major index)
  int b, first, step;
  int count;         // units of the CTA
  bool round_robin;
};
__host__ __device__ inline FusedUnits fused_units(int c, int grid, int nb, int tiles) {
  FusedUnits f;
  f.u0 = 0;
  f.b = 0;
  f.first = 0;
  f.step = 1;
  f.round_robin = grid >= nb;
  if (f.round_robin) {
    const int b = (int)((int64_t)c * nb / grid);
    const int c_lo = (int)(((int64_t)b * grid + nb - 1) / nb);
    const int c_hi = (int)(((int64_t)(b + 1) * grid + nb - 1) / nb);
    const int m = c_hi - c_lo, i = c - c_lo;
    f.b = b;
    f.first = i;
    f.step = m;
    f.count = i < tiles ? (tiles - i + m - 1) / m : 0;
  } else {
    int64_t u1;
    unit_range(c, grid, nb, tiles, &f.u0, &u1);
    f.count = (int)(u1 - f.u0);
  }
  return f;
}
__host__ __device__ inline void fused_unit(const FusedUnits& f, int j, int tiles, int* b, int* tile) {
  if (f.round_robin) {
    *b = f.b;
    *tile = f.first + j * f.step;
  } else {
    const int64_t u = f.u0 + j;
    *b = (int)(u / tiles);
    *tile = (int)(u % tiles);
  }
}

__device__ __forceinline__ uint32_t bf16x2_bits(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Split the fp32 K x K group matrix into bf16 H, M, L in the MMA's 128B-swizzled K-major layout;
// `ct` is the thread's index among the converter threads.  The group matrix is block-diagonal with
// kb x kb blocks (kb divides K; kb = K: one block): Ab points to the group's K rows in the [rows][kb]
// layout of the blocks (row i = output i), and entry (i, j) is Ab[i][j % kb] when i and j lie in the
// same block, 0 otherwise.  A block-diagonal T thus runs on the K-wide kernels exactly: the zeros
// add exact zeros to the fp32 sums.
template <int N, int KD>
__device__ __forceinline__ void split_block(const float* __restrict__ Ab, int kb, uint8_t* ts, int ct) {
  constexpr uint32_t kSplit = N * KD * 2;                     // one plane
  static_assert((N * KD / 8) % (kCvtWarps * 32) == 0, "converter items must divide evenly");
  // all loads first (the block is read from L2/HBM once per block change: keep them in flight together)
  constexpr int kIt = N * KD / 8 / (kCvtWarps * 32);
  float4 pv[kIt], qv[kIt];
#pragma unroll
  for (int it = 0; it < kIt; ++it) {  // 8 consecutive inputs of one output row per item (kb >= 16)
    const int ch = ct + it * kCvtWarps * 32;
    const int i = ch / (KD / 8), j0 = (ch % (KD / 8)) * 8;
    if (i / kb == j0 / kb) {
      pv[it] = __ldg(reinterpret_cast<const float4*>(Ab + (size_t)i * kb + (j0 % kb)));
      qv[it] = __ldg(reinterpret_cast<const float4*>(Ab + (size_t)i * kb + (j0 % kb) + 4));
    } else {
      pv[it] = qv[it] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
  }
#pragma unroll
  for (int it = 0; it < kIt; ++it) {
    const int ch = ct + it * kCvtWarps * 32;
    const int i = ch / (KD / 8), j0 = (ch % (KD / 8)) * 8;
    const float4 p = pv[it], q = qv[it];
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
    const uint32_t off = atom * (N * 128) + i * 128 + ((chunk ^ (i & 7)) << 4);
    *reinterpret_cast<uint4*>(ts + off) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
    *reinterpret_cast<uint4*>(ts + kSplit + off) = make_uint4(mw[0], mw[1], mw[2], mw[3]);
    *reinterpret_cast<uint4*>(ts + 2 * kSplit + off) = make_uint4(lw[0], lw[1], lw[2], lw[3]);
  }
}

// The three planes of T_b, pre-split by cat_split_transform into exactly the shared-memory image
// split_block writes, fetched with one bulk copy per plane (counted on `bar`).
__device__ __forceinline__ void bulk_copy_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   smem_u32(dst)),
               "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(smem_u32(bar))
               : "memory");
}
template <int N, int KD>
__device__ __forceinline__ void fetch_planes(const uint8_t* __restrict__ planes, int g, uint8_t* ts, uint64_t* bar) {
  constexpr uint32_t kSplit = N * KD * 2;
  mbar_arrive_expect_tx(bar, 3 * kSplit);
  const uint8_t* src = planes + (size_t)g * 3 * kSplit;
#pragma unroll
  for (int sp = 0; sp < 3; ++sp) bulk_copy_g2s(ts + sp * kSplit, src + sp * kSplit, kSplit, bar);
}

// The three bf16 planes of every group (N outputs x KD inputs), in the MMA's shared-memory layout
// (cat_split_transform).
template <int N, int KD>
__global__ void __launch_bounds__(kCvtWarps * 32)
    split_planes_kernel(const float* __restrict__ A, int kb, uint8_t* __restrict__ planes) {
  split_block<N, KD>(A + (size_t)blockIdx.x * N * kb, kb, planes + (size_t)blockIdx.x * 3 * N * KD * 2, threadIdx.x);
}

// Four two's-complement bytes in [-7, 7] -> the SM4x8 sign-magnitude bytes (sign << 7 | magnitude).
__device__ __forceinline__ uint32_t twos_to_sm(uint32_t w) {
  const uint32_t s = (w >> 7) & 0x01010101u;        // 1 in every negative byte
  const uint32_t m = (s << 8) - s;                   // 0xFF in every negative byte
  return ((w ^ m) + s) | (s << 7);                   // |q| (no carry leaves a byte) and the sign bit
}

// qcode_exact out of line: the rare near-tie route then costs a call, not 32 inlined copies.
__device__ __noinline__ int qcode_exact_call(float v, QRow qr) { return qcode_exact(v, qr, 7.0f); }

// The codes of the 32 values v_e in tensor memory at taddr (this lane's row, 32 columns) on the row
// described by qr (|v_e| <= max|v|), as eight words of E4M3 code bytes (codes 4i .. 4i+3 in word i,
// little-endian); called by the whole warp.  Fast route:
// adding 1.5 * 2^23 to p = fl(v_e * inv) rounds it to an integer (half to even) that sits, two's
// complement, in the low byte of the sum's bits; the bytes are gathered four to a word and turned
// into sign-magnitude.  The products and sums run as f32x2 pairs, with the same rounding as the scalar
// operations.  If any lane has a p within 2^-18 of a half-integer (an exact tie included), or a
// rescaled row, the warp reloads the chunk and the lanes concerned decide those values' codes exactly
// (qcode_exact): the values are not kept live across that rare branch, which leaves the fast route
// its registers, and the branch costs about one exact decision rather than 32.
// qr.inv == 0 (an all-zero or non-finite row): all codes 0.
__device__ __forceinline__ void quant_chunk(uint32_t taddr, const QRow& qr, uint32_t (&out)[8]) {
  constexpr float kMagic = 12582912.0f;
  uint32_t bq[32];
  bool near = qr.exact;
  {
    uint32_t r[32];
    __syncwarp();
    CAT_TMEM_LD32(taddr, r);
    tmem_ld_wait();
    uint64_t inv2, mg2;
    asm("mov.b64 %0, {%1, %1};" : "=l"(inv2) : "f"(qr.inv));
    asm("mov.b64 %0, {%1, %1};" : "=l"(mg2) : "f"(kMagic));
#pragma unroll
    for (int e = 0; e < 32; e += 2) {
      uint64_t v2, p2, rb2, d2;
      asm("mov.b64 %0, {%1, %2};" : "=l"(v2) : "r"(r[e]), "r"(r[e + 1]));
      asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(p2) : "l"(v2), "l"(inv2));
      asm("add.rn.f32x2 %0, %1, %2;" : "=l"(rb2) : "l"(p2), "l"(mg2));
      asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(d2) : "l"(rb2), "l"(mg2));
      asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(d2) : "l"(d2), "l"(p2));
      float d0, d1;
      asm("mov.b64 {%0, %1}, %2;" : "=f"(d0), "=f"(d1) : "l"(d2));
      asm("mov.b64 {%0, %1}, %2;" : "=r"(bq[e]), "=r"(bq[e + 1]) : "l"(rb2));
      near |= fmaxf(fabsf(d0), fabsf(d1)) > kNearTie;
    }
  }
  if (__any_sync(0xFFFFFFFFu, near)) {
    uint32_t r[32];
    __syncwarp();
    CAT_TMEM_LD32(taddr, r);
    tmem_ld_wait();
    if (near) {                                  // patch the codes of this lane's near values only
#pragma unroll
      for (int e = 0; e < 32; ++e) {
        const float v = __uint_as_float(r[e]);
        const float p = __fmul_rn(v, qr.inv);
        if (qr.exact || fabsf(__fsub_rn(__fsub_rn(__fadd_rn(p, kMagic), kMagic), p)) > kNearTie)
          bq[e] = (bq[e] & ~0xFFu) | ((uint32_t)qcode_exact_call(v, qr) & 0xFFu);
      }
    }
  }
  const bool zero = qr.inv == 0.f;
#pragma unroll
  for (int g = 0; g < 8; ++g) {
    const uint32_t* bg = bq + 4 * g;
    const uint32_t e =
        twos_to_sm(__byte_perm(__byte_perm(bg[0], bg[1], 0x0040), __byte_perm(bg[2], bg[3], 0x0040), 0x5410));
    out[g] = zero ? 0u : e;
  }
}

// The four SM4x8 words of a chunk's 32 code bytes (codes 8g .. 8g+7 in word g).
__device__ __forceinline__ uint4 sm4_words(const uint32_t (&e)[8]) {
  return make_uint4(e[0] | __funnelshift_l(e[1], e[1], 4), e[2] | __funnelshift_l(e[3], e[3], 4),
                    e[4] | __funnelshift_l(e[5], e[5], 4), e[6] | __funnelshift_l(e[7], e[7], 4));
}

// Running maximum of |v| over 32 values, on their bit patterns: for non-negative floats the bit
// order is the value order, and every NaN pattern lies above the infinity 0x7F800000, so the result
// is below 0x7F800000 exactly when all 32 values are finite.
__device__ __forceinline__ uint32_t absmax_bits32(const uint32_t (&r)[32], uint32_t m) {
#pragma unroll
  for (int e = 0; e < 32; ++e) m = max(m, r[e] & 0x7FFFFFFFu);
  return m;
}

template <int K, int PASS>
__global__ void __launch_bounds__(kThreads, 1)
    transform_quant_tc_kernel(const __grid_constant__ CUtensorMap tmX, const float* __restrict__ A,
                              const uint8_t* __restrict__ planes, int n, int d, int kb, uint32_t* __restrict__ amax_bits,
                              uint32_t* __restrict__ codes, float* __restrict__ scale, uint32_t* __restrict__ exit_ctr,
                              uint32_t* __restrict__ status) {
  // scale != nullptr (pass 1 with the maxima in a scratch slot): the CTAs holding block 0 write the
  // steps s = max / 7, and the last CTA out zeroes the slot's maxima and its exit counter
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
  int64_t u0, u1;
  unit_range(blockIdx.x, gridDim.x, nb, num_tiles, &u0, &u1);

  if (tid == 0) {
    for (int s = 0; s < kXStages; ++s) {
      mbar_init(&bars->x_full[s], 1);
      mbar_init(&bars->x_empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&bars->d_full[s], 1);
      mbar_init(&bars->d_empty[s], 4);
    }
    mbar_init(&bars->t_first, planes ? 1 : kCvtWarps);   // pre-split planes: one copying thread
    mbar_init(&bars->t_full, planes ? 1 : kCvtWarps);
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
        // the first unit's x tile goes out with T_b's loads, the others once T_b is split (T_b would
        // otherwise queue behind them in HBM)
        if (j == 1 && !(ok = mbar_wait_bounded(&bars->t_first, 0, abort_flag, __LINE__))) break;
        if (j >= kXStages && !(ok = mbar_wait_bounded(&bars->x_empty[s], ((j / kXStages) - 1) & 1, abort_flag, __LINE__))) break;
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
          if (!(ok = mbar_wait_bounded(&bars->t_full, version & 1, abort_flag, __LINE__))) break;
          ++version;
          cur_b = b;
        }
        const uint32_t s = j % kXStages, sd = j & 1;
        if (!(ok = mbar_wait_bounded(&bars->x_full[s], (j / kXStages) & 1, abort_flag, __LINE__))) break;
        if (j >= 2 && !(ok = mbar_wait_bounded(&bars->d_empty[sd], ((j >> 1) - 1) & 1, abort_flag, __LINE__))) break;
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
      if (version > 0 && !(ok = mbar_wait_bounded(&bars->t_empty, (version - 1) & 1, abort_flag, __LINE__))) break;
      cur_b = b;
      if (planes) {                                    // one thread copies the pre-split planes
        if (ct == 0) {
          fetch_planes<K, K>(planes, b, ts, &bars->t_full);
          if (version == 0) mbar_arrive(&bars->t_first);
        }
      } else {
        split_block<K, K>(A + (size_t)b * K * kb, kb, ts, ct);
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(&bars->t_full);
          if (version == 0) mbar_arrive(&bars->t_first);
        }
      }
      ++version;
    }
  } else if (warp >= kEpiWarp0) {
    // ---------------------------------------------------------------- epilogue: one row per thread
    const int quad = warp & 3;
    const int64_t words_per_row = d / 8;
    bool ok = true, finite = true;
    uint32_t j = 0;
    // pass 1: this lane's row maximum for the next unit is loaded while the current unit is quantized
    auto row_of = [&](int64_t uu) { return (int)(uu % num_tiles) * TM + quad * 32 + lane; };
    float a_next = 0.f;
    if (PASS == 1 && u0 < u1 && row_of(u0) < n) a_next = __uint_as_float(__ldcg(&amax_bits[row_of(u0)]));
    for (int64_t u = u0; u < u1 && ok; ++u, ++j) {
      const int b = (int)(u / num_tiles), tile = (int)(u % num_tiles);
      const uint32_t sd = j & 1;
      const int t = tile * TM + quad * 32 + lane;
      QRow qr = qrow_setup(0.f, 7.0f);
      if (PASS == 1) {
        const float a = a_next;
        if (u + 1 < u1 && row_of(u + 1) < n) a_next = __uint_as_float(__ldcg(&amax_bits[row_of(u + 1)]));
        if (t < n) qr = qrow_setup(a, 7.0f);
        if (scale && b == 0 && t < n) {               // each row's one unit of block 0 writes its step
          float sc = 0.f;
          if (isfinite(a))
            sc = __fdiv_rn(a, 7.0f);
          else
            report(status, kStatusNonFinite);
          scale[t] = sc;
        }
      }
      if (!(ok = mbar_wait_bounded(&bars->d_full[sd], (j >> 1) & 1, abort_flag, __LINE__))) break;
      __syncwarp();
      tc_fence_after();
      float m = 0.f;
      bool row_finite = true;
#pragma unroll 1
      for (int c = 0; c < K / 32; ++c) {
        const uint32_t taddr = tmem + ((uint32_t)(quad * 32) << 16) + sd * K + c * 32;
        if (PASS == 0) {
          uint32_t r[32];
          __syncwarp();
          CAT_TMEM_LD32(taddr, r);
          tmem_ld_wait();
#pragma unroll
          for (int e = 0; e < 32; ++e) {
            const float v = __uint_as_float(r[e]);
            row_finite &= isfinite(v);
            m = fmaxf(m, fabsf(v));
          }
        } else {
          // the row's codes with the final maximum (|v * inv| <= 7 for a finite row; inv = 0 gives
          // 0 codes for an all-zero or non-finite row)
          uint32_t e[8];
          quant_chunk(taddr, qr, e);
          if (t < n)
            *reinterpret_cast<uint4*>(codes + (int64_t)t * words_per_row + ((int64_t)b * K + c * 32) / 8) = sm4_words(e);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars->d_empty[sd]);
      // a non-finite value makes the row's maximum the largest NaN pattern: its codes and step become 0
      finite &= row_finite;
      if (PASS == 0 && t < n) atomicMax(&amax_bits[t], row_finite ? __float_as_uint(m) : 0x7FFFFFFFu);
    }
    if (PASS == 0 && !finite) report(status, kStatusNonFinite);
  }

  __syncthreads();
  if (PASS == 1 && exit_ctr) {
    // the last CTA out returns the slot to zero: every CTA has read its maxima before it counts out
    __shared__ int last_out;
    if (tid == 0) {
      __threadfence();
      last_out = atomicAdd(exit_ctr, 1u) == gridDim.x - 1;
    }
    __syncthreads();
    if (last_out) {
      __threadfence();
      for (int t = tid; t < n; t += kThreads) amax_bits[t] = 0u;
      __threadfence();
      __syncthreads();
      if (tid == 0) *exit_ctr = 0u;
    }
  }
  if (bars->abort && tid == 0) report(status, timeout_bits(kWhereTransform2Pass, bars->abort));
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

// ---- single-launch variant: x' stays in tensor memory between the two row-wide phases ---------
//
// When every CTA's units fit in tensor memory at once (units per CTA x K <= 512 columns), one
// cooperative launch does both passes.  Phase A runs the MMAs once, keeps each unit's x' tile in its
// own TMEM columns and publishes the tile's row maxima (atomicMax into the launch's scratch, then a
// count on the tile's record).  Phase B needs a row's maximum over all blocks, i.e. all nb units of a
// row tile, but not the rest of the grid: a watcher warp per CTA waits for each of its tiles' counts
// in turn, copies the final maxima to shared memory and releases the quantizer warps for that unit,
// while later units are still in phase A.  The CTAs holding block 0 write the steps s = max / 7.
//
// Scratch: each slot (up to kSyncSlots launches may run at once on different streams; slots are
// handed out round robin) has two sets of maxima and tile records, used by alternate launches on the
// slot.  A launch reads the slot's epoch at start (parity = its set), zeroes the other set (left by
// the previous launch on the slot, which has finished: a launch that gave up is cleaned up the same
// way), and the last of its CTAs to start moves the epoch on and records how many tiles its set
// holds.  The state lives on the device, so graph replays alternate too, and no CTA has to wait for
// the others at the end.  Every wait is bounded.
constexpr int kSyncSlots = 8;
constexpr int kAmaxRows = 1 << 17;             // rows the fused path can have (<= 1024 tiles of 128 rows)
constexpr int kAmaxTiles = kAmaxRows / TM;
constexpr int kTileWords = 32;                 // a tile's record ([0]: units' maxima published, 4 per unit)
__device__ __align__(16) uint32_t g_tq_sync[kSyncSlots][4];          // two-pass kernel: [1] exit counter
__device__ uint32_t g_tq_amax[kSyncSlots][kAmaxRows];                // two-pass kernel: row maxima
// fused kernel: [0] epoch, [1] CTAs started, [2 + s] tiles set s holds
__device__ __align__(16) uint32_t g_tqf_state[kSyncSlots][4];
__device__ uint32_t g_tqf_amax[kSyncSlots][2][kAmaxRows];
__device__ __align__(128) uint32_t g_tqf_tiles[kSyncSlots][2][kAmaxTiles * kTileWords];

__device__ __forceinline__ uint32_t ld_acquire_gpu(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Bounded poll of a counter in global memory until it reaches `expected` (one thread).
__device__ __forceinline__ bool wait_count(const uint32_t* ctr, uint32_t expected, volatile int* abort_flag, int site) {
  if (ld_acquire_gpu(ctr) >= expected) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t it = 1;; ++it) {
    __nanosleep(32);
    if (ld_acquire_gpu(ctr) >= expected) return true;
    if ((it & 63u) == 0u && (*abort_flag || globaltimer_ns() - t0 > kWaitLimitNs)) {
      if (*abort_flag == 0) *abort_flag = site;
      return false;
    }
  }
}

// Phase B of one quantizer warp (slot 0: the quadrant's epilogue warp, 1 and 2: its converter
// warps).  Units are taken in order, each once the watcher has put its final row maxima in shared
// memory; a unit's 32-column chunk c goes to slot 1 + (c & 1) except in the CTA's last unit, which the
// three warps share (slot (c + 1) % 3): the epilogue warp joins when its phase A is done.
__device__ __forceinline__ int chunk_slot(int c, bool last) { return last ? (c + 1) % 3 : 1 + (c & 1); }

template <int N, int KD, bool WAVES>
__device__ __forceinline__ void quantize_units(uint32_t tmem, uint8_t* smem, const FusedUnits& fu, int num_tiles,
                                               int n, int d, uint64_t* maxima_ready, uint64_t* tmem_free,
                                               uint32_t* __restrict__ codes, int e8, volatile int* abort_flag,
                                               int slot) {
  // unit j sits in tensor-memory slot j % U (phase (j / U) & 1 of the slot's barriers); with WAVES the
  // converter warps (slots 1 and 2) hand the slot back once their chunks of the unit are done
  using F = FusedCfg<N, KD, WAVES>;
  const int lane = threadIdx.x & 31, quad = (threadIdx.x >> 5) & 3;
  const int64_t words_per_row = d / 8;
  const int nu = fu.count;
  for (int j = 0; j < nu; ++j) {
    const int us = j % F::U;
    const uint32_t ph = (uint32_t)(j / F::U) & 1u;
    const bool last = j == nu - 1;
    bool mine = false;
#pragma unroll
    for (int c = 0; c < N / 32; ++c) mine |= chunk_slot(c, last) == slot;
    if (mine) {
      const bool got = !*abort_flag && mbar_wait_bounded(&maxima_ready[us], ph, abort_flag, __LINE__);
      if (!__all_sync(0xFFFFFFFFu, got)) return;
      int b, tile;
      fused_unit(fu, j, num_tiles, &b, &tile);
      const int t = tile * TM + quad * 32 + lane;
      const float a = F::amax_slot(smem, us)[quad * 32 + lane];
      const QRow qr = qrow_setup(a, 7.0f);     // inv == 0: zero or non-finite row, all codes 0
      tc_fence_after();
#pragma unroll 1
      for (int c = 0; c < N / 32; ++c) {
        if (chunk_slot(c, last) != slot) continue;
        uint32_t e[8];
        quant_chunk(tmem + ((uint32_t)(quad * 32) << 16) + us * N + c * 32, qr, e);
        if (t < n) {
          if (e8) {                            // byte codes: 32 bytes of row t
            uint4* dst = reinterpret_cast<uint4*>(reinterpret_cast<uint8_t*>(codes) + (int64_t)t * d + (int64_t)b * N +
                                                  c * 32);
            dst[0] = make_uint4(e[0], e[1], e[2], e[3]);
            dst[1] = make_uint4(e[4], e[5], e[6], e[7]);
          } else {
            *reinterpret_cast<uint4*>(codes + (int64_t)t * words_per_row + ((int64_t)b * N + c * 32) / 8) = sm4_words(e);
          }
        }
      }
    }
    if (WAVES && slot != 0) {                  // the slot's tensor memory (and maxima) are free again
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tmem_free[us]);
    }
  }
}

template <int N, int KD, bool WAVES>
__global__ void __launch_bounds__(kThreads, 1)
    transform_quant_tc_fused_kernel(const __grid_constant__ CUtensorMap tmX, const float* __restrict__ A,
                                    const uint8_t* __restrict__ planes, int n, int d, int kb, float* __restrict__ scale,
                                    uint32_t* __restrict__ codes, int e8, uint32_t* __restrict__ state,
                                    uint32_t* __restrict__ amax_sets, uint32_t* __restrict__ rec_sets,
                                    uint32_t* __restrict__ status) {
  // state: the slot's epoch, start counter and tiles per set; amax_sets: two sets of kAmaxRows row
  // maxima (float bits); rec_sets: two sets of kAmaxTiles tile records
  using F = FusedCfg<N, KD, WAVES>;
  constexpr int U = F::U;                              // tensor-memory slots (units resident at once)
  static_assert(sizeof(TcBars) + (4 * U + 4) * sizeof(uint64_t) + 8 <= F::BAR_BYTES, "barrier room");
  static_assert(!F::AMAX_IN_X || U <= F::XS, "in one wave at k = 128 unit j's x stage holds its maxima");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* xs = smem + F::X_OFF;
  uint8_t* ts = smem + F::T_OFF;
  TcBars* bars = reinterpret_cast<TcBars*>(smem + F::BAR_OFF);
  // per tensor-memory slot (unit j: slot j % U, phase (j / U) & 1)
  uint64_t* unit_full = reinterpret_cast<uint64_t*>(bars + 1);   // the unit's MMAs are done
  uint64_t* epi_done = unit_full + U;                             // its row maxima's atomics are issued
  uint64_t* maxima_ready = epi_done + U;                          // its final maxima are in shared memory
  uint64_t* tmem_free = maxima_ready + U;                         // WAVES: quantized, the slot is free
  uint64_t* plane_full = tmem_free + U;                           // per plane of T_b (producer-fetched planes)
  uint64_t* set_ready = plane_full + 3;                           // the launch's scratch set is known
  volatile int* set_sel = reinterpret_cast<int*>(set_ready + 1);  // ... and it is set_sel (0 or 1)
  volatile int* abort_flag = &bars->abort;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nb = d / N;                                // groups of N output channels
  const int num_tiles = (n + TM - 1) / TM;
  FusedUnits fu = fused_units(blockIdx.x, gridDim.x, nb, num_tiles);
  if (!WAVES && fu.count > U) fu.count = U;            // the launcher guarantees this never cuts
  const int nu = fu.count;
  // With pre-split planes and one block per CTA, the producer fetches the planes itself, in the order
  // H, (unit 0's x tile), M, L, and unit 0's MMAs start on H while M and L are still on their way.
  const bool own_planes = planes != nullptr && fu.round_robin;

  if (tid == 0) {
    for (int st = 0; st < kXStages; ++st) {
      mbar_init(&bars->x_full[st], 1);
      mbar_init(&bars->x_empty[st], 1);
    }
    for (int j = 0; j < U; ++j) {
      mbar_init(&unit_full[j], 1);
      mbar_init(&epi_done[j], 4);                       // the four epilogue warps
      mbar_init(&maxima_ready[j], 1);
      mbar_init(&tmem_free[j], kCvtWarps);              // the converter warps, after their chunks
    }
    for (int sp = 0; sp < 3; ++sp) mbar_init(&plane_full[sp], 1);
    mbar_init(set_ready, 1);
    mbar_init(&bars->t_first, planes ? 1 : kCvtWarps);   // pre-split planes: one copying thread
    mbar_init(&bars->t_full, planes ? 1 : kCvtWarps);
    mbar_init(&bars->t_empty, 1);
    mbar_init(&bars->mma_done, 1);
    bars->abort = 0;
    fence_mbar_init();
  }
  __syncwarp();
  pdl_wait_then_release();                        // nothing global or in tensor memory before this
  if (warp == 0) tmem_alloc(&bars->tmem_addr, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem_addr;

  if (warp == 0) {
    // ---------------------------------------------------------------- TMA producer
    if (lane == 0) {
      prefetch_tensormap(&tmX);
      bool ok = true;
      const uint8_t* src = own_planes ? planes + (size_t)fu.b * 3 * F::SPLIT : nullptr;
      if (own_planes) {
        mbar_arrive_expect_tx(&plane_full[0], F::SPLIT);
        bulk_copy_g2s(ts, src, F::SPLIT, &plane_full[0]);
      }
      // stage q = j XH + h: half h of unit j's x tile (the whole tile below KD = 256)
      int q = 0;
      const int nq = nu * F::XH;
      for (; q < nq; ++q) {
        const int j = q / F::XH, h = q % F::XH;
        int g, tile;
        fused_unit(fu, j, num_tiles, &g, &tile);
        const int in0 = (g * N / KD) * KD + h * F::XW;   // first input channel of this stage
        const uint32_t st = q % F::XS;
        if (own_planes) {
          // M and L after the first stage; the stages from the third on after all of T's planes are in
          if (q == 2 && !(ok = mbar_wait_bounded(&plane_full[2], 0, abort_flag, __LINE__))) break;
        } else {
          // the first two stages go out with T's loads; the others wait until T is in shared memory,
          // so that T does not queue behind them and unit 0's MMAs start as early as they can
          if (q == 2 && !(ok = mbar_wait_bounded(&bars->t_first, 0, abort_flag, __LINE__))) break;
        }
        if (q >= F::XS && !(ok = mbar_wait_bounded(&bars->x_empty[st], ((q / F::XS) - 1) & 1, abort_flag, __LINE__))) break;
        mbar_arrive_expect_tx(&bars->x_full[st], F::X_STAGE);
#pragma unroll
        for (int a = 0; a < F::XATOMS; ++a)
          tma_load_2d(xs + st * F::X_STAGE + a * (TM * 128), &tmX, in0 + 64 * a, tile * TM, &bars->x_full[st]);
        if (own_planes && q == 0) {
#pragma unroll
          for (int sp = 1; sp < 3; ++sp) {
            mbar_arrive_expect_tx(&plane_full[sp], F::SPLIT);
            bulk_copy_g2s(ts + sp * F::SPLIT, src + sp * F::SPLIT, F::SPLIT, &plane_full[sp]);
          }
        }
      }
      const int issued = q, first = issued > F::XS ? issued - F::XS : 0;
      volatile int no_abort = 0;
      for (int r = first; r < issued; ++r) mbar_wait_bounded(&bars->x_full[r % F::XS], (r / F::XS) & 1, &no_abort);
      if (own_planes)
        for (int sp = 0; sp < 3; ++sp) mbar_wait_bounded(&plane_full[sp], 0, &no_abort);
      (void)ok;
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer: unit j -> slot j % U
    // D = V H^T + V M^T + V L^T, plane by plane
    if (lane == 0) {
      bool ok = true;
      uint32_t version = 0;
      int cur_b = -1;
      for (int j = 0; j < nu && ok; ++j) {
        int b, tile;
        fused_unit(fu, j, num_tiles, &b, &tile);
        if (b != cur_b) {
          if (!own_planes && !(ok = mbar_wait_bounded(&bars->t_full, version & 1, abort_flag, __LINE__))) break;
          ++version;
          cur_b = b;
        }
        // WAVES: the unit U back in this slot must be quantized before its columns are overwritten
        if (WAVES && j >= U && !(ok = mbar_wait_bounded(&tmem_free[j % U], ((j / U) - 1) & 1, abort_flag, __LINE__))) break;
        const uint32_t dcol = tmem + (j % U) * N;
        const uint32_t tbase = smem_u32(ts);
        for (int h = 0; h < F::XH && ok; ++h) {       // the unit's x stages (two K halves at KD = 256)
          const int q = j * F::XH + h;
          const uint32_t st = q % F::XS;
          if (!(ok = mbar_wait_bounded(&bars->x_full[st], (q / F::XS) & 1, abort_flag, __LINE__))) break;
          tc_fence_after();
          const uint32_t xbase = smem_u32(xs + st * F::X_STAGE);
#pragma unroll
          for (int sp = 0; sp < 3; ++sp) {
            if (own_planes && q == 0) {                 // later stages find every plane in place
              if (!(ok = mbar_wait_bounded(&plane_full[sp], 0, abort_flag, __LINE__))) break;
              tc_fence_after();
            }
#pragma unroll
            for (int kk = 0; kk < F::XW / 16; ++kk) {
              const int kg = h * (F::XW / 16) + kk;       // the K step within the group's KD inputs
              const uint32_t a_off = (kk >> 2) * (TM * 128) + (kk & 3) * 32;
              const uint32_t b_off = (kg >> 2) * (N * 128) + (kg & 3) * 32;
              mma_bf16(dcol, sdesc_kmajor_sw128(xbase + a_off), sdesc_kmajor_sw128(tbase + sp * F::SPLIT + b_off),
                       F::IDESC, (h | kk | sp) != 0);
            }
          }
          if (!ok) break;
          mma_commit(&bars->x_empty[st]);
        }
        if (!ok) break;
        mma_commit(&unit_full[j % U]);
        int nb_next = -1, tile_next;
        if (j + 1 < nu) fused_unit(fu, j + 1, num_tiles, &nb_next, &tile_next);
        if (nb_next != b) mma_commit(&bars->t_empty);     // the CTA's last unit of block b
      }
      mma_commit(&bars->mma_done);
      volatile int no_abort = 0;
      mbar_wait_bounded(&bars->mma_done, 0, &no_abort);
    }
  } else if (warp == 2) {
    // ---------------------------------------------------------------- watcher: final maxima, unit by unit
    const bool have_set = __all_sync(0xFFFFFFFFu, mbar_wait_bounded(set_ready, 0, abort_flag, __LINE__));
    const int P = *set_sel;
    const uint32_t* amax_bits = amax_sets + (size_t)P * kAmaxRows;
    const uint32_t* tile_rec = rec_sets + (size_t)P * kAmaxTiles * kTileWords;
    for (int j = 0; j < nu && have_set; ++j) {
      int b, tile;
      fused_unit(fu, j, num_tiles, &b, &tile);
      bool ok = true;
      if (lane == 0) ok = wait_count(tile_rec + (size_t)tile * kTileWords, 4u * (uint32_t)nb, abort_flag, __LINE__);
      if (!__shfl_sync(0xFFFFFFFFu, (int)ok, 0)) break;
      // unit j's MMAs are done (this CTA counted the tile after them): in one wave at k = 128 its x
      // stage is free for the maxima
      if (F::AMAX_IN_X) {
        if (!__all_sync(0xFFFFFFFFu, mbar_wait_bounded(&unit_full[j], 0, abort_flag, __LINE__))) break;
        fence_proxy_async_smem();
      }
      uint32_t v[TM / 32];
#pragma unroll
      for (int i = 0; i < TM / 32; ++i) v[i] = __ldcg(&amax_bits[tile * TM + 32 * i + lane]);  // < kAmaxRows
      float* am = F::amax_slot(smem, j % U);
#pragma unroll
      for (int i = 0; i < TM / 32; ++i) am[32 * i + lane] = __uint_as_float(v[i]);
      __syncwarp();
      if (lane == 0) mbar_arrive(&maxima_ready[j % U]);
      if (b == 0) {                                      // the CTAs holding block 0 write the steps
#pragma unroll
        for (int i = 0; i < TM / 32; ++i) {
          const int t = tile * TM + 32 * i + lane;
          const float a = __uint_as_float(v[i]);
          if (t >= n) continue;
          float sc = 0.f;
          if (isfinite(a))
            sc = __fdiv_rn(a, 7.0f);
          else
            report(status, kStatusNonFinite);
          scale[t] = sc;
        }
      }
    }
  } else if (warp == 3) {
    // ---------------------------------------------------------------- publisher
    // Start: the slot's epoch gives this launch's scratch set; this CTA's share of the other set (left
    // by the previous launch on the slot, finished) goes back to zero; the last CTA to start moves the
    // epoch on (every CTA has read it by then) and records the tiles this launch's set holds.
    uint32_t E = 0, prev_tiles = 0;
    if (lane == 0) E = ld_acquire_gpu(&state[0]);
    E = __shfl_sync(0xFFFFFFFFu, E, 0);
    const int P = (int)(E & 1u);
    if (lane == 0) {
      *set_sel = P;
      mbar_arrive(set_ready);
      prev_tiles = state[2 + (P ^ 1)];
    }
    prev_tiles = min(__shfl_sync(0xFFFFFFFFu, prev_tiles, 0), (uint32_t)kAmaxTiles);
    {
      uint32_t* amax_o = amax_sets + (size_t)(P ^ 1) * kAmaxRows;
      uint32_t* rec_o = rec_sets + (size_t)(P ^ 1) * kAmaxTiles * kTileWords;
      const int64_t rows = (int64_t)prev_tiles * TM, words = (int64_t)prev_tiles * kTileWords;
      const int64_t r0 = rows * blockIdx.x / gridDim.x, r1 = rows * (blockIdx.x + 1) / gridDim.x;
      const int64_t w0 = words * blockIdx.x / gridDim.x, w1 = words * (blockIdx.x + 1) / gridDim.x;
      for (int64_t i = r0 + lane; i < r1; i += 32) amax_o[i] = 0u;
      for (int64_t i = w0 + lane; i < w1; i += 32) rec_o[i] = 0u;
    }
    __syncwarp();
    uint32_t* tile_rec = rec_sets + (size_t)P * kAmaxTiles * kTileWords;
    if (lane == 0) {
      __threadfence();
      if (atomicAdd(&state[1], 1u) == gridDim.x - 1) {
        state[2 + P] = (uint32_t)num_tiles;
        state[1] = 0u;
        __threadfence();
        state[0] = E + 1u;
      }
      // A unit's count: the four epilogue warps of unit j arrive on epi_done[j] after issuing the
      // unit's atomicMax; the fence here (after that CTA-scope synchronization) orders them before the
      // count at GPU scope, so the epilogue warps never wait on a fence themselves.
      for (int j = 0; j < nu; ++j) {
        int b, tile;
        fused_unit(fu, j, num_tiles, &b, &tile);
        if (!mbar_wait_bounded(&epi_done[j % U], (j / U) & 1, abort_flag, __LINE__)) break;
        __threadfence();
        atomicAdd(&tile_rec[(size_t)tile * kTileWords], 4u);
      }
    }
  } else if (warp >= kCvtWarp0) {
    // ---------------------------------------------------------------- T_b into shared memory, then phase B
    if (!own_planes) {
      const int ct = tid - kCvtWarp0 * 32;
      bool ok = true;
      uint32_t version = 0;
      int cur_b = -1;
      for (int j = 0; j < nu && ok; ++j) {
        int b, tile;
        fused_unit(fu, j, num_tiles, &b, &tile);
        if (b == cur_b) continue;
        if (version > 0 && !(ok = mbar_wait_bounded(&bars->t_empty, (version - 1) & 1, abort_flag, __LINE__))) break;
        cur_b = b;
        if (planes) {                                  // one thread copies the pre-split planes
          if (ct == 0) {
            fetch_planes<N, KD>(planes, b, ts, &bars->t_full);
            if (version == 0) mbar_arrive(&bars->t_first);
          }
        } else {
          split_block<N, KD>(A + (size_t)b * N * kb, kb, ts, ct);
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            mbar_arrive(&bars->t_full);
            if (version == 0) mbar_arrive(&bars->t_first);
          }
        }
        ++version;
      }
    }
    quantize_units<N, KD, WAVES>(tmem, smem, fu, num_tiles, n, d, maxima_ready, tmem_free, codes, e8, abort_flag,
                                 1 + ((warp - kCvtWarp0) >> 2));
    tc_fence_before();
  } else if (warp >= kEpiWarp0) {
    // ---------------------------------------------------------------- phase A: one row per thread
    const int quad = warp & 3;
    bool finite = true;
    const bool have_set = __all_sync(0xFFFFFFFFu, mbar_wait_bounded(set_ready, 0, abort_flag, __LINE__));
    uint32_t* amax_bits = amax_sets + (size_t)(*set_sel) * kAmaxRows;
    for (int j = 0; j < nu && have_set; ++j) {
      int b, tile;
      fused_unit(fu, j, num_tiles, &b, &tile);
      const int t = tile * TM + quad * 32 + lane;
      const bool got = !*abort_flag && mbar_wait_bounded(&unit_full[j % U], (j / U) & 1, abort_flag, __LINE__);
      if (!__all_sync(0xFFFFFFFFu, got)) break;        // warp-uniform: TMEM loads need the whole warp
      tc_fence_after();
      uint32_t mb = 0;
#pragma unroll 1
      for (int c = 0; c < N / 32; c += 2) {            // two loads in flight
        uint32_t r0[32], r1[32];
        __syncwarp();
        CAT_TMEM_LD32(tmem + ((uint32_t)(quad * 32) << 16) + (j % U) * N + c * 32, r0);
        CAT_TMEM_LD32(tmem + ((uint32_t)(quad * 32) << 16) + (j % U) * N + (c + 1) * 32, r1);
        tmem_ld_wait();
        mb = absmax_bits32(r1, absmax_bits32(r0, mb));
      }
      const bool row_finite = mb < 0x7F800000u;
      finite &= row_finite;
      // a non-finite value makes the row's maximum the largest NaN pattern: its codes and step become 0
      if (t < n) atomicMax(&amax_bits[t], row_finite ? mb : 0x7FFFFFFFu);
      __syncwarp();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&epi_done[j % U]);
    }
    if (!finite) report(status, kStatusNonFinite);
    quantize_units<N, KD, WAVES>(tmem, smem, fu, num_tiles, n, d, maxima_ready, tmem_free, codes, e8, abort_flag, 0);
    tc_fence_before();
  }

  __syncthreads();
  if (bars->abort && tid == 0) report(status, timeout_bits(kWhereTransformFused, bars->abort));
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
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

// The device's scratch arrays, looked up once per device.
struct TqScratch {
  uint32_t* sync;       // two-pass kernel: [kSyncSlots][4]
  uint32_t* amax;       // two-pass kernel: [kSyncSlots][kAmaxRows]
  uint32_t* state;      // fused kernel: [kSyncSlots][4]
  uint32_t* amax_sets;  // fused kernel: [kSyncSlots][2][kAmaxRows]
  uint32_t* rec_sets;   // fused kernel: [kSyncSlots][2][kAmaxTiles * kTileWords]
};
const TqScratch* tq_scratch(cudaError_t* err);

// Slots of the transform's device scratch, handed out round robin to every launch that uses one
// (fused or two-pass), so that up to kSyncSlots such launches may be in flight at once.
uint32_t next_tq_slot() {
  static std::atomic<uint32_t> next{0};
  return next.fetch_add(1) % kSyncSlots;
}

// scale != nullptr and n <= kAmaxRows: the maxima go to a slot of device scratch and pass 1 writes
// the steps and returns the slot to zero (no memset, no finalize launch); cudaErrorNotSupported
// otherwise, when the caller zeroes `amax` (its scale buffer) and finalizes the steps itself.
template <int K>
cudaError_t launch_k(const __nv_bfloat16* x, int64_t n, int64_t d, int kb, const float* A, const uint8_t* planes,
                     uint32_t* amax, uint32_t* words, float* scale, uint32_t* status, cudaStream_t stream) {
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
  uint32_t* exit_ctr = nullptr;
  if (scale) {
    if (n > kAmaxRows) return cudaErrorNotSupported;
    cudaError_t es;
    const TqScratch* sc = tq_scratch(&es);
    if (!sc) return es;
    const uint32_t slot = next_tq_slot();
    exit_ctr = sc->sync + 4 * slot + 1;
    amax = sc->amax + (size_t)kAmaxRows * slot;
  }
  note_launch();
  k0<<<grid, kThreads, C::SMEM, stream>>>(map, A, planes, (int)n, (int)d, kb, amax, words, nullptr, nullptr, status);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  note_launch();
  k1<<<grid, kThreads, C::SMEM, stream>>>(map, A, planes, (int)n, (int)d, kb, amax, words, scale, exit_ctr, status);
  return cudaGetLastError();
}

const TqScratch* tq_scratch(cudaError_t* err) {
  static std::mutex mu;
  static TqScratch cache[64];
  static bool have[64] = {false};
  int dev = 0;
  *err = cudaGetDevice(&dev);
  if (*err != cudaSuccess) return nullptr;
  if (dev < 0 || dev >= 64) {
    *err = cudaErrorInvalidDevice;
    return nullptr;
  }
  std::lock_guard<std::mutex> lock(mu);
  if (!have[dev]) {
    void* p[5] = {nullptr, nullptr, nullptr, nullptr, nullptr};
    if ((*err = cudaGetSymbolAddress(&p[0], g_tq_sync)) != cudaSuccess) return nullptr;
    if ((*err = cudaGetSymbolAddress(&p[1], g_tq_amax)) != cudaSuccess) return nullptr;
    if ((*err = cudaGetSymbolAddress(&p[2], g_tqf_state)) != cudaSuccess) return nullptr;
    if ((*err = cudaGetSymbolAddress(&p[3], g_tqf_amax)) != cudaSuccess) return nullptr;
    if ((*err = cudaGetSymbolAddress(&p[4], g_tqf_tiles)) != cudaSuccess) return nullptr;
    cache[dev] = TqScratch{static_cast<uint32_t*>(p[0]), static_cast<uint32_t*>(p[1]), static_cast<uint32_t*>(p[2]),
                           static_cast<uint32_t*>(p[3]), static_cast<uint32_t*>(p[4])};
    have[dev] = true;
  }
  return &cache[dev];
}

bool cooperative_ok() {
  int dev = 0, v = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  return cudaDeviceGetAttribute(&v, cudaDevAttrCooperativeLaunch, dev) == cudaSuccess && v != 0;
}

template <int N, int KD>
cudaError_t launch_fused_k(const __nv_bfloat16* x, int64_t n, int64_t d, int kb, const float* A, const uint8_t* planes,
                           uint32_t* amax, uint32_t* words, int e8, uint32_t* status, cudaStream_t stream) {
  const int nb = (int)(d / N);                         // groups of N output channels
  const int tiles = (int)((n + TM - 1) / TM);
  const int64_t units = (int64_t)nb * tiles;
  const int sms = num_sms();
  // One wave when every CTA's units fit in tensor memory at once; otherwise waves, with the same
  // number m of CTAs on every block (then a tile sits at the same position t / m in every CTA that
  // holds it, and no CTA can wait on a tile that another CTA reaches only after a later wave of its
  // own); beyond one CTA per block the caller takes the two-pass path.
  int grid = (int)(units < sms ? units : sms);
  bool waves = false;
  for (int c = 0; c < grid && !waves; ++c)
    if (fused_units(c, grid, nb, tiles).count > 512 / N) waves = true;
  if (waves) {
    if (nb > sms) return cudaErrorNotSupported;
    const int m = std::min(sms / nb, tiles);
    grid = m * nb;
  }
  if (!cooperative_ok()) return cudaErrorNotSupported;
  EncodeTiledFn fn = encode_fn();
  if (!fn) return cudaErrorNotSupported;
  if (n > kAmaxRows) return cudaErrorNotSupported;
  cudaError_t e;
  const TqScratch* sc = tq_scratch(&e);
  if (!sc) return e;
  const uint32_t slot = next_tq_slot();
  uint32_t* state = sc->state + 4 * slot;
  uint32_t* amax_sets = sc->amax_sets + (size_t)2 * kAmaxRows * slot;
  uint32_t* rec_sets = sc->rec_sets + (size_t)2 * kAmaxTiles * kTileWords * slot;
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
  static std::once_flag once;
  static cudaError_t attr = cudaSuccess;
  std::call_once(once, [] {
    attr = cudaFuncSetAttribute(transform_quant_tc_fused_kernel<N, KD, false>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, (int)FusedCfg<N, KD, false>::SMEM);
    if (attr == cudaSuccess)
      attr = cudaFuncSetAttribute(transform_quant_tc_fused_kernel<N, KD, true>,
                                  cudaFuncAttributeMaxDynamicSharedMemorySize, (int)FusedCfg<N, KD, true>::SMEM);
  });
  if (attr != cudaSuccess) return attr;
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = dim3((unsigned)grid, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = waves ? FusedCfg<N, KD, true>::SMEM : FusedCfg<N, KD, false>::SMEM;
  cfg.stream = stream;
  // not a programmatic dependent launch: measured, one cost the c2 step ~4 us (the kernel still
  // releases its dependents early, so a programmatic GEMM launch after it gets going sooner)
  cudaLaunchAttribute attrs[1];
  attrs[0].id = cudaLaunchAttributeCooperative;
  attrs[0].val.cooperative = 1;
  cfg.attrs = attrs;
  cfg.numAttrs = 1;
  note_launch();
  if (waves)
    return cudaLaunchKernelEx(&cfg, transform_quant_tc_fused_kernel<N, KD, true>, map, A, planes, (int)n, (int)d, kb,
                              reinterpret_cast<float*>(amax), words, e8, state, amax_sets, rec_sets, status);
  return cudaLaunchKernelEx(&cfg, transform_quant_tc_fused_kernel<N, KD, false>, map, A, planes, (int)n, (int)d, kb,
                            reinterpret_cast<float*>(amax), words, e8, state, amax_sets, rec_sets, status);
}

}  // namespace

// The tensor-core transform's input width KD per group (the plane split's group: N = KD outputs,
// except N = 64 at KD = 256) for block size k on d channels: 128 when 128 divides d and k <= 128 (a
// k < 128 runs block-diagonal inside each 128-channel group: 2-8x the MMAs of a k-wide kernel, but
// the 128-wide kernels are the faster ones, e.g. c5 at k = 64: 64 against 87 us), 64 for k = 64
// otherwise, 256 for k = 256 (a group is a quarter of a block's outputs: a whole block's three bf16
// planes would not fit in shared memory), 0 when no tensor-core kernel applies.
int transform_tc_group(int k, int64_t d) {
  if ((k == 16 || k == 32 || k == 64 || k == 128) && d % 128 == 0) return 128;
  if (k == 64 && d % 64 == 0) return 64;
  if (k == 256 && d % 256 == 0) return 256;
  return 0;
}

bool transform_quantize_tc_supported(int dtype, int k, int64_t n, int64_t d) {
  return dtype == 1 && transform_tc_group(k, d) != 0 && n <= 0x7FFFFFFF && d <= 0x7FFFFFFF;
}

// Passes 0 and 1; the caller zeroes the scale buffer before and finalizes it after.
cudaError_t launch_transform_quantize_tc(const void* x, int64_t n, int64_t d, int k, const float* A,
                                         const uint8_t* planes, uint32_t* amax, uint32_t* words, float* scale,
                                         uint32_t* status, cudaStream_t stream) {
  const __nv_bfloat16* xb = static_cast<const __nv_bfloat16*>(x);
  const int K = transform_tc_group(k, d);
  if (K == 64) return launch_k<64>(xb, n, d, k, A, planes, amax, words, scale, status, stream);
  if (K == 128) return launch_k<128>(xb, n, d, k, A, planes, amax, words, scale, status, stream);
  return cudaErrorNotSupported;                      // k = 256: the fused kernel only
}

// T_blocks -> the three bf16 planes of every group (KD = transform_tc_group(k, d) inputs, N outputs)
// in the transform kernels' shared-memory layout ([d/N][3][N*KD] bf16, 6 d KD bytes).
cudaError_t launch_split_transform(const float* A, int64_t d, int k, uint8_t* planes, cudaStream_t stream) {
  const int KD = transform_tc_group(k, d);
  if (KD == 0) return cudaErrorNotSupported;
  note_launch();
  if (KD == 64) split_planes_kernel<64, 64><<<(unsigned)(d / 64), kCvtWarps * 32, 0, stream>>>(A, k, planes);
  else if (KD == 128) split_planes_kernel<128, 128><<<(unsigned)(d / 128), kCvtWarps * 32, 0, stream>>>(A, k, planes);
  else split_planes_kernel<64, 256><<<(unsigned)(d / 64), kCvtWarps * 32, 0, stream>>>(A, k, planes);
  return cudaGetLastError();
}

}  // namespace cat

namespace cat {
// Both phases and the steps in one cooperative launch when every CTA's units fit in tensor memory
// (the row maxima go to a slot of device scratch that the launch leaves zeroed); cudaErrorNotSupported
// otherwise (the caller takes the two-pass path).  e8: the codes as bytes ([n][d], one E4M3 byte per
// code) instead of SM4x8 words.
cudaError_t launch_transform_quantize_tc_fused(const void* x, int64_t n, int64_t d, int k, const float* A,
                                               const uint8_t* planes, uint32_t* amax, uint32_t* words, int e8,
                                               uint32_t* status, cudaStream_t stream) {
  const __nv_bfloat16* xb = static_cast<const __nv_bfloat16*>(x);
  const int KD = transform_tc_group(k, d);
  if (KD == 64) return launch_fused_k<64, 64>(xb, n, d, k, A, planes, amax, words, e8, status, stream);
  if (KD == 128) return launch_fused_k<128, 128>(xb, n, d, k, A, planes, amax, words, e8, status, stream);
  if (KD == 256) return launch_fused_k<64, 256>(xb, n, d, k, A, planes, amax, words, e8, status, stream);
  return cudaErrorNotSupported;
}
}  // namespace cat
