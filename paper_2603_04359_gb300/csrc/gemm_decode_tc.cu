// W4A4 GEMM for a few tokens (decode, n <= 32) on 5th-generation tensor cores (sm_103a).
//
//   acc[t, o] = sum_i q_x[t, i] q_w[o, i],   y[t, o] = acc * s_x[t] * s_w[o]   (Sec. 3, Eq. 5)
//
// With a handful of tokens the packed weight stream (d_out x d_in / 2 bytes) is the whole cost, and
// the legacy mma.sync path of this GPU is too slow to keep up with HBM, so the weights are the MMA's
// M dimension (128 rows per unit) and the tokens its N dimension (16 or 32):
//   * the tokens are decoded once per CTA into a resident K-major, 128B-swizzled E4M3 operand, with
//     every staging thread's loads in flight at once (the first MMA waits for the whole operand);
//   * two producer warps stream 16 KiB packed weight tiles (128 rows x 128 bytes = 256 codes,
//     128-byte swizzle) through a TMA ring -- two issuers, because one issuer's TMA rate is below
//     the per-SM share of HBM bandwidth;
//   * sixteen decode warps, in four groups taking every fourth K step (the decode of a step is a
//     latency chain), turn each tile into E4M3 in tensor memory (thread = weight row = TMEM lane,
//     the whole 256 codes);
//   * one thread issues tcgen05.mma (A from tensor memory, B from shared memory), accumulating the
//     exact products q_x q_w 2^-18 in fp32 (|acc| <= 49 d_in < 2^24);
//   * four epilogue warps read the double-buffered accumulator (thread = output channel) and write
//     y[t][o] with consecutive o across a warp; y_ref, when given, is loaded while the MMAs run.
// Work split (stream-K): the (unit, K step) sequence -- unit-major, num_units x num_ks steps of
// 16 KiB -- is cut into one contiguous, equal range per CTA, one CTA per SM, so every SM streams
// the same number of weight bytes whatever the number of units (with 128-row units alone, 112 units
// at d_out = 14336 left 40 of 152 SMs idle).  A unit whose steps fall into one CTA's range is
// finished there.  A unit cut between CTAs is owned by the CTA holding its first step, where it is
// the last segment of the range; every other part is the first segment of its CTA's range, so it
// is done early: it stores its raw accumulators (integers times 2^-18, exact in fp32) to its CTA's
// slice of device scratch and bumps the unit's per-warp counter.  The owner waits (bounded) for the
// counter while its own MMAs run, loads the other slices, adds them (an exact sum in any order),
// writes y and resets the counter.  The launch is cooperative, so all parts are resident while the
// owners wait.  Every mbarrier wait is bounded; a wait that gives up raises the device status word
// and all roles drain and exit.
#include <atomic>
#include <cstring>
#include <mutex>

#include "common.cuh"
#include "sqnr_slot.cuh"

namespace cat {
namespace {

constexpr int UM = 128;                      // weight rows per unit (MMA M)
constexpr int KSB = 128;                     // packed bytes per row per K step (256 codes)
constexpr uint32_t kPkStage = UM * KSB;      // 16 KiB packed tile
constexpr int kMaxSP = 8;                    // packed stages (runtime count <= this)
constexpr int kMaxSE = 8;                    // decoded A stages in tensor memory, 64 columns each
constexpr int kThreads = 768;
constexpr int kProd0 = 0, kProd1 = 2;
constexpr int kStageWarp0 = 3;               // warps 3.. stage the token operand at the start
constexpr int kDecWarp0 = 4, kDecWarps = 16, kDecGroups = 4;
constexpr int kEpiWarp0 = 20, kEpiWarps = 4;
constexpr int kTokLoads = 4;                 // token loads in flight per staging thread
constexpr int kGroupBar0 = 4;                // named barriers 4..7: the four warps of a decode group

// Tensor memory: accumulator (group g, buffer b) at column (b * kDecGroups + g) * NTOK, then the
// decoded A stages of 64 columns.  Stage s is only ever used by group s % kDecGroups, and packed
// stage ps only by group ps % kDecGroups (both counts are multiples of the group count): every
// mbarrier phase a group waits for is then the one after the phase it last saw.
template <int NTOK>
struct TmemPlan {
  static constexpr uint32_t kAccCols = 2u * kDecGroups * NTOK;
  // two stages per group where they fit (a group decodes its next step while the MMAs of the last
  // one run), else one
  static constexpr int kSE = kAccCols + 64u * 2 * kDecGroups <= 512u ? 2 * kDecGroups : kDecGroups;
  static_assert(kAccCols + 64u * kSE <= 512u && kSE <= kMaxSE, "tensor memory plan");
};
constexpr uint32_t kTmemCols = 512;
constexpr size_t kSmemBudget = 220 * 1024;

// Partial accumulators of the non-owner parts of cut units: slice (slot, CTA) holds [NTOK <= 32][128]
// floats (a CTA is a non-owner part only of the first unit of its range); counters per (slot, unit,
// epilogue warp).  Slots are handed out round robin per launch.
constexpr int kDecSlots = 2;
constexpr int kDecMaxGrid = 192;
constexpr int kDecMaxUnits = 4096;
__device__ float4 g_dec_part[kDecSlots][kDecMaxGrid][32][UM / 4];
__device__ uint32_t g_dec_cnt[kDecSlots][kDecMaxUnits][kEpiWarps];

// Bound of the pipeline waits (ns); kWaitLimitNs unless a test shortens it (cat_set_wait_limit_ns).
__device__ uint64_t g_dec_wait_limit = kWaitLimitNs;

__device__ __forceinline__ uint32_t ld_acquire_u32(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Range of (unit, K step) steps of CTA c out of g: [s0, s1).  split: equal cuts of all T steps;
// otherwise whole units, contiguous.
__host__ __device__ __forceinline__ int range_begin(int c, int g, int units, int num_ks, bool split) {
  if (split) return (int)((int64_t)c * units * num_ks / g);
  return (int)((int64_t)c * units / g) * num_ks;
}
// The CTA whose range holds step s (split mode): the largest c with range_begin(c) <= s.
__device__ __forceinline__ int cta_of_step(int s, int g, int total) {
  return (int)(((int64_t)(s + 1) * g + total - 1) / total) - 1;
}

struct DecBars {
  uint64_t p_full[kMaxSP], p_empty[kMaxSP], empty[kMaxSE], acc_full[2], acc_empty[2], tok_ready, mma_done;
  f32x2 sums[4][2];                            // SQNR sums of the four epilogue warps
  uint32_t tmem_addr;
  int abort;
};

#define DEC_TMEM_ST32(taddr, v)                                                                                 \
  asm volatile("tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16," \
               "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),                   \
               "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]),      \
               "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15]), "r"(v[16]),          \
               "r"(v[17]), "r"(v[18]), "r"(v[19]), "r"(v[20]), "r"(v[21]), "r"(v[22]), "r"(v[23]), "r"(v[24]),         \
               "r"(v[25]), "r"(v[26]), "r"(v[27]), "r"(v[28]), "r"(v[29]), "r"(v[30]), "r"(v[31])                     \
               : "memory")

#define DEC_TMEM_LD16(taddr, r)                                                                                \
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];" \
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),      \
                 "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]) \
               : "r"(taddr))

__device__ __forceinline__ void dec_tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// Named barrier over the 128 threads of a decode group; true on every thread if pred is true on any.
__device__ __forceinline__ bool group_barrier_any(int id, bool pred) {
  uint32_t r;
  asm volatile("{ .reg .pred q, p; setp.ne.u32 q, %1, 0; bar.red.or.pred p, %2, 128, q; selp.u32 %0, 1, 0, p; }"
               : "=r"(r)
               : "r"((uint32_t)pred), "r"(id)
               : "memory");
  return r != 0;
}

__device__ __forceinline__ void dec_mma_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                           uint32_t accumulate) {
  asm volatile(
      "{ .reg .pred p; setp.ne.b32 p, %4, 0; "
      "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], [%1], %2, %3, p; }" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Bytes of the resident token operand: one [NTOK rows x 128 B] block per 128-code slab.
__host__ __device__ constexpr size_t tok_bytes(int ntok, int num_ks) { return (size_t)num_ks * 2 * ntok * 128; }

template <int NTOK, bool SPLIT>
__global__ void __launch_bounds__(kThreads, 1)
    w4a4_gemm_decode_tc_kernel(const __grid_constant__ CUtensorMap tmW, const uint8_t* __restrict__ xq,
                               const float* __restrict__ sx, const float* __restrict__ sw, int n, int d_in, int d_out,
                               int sp, float* __restrict__ y, int32_t* __restrict__ acc_out,
                               const float* __restrict__ y_ref, double* __restrict__ sums3, int sqnr_slot,
                               int part_slot, uint32_t* __restrict__ status) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int row_bytes = d_in / 2;
  const int num_ks = (row_bytes + KSB - 1) / KSB;
  const int num_units = (d_out + UM - 1) / UM;
  const int total = num_units * num_ks;
  const int s0 = range_begin(blockIdx.x, gridDim.x, num_units, num_ks, SPLIT);
  const int s1 = range_begin(blockIdx.x + 1, gridDim.x, num_units, num_ks, SPLIT);
  constexpr int kSE = TmemPlan<NTOK>::kSE;
  constexpr uint32_t kAStage0 = TmemPlan<NTOK>::kAccCols;
  uint8_t* bst = smem;                                            // tokens, E4M3
  uint8_t* pk = smem + tok_bytes(NTOK, num_ks);                   // sp x 16 KiB packed weight tiles
  DecBars* bars = reinterpret_cast<DecBars*>(pk + (size_t)sp * kPkStage);
  float* sxs = reinterpret_cast<float*>(bars + 1);                // NTOK token steps
  volatile int* abort_flag = &bars->abort;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint64_t lim = g_dec_wait_limit;

  if (tid == 0) {
    for (int s = 0; s < sp; ++s) {
      mbar_init(&bars->p_full[s], 1);
      mbar_init(&bars->p_empty[s], kDecWarps / kDecGroups);   // the decode group of that K step
    }
    for (int s = 0; s < kSE; ++s) mbar_init(&bars->empty[s], 1);
    for (int b = 0; b < 2; ++b) {
      mbar_init(&bars->acc_full[b], kDecGroups);  // every group commits once per segment
      mbar_init(&bars->acc_empty[b], kEpiWarps);
    }
    mbar_init(&bars->tok_ready, kThreads / 32 - kStageWarp0);
    mbar_init(&bars->mma_done, kDecGroups);
    bars->abort = 0;
    fence_mbar_init();
  }
  pdl_wait_then_release();                        // nothing global or in tensor memory before this
  if (warp == 0) tmem_alloc(&bars->tmem_addr, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem_addr;

  if (warp >= kStageWarp0) {
    // resident token operand, staged by warps 3.. while the weight tiles start to stream (all of a
    // thread's loads in flight at once: the first MMA waits for the whole operand): slab a (codes
    // 128a .. 128a+127) of token t at a*NTOK*128 + t*128, 16-byte chunk c at c ^ (t % 8); tokens >= n
    // and codes >= d_in are zero
    // Only the K steps of this CTA's range are staged: with fewer steps than a row has, they are the
    // num_ks-periodic run starting at s0 % num_ks.  Item e = 16-byte chunk c of token t's packed row
    // (e = t * row_chunks + c); (t, c) advance incrementally, with no division inside the loops.
    const int span = s1 - s0, ks_lo = s0 % num_ks;
    const int row_chunks = 8 * num_ks;                            // 16-byte chunks per (padded) packed row
    const int st = tid - kStageWarp0 * 32, nst = kThreads - kStageWarp0 * 32;
    const float sx_pre = (st < NTOK && st < n) ? sx[st] * kAccScale : 0.f;   // loaded beside the token rows
    const int items = NTOK * row_chunks;
    const int step_t = nst / row_chunks, step_c = nst % row_chunks;
    int t_cur = st / row_chunks, c_cur = st % row_chunks;
    auto needed = [&](int c) {
      if (!SPLIT) return true;
      int dk = (c >> 3) - ks_lo;
      if (dk < 0) dk += num_ks;
      return span >= num_ks || dk < span;
    };
    for (int e0 = st; e0 < items; e0 += kTokLoads * nst) {
      uint4 w[kTokLoads];
      int tc[kTokLoads];                                          // t << 16 | c of each item, -1 past the end
#pragma unroll
      for (int q = 0; q < kTokLoads; ++q) {
        const int e = e0 + q * nst;
        const int t = t_cur, c = c_cur;
        tc[q] = e < items ? (t << 16 | c) : -1;
        const int off = c * 16;                                   // packed byte offset in the row
        w[q] = make_uint4(0u, 0u, 0u, 0u);
        if (e < items && t < n && off < row_bytes && needed(c))
          w[q] = *reinterpret_cast<const uint4*>(xq + (int64_t)t * row_bytes + off);
        c_cur += step_c;
        t_cur += step_t;
        if (c_cur >= row_chunks) {
          c_cur -= row_chunks;
          ++t_cur;
        }
      }
#pragma unroll
      for (int q = 0; q < kTokLoads; ++q) {
        if (tc[q] < 0) break;
        const int t = tc[q] >> 16, c = tc[q] & 0xFFFF;
        if (!needed(c)) continue;
        const int a = c >> 2, j = c & 3;                          // 64-byte slab a, 16-byte chunk j in it
        uint8_t* dst = bst + (size_t)a * NTOK * 128 + t * 128;
        const int swz = t & 7;
        *reinterpret_cast<uint4*>(dst + (((2 * j) ^ swz) << 4)) =
            make_uint4(sm4_lo(w[q].x), sm4_hi(w[q].x), sm4_lo(w[q].y), sm4_hi(w[q].y));
        *reinterpret_cast<uint4*>(dst + (((2 * j + 1) ^ swz) << 4)) =
            make_uint4(sm4_lo(w[q].z), sm4_hi(w[q].z), sm4_lo(w[q].w), sm4_hi(w[q].w));
      }
    }
    if (st < NTOK) sxs[st] = sx_pre;
    fence_proxy_async_smem();                                     // the MMA reads the tokens via the async proxy
    __syncwarp();
    if (lane == 0) mbar_arrive(&bars->tok_ready);
  }

  if (warp == kProd0 || warp == kProd1) {
    // ---------------------------------------------------------------- TMA producers (alternate K steps)
    if (lane == 0) {
      const uint32_t me = warp == kProd0 ? 0u : 1u;
      if (me == 0) prefetch_tensormap(&tmW);
      // it = the CTA-local step index (step s0 + it of the (unit, K step) sequence)
      uint32_t it = 0, issued_end = 0;                  // this producer issued every K step of its parity below issued_end
      bool ok = true;
      for (int sg = s0; sg < s1 && ok; ++sg, ++it) {
        if ((it & 1u) != me) continue;
        const int u = sg / num_ks, ks = sg % num_ks;
        const uint32_t s = it % sp, use = it / sp;
        if (use > 0 && !(ok = mbar_wait_bounded(&bars->p_empty[s], (use - 1) & 1, abort_flag, __LINE__, lim))) break;
        mbar_arrive_expect_tx(&bars->p_full[s], kPkStage);
        tma_load_2d(pk + s * kPkStage, &tmW, ks * KSB, u * UM, &bars->p_full[s]);
        issued_end = it + 1;
      }
      // loads still in flight land before the CTA exits: only the last sp K steps of the whole walk
      // (`it` steps) have stages that were not reused, so only their barriers still hold the phase
      // to wait for; this producer waits for the ones it issued
      volatile int no_abort = 0;
      for (uint32_t q = it > (uint32_t)sp ? it - sp : 0; q < it && q < issued_end; ++q)
        if ((q & 1u) == me) mbar_wait_bounded(&bars->p_full[q % sp], (q / sp) & 1, &no_abort);
    }
  } else if (warp >= kDecWarp0 && warp < kDecWarp0 + kDecWarps) {
    // ---------------------------------------------------------------- decode + MMA: weight row = TMEM lane
    // Four groups of four warps (one per TMEM lane quadrant) take every fourth step of the CTA's
    // range (group = local step index mod 4, so every stage has one consumer).  A thread decodes its
    // whole 128-byte row (256 codes, 64 TMEM columns); then the group's leader thread issues the
    // step's eight MMAs into the group's own accumulator.  One thread issues an MMA about every 55
    // cycles whatever N is, so four issuers keep the tensor core fed at N = 16; the partial
    // accumulators of a segment (the range's steps of one unit) are added in the epilogue (integers
    // times 2^-18: exact).  Every group commits the segment's accumulator barrier once, with or
    // without steps in it, after waiting for that buffer to be drained.
    const int quad = warp & 3, grp = (warp - kDecWarp0) >> 2;
    const bool leader = quad == 0 && lane == 0;
    const int r = quad * 32 + lane;
    constexpr uint32_t kIdesc = idesc_e4m3_f32(UM, NTOK);
    const uint32_t bbase = smem_u32(bst);
    bool stop = false;
    if (leader) {
      mbar_wait_bounded(&bars->tok_ready, 0, abort_flag, __LINE__, lim);
      tc_fence_after();
    }
    uint32_t seg = 0;
    for (int sb = s0; sb < s1 && !stop; ++seg) {
      const int u = sb / num_ks;
      const int se = min(s1, (u + 1) * num_ks);        // segment [sb, se): the range's steps of unit u
      const uint32_t ab = seg & 1;
      const uint32_t d_acc = tmem + (ab * kDecGroups + grp) * NTOK;
      bool first = true;                                 // the group's first step of the segment
      for (int sg = sb + ((grp - (sb - s0)) % kDecGroups + kDecGroups) % kDecGroups; sg < se; sg += kDecGroups) {
        const uint32_t it = (uint32_t)(sg - s0);         // it % kDecGroups == grp
        const int ks = sg % num_ks;
        const uint32_t ps = it % sp, sa = it % kSE;
        const bool good = mbar_wait_bounded(&bars->p_full[ps], (it / sp) & 1, abort_flag, __LINE__, lim) &&
                          (it < (uint32_t)kSE || mbar_wait_bounded(&bars->empty[sa], ((it / kSE) - 1) & 1, abort_flag, __LINE__, lim));
        if (good) {
          tc_fence_after();
          const uint8_t* prow = pk + ps * kPkStage + r * 128;
#pragma unroll
          for (int half = 0; half < 2; ++half) {
            uint32_t av[32];
#pragma unroll
            for (int jj = 0; jj < 4; ++jj) {  // 16-byte chunk j of the 128-byte row, at j ^ (r % 8)
              const int j = 4 * half + jj;
              const uint4 w = *reinterpret_cast<const uint4*>(prow + ((j ^ (r & 7)) << 4));
              av[8 * jj + 0] = sm4_lo(w.x); av[8 * jj + 1] = sm4_hi(w.x);
              av[8 * jj + 2] = sm4_lo(w.y); av[8 * jj + 3] = sm4_hi(w.y);
              av[8 * jj + 4] = sm4_lo(w.z); av[8 * jj + 5] = sm4_hi(w.z);
              av[8 * jj + 6] = sm4_lo(w.w); av[8 * jj + 7] = sm4_hi(w.w);
            }
            __syncwarp();
            DEC_TMEM_ST32(tmem + ((uint32_t)(quad * 32) << 16) + kAStage0 + 64u * sa + 32u * half, av);
          }
          dec_tmem_st_wait();
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0 && good) mbar_arrive(&bars->p_empty[ps]);
        // the group's four warps have stored the stage (and agree on whether to go on)
        stop = group_barrier_any(kGroupBar0 + grp, *abort_flag != 0);
        if (stop) break;
        if (leader) {
          tc_fence_after();
          if (first && seg >= 2) mbar_wait_bounded(&bars->acc_empty[ab], ((seg >> 1) - 1) & 1, abort_flag, __LINE__, lim);
          tc_fence_after();
          const uint32_t ta = tmem + kAStage0 + 64u * sa;
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) {  // K = 32 codes per MMA: 8 TMEM columns of A; B slab 2ks + kk/4, +32 B
            const uint64_t db = sdesc_kmajor_sw128(bbase + (uint32_t)((2 * ks + (kk >> 2)) * NTOK * 128)) + 2 * (kk & 3);
            dec_mma_ts(d_acc, ta + 8u * kk, db, kIdesc, (first && kk == 0) ? 0u : 1u);
          }
          mma_commit(&bars->empty[sa]);
        }
        first = false;
      }
      if (stop) break;
      if (leader) {
        // a group without steps in this segment still waits for the buffer to be drained before it
        // commits, so its arrivals can never run a phase ahead
        if (first && seg >= 2) mbar_wait_bounded(&bars->acc_empty[ab], ((seg >> 1) - 1) & 1, abort_flag, __LINE__, lim);
        mma_commit(&bars->acc_full[ab]);
      }
      sb = se;
    }
    if (leader) {
      mma_commit(&bars->mma_done);  // all MMAs complete before tensor memory is released
      volatile int no_abort = 0;
      mbar_wait_bounded(&bars->mma_done, 0, &no_abort);
    }
  } else if (warp >= kEpiWarp0) {
    // ---------------------------------------------------------------- epilogue: output channel = TMEM lane
    const int quad = warp & 3;
    const int ch = quad * 32 + lane;                 // channel within the unit
    bool ok = true;
    f32x2 sig = {0.f, 0.f}, err = {0.f, 0.f};      // SQNR sums (Sec. 2, Eq. 1) when y_ref is given
    uint32_t seg = 0;
    for (int sb = s0; sb < s1 && ok; ++seg) {
      const int u = sb / num_ks;
      const int se = min(s1, (u + 1) * num_ks);
      const uint32_t ab = seg & 1;
      const bool whole = !SPLIT || se - sb == num_ks;  // the unit is finished in this CTA
      const int o = u * UM + ch;
      const bool o_ok = o < d_out;
      const float swo = o_ok ? sw[o] : 0.f;
      const int cf = whole ? (int)blockIdx.x : cta_of_step(u * num_ks, gridDim.x, total);
      const int cl = whole ? (int)blockIdx.x : cta_of_step((u + 1) * num_ks - 1, gridDim.x, total);
      const bool owner = cf == (int)blockIdx.x;       // writes the unit's outputs
      // y_ref in flight while the MMAs of the segment run, where this CTA writes the unit
      const bool pre = y_ref && o_ok && owner;
      float yr[NTOK];
#pragma unroll
      for (int t = 0; t < NTOK; ++t) yr[t] = (pre && t < n) ? __ldcs(y_ref + (int64_t)t * d_out + o) : 0.f;
      if (!(ok = mbar_wait_bounded(&bars->acc_full[ab], (seg >> 1) & 1, abort_flag, __LINE__, lim))) break;
      __syncwarp();
      tc_fence_after();
      // the groups with steps in the segment: local steps sb - s0 .. se - s0 - 1, group = step % 4
      const int nact = se - sb < kDecGroups ? se - sb : kDecGroups;
      uint32_t* cnt = &g_dec_cnt[part_slot][u][quad];
      float s_run = 0.f, e_run = 0.f;
      auto emit = [&](int t, float a) {                // y (and acc_out, SQNR terms) of token t
        const float v = a * sxs[t] * swo;              // consecutive o across the warp: coalesced stores
        y[(int64_t)t * d_out + o] = v;
        if (acc_out) acc_out[(int64_t)t * d_out + o] = __float2int_rn(a * kAccScale);
        const float e = yr[t] - v;
        s_run += yr[t] * yr[t];
        e_run += e * e;
      };
      // owner of a cut unit: the other parts ran first in their CTAs; wait for their counts and
      // sum their slices while this segment's MMAs run (16 tokens), or after them (32)
      constexpr bool kEarly = SPLIT && NTOK == 16;
      float ext[kEarly ? NTOK : 1];
      auto wait_parts = [&]() -> bool {              // warp-uniform
        uint32_t good = 1u;
        if (lane == 0) {
          const uint64_t t0 = globaltimer_ns();
          for (uint32_t it = 0; ld_acquire_u32(cnt) < (uint32_t)(cl - cf); ++it) {
            __nanosleep(32);
            if ((it & 63u) == 63u && (*abort_flag || globaltimer_ns() - t0 > lim)) {
              if (*abort_flag == 0) *abort_flag = __LINE__;
              good = 0u;
              break;
            }
          }
          if (good) *cnt = 0u;                         // every part has counted: clean for the next launch
        }
        good = __shfl_sync(0xFFFFFFFFu, good, 0);
        __threadfence();
        return good != 0u;
      };
      auto slice_of = [&](int c) { return reinterpret_cast<const float*>(&g_dec_part[part_slot][c][0][0]) + ch; };
      if (kEarly && !whole && owner) {
        if (!(ok = wait_parts())) break;
#pragma unroll
        for (int t = 0; t < (kEarly ? NTOK : 1); ++t) ext[t] = 0.f;
        for (int c = cf + 1; c <= cl; ++c) {
          const float* src = slice_of(c);
#pragma unroll
          for (int t = 0; t < (kEarly ? NTOK : 1); ++t) ext[t] += __ldcg(src + t * UM);  // exact in any order
        }
      }
      if (!(ok = mbar_wait_bounded(&bars->acc_full[ab], (seg >> 1) & 1, abort_flag, __LINE__, lim))) break;
      __syncwarp();
      tc_fence_after();
      if (!kEarly && !whole && owner && !(ok = wait_parts())) break;
      float* my_slice = reinterpret_cast<float*>(&g_dec_part[part_slot][blockIdx.x][0][0]) + ch;
#pragma unroll
      for (int c = 0; c < NTOK / 16; ++c) {          // 16 accumulator columns at a time
        float acc[16];
#pragma unroll
        for (int j = 0; j < 16; ++j) acc[j] = 0.f;
        for (int i = 0; i < nact; ++i) {
          const int g = (sb - s0 + i) % kDecGroups;
          uint32_t part[16];
          DEC_TMEM_LD16(tmem + ((uint32_t)(quad * 32) << 16) + (ab * kDecGroups + g) * NTOK + 16u * c, part);
          tmem_ld_wait();
#pragma unroll
          for (int j = 0; j < 16; ++j) acc[j] += __uint_as_float(part[j]);  // integers times 2^-18: exact
        }
        if (c == NTOK / 16 - 1) {
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&bars->acc_empty[ab]);
        }
        if (owner) {
          if (!whole) {
            if constexpr (kEarly) {
#pragma unroll
              for (int j = 0; j < 16; ++j) acc[j] += ext[16 * c + j];
            } else {
              for (int p = cf + 1; p <= cl; ++p) {
                const float* src = slice_of(p);
#pragma unroll
                for (int j = 0; j < 16; ++j) acc[j] += __ldcg(src + (16 * c + j) * UM);
              }
            }
          }
          if (o_ok) {
#pragma unroll
            for (int j = 0; j < 16; ++j)
              if (16 * c + j < n) emit(16 * c + j, acc[j]);
          }
        } else {
#pragma unroll
          for (int j = 0; j < 16; ++j) __stcg(my_slice + (16 * c + j) * UM, acc[j]);
        }
      }
      if (!owner) {                                    // a non-owner part: stored; count it
        __threadfence();
        __syncwarp();
        if (lane == 0) atomicAdd(cnt, 1u);
      }
      sig = f2_add(sig, s_run);
      err = f2_add(err, e_run);
      sb = se;
    }
    if (y_ref) {
      // the four warps' sums meet in shared memory; one warp hands the CTA's pair to the slot
      sig = f2_warp_sum(sig);
      err = f2_warp_sum(err);
      if (lane == 0) {
        bars->sums[quad][0] = sig;
        bars->sums[quad][1] = err;
      }
      asm volatile("bar.sync 2, 128;" ::: "memory");  // this CTA's four epilogue warps have written theirs
      if (warp == kEpiWarp0) {
        const f32x2 s_cta = f2_add(f2_add(bars->sums[0][0], bars->sums[1][0]), f2_add(bars->sums[2][0], bars->sums[3][0]));
        const f32x2 e_cta = f2_add(f2_add(bars->sums[0][1], bars->sums[1][1]), f2_add(bars->sums[2][1], bars->sums[3][1]));
        sqnr_cta_done(sqnr_slot, s_cta, e_cta, sums3);
      }
    }
  }

  __syncthreads();
  if (bars->abort && tid == 0) report(status, timeout_bits(kWhereGemmDecode, bars->abort));
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

size_t smem_bytes(int ntok, int num_ks, int sp) {
  return 1024 + tok_bytes(ntok, num_ks) + (size_t)sp * kPkStage + sizeof(DecBars) + 32 * sizeof(float);
}

// Whether one CTA per SM of the kernel is resident at once on this device under a cooperative launch
// (checked once per token count; the grid never exceeds the SM count).
template <int NTOK>
bool coop_fits(size_t smem) {
  static int ok = -1;
  static std::mutex mu;
  std::lock_guard<std::mutex> lock(mu);
  if (ok < 0) {
    int dev = 0, coop = 0, blocks = 0;
    ok = cudaGetDevice(&dev) == cudaSuccess &&
         cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, dev) == cudaSuccess && coop &&
         cudaFuncSetAttribute(w4a4_gemm_decode_tc_kernel<NTOK, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)kSmemBudget + 4096) == cudaSuccess &&
         cudaOccupancyMaxActiveBlocksPerMultiprocessor(&blocks, w4a4_gemm_decode_tc_kernel<NTOK, true>, kThreads,
                                                       kSmemBudget + 4096) == cudaSuccess &&
         blocks >= 1;
    cudaGetLastError();
  }
  (void)smem;
  return ok == 1;
}

template <int NTOK>
cudaError_t launch_ntok(const uint8_t* xq, const float* sx, const uint8_t* wq, const float* sw, int64_t n,
                        int64_t d_in, int64_t d_out, float* y, int32_t* acc_out, const float* y_ref, double* sums3,
                        uint32_t* status, int sp, cudaStream_t stream) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return cudaErrorNotSupported;
  const int64_t row_bytes = d_in / 2;
  CUtensorMap map;
  memset(&map, 0, sizeof(map));
  cuuint64_t dims[2] = {(cuuint64_t)row_bytes, (cuuint64_t)d_out};
  cuuint64_t strides[1] = {(cuuint64_t)row_bytes};
  cuuint32_t box[2] = {(cuuint32_t)KSB, (cuuint32_t)UM};
  cuuint32_t estr[2] = {1, 1};
  if (fn(&map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<uint8_t*>(wq), dims, strides, box, estr,
         CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  const int num_ks = (int)((row_bytes + KSB - 1) / KSB);
  const size_t smem = smem_bytes(NTOK, num_ks, sp);
  static std::mutex mu;
  static size_t configured = 0;
  {
    std::lock_guard<std::mutex> lock(mu);
    if (smem > configured) {
      cudaError_t e = cudaFuncSetAttribute(w4a4_gemm_decode_tc_kernel<NTOK, false>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (e == cudaSuccess)
        e = cudaFuncSetAttribute(w4a4_gemm_decode_tc_kernel<NTOK, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)smem);
      if (e != cudaSuccess) return e;
      configured = smem;
    }
  }
  const int64_t units = (d_out + UM - 1) / UM;
  const int64_t sms = num_sms() < kDecMaxGrid ? num_sms() : kDecMaxGrid;
  // Stream-K over all (unit, K step) steps when there are more units than SMs: every CTA's range is
  // then at least one unit long, so no CTA lies inside a unit and every part of a cut unit other
  // than the owner's is the head of its CTA's range, done early.  With fewer units than SMs a range
  // would be shorter than a unit; CTAs inside a unit finish together with the unit's owner, and the
  // exchange through global memory then sits on the tail (measured at 16 tokens, 4096 -> 14336:
  // 15.8 us on 152 CTAs against 12.8 us for whole units on 112).  Whole units per CTA in that case.
  const int split = units > sms && units <= kDecMaxUnits && coop_fits<NTOK>(smem) ? 1 : 0;
  const int64_t work = split ? units * num_ks : units;
  const unsigned grid = (unsigned)(work < sms ? work : sms);
  if (grid > (unsigned)kSqnrMaxCtas) return cudaErrorInvalidConfiguration;
  const int slot = y_ref ? next_sqnr_slot() : 0;
  static std::atomic<unsigned> next_part{0};
  const int part_slot = split ? (int)(next_part.fetch_add(1, std::memory_order_relaxed) % kDecSlots) : 0;
  note_launch();
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = dim3(grid, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attrs[2] = {pdl_attr(), {}};
  attrs[1].id = cudaLaunchAttributeCooperative;       // the owners of cut units wait for the other parts
  attrs[1].val.cooperative = 1;
  cfg.attrs = attrs;
  cfg.numAttrs = split ? 2 : 1;
  if (split)
    return cudaLaunchKernelEx(&cfg, w4a4_gemm_decode_tc_kernel<NTOK, true>, map, xq, sx, sw, (int)n, (int)d_in,
                              (int)d_out, sp, y, acc_out, y_ref, sums3, slot, part_slot, status);
  return cudaLaunchKernelEx(&cfg, w4a4_gemm_decode_tc_kernel<NTOK, false>, map, xq, sx, sw, (int)n, (int)d_in,
                            (int)d_out, sp, y, acc_out, y_ref, sums3, slot, part_slot, status);
}

}  // namespace

cudaError_t set_decode_wait_limit(uint64_t ns) {
  return cudaMemcpyToSymbol(g_dec_wait_limit, &ns, sizeof(ns));
}

// Packed stages that fit beside the resident tokens; 0 when this kernel does not apply.
int decode_tc_stages(int64_t n, int64_t d_in) {
  if (n < 1 || n > 32) return 0;
  const int ntok = n <= 16 ? 16 : 32;
  const int num_ks = (int)((d_in / 2 + KSB - 1) / KSB);
  const size_t fixed = smem_bytes(ntok, num_ks, 0);
  if (fixed >= kSmemBudget) return 0;
  int sp = (int)((kSmemBudget - fixed) / kPkStage);
  if (sp > kMaxSP) sp = kMaxSP;
  sp -= sp % kDecGroups;                      // a multiple of the decode groups (see TmemPlan)
  return sp >= kDecGroups ? sp : 0;
}

// y_ref != nullptr: the epilogue also forms the SQNR sums of y against y_ref and writes
// sums3 = {sum y_ref^2, sum (y_ref - y)^2, dB} (sums3 needs no zeroing).
cudaError_t launch_w4a4_gemm_decode_tc(const uint8_t* xq, const float* sx, const uint8_t* wq, const float* sw,
                                       int64_t n, int64_t d_in, int64_t d_out, float* y, int32_t* acc_out,
                                       const float* y_ref, double* sums3, uint32_t* status, cudaStream_t stream) {
  const int sp = decode_tc_stages(n, d_in);
  if (sp == 0) return cudaErrorInvalidValue;
  if (n <= 16) return launch_ntok<16>(xq, sx, wq, sw, n, d_in, d_out, y, acc_out, y_ref, sums3, status, sp, stream);
  return launch_ntok<32>(xq, sx, wq, sw, n, d_in, d_out, y, acc_out, y_ref, sums3, status, sp, stream);
}

}  // namespace cat
