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
// Two operand formats share this kernel (template parameter E8):
//   * byte codes (E8): the codes are stored one E4M3 byte each, so TMA loads them into 128B-swizzled
//     shared memory as they are and the pair MMAs read both operands there -- no decode warps.  Tiles
//     are 256 x 128 (four 48 KB stages) or 256 x 256 (NB = 256: three 64 KB stages, the two
//     accumulators filling tensor memory), chosen per shape by e8_wide_tiles;
//   * SM4x8 codes: the packed codes are decoded in the kernel, as described below (tiles 256 x 128).
// Both walk the tiles in bands of kBandM token tiles, and both split a last wave that is at most half
// full along K.
//
// Data path of the SM4x8 kernel.  The tensor cores read their shared-memory operands on a path of
// their own (their rate does not change under concurrent LSU shared-memory traffic) and an MMA with
// A in tensor
// memory runs at ~93% of peak, while the decode of the packed B operand into shared memory is the
// costliest step.  So two SMs share each output tile (a cluster pair and tcgen05.mma.cta_group::2):
//   * the pair tile is 256 tokens x 128 channels; each CTA owns 128 tokens (the A rows, in its own
//     tensor memory) and 64 channels (half of B, in its own shared memory), so every decoded B row
//     serves 256 tokens and each SM decodes half the B rows a single-SM tile would need;
//   * each K step covers 256 codes: packed A (128 x 128 B) and B (64 x 128 B) tiles arrive by TMA
//     with a 128-byte swizzle, from two issuing warps (one per operand);
//   * A is decoded one row per thread and written to tensor memory; B is decoded into 128B-swizzled
//     shared memory; two groups of decode warps take alternate K steps;
//   * the decode warps of both CTAs arrive on the even CTA's stage barrier; its MMA thread issues the
//     pair MMAs and multicasts the completions (stage free, accumulator full) to both CTAs;
//   * four decoded stages: the decode of a K step takes several times longer (latency: loads, fences,
//     tensor-memory stores) than its MMAs, so four steps are decoded while one is multiplied;
//   * the accumulator is double-buffered (2 x 128 columns), so the epilogue of one tile overlaps the
//     MMAs of the next; each CTA drains its own 128 rows.
//
// Persistent CTA pairs (one CTA per SM, 512 threads each):
//   warp 0       TMA producer of A tiles and TMEM allocator
//   warp 1       lane 0 of the even CTA issues tcgen05.mma (8 x K=32 per K step) and commits
//   warps 1, 3   lane 0 of the odd CTA forwards its decode groups' stage readiness to the even CTA
//   warp 2       TMA producer of B tiles
//   warps 4..7   epilogue: tcgen05.ld of their TMEM lane quadrant, scale, stage the rows in
//                128B-swizzled shared memory, TMA store (plain stores when the TMA rules don't hold)
//   warps 8..15  decode, two groups of four warps taking alternate K steps: a whole A row per
//                thread, and B chunks
// TMEM: accumulators at columns [0, 128) and [128, 256), A stages at 256 + 64 s.  A last wave that is at
// most half full is split along K (see the split-tail section below).  Every wait is bounded; a wait
// that gives up raises the device status word and all roles drain and exit.
#include <cstring>
#include <mutex>
#include <type_traits>

#include "common.cuh"
#include "sqnr_slot.cuh"

namespace cat {
namespace {

constexpr int BM = 128;                    // tokens per CTA (256 per pair)
constexpr int BN = 128;                    // channels per pair tile
constexpr int BNC = BN / 2;                // channels (B rows) held by each CTA
constexpr int BK = 256;
constexpr int BKP = BK / 2;                 // packed bytes per row per K step (128)
constexpr int SP = 3;                       // packed stages (TMA)
constexpr int SE = 4;                       // decoded stages (A in TMEM, B in shared memory)
constexpr uint32_t kPackedA = BM * BKP;     // 16 KiB
constexpr uint32_t kPackedB = BNC * BKP;    // 8 KiB
constexpr uint32_t kPackedStage = kPackedA + kPackedB;
constexpr uint32_t kAtomB = BNC * 128;      // one 128-code K atom of decoded B (64 rows x 128 B)
constexpr uint32_t kStageB = BNC * BK;      // 16 KiB of E4M3 per stage (two atoms)
constexpr int kThreads = 512;
constexpr int kProdA = 0, kMmaWarp = 1, kProdB = 2, kFwdWarp = 3;
constexpr int kDecWarp0 = 8, kGroupWarps = 4, kGroupThreads = kGroupWarps * 32;  // two decode groups
constexpr int kDecGroups = 2;                // the groups take alternate K steps
// The packed stages are not a multiple of the groups, so one packed stage is consumed by both groups
// in turn.  Each group therefore gets its own full-barrier per packed stage: a barrier's phases are
// then consumed by one group only, which has seen the previous phase complete before it waits for
// the next one.  (With one barrier per stage, a group could wait for a phase two ahead of the
// barrier, when the other group's load is late, and the parity wait would return at once.)
// Loads into barrier (g, s) come every kPFullPeriod K steps.
constexpr int kPFullPeriod = SP % kDecGroups == 0 ? SP : SP * kDecGroups;
constexpr int kEpiWarp0 = 4, kEpiWarps = 4;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kAccCols = 2 * BN;       // two accumulators
constexpr uint32_t kEpiStage = 32 * 32 * 4;                 // 32 rows x 32 fp32 columns, 4 KiB
constexpr int kEpiBufs = 2;                                  // TMA-store staging buffers per epilogue warp
constexpr uint32_t kPkOffset = SE * kStageB;                 // after the decoded B stages
constexpr uint32_t kBarBytes = 1024;                         // room reserved for the barrier block
// Byte codes (E8): one E4M3 byte per code (sign << 7 | magnitude, i.e. q * 2^-9), loaded by TMA as
// they are and multiplied from shared memory: no decode warps, no packed ring, and SE stages of
// A (128 rows x 256 B) and B (64 rows x 256 B).
constexpr uint32_t kAtomA8 = BM * 128;      // one 128-code K atom of A (128 rows x 128 B)
constexpr uint32_t kStageA8 = BM * BK;      // 32 KiB
constexpr uint32_t kStage8 = kStageA8 + kStageB;   // 48 KiB
constexpr int kStages8 = 4;                 // byte-code stages
constexpr int kEpiBufs8 = 1;                // byte codes: y and y_ref staging buffers per epilogue warp
// Shared memory and tensor memory of the two operand formats.  The byte-code stages leave room for
// one y and one y_ref staging buffer per epilogue warp, and the output-channel steps of a chunk go
// through registers instead of shared memory.
template <bool E8, int NB = BN>
struct GemmLayout {
  // byte codes at NB = 256: three 64 KB stages; NB = 128: kStages8 stages of 48 KB
  static constexpr int S = E8 ? (NB == 256 ? 3 : kStages8) : SE;   // operand stages the MMA consumes
  static constexpr uint32_t kStageOp = kStageA8 + (uint32_t)(NB / 2) * BK;
  static constexpr int EB = E8 ? kEpiBufs8 : kEpiBufs;   // y staging buffers per epilogue warp
  static constexpr int RB = E8 ? kEpiBufs8 : kEpiBufs;   // y_ref staging buffers per epilogue warp
  static constexpr uint32_t kOperands = E8 ? S * kStageOp : kPkOffset + SP * kPackedStage;
  static constexpr uint32_t kEpiOffset = kOperands;
  static constexpr uint32_t kRefOffset = kEpiOffset + kEpiWarps * EB * kEpiStage;   // y_ref tiles (SQNR)
  static constexpr uint32_t kScaleOffset = kRefOffset + kEpiWarps * RB * kEpiStage;
  static constexpr uint32_t kBarOffset = kScaleOffset + (E8 ? 0u : kEpiWarps * NB * 4);
  static constexpr uint32_t kBarRoom = E8 ? 512u : kBarBytes;
  static constexpr size_t kSmemBytes = kBarOffset + kBarRoom + 1024;  // + barriers + alignment slack
  static constexpr uint32_t kTmem = E8 ? 2 * NB : kTmemCols;   // E8: the two accumulators
  static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");
  static_assert(S <= SE && EB <= kEpiBufs && RB <= kEpiBufs, "barrier arrays");
  static_assert(E8 || S % kDecGroups == 0, "a decode group's steps keep to the stages of one parity");
  static_assert((E8 && (NB == 128 || NB == 256)) || NB == BN, "tile widths");
  static_assert(kStageOp % 1024 == 0, "128B-swizzle alignment");
};
static_assert(kAccCols + SE * 64 <= kTmemCols, "tensor memory budget");
static_assert(kPackedStage % 1024 == 0 && kAtomB % 1024 == 0 && kPackedA % 1024 == 0, "128B-swizzle alignment");
static_assert(kStage8 % 1024 == 0 && kAtomA8 % 1024 == 0 && kStageA8 % 1024 == 0, "128B-swizzle alignment");
static_assert((BNC * 8) % kGroupThreads == 0, "B chunks per decode thread");


struct Bars {
  uint64_t p_full[kDecGroups][SP], p_empty[SP], full[SE], ready[SE], empty[SE], acc_full[2], acc_empty[2], mma_done;
  uint64_t ref_full[kEpiWarps][kEpiBufs];      // y_ref tile loads of each epilogue warp
  uint32_t fwd_word[SE];                         // even CTA: targets of the odd CTA's st.async per stage
  uint32_t tmem_addr;
  int abort;
  f32x2 sums[kEpiWarps][2];                      // SQNR sums of the epilogue warps
};
static_assert(sizeof(Bars) <= GemmLayout<false>::kBarRoom && sizeof(Bars) <= GemmLayout<true>::kBarRoom &&
                  sizeof(Bars) <= GemmLayout<true, 256>::kBarRoom,
              "barrier block must fit its reserved room");

// ---- tensor-memory stores and the TMA store path -------------------------------------------
#define CAT_TMEM_ST32(taddr, v)                                                                                 \
  asm volatile("tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16," \
               "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),                   \
               "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]),      \
               "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15]), "r"(v[16]),          \
               "r"(v[17]), "r"(v[18]), "r"(v[19]), "r"(v[20]), "r"(v[21]), "r"(v[22]), "r"(v[23]), "r"(v[24]),         \
               "r"(v[25]), "r"(v[26]), "r"(v[27]), "r"(v[28]), "r"(v[29]), "r"(v[30]), "r"(v[31])                     \
               : "memory")

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// arrive on the mbarrier at the same shared-memory offset in CTA `rank` of the cluster
__device__ __forceinline__ void mbar_arrive_cluster(uint64_t* bar, uint32_t rank) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(bar)), "r"(rank));
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(remote) : "memory");
}
// Asynchronous 4-byte store into CTA `rank`'s shared memory whose completion is counted (complete_tx,
// release at cluster scope) on that CTA's mbarrier; the issuing thread does not wait for it.
__device__ __forceinline__ void st_async_signal(uint32_t* word, uint64_t* bar, uint32_t rank) {
  uint32_t rw, rb;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(rw) : "r"(smem_u32(word)), "r"(rank));
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(rb) : "r"(smem_u32(bar)), "r"(rank));
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.u32 [%0], %1, [%2];" ::"r"(rw), "r"(1u), "r"(rb)
               : "memory");
}
__device__ __forceinline__ void tmem_alloc_pair(uint32_t* dst, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(dst)), "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
// the pair MMA: D (both CTAs' TMEM) (+)= A (both CTAs' TMEM) x B (both CTAs' shared memory)
__device__ __forceinline__ void mma_pair_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{ .reg .pred p; setp.ne.b32 p, %4, 0; "
      "tcgen05.mma.cta_group::2.kind::f8f6f4 [%0], [%1], %2, %3, p; }" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// the pair MMA with both operands in shared memory (each CTA: its 128 A rows and its half of B)
__device__ __forceinline__ void mma_pair_ss(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{ .reg .pred p; setp.ne.b32 p, %4, 0; "
      "tcgen05.mma.cta_group::2.kind::f8f6f4 [%0], %1, %2, %3, p; }" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// arrive once on the mbarrier at this offset in both CTAs when the pair MMAs issued so far complete
__device__ __forceinline__ void mma_commit_pair(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(
                   smem_u32(bar)),
               "h"((uint16_t)3)
               : "memory");
}

__device__ __forceinline__ void tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, const void* smem_src, int32_t x, int32_t y) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(x), "r"(y), "r"(smem_u32(smem_src))
               : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read_le1() { asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read_all() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// ---- the last wave's tiles split along K -----------------------------------------------------
// With T pair tiles on P pairs the last wave holds T mod P tiles and the other pairs idle through
// it.  When it is at most half full, each of its tiles is split into S parts of its K steps (S a
// power of two, at most 16), one part per pair.  Every part writes its raw accumulators to its own
// slice of device scratch with plain stores (float32 atomics from many SMs onto one tile are an
// order of magnitude slower), waits until all S parts of the tile have arrived (bounded; the launch
// is cooperative, so all parts are resident), and then finishes NB / S of the tile's channels:
// the sum over the parts (exact in any order: integer multiples of 2^-18 below 2^6 in magnitude),
// the scaling, y, acc_out and the SQNR sums.  Counters are per (tile, CTA, epilogue warp); the last
// part to finish sets them back to zero.  Slots of this scratch are handed out round robin per launch.
constexpr int kSplitSlots = 2;
constexpr int kMaxSplitTiles = 38;            // half a wave of 76 pairs
constexpr int kMaxSplitUnits = 80;            // tail tiles x parts x NB / 128 <= pairs
constexpr int kMaxSplit = 16;
// Per slot: [part][channel/4][row] float4 slices of NB / 4 x 2 BM, room for kMaxSplitUnits 128-wide parts
// (half as many 256-wide ones).
constexpr size_t kSplitSlotF4 = (size_t)kMaxSplitUnits * (BN / 4) * (2 * BM);
__device__ float4 g_split_part[kSplitSlots * kSplitSlotF4];
__device__ uint32_t g_split_cnt[kSplitSlots][kMaxSplitTiles][2][kEpiWarps][2];   // arrived, finished

__device__ __forceinline__ uint32_t ld_acquire_gpu(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Tile t of the launch -> (token tile m, channel tile nn).  Tiles go in bands of kBandM token tiles,
// m fastest within a band, so the tiles a wave of pairs works on at once cover ~kBandM token tiles by
// a few channel tiles rather than every token tile by ~2 channel tiles: at 8192 x 8192 x 28672 on 76
// pairs, ~35 MB of operand rows per wave instead of ~70 MB, all read from DRAM again each wave.
constexpr int kBandM = 8;
__device__ __forceinline__ void tile_coords(int t, int num_m, int num_n, int* m, int* nn) {
  const int m0 = (t / (kBandM * num_n)) * kBandM;     // the band's first token tile
  const int bm = min(kBandM, num_m - m0);             // token tiles in this band (fewer in the last)
  const int r = t - m0 * num_n;                       // the tile's index within its band
  *m = m0 + r % bm;
  *nn = r / bm;
}

// Work unit u of the launch: the n_split = tail x split parts come first (part u % split of tail
// tile num_full + u / split, on pairs 0 .. n_split - 1, one each), then the whole tiles (tile
// u - n_split).  All parts run at the same time, as their pairs' first units, and each part's share
// of the tile is finished while the MMAs of its pair's first whole tile run (the epilogue is idle
// then).
struct Unit {
  int tile, k0, k1, part;                     // part < 0: the whole tile
};
__device__ __forceinline__ Unit unit_at(int u, int num_full, int split, int num_k, int n_split) {
  if (u >= n_split) return {u - n_split, 0, num_k, -1};
  const int part = u % split;
  return {num_full + u / split, part * num_k / split, (part + 1) * num_k / split, part};
}

template <bool E8, int NB>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    w4a4_gemm_tc_kernel(const __grid_constant__ CUtensorMap tmY, const __grid_constant__ CUtensorMap tmA,
                        const __grid_constant__ CUtensorMap tmB, const __grid_constant__ CUtensorMap tmR,
                        const float* __restrict__ y_ref, double* __restrict__ sums3, int sqnr_slot,
                        const float* __restrict__ sx,
                        const float* __restrict__ sw, int n, int d_in, int d_out, float* __restrict__ y,
                        int32_t* __restrict__ acc_out, int use_tma_store, int num_full, int split, int split_slot,
                        uint32_t* __restrict__ status) {
  using L = GemmLayout<E8, NB>;
  // the pair tile: 256 tokens x NB channels; each CTA holds NB / 2 rows of B
  constexpr uint32_t kAtomBn = (uint32_t)(NB / 2) * 128;   // one 128-code K atom of B
  constexpr uint32_t kStageBn = (uint32_t)(NB / 2) * BK;   // a stage's B (two atoms)
  constexpr uint32_t kIdescN = idesc_e4m3_f32(2 * BM, NB);
  static_assert(NB == NB || E8, "the packed-code path uses 128-channel tiles");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  // packed codes: SE x 2 atoms x [64 rows x 128 B] decoded B; byte codes: SE x [A 2 atoms x [128 rows x
  // 128 B] | B 2 atoms x [64 rows x 128 B]] as loaded; all E4M3, 128B-swizzled
  uint8_t* bst = smem;
  uint8_t* pk = smem + kPkOffset;              // packed codes: SP x [A 128 x 128 B | B 64 x 128 B], 128B-swizzled
  uint8_t* epi = smem + L::kEpiOffset;         // 4 warps x EB x [32 rows x 128 B], 128B-swizzled
  uint8_t* refb = smem + L::kRefOffset;        // 4 warps x RB x [32 rows x 128 B] y_ref, 128B-swizzled
  float* scl = reinterpret_cast<float*>(smem + L::kScaleOffset);  // packed codes: 4 warps x 128 channel steps
  Bars* bars = reinterpret_cast<Bars*>(smem + L::kBarOffset);
  volatile int* abort_flag = &bars->abort;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t rank = cluster_rank();         // 0: the pair's MMA issuer
  const int pair = blockIdx.x >> 1, num_pairs = gridDim.x >> 1;
  const int num_m = (n + 2 * BM - 1) / (2 * BM);  // 256-token pair tiles
  const int num_n = (d_out + NB - 1) / NB;
  const int num_k = (d_in + BK - 1) / BK;
  const int num_tiles = num_m * num_n;
  const int n_split = (num_tiles - num_full) * split;   // 0 without a split
  const int total_units = num_full + n_split;

  if (tid == 0) {
    for (int s = 0; s < SP; ++s) {
      for (int g = 0; g < kDecGroups; ++g)
        mbar_init(&bars->p_full[g][s], 2);     // the A and the B producer each arrive with their bytes
      mbar_init(&bars->p_empty[s], kGroupWarps);    // the decode group of that stage
    }
    for (int s = 0; s < SE; ++s) {
      // even CTA: its decode group, or with byte codes its two producers (+ 4 bytes from the odd CTA);
      // odd CTA: the same locally, then forwarded
      mbar_init(&bars->full[s], E8 ? 2 : kGroupWarps);
      mbar_init(&bars->ready[s], E8 ? 2 : kGroupWarps);
      mbar_init(&bars->empty[s], 1);              // the pair MMA's multicast commit
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&bars->acc_full[b], 1);
      mbar_init(&bars->acc_empty[b], 2 * kEpiWarps);  // the epilogue warps of both CTAs (even CTA)
    }
    mbar_init(&bars->mma_done, 1);
    for (int w = 0; w < kEpiWarps; ++w)
      for (int b = 0; b < L::RB; ++b) mbar_init(&bars->ref_full[w][b], 1);
    bars->abort = 0;
    fence_mbar_init();
  }
  __syncwarp();
  pdl_wait_then_release();                        // nothing global or in tensor memory before this
  if (warp == 0) tmem_alloc_pair(&bars->tmem_addr, L::kTmem);
  tc_fence_before();
  cluster_sync();                                 // both CTAs' barriers are initialized before any remote arrive
  tc_fence_after();
  const uint32_t tmem = bars->tmem_addr;

  if (warp == kProdA || warp == kProdB) {
    // ---------------------------------------------------------------- TMA producers (A: warp 0, B: warp 2)
    if (lane == 0) {
      const bool is_a = warp == kProdA;
      const CUtensorMap* map = is_a ? &tmA : &tmB;
      prefetch_tensormap(map);
      uint32_t it = 0;
      bool ok = true;
      for (int u = pair; u < total_units && ok; u += num_pairs) {
        const Unit w = unit_at(u, num_full, split, num_k, n_split);
        int m, nn;
        tile_coords(w.tile, num_m, num_n, &m, &nn);
        const int row = is_a ? m * 2 * BM + (int)rank * BM : nn * NB + (int)rank * (NB / 2);
        for (int ks = w.k0; ks < w.k1; ++ks, ++it) {
          if constexpr (E8) {
            // the stage's two K atoms; the even CTA's A producer also expects the odd CTA's 4-byte signal
            const uint32_t s = it % L::S, use = it / L::S;
            if (use > 0 && !(ok = mbar_wait_bounded(&bars->empty[s], (use - 1) & 1, abort_flag, __LINE__))) break;
            uint8_t* dst = bst + s * L::kStageOp + (is_a ? 0u : kStageA8);
            uint64_t* fb = rank == 0 ? &bars->full[s] : &bars->ready[s];
            mbar_arrive_expect_tx(fb, is_a ? kStageA8 + (rank == 0 ? 4u : 0u) : kStageBn);
            tma_load_2d(dst, map, ks * BK, row, fb);
            tma_load_2d(dst + (is_a ? kAtomA8 : kAtomBn), map, ks * BK + 128, row, fb);
          } else {
            const uint32_t s = it % SP, use = it / SP;
            if (use > 0 && !(ok = mbar_wait_bounded(&bars->p_empty[s], (use - 1) & 1, abort_flag, __LINE__))) break;
            uint8_t* dst = pk + s * kPackedStage + (is_a ? 0 : kPackedA);
            uint64_t* pf = &bars->p_full[it % kDecGroups][s];   // the barrier of the group that decodes it
            mbar_arrive_expect_tx(pf, is_a ? kPackedA : kPackedB);
            tma_load_2d(dst, map, ks * BKP, row, pf);
          }
        }
      }
      // the copies in flight land before the CTA exits (they have, unless a wait gave up)
      volatile int no_abort = 0;
      if constexpr (E8) {
        for (uint32_t j = it > (uint32_t)L::S ? it - L::S : 0; j < it; ++j)
          mbar_wait_bounded(rank == 0 ? &bars->full[j % L::S] : &bars->ready[j % L::S], (j / L::S) & 1, &no_abort);
      } else {
        for (uint32_t j = it > (uint32_t)SP ? it - SP : 0; j < it; ++j)
          mbar_wait_bounded(&bars->p_full[j % kDecGroups][j % SP], (j / kPFullPeriod) & 1, &no_abort);
      }
    }
  } else if ((warp == kMmaWarp || warp == kFwdWarp) && rank == 1) {
    // ---------------------------------------------------------------- odd CTA: forward stage readiness
    // An arrive on the even CTA's barrier from a thread that has just written shared and tensor
    // memory stalls it for ~1.5k cycles (the cluster-scope release drains its writes), so the decode
    // warps arrive locally and one thread per decode group carries the stage's readiness over with an
    // asynchronous 4-byte store that completes bytes on the even CTA's stage barrier.  Each forwarder
    // takes the stages of one parity, so every barrier's phases are waited for in order by one thread
    // (a thread that skipped a phase would wait for one two ahead, which a parity wait returns at
    // once); with an even number of stages that is also the decode group of the step.
    if (lane == 0) {
      const uint32_t grp = warp == kMmaWarp ? 0u : 1u;
      uint32_t it = 0;
      bool ok = true;
      for (int u = pair; u < total_units && ok; u += num_pairs) {
        const Unit w = unit_at(u, num_full, split, num_k, n_split);
        for (int ks = w.k0; ks < w.k1; ++ks, ++it) {
          const uint32_t s = it % L::S;
          if ((s & 1u) != grp) continue;
          if (!(ok = mbar_wait_bounded(&bars->ready[s], (it / L::S) & 1, abort_flag, __LINE__))) break;
          tc_fence_after();
          st_async_signal(&bars->fwd_word[s], &bars->full[s], 0);
        }
      }
    }
  } else if (warp == kMmaWarp) {
    // ---------------------------------------------------------------- MMA issuer (even CTA)
    if (lane == 0 && rank == 0) {
      uint32_t it = 0, tcount = 0;
      bool ok = true;
      for (int u = pair; u < total_units && ok; u += num_pairs, ++tcount) {
        const Unit w = unit_at(u, num_full, split, num_k, n_split);
        const uint32_t ab = tcount & 1;
        // the epilogue must have drained this accumulator (used two units ago)
        if (tcount >= 2 && !(ok = mbar_wait_bounded(&bars->acc_empty[ab], ((tcount >> 1) - 1) & 1, abort_flag, __LINE__))) break;
        tc_fence_after();
        for (int ks = w.k0; ks < w.k1; ++ks, ++it) {
          const uint32_t s = it % L::S;
          if (!(ok = mbar_wait_bounded(&bars->full[s], (it / L::S) & 1, abort_flag, __LINE__))) break;
          tc_fence_after();
          if constexpr (E8) {
            const uint32_t abase = smem_u32(bst + s * L::kStageOp), bbase = abase + kStageA8;
#pragma unroll
            for (int kk = 0; kk < BK / 32; ++kk) {  // K = 32 codes per MMA: atom kk/4 of A and of B, +32 B
              const uint64_t da = sdesc_kmajor_sw128(abase + (uint32_t)(kk >> 2) * kAtomA8) + 2 * (kk & 3);
              const uint64_t db = sdesc_kmajor_sw128(bbase + (uint32_t)(kk >> 2) * kAtomBn) + 2 * (kk & 3);
              mma_pair_ss(tmem + ab * NB, da, db, kIdescN, (ks != w.k0 || kk != 0) ? 1u : 0u);
            }
          } else {
            const uint32_t bbase = smem_u32(bst + s * kStageBn);
            const uint32_t ta = tmem + kAccCols + 64u * s;
#pragma unroll
            for (int kk = 0; kk < BK / 32; ++kk) {  // K = 32 codes per MMA: 8 TMEM columns of A; B atom kk/4, +32 B
              const uint64_t db = sdesc_kmajor_sw128(bbase + (uint32_t)(kk >> 2) * kAtomBn) + 2 * (kk & 3);
              mma_pair_ts(tmem + ab * NB, ta + 8u * kk, db, kIdescN, (ks != w.k0 || kk != 0) ? 1u : 0u);
            }
          }
          mma_commit_pair(&bars->empty[s]);
        }
        if (ok) mma_commit_pair(&bars->acc_full[ab]);
      }
      mma_commit_pair(&bars->mma_done);  // all MMAs complete before TMEM is released
      volatile int no_abort = 0;
      mbar_wait_bounded(&bars->mma_done, 0, &no_abort);
    }
  } else if (warp >= kEpiWarp0 && warp < kEpiWarp0 + kEpiWarps) {
    // ---------------------------------------------------------------- epilogue
    const int quad = warp & 3, ew = warp - kEpiWarp0;
    uint8_t* stage0 = epi + ew * L::EB * kEpiStage;
    uint8_t* rstage0 = refb + ew * L::RB * kEpiStage;
    float* wsc = scl + ew * NB;
    const bool with_ref = sums3 != nullptr;
    f32x2 sig = {0.f, 0.f}, err = {0.f, 0.f};      // SQNR sums of this thread's outputs
    uint32_t tcount = 0, nstore = 0;
    bool ok = true;
    // y_ref tiles of whole-tile units: chunk c of every such tile goes through buffer c % RB, loaded RB
    // chunks ahead; all four are loaded (out-of-range parts read as zero), so the buffer phases advance
    // regularly.  The epilogue of a split tail tile reads y_ref with plain loads.
    uint32_t nref[kEpiBufs] = {0u, 0u}, nused[kEpiBufs] = {0u, 0u};  // loads issued / consumed per buffer
    auto load_ref = [&](int tile_, int c_) {        // called by the whole warp; lane 0 issues
      int m_, nn_;
      tile_coords(tile_, num_m, num_n, &m_, &nn_);
      const int rb_ = c_ % L::RB;
      uint64_t* bar = &bars->ref_full[ew][rb_];
      if (lane == 0) {
        mbar_arrive_expect_tx(bar, kEpiStage);
        tma_load_2d(rstage0 + rb_ * kEpiStage, &tmR, nn_ * NB + c_ * 32, m_ * 2 * BM + (int)rank * BM + quad * 32,
                    bar);
      }
      ++nref[rb_];
    };
    // y (and acc_out) of one chunk: 32 rows from row0_ (this lane: t_) x 32 channels from o0; v the
    // outputs, a the raw accumulators
    auto store_chunk = [&](int o0, int row0_, int t_, const float (&v)[32], const float (&a)[32]) {
      if (o0 >= d_out || row0_ >= n) return;      // warp-uniform: nothing of this chunk is in range
      if (use_tma_store) {
        uint8_t* buf = stage0 + (nstore % L::EB) * kEpiStage;
        if (lane == 0) {                       // the store issued EB chunks ago has read this buffer
          if (L::EB == 1)
            bulk_wait_read_all();
          else
            bulk_wait_read_le1();
        }
        __syncwarp();
#pragma unroll
        for (int q = 0; q < 8; ++q)  // row `lane`, 16-byte chunk q at q ^ (lane % 8)
          *reinterpret_cast<float4*>(buf + lane * 128 + ((q ^ (lane & 7)) << 4)) =
              make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          tma_store_2d(&tmY, buf, o0, row0_);
          bulk_commit();
        }
        ++nstore;
      } else if (t_ < n) {
        float* yrow = y + (size_t)t_ * d_out;
#pragma unroll
        for (int i = 0; i < 32; ++i)
          if (o0 + i < d_out) yrow[o0 + i] = v[i];
      }
      if (acc_out && t_ < n) {
        int32_t* arow = acc_out + (size_t)t_ * d_out;
#pragma unroll
        for (int i = 0; i < 32; ++i)
          if (o0 + i < d_out) arow[o0 + i] = __float2int_rn(a[i] * kAccScale);
      }
    };
    // tail tiles: this lane's row of part j's partial accumulators, the counters of this warp's
    // 32-row slice of tail tile tj, and the bounded wait for all parts of the tile
    const int my_row = (int)rank * BM + quad * 32 + lane;
    // part j's partial accumulators of channel group g (4 channels), this lane's row
    auto split_at = [&](int j, int g) {
      return g_split_part + (size_t)split_slot * kSplitSlotF4 + ((size_t)j * (NB / 4) + g) * (2 * BM) + my_row;
    };
    auto cnt_of = [&](int tj, int which) { return &g_split_cnt[split_slot][tj][rank][ew][which]; };
    auto arrive_part = [&](int tj) {                // after this lane's partial stores
      __threadfence();
      __syncwarp();
      if (lane == 0) atomicAdd(cnt_of(tj, 0), 1u);
    };
    auto wait_parts = [&](int tj) -> bool {         // warp-uniform: true once all parts have arrived
      uint32_t good = 1u;
      if (lane == 0) {
        const uint64_t t0 = globaltimer_ns();
        for (uint32_t it = 0; ld_acquire_gpu(cnt_of(tj, 0)) < (uint32_t)split; ++it) {
          __nanosleep(64);
          if ((it & 63u) == 63u && (*abort_flag || globaltimer_ns() - t0 > kWaitLimitNs)) {
            if (*abort_flag == 0) *abort_flag = __LINE__;
            good = 0u;
            break;
          }
        }
      }
      good = __shfl_sync(0xFFFFFFFFu, good, 0);
      __threadfence();                              // the other parts' stores are seen from here on
      return good != 0u;
    };
    auto finish_part = [&](int tj) {                // the last part to finish clears the counters
      __syncwarp();
      if (lane == 0 && atomicAdd(cnt_of(tj, 1), 1u) == (uint32_t)(split - 1)) {
        *cnt_of(tj, 0) = 0u;
        *cnt_of(tj, 1) = 0u;
      }
    };
    // the share of split unit uu's tile that its part finishes: channels [NB / S * part, ...) of the
    // tile, once all S parts' partials are out
    auto finish_share = [&](int uu) {
      const Unit w = unit_at(uu, num_full, split, num_k, n_split);
      const int tj = w.tile - num_full;
      int m, nn;
      tile_coords(w.tile, num_m, num_n, &m, &nn);
      const int t = m * 2 * BM + (int)rank * BM + quad * 32 + lane;
      const float sxt = (t < n) ? sx[t] * kAccScale : 0.f;
      if (wait_parts(tj)) {
        float s_run = 0.f, e_run = 0.f;
        auto fixup = [&](auto split_c) {
          constexpr int S = decltype(split_c)::value;
          constexpr int L = S >= 4 ? 16 : 8;      // loads of parts per batch
          constexpr int G = NB / 4 / S, PB = L / S;   // groups of the share, groups per batch
          const int g0 = w.part * G;
#pragma unroll 1
          for (int b = 0; b < G; b += PB) {
            float4 pq[L], yr[PB];
#pragma unroll
            for (int i = 0; i < L; ++i)
              pq[i] = __ldcg(split_at(tj * S + i % S, g0 + b + i / S));
#pragma unroll
            for (int k = 0; k < PB; ++k) {
              const int o = nn * NB + 4 * (g0 + b + k);
              yr[k] = (with_ref && t < n && o < d_out)
                          ? __ldcs(reinterpret_cast<const float4*>(y_ref + (size_t)t * d_out + o))
                          : make_float4(0.f, 0.f, 0.f, 0.f);
            }
#pragma unroll
            for (int k = 0; k < PB; ++k) {
              float4 acc4 = pq[k * S];
#pragma unroll
              for (int q = 1; q < S; ++q) {   // exact in any order
                acc4.x += pq[k * S + q].x;
                acc4.y += pq[k * S + q].y;
                acc4.z += pq[k * S + q].z;
                acc4.w += pq[k * S + q].w;
              }
              const int gl = g0 + b + k, o = nn * NB + 4 * gl;
              const float a[4] = {acc4.x, acc4.y, acc4.z, acc4.w};
              float v[4];
#pragma unroll
              for (int i = 0; i < 4; ++i) v[i] = a[i] * sxt * ((o + i < d_out) ? __ldg(sw + o + i) : 0.f);
              if (t < n && o < d_out) {
                float* yp = y + (size_t)t * d_out + o;
                if ((d_out & 3) == 0) {               // a float4 is wholly in or out of range
                  *reinterpret_cast<float4*>(yp) = make_float4(v[0], v[1], v[2], v[3]);
                  const float e0 = yr[k].x - v[0], e1 = yr[k].y - v[1], e2 = yr[k].z - v[2], e3 = yr[k].w - v[3];
                  s_run += yr[k].x * yr[k].x + yr[k].y * yr[k].y + yr[k].z * yr[k].z + yr[k].w * yr[k].w;
                  e_run += e0 * e0 + e1 * e1 + e2 * e2 + e3 * e3;
                } else {
#pragma unroll
                  for (int i = 0; i < 4; ++i)
                    if (o + i < d_out) yp[i] = v[i];
                }
                if (acc_out) {
#pragma unroll
                  for (int i = 0; i < 4; ++i)
                    if (o + i < d_out) acc_out[(size_t)t * d_out + o + i] = __float2int_rn(a[i] * kAccScale);
                }
              }
            }
          }
        };
        switch (split) {
          case 2: fixup(std::integral_constant<int, 2>{}); break;
          case 4: fixup(std::integral_constant<int, 4>{}); break;
          case 8: fixup(std::integral_constant<int, 8>{}); break;
          default: fixup(std::integral_constant<int, 16>{}); break;
        }
        if (with_ref) {
          sig = f2_add(sig, s_run);
          err = f2_add(err, e_run);
        }
      }
      finish_part(tj);
    };
    // this pair's first whole tile comes after its split part, if it has one; y_ref loads and uses
    // count whole tiles only (fcount)
    const int u_full0 = pair < n_split ? pair + num_pairs : pair;
    if (with_ref && u_full0 < total_units)
      for (int c0 = 0; c0 < L::RB; ++c0) load_ref(u_full0 - n_split, c0);
    uint32_t fcount = 0;
    int split_state = 0;                            // this pair's split part: 1 partials out, 2 share done
    int u = pair;
    for (; u < total_units; u += num_pairs, ++tcount) {
      const Unit w = unit_at(u, num_full, split, num_k, n_split);
      const uint32_t ab = tcount & 1;
      int m, nn;
      tile_coords(w.tile, num_m, num_n, &m, &nn);
      const int row0 = m * 2 * BM + (int)rank * BM + quad * 32;
      const int t = row0 + lane;
      const float sxt = (t < n) ? sx[t] * kAccScale : 0.f;
      if constexpr (!E8) {
        __syncwarp();
#pragma unroll
        for (int i = 0; i < NB / 32; ++i) {  // this tile's output-channel steps, staged once per unit
          const int o = nn * NB + 32 * i + lane;
          wsc[32 * i + lane] = (o < d_out) ? sw[o] : 0.f;
        }
        __syncwarp();
      }
      if (!(ok = mbar_wait_bounded(&bars->acc_full[ab], (tcount >> 1) & 1, abort_flag, __LINE__))) break;
      __syncwarp();
      tc_fence_after();
      if (w.part < 0) {
#pragma unroll 1
        for (int c = 0; c < NB / 32; ++c) {
          uint32_t r[32];
          __syncwarp();
          CAT_TMEM_LD32(tmem + ((uint32_t)(quad * 32) << 16) + ab * NB + c * 32, r);
          tmem_ld_wait();
          if (c == NB / 32 - 1) {  // accumulator fully read: the MMAs of unit + 2 may use it
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_cluster(&bars->acc_empty[ab], 0);
          }
          const int o0 = nn * NB + c * 32;
          float a[32], v[32];
          if constexpr (E8) {                    // the chunk's 32 channel steps, one per lane
            const float swl = (o0 + lane < d_out) ? __ldg(sw + o0 + lane) : 0.f;
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              a[i] = __uint_as_float(r[i]);
              v[i] = a[i] * sxt * __shfl_sync(0xFFFFFFFFu, swl, i);
            }
          } else {
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              a[i] = __uint_as_float(r[i]);
              v[i] = a[i] * sxt * wsc[c * 32 + i];
            }
          }
          if (with_ref) {
            // SQNR sums (Sec. 2, Eq. 1) from the y_ref tile of this chunk; out-of-range entries are zero
            // on both sides.  Squares are summed in fp32 over the chunk's 32 values, then as float pairs.
            const int rbuf = c % L::RB;
            const uint32_t use = (NB / 32 / L::RB) * fcount + c / L::RB;  // the use-th load into buffer rbuf
            if (!(ok = mbar_wait_bounded(&bars->ref_full[ew][rbuf], use & 1, abort_flag, __LINE__))) break;
            ++nused[rbuf];
            const uint8_t* rb = rstage0 + rbuf * kEpiStage + lane * 128;
            float s_run = 0.f, e_run = 0.f;
#pragma unroll
            for (int q = 0; q < 8; ++q) {
              const float4 yr = *reinterpret_cast<const float4*>(rb + ((q ^ (lane & 7)) << 4));
              const float e0 = yr.x - v[4 * q], e1 = yr.y - v[4 * q + 1], e2 = yr.z - v[4 * q + 2], e3 = yr.w - v[4 * q + 3];
              s_run += yr.x * yr.x + yr.y * yr.y + yr.z * yr.z + yr.w * yr.w;
              e_run += e0 * e0 + e1 * e1 + e2 * e2 + e3 * e3;
            }
            sig = f2_add(sig, s_run);
            err = f2_add(err, e_run);
            // refill this buffer with the chunk RB ahead (this tile or the next: whole tiles follow)
            int nu = u, nc = c + L::RB;
            if (nc >= NB / 32) {
              nc -= NB / 32;
              nu = u + num_pairs;
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (nu < total_units) load_ref(nu - n_split, nc);
          }
          store_chunk(o0, row0, t, v, a);
        }
        ++fcount;
        if (!ok) break;
      } else {
        // a K part of a tail tile: this warp's 32 rows of raw accumulators to the part's slice
        const int tj = w.tile - num_full, j = u;
#pragma unroll 1
        for (int c = 0; c < NB / 32; ++c) {
          uint32_t r[32];
          __syncwarp();
          CAT_TMEM_LD32(tmem + ((uint32_t)(quad * 32) << 16) + ab * NB + c * 32, r);
          tmem_ld_wait();
          if (c == NB / 32 - 1) {
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_cluster(&bars->acc_empty[ab], 0);
          }
#pragma unroll
          for (int q = 0; q < 8; ++q)   // a warp stores 32 consecutive rows of one channel group: 512 B
            __stcg(split_at(j, 8 * c + q),
                   make_float4(__uint_as_float(r[4 * q]), __uint_as_float(r[4 * q + 1]), __uint_as_float(r[4 * q + 2]),
                               __uint_as_float(r[4 * q + 3])));
        }
        arrive_part(tj);
        split_state = 1;
        // the sibling parts run at the same time, on other pairs, as their first unit: the share is
        // finished while this pair's first whole tile is still in its MMAs
        finish_share(pair);
        split_state = 2;
      }
    }
    if (!ok && pair < n_split) {
      // a wait gave up: settle this warp's split part all the same (without data: the launch's
      // outputs are void), so that every counter of the launch ends at zero
      const int tj = unit_at(pair, num_full, split, num_k, n_split).tile - num_full;
      if (split_state == 0) arrive_part(tj);
      if (split_state <= 1) finish_part(tj);
    }
    if (with_ref) {
      // y_ref loads issued but not consumed (only after a wait gave up) land before the CTA exits
      volatile int no_abort = 0;
      for (int bb = 0; bb < L::RB; ++bb)
        if (nref[bb] > nused[bb]) mbar_wait_bounded(&bars->ref_full[ew][bb], (nref[bb] - 1) & 1, &no_abort);
      sig = f2_warp_sum(sig);
      err = f2_warp_sum(err);
      if (lane == 0) {
        bars->sums[ew][0] = sig;
        bars->sums[ew][1] = err;
      }
      asm volatile("bar.sync 2, 128;" ::: "memory");  // this CTA's four epilogue warps have written theirs
      if (ew == 0) {
        const f32x2 s_cta = f2_add(f2_add(bars->sums[0][0], bars->sums[1][0]), f2_add(bars->sums[2][0], bars->sums[3][0]));
        const f32x2 e_cta = f2_add(f2_add(bars->sums[0][1], bars->sums[1][1]), f2_add(bars->sums[2][1], bars->sums[3][1]));
        sqnr_cta_done(sqnr_slot, s_cta, e_cta, sums3);
      }
    }
    if (lane == 0) bulk_wait_all();
    __syncwarp();
  } else if (!E8 && warp >= kDecWarp0) {
    // ---------------------------------------------------------------- decode (packed codes)
    // Two groups of four warps (one warp per TMEM lane quadrant each) decode alternate K steps: the
    // decode of one step is latency-bound (shared-memory loads, tensor-memory stores and their wait,
    // the proxy fence), so two steps are kept in flight.
    const int grp = (warp - kDecWarp0) >> 2;      // 0: even K steps, 1: odd K steps
    const int quad = warp & 3;
    const int gt = (warp - kDecWarp0 - 4 * grp) * 32 + lane;  // 0..127 within the group
    const int a_row = quad * 32 + lane;           // this thread's A row = TMEM lane
    uint32_t it = 0;
    bool ok = true;
    for (int u = pair; u < total_units && ok; u += num_pairs) {
      const Unit w = unit_at(u, num_full, split, num_k, n_split);
      for (int ks = w.k0; ks < w.k1; ++ks, ++it) {
        if ((it & 1u) != (uint32_t)grp) continue;
        const uint32_t ps = it % SP, s = it % SE;
        if (!(ok = mbar_wait_bounded(&bars->p_full[grp][ps], (it / kPFullPeriod) & 1, abort_flag, __LINE__))) break;
        if (it >= SE && !(ok = mbar_wait_bounded(&bars->empty[s], ((it / SE) - 1) & 1, abort_flag, __LINE__))) break;
        tc_fence_after();
        const uint8_t* pa = pk + ps * kPackedStage;
        const uint8_t* pb = pa + kPackedA;
        const uint8_t* prow = pa + a_row * 128;
#pragma unroll
        for (int half = 0; half < 2; ++half) {  // A: one 128-byte row per thread -> 64 TMEM columns
          uint32_t av[32];
#pragma unroll
          for (int jj = 0; jj < 4; ++jj) {
            const int j = 4 * half + jj;
            const uint4 w = *reinterpret_cast<const uint4*>(prow + ((j ^ (a_row & 7)) << 4));
            av[8 * jj + 0] = sm4_lo(w.x); av[8 * jj + 1] = sm4_hi(w.x);
            av[8 * jj + 2] = sm4_lo(w.y); av[8 * jj + 3] = sm4_hi(w.y);
            av[8 * jj + 4] = sm4_lo(w.z); av[8 * jj + 5] = sm4_hi(w.z);
            av[8 * jj + 6] = sm4_lo(w.w); av[8 * jj + 7] = sm4_hi(w.w);
          }
          __syncwarp();
          CAT_TMEM_ST32(tmem + ((uint32_t)(quad * 32) << 16) + kAccCols + 64u * s + 32u * half, av);
        }
        // B: 512 chunks of 16 packed bytes (64 rows x 8), 4 per thread; 8 consecutive threads read
        // one 128-byte row.  Chunk j (codes 32j .. 32j+31) becomes the 16-byte E4M3 chunks 2(j%4) and
        // 2(j%4)+1 of atom j/4; threads of atom 1 store their odd chunk first, so the 8 threads of a
        // row never hit the same bank group in one store
        uint8_t* bs = bst + s * kStageBn;
#pragma unroll
        for (int i = 0; i < (NB / 2) * 8 / kGroupThreads; ++i) {
          const int id = gt + kGroupThreads * i;
          const int row = id >> 3, j = id & 7, swz = row & 7;
          const uint4 w = *reinterpret_cast<const uint4*>(pb + row * 128 + ((j ^ swz) << 4));
          uint8_t* dst = bs + (j >> 2) * kAtomBn + row * 128;
          const uint4 lo = make_uint4(sm4_lo(w.x), sm4_hi(w.x), sm4_lo(w.y), sm4_hi(w.y));
          const uint4 hi = make_uint4(sm4_lo(w.z), sm4_hi(w.z), sm4_lo(w.w), sm4_hi(w.w));
          const int c0 = 2 * (j & 3);
          if (j < 4) {
            *reinterpret_cast<uint4*>(dst + ((c0 ^ swz) << 4)) = lo;
            *reinterpret_cast<uint4*>(dst + (((c0 + 1) ^ swz) << 4)) = hi;
          } else {
            *reinterpret_cast<uint4*>(dst + (((c0 + 1) ^ swz) << 4)) = hi;
            *reinterpret_cast<uint4*>(dst + ((c0 ^ swz) << 4)) = lo;
          }
        }
        tmem_st_wait();
        fence_proxy_async_smem();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(&bars->p_empty[ps]);
          if (rank == 1)
            mbar_arrive(&bars->ready[s]);          // local arrives only: cheap
          else if (quad == 0)
            mbar_arrive_expect_tx(&bars->full[s], 4u);  // the odd CTA's 4-byte signal completes the stage
          else
            mbar_arrive(&bars->full[s]);
        }
      }
    }
  }

  tc_fence_before();
  cluster_sync();                                 // the pair's MMAs and both epilogues are done with TMEM
  if (bars->abort && tid == 0) report(status, timeout_bits(kWhereGemm, bars->abort));
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, L::kTmem);
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

// Packed codes [rows][row_bytes], box [box_rows][128 bytes], 128-byte swizzle, out-of-range reads zero.
bool make_packed_map(CUtensorMap* map, const uint8_t* base, int64_t rows, int64_t row_bytes, int box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {(cuuint64_t)row_bytes, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)row_bytes};
  cuuint32_t box[2] = {(cuuint32_t)BKP, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<uint8_t*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int num_sms() {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 148;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0) return 148;
  return sms;
}

// Whether a cooperative launch of `pairs` CTA pairs of the GEMM kernel fits on this device (checked
// once per process and operand format, on the first device asked).
template <bool E8, int NB>
bool split_launch_ok(int64_t pairs) {
  using L = GemmLayout<E8, NB>;
  static int ok = -1;
  static std::mutex mu;
  std::lock_guard<std::mutex> lock(mu);
  if (ok < 0) {
    int dev = 0, coop = 0, clusters = 0;
    ok = 0;
    if (cudaGetDevice(&dev) == cudaSuccess &&
        cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, dev) == cudaSuccess && coop &&
        cudaFuncSetAttribute(w4a4_gemm_tc_kernel<E8, NB>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)L::kSmemBytes) == cudaSuccess) {
      cudaLaunchConfig_t cfg;
      memset(&cfg, 0, sizeof(cfg));
      cfg.gridDim = dim3((unsigned)(2 * pairs), 1, 1);
      cfg.blockDim = dim3(kThreads, 1, 1);
      cfg.dynamicSmemBytes = L::kSmemBytes;
      if (cudaOccupancyMaxActiveClusters(&clusters, w4a4_gemm_tc_kernel<E8, NB>, &cfg) == cudaSuccess &&
          clusters >= pairs)
        ok = 1;
    }
    cudaGetLastError();
  }
  return ok == 1;
}

// y_ref != nullptr: the epilogue also forms the SQNR sums of y against y_ref and writes
// sums3 = {sum y_ref^2, sum (y_ref - y)^2, dB} (sums3 needs no zeroing).  Needs d_out % 4 == 0
// (TMA row pitch).  E8: xq and wq hold one code per byte, else SM4x8 (two per byte).  NB: channels per
// pair tile (256 only with byte codes; the last wave is then not split along K).
template <bool E8, int NB>
cudaError_t launch_gemm_tc(const uint8_t* xq, const float* sx, const uint8_t* wq, const float* sw, int64_t n,
                           int64_t d_in, int64_t d_out, float* y, int32_t* acc_out, const float* y_ref, double* sums3,
                           uint32_t* status, cudaStream_t stream) {
  using L = GemmLayout<E8, NB>;
  CUtensorMap ty, ta, tb, tr;
  memset(&ty, 0, sizeof(ty));
  memset(&tr, 0, sizeof(tr));
  int use_tma = (d_out % 4 == 0) ? 1 : 0;
  if (use_tma && !make_output_map(&ty, y, n, d_out)) use_tma = 0;
  if (y_ref) {
    if (d_out % 4 != 0 || !sums3 || !make_output_map(&tr, const_cast<float*>(y_ref), n, d_out))
      return cudaErrorInvalidValue;
  }
  const int64_t row_bytes = E8 ? d_in : d_in / 2;
  if (!make_packed_map(&ta, xq, n, row_bytes, BM) || !make_packed_map(&tb, wq, d_out, row_bytes, NB / 2))
    return cudaErrorInvalidValue;
  static std::once_flag attr_once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(attr_once, [] {
    attr_err = cudaFuncSetAttribute(w4a4_gemm_tc_kernel<E8, NB>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)L::kSmemBytes);
  });
  if (attr_err != cudaSuccess) return attr_err;
  const int64_t tiles = ((n + 2 * BM - 1) / (2 * BM)) * ((d_out + NB - 1) / NB);
  const int64_t num_k = (d_in + BK - 1) / BK;
  const int64_t pairs_max = num_sms() / 2;
  // the last wave's tiles, split along K into a power-of-two number of parts when that wave is at
  // most half full (the parts wait for one another: only with a cooperative launch)
  const int64_t tail = tiles >= pairs_max ? tiles % pairs_max : tiles;
  int split = 1;
  constexpr int64_t kWide = NB / BN;             // a part's scratch, in 128-wide parts
  if (tail > 0 && tail <= kMaxSplitTiles && 2 * tail <= pairs_max && split_launch_ok<E8, NB>(pairs_max))
    while (2 * split <= kMaxSplit && 2 * split * tail <= pairs_max && 2 * split <= num_k &&
           2 * split * tail * kWide <= kMaxSplitUnits)
      split *= 2;
  // a single partial wave has no whole tiles to hide the parts' exchange behind: split it only
  // when that saves ten K steps or more
  if (split > 1 && tiles < pairs_max && num_k - num_k / split < 10) split = 1;
  const int64_t num_full = split > 1 ? tiles - tail : tiles;
  const int64_t units = num_full + (tiles - num_full) * split;
  if (split > 1 && ((units - num_full) * kWide > kMaxSplitUnits || num_full % pairs_max != 0))
    return cudaErrorInvalidConfiguration;
  const int grid = 2 * (int)(units < pairs_max ? units : pairs_max);  // CTA pairs (cluster of 2)
  if (grid > kSqnrMaxCtas) return cudaErrorInvalidConfiguration;
  static std::atomic<unsigned> next_split{0};
  const int split_slot = split > 1 ? (int)(next_split.fetch_add(1, std::memory_order_relaxed) % kSplitSlots) : 0;
  const int slot = y_ref ? next_sqnr_slot() : 0;
  const double* sums = y_ref ? sums3 : nullptr;
  note_launch();
  cudaLaunchConfig_t cfg;
  memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = dim3((unsigned)grid, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = L::kSmemBytes;
  cfg.stream = stream;
  cudaLaunchAttribute attrs[2];
  attrs[0] = pdl_attr();
  attrs[1].id = cudaLaunchAttributeCooperative;   // the split parts wait for one another
  attrs[1].val.cooperative = 1;
  cfg.attrs = attrs;
  cfg.numAttrs = split > 1 ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, w4a4_gemm_tc_kernel<E8, NB>, ty, ta, tb, tr, y_ref, const_cast<double*>(sums), slot, sx,
                            sw, (int)n, (int)d_in, (int)d_out, y, acc_out, use_tma, (int)num_full, split, split_slot,
                            status);
}

// Byte codes: 256-channel pair tiles where they take less time than 128-channel ones.  The MMA thread's
// wait for each stage idles the tensor core for ~200-300 cycles, whatever the tile width, so a 256-wide
// tile (twice the MMA work per stage) costs kWideTileCost of two 128-wide tiles (measured: 0.78 on the
// 8192 x 8192 x 28672 and 4096 x 14336 x 4096 layers); but there are half as many tiles to spread over
// the pairs, and the last wave is not split along K.
constexpr double kWideTileCost = 0.78;
bool e8_wide_tiles(int64_t n, int64_t d_out) {
  const int64_t pairs = num_sms() / 2, m_tiles = (n + 2 * BM - 1) / (2 * BM);
  const int64_t t128 = m_tiles * ((d_out + BN - 1) / BN), t256 = m_tiles * ((d_out + 255) / 256);
  // a last wave at most half full is split along K over the idle pairs (in about that proportion),
  // when the scratch holds at least two parts of each of its tiles (as the launcher decides)
  auto waves = [&](int64_t tiles, int64_t wide) {
    const int64_t tail = tiles % pairs;
    const bool split = tail > 0 && 2 * tail <= pairs && tail <= kMaxSplitTiles && 2 * tail * wide <= kMaxSplitUnits;
    return split ? (double)tiles / pairs : (double)((tiles + pairs - 1) / pairs);
  };
  const double w128 = waves(t128, 1), w256 = 2.0 * kWideTileCost * waves(t256, 2);
  return w256 < w128;
}

}  // namespace

cudaError_t launch_w4a4_gemm_tc(const uint8_t* xq, const float* sx, const uint8_t* wq, const float* sw, int64_t n,
                                int64_t d_in, int64_t d_out, float* y, int32_t* acc_out, const float* y_ref,
                                double* sums3, uint32_t* status, cudaStream_t stream) {
  return launch_gemm_tc<false, BN>(xq, sx, wq, sw, n, d_in, d_out, y, acc_out, y_ref, sums3, status, stream);
}

cudaError_t launch_w4a4_gemm_tc_e8(const uint8_t* xq8, const float* sx, const uint8_t* wq8, const float* sw, int64_t n,
                                   int64_t d_in, int64_t d_out, float* y, int32_t* acc_out, const float* y_ref,
                                   double* sums3, uint32_t* status, cudaStream_t stream) {
  if (e8_wide_tiles(n, d_out))
    return launch_gemm_tc<true, 256>(xq8, sx, wq8, sw, n, d_in, d_out, y, acc_out, y_ref, sums3, status, stream);
  return launch_gemm_tc<true, BN>(xq8, sx, wq8, sw, n, d_in, d_out, y, acc_out, y_ref, sums3, status, stream);
}

// SM4x8 codes -> byte codes.  Every 16 packed bytes (32 codes of a row) become 32 bytes: the masks of
// the format give the E4M3 bytes of codes 0..3 and 4..7 of each word directly.
__global__ void __launch_bounds__(256) codes_to_e4m3_kernel(const uint4* __restrict__ in, uint4* __restrict__ out,
                                                            int64_t chunks) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < chunks; i += stride) {
    const uint4 w = __ldcs(in + i);
    out[2 * i] = make_uint4(sm4_lo(w.x), sm4_hi(w.x), sm4_lo(w.y), sm4_hi(w.y));
    out[2 * i + 1] = make_uint4(sm4_lo(w.z), sm4_hi(w.z), sm4_lo(w.w), sm4_hi(w.w));
  }
}

// rows x d codes (d a multiple of 32): codes [rows][d/2] -> out [rows][d].
cudaError_t launch_codes_to_e4m3(const uint8_t* codes, int64_t rows, int64_t d, uint8_t* out, cudaStream_t stream) {
  const int64_t chunks = rows * (d / 32);
  if (chunks == 0) return cudaSuccess;
  const int64_t cap = (int64_t)num_sms() * 8;
  const int64_t blocks = (chunks + 255) / 256;
  note_launch();
  codes_to_e4m3_kernel<<<(unsigned)(blocks < cap ? blocks : cap), 256, 0, stream>>>(
      reinterpret_cast<const uint4*>(codes), reinterpret_cast<uint4*>(out), chunks);
  return cudaGetLastError();
}

}  // namespace cat
