// Device helpers shared by the CAT W4A4 kernels (sm_103a): status reporting, the SM4x8 code
// format, bounded mbarrier waits, TMA and tcgen05 wrappers.
#pragma once
#include <atomic>

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace cat {

// Kernels this library has launched in this process (host counter, bumped at every launch site).
extern std::atomic<unsigned long long> g_kernel_launches;
inline void note_launch() { g_kernel_launches.fetch_add(1, std::memory_order_relaxed); }


// ------------------------------------------------------------------------------------------
// Device status word (one per device, owned by api.cu; kernels get its address).
// ------------------------------------------------------------------------------------------
enum : uint32_t {
  kStatusTimeout = 1u,     // a bounded wait gave up
  kStatusNonFinite = 2u,   // a non-finite value reached a quantizer
  // with kStatusTimeout: the kernel (bits 8..12) and, in bits 16..31, the source line of the first
  // wait that gave up
  kWhereTransform2Pass = 1u << 8,
  kWhereTransformFused = 1u << 9,
  kWhereGemm = 1u << 10,
  kWhereGemmDecode = 1u << 11,
  kWhereCalib = 1u << 12,
  kWhereGemmDp = 1u << 13,
};

// The status bits a kernel raises when a wait gave up: abort holds the line of the first one.
__host__ __device__ constexpr uint32_t timeout_bits(uint32_t where, int abort) {
  return kStatusTimeout | where | ((uint32_t)(abort & 0xFFFF) << 16);
}

// Upper bound of any single pipeline wait, in nanoseconds of %globaltimer.
constexpr uint64_t kWaitLimitNs = 1000000000ull;

// Programmatic dependent launch.  A kernel launched with pdl_attr() (the two GEMMs) may be scheduled
// while the previous kernel in the stream is still running; before its first access to global or
// tensor memory it calls pdl_wait_then_release(), which waits until that grid has completed with
// its writes visible, then lets the next dependent grid be scheduled.  The transform and SYRK
// kernels call it too (without the attribute the wait returns at once) so that a GEMM after them
// is scheduled early.  A dependent grid is scheduled
// only once every CTA of this grid has passed that point, i.e. is resident, so waiting CTAs of
// the next grid can never keep a CTA of this one from an SM.
inline cudaLaunchAttribute pdl_attr() {
  cudaLaunchAttribute a;
  a.id = cudaLaunchAttributeProgrammaticStreamSerialization;
  a.val.programmaticStreamSerializationAllowed = 1;
  return a;
}
__device__ __forceinline__ void pdl_wait_then_release() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

__device__ __forceinline__ void report(uint32_t* status, uint32_t bits) {
  if (status) atomicOr(status, bits);
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
  return t;
}

// ------------------------------------------------------------------------------------------
// SM4x8 code format.  A code q in [-7, 7] is the FP8 E4M3 byte (q < 0) << 7 | |q|, i.e. the
// subnormal value q * 2^-9.  Eight consecutive codes e0..e7 share one 32-bit word
//   w = E(e0..e3) | rotl(E(e4..e7), 4)
// where E(.) packs four E4M3 bytes little-endian; then E(e0..e3) = w & 0x87878787 and
// E(e4..e7) = rotr(w, 4) & 0x87878787.
// ------------------------------------------------------------------------------------------
constexpr uint32_t kSm4Mask = 0x87878787u;

__device__ __forceinline__ uint32_t sm4_lo(uint32_t w) { return w & kSm4Mask; }
__device__ __forceinline__ uint32_t sm4_hi(uint32_t w) { return __funnelshift_r(w, w, 4) & kSm4Mask; }

__device__ __forceinline__ uint32_t e4m3_code_byte(int q) {
  return (q < 0 ? 0x80u : 0u) | (uint32_t)(q < 0 ? -q : q);
}

// Pack eight codes (each in [-7, 7]) into one SM4x8 word.
__device__ __forceinline__ uint32_t sm4_pack(const int (&q)[8]) {
  uint32_t lo = e4m3_code_byte(q[0]) | (e4m3_code_byte(q[1]) << 8) | (e4m3_code_byte(q[2]) << 16) |
                (e4m3_code_byte(q[3]) << 24);
  uint32_t hi = e4m3_code_byte(q[4]) | (e4m3_code_byte(q[5]) << 8) | (e4m3_code_byte(q[6]) << 16) |
                (e4m3_code_byte(q[7]) << 24);
  return lo | __funnelshift_l(hi, hi, 4);
}

// The accumulators hold sum(q_x * 2^-9 * q_w * 2^-9); multiply by 2^18 to get the integer.
constexpr float kAccScale = 262144.0f;

// ------------------------------------------------------------------------------------------
// Exact symmetric round-to-nearest code decision (Lemma 2 range, Sec. 6 RTN):
//   q = clamp(round_half_even(qmax * v / a), -qmax, qmax),   a = max|v| of the row.
// The fast estimate p = fl(v * fl(qmax / a)) is within qmax * 2^-22 of the quotient, so rint(p) is
// the exact code unless p lies within 2^-18 of a half-integer; there the decision is redone
// exactly: with f = floor(p) and the boundary h = f + 1/2, the sign of qmax*|v| - h*a is found from
// a two-product (qmax*|v| = prod + err, both fp32, err by fma) and one fma for prod - h*a, which
// is exact whenever it is small and otherwise far from zero, so its sum with err has the true
// sign, and is zero only on an exact tie.  Rows whose maximum lies outside [2^-60, 2^100] are
// rescaled by a power of two first (exact), so qmax*|v| cannot overflow and no product loses bits
// to underflow; such rows always take the exact route.
// ------------------------------------------------------------------------------------------
struct QRow {
  float inv;   // fl(qmax / a_s), 0 for a row whose codes are all 0 (zero or non-finite maximum)
  float a;     // a_s = a * sc
  float sc;    // power-of-two rescale (1 for ordinary rows)
  bool exact;  // always decide exactly (rescaled rows)
};

__device__ __forceinline__ QRow qrow_setup(float a, float qmax) {
  QRow r;
  r.sc = 1.f;
  r.exact = false;
  if (!(isfinite(a) && a > 0.f)) {
    r.inv = 0.f;
    r.a = 0.f;
    return r;
  }
  if (a > 0x1p100f) {
    r.sc = 0x1p-64f;
    r.exact = true;
  } else if (a < 0x1p-60f) {
    r.sc = 0x1p64f;
    r.exact = true;
  }
  r.a = a * r.sc;
  r.inv = __fdiv_rn(qmax, r.a);
  return r;
}

// round_half_even(qmax * u / a) for 0 <= u <= a (both already rescaled, a in [2^-60, 2^100]).
__device__ __forceinline__ int qmag_exact(float u, float a, float inv, float qmax) {
  const float p = __fmul_rn(u, inv);
  const float f = floorf(p);
  const float h = __fadd_rn(f, 0.5f);
  const float prod = __fmul_rn(qmax, u);
  const float err = __fmaf_rn(qmax, u, -prod);
  const float dd = __fmaf_rn(-h, a, prod);
  const float tot = __fadd_rn(dd, err);
  int q = (int)f;
  q += (tot > 0.f || (tot == 0.f && (q & 1))) ? 1 : 0;
  return q > (int)qmax ? (int)qmax : q;
}

// The signed code of one value of a row (0 for a non-finite value or a zero row).
__device__ __forceinline__ int qcode_exact(float v, const QRow& r, float qmax) {
  if (r.inv == 0.f || !isfinite(v)) return 0;
  const int m = qmag_exact(fabsf(v) * r.sc, r.a, r.inv, qmax);
  return v < 0.f ? -m : m;
}

// |rint(p) - p| beyond this marks a value whose fast code may differ from the exact one.
constexpr float kNearTie = 0.5f - 0x1p-18f;

// ------------------------------------------------------------------------------------------
// Shared-memory addresses, mbarriers (all waits bounded).
// ------------------------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t done;
  asm volatile(
      "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
      : "=r"(done)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return done != 0;
}

// Wait until the phase with the given parity has completed.  Returns false (and raises
// `*abort`, to `site` if it was not raised yet) if `*abort` was already raised by another thread or
// the wait exceeded the limit.
// `limit`: the wait's bound in ns (kernels whose pipeline waits take a test-settable bound pass it;
// waits that drain copies or MMAs in flight before exit always keep kWaitLimitNs).
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity, volatile int* abort, int site = 1,
                                                  uint64_t limit = kWaitLimitNs) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    // the clock is read on the first poll and every 64th (a try_wait may itself suspend for a while)
    if (it == 1u || (it & 63u) == 0u) {
      if (*abort) return false;
      if (globaltimer_ns() - t0 > limit) {
        if (*abort == 0) *abort = site;
        return false;
      }
    }
  }
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}

// ------------------------------------------------------------------------------------------
// TMA (tiled tensor copies global -> shared, completion counted on an mbarrier).
// ------------------------------------------------------------------------------------------
__device__ __forceinline__ void tma_load_2d(void* smem_dst, const CUtensorMap* map, int32_t x, int32_t y,
                                            uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
          smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void prefetch_tensormap(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// ------------------------------------------------------------------------------------------
// tcgen05 (5th-generation tensor cores, accumulators in tensor memory).
// ------------------------------------------------------------------------------------------
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// Whole warp: allocate `ncols` TMEM columns, address written to *dst (shared memory).
__device__ __forceinline__ void tmem_alloc(uint32_t* dst, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(dst)), "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

// Arrive on an mbarrier once every tcgen05.mma issued so far by this thread has completed.
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
               : "memory");
}

// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle, 8-row groups 1024 B apart.
__device__ __forceinline__ uint64_t sdesc_kmajor_sw128(uint32_t saddr) {
  return (uint64_t)((saddr >> 4) & 0x3FFFu) | (1ull << 16) | (64ull << 32) | (1ull << 46) | (2ull << 61);
}

// Instruction descriptor: dense, D fp32, A/B E4M3, both K-major, shape M x N.
__host__ __device__ constexpr uint32_t idesc_e4m3_f32(int M, int N) {
  return (1u << 4) | (0u << 7) | (0u << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

// 32 lanes x 32 consecutive 32-bit columns: thread i of the warp gets lane (base lane + i).
#define CAT_TMEM_LD32(taddr, r)                                                                                  \
  asm volatile(                                                                                                   \
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18," \
      "%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"                                              \
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),          \
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),    \
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),  \
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])   \
      : "r"(taddr))

__device__ __forceinline__ void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// ------------------------------------------------------------------------------------------
// Misc
// ------------------------------------------------------------------------------------------
template <typename T>
__device__ __forceinline__ float to_f32(T v);
template <>
__device__ __forceinline__ float to_f32<float>(float v) { return v; }
template <>
__device__ __forceinline__ float to_f32<__nv_bfloat16>(__nv_bfloat16 v) { return __bfloat162float(v); }

}  // namespace cat

// Host-side launchers implemented by the kernel translation units (all return cudaError_t).
namespace cat {
cudaError_t launch_calib_cov(const void* x, int dtype, int64_t n, int64_t d, int k, double* sigma, int accumulate,
                             uint32_t* status, cudaStream_t stream);
cudaError_t launch_transform_quantize(const void* x, int dtype, int64_t n, int64_t d, int k, const float* T,
                                      uint8_t* codes, float* scale, uint32_t* status, cudaStream_t stream,
                                      const uint8_t* planes = nullptr);
cudaError_t launch_transform_quantize_e8(const void* x, int dtype, int64_t n, int64_t d, int k, const float* A,
                                         uint8_t* codes8, float* scale, uint32_t* status, cudaStream_t stream,
                                         const uint8_t* planes);
cudaError_t launch_split_transform(const float* T, int64_t d, int k, uint8_t* planes, cudaStream_t stream);
// the group width K of the tensor-core transform for block size k on d channels (0: none applies);
// the pre-split planes take 6 d K bytes
int transform_tc_group(int k, int64_t d);
cudaError_t launch_w4a4_gemm(const uint8_t* xq, const float* sx, const uint8_t* wq, const float* sw, int64_t n,
                             int64_t d_in, int64_t d_out, float* y, int32_t* acc_out, uint32_t* status,
                             cudaStream_t stream);
cudaError_t launch_sqnr(const float* y_ref, const float* y_hat, int64_t numel, double* out3, cudaStream_t stream);
}  // namespace cat
