// W4A4 GEMM for a few tokens (decode) on the legacy mma.sync path: the fallback of the tcgen05
// weight-streaming kernel (gemm_decode_tc.cu) for token operands too large for its shared memory
// (d_in beyond ~10k codes at 16 tokens).  The packed weight stream is read once from HBM.
//
//   acc[t, o] = sum_i q_x[t, i] q_w[o, i],   y[t, o] = acc * s_x[t] * s_w[o]   (Sec. 3, Eq. 5)
//
// One CTA owns 16 weight rows; its 8 warps split d_in into 128-code chunks (chunk c -> warp c % 8,
// so the 8 warps read 512 consecutive bytes of every row per round).  A thread (group g = lane/4,
// t = lane%4) loads 16 packed bytes of rows g and g+8 per chunk with 128-bit loads and decodes
// each SM4x8 word in registers into the E4M3 operand fragments of mma.sync.m16n8k32: for the
// word u (codes 32t+8u .. +7) the low half feeds the k-slots 4t..4t+3 and the high half the
// k-slots 16+4t..16+4t+3.  The tokens use the same words and slots, so A and B agree on k.
// Each chunk accumulates from zero (|chunk sum| <= 49 * 128 * 2^-18) and is added to a running
// fp32 total; all partial sums are integers times 2^-18 below 2^24, hence exact.
#include "common.cuh"

namespace cat {
namespace {

constexpr int kWarps = 8;
constexpr int kRowsPerCta = 16;
constexpr int kChunkBytes = 64;  // 128 codes per row

__device__ __forceinline__ uint4 ldg_stream(const uint8_t* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ void mma_e4m3_16832(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                               uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k32.row.col.f32.e4m3.e4m3.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

template <int NT8>  // number of 8-token column tiles (n <= 8 * NT8 <= 32)
__global__ void __launch_bounds__(kWarps * 32) w4a4_gemm_decode_kernel(
    const uint8_t* __restrict__ xq, const float* __restrict__ sx, const uint8_t* __restrict__ wq,
    const float* __restrict__ sw, int n, int d_in, int d_out, float* __restrict__ y, int32_t* __restrict__ acc_out) {
  __shared__ float red[kWarps][kRowsPerCta][NT8 * 8];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, t = lane & 3;
  const int o0 = blockIdx.x * kRowsPerCta;
  const int64_t row_bytes = d_in / 2;
  const int num_chunks = (int)((row_bytes + kChunkBytes - 1) / kChunkBytes);
  const bool rlo_ok = o0 + g < d_out, rhi_ok = o0 + g + 8 < d_out;
  const uint8_t* wlo = wq + (int64_t)(o0 + g) * row_bytes + t * 16;
  const uint8_t* whi = wq + (int64_t)(o0 + g + 8) * row_bytes + t * 16;

  float tot[NT8][4];
#pragma unroll
  for (int j = 0; j < NT8; ++j) tot[j][0] = tot[j][1] = tot[j][2] = tot[j][3] = 0.f;

  const uint4 zero = make_uint4(0u, 0u, 0u, 0u);
  auto load_w = [&](int c, uint4& lo, uint4& hi) {
    const int64_t off = (int64_t)c * kChunkBytes;
    const bool in_k = off + t * 16 < row_bytes;
    lo = (rlo_ok && in_k) ? ldg_stream(wlo + off) : zero;
    hi = (rhi_ok && in_k) ? ldg_stream(whi + off) : zero;
  };

  int c = warp;
  uint4 wl, wh;
  if (c < num_chunks) load_w(c, wl, wh);
  for (; c < num_chunks; c += kWarps) {
    uint4 nl = zero, nh = zero;
    if (c + kWarps < num_chunks) load_w(c + kWarps, nl, nh);  // prefetch the warp's next chunk
    const int64_t off = (int64_t)c * kChunkBytes + t * 16;
    const bool in_k = off < row_bytes;
    uint4 xb[NT8];
#pragma unroll
    for (int j = 0; j < NT8; ++j) {
      const int tok = 8 * j + g;
      xb[j] = (in_k && tok < n) ? *reinterpret_cast<const uint4*>(xq + (int64_t)tok * row_bytes + off) : zero;
    }
    float part[NT8][4];
#pragma unroll
    for (int j = 0; j < NT8; ++j) part[j][0] = part[j][1] = part[j][2] = part[j][3] = 0.f;
    const uint32_t wlw[4] = {wl.x, wl.y, wl.z, wl.w};
    const uint32_t whw[4] = {wh.x, wh.y, wh.z, wh.w};
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const uint32_t a0 = sm4_lo(wlw[u]), a1 = sm4_lo(whw[u]), a2 = sm4_hi(wlw[u]), a3 = sm4_hi(whw[u]);
#pragma unroll
      for (int j = 0; j < NT8; ++j) {
        const uint32_t xw = u == 0 ? xb[j].x : (u == 1 ? xb[j].y : (u == 2 ? xb[j].z : xb[j].w));
        mma_e4m3_16832(part[j], a0, a1, a2, a3, sm4_lo(xw), sm4_hi(xw));
      }
    }
#pragma unroll
    for (int j = 0; j < NT8; ++j)
#pragma unroll
      for (int q = 0; q < 4; ++q) tot[j][q] += part[j][q];
    wl = nl;
    wh = nh;
  }

  // C fragment: tot[j][0..1] -> row g, tokens 8j+2t, 8j+2t+1; tot[j][2..3] -> row g+8, same tokens.
#pragma unroll
  for (int j = 0; j < NT8; ++j) {
    red[warp][g][8 * j + 2 * t] = tot[j][0];
    red[warp][g][8 * j + 2 * t + 1] = tot[j][1];
    red[warp][g + 8][8 * j + 2 * t] = tot[j][2];
    red[warp][g + 8][8 * j + 2 * t + 1] = tot[j][3];
  }
  __syncthreads();
  for (int e = threadIdx.x; e < kRowsPerCta * NT8 * 8; e += kWarps * 32) {
    const int tok = e / kRowsPerCta, r = e % kRowsPerCta;  // consecutive threads: consecutive rows
    const int o = o0 + r;
    if (tok >= n || o >= d_out) continue;
    float s = 0.f;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) s += red[w][r][tok];  // integers * 2^-18, exact
    y[(int64_t)tok * d_out + o] = s * kAccScale * sx[tok] * sw[o];
    if (acc_out) acc_out[(int64_t)tok * d_out + o] = __float2int_rn(s * kAccScale);
  }
}

}  // namespace

int decode_tc_stages(int64_t n, int64_t d_in);
cudaError_t launch_w4a4_gemm_decode_tc(const uint8_t* xq, const float* sx, const uint8_t* wq, const float* sw,
                                       int64_t n, int64_t d_in, int64_t d_out, float* y, int32_t* acc_out,
                                       const float* y_ref, double* sums3, uint32_t* status, cudaStream_t stream);

// n <= 32: tcgen05 weight streaming when the decoded tokens fit in shared memory, else mma.sync
// weight streaming with registers.
// y_ref != nullptr: also the SQNR sums of y against y_ref into sums3 (in the tcgen05 kernel's
// epilogue, else by the separate reduction after the GEMM).
cudaError_t launch_w4a4_gemm_decode(const uint8_t* xq, const float* sx, const uint8_t* wq, const float* sw, int64_t n,
                                    int64_t d_in, int64_t d_out, float* y, int32_t* acc_out, const float* y_ref,
                                    double* sums3, uint32_t* status, cudaStream_t stream) {
  if (decode_tc_stages(n, d_in) > 0)
    return launch_w4a4_gemm_decode_tc(xq, sx, wq, sw, n, d_in, d_out, y, acc_out, y_ref, sums3, status, stream);
  if (y_ref) {
    const cudaError_t e = launch_w4a4_gemm_decode(xq, sx, wq, sw, n, d_in, d_out, y, acc_out, nullptr, nullptr, status,
                                                  stream);
    return e != cudaSuccess ? e : launch_sqnr(y_ref, y, n * d_out, sums3, stream);
  }
  const int nt8 = (int)((n + 7) / 8);
#define CAT_DECODE_CASE(NT)                                                                                     \
  case NT: {                                                                                                    \
    const unsigned grid = (unsigned)((d_out + kRowsPerCta - 1) / kRowsPerCta);                                  \
    note_launch();                                                                                               \
    w4a4_gemm_decode_kernel<NT><<<grid, kWarps * 32, 0, stream>>>(xq, sx, wq, sw, (int)n, (int)d_in, (int)d_out, \
                                                                   y, acc_out);                                \
    break;                                                                                                      \
  }
  switch (nt8) {
    CAT_DECODE_CASE(1)
    CAT_DECODE_CASE(2)
    CAT_DECODE_CASE(3)
    CAT_DECODE_CASE(4)
    default:
      return cudaErrorInvalidValue;
  }
#undef CAT_DECODE_CASE
  return cudaGetLastError();
}

}  // namespace cat
