// C ABI of the CAT W4A4 library (declarations and contracts: include/cat_w4a4.h).
// Host-side validation, dispatch to the kernels and the per-device status word.
#include <cmath>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "../../include/cat_w4a4.h"
#include "common.cuh"
#include "transform_host.h"

namespace cat {
std::atomic<unsigned long long> g_kernel_launches{0};

cudaError_t launch_w4a4_gemm_tc(const uint8_t* xq, const float* sx, const uint8_t* wq, const float* sw, int64_t n,
                                int64_t d_in, int64_t d_out, float* y, int32_t* acc_out, const float* y_ref,
                                double* sums3, uint32_t* status, cudaStream_t stream);
cudaError_t launch_w4a4_gemm_decode(const uint8_t* xq, const float* sx, const uint8_t* wq, const float* sw, int64_t n,
                                    int64_t d_in, int64_t d_out, float* y, int32_t* acc_out, const float* y_ref,
                                    double* sums3, uint32_t* status, cudaStream_t stream);
cudaError_t launch_w4a4_gemm_tc_e8(const uint8_t* xq8, const float* sx, const uint8_t* wq8, const float* sw, int64_t n,
                                   int64_t d_in, int64_t d_out, float* y, int32_t* acc_out, const float* y_ref,
                                   double* sums3, uint32_t* status, cudaStream_t stream);
cudaError_t launch_codes_to_e4m3(const uint8_t* codes, int64_t rows, int64_t d, uint8_t* out, cudaStream_t stream);
cudaError_t launch_block_row_stats(const void* V, int dtype, int64_t rows, int64_t d, int k, const float* M,
                                   int transpose, float* row_sumsq, float* row_amax, double* out3,
                                   cudaStream_t stream);
int dp_planes(int bits, int asym);
cudaError_t launch_block_transform(const void* V, int dtype, int64_t rows, int64_t d, int k, const float* M,
                                   int transpose, float* Vt, cudaStream_t stream);
cudaError_t launch_dequantize_sm4x8(const uint8_t* codes, const float* scale, int64_t rows, int64_t d, float* out,
                                    cudaStream_t stream);
cudaError_t launch_gemm_f32_nt(const float* A, const float* B, float* C, int64_t M, int64_t N, int64_t K,
                               cudaStream_t stream);
cudaError_t launch_fwht_rows(float* V, int64_t rows, int64_t d, cudaStream_t stream);
cudaError_t launch_gram_f32(const void* X, int dtype, int64_t n, int64_t d, float* C, cudaStream_t stream);
cudaError_t set_decode_wait_limit(uint64_t ns);
cudaError_t set_dp_wait_limit(uint64_t ns);
size_t dp_l24_work_bytes(int64_t n);
cudaError_t launch_transform_quantize_dp(const void* x, int dtype, int64_t n, int64_t d, int k, const float* A, int bits,
                                         int asym, int l24, uint8_t* planes, float* scale, int32_t* zero,
                                         int32_t* rowsum, void* work, uint32_t* status, cudaStream_t stream);
cudaError_t launch_dp_gemm(const uint8_t* x_planes, int DX, const float* sx, const int32_t* zx, const uint8_t* w_planes,
                           int DW, const float* sw, const int32_t* w_rowsum, int64_t n, int64_t d_in, int64_t d_out,
                           float* y, int32_t* acc_out, uint32_t* status, cudaStream_t stream);
}  // namespace cat

namespace {

constexpr int kVersion = 10000;        // 1.0.0
constexpr int64_t kMaxDecodeTokens = 32;   // n <= 32: weight-streaming kernel; else tcgen05 tiles
constexpr int64_t kMaxDin = 262144;    // 49 * d_in < 2^24 keeps fp32 accumulation exact
// digit planes: an accumulator sums up to 2 d_in digit products of at most 15 * 8, and the int32
// result |sum (q_x - z) q_w| <= 255 * 127 * d_in: both bounded for d_in <= 2^16
constexpr int64_t kMaxDinDp = 65536;

// Device status word (one per device that loads the library).
__device__ uint32_t g_device_status;

thread_local std::string t_last_error;

cat_status fail(cat_status s, const std::string& msg) {
  t_last_error = msg;
  return s;
}

cat_status ok() {
  t_last_error.clear();
  return CAT_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

bool valid_k(int32_t k) { return k == 16 || k == 32 || k == 64 || k == 128 || k == 256; }

cat_status cuda_fail(cudaError_t e, const char* where) {
  return fail(CAT_ERR_CUDA, std::string(where) + ": " + cudaGetErrorString(e));
}

// Address of this device's status word (cached per device).
uint32_t* status_word(cudaError_t* err) {
  static std::mutex mu;
  static uint32_t* cache[64] = {nullptr};
  int dev = 0;
  *err = cudaGetDevice(&dev);
  if (*err != cudaSuccess) return nullptr;
  if (dev < 0 || dev >= 64) {
    *err = cudaErrorInvalidDevice;
    return nullptr;
  }
  std::lock_guard<std::mutex> lock(mu);
  if (!cache[dev]) {
    void* p = nullptr;
    *err = cudaGetSymbolAddress(&p, g_device_status);
    if (*err != cudaSuccess) return nullptr;
    cache[dev] = static_cast<uint32_t*>(p);
  }
  return cache[dev];
}

// Scratch of cat_quantize_weights_noalloc: it makes no device allocation of its own.
constexpr int64_t kPrepMaxDK = CAT_PREP_NOALLOC_MAX_DK;                 // largest d_in * k
constexpr size_t kPrepSigmaBytes = (size_t)kPrepMaxDK * sizeof(double);  // Sigma_w blocks
constexpr size_t kPrepScratchBytes = kPrepSigmaBytes + (size_t)kPrepMaxDK * sizeof(float);  // + A_w blocks

}  // namespace

// 12 MiB on each device where this module is loaded.  With lazy module loading (CUDA's default)
// that happens at the first use of this translation unit on the device -- in practice the first
// entry-point call there -- not when the library is loaded into the process.
static __device__ __align__(256) unsigned char g_prep_scratch[kPrepScratchBytes];

namespace {

// Address of this device's prep scratch.  Looked up once per device with that device current;
// the first cat_quantize_weights_noalloc call on a device does the lookup.
unsigned char* prep_scratch(cudaError_t* err) {
  static std::mutex mu;
  static unsigned char* cache[64] = {nullptr};
  int dev = 0;
  *err = cudaGetDevice(&dev);
  if (*err != cudaSuccess) return nullptr;
  if (dev < 0 || dev >= 64) {
    *err = cudaErrorInvalidDevice;
    return nullptr;
  }
  std::lock_guard<std::mutex> lock(mu);
  if (!cache[dev]) {
    void* p = nullptr;
    *err = cudaGetSymbolAddress(&p, g_prep_scratch);
    if (*err != cudaSuccess) return nullptr;
    cache[dev] = static_cast<unsigned char*>(p);
  }
  return cache[dev];
}

// The kernels are built for sm_103a only.
cat_status check_device() {
  int dev = 0, major = 0, minor = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if ((e = cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev)) != cudaSuccess)
    return cuda_fail(e, "cudaDeviceGetAttribute");
  if ((e = cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev)) != cudaSuccess)
    return cuda_fail(e, "cudaDeviceGetAttribute");
  if (major != 10 || minor != 3)
    return fail(CAT_ERR_UNSUPPORTED, "this library is built for sm_103a (GB300); device is sm_" +
                                         std::to_string(major) + std::to_string(minor));
  return CAT_OK;
}

cat_status check_din(int64_t d_in) {
  if (d_in <= 0 || d_in % 32 != 0) return fail(CAT_ERR_SHAPE, "d_in must be a positive multiple of 32");
  if (d_in > kMaxDin) return fail(CAT_ERR_SHAPE, "d_in exceeds 262144 (exact fp32 accumulation bound)");
  return CAT_OK;
}

// v' = H_d (A_b v_b) for every row (blocks applied as v'_b = A_b v_b, or A_b^T v_b with transpose), then
// the per-row symmetric INT4 codes of the float32 rows (identity blocks of 16).  Float32 scratch taken
// from the stream-ordered pool.
cudaError_t transform_fwht_quantize(const void* V, int dtype, int64_t rows, int64_t d, int k, const float* A,
                                    int transpose, uint8_t* codes, float* scale, uint32_t* status, cudaStream_t s) {
  float* tmp = nullptr;
  float* eye = nullptr;
  const size_t eye_elems = (size_t)(d / 16) * 256;
  cudaError_t e = cudaMallocAsync((void**)&tmp, (size_t)rows * d * sizeof(float), s);
  if (e != cudaSuccess) return e;
  if ((e = cudaMallocAsync((void**)&eye, eye_elems * sizeof(float), s)) != cudaSuccess) {
    cudaFreeAsync(tmp, s);
    return e;
  }
  std::vector<float> eye_h(eye_elems, 0.f);
  for (size_t b = 0; b < (size_t)(d / 16); ++b)
    for (int i = 0; i < 16; ++i) eye_h[b * 256 + (size_t)i * 16 + i] = 1.f;
  e = cudaMemcpyAsync(eye, eye_h.data(), eye_elems * sizeof(float), cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess) e = cat::launch_block_transform(V, dtype, rows, d, k, A, transpose, tmp, s);
  if (e == cudaSuccess) e = cat::launch_fwht_rows(tmp, rows, d, s);
  if (e == cudaSuccess) e = cat::launch_transform_quantize(tmp, 0, rows, d, 16, eye, codes, scale, status, s);
  cudaError_t e2 = cudaStreamSynchronize(s);   // eye_h is read by the copy above
  cudaFreeAsync(tmp, s);
  cudaFreeAsync(eye, s);
  return e != cudaSuccess ? e : e2;
}

}  // namespace

extern "C" {

const char* cat_status_string(cat_status status) {
  switch (status) {
    case CAT_OK: return "CAT_OK";
    case CAT_ERR_INVALID_ARG: return "CAT_ERR_INVALID_ARG";
    case CAT_ERR_SHAPE: return "CAT_ERR_SHAPE";
    case CAT_ERR_ALIGNMENT: return "CAT_ERR_ALIGNMENT";
    case CAT_ERR_NUMERIC: return "CAT_ERR_NUMERIC";
    case CAT_ERR_UNSUPPORTED: return "CAT_ERR_UNSUPPORTED";
    case CAT_ERR_CUDA: return "CAT_ERR_CUDA";
    case CAT_ERR_TIMEOUT: return "CAT_ERR_TIMEOUT";
  }
  return "CAT_ERR_UNKNOWN";
}

const char* cat_last_error(void) { return t_last_error.c_str(); }

int cat_version(void) { return kVersion; }

unsigned long long cat_kernel_launches(void) { return cat::g_kernel_launches.load(); }

cat_status cat_calib_cov(const void* x, cat_dtype dtype, int64_t n, int64_t d, int32_t k, double* sigma_blocks,
                         int accumulate, cat_stream_t stream) {
  if (dtype != CAT_F32 && dtype != CAT_BF16) return fail(CAT_ERR_INVALID_ARG, "unknown dtype");
  if (n < 0 || d <= 0) return fail(CAT_ERR_SHAPE, "n must be >= 0 and d > 0");
  if (!valid_k(k)) return fail(CAT_ERR_SHAPE, "k must be one of 16, 32, 64, 128, 256");
  if (d % k != 0) return fail(CAT_ERR_SHAPE, "k must divide d");
  if (!sigma_blocks || (n > 0 && !x)) return fail(CAT_ERR_INVALID_ARG, "NULL pointer");
  if (!aligned16(sigma_blocks) || (x && !aligned16(x))) return fail(CAT_ERR_ALIGNMENT, "pointers must be 16-byte aligned");
  if (d / k > 0x7FFFFFFF) return fail(CAT_ERR_SHAPE, "too many blocks");
  cat_status st = check_device();
  if (st != CAT_OK) return st;
  cudaError_t e;
  uint32_t* status = status_word(&e);
  if (!status) return cuda_fail(e, "status word");
  e = cat::launch_calib_cov(x, (int)dtype, n, d, k, sigma_blocks, accumulate, status, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "cat_calib_cov launch");
  return ok();
}

cat_status cat_build_transform_host(cat_tkind kind, int64_t d_in, int32_t k, const double* sigma_x_blocks,
                                    int64_t n_calib, const double* sigma_w_blocks, const float* rht_signs,
                                    double* T_out, double* Tinv_out) {
  if (kind != CAT_T_IDENTITY && kind != CAT_T_RHT && kind != CAT_T_CAT && kind != CAT_T_DIAG && kind != CAT_T_CAT_HD)
    return fail(CAT_ERR_INVALID_ARG, "unknown kind");
  if (!valid_k(k)) return fail(CAT_ERR_SHAPE, "k must be one of 16, 32, 64, 128, 256");
  if (d_in <= 0 || d_in % k != 0) return fail(CAT_ERR_SHAPE, "d_in must be a positive multiple of k");
  if (!T_out || !Tinv_out) return fail(CAT_ERR_INVALID_ARG, "NULL output");
  if (kind == CAT_T_RHT) {
    if (!rht_signs) return fail(CAT_ERR_INVALID_ARG, "RHT needs rht_signs");
    for (int64_t i = 0; i < d_in; ++i)
      if (rht_signs[i] != 1.0f && rht_signs[i] != -1.0f) return fail(CAT_ERR_INVALID_ARG, "rht_signs must be +-1");
  }
  if (kind == CAT_T_CAT || kind == CAT_T_DIAG || kind == CAT_T_CAT_HD) {
    if (!sigma_x_blocks || !sigma_w_blocks) return fail(CAT_ERR_INVALID_ARG, "CAT needs sigma_x and sigma_w blocks");
    if (n_calib < 1) return fail(CAT_ERR_INVALID_ARG, "n_calib must be >= 1");
    const size_t cnt = (size_t)d_in * (size_t)k;
    for (size_t i = 0; i < cnt; ++i)
      if (!std::isfinite(sigma_x_blocks[i]) || !std::isfinite(sigma_w_blocks[i]))
        return fail(CAT_ERR_NUMERIC, "non-finite calibration statistics");
  }
  std::string err;
  if (cat::build_transform_host((int)kind, d_in, k, sigma_x_blocks, n_calib, sigma_w_blocks, rht_signs, T_out,
                                Tinv_out, &err) != 0)
    return fail(CAT_ERR_NUMERIC, err);
  return ok();
}

cat_status cat_quantize_weights(const void* W, cat_dtype dtype, int64_t d_out, int64_t d_in, int32_t k,
                                cat_tkind kind, const double* sigma_x_blocks, int64_t n_calib,
                                const float* rht_signs, float* T_blocks, uint8_t* Wq, float* w_scale,
                                cat_stream_t stream) {
  if (dtype != CAT_F32 && dtype != CAT_BF16) return fail(CAT_ERR_INVALID_ARG, "unknown dtype");
  if (kind != CAT_T_IDENTITY && kind != CAT_T_RHT && kind != CAT_T_CAT && kind != CAT_T_DIAG && kind != CAT_T_CAT_HD)
    return fail(CAT_ERR_INVALID_ARG, "unknown kind");
  if (kind == CAT_T_CAT_HD && (d_in & (d_in - 1)) != 0) return fail(CAT_ERR_SHAPE, "the full-size Hadamard needs d_in = 2^m");
  if (kind == CAT_T_CAT_HD && d_in > 32768) return fail(CAT_ERR_SHAPE, "the full-size Hadamard needs d_in <= 32768");
  if (d_out <= 0) return fail(CAT_ERR_SHAPE, "d_out must be >= 1");
  cat_status st = check_din(d_in);
  if (st != CAT_OK) return st;
  if (!valid_k(k) || d_in % k != 0) return fail(CAT_ERR_SHAPE, "k must be one of 16..256 (power of two) and divide d_in");
  if (!W || !T_blocks || !Wq || !w_scale) return fail(CAT_ERR_INVALID_ARG, "NULL pointer");
  const bool cat_like = kind == CAT_T_CAT || kind == CAT_T_DIAG || kind == CAT_T_CAT_HD;
  if (cat_like && (!sigma_x_blocks || n_calib < 1))
    return fail(CAT_ERR_INVALID_ARG, "CAT needs sigma_x_blocks and n_calib >= 1");
  if (kind == CAT_T_RHT && !rht_signs) return fail(CAT_ERR_INVALID_ARG, "RHT needs rht_signs");
  if (!aligned16(W) || !aligned16(T_blocks) || !aligned16(Wq) || !aligned16(w_scale) ||
      (sigma_x_blocks && !aligned16(sigma_x_blocks)))
    return fail(CAT_ERR_ALIGNMENT, "pointers must be 16-byte aligned");
  if ((st = check_device()) != CAT_OK) return st;

  cudaStream_t s = (cudaStream_t)stream;
  const int64_t nb = d_in / k;
  const size_t kk = (size_t)k * k, nblk = (size_t)nb * kk;
  std::vector<double> sx_h, sw_h;
  cudaError_t e;
  if (cat_like) {
    double* sw_d = nullptr;
    if ((e = cudaMallocAsync((void**)&sw_d, nblk * sizeof(double), s)) != cudaSuccess) return cuda_fail(e, "cudaMallocAsync");
    uint32_t* st_word = status_word(&e);
    if (!st_word) return cuda_fail(e, "status word");
    e = cat::launch_calib_cov(W, (int)dtype, d_out, d_in, k, sw_d, 0, st_word, s);  // Sigma_w = W^T W blocks
    sx_h.resize(nblk);
    sw_h.resize(nblk);
    if (e == cudaSuccess) e = cudaMemcpyAsync(sx_h.data(), sigma_x_blocks, nblk * sizeof(double), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaMemcpyAsync(sw_h.data(), sw_d, nblk * sizeof(double), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    cudaFreeAsync(sw_d, s);
    if (e != cudaSuccess) return cuda_fail(e, "Sigma_w / Sigma_x readback");
  }
  std::vector<double> T(nblk), Ti(nblk);
  st = cat_build_transform_host(kind, d_in, k, sx_h.empty() ? nullptr : sx_h.data(), n_calib,
                                sw_h.empty() ? nullptr : sw_h.data(), rht_signs, T.data(), Ti.data());
  if (st != CAT_OK) return st;
  // Upload T (online transform) and A_w = (T^{-1})^T, which maps a weight row w to (W T^{-1}) row.
  std::vector<float> Tf(nblk), Awf(nblk);
  for (int64_t b = 0; b < nb; ++b)
    for (int i = 0; i < k; ++i)
      for (int j = 0; j < k; ++j) {
        Tf[b * kk + (size_t)i * k + j] = (float)T[b * kk + (size_t)i * k + j];
        Awf[b * kk + (size_t)i * k + j] = (float)Ti[b * kk + (size_t)j * k + i];
      }
  float* aw_d = nullptr;
  uint32_t* status = status_word(&e);
  if (!status) return cuda_fail(e, "status word");
  if ((e = cudaMallocAsync((void**)&aw_d, nblk * sizeof(float), s)) != cudaSuccess) return cuda_fail(e, "cudaMallocAsync");
  e = cudaMemcpyAsync(T_blocks, Tf.data(), nblk * sizeof(float), cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess) e = cudaMemcpyAsync(aw_d, Awf.data(), nblk * sizeof(float), cudaMemcpyHostToDevice, s);
  if (kind == CAT_T_CAT_HD) {
    // W' = W M^{-1} H_d: the rows through the blocks (M_b^{-1})^T, the full-size Hadamard, then the
    // codes of the float32 rows (identity blocks)
    if (e == cudaSuccess) e = transform_fwht_quantize(W, (int)dtype, d_out, d_in, k, aw_d, 1, Wq, w_scale, status, s);
  } else if (e == cudaSuccess) {
    e = cat::launch_transform_quantize(W, (int)dtype, d_out, d_in, k, aw_d, Wq, w_scale, status, s);
  }
  cudaFreeAsync(aw_d, s);
  cudaError_t e2 = cudaStreamSynchronize(s);  // host buffers above must outlive the copies
  if (e != cudaSuccess) return cuda_fail(e, "weight quantization");
  if (e2 != cudaSuccess) return cuda_fail(e2, "cudaStreamSynchronize");
  return ok();
}

// Weight preparation that takes no device memory (no counterpart in the paper).  Same steps and
// results as cat_quantize_weights; its two temporaries live in g_prep_scratch instead of
// stream-ordered allocations.  Callers that cannot allocate: a process that has handed all free
// device memory to its own pool up front (a serving engine's cache pool) and re-quantizes a
// layer later, e.g. after re-calibration -- a new allocation there fails or has to evict the
// pool.  The scratch is shared by every call on a device, so overlapping calls race.
cat_status cat_quantize_weights_noalloc(const void* W, cat_dtype dtype, int64_t d_out, int64_t d_in, int32_t k,
                                        cat_tkind kind, const double* sigma_x_blocks, int64_t n_calib,
                                        const float* rht_signs, float* T_blocks, uint8_t* Wq, float* w_scale,
                                        cat_stream_t stream) {
  if (dtype != CAT_F32 && dtype != CAT_BF16) return fail(CAT_ERR_INVALID_ARG, "unknown dtype");
  if (kind != CAT_T_IDENTITY && kind != CAT_T_RHT && kind != CAT_T_CAT) return fail(CAT_ERR_INVALID_ARG, "unknown kind");
  if (d_out <= 0) return fail(CAT_ERR_SHAPE, "d_out must be >= 1");
  cat_status st = check_din(d_in);
  if (st != CAT_OK) return st;
  if (!valid_k(k) || d_in % k != 0) return fail(CAT_ERR_SHAPE, "k must be one of 16..256 (power of two) and divide d_in");
  if (d_in * (int64_t)k > kPrepMaxDK)
    return fail(CAT_ERR_SHAPE, "cat_quantize_weights_noalloc: d_in * k = " + std::to_string(d_in * (int64_t)k) +
                                   " exceeds the static scratch limit CAT_PREP_NOALLOC_MAX_DK = " +
                                   std::to_string(kPrepMaxDK) + "; use cat_quantize_weights");
  if (!W || !T_blocks || !Wq || !w_scale) return fail(CAT_ERR_INVALID_ARG, "NULL pointer");
  if (kind == CAT_T_CAT && (!sigma_x_blocks || n_calib < 1))
    return fail(CAT_ERR_INVALID_ARG, "CAT needs sigma_x_blocks and n_calib >= 1");
  if (kind == CAT_T_RHT && !rht_signs) return fail(CAT_ERR_INVALID_ARG, "RHT needs rht_signs");
  if (!aligned16(W) || !aligned16(T_blocks) || !aligned16(Wq) || !aligned16(w_scale) ||
      (sigma_x_blocks && !aligned16(sigma_x_blocks)))
    return fail(CAT_ERR_ALIGNMENT, "pointers must be 16-byte aligned");
  if ((st = check_device()) != CAT_OK) return st;

  cudaStream_t s = (cudaStream_t)stream;
  cudaError_t e;
  unsigned char* scratch = prep_scratch(&e);
  if (!scratch) return cuda_fail(e, "cudaGetSymbolAddress(prep scratch)");
  uint32_t* status = status_word(&e);
  if (!status) return cuda_fail(e, "status word");
  double* sw_d = reinterpret_cast<double*>(scratch);                    // Sigma_w blocks, float64
  float* aw_d = reinterpret_cast<float*>(scratch + kPrepSigmaBytes);    // (T_b^{-1})^T blocks, float32
  const int64_t nb = d_in / k;
  const size_t kk = (size_t)k * k, nblk = (size_t)nb * kk;
  std::vector<double> sx_h, sw_h;
  if (kind == CAT_T_CAT) {
    // The Sigma_w sums accumulate into the scratch, so it must start at zero on every call.
    e = cudaMemsetAsync(sw_d, 0, nblk * sizeof(double), s);
    if (e == cudaSuccess) e = cat::launch_calib_cov(W, (int)dtype, d_out, d_in, k, sw_d, 1, status, s);
    sx_h.resize(nblk);
    sw_h.resize(nblk);
    if (e == cudaSuccess) e = cudaMemcpyAsync(sx_h.data(), sigma_x_blocks, nblk * sizeof(double), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaMemcpyAsync(sw_h.data(), sw_d, nblk * sizeof(double), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(e, "Sigma_w / Sigma_x readback");
  }
  std::vector<double> T(nblk), Ti(nblk);
  st = cat_build_transform_host(kind, d_in, k, sx_h.empty() ? nullptr : sx_h.data(), n_calib,
                                sw_h.empty() ? nullptr : sw_h.data(), rht_signs, T.data(), Ti.data());
  if (st != CAT_OK) return st;
  std::vector<float> Tf(nblk), Awf(nblk);
  for (int64_t b = 0; b < nb; ++b)
    for (int i = 0; i < k; ++i)
      for (int j = 0; j < k; ++j) {
        Tf[b * kk + (size_t)i * k + j] = (float)T[b * kk + (size_t)i * k + j];
        Awf[b * kk + (size_t)i * k + j] = (float)Ti[b * kk + (size_t)j * k + i];
      }
  e = cudaMemcpyAsync(T_blocks, Tf.data(), nblk * sizeof(float), cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess) e = cudaMemcpyAsync(aw_d, Awf.data(), nblk * sizeof(float), cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess) e = cat::launch_transform_quantize(W, (int)dtype, d_out, d_in, k, aw_d, Wq, w_scale, status, s);
  cudaError_t e2 = cudaStreamSynchronize(s);  // host buffers and the scratch are in use until here
  if (e != cudaSuccess) return cuda_fail(e, "weight quantization");
  if (e2 != cudaSuccess) return cuda_fail(e2, "cudaStreamSynchronize");
  return ok();
}

// ---- b-bit codes as E4M3 digit planes (bit widths; Sec. 6's asymmetric activations and L_2.4 range)

int32_t cat_dp_planes(int32_t bits) { return (bits >= 2 && bits <= 8) ? (int32_t)cat::dp_planes(bits, 0) : 0; }

cat_status cat_transform_quantize_act_dp(const void* x, cat_dtype dtype, int64_t n, int64_t d_in, int32_t k,
                                         const float* T_blocks, int32_t bits, int32_t asymmetric, uint8_t* planes,
                                         float* x_scale, int32_t* x_zero, cat_stream_t stream) {
  if (dtype != CAT_F32 && dtype != CAT_BF16) return fail(CAT_ERR_INVALID_ARG, "unknown dtype");
  if (bits < 2 || bits > 8) return fail(CAT_ERR_SHAPE, "bits must be in 2..8");
  if (asymmetric != 0 && asymmetric != 1) return fail(CAT_ERR_INVALID_ARG, "asymmetric must be 0 or 1");
  if (n < 0) return fail(CAT_ERR_SHAPE, "n must be >= 0");
  cat_status st = check_din(d_in);
  if (st != CAT_OK) return st;
  if (d_in > kMaxDinDp) return fail(CAT_ERR_SHAPE, "d_in exceeds 65536 (exact digit-plane accumulation bound)");
  if (!valid_k(k) || d_in % k != 0) return fail(CAT_ERR_SHAPE, "k must be one of 16..256 (power of two) and divide d_in");
  if (n == 0) return ok();
  if (!x || !T_blocks || !planes || !x_scale || (asymmetric && !x_zero)) return fail(CAT_ERR_INVALID_ARG, "NULL pointer");
  if (!aligned16(x) || !aligned16(T_blocks) || !aligned16(planes) || !aligned16(x_scale) || (x_zero && !aligned16(x_zero)))
    return fail(CAT_ERR_ALIGNMENT, "pointers must be 16-byte aligned");
  if ((n + 63) / 64 > 0x7FFFFFFF) return fail(CAT_ERR_SHAPE, "n too large");
  if ((st = check_device()) != CAT_OK) return st;
  cudaError_t e;
  uint32_t* status = status_word(&e);
  if (!status) return cuda_fail(e, "status word");
  e = cat::launch_transform_quantize_dp(x, (int)dtype, n, d_in, k, T_blocks, bits, asymmetric, 0, planes, x_scale,
                                        asymmetric ? x_zero : nullptr, nullptr, nullptr, status, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "cat_transform_quantize_act_dp launch");
  return ok();
}

cat_status cat_quantize_weights_dp(const void* W, cat_dtype dtype, int64_t d_out, int64_t d_in, int32_t k,
                                   cat_tkind kind, const double* sigma_x_blocks, int64_t n_calib,
                                   const float* rht_signs, int32_t bits, int32_t l24_range, float* T_blocks,
                                   uint8_t* planes, float* w_scale, int32_t* w_rowsum, cat_stream_t stream) {
  if (dtype != CAT_F32 && dtype != CAT_BF16) return fail(CAT_ERR_INVALID_ARG, "unknown dtype");
  if (kind != CAT_T_IDENTITY && kind != CAT_T_RHT && kind != CAT_T_CAT) return fail(CAT_ERR_INVALID_ARG, "unknown kind");
  if (bits < 2 || bits > 8) return fail(CAT_ERR_SHAPE, "bits must be in 2..8");
  if (l24_range != 0 && l24_range != 1) return fail(CAT_ERR_INVALID_ARG, "l24_range must be 0 or 1");
  if (d_out <= 0 || d_out > 0x7FFFFFFF) return fail(CAT_ERR_SHAPE, "d_out must be in [1, 2^31)");
  cat_status st = check_din(d_in);
  if (st != CAT_OK) return st;
  if (d_in > kMaxDinDp) return fail(CAT_ERR_SHAPE, "d_in exceeds 65536 (exact digit-plane accumulation bound)");
  if (!valid_k(k) || d_in % k != 0) return fail(CAT_ERR_SHAPE, "k must be one of 16..256 (power of two) and divide d_in");
  if (!W || !T_blocks || !planes || !w_scale) return fail(CAT_ERR_INVALID_ARG, "NULL pointer");
  if (kind == CAT_T_CAT && (!sigma_x_blocks || n_calib < 1))
    return fail(CAT_ERR_INVALID_ARG, "CAT needs sigma_x_blocks and n_calib >= 1");
  if (kind == CAT_T_RHT && !rht_signs) return fail(CAT_ERR_INVALID_ARG, "RHT needs rht_signs");
  if (!aligned16(W) || !aligned16(T_blocks) || !aligned16(planes) || !aligned16(w_scale) ||
      (w_rowsum && !aligned16(w_rowsum)) || (sigma_x_blocks && !aligned16(sigma_x_blocks)))
    return fail(CAT_ERR_ALIGNMENT, "pointers must be 16-byte aligned");
  if ((st = check_device()) != CAT_OK) return st;

  cudaStream_t s = (cudaStream_t)stream;
  const int64_t nb = d_in / k;
  const size_t kk = (size_t)k * k, nblk = (size_t)nb * kk;
  std::vector<double> sx_h, sw_h;
  cudaError_t e;
  if (kind == CAT_T_CAT) {
    double* sw_d = nullptr;
    if ((e = cudaMallocAsync((void**)&sw_d, nblk * sizeof(double), s)) != cudaSuccess) return cuda_fail(e, "cudaMallocAsync");
    uint32_t* st_word = status_word(&e);
    if (!st_word) return cuda_fail(e, "status word");
    e = cat::launch_calib_cov(W, (int)dtype, d_out, d_in, k, sw_d, 0, st_word, s);  // Sigma_w = W^T W blocks
    sx_h.resize(nblk);
    sw_h.resize(nblk);
    if (e == cudaSuccess) e = cudaMemcpyAsync(sx_h.data(), sigma_x_blocks, nblk * sizeof(double), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaMemcpyAsync(sw_h.data(), sw_d, nblk * sizeof(double), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    cudaFreeAsync(sw_d, s);
    if (e != cudaSuccess) return cuda_fail(e, "Sigma_w / Sigma_x readback");
  }
  std::vector<double> T(nblk), Ti(nblk);
  st = cat_build_transform_host(kind, d_in, k, sx_h.empty() ? nullptr : sx_h.data(), n_calib,
                                sw_h.empty() ? nullptr : sw_h.data(), rht_signs, T.data(), Ti.data());
  if (st != CAT_OK) return st;
  std::vector<float> Tf(nblk), Awf(nblk);
  for (int64_t b = 0; b < nb; ++b)
    for (int i = 0; i < k; ++i)
      for (int j = 0; j < k; ++j) {
        Tf[b * kk + (size_t)i * k + j] = (float)T[b * kk + (size_t)i * k + j];
        Awf[b * kk + (size_t)i * k + j] = (float)Ti[b * kk + (size_t)j * k + i];
      }
  uint32_t* status = status_word(&e);
  if (!status) return cuda_fail(e, "status word");
  float* aw_d = nullptr;
  void* work = nullptr;
  const size_t work_bytes = l24_range ? cat::dp_l24_work_bytes(d_out) : 0;
  if ((e = cudaMallocAsync((void**)&aw_d, nblk * sizeof(float), s)) != cudaSuccess) return cuda_fail(e, "cudaMallocAsync");
  if (work_bytes && (e = cudaMallocAsync(&work, work_bytes, s)) != cudaSuccess) {
    cudaFreeAsync(aw_d, s);
    return cuda_fail(e, "cudaMallocAsync");
  }
  if (work_bytes) e = cudaMemsetAsync(work, 0, work_bytes, s);
  if (e == cudaSuccess) e = cudaMemcpyAsync(T_blocks, Tf.data(), nblk * sizeof(float), cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess) e = cudaMemcpyAsync(aw_d, Awf.data(), nblk * sizeof(float), cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess)
    e = cat::launch_transform_quantize_dp(W, (int)dtype, d_out, d_in, k, aw_d, bits, 0, l24_range, planes, w_scale,
                                          nullptr, w_rowsum, work, status, s);
  cudaFreeAsync(aw_d, s);
  if (work) cudaFreeAsync(work, s);
  cudaError_t e2 = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(e, "weight quantization (digit planes)");
  if (e2 != cudaSuccess) return cuda_fail(e2, "cudaStreamSynchronize");
  return ok();
}

cat_status cat_linear_dp(const uint8_t* x_planes, int32_t bits_x, int32_t asym_x, const float* x_scale,
                         const int32_t* x_zero, const uint8_t* w_planes, int32_t bits_w, const float* w_scale,
                         const int32_t* w_rowsum, int64_t n, int64_t d_in, int64_t d_out, float* y, int32_t* acc_out,
                         cat_stream_t stream) {
  if (bits_x < 2 || bits_x > 8 || bits_w < 2 || bits_w > 8) return fail(CAT_ERR_SHAPE, "bits must be in 2..8");
  if (asym_x != 0 && asym_x != 1) return fail(CAT_ERR_INVALID_ARG, "asym_x must be 0 or 1");
  if (n < 0 || d_out <= 0) return fail(CAT_ERR_SHAPE, "n must be >= 0 and d_out >= 1");
  cat_status st = check_din(d_in);
  if (st != CAT_OK) return st;
  if (d_in > kMaxDinDp) return fail(CAT_ERR_SHAPE, "d_in exceeds 65536 (exact digit-plane accumulation bound)");
  if (n > 0x7FFFFFFF || d_out > 0x7FFFFFFF || (n + 127) / 128 > 65535) return fail(CAT_ERR_SHAPE, "n or d_out too large");
  if (n == 0) return ok();
  if (!x_planes || !x_scale || !w_planes || !w_scale || !y || (asym_x && (!x_zero || !w_rowsum)))
    return fail(CAT_ERR_INVALID_ARG, "NULL pointer (asymmetric activations need x_zero and w_rowsum)");
  if (!aligned16(x_planes) || !aligned16(x_scale) || !aligned16(w_planes) || !aligned16(w_scale) || !aligned16(y) ||
      (x_zero && !aligned16(x_zero)) || (w_rowsum && !aligned16(w_rowsum)) || (acc_out && !aligned16(acc_out)))
    return fail(CAT_ERR_ALIGNMENT, "pointers must be 16-byte aligned");
  if ((st = check_device()) != CAT_OK) return st;
  cudaError_t e;
  uint32_t* status = status_word(&e);
  if (!status) return cuda_fail(e, "status word");
  e = cat::launch_dp_gemm(x_planes, cat::dp_planes(bits_x, asym_x), x_scale, asym_x ? x_zero : nullptr, w_planes,
                          cat::dp_planes(bits_w, 0), w_scale, asym_x ? w_rowsum : nullptr, n, d_in, d_out, y, acc_out,
                          status, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "cat_linear_dp launch");
  return ok();
}

cat_status cat_transform_quantize_act(const void* x, cat_dtype dtype, int64_t n, int64_t d_in, int32_t k,
                                      const float* T_blocks, uint8_t* xq, float* x_scale, cat_stream_t stream) {
  if (dtype != CAT_F32 && dtype != CAT_BF16) return fail(CAT_ERR_INVALID_ARG, "unknown dtype");
  if (n < 0) return fail(CAT_ERR_SHAPE, "n must be >= 0");
  cat_status st = check_din(d_in);
  if (st != CAT_OK) return st;
  if (!valid_k(k) || d_in % k != 0) return fail(CAT_ERR_SHAPE, "k must be one of 16..256 (power of two) and divide d_in");
  if (n == 0) return ok();
  if (!x || !T_blocks || !xq || !x_scale) return fail(CAT_ERR_INVALID_ARG, "NULL pointer");
  if (!aligned16(x) || !aligned16(T_blocks) || !aligned16(xq) || !aligned16(x_scale))
    return fail(CAT_ERR_ALIGNMENT, "pointers must be 16-byte aligned");
  if ((n + 63) / 64 > 0x7FFFFFFF) return fail(CAT_ERR_SHAPE, "n too large");
  if ((st = check_device()) != CAT_OK) return st;
  cudaError_t e;
  uint32_t* status = status_word(&e);
  if (!status) return cuda_fail(e, "status word");
  e = cat::launch_transform_quantize(x, (int)dtype, n, d_in, k, T_blocks, xq, x_scale, status, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "cat_transform_quantize_act launch");
  return ok();
}

int64_t cat_split_transform_bytes(int64_t d_in, int32_t k) {
  if (d_in <= 0 || !valid_k(k) || d_in % k != 0) return 0;
  return 6 * d_in * (int64_t)cat::transform_tc_group(k, d_in);
}

cat_status cat_split_transform(const float* T_blocks, int64_t d_in, int32_t k, uint8_t* planes, cat_stream_t stream) {
  cat_status st = check_din(d_in);
  if (st != CAT_OK) return st;
  if (!valid_k(k) || d_in % k != 0) return fail(CAT_ERR_SHAPE, "k must be one of 16..256 (power of two) and divide d_in");
  if (cat::transform_tc_group(k, d_in) == 0)
    return fail(CAT_ERR_UNSUPPORTED, "pre-split planes serve the tensor-core transform: k <= 128 with 128 | d_in, or k = 64");
  if (!T_blocks || !planes) return fail(CAT_ERR_INVALID_ARG, "NULL pointer");
  if (!aligned16(T_blocks) || !aligned16(planes)) return fail(CAT_ERR_ALIGNMENT, "pointers must be 16-byte aligned");
  if ((st = check_device()) != CAT_OK) return st;
  cudaError_t e = cat::launch_split_transform(T_blocks, d_in, k, planes, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "cat_split_transform launch");
  return ok();
}

cat_status cat_transform_quantize_act_split(const void* x, cat_dtype dtype, int64_t n, int64_t d_in, int32_t k,
                                            const float* T_blocks, const uint8_t* T_planes, uint8_t* xq, float* x_scale,
                                            cat_stream_t stream) {
  if (dtype != CAT_F32 && dtype != CAT_BF16) return fail(CAT_ERR_INVALID_ARG, "unknown dtype");
  if (n < 0) return fail(CAT_ERR_SHAPE, "n must be >= 0");
  cat_status st = check_din(d_in);
  if (st != CAT_OK) return st;
  if (!valid_k(k) || d_in % k != 0) return fail(CAT_ERR_SHAPE, "k must be one of 16..256 (power of two) and divide d_in");
  if (n == 0) return ok();
  if (!x || !T_blocks || !xq || !x_scale) return fail(CAT_ERR_INVALID_ARG, "NULL pointer");
  if (!aligned16(x) || !aligned16(T_blocks) || !aligned16(xq) || !aligned16(x_scale) || (T_planes && !aligned16(T_planes)))
    return fail(CAT_ERR_ALIGNMENT, "pointers must be 16-byte aligned");
  if ((n + 63) / 64 > 0x7FFFFFFF) return fail(CAT_ERR_SHAPE, "n too large");
  if ((st = check_device()) != CAT_OK) return st;
  cudaError_t e;
  uint32_t* status = status_word(&e);
  if (!status) return cuda_fail(e, "status word");
  e = cat::launch_transform_quantize(x, (int)dtype, n, d_in, k, T_blocks, xq, x_scale, status, (cudaStream_t)stream,
                                     cat::transform_tc_group(k, d_in) != 0 ? T_planes : nullptr);
  if (e != cudaSuccess) return cuda_fail(e, "cat_transform_quantize_act_split launch");
  return ok();
}

cat_status cat_w4a4_linear(const uint8_t* xq, const float* x_scale, const uint8_t* Wq, const float* w_scale,
                           int64_t n, int64_t d_in, int64_t d_out, float* y, int32_t* acc_out, cat_stream_t stream) {
  if (n < 0 || d_out <= 0) return fail(CAT_ERR_SHAPE, "n must be >= 0 and d_out >= 1");
  cat_status st = check_din(d_in);
  if (st != CAT_OK) return st;
  if (n > 0x7FFFFFFF || d_out > 0x7FFFFFFF) return fail(CAT_ERR_SHAPE, "n and d_out must fit in int32");
  if (n == 0) return ok();
  if (!xq || !x_scale || !Wq || !w_scale || !y) return fail(CAT_ERR_INVALID_ARG, "NULL pointer");
  if (!aligned16(xq) || !aligned16(x_scale) || !aligned16(Wq) || !aligned16(w_scale) || !aligned16(y) ||
      (acc_out && !aligned16(acc_out)))
    return fail(CAT_ERR_ALIGNMENT, "pointers must be 16-byte aligned");
  if ((st = check_device()) != CAT_OK) return st;
  cudaError_t e;
  uint32_t* status = status_word(&e);
  if (!status) return cuda_fail(e, "status word");
  if (n <= kMaxDecodeTokens)
    e = cat::launch_w4a4_gemm_decode(xq, x_scale, Wq, w_scale, n, d_in, d_out, y, acc_out, nullptr, nullptr, status,
                                     (cudaStream_t)stream);
  else
    e = cat::launch_w4a4_gemm_tc(xq, x_scale, Wq, w_scale, n, d_in, d_out, y, acc_out, nullptr, nullptr, status,
                                 (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "cat_w4a4_linear launch");
  return ok();
}

cat_status cat_w4a4_linear_sqnr(const uint8_t* xq, const float* x_scale, const uint8_t* Wq, const float* w_scale,
                                int64_t n, int64_t d_in, int64_t d_out, float* y, const float* y_ref, double* out3,
                                cat_stream_t stream) {
  if (n < 0 || d_out <= 0) return fail(CAT_ERR_SHAPE, "n must be >= 0 and d_out >= 1");
  cat_status st = check_din(d_in);
  if (st != CAT_OK) return st;
  if (n > 0x7FFFFFFF || d_out > 0x7FFFFFFF) return fail(CAT_ERR_SHAPE, "n and d_out must fit in int32");
  if (!out3 || (n > 0 && (!xq || !x_scale || !Wq || !w_scale || !y || !y_ref)))
    return fail(CAT_ERR_INVALID_ARG, "NULL pointer");
  if (!aligned16(out3) || (n > 0 && (!aligned16(xq) || !aligned16(x_scale) || !aligned16(Wq) || !aligned16(w_scale) ||
                                     !aligned16(y) || !aligned16(y_ref))))
    return fail(CAT_ERR_ALIGNMENT, "pointers must be 16-byte aligned");
  if ((st = check_device()) != CAT_OK) return st;
  cudaError_t e;
  uint32_t* status = status_word(&e);
  if (!status) return cuda_fail(e, "status word");
  cudaStream_t s = (cudaStream_t)stream;
  if (n > kMaxDecodeTokens && d_out % 4 == 0) {  // SQNR sums fused into the GEMM epilogue
    e = cat::launch_w4a4_gemm_tc(xq, x_scale, Wq, w_scale, n, d_in, d_out, y, nullptr, y_ref, out3, status, s);
  } else if (n > 0 && n <= kMaxDecodeTokens) {  // weight streaming; sums in its epilogue where it can
    e = cat::launch_w4a4_gemm_decode(xq, x_scale, Wq, w_scale, n, d_in, d_out, y, nullptr, y_ref, out3, status, s);
  } else {  // the GEMM, then the separate reduction
    e = n == 0 ? cudaSuccess
               : cat::launch_w4a4_gemm_tc(xq, x_scale, Wq, w_scale, n, d_in, d_out, y, nullptr, nullptr, nullptr,
                                          status, s);
    if (e == cudaSuccess) e = cat::launch_sqnr(y_ref, y, n * d_out, out3, s);
  }
  if (e != cudaSuccess) return cuda_fail(e, "cat_w4a4_linear_sqnr launch");
  return ok();
}

// ---- byte codes: one E4M3 byte per code, for the tensor cores to read as they are

cat_status cat_codes_to_e4m3(const uint8_t* codes, int64_t rows, int64_t d, uint8_t* out, cat_stream_t stream) {
  if (rows < 0 || d <= 0 || d % 32 != 0) return fail(CAT_ERR_SHAPE, "rows >= 0 and d a positive multiple of 32");
  if (rows > ((int64_t)1 << 40) / d) return fail(CAT_ERR_SHAPE, "rows x d too large");
  if (rows == 0) return ok();
  if (!codes || !out) return fail(CAT_ERR_INVALID_ARG, "NULL pointer");
  if (!aligned16(codes) || !aligned16(out)) return fail(CAT_ERR_ALIGNMENT, "pointers must be 16-byte aligned");
  cat_status st = check_device();
  if (st != CAT_OK) return st;
  cudaError_t e = cat::launch_codes_to_e4m3(codes, rows, d, out, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "cat_codes_to_e4m3 launch");
  return ok();
}

cat_status cat_transform_quantize_act_e8(const void* x, cat_dtype dtype, int64_t n, int64_t d_in, int32_t k,
                                         const float* T_blocks, const uint8_t* T_planes, uint8_t* xq8, float* x_scale,
                                         cat_stream_t stream) {
  if (dtype != CAT_F32 && dtype != CAT_BF16) return fail(CAT_ERR_INVALID_ARG, "unknown dtype");
  if (n < 0) return fail(CAT_ERR_SHAPE, "n must be >= 0");
  cat_status st = check_din(d_in);
  if (st != CAT_OK) return st;
  if (!valid_k(k) || d_in % k != 0) return fail(CAT_ERR_SHAPE, "k must be one of 16..256 (power of two) and divide d_in");
  if (n == 0) return ok();
  if (!x || !T_blocks || !xq8 || !x_scale) return fail(CAT_ERR_INVALID_ARG, "NULL pointer");
  if (!aligned16(x) || !aligned16(T_blocks) || !aligned16(xq8) || !aligned16(x_scale) || (T_planes && !aligned16(T_planes)))
    return fail(CAT_ERR_ALIGNMENT, "pointers must be 16-byte aligned");
  if ((n + 63) / 64 > 0x7FFFFFFF) return fail(CAT_ERR_SHAPE, "n too large");
  if ((st = check_device()) != CAT_OK) return st;
  cudaError_t e;
  uint32_t* status = status_word(&e);
  if (!status) return cuda_fail(e, "status word");
  cudaStream_t s = (cudaStream_t)stream;
  const uint8_t* planes = cat::transform_tc_group(k, d_in) != 0 ? T_planes : nullptr;
  e = cat::launch_transform_quantize_e8(x, (int)dtype, n, d_in, k, T_blocks, xq8, x_scale, status, s, planes);
  if (e == cudaErrorNotSupported) {
    // no kernel writes byte codes here: SM4x8 codes into stream-ordered scratch, then converted
    uint8_t* tmp = nullptr;
    if ((e = cudaMallocAsync((void**)&tmp, (size_t)n * (size_t)(d_in / 2), s)) != cudaSuccess)
      return cuda_fail(e, "cudaMallocAsync");
    e = cat::launch_transform_quantize(x, (int)dtype, n, d_in, k, T_blocks, tmp, x_scale, status, s, planes);
    if (e == cudaSuccess) e = cat::launch_codes_to_e4m3(tmp, n, d_in, xq8, s);
    const cudaError_t ef = cudaFreeAsync(tmp, s);
    if (e == cudaSuccess) e = ef;
  }
  if (e != cudaSuccess) return cuda_fail(e, "cat_transform_quantize_act_e8 launch");
  return ok();
}

cat_status cat_w4a4_linear_e8(const uint8_t* xq8, const float* x_scale, const uint8_t* Wq8, const float* w_scale,
                              int64_t n, int64_t d_in, int64_t d_out, float* y, int32_t* acc_out, cat_stream_t stream) {
  if (n < 0 || d_out <= 0) return fail(CAT_ERR_SHAPE, "n must be >= 0 and d_out >= 1");
  cat_status st = check_din(d_in);
  if (st != CAT_OK) return st;
  if (n > 0x7FFFFFFF || d_out > 0x7FFFFFFF) return fail(CAT_ERR_SHAPE, "n and d_out must fit in int32");
  if (n == 0) return ok();
  if (!xq8 || !x_scale || !Wq8 || !w_scale || !y) return fail(CAT_ERR_INVALID_ARG, "NULL pointer");
  if (!aligned16(xq8) || !aligned16(x_scale) || !aligned16(Wq8) || !aligned16(w_scale) || !aligned16(y) ||
      (acc_out && !aligned16(acc_out)))
    return fail(CAT_ERR_ALIGNMENT, "pointers must be 16-byte aligned");
  if ((st = check_device()) != CAT_OK) return st;
  cudaError_t e;
  uint32_t* status = status_word(&e);
  if (!status) return cuda_fail(e, "status word");
  e = cat::launch_w4a4_gemm_tc_e8(xq8, x_scale, Wq8, w_scale, n, d_in, d_out, y, acc_out, nullptr, nullptr, status,
                                  (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "cat_w4a4_linear_e8 launch");
  return ok();
}

cat_status cat_w4a4_linear_sqnr_e8(const uint8_t* xq8, const float* x_scale, const uint8_t* Wq8, const float* w_scale,
                                   int64_t n, int64_t d_in, int64_t d_out, float* y, const float* y_ref, double* out3,
                                   cat_stream_t stream) {
  if (n < 0 || d_out <= 0) return fail(CAT_ERR_SHAPE, "n must be >= 0 and d_out >= 1");
  cat_status st = check_din(d_in);
  if (st != CAT_OK) return st;
  if (n > 0x7FFFFFFF || d_out > 0x7FFFFFFF) return fail(CAT_ERR_SHAPE, "n and d_out must fit in int32");
  if (!out3 || (n > 0 && (!xq8 || !x_scale || !Wq8 || !w_scale || !y || !y_ref)))
    return fail(CAT_ERR_INVALID_ARG, "NULL pointer");
  if (!aligned16(out3) || (n > 0 && (!aligned16(xq8) || !aligned16(x_scale) || !aligned16(Wq8) ||
                                     !aligned16(w_scale) || !aligned16(y) || !aligned16(y_ref))))
    return fail(CAT_ERR_ALIGNMENT, "pointers must be 16-byte aligned");
  if ((st = check_device()) != CAT_OK) return st;
  cudaError_t e;
  uint32_t* status = status_word(&e);
  if (!status) return cuda_fail(e, "status word");
  cudaStream_t s = (cudaStream_t)stream;
  if (n > 0 && d_out % 4 == 0) {  // SQNR sums fused into the GEMM epilogue
    e = cat::launch_w4a4_gemm_tc_e8(xq8, x_scale, Wq8, w_scale, n, d_in, d_out, y, nullptr, y_ref, out3, status, s);
  } else {                        // the GEMM, then the separate reduction
    e = n == 0 ? cudaSuccess
               : cat::launch_w4a4_gemm_tc_e8(xq8, x_scale, Wq8, w_scale, n, d_in, d_out, y, nullptr, nullptr, nullptr,
                                             status, s);
    if (e == cudaSuccess) e = cat::launch_sqnr(y_ref, y, n * d_out, out3, s);
  }
  if (e != cudaSuccess) return cuda_fail(e, "cat_w4a4_linear_sqnr_e8 launch");
  return ok();
}

cat_status cat_sqnr(const float* y_ref, const float* y_hat, int64_t numel, double* out3, cat_stream_t stream) {
  if (numel < 0) return fail(CAT_ERR_SHAPE, "numel must be >= 0");
  if (!out3 || (numel > 0 && (!y_ref || !y_hat))) return fail(CAT_ERR_INVALID_ARG, "NULL pointer");
  if (!aligned16(out3) || (y_ref && !aligned16(y_ref)) || (y_hat && !aligned16(y_hat)))
    return fail(CAT_ERR_ALIGNMENT, "pointers must be 16-byte aligned");
  cat_status st = check_device();
  if (st != CAT_OK) return st;
  cudaError_t e = cat::launch_sqnr(y_ref, y_hat, numel, out3, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "cat_sqnr launch");
  return ok();
}

cat_status cat_set_wait_limit_ns(uint64_t ns) {
  if (ns > cat::kWaitLimitNs) return fail(CAT_ERR_INVALID_ARG, "the wait limit is at most 1 s (1e9 ns)");
  const uint64_t v = ns == 0 ? cat::kWaitLimitNs : ns;
  cat_status st = check_device();
  if (st != CAT_OK) return st;
  cudaError_t e = cat::set_decode_wait_limit(v);
  if (e == cudaSuccess) e = cat::set_dp_wait_limit(v);
  if (e != cudaSuccess) return cuda_fail(e, "cat_set_wait_limit_ns");
  return ok();
}

cat_status cat_device_status(cat_stream_t stream, uint32_t* detail) {
  cudaError_t e = cudaStreamSynchronize((cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
  uint32_t v = 0, zero = 0;
  if ((e = cudaMemcpyFromSymbol(&v, g_device_status, sizeof(v))) != cudaSuccess) return cuda_fail(e, "read status");
  if ((e = cudaMemcpyToSymbol(g_device_status, &zero, sizeof(zero))) != cudaSuccess) return cuda_fail(e, "clear status");
  if (detail) *detail = v;
  if (v & cat::kStatusTimeout) return fail(CAT_ERR_TIMEOUT, "a bounded device wait gave up");
  if (v & cat::kStatusNonFinite) return fail(CAT_ERR_NUMERIC, "a kernel met a non-finite value");
  return ok();
}

}  // extern "C"

cat_status cat_block_row_stats(const void* V, cat_dtype dtype, int64_t rows, int64_t d, int32_t k,
                               const float* M_blocks, int transpose, float* row_sumsq, float* row_amax, double* out3,
                               cat_stream_t stream) {
  if (dtype != CAT_F32 && dtype != CAT_BF16) return fail(CAT_ERR_INVALID_ARG, "unknown dtype");
  if (rows < 1 || rows > 0x7FFFFFFF) return fail(CAT_ERR_SHAPE, "rows must be in [1, 2^31)");
  cat_status st = check_din(d);
  if (st != CAT_OK) return st;
  if (!valid_k(k) || d % k != 0) return fail(CAT_ERR_SHAPE, "k must be one of 16..256 (power of two) and divide d");
  if (transpose != 0 && transpose != 1) return fail(CAT_ERR_INVALID_ARG, "transpose must be 0 or 1");
  if (!V || !M_blocks || !row_sumsq || !row_amax || !out3) return fail(CAT_ERR_INVALID_ARG, "NULL pointer");
  if (!aligned16(V) || !aligned16(M_blocks) || !aligned16(row_sumsq) || !aligned16(row_amax) || !aligned16(out3))
    return fail(CAT_ERR_ALIGNMENT, "pointers must be 16-byte aligned");
  if ((st = check_device()) != CAT_OK) return st;
  cudaError_t e = cat::launch_block_row_stats(V, (int)dtype, rows, d, k, M_blocks, transpose, row_sumsq, row_amax, out3,
                                              (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "cat_block_row_stats launch");
  return ok();
}

// ---- building blocks of the one-sided SQNRs (Lemmas 2 and 3), off the hot path

cat_status cat_block_transform(const void* V, cat_dtype dtype, int64_t rows, int64_t d, int32_t k,
                               const float* M_blocks, int transpose, float* out, cat_stream_t stream) {
  if (dtype != CAT_F32 && dtype != CAT_BF16) return fail(CAT_ERR_INVALID_ARG, "unknown dtype");
  if (rows < 1 || rows > 0x7FFFFFFF) return fail(CAT_ERR_SHAPE, "rows must be in [1, 2^31)");
  cat_status st = check_din(d);
  if (st != CAT_OK) return st;
  if (!valid_k(k) || d % k != 0) return fail(CAT_ERR_SHAPE, "k must be one of 16..256 (power of two) and divide d");
  if ((rows + 63) / 64 > 0x7FFFFFFF || d / k > 65535) return fail(CAT_ERR_SHAPE, "too many rows or blocks");
  if (transpose != 0 && transpose != 1) return fail(CAT_ERR_INVALID_ARG, "transpose must be 0 or 1");
  if (!V || !M_blocks || !out) return fail(CAT_ERR_INVALID_ARG, "NULL pointer");
  if (!aligned16(V) || !aligned16(M_blocks) || !aligned16(out)) return fail(CAT_ERR_ALIGNMENT, "pointers must be 16-byte aligned");
  if ((st = check_device()) != CAT_OK) return st;
  cudaError_t e = cat::launch_block_transform(V, (int)dtype, rows, d, k, M_blocks, transpose, out, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "cat_block_transform launch");
  return ok();
}

cat_status cat_dequantize_codes(const uint8_t* codes, const float* scale, int64_t rows, int64_t d, float* out,
                                cat_stream_t stream) {
  if (rows < 0) return fail(CAT_ERR_SHAPE, "rows must be >= 0");
  cat_status st = check_din(d);
  if (st != CAT_OK) return st;
  if (rows == 0) return ok();
  if (rows * (d / 8) / 256 + 1 > 0x7FFFFFFF) return fail(CAT_ERR_SHAPE, "too many codes");
  if (!codes || !scale || !out) return fail(CAT_ERR_INVALID_ARG, "NULL pointer");
  if (!aligned16(codes) || !aligned16(scale) || !aligned16(out)) return fail(CAT_ERR_ALIGNMENT, "pointers must be 16-byte aligned");
  if ((st = check_device()) != CAT_OK) return st;
  cudaError_t e = cat::launch_dequantize_sm4x8(codes, scale, rows, d, out, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "cat_dequantize_codes launch");
  return ok();
}

cat_status cat_gemm_f32(const float* A, const float* B, int64_t m, int64_t n, int64_t kdim, float* C,
                        cat_stream_t stream) {
  if (m < 0 || n < 0 || kdim < 1 || m > 0x7FFFFFFF || n > 0x7FFFFFFF || kdim > 0x7FFFFFFF)
    return fail(CAT_ERR_SHAPE, "m, n >= 0 and k >= 1, each below 2^31");
  if ((m + 127) / 128 > 65535) return fail(CAT_ERR_SHAPE, "m too large");
  if (m == 0 || n == 0) return ok();
  if (!A || !B || !C) return fail(CAT_ERR_INVALID_ARG, "NULL pointer");
  if (!aligned16(A) || !aligned16(B) || !aligned16(C)) return fail(CAT_ERR_ALIGNMENT, "pointers must be 16-byte aligned");
  cat_status st = check_device();
  if (st != CAT_OK) return st;
  cudaError_t e = cat::launch_gemm_f32_nt(A, B, C, m, n, kdim, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "cat_gemm_f32 launch");
  return ok();
}

// ---- the alignment ceiling and the full-size Hadamard (Sec. 4: Eq. 9; T = H_d M_hat_block)

cat_status cat_transform_quantize_act_hd(const void* x, cat_dtype dtype, int64_t n, int64_t d_in, int32_t k,
                                         const float* M_blocks, uint8_t* xq, float* x_scale, cat_stream_t stream) {
  if (dtype != CAT_F32 && dtype != CAT_BF16) return fail(CAT_ERR_INVALID_ARG, "unknown dtype");
  if (n < 0) return fail(CAT_ERR_SHAPE, "n must be >= 0");
  cat_status st = check_din(d_in);
  if (st != CAT_OK) return st;
  if ((d_in & (d_in - 1)) != 0 || d_in > 32768) return fail(CAT_ERR_SHAPE, "the full-size Hadamard needs d_in = 2^m <= 32768");
  if (!valid_k(k) || d_in % k != 0) return fail(CAT_ERR_SHAPE, "k must be one of 16..256 (power of two) and divide d_in");
  if (n == 0) return ok();
  if (n > 0x7FFFFFFF) return fail(CAT_ERR_SHAPE, "n too large");
  if (!x || !M_blocks || !xq || !x_scale) return fail(CAT_ERR_INVALID_ARG, "NULL pointer");
  if (!aligned16(x) || !aligned16(M_blocks) || !aligned16(xq) || !aligned16(x_scale))
    return fail(CAT_ERR_ALIGNMENT, "pointers must be 16-byte aligned");
  if ((st = check_device()) != CAT_OK) return st;
  cudaError_t e;
  uint32_t* status = status_word(&e);
  if (!status) return cuda_fail(e, "status word");
  e = transform_fwht_quantize(x, (int)dtype, n, d_in, k, M_blocks, 0, xq, x_scale, status, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "cat_transform_quantize_act_hd");
  return ok();
}

cat_status cat_fwht_rows(float* V, int64_t rows, int64_t d, cat_stream_t stream) {
  if (rows < 0 || rows > 0x7FFFFFFF) return fail(CAT_ERR_SHAPE, "rows must be in [0, 2^31)");
  if (d < 2 || (d & (d - 1)) != 0 || d > 32768) return fail(CAT_ERR_SHAPE, "d must be a power of two in 2..32768");
  if (rows == 0) return ok();
  if (!V) return fail(CAT_ERR_INVALID_ARG, "NULL pointer");
  if (!aligned16(V)) return fail(CAT_ERR_ALIGNMENT, "pointers must be 16-byte aligned");
  cat_status st = check_device();
  if (st != CAT_OK) return st;
  cudaError_t e = cat::launch_fwht_rows(V, rows, d, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "cat_fwht_rows launch");
  return ok();
}

cat_status cat_gram_f32(const void* X, cat_dtype dtype, int64_t n, int64_t d, float* C, cat_stream_t stream) {
  if (dtype != CAT_F32 && dtype != CAT_BF16) return fail(CAT_ERR_INVALID_ARG, "unknown dtype");
  if (n < 1 || n > 0x7FFFFFFF || d < 1 || d > 65536) return fail(CAT_ERR_SHAPE, "n in [1, 2^31), d in [1, 65536]");
  if (!X || !C) return fail(CAT_ERR_INVALID_ARG, "NULL pointer");
  if (!aligned16(X) || !aligned16(C)) return fail(CAT_ERR_ALIGNMENT, "pointers must be 16-byte aligned");
  cat_status st = check_device();
  if (st != CAT_OK) return st;
  cudaError_t e = cat::launch_gram_f32(X, (int)dtype, n, d, C, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "cat_gram_f32 launch");
  return ok();
}

cat_status cat_alignment_ceiling_host(const double* sigma_x, const double* sigma_w, int64_t d, double* out3) {
  if (d < 1 || d > 4096) return fail(CAT_ERR_SHAPE, "d must be in [1, 4096] (a host eigen-decomposition of d x d)");
  if (!sigma_x || !sigma_w || !out3) return fail(CAT_ERR_INVALID_ARG, "NULL pointer");
  for (int64_t i = 0; i < d * d; ++i)
    if (!std::isfinite(sigma_x[i]) || !std::isfinite(sigma_w[i])) return fail(CAT_ERR_NUMERIC, "non-finite statistics");
  if (!cat::alignment_ceiling_host(sigma_x, sigma_w, d, &out3[0], &out3[1], &out3[2]))
    return fail(CAT_ERR_NUMERIC, "Sigma_x is not positive definite");
  return ok();
}
