/*
 * cat_w4a4.h -- C ABI of the block Concentration-Alignment Transform (CAT) W4A4 linear layer
 * on NVIDIA GB300 (sm_103a).
 *
 * The layer follows "Dissecting Quantization Error: A Concentration-Alignment Perspective":
 *   y = W x = (W T^{-1}) (T x) ~ Q(W T^{-1}) Q(T x)                      (Sec. 3, Eq. 5)
 * with a block-diagonal transform T = H_k M_block (Sec. 4, Eq. 10), where every k x k block
 * M_b = (Sigma_w_b # Sigma_x_b^{-1})^{1/2} maximises alignment on its own sub-problem (Eq. 7),
 * Sigma_x = E[x x^T] over calibration tokens and Sigma_w = W^T W.  Activations are quantized
 * per token and weights per output channel with a symmetric uniform round-to-nearest INT4
 * quantizer (Lemma 2 range, Sec. 6 set-up); the layer's quality is its SQNR (Sec. 2, Eq. 1).
 *
 * Conventions shared by every call
 * --------------------------------
 *  - Matrices are row-major and dense.  A token is a row of x [n][d_in]; W is [d_out][d_in];
 *    y is [n][d_out] float32.  T acts on activations (x' = T x); T_blocks[b] is the k x k block
 *    acting on channels b*k .. b*k+k-1, stored row-major ([d_in/k][k][k] float32).
 *  - Unless a parameter says "host", pointers are device pointers owned by the caller; the
 *    library never frees them.  Device pointers must be 16-byte aligned.
 *  - Calls are asynchronous on `stream` (NULL = the legacy default stream) unless stated.
 *    Launch failures return CAT_ERR_CUDA.  Conditions detected on the device (a bounded wait
 *    that gave up, a non-finite input) are recorded in a device status word that
 *    cat_device_status() reads; kernels never trap.
 *  - Arguments are validated on the host before anything is launched; an invalid call returns
 *    an error code, launches nothing and touches no output.  cat_last_error() gives a message.
 *  - Shapes: d_in % 32 == 0 (a packed row is a whole number of 16-byte chunks); k is one of
 *    16, 32, 64, 128, 256 and divides d_in; n, d_out >= 1 (n == 0 is accepted and does nothing).
 *  - Thread safety: calls keep no host state between calls except the error message of the
 *    calling thread and, per device, the cached device addresses of the library's static device
 *    scratch (looked up once under a lock).  Exception: cat_quantize_weights_noalloc uses one
 *    shared device scratch area per device, so its calls must be serialized by the caller.
 *
 * INT4 code format ("SM4x8")
 * --------------------------
 *  Codes q are integers in [-7, 7] (the restricted symmetric INT4 grid: step s = max|v| / 7,
 *  round half to even, so the largest magnitude maps to +-7 and zero is exact).  Each code is a
 *  4-bit sign-magnitude value: sign s = (q < 0), magnitude m = |q| (3 bits).  A row of d_in codes
 *  occupies d_in/2 bytes; every 8 consecutive codes e0..e7 of a row (along d_in) form one
 *  little-endian 32-bit word w whose byte i (i = 0..3) holds
 *      bits 0-2: m(e_i)     bit 7: s(e_i)     bits 4-6: m(e_{4+i})     bit 3: s(e_{4+(i+3)%4}).
 *  With this layout  (w & 0x87878787)  and  (rotr32(w, 4) & 0x87878787)  are, byte for byte,
 *  the FP8 E4M3 encodings (s << 7 | m) of e0..e3 and e4..e7, i.e. the subnormal values
 *  (-1)^s * m * 2^-9.  The GEMM feeds these bytes to the FP8 tensor cores and rescales the
 *  exactly accumulated result by 2^18.
 */
#ifndef CAT_W4A4_H
#define CAT_W4A4_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t. */
typedef struct CUstream_st* cat_stream_t;

typedef enum {
  CAT_OK = 0,
  CAT_ERR_INVALID_ARG = 1,   /* NULL pointer, unknown enum value, negative size */
  CAT_ERR_SHAPE = 2,         /* sizes violate the shape rules above */
  CAT_ERR_ALIGNMENT = 3,     /* a device pointer is not 16-byte aligned */
  CAT_ERR_NUMERIC = 4,       /* non-finite input, or a calibration block that is not positive definite */
  CAT_ERR_UNSUPPORTED = 5,   /* valid request this build does not implement (e.g. no sm_103a device) */
  CAT_ERR_CUDA = 6,          /* a CUDA runtime call failed */
  CAT_ERR_TIMEOUT = 7        /* a bounded device-side wait gave up */
} cat_status;

typedef enum { CAT_F32 = 0, CAT_BF16 = 1 } cat_dtype;

typedef enum {
  CAT_T_IDENTITY = 0,        /* T = I: plain W4A4 RTN */
  CAT_T_RHT = 1,             /* T_b = H_k Diag(sigma_b): randomized Hadamard rotation, signs given by the caller */
  CAT_T_CAT = 2,             /* T_b = H_k M_b, M_b = (Sigma_w_b # Sigma_x_b^{-1})^{1/2} (Sec. 4, Eq. 7, Eq. 10) */
  CAT_T_DIAG = 3,            /* the k = 1 optimum (end of Sec. 4): T = Diag(m), m_i = (Sigma_w_ii / Sigma_x_ii)^{1/4},
                                stored as k x k diagonal blocks */
  CAT_T_CAT_HD = 4           /* T = H_d M_block (Sec. 4, "approximately optimal transform" with the full-size
                                Hadamard over all d_in = 2^m channels): T_blocks hold the M_b; the online path
                                is cat_transform_quantize_act_hd */
} cat_tkind;

/* Human-readable name of a status code (static string). */
const char* cat_status_string(cat_status status);

/* Message of the last error returned to the calling thread ("" if none). */
const char* cat_last_error(void);

/* Library version: major * 10000 + minor * 100 + patch. */
int cat_version(void);

/* Number of kernels the library has launched in this process so far (a host counter bumped at
 * every launch site, also during stream capture).  Diagnostic; no counterpart in the paper. */
unsigned long long cat_kernel_launches(void);

/*
 * cat_calib_cov -- calibration autocorrelation blocks (Sec. 4: Sigma_x = E[x x^T]; Eq. 10 uses its
 * k x k diagonal blocks).
 *   x            device [n][d] in `dtype` (calibration tokens, or weight rows for Sigma_w = W^T W).
 *   sigma_blocks device [d/k][k][k] float64: receives sum_t x_{t,b} x_{t,b}^T for every block b
 *                (a plain sum over tokens: divide by the token count for E[x x^T]).  With
 *                accumulate == 0 the buffer is overwritten, otherwise the sums are added to it, so
 *                calibration sets larger than one batch can be streamed through.
 * bf16 rows run on tensor cores: products are exact and tokens accumulate in fp32 (relative error
 * ~1e-7, which moves the block transform by ~1e-7).  fp32 rows accumulate products and their FMA
 * errors in compensated (double-float) fp32 arithmetic, matching float64 to ~1e-12.  Sums are
 * stored as float64.
 */
cat_status cat_calib_cov(const void* x, cat_dtype dtype, int64_t n, int64_t d, int32_t k,
                         double* sigma_blocks, int accumulate, cat_stream_t stream);

/*
 * cat_quantize_weights -- offline weight preparation (Sec. 3 Eq. 5: W' = W T^{-1}; Sec. 4 Eq. 7
 * and Eq. 10: the block transform; Sec. 6: per-output-channel symmetric RTN).
 *   W              device [d_out][d_in] in `dtype`.
 *   kind           transform family.  CAT_T_DIAG and CAT_T_CAT_HD need sigma_x_blocks as CAT does;
 *                  CAT_T_CAT_HD needs d_in = 2^m <= 32768, returns the M_b blocks in T_blocks and the
 *                  codes of W M^{-1} H_d (through a float32 scratch from the stream-ordered pool).
 *   sigma_x_blocks device [d_in/k][k][k] float64 sums from cat_calib_cov (CAT only; else may be NULL).
 *   n_calib        number of tokens behind sigma_x_blocks (CAT only, >= 1).
 *   rht_signs      HOST [d_in] float32, each +1 or -1 (RHT only; else may be NULL).
 *   T_blocks       out, device [d_in/k][k][k] float32: the online activation transform T.
 *   Wq             out, device [d_out][d_in/2] bytes: SM4x8 codes of W T^{-1}.
 *   w_scale        out, device [d_out] float32: per-output-channel step s_w = max_i |W'_{o,i}| / 7.
 * Synchronous: it reads the calibration sums back, builds T and T^{-1} in float64 on the host
 * (per block, in parallel over host threads), uploads them, and runs the weight kernels; it
 * returns after the outputs are written.  It allocates and frees its own temporaries.
 * Returns CAT_ERR_NUMERIC if a Sigma_x or Sigma_w block is not positive definite.
 */
cat_status cat_quantize_weights(const void* W, cat_dtype dtype, int64_t d_out, int64_t d_in, int32_t k,
                                cat_tkind kind, const double* sigma_x_blocks, int64_t n_calib,
                                const float* rht_signs, float* T_blocks, uint8_t* Wq, float* w_scale,
                                cat_stream_t stream);

/*
 * cat_quantize_weights_noalloc -- cat_quantize_weights without device allocation.  No counterpart
 * in the paper: it exists for callers that cannot take new device memory mid-run, e.g. a process
 * that has handed all free device memory to its own pool and re-quantizes a layer later (after
 * re-calibration), where a new allocation would fail or evict that pool.
 * Same arguments, steps and results as cat_quantize_weights.  Its two temporaries (the float64
 * Sigma_w blocks and the float32 blocks (T_b^{-1})^T, 12 bytes per element of d_in * k) live in a
 * fixed 12 MiB scratch area that the library reserves statically on every device it is loaded on.
 *   Limit: d_in * k <= CAT_PREP_NOALLOC_MAX_DK; a larger call returns CAT_ERR_SHAPE before any
 *   CUDA call and writes nothing.
 *   Setup: the first call on a device looks up the scratch address (cudaGetSymbolAddress) with
 *   that device current; make that first call before any stream capture.  Under CUDA's default
 *   lazy module loading (CUDA_MODULE_LOADING=LAZY) the 12 MiB array and the kernels this call
 *   launches are only loaded onto the device by that first call (or by the first use of another
 *   entry point in the same module), and loading them takes device memory.  A caller that will
 *   later hand all free device memory to its own pool must therefore make one call (any valid
 *   size) before reserving it; later calls then take no device memory at all.
 *   Concurrency: every call on a device shares the one scratch area, so calls that overlap in
 *   time (other host threads or streams) race; the caller must serialize them.  Each call
 *   synchronizes its stream before returning, so consecutive calls are safe.
 */
#define CAT_PREP_NOALLOC_MAX_DK 1048576
cat_status cat_quantize_weights_noalloc(const void* W, cat_dtype dtype, int64_t d_out, int64_t d_in, int32_t k,
                                        cat_tkind kind, const double* sigma_x_blocks, int64_t n_calib,
                                        const float* rht_signs, float* T_blocks, uint8_t* Wq, float* w_scale,
                                        cat_stream_t stream);

/*
 * cat_build_transform_host -- the host part of cat_quantize_weights, exposed for inspection: the
 * block transform T and its inverse in float64 (Sec. 4, Eq. 7 and Eq. 10).  All pointers are HOST.
 *   sigma_x_blocks [d_in/k][k][k] sums over n_calib tokens (CAT only); sigma_w_blocks [d_in/k][k][k]
 *   (= diagonal blocks of W^T W, CAT only); rht_signs [d_in] (RHT only).
 *   T_out, Tinv_out [d_in/k][k][k] float64.
 * Runs on the calling thread's host cores only; no CUDA call is made.
 */
cat_status cat_build_transform_host(cat_tkind kind, int64_t d_in, int32_t k, const double* sigma_x_blocks,
                                    int64_t n_calib, const double* sigma_w_blocks, const float* rht_signs,
                                    double* T_out, double* Tinv_out);

/*
 * cat_transform_quantize_act -- online activation path (Sec. 3 Eq. 5: x' = T x; Lemma 2 symmetric
 * range; Sec. 6: dynamic per-token quantization, round to nearest).
 *   x        device [n][d_in] in `dtype`.
 *   T_blocks device [d_in/k][k][k] float32 (from cat_quantize_weights).
 *   xq       out, device [n][d_in/2] bytes: SM4x8 codes of x' = T x.
 *   x_scale  out, device [n] float32: per-token step s_x = max_i |x'_i| / 7 (0 for an all-zero token).
 * Codes are q = clamp(round_half_even(7 x'_i / max|x'|), -7, 7), x' accumulated in float32; the
 * rounding decision is exact for the float32 x' (ties included), not a float32 approximation of it.
 */
cat_status cat_transform_quantize_act(const void* x, cat_dtype dtype, int64_t n, int64_t d_in, int32_t k,
                                      const float* T_blocks, uint8_t* xq, float* x_scale,
                                      cat_stream_t stream);

/*
 * cat_split_transform_bytes -- the size of cat_split_transform's planes for d_in channels and block
 * size k: 6 * d_in * K bytes, K the width of the tensor-core transform's channel groups (128 when
 * 128 divides d_in and k <= 128; 64 for k = 64 otherwise); 0 when no tensor-core transform applies
 * (k = 256, or a shape the arguments do not allow).  No device access.
 */
int64_t cat_split_transform_bytes(int64_t d_in, int32_t k);

/*
 * cat_split_transform -- T_blocks [d_in/k][k][k] float32 into the three bf16 planes of every K-wide
 * channel group (K as in cat_split_transform_bytes; a group holds K/k blocks of the block-diagonal T
 * on its diagonal and zeros elsewhere), T = H + M + L with H = bf16(T), M = bf16(T - H),
 * L = bf16(T - H - M) (24 significant bits: the tensor-core transform's fp32-accurate products),
 * laid out exactly as that kernel's shared-memory operand (K-major, 128-byte swizzle).
 *   planes: device, cat_split_transform_bytes(d_in, k) bytes.
 * CAT_ERR_UNSUPPORTED when that size is 0.  Run once per layer after weight preparation; no
 * counterpart in the paper (a layout of T).
 */
cat_status cat_split_transform(const float* T_blocks, int64_t d_in, int32_t k, uint8_t* planes, cat_stream_t stream);

/*
 * cat_transform_quantize_act_split -- cat_transform_quantize_act with T's pre-split planes
 * (cat_split_transform; may be NULL): on the tensor-core path (bf16 rows, cat_split_transform_bytes
 * nonzero) each CTA fetches its group's planes with three bulk copies instead of splitting them
 * itself.  Same results.
 */
cat_status cat_transform_quantize_act_split(const void* x, cat_dtype dtype, int64_t n, int64_t d_in, int32_t k,
                                            const float* T_blocks, const uint8_t* T_planes, uint8_t* xq, float* x_scale,
                                            cat_stream_t stream);

/*
 * cat_w4a4_linear -- integer GEMM and dequantization (Sec. 3 Eq. 5: y ~ Q(W T^{-1}) Q(T x)).
 *   xq [n][d_in/2], x_scale [n]; Wq [d_out][d_in/2], w_scale [d_out]  (SM4x8 codes and steps).
 *   y        out, device [n][d_out] float32: y[t][o] = acc[t][o] * x_scale[t] * w_scale[o], with
 *            acc[t][o] = sum_i q_x[t][i] q_w[o][i] computed exactly (FP8 tensor cores, fp32
 *            accumulators holding integers |acc| <= 49 * d_in < 2^24).
 *   acc_out  optional out (NULL to skip), device [n][d_out] int32: the integer accumulators.
 * Exactness needs 49 * d_in < 2^24, so d_in <= 262144 is required (CAT_ERR_SHAPE otherwise).
 */
cat_status cat_w4a4_linear(const uint8_t* xq, const float* x_scale, const uint8_t* Wq, const float* w_scale,
                           int64_t n, int64_t d_in, int64_t d_out, float* y, int32_t* acc_out,
                           cat_stream_t stream);

/*
 * cat_w4a4_linear_sqnr -- cat_w4a4_linear and cat_sqnr in one call (Sec. 3 Eq. 5; Sec. 2 Eq. 1).
 *   Same arguments as cat_w4a4_linear (without acc_out), plus
 *   y_ref  device [n][d_out] float32: the full-precision output y = W x;
 *   out3   out, device [3] float64: { sum y_ref^2, sum (y_ref - y)^2, 10 log10(ratio) dB }, as cat_sqnr.
 * y is written exactly as cat_w4a4_linear writes it.  The sums are formed in the GEMM's epilogue while
 * y is produced (y is not read back) -- for n > 32 when d_out % 4 == 0, for n <= 32 when the decoded
 * tokens fit in the weight-streaming kernel's shared memory; otherwise the GEMM is followed by the
 * cat_sqnr reduction.  Squares are summed in fp32 over runs of at most 32 outputs, the runs as float pairs
 * (hi + lo, ~48 significant bits); the result does not depend on CTA timing.
 */
cat_status cat_w4a4_linear_sqnr(const uint8_t* xq, const float* x_scale, const uint8_t* Wq, const float* w_scale,
                                int64_t n, int64_t d_in, int64_t d_out, float* y, const float* y_ref, double* out3,
                                cat_stream_t stream);

/*
 * Byte codes ("E8")
 * -----------------
 *  The same codes q in [-7, 7], one per byte: byte = (q < 0) << 7 | |q|, the FP8 E4M3 encoding of
 *  the subnormal q * 2^-9 (the bytes the SM4x8 masks produce).  A row of d codes occupies d bytes,
 *  twice the SM4x8 size.  The byte-code GEMM loads them into shared memory as they are and runs the
 *  FP8 tensor cores on them directly, with no decode step; the weights are converted once per layer
 *  (cat_codes_to_e4m3), the activations are written in this form by cat_transform_quantize_act_e8.
 *  Its results are identical to the SM4x8 GEMM's (same exact integer accumulators, same scaling).
 */

/*
 * cat_codes_to_e4m3 -- SM4x8 codes to byte codes (a layout change; no arithmetic).
 *   codes  device [rows][d/2] bytes, SM4x8;   out  out, device [rows][d] bytes, byte codes.
 *   d must be a positive multiple of 32 (CAT_ERR_SHAPE).  rows == 0 is a no-op.  Asynchronous on stream.
 */
cat_status cat_codes_to_e4m3(const uint8_t* codes, int64_t rows, int64_t d, uint8_t* out, cat_stream_t stream);

/*
 * cat_transform_quantize_act_e8 -- cat_transform_quantize_act_split with byte codes out (Sec. 3 Eq. 5:
 * x' = T x; Sec. 2 Lemma 2 range, Sec. 6 round to nearest).
 *   Arguments as cat_transform_quantize_act_split, except
 *   xq8  out, device [n][d_in] bytes: the codes of x' as byte codes.
 *   x_scale and the codes are those cat_transform_quantize_act_split writes (the same code decisions).
 *   bf16 rows on the fused tensor-core kernel write the bytes directly; elsewhere the SM4x8 codes go
 *   to stream-ordered scratch (n * d_in / 2 bytes, cudaMallocAsync) and are converted.
 */
cat_status cat_transform_quantize_act_e8(const void* x, cat_dtype dtype, int64_t n, int64_t d_in, int32_t k,
                                         const float* T_blocks, const uint8_t* T_planes, uint8_t* xq8, float* x_scale,
                                         cat_stream_t stream);

/*
 * cat_w4a4_linear_e8 -- cat_w4a4_linear on byte codes (Sec. 3 Eq. 5).
 *   xq8 [n][d_in], Wq8 [d_out][d_in] byte codes; x_scale, w_scale, y, acc_out as cat_w4a4_linear.
 *   Same results as cat_w4a4_linear on the SM4x8 form of the same codes, for every n >= 1 (it
 *   always runs the 256 x 128 tile kernel: for n <= 32 the SM4x8 weight-streaming kernel reads half
 *   the bytes).  Asynchronous on stream; errors as cat_w4a4_linear.
 */
cat_status cat_w4a4_linear_e8(const uint8_t* xq8, const float* x_scale, const uint8_t* Wq8, const float* w_scale,
                              int64_t n, int64_t d_in, int64_t d_out, float* y, int32_t* acc_out, cat_stream_t stream);

/*
 * cat_w4a4_linear_sqnr_e8 -- cat_w4a4_linear_sqnr on byte codes (Sec. 3 Eq. 5; Sec. 2 Eq. 1).
 *   Arguments as cat_w4a4_linear_e8 (without acc_out) plus y_ref and out3 as cat_w4a4_linear_sqnr.
 *   The sums are formed in the GEMM's epilogue when d_out % 4 == 0, else by the cat_sqnr reduction;
 *   the same sums as cat_w4a4_linear_sqnr for n > 32.
 */
cat_status cat_w4a4_linear_sqnr_e8(const uint8_t* xq8, const float* x_scale, const uint8_t* Wq8, const float* w_scale,
                                   int64_t n, int64_t d_in, int64_t d_out, float* y, const float* y_ref, double* out3,
                                   cat_stream_t stream);

/*
 * cat_sqnr -- signal-to-quantization-noise ratio of the layer output (Sec. 2, Eq. 1).
 *   y_ref, y_hat device [numel] float32 (full-precision and quantized outputs).
 *   out3         out, device [3] float64: { sum y_ref^2, sum (y_ref - y_hat)^2, 10 log10(ratio) dB }.
 * Squares are summed in fp32 over short runs and the run sums as float pairs (hi + lo, ~48 significant
 * bits); the dB value is formed in fp32 from the high parts (|error| ~1e-5 dB).  The per-CTA partial sums
 * are added in a fixed order, so the three values are the same on every run of the same inputs.
 * out3 is written, never read: it needs no zeroing.  The cross-CTA reduction uses one of eight
 * slots of device scratch per kernel, handed out round robin, so at most eight SQNR-forming
 * launches of one kernel may run concurrently.
 */
cat_status cat_sqnr(const float* y_ref, const float* y_hat, int64_t numel, double* out3, cat_stream_t stream);

/*
 * cat_block_row_stats -- per-layer diagnostics (Sec. 2, Lemmas 2 and 3): the row statistics of a
 * block-transformed matrix that the concentration C(v) = E||v||^2 / E r(v)^2 (symmetric range
 * r(v) = 2 max_i |v_i|) and the alignment A(x, W) = E||W x||^2 / (||W||_F^2 E||x||^2) are made of.
 *   V          device [rows][d] in `dtype`: activations x (one token per row) or weights W (one
 *              output channel per row).
 *   M_blocks   device [d/k][k][k] float32.  transpose = 0: v'_b = M_b v_b (activations with
 *              M = T, x' = T x); transpose = 1: v'_b = M_b^T v_b (weight rows with M = T^{-1},
 *              w' = w T^{-1}).
 *   row_sumsq  out, device [rows] float32: ||v'_r||^2 (fp32 sums).
 *   row_amax   out, device [rows] float32: max_i |v'_ri|.
 *   out3       out, device [3] float64: { sum_r ||v'_r||^2, sum_r (2 max_i |v'_ri|)^2,
 *              10 log10 of their ratio, i.e. C(v') in dB }.
 * Then C(x') = out3x[0] / out3x[1], C(W') = out3w[0] / out3w[1], and with sum y^2 over the layer's
 * outputs (cat_sqnr's first word) A = sum y^2 / (out3w[0] * out3x[0]) (the 1/n of both expectations
 * cancels).  Diagnostics, off the layer's hot path: a SIMT kernel plus a reduction; the row
 * outputs are zeroed with two memsets.  Requires rows in [1, 2^31), k in 16..256 (power of two)
 * dividing d, and 16-byte aligned pointers.
 */
cat_status cat_block_row_stats(const void* V, cat_dtype dtype, int64_t rows, int64_t d, int32_t k,
                               const float* M_blocks, int transpose, float* row_sumsq, float* row_amax, double* out3,
                               cat_stream_t stream);

/*
 * ---------------------------------------------------------------------------------------------
 * b-bit codes as E4M3 digit planes: the bit widths of Sec. 2 ("Bit width": each bit ~6 dB; Fig. 1
 * and Fig. 6 compare W4A4 with W6A6) and the experimental set-up of Sec. 6 (activations per token,
 * asymmetric; weights per output channel, symmetric, range by the L_2.4 error following GPTQ).
 *
 * Code grids (b in 2..8):
 *   symmetric  q = clamp(round(qmax v / a), -qmax, qmax), qmax = 2^(b-1) - 1, a = max|v| of the row
 *              (or the L_2.4 range for weights); step s = a / qmax.
 *   asymmetric lo = min(min v, 0), hi = max(max v, 0), N = 2^b - 1, s = (hi - lo) / N,
 *              zero point z = round(-lo / s), q = clamp(round(v / s) + z, 0, N); Q(v) = s (q - z).
 *   Rounding is half to even; every decision is exact for the float32 transformed value.
 * Digit-plane format: D = cat_dp_planes(b) planes (1 for b <= 4, else 2); a code is q = d0 + 16 d1 with
 *   symmetric d0 = ((q + 8) mod 16) - 8, d1 = (q - d0) / 16 (|d| <= 8), asymmetric d0 = q mod 16,
 *   d1 = q div 16 (one plane: d0 = q).  Each digit is one byte, the FP8 E4M3 encoding
 *   (d < 0) << 7 | |d|, which is exactly d * 2^-9 for |d| <= 16.  Plane p of an [R][d_in] code
 *   matrix is the [R][d_in] byte matrix at planes + p * R * d_in.
 * The GEMM accumulates every digit product on the FP8 tensor cores exactly; these calls need
 * d_in <= 65536 (CAT_ERR_SHAPE otherwise) on top of the shape rules above.
 * ---------------------------------------------------------------------------------------------
 */

/* Number of digit planes of b-bit codes (1 or 2); 0 if b is outside 2..8. */
int32_t cat_dp_planes(int32_t bits);

/*
 * cat_transform_quantize_act_dp -- online activation path at b bits (Sec. 3 Eq. 5: x' = T x; Sec. 6:
 * dynamic per-token quantization, symmetric or asymmetric).
 *   x, T_blocks  as cat_transform_quantize_act.
 *   planes       out, device [D][n][d_in] bytes (digit planes of the codes of x').
 *   x_scale      out, device [n] float32 steps (0 for an all-zero or non-finite token).
 *   x_zero       out, device [n] int32 zero points (asymmetric only; may be NULL when symmetric).
 * x_scale and x_zero also serve as the row statistics' scratch while the call runs.  Runs on SIMT
 * cores (transform, row statistics, codes: four launches).
 */
cat_status cat_transform_quantize_act_dp(const void* x, cat_dtype dtype, int64_t n, int64_t d_in, int32_t k,
                                         const float* T_blocks, int32_t bits, int32_t asymmetric, uint8_t* planes,
                                         float* x_scale, int32_t* x_zero, cat_stream_t stream);

/*
 * cat_quantize_weights_dp -- cat_quantize_weights at b bits with digit-plane output (Sec. 4 Eq. 7 and
 * Eq. 10: the transform; Sec. 6: per-output-channel symmetric codes).
 *   l24_range  0: a = max|w'| per row; 1: the L_2.4 range search (Sec. 6): candidates
 *              a_i = max|w'| (100 - i) / 100, i = 0..79, scored by sum |w' - s_i q_i|^2.4 (float32 terms
 *              summed in float64), the first smallest score wins.
 *   planes     out, device [D][d_out][d_in] bytes; w_scale out, device [d_out] float32.
 *   w_rowsum   optional out (NULL to skip), device [d_out] int32: sum_i q_w[o][i], the zero-point
 *              correction that cat_linear_dp needs for asymmetric activations.
 * Other arguments, synchronization, allocation and errors as cat_quantize_weights.
 */
cat_status cat_quantize_weights_dp(const void* W, cat_dtype dtype, int64_t d_out, int64_t d_in, int32_t k,
                                   cat_tkind kind, const double* sigma_x_blocks, int64_t n_calib,
                                   const float* rht_signs, int32_t bits, int32_t l24_range, float* T_blocks,
                                   uint8_t* planes, float* w_scale, int32_t* w_rowsum, cat_stream_t stream);

/*
 * cat_linear_dp -- integer GEMM of digit-plane codes and dequantization (Sec. 3 Eq. 5).
 *   acc[t][o] = sum_i (q_x[t][i] - z[t]) q_w[o][i]  (z = 0 unless asym_x), exactly;
 *   y[t][o]   = acc * x_scale[t] * w_scale[o] (float32, device [n][d_out]);
 *   acc_out   optional int32 [n][d_out] (NULL to skip).
 * asym_x = 1 needs x_zero [n] and w_rowsum [d_out] (from cat_quantize_weights_dp).  tcgen05 FP8 MMAs
 * (kind::f8f6f4) on TMA-loaded digit planes, one fp32 tensor-memory accumulator per digit weight 16^g.
 */
cat_status cat_linear_dp(const uint8_t* x_planes, int32_t bits_x, int32_t asym_x, const float* x_scale,
                         const int32_t* x_zero, const uint8_t* w_planes, int32_t bits_w, const float* w_scale,
                         const int32_t* w_rowsum, int64_t n, int64_t d_in, int64_t d_out, float* y, int32_t* acc_out,
                         cat_stream_t stream);

/*
 * cat_set_wait_limit_ns -- testing aid, no counterpart in the paper.  Sets, on the current device, the
 * bound of the pipeline waits of the weight-streaming W4A4 GEMM (cat_w4a4_linear, n <= 32) and of the
 * digit-plane GEMM (cat_linear_dp); 0 restores the default of 1 s (1e9 ns, also the largest value
 * accepted).  A wait that exceeds its bound gives up: the kernel drains its copies and MMAs in flight
 * (those waits keep the 1 s bound), frees its tensor memory, returns, and raises CAT_ERR_TIMEOUT in the
 * device status word with the kernel's bit (1 << 11 weight-streaming GEMM, 1 << 13 digit-plane GEMM)
 * and the source line of the first wait that gave up in bits 16..31.  Its outputs are then undefined.
 * Synchronous (a blocking copy to the device); not for use while those kernels run.
 */
cat_status cat_set_wait_limit_ns(uint64_t ns);

/*
 * One-sided SQNRs (Sec. 2: Lemma 2, SQNR(W x~), only activations quantized; Lemma 3, SQNR(W~ x), only
 * weights quantized; Lemma 1 combines the two into Theorem 1).  Off the hot path, three building
 * blocks on SIMT cores; with x' = T x and W' = W T^{-1} (so W' x' = W x):
 *   activation side: y_x = Q(x') W'^T  = cat_gemm_f32(cat_dequantize_codes(xq, x_scale), W')
 *   weight side:     y_w = x' Q(W')^T  = cat_gemm_f32(x', cat_dequantize_codes(Wq, w_scale))
 *   x' and W' from cat_block_transform; each SQNR then from cat_sqnr against y = W x.
 */

/*
 * cat_block_transform -- v'_b = M_b v_b (transpose = 0; activations with M = T) or M_b^T v_b
 * (transpose = 1; weight rows with M = T^{-1}, w' = w T^{-1}) for every row (Sec. 3, Eq. 5).
 *   V device [rows][d] in `dtype`; M_blocks device [d/k][k][k] float32; out device [rows][d] float32.
 * fp32 products and sums.
 */
cat_status cat_block_transform(const void* V, cat_dtype dtype, int64_t rows, int64_t d, int32_t k,
                               const float* M_blocks, int transpose, float* out, cat_stream_t stream);

/*
 * cat_dequantize_codes -- Q(v) = s_r q (Sec. 2): SM4x8 codes [rows][d/2] and steps [rows] float32 to
 * out [rows][d] float32.  All device pointers.
 */
cat_status cat_dequantize_codes(const uint8_t* codes, const float* scale, int64_t rows, int64_t d, float* out,
                                cat_stream_t stream);

/*
 * cat_gemm_f32 -- C[i][j] = sum_l A[i][l] B[j][l] in float32 (A [m][kdim], B [n][kdim], C [m][n], row-major
 * device arrays): the float GEMMs of the one-sided SQNRs.  A tiled SIMT kernel.
 */
cat_status cat_gemm_f32(const float* A, const float* B, int64_t m, int64_t n, int64_t kdim, float* C,
                        cat_stream_t stream);

/*
 * The alignment ceiling and the full-size Hadamard (Sec. 4: "Optimizing alignment", Eq. 9; the
 * approximately optimal transform T = H M with H over all channels).
 */

/*
 * cat_transform_quantize_act_hd -- online activations under CAT_T_CAT_HD: x' = H_d (M_block x) with the
 * orthonormal Sylvester H_d over all d_in = 2^m <= 32768 channels, then per-token symmetric INT4 codes
 * (as cat_transform_quantize_act).  M_blocks: the T_blocks of cat_quantize_weights(kind = CAT_T_CAT_HD).
 * Takes float32 scratch from the stream-ordered pool; synchronizes the stream before returning.
 */
cat_status cat_transform_quantize_act_hd(const void* x, cat_dtype dtype, int64_t n, int64_t d_in, int32_t k,
                                         const float* M_blocks, uint8_t* xq, float* x_scale, cat_stream_t stream);

/* cat_fwht_rows -- in place, V[r] <- H_d V[r] / sqrt(d) for every row (Sylvester order), V device [rows][d]
 * float32, d = 2^m in 2..32768.  One shared-memory row per CTA, log2(d) butterfly stages. */
cat_status cat_fwht_rows(float* V, int64_t rows, int64_t d, cat_stream_t stream);

/* cat_gram_f32 -- C = X^T X (C[i][j] = sum_t X[t][i] X[t][j]) in float32, X device [n][d] in `dtype`,
 * C device [d][d]: the full Sigma_x (over n) and Sigma_w that the ceiling needs. */
cat_status cat_gram_f32(const void* X, cat_dtype dtype, int64_t n, int64_t d, float* C, cat_stream_t stream);

/*
 * cat_alignment_ceiling_host -- the largest alignment any invertible transform reaches (Eq. 9):
 *   A_max = sum_i mu_i / (sum_i sqrt(mu_i))^2,  mu = eigenvalues of Sigma_x^{1/2} Sigma_w Sigma_x^{1/2}
 *   (equivalently of W Sigma_x W^T).  All pointers HOST: Sigma_x, Sigma_w [d][d] float64 (Sigma_x
 *   positive definite), out3 = { A_max, sum mu, sum sqrt(mu) }.  d <= 4096 (a Jacobi eigen-decomposition
 *   on the calling thread).  CAT_ERR_NUMERIC if Sigma_x is not positive definite.
 */
cat_status cat_alignment_ceiling_host(const double* sigma_x, const double* sigma_w, int64_t d, double* out3);

/*
 * cat_device_status -- synchronizes `stream`, then reads and clears the device status word.
 * Returns CAT_OK, CAT_ERR_TIMEOUT (a bounded wait in a kernel gave up and the kernel returned
 * early; its outputs are undefined) or CAT_ERR_NUMERIC (a kernel met a non-finite value; the
 * affected codes are 0).  `detail` (HOST, may be NULL) receives the raw status word.
 */
cat_status cat_device_status(cat_stream_t stream, uint32_t* detail);

#ifdef __cplusplus
}
#endif

#endif /* CAT_W4A4_H */
