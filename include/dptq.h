/*
 * dptq.h -- C ABI of the GB300 (sm_103a) quantized linear layer of DynamicPTQ
 * (arxiv 2606.12487): online block-Hadamard rotation of fp16 activations, symmetric
 * per-token 4/8-bit activation quantization chosen by a per-layer mask, and a GEMM of
 * packed int4 per-channel weights against the integer codes with exact 32-bit
 * integer accumulation and a per-token x per-channel scale epilogue to fp16.
 *
 * Paper passages the operations follow:
 *   Section 2, "Low-Bit Quantization of LLMs": Y = X W^T; Q_b(x) = s * round(x / s)
 *       (Eq. 2); quantization error x - Q_b(x) (Eq. 3).
 *   Section 2, "Rotation-based Activation Transformation": quantize X R with
 *       R^T R = I (Eq. 4); fold R into the weight offline, X W^T = (XR)(WR)^T (Eq. 5).
 *   Section 4.2, "Implementation and Quantization Details": weights per-channel
 *       symmetric (RTN), activations per-token symmetric, 4 bits by default.
 *   Section 3.3, Algorithm 1 steps 1-2: weights 4-bit; activations 8-bit on the
 *       sensitive layers of the mask, 4-bit elsewhere.
 *
 * Numerics (readings where the paper is silent):
 *   R = blockdiag(H_B, ..., H_B, H_r) / sqrt(block) along K, H the Sylvester
 *   Hadamard matrix in natural order, B = had_block a power of two, r = K mod B.
 *   A tail r that is not a power of two takes H_r = H_p (x) H_(2^k) with r = p 2^k
 *   and H_p the Paley type-I matrix of order p (p - 1 prime, p = 3 mod 4; the
 *   smallest such p, so that 2^k is largest), H_p = I + S, S[0][j>0] = 1, S[i>0][0] = -1,
 *   S[i][j] = chi(j - i) for i, j >= 1 with chi the quadratic character mod p - 1
 *   (Paley's first construction); the tail is scaled by 1/sqrt(r).  Scales s = max|row| / (2^(b-1) - 1) in fp32 (IEEE
 *   division); codes round half to even, clamped to [-2^(b-1), 2^(b-1) - 1];
 *   an all-zero row has s = 0 and all codes 0.  Output
 *   out[m][n] = fp16_rne( fp32( fp32(acc[m][n]) * s_a[m] ) * s_w[n] ).
 *
 * Conventions for every call:
 *   - Pointers passed to the online calls are DEVICE pointers owned by the caller;
 *     the library never frees them.  fp16 buffers are raw IEEE binary16 (uint16_t).
 *     Activation and output matrices are row-major and dense; x and codes rows must
 *     start 16-byte aligned (true for dense rows when K % 32 == 0 and the base
 *     pointer is 16-byte aligned).
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *     Online calls are asynchronous and stream-ordered; they do not synchronize the
 *     host.  Calls that share one handle, or the library scratch of one device,
 *     must not run concurrently on different streams.
 *   - Shape rules: 1 <= K <= 49152, K % 32 == 0, N % 16 == 0, had_block a power of
 *     two <= 4096, K splits into blocks of had_block plus a tail r that is a power of
 *     two or p 2^k with a Paley order p <= 256 (r = 2816 = 44 x 64 at K = 11008 and
 *     had_block 4096; r = 96 = 12 x 8, but not r = 736 = 23 x 32), bits in {4, 8}.
 *     Layers with a non-power-of-two tail run dptq_qlinear as two launches
 *     (rotate-quantize, then GEMM); dptq_qlinear_static rejects them.  Violations return
 *     DPTQ_ERR_INVALID_ARG (bits, null pointers, negative sizes) or
 *     DPTQ_ERR_UNSUPPORTED (shape).  M == 0 is a no-op.
 *   - No exception crosses this boundary.  CUDA errors map to DPTQ_ERR_CUDA (failed
 *     device allocations to DPTQ_ERR_OOM); the message of the last failure on the calling
 *     thread is dptq_last_error_message().  For tests of the out-of-memory path, the
 *     environment variable DPTQ_FAULT_ALLOC=n makes the n-th device allocation the
 *     library attempts in the process fail as out of memory (no cudaMalloc is made).
 *   - Device-side waits are bounded: a pipeline wait that exceeds about one second
 *     makes the kernel record an error word and return; dptq_last_device_error()
 *     reports it as DPTQ_ERR_TIMEOUT.
 */
#ifndef DPTQ_H_
#define DPTQ_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  DPTQ_OK = 0,
  DPTQ_ERR_INVALID_ARG = 1,
  DPTQ_ERR_UNSUPPORTED = 2,
  DPTQ_ERR_CUDA = 3,
  DPTQ_ERR_OOM = 4,
  DPTQ_ERR_TIMEOUT = 5
} dptq_status;

/* Opaque handle of one quantized linear layer.  It owns the packed weights, the
 * per-channel scales and the shape; it is created by dptq_pack_weights and released
 * by dptq_destroy. */
typedef struct dptq_linear* dptq_handle;

/* Offline weight packing (Section 2 Eq. 5; Section 4.2 RTN per-channel symmetric).
 * W_fp16: [N][K] row-major binary16 weights, on the device if w_on_device != 0,
 *   else in host memory.  Read only; not retained.
 * Computes W' = W R, s_w[n] = max_k |W'[n][k]| / 7, q = clamp(rint(W'/s_w), -8, 7)
 * on the GPU and keeps q (4 bits per weight, in a tiled device layout) and s_w in
 * device memory owned by the handle.  Synchronous (returns after packing).
 * Errors: INVALID_ARG for null pointers or sizes <= 0, UNSUPPORTED for shapes, OOM
 * when device memory runs out, CUDA for other CUDA failures. */
dptq_status dptq_pack_weights(const void* W_fp16, int N, int K, int had_block, int w_on_device,
                              dptq_handle* out);

/* Randomized Hadamard variant (QuaRot's rotation, named in Section 1 and Section 4.2):
 * R' = D R with D = diag(signs), signs_host[k] in {+1, -1} for k < K (host memory, read
 * only, copied into the handle).  D is orthogonal, so R'^T R' = I (Eq. 4) and folding
 * R' into W keeps X W^T (Eq. 5).  Packs W' = W R' like dptq_pack_weights; every
 * qlinear call on the returned handle then rotates x by the same R'.  INVALID_ARG if a
 * sign is neither +1 nor -1. */
dptq_status dptq_pack_weights_rh(const void* W_fp16, int N, int K, int had_block, const int8_t* signs_host,
                                 int w_on_device, dptq_handle* out);

/* Online rotation + quantization of activations (Section 2 Eq. 4 then Eq. 2).
 * x_fp16: device [M][K] binary16.  bits: 4 or 8 (the mask entry of the layer).
 * codes (device, written): bits == 4: uint8 [M][K/2], byte j of a row holds code 2j in
 *   bits 0-3 and code 2j+1 in bits 4-7, each 4-bit two's complement;
 *   bits == 8: int8 [M][K].
 * scales (device, written): float [M], s_a per token.
 * One fused kernel: 128-bit loads, Walsh-Hadamard butterflies on exact 64-bit fixed
 * point, one correctly rounded conversion to fp32, row absmax, rounding, packing. */
dptq_status dptq_rotate_quant_act(const void* x_fp16, int M, int K, int had_block, int bits,
                                  void* codes, float* scales, void* stream);

/* Test hook: the rotated activations y = x R as fp32 [M][K] (device), the value the
 * quantizer of dptq_rotate_quant_act sees. */
dptq_status dptq_rotate_act(const void* x_fp16, int M, int K, int had_block, float* y_f32,
                            void* stream);

/* dptq_rotate_quant_act and dptq_rotate_act with the randomized Hadamard R' = D R:
 * signs_dev is a DEVICE array of K int8 values, 16-byte aligned (a value below zero
 * means -1, any other +1), or NULL for the plain block Hadamard.  INVALID_ARG if
 * signs_dev is not 16-byte aligned. */
dptq_status dptq_rotate_quant_act_rh(const void* x_fp16, int M, int K, int had_block, int bits,
                                     const int8_t* signs_dev, void* codes, float* scales, void* stream);
dptq_status dptq_rotate_act_rh(const void* x_fp16, int M, int K, int had_block, const int8_t* signs_dev,
                               float* y_f32, void* stream);

/* KV-cache quantization (Section 4.2: 4-bit KV cache, quantized in groups of 128
 * values).  kv_fp16: device [rows][cols] binary16 (16-byte aligned).  Each row is
 * cut into groups of `group` consecutive columns, each quantized on its own,
 * symmetrically (the paper does not say symmetric or asymmetric): s = max|x| / 7 in
 * fp32 (IEEE division), c = clamp(round-half-even(x / s), -8, 7) (never -8), an
 * all-zero group has s = 0 and codes 0.
 * codes (device, written): uint8 [rows][cols/2] in the A4 format of
 * dptq_rotate_quant_act (low nibble = even column); scales (device, written): float
 * [rows][cols / group].  group: a multiple of 128 up to 1024 that divides cols (the
 * paper's 128).  Asynchronous.  INVALID_ARG for null pointers, negative sizes or a
 * misaligned kv_fp16; UNSUPPORTED for other group sizes.  rows == 0 is a no-op. */
dptq_status dptq_kv4_quantize(const void* kv_fp16, int rows, int cols, int group, void* codes, float* scales,
                              void* stream);

/* Sensitive-layer policy: the statistics of Section 3.1 and the set of Section 3.3
 * (Eq. 20), giving the activation bits of Algorithm 1 step 2.  For layer l with
 * residual state x_t (entering the layer) and update dx_t of token t:
 *   Jump Ratio        JR_l  = mean_t ||dx_t|| / (||x_t|| + eps)                 (Eqs. 8-9)
 *   historical SNR    SNR_l = mean_t 10 log10(||x_t||^2 / (||xhat_t - x_t||^2 + eps)),
 *                     xhat_t = Q_b(x_t + dx_t) - dx_t, Q_b the per-token symmetric
 *                     quantizer at `bits` on the fp32 sum x_t + dx_t     (Eqs. 10-11)
 *   bits_out[l] = 8 if JR_l > tau_jr and SNR_l < tau_snr, else 4.          (Eq. 20)
 * x, dx: device fp32 [L][T][d], 16-byte aligned, d % 4 == 0; jr, snr: device double
 * [L] (written); bits_out: device uint8 [L] (written).  bits in {4, 8}; eps >= 0 (the
 * paper's epsilon; its value is not given).  Norms and errors are evaluated in fp32 per
 * element and summed per token (in fp32 for d <= 4096: sums of non-negative terms, a
 * relative error below 2^-19) and the per-layer means accumulate in fp64: JR within
 * 1e-5 relative and SNR within 1e-3 dB of the exact statistics.  Asynchronous.  INVALID_ARG for bad sizes, bits, eps, null or misaligned pointers.  The
 * first call on a device allocates the library's small per-device scratch (its error
 * word), which is refused (UNSUPPORTED) during stream capture: call dptq_reserve first.
 * A bounded in-kernel wait that gave up leaves jr/snr unspecified and is reported by
 * dptq_last_device_error (TIMEOUT). */
dptq_status dptq_sensitivity_policy(const float* x, const float* dx, int L, int T, int d, int bits, double eps,
                                    double tau_jr, double tau_snr, double* jr, double* snr, uint8_t* bits_out,
                                    void* stream);

/* The quantized linear layer: out = fp16( Q(x R) (W R)^T scaled ), i.e. rotate and
 * quantize x with `bits` (4 or 8, the layer's mask entry), multiply by the packed
 * int4 weights of `h` with exact int32 accumulation, apply s_a[m] * s_w[n].
 * x_fp16: device [M][K]; out_fp16: device [M][N] (written; any alignment, a 16-byte
 * aligned pointer is written 8 bytes at a time).  Asynchronous.
 * Uses the library's per-device scratch (grown on demand; call dptq_reserve before
 * capturing into a CUDA graph so that no allocation happens during capture).  Growth
 * never frees memory: a call that needs more scratch than the device holds allocates new,
 * at least twice larger buffers and keeps the superseded ones allocated until the process
 * exits, so work enqueued earlier and graphs captured earlier (which keep the old
 * addresses) stay valid.
 * For token tiles of up to 64 rows (M <= 64), K <= 16384 and a power-of-two tail block,
 * rotation, quantization and GEMM run as ONE kernel launch: each token row is split over
 * two or four CTAs of the GEMM grid, each rotating and quantizing its own share of the
 * row, and the row maxima are exchanged between them (the environment variable
 * DPTQ_FUSED=0 selects the two-launch sequence of dptq_qlinear_quantize +
 * dptq_qlinear_gemm); both give the same bits. */
dptq_status dptq_qlinear(dptq_handle h, const void* x_fp16, int M, int bits, void* out_fp16,
                         void* stream);

/* The two halves of dptq_qlinear, for callers that feed one quantized activation
 * matrix to several layers with the same K and had_block (for example q, k and v):
 * dptq_qlinear_quantize rotates and quantizes x into the device's scratch (the same
 * kernel as dptq_rotate_quant_act, writing the GEMM's operand layout), and
 * dptq_qlinear_gemm multiplies those codes by the weights of `h`.  The codes stay in
 * the scratch until the next quantize call on the device; a gemm call must use the
 * M and bits of the preceding quantize call and a handle with its K and had_block. */
dptq_status dptq_qlinear_quantize(dptq_handle h, const void* x_fp16, int M, int bits, void* stream);
dptq_status dptq_qlinear_gemm(dptq_handle h, int M, int bits, void* out_fp16, void* stream);

/* dptq_qlinear for callers that cannot allocate device memory when they call it:
 * runtimes whose own memory pool owns all device memory, or hosts that forbid
 * cudaMalloc once they are serving.  The paper has no counterpart: this is a property
 * of the library, not of the method.
 * Same arguments and results as dptq_qlinear, but its scratch lives in one fixed
 * device array of about 5 MiB inside the library, which every GPU that loads the
 * library holds until the process exits.  The call never runs cudaMalloc, cudaFree or
 * an allocating library routine.
 * Limits: M <= 32 tokens, K <= 16384 and a power-of-two tail block (K mod had_block);
 * other shapes return DPTQ_ERR_UNSUPPORTED.
 * The first call on a device looks the array up (cudaGetSymbolAddress) and zeroes it,
 * synchronously; make that first call before any stream capture.  That first call is
 * also when the CUDA driver brings the array's device memory in (modules load lazily),
 * so make it, or a warm-up call, before the caller's own pool takes the device memory.
 * All calls share the array: calls whose kernels overlap on the GPU (for example on
 * two streams without ordering between them) race and corrupt each other's results.
 * A bounded-wait timeout inside this call is recorded in the array's own error word;
 * dptq_last_device_error reports it (TIMEOUT) and clears the array's error word, split-tile
 * sums and counters, without allocating. */
dptq_status dptq_qlinear_static(dptq_handle h, const void* x_fp16, int M, int bits, void* out_fp16,
                                void* stream);

/* GEMM + epilogue on caller-provided codes (the format dptq_rotate_quant_act writes)
 * and per-token scales.  acc_i32: optional device int32 [M][N] that receives the
 * exact integer accumulators (test hook); NULL to skip. */
dptq_status dptq_qgemm_codes(dptq_handle h, const void* codes, const float* scales, int M, int bits,
                             void* out_fp16, int32_t* acc_i32, void* stream);

/* Pre-size the per-device scratch for calls with up to max_M tokens and up to max_K
 * inputs / max_N outputs, so that later calls allocate nothing.  Synchronous. */
dptq_status dptq_reserve(int max_M, int max_K, int max_N);

/* The GEMM launch plan the library would use for M tokens, N outputs, K inputs at
 * `bits` activation bits on a GPU with num_sms SMs (host only: no GPU is needed or
 * touched).  fused != 0 plans the one-launch decode kernel that rotates and quantizes
 * the token rows itself (dptq_qlinear additionally uses it only for K <= 16384 and
 * when its token padding equals the two-launch plan's).  Writes DPTQ_PLAN_INFO_LEN
 * ints to info (host memory, caller-owned), in this order:
 *   0 token tile NT (MMA N)         1 k-blocks of 128 per stage     2 padded tokens M_pad
 *   3 grid (CTAs)                   4 dynamic shared memory bytes   5 bulk-copy stages
 *   6 widened-weight slots          7 widened weights in TMEM (1) or shared memory (0)
 *   8 TMEM accumulator buffers      9 exact-accumulation segments   10 stages per segment
 *   11 TMEM columns allocated       12 first TMEM column of the weight slots (= the
 *   accumulators' columns)          13 stages per tile (KI)         14 weight tiles (N/128)
 *   15 token tiles                  16 tiles processed whole        17 stream-K stages
 *   (saturated at INT_MAX)          18 parts per token row (fused)  19 fused (1/0).
 * INVALID_ARG for sizes < 1, bits not 4/8, a null or short info; UNSUPPORTED when no
 * plan fits (e.g. a fused plan for more than 64 tokens). */
#define DPTQ_PLAN_INFO_LEN 20
dptq_status dptq_plan_info(int M, int N, int K, int bits, int num_sms, int fused, int* info, int info_len);

/* Copy the packed weights out in the public layout: wq_host uint8 [N][K/2] (same
 * nibble format as 4-bit activation codes) and sw_host float [N].  Either may be
 * NULL.  Synchronous (test access). */
dptq_status dptq_get_packed(dptq_handle h, void* wq_host, float* sw_host);

/* Shape of a handle (any pointer may be NULL). */
dptq_status dptq_get_shape(dptq_handle h, int* N, int* K, int* had_block);

/* Synchronize the device and report (and clear) the device error word set by a
 * bounded wait that gave up: DPTQ_OK or DPTQ_ERR_TIMEOUT.  `h` may be NULL.  Covers the
 * per-device scratch of the allocating calls and the fixed array of dptq_qlinear_static;
 * after a timeout it also zeroes the split-tile sums and counters the aborted kernel may
 * have left, so that later calls start clean. */
dptq_status dptq_last_device_error(dptq_handle h);

/* Test hook: the activation-plane and scale buffers of the current device's scratch,
 * current ones first, then the ones that growth superseded (newest first).  Writes up to
 * `max` entries: ptrs[i] (device address), bytes[i], and allocated[i] = 1 when the CUDA
 * runtime still reports ptrs[i] as a device allocation; *count = the number of buffers
 * held.  Host memory, caller-owned.  INVALID_ARG for a null count, or null arrays with
 * max > 0. */
dptq_status dptq_scratch_buffers(void** ptrs, size_t* bytes, int* allocated, int max, int* count);

/* Release a handle and its device memory.  NULL is ignored.  Must not be called
 * while work using the handle is still running. */
void dptq_destroy(dptq_handle h);

/* Static description of a status code. */
const char* dptq_status_str(dptq_status s);

/* Message of the last failing call on this thread ("" if none). */
const char* dptq_last_error_message(void);

#ifdef __cplusplus
}
#endif

#endif /* DPTQ_H_ */
