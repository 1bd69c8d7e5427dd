/*
 * fqvit.h -- C ABI of libfqvit.so: the integer inference hot path of
 * FQ-ViT ("Post-Training Quantization for Fully Quantized Vision
 * Transformer", IJCAI 2022) on one GB300 GPU (sm_103a).
 *
 * Conventions for every entry point
 *   - Pointers are DEVICE pointers owned by the caller unless stated
 *     otherwise.  Nothing is retained after the call returns; the library
 *     allocates no device memory.
 *   - Every call is asynchronous on `stream` (a cudaStream_t passed as
 *     void*; NULL is the legacy default stream).  Results are ready when
 *     the stream reaches the call.
 *   - Matrices are row-major.  ld_* are row strides in ELEMENTS of the
 *     matrix's type (bytes for 8-bit data).
 *   - Return value: FQVIT_OK or one of the error codes below.  Arguments
 *     are validated on the host before anything is launched; on error
 *     nothing is launched and fqvit_last_error() describes the problem.
 *   - Scalars that the paper computes offline after calibration (s, zp,
 *     s_out, zp_out, s_logit) are passed by value.
 */
#ifndef FQVIT_H
#define FQVIT_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define FQVIT_API __attribute__((visibility("default")))
#else
#define FQVIT_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

#define FQVIT_OK 0
#define FQVIT_ERR_INVALID_ARG 1 /* NULL, bad size, stride or alignment            */
#define FQVIT_ERR_UNSUPPORTED 2 /* valid in the paper, not handled by this build  */
#define FQVIT_ERR_RANGE 3       /* reserved: a value outside an exactness bound   */
#define FQVIT_ERR_CUDA 4        /* a CUDA launch or runtime call failed           */
#define FQVIT_ERR_TIMEOUT 5     /* a kernel gave up a bounded wait (see below)    */

/* Library version, (major << 16) | minor. */
FQVIT_API int fqvit_version(void);

/* Thread-local description of the last non-OK status returned on this
 * thread (empty string if none).  Valid until the next call on the thread. */
FQVIT_API const char *fqvit_last_error(void);

/* Synchronizes `stream` and reports the library's device status word:
 * FQVIT_ERR_TIMEOUT if a kernel of this library abandoned a bounded wait
 * (every wait on an asynchronous copy or tensor-core operation gives up after
 * two seconds, drains what it issued and returns) since the last call,
 * FQVIT_ERR_INVALID_ARG if fqvit_linear_q met a per-channel weight scale that
 * is not positive and finite (device data the host does not see),
 * FQVIT_ERR_UNSUPPORTED if a kernel found its shared-memory layout different
 * from the one the host computed and returned without writing its output,
 * FQVIT_ERR_CUDA if the stream reports an error, else FQVIT_OK.  The word is
 * cleared.  Not part of the paper; a diagnostic of this implementation. */
FQVIT_API int fqvit_sync_status(void *stream);

/* Exercises the failure path of the bounded waits without a fault: launches
 * one CTA on `stream` whose thread waits, through the same bounded wait the
 * kernels use, on an mbarrier that nothing completes.  The wait gives up
 * after two seconds and records the timeout; the next fqvit_sync_status
 * returns FQVIT_ERR_TIMEOUT and the context stays usable.  Returns
 * FQVIT_ERR_CUDA if the launch fails.  Not part of the paper. */
FQVIT_API int fqvit_selftest_bounded_wait(void *stream);

/* ------------------------------------------------------------------ */
/* Power-of-Two Factor calibration (Sec. 3.2, Eqs. 8-10)              */
/* ------------------------------------------------------------------ */

/* Bytes of device workspace fqvit_calibrate_ptf needs (a few KB). */
FQVIT_API size_t fqvit_calibrate_workspace_size(int64_t rows, int32_t C, int32_t K);

/* The same size under the name of the planned interface: the workspace does not depend on the
 * number of calibration rows (the min / max pass keeps at most 1024 block partials), so
 * fqvit_workspace_size(C, K) == fqvit_calibrate_workspace_size(rows, C, K) for every rows >= 1.
 * 0 for C < 1 or K outside 0..7. */
FQVIT_API size_t fqvit_workspace_size(int32_t C, int32_t K);

/*
 * Layer-wise scale s and zero point zp (Eqs. 8-9) and per-channel factors
 * alpha_c in {0..K} (Eq. 10) from a calibration batch x [rows, C] fp32.
 *   s0 = (max x - min x) / (2^bits - 1) in fp32 (a zero range counts as 1),
 *   s  = s0 / 2^K,  zp = clip(rint(-min x / s0), 0, 2^bits - 1).
 *   err_c(a) = sum over rows, in ascending row order, in fp64, of
 *     (x - clip(rint(x / (2^a s)), -zp, 255 - zp) * 2^a s)^2,
 *   the quotient, rint, product and difference being fp32; alpha_c is the
 *   smallest a with the least error.
 * Outputs (device): s[1], zp[1], alpha[C]; sse_opt[C][K+1] if not NULL.
 * workspace: device buffer of fqvit_calibrate_workspace_size() bytes,
 *   8-byte aligned; its contents on entry do not matter.
 * Supported: bits == 8, 0 <= K <= 7, 1 <= C <= 8192, ld_x >= C, rows >= 1.
 * x must be finite.
 */
FQVIT_API int fqvit_calibrate_ptf(const float *x, int64_t rows, int32_t C, int64_t ld_x,
                        int32_t bits, int32_t K, float *s, int32_t *zp, uint8_t *alpha,
                        double *sse_opt, void *workspace, size_t ws_bytes, void *stream);

/*
 * Same calibration as fqvit_calibrate_ptf, for callers that cannot allocate
 * device memory: code that must not allocate once it runs (real-time or
 * certified inference with a fixed memory budget) and code whose device memory
 * is owned by another allocator that gives out no extra buffer.  There is no
 * counterpart in the paper; it is an interface of this library.
 *   - No workspace argument: the kernels use a fixed 160 KiB array of device
 *     memory that belongs to the library, one per GPU, kept until the process
 *     ends or the context is reset.  The call itself allocates nothing.
 *   - The array is reserved when the library's code is loaded on a GPU.  With
 *     CUDA's default lazy module loading that is the first call on that GPU
 *     (its lookup of the array's address loads the code), so that first call
 *     may take device memory: make it at start-up, before the memory budget is
 *     fixed and before any stream capture (or set CUDA_MODULE_LOADING=EAGER).
 *     Later calls take none.
 *   - Limit, when sse_opt is NULL (the error sums are then kept in the array):
 *     C * (K + 1) <= 16384 (e.g. C = 4096 at K = 3); larger problems return
 *     FQVIT_ERR_UNSUPPORTED -- pass sse_opt, or use fqvit_calibrate_ptf with a
 *     workspace.  With sse_opt any supported C and K fit.
 *   - All calls share the array, which keeps the last call's contents (no
 *     call needs it zeroed).  Calls whose kernels overlap on the GPU race on
 *     it: do not run two of them concurrently.
 * Arguments, outputs and results are those of fqvit_calibrate_ptf.
 */
FQVIT_API int fqvit_calibrate_ptf_noalloc(const float *x, int64_t rows, int32_t C, int64_t ld_x,
                                          int32_t bits, int32_t K, float *s, int32_t *zp,
                                          uint8_t *alpha, double *sse_opt, void *stream);

/*
 * Sharded calibration: the batch of fqvit_calibrate_ptf split by rows over
 * `world` ranks (one GPU each), with the same s, zp and alpha on every rank.
 * Eqs. 8-9 need the global range and Eq. 10 sums over all rows, so the batch
 * is calibrated in three stages with two exchanges in between (done by the
 * caller, e.g. torch.distributed):
 *   1. fqvit_calibrate_minmax on each rank's rows -> its (min, max);
 *      all-reduce MIN / MAX -> the global range (exact: any split gives the
 *      unsplit range, hence the unsplit s and zp);
 *   2. fqvit_calibrate_sse_partial on each rank's rows with the global range
 *      -> its err_c(a) sums (ascending row order within the rank, fp64);
 *      all-gather;
 *   3. fqvit_calibrate_combine (host) -> the per-rank sums added in rank
 *      order starting from 0.0, alpha_c = the smallest a with the least
 *      total, and s, zp of the global range.
 * Every rank combining the same gathered sums gets identical results; one
 * rank reproduces fqvit_calibrate_ptf exactly.  Sums of several ranks differ
 * from the unsplit sequential sum only by fp64 rounding.
 */

/* Stage 1.  mnmx (device, float[2]) <- exact (min, max) of x [rows, C].
 * workspace: device, >= fqvit_calibrate_workspace_size(rows, C, 0) bytes,
 * 8-byte aligned.  Shapes as fqvit_calibrate_ptf; x must be finite. */
FQVIT_API int fqvit_calibrate_minmax(const float *x, int64_t rows, int32_t C, int64_t ld_x, float *mnmx,
                                     void *workspace, size_t ws_bytes, void *stream);

/* Stage 2.  sse (device, double[C][K+1]) <- err_c(a) of Eq. 10 over the
 * rows of x for the global range mnmx (device, float[2], min <= max).
 * workspace: device, >= 64 bytes, 8-byte aligned.  bits == 8, 0 <= K <= 7. */
FQVIT_API int fqvit_calibrate_sse_partial(const float *x, int64_t rows, int32_t C, int64_t ld_x, int32_t bits,
                                          int32_t K, const float *mnmx, double *sse, void *workspace,
                                          size_t ws_bytes, void *stream);

/* Stage 3, host only (no GPU call).  sse_parts: host double[world][C][K+1]
 * in rank order; (mn, mx): the global range.  Outputs (host): s, zp,
 * alpha[C]; sse_total[C][K+1] if not NULL.  INVALID_ARG if mn > mx. */
FQVIT_API int fqvit_calibrate_combine(const double *sse_parts, int32_t world, int32_t C, int32_t K, float mn,
                                      float mx, float *s, int32_t *zp, uint8_t *alpha, double *sse_total);

/*
 * PTF quantizer (Eq. 7): xq[r][c] = clip(rint(x[r][c] / (2^alpha_c s)) + zp, 0, 255),
 * fp32 quotient, ties to even.  x [rows, C] fp32, alpha [C] (device),
 * xq [rows, C] uint8 with stride ld_q.
 */
FQVIT_API int fqvit_ptf_quantize(const float *x, int64_t rows, int32_t C, int64_t ld_x, float s,
                       int32_t zp, const uint8_t *alpha, uint8_t *xq, int64_t ld_q,
                       void *stream);

/* ------------------------------------------------------------------ */
/* Integer LayerNorm on PTF-quantized input (supplement, "Quantized    */
/* Inference of LayerNorm", Eqs. 11-13 and the dyadic requantization)  */
/* ------------------------------------------------------------------ */

/*
 * Per row of xq [rows, C] (uint8, stride ld_in):
 *   Xh_c = (xq_c - zp_in) * 2^alpha_c;  M1 = sum Xh;  M2 = sum Xh^2 (int64);
 *   D = C M2 - M1^2;  sd = sqrtf((float)D);  r = C / sd;  t = (float)M1 / sd
 *   (fp32, correctly rounded; r = t = 0 when D == 0, i.e. a constant row);
 *   gs_c = gamma_c / s_out, bs_c = beta_c / s_out (fp32);
 *   A = gs_c r, B = bs_c - gs_c t (fp32, no fused multiply-add);
 *   N1 = min(7 - floor(log2 |A|), 31), N2 = floor(|A| 2^N1) (A == 0: 0, 0);
 *   Bq = rint(B 2^N1);  Y = clip(round_half_up((sign(A) N2 Xh + Bq) / 2^N1)
 *                              + zp_out, 0, 255)   (N1 < 0 multiplies).
 * The input scale s cancels (A and B are independent of it) and is not an
 * argument.  Output yq [rows, C] uint8, stride ld_out.  m1_opt / m2_opt
 * (int64 [rows]) receive M1 / M2 when not NULL.
 * Supported: 1 <= C <= 8192, alpha_c <= 7, s_out > 0 and finite.
 */
FQVIT_API int fqvit_ptf_layernorm(const uint8_t *xq, int64_t rows, int32_t C, int64_t ld_in,
                        int32_t zp_in, const uint8_t *alpha, const float *gamma,
                        const float *beta, float s_out, int32_t zp_out, uint8_t *yq,
                        int64_t ld_out, int64_t *m1_opt, int64_t *m2_opt, void *stream);

/* ------------------------------------------------------------------ */
/* Log-Int-Softmax (Sec. 3.3, Eqs. 16-17; supplement Algorithms 1-2)  */
/* ------------------------------------------------------------------ */

/* Relative-position bias for windowed (Swin) attention, not in the paper:
 * table [heads][(2 window - 1)^2] int8 (device), same scale as the
 * logits; the entry for query i, key j of a window is at
 * (y_i - y_j + window - 1)(2 window - 1) + (x_i - x_j + window - 1)
 * with y = index / window, x = index % window. */
typedef struct fqvit_relpos_bias {
    const int8_t *table;
    int32_t heads;
    int32_t window;
} fqvit_relpos_bias;

/* Shifted-window attention mask (Swin, not in the paper): region ids
 * [n_windows][L] uint8 (device); rows are ordered [batch][window][head]
 * [query], so row r belongs to window (r / (L heads)) % n_windows.  Key j of
 * query i gets mask_value (logit units, -32768 .. 0) added to its logit when
 * region[w][i] != region[w][j]; the bias, if any, is added too. */
typedef struct fqvit_window_mask {
    const uint8_t *region;
    int32_t n_windows;
    int32_t mask_value;
} fqvit_window_mask;

/*
 * Log-Int-Softmax of n_rows rows of int8 logits (stride ld_logit bytes,
 * L keys per row; rows ordered [batch][head][query]):
 *   q~ = q (+ bias) - max;  e = i-exp(q~) with q_ln2 = floor(-ln2/s),
 *   q_b = floor(1.353/s), q_c = floor(0.344/(0.3585 s^2)) in fp64, the
 *   clamp q~ >= n q_ln2, z = q~ / q_ln2, q_p = q~ - z q_ln2,
 *   e = ((q_p + q_b)^2 + q_c) << (n - z)   (Algorithm 1);
 *   S = sum e;  q_rev = floor((2S + e) / (2e))  (round half up);
 *   code = min(I-Log2(q_rev), 15)  (Algorithm 2, Eq. 33; I-Log2(x) = M + bit
 *   M-1 of x, M the index of the leading one).
 * The code is Attn_Q (4 bits); the LIS output of Eq. 17 is 15 - code with
 * scale 1/2^15.  codes: packed nibbles, code of key j in byte j/2 of the
 * row (low nibble for even j), row stride ld_codes >= ceil(L/2) bytes; a
 * pad nibble of odd L is written as 0.  rowsum_opt (uint64 [n_rows])
 * receives S when not NULL.
 * Supported: n_shift == 15 (the exponent headroom n of Algorithm 1), 1 <= L
 * <= 1024, s_logit in [2^-7, 0.5] (the range where every i-exp value fits 31
 * bits), ld_logit a multiple of 4 and >= L.  With bias_opt: window^2 == L,
 * heads >= 1, n_rows a multiple of heads * L.
 */
FQVIT_API int fqvit_lis_softmax(const int8_t *logits, int64_t n_rows, int32_t L, int64_t ld_logit,
                      float s_logit, int32_t n_shift, const fqvit_relpos_bias *bias_opt,
                      uint8_t *codes, int64_t ld_codes, uint64_t *rowsum_opt, void *stream);

/*
 * BitShift attention times values (Eq. 15; supplement Attn.V):
 *   acc[bh][i][t] = sum_j (v[bh][j][t] - zp_v) << (15 - code[bh][i][j])
 * (a left shift of a negative value is a multiplication by 2^(15 - code));
 * the real result is acc * s_V / 2^15.
 * codes: packed nibbles as written by fqvit_lis_softmax, [BH * L] rows of
 * ld_codes bytes.  v: int8 [BH][L][ld_v] (head stride L * ld_v).  acc: int32
 * [BH][L][ld_acc] (head stride L * ld_acc).  range_flag_opt (device int32)
 * is set to 1 if some row's sum could leave int32 (arbitrary codes only;
 * never for codes made by fqvit_lis_softmax); it is not cleared.
 * Supported: d in {32, 64}, 1 <= L <= 1024, |zp_v| <= 255.
 */
FQVIT_API int fqvit_lis_attn_v(const uint8_t *codes, int64_t ld_codes, const int8_t *v, int64_t ld_v,
                     int32_t zp_v, int64_t BH, int32_t L, int32_t d, int32_t *acc,
                     int64_t ld_acc, int32_t *range_flag_opt, void *stream);

/*
 * Fused Log-Int-Softmax and BitShift attention times values: the same
 * result as fqvit_lis_softmax followed by fqvit_lis_attn_v, without the
 * codes leaving the chip unless codes_opt is not NULL (then they are also
 * written, packed as above).  logits [BH * L] rows of ld_logit bytes, v and
 * acc as in fqvit_lis_attn_v.
 * Supported: as fqvit_lis_softmax and fqvit_lis_attn_v.
 */
FQVIT_API int fqvit_lis_attention(const int8_t *logits, int64_t ld_logit, float s_logit,
                        int32_t n_shift, const fqvit_relpos_bias *bias_opt, const int8_t *v,
                        int64_t ld_v, int32_t zp_v, int64_t BH, int32_t L, int32_t d,
                        int32_t *acc, int64_t ld_acc, uint8_t *codes_opt, int64_t ld_codes,
                        void *stream);

/*
 * The fused attention with its output requantized to 8 bits for the next
 * layer (the activation quantizer of Eq. 3, scale s_out, zero point zp_out),
 * evaluated with the dyadic multiplier of the supplement's LayerNorm output
 * stage: the real output acc * s_v / 2^15 (Eq. 15) becomes
 *   M  = (s_v / s_out) / 2^15   (one fp32 division, then an exact scaling),
 *   N1 = 7 - floor(log2 M) (at most 31),  N2 = floor(M 2^N1)  (8 bits),
 *   out = clip(floor((N2 acc + 2^(N1-1)) / 2^N1) + zp_out, 0, 255)  (N1 > 0),
 *   out = clip(N2 acc 2^min(-N1, 10) + zp_out, 0, 255)             (N1 <= 0).
 * The int32 accumulators are not written.  out: uint8 [BH][L][ld_out]
 * (device, caller-owned), ld_out >= d.  Other arguments as in
 * fqvit_lis_attention.  Errors: INVALID_ARG for a NULL out, ld_out < d,
 * s_v or s_out not positive and finite, zp_out outside 0..255; UNSUPPORTED
 * when M leaves the fp32 range; otherwise as fqvit_lis_attention.
 */
FQVIT_API int fqvit_lis_attention_q(const int8_t *logits, int64_t ld_logit, float s_logit,
                          int32_t n_shift, const fqvit_relpos_bias *bias_opt, const int8_t *v,
                          int64_t ld_v, int32_t zp_v, int64_t BH, int32_t L, int32_t d,
                          float s_v, float s_out, int32_t zp_out, uint8_t *out, int64_t ld_out,
                          void *stream);

/*
 * fqvit_lis_softmax and fqvit_lis_attention with a shifted-window mask
 * (mask may be NULL: then they are those functions).  The mask requires
 * n_rows (BH * L) to be a multiple of heads * L * n_windows, heads from
 * bias_opt (1 without a bias).  Errors as those functions, plus INVALID_ARG
 * for a NULL region, n_windows < 1, a row count that is not such a multiple,
 * and UNSUPPORTED for mask_value outside -32768 .. 0.
 */
FQVIT_API int fqvit_lis_softmax_masked(const int8_t *logits, int64_t n_rows, int32_t L, int64_t ld_logit,
                      float s_logit, int32_t n_shift, const fqvit_relpos_bias *bias_opt,
                      const fqvit_window_mask *mask, uint8_t *codes, int64_t ld_codes,
                      uint64_t *rowsum_opt, void *stream);
FQVIT_API int fqvit_lis_attention_masked(const int8_t *logits, int64_t ld_logit, float s_logit,
                        int32_t n_shift, const fqvit_relpos_bias *bias_opt,
                        const fqvit_window_mask *mask, const int8_t *v, int64_t ld_v, int32_t zp_v,
                        int64_t BH, int32_t L, int32_t d, int32_t *acc, int64_t ld_acc,
                        uint8_t *codes_opt, int64_t ld_codes, void *stream);
/* fqvit_lis_attention_q with a shifted-window mask (mask may be NULL); the
 * mask's requirements and errors as fqvit_lis_attention_masked. */
FQVIT_API int fqvit_lis_attention_masked_q(const int8_t *logits, int64_t ld_logit, float s_logit,
                          int32_t n_shift, const fqvit_relpos_bias *bias_opt,
                          const fqvit_window_mask *mask, const int8_t *v, int64_t ld_v, int32_t zp_v,
                          int64_t BH, int32_t L, int32_t d, float s_v, float s_out, int32_t zp_out,
                          uint8_t *out, int64_t ld_out, void *stream);

/* ------------------------------------------------------------------ */
/* The MatMul Q K^T and its 8-bit output (Sec. 3 MinMax; Sec. 4.1)     */
/* ------------------------------------------------------------------ */

/*
 * Logits of attention from 8-bit Q and K codes.  Sec. 3 quantizes MatMul
 * outputs with uniform MinMax and Sec. 4.1 takes activations asymmetric, so Q
 * and K come with zero points and the product is quantized to 8 bits:
 *   P[bh][i][j] = sum_t (q[bh][i][t] - zp_q) (k[bh][j][t] - zp_k)   (exact)
 *   M  = (s_q s_k) / (sqrt(d) s_logit)  (fp32: a = s_q s_k, r = sqrtf(d),
 *        c = r s_logit, M = a / c),
 *   N1 = 7 - floor(log2 M) (at most 31), N2 = floor(M 2^N1)  (the dyadic
 *        multiplier of the supplement's LayerNorm output stage),
 *   logit = clip(floor((N2 P + 2^(N1-1)) / 2^N1) + zp_logit, -128, 127)
 *        (N1 <= 0: clip(N2 P 2^min(-N1, 10) + zp_logit, ...)).
 * Logits are signed (the 8-bit code minus 128; zp_logit likewise): the form
 * fqvit_lis_softmax and fqvit_lis_attention take.
 * q [BH][L][ld_q], k [BH][L][ld_k] int8 (device), d values per row;
 * logits [BH*L][ld_logit] int8 (device, caller-owned): row i of head bh at
 * bh*L + i, key j at byte j, bytes L .. ld_logit-1 of a row written as 0.
 * Supported: 1 <= L <= 640, d <= 64 a multiple of 8, ld_q and ld_k multiples
 * of 8 with 8-byte aligned bases, ld_logit a multiple of 16 with a 16-byte
 * aligned base, zero points in -128..127.  Errors: INVALID_ARG (NULL, shapes,
 * strides, alignment, zero points, scales not positive and finite),
 * UNSUPPORTED (L, d, or M outside the fp32 range).
 */
FQVIT_API int fqvit_qk_logits(const int8_t *q, int64_t ld_q, int32_t zp_q, const int8_t *k, int64_t ld_k,
                              int32_t zp_k, int64_t BH, int32_t L, int32_t d, float s_q, float s_k,
                              float s_logit, int32_t zp_logit, int8_t *logits, int64_t ld_logit, void *stream);

/* Bytes of logits workspace fqvit_qk_lis_attention needs for groups of
 * group_heads heads (<= 0: the library's choice, every head in one group up to
 * 1 GiB of logits; a smaller group bounds the workspace at the cost of more
 * launches): group x L x ld with ld = L rounded up to 16.  0 for a bad shape. */
FQVIT_API size_t fqvit_qk_workspace_size(int64_t BH, int32_t L, int64_t group_heads);

/*
 * Attention from 8-bit Q, K and V: fqvit_qk_logits, then
 * fqvit_lis_attention_masked on those logits (same arguments, bias and mask
 * optional), group after group of heads on the caller's stream; the logits of
 * a group live in `workspace` (device, caller-owned, at least one group:
 * fqvit_qk_workspace_size) and are overwritten by the next group.  Groups are
 * multiples of heads (bias) x n_windows (mask), at most group_heads (<= 0: the
 * library's choice) and what the workspace holds.  acc as in
 * fqvit_lis_attention.  Errors: those of the two functions; INVALID_ARG when
 * the workspace holds less than one group.
 */
FQVIT_API int fqvit_qk_lis_attention(const int8_t *q, int64_t ld_q, int32_t zp_q, const int8_t *k, int64_t ld_k,
                              int32_t zp_k, float s_q, float s_k, float s_logit, int32_t zp_logit,
                              int32_t n_shift, const fqvit_relpos_bias *bias_opt,
                              const fqvit_window_mask *mask_opt, const int8_t *v, int64_t ld_v,
                              int32_t zp_v, int64_t BH, int32_t L, int32_t d, int32_t *acc, int64_t ld_acc,
                              int8_t *workspace, size_t workspace_bytes, int64_t group_heads, void *stream);

/* ------------------------------------------------------------------ */
/* MinMax Linear layers of the block (Sec. 3; Sec. 4.1)                */
/* ------------------------------------------------------------------ */

/*
 * Weights of a Linear layer in the form fqvit_linear_q takes: int8 codes
 * w [N][ld_w] (symmetric, channel-wise; device) -> fp16 w_h [N][K] (device,
 * caller-owned, written once and kept with the model).  Every code is exact
 * in fp16.  Supported: K a multiple of 8, ld_w a multiple of 8 with an 8-byte
 * aligned base, w_h 16-byte aligned.  Errors: INVALID_ARG (NULL, shapes,
 * alignment), UNSUPPORTED (K).
 */
FQVIT_API int fqvit_linear_pack_weight(const int8_t *w, int32_t N, int32_t K, int64_t ld_w, uint16_t *w_h,
                                       void *stream);

/* Bytes of workspace fqvit_linear_q needs: the fp16 copy of the activations
 * (M x K x 2, rounded up to 256) and 4096 int32 per-channel weight sums.
 * 0 for a bad shape. */
FQVIT_API size_t fqvit_linear_workspace_size(int64_t M, int32_t K);

/*
 * A Linear layer of the fully quantized block.  Sec. 3 quantizes Linear
 * layers with uniform MinMax; Sec. 4.1 takes the weights symmetric and
 * channel-wise, the activations asymmetric and layer-wise:
 *   acc[m][n] = sum_k (x[m][k] - zp_x) w[n][k] + bias[n]        (exact, int32)
 *   M_n = (s_x s_w[n]) / s_y     (fp32, in this order)
 *   N1 = 7 - floor(log2 M_n) (at most 31), N2 = floor(M_n 2^N1)  (the dyadic
 *        multiplier of the supplement's LayerNorm output stage, per channel)
 *   y[m][n] = clip(floor((N2 acc + 2^(N1-1)) / 2^N1) + zp_y, 0, 255)
 *        (N1 <= 0: clip(N2 acc 2^min(-N1, 10) + zp_y, 0, 255)).
 * The bias is the integer bias at scale s_x s_w[n] (|bias[n]| <= 2^30).
 * x [M][ld_x] uint8 (device); w_h [N][K] from fqvit_linear_pack_weight;
 * s_w [N] float and bias_opt [N] int32 (device; bias NULL = none);
 * y [M][ld_y] uint8 (device, caller-owned); acc_opt [M][ld_acc] int32
 * (device, may be NULL) receives acc; workspace (device, caller-owned, at
 * least fqvit_linear_workspace_size(M, K) bytes, 16-byte aligned) is
 * overwritten.  Three launches on `stream`: the per-channel weight sums, the
 * fp16 copy of x - 128 (the product runs on x - 128 and adds
 * (128 - zp_x) sum_k w[n][k] to the bias, the same integer), then the
 * tensor-core product and its requantization.
 * Supported: K <= 16384 a multiple of 8, N <= 4096 a multiple of 16,
 * ld_x a multiple of 8 with an 8-byte aligned base, ld_y a multiple of 16 and
 * ld_acc of 4 with 16-byte aligned bases, zero points in 0..255.  Errors:
 * INVALID_ARG (NULL, shapes, strides, alignment, zero points, s_x or s_y not
 * positive and finite, a small workspace), UNSUPPORTED (K, N, M >= 2^31).  A
 * weight scale that is not positive and finite is device data: its channel
 * holds zp_y and fqvit_sync_status reports INVALID_ARG.
 */
FQVIT_API int fqvit_linear_q(const uint8_t *x, int64_t M, int32_t K, int64_t ld_x, int32_t zp_x, float s_x,
                             const uint16_t *w_h, int32_t N, const float *s_w, const int32_t *bias_opt, float s_y,
                             int32_t zp_y, uint8_t *y, int64_t ld_y, int32_t *acc_opt, int64_t ld_acc,
                             void *workspace, size_t workspace_bytes, void *stream);

/* ------------------------------------------------------------------ */
/* Head split and merge around the attention core (Fig. 4 dataflow)   */
/* ------------------------------------------------------------------ */

/*
 * The QKV Linear's token-major output to head-major Q, K and V codes for
 * fqvit_qk_logits and the attention calls: qkv [B*L][ld_qkv] uint8 (device),
 * part p (0 Q, 1 K, 2 V) in columns p*H*d .. p*H*d + H*d - 1, head h at
 * + h*d; q, k, v [B*H][L][ld_head] int8 (device, caller-owned), row
 * (b*H + h)*L + i = the code of token b*L + i minus 128 (the signed form
 * those calls take; the zero point moves by -128 with it).  Bytes past d of
 * an output row are not written.  Supported: d a multiple of 16, ld_qkv and
 * ld_head multiples of 16 with 16-byte aligned bases.  Errors: INVALID_ARG
 * (NULL, shapes, strides, alignment), UNSUPPORTED (d).
 */
FQVIT_API int fqvit_split_qkv(const uint8_t *qkv, int64_t B, int32_t L, int32_t H, int32_t d, int64_t ld_qkv,
                              int8_t *q, int8_t *k, int8_t *v, int64_t ld_head, void *stream);

/*
 * The attention output's head-major rows back to token rows for the
 * projection Linear: heads [B*H][L][ld_head] uint8 (device; the 8-bit output
 * of fqvit_lis_attention_q) -> out [B*L][ld_out] uint8 (device,
 * caller-owned), head h in columns h*d .. h*d + d - 1 (codes unchanged).
 * Supported and errors as fqvit_split_qkv.
 */
FQVIT_API int fqvit_merge_heads(const uint8_t *heads, int64_t B, int32_t L, int32_t H, int32_t d,
                                int64_t ld_head, uint8_t *out, int64_t ld_out, void *stream);

/* ------------------------------------------------------------------ */
/* One layer: norm1 LayerNorm and the attention core (Fig. 4 dataflow) */
/* ------------------------------------------------------------------ */

typedef struct fqvit_block_desc {
    /* PTF LayerNorm (see fqvit_ptf_layernorm), contiguous rows */
    const uint8_t *xq;
    int64_t rows;
    int32_t C;
    int32_t zp_in;
    const uint8_t *alpha;
    const float *gamma;
    const float *beta;
    float s_out;
    int32_t zp_out;
    uint8_t *yq;
    /* attention core (see fqvit_lis_attention); logits rows padded to ld_logit */
    const int8_t *logits;
    int64_t ld_logit;
    float s_logit;
    const int8_t *v;   /* [BH][L][d] contiguous */
    int32_t zp_v;
    int64_t BH;
    int32_t L;
    int32_t d;
    const fqvit_relpos_bias *bias; /* NULL = none */
    int32_t *acc;      /* [BH][L][d] contiguous */
} fqvit_block_desc;

/* Runs the LayerNorm and the fused attention of one layer on `stream`
 * (two launches, in that order).  Supported: as the two calls. */
FQVIT_API int fqvit_block_int(const fqvit_block_desc *desc, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* FQVIT_H */
