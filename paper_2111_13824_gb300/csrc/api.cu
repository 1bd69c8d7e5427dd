// api.cu -- extern "C" entry points of libfqvit.so (declared in
// include/fqvit.h): host-side validation, then launches on the caller's
// stream.  Nothing is allocated and nothing is retained.
#include "fqvit.h"
#include "fqvit_internal.cuh"

#include <cstdarg>
#include <cstdio>
#include <cstring>

namespace {

thread_local char g_err[512] = "";

int fail(int code, const char *fmt, ...)
{
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
    return code;
}

int ok()
{
    g_err[0] = '\0';
    return FQVIT_OK;
}

int cuda_status(cudaError_t e, const char *what)
{
    if (e != cudaSuccess) return fail(FQVIT_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
    return ok();
}

bool aligned(const void *p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

cudaStream_t as_stream(void *s) { return reinterpret_cast<cudaStream_t>(s); }

// s_logit range in which every i-exp value fits 31 bits (see lis.cu)
bool logit_scale_ok(float s) { return s >= 0.0078125f && s <= 0.5f; }

}  // namespace

namespace fqvit {

int sm_count()
{
    static int cached[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
    if (cached[dev] == 0) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
        cached[dev] = n;
    }
    return cached[dev];
}

cudaError_t check_smem_fits(const void *kernel, size_t dynamic)
{
    cudaFuncAttributes fa;
    cudaError_t e = cudaFuncGetAttributes(&fa, kernel);
    if (e != cudaSuccess) return e;
    int dev = 0, optin = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev)) != cudaSuccess) return e;
    return fa.sharedSizeBytes + dynamic <= (size_t)optin ? cudaSuccess : cudaErrorInvalidConfiguration;
}

int record_error(int code, const char *msg)
{
    if (code == FQVIT_OK) return ok();
    return fail(code, "%s", msg);
}

}  // namespace fqvit

extern "C" {

int fqvit_version(void) { return (0 << 16) | 1; }

const char *fqvit_last_error(void) { return g_err; }

int fqvit_sync_status(void *stream)
{
    int status = 0;
    cudaError_t e = fqvit::read_clear_device_status(&status, as_stream(stream));
    if (e != cudaSuccess) return fail(FQVIT_ERR_CUDA, "sync_status: %s", cudaGetErrorString(e));
    int lst = 0;  // the Linear layers' status word (linear_tc.cu)
    e = fqvit::read_clear_linear_status(&lst);
    if (e != cudaSuccess) return fail(FQVIT_ERR_CUDA, "sync_status: %s", cudaGetErrorString(e));
    if (status == 0 || (status == FQVIT_ERR_INVALID_ARG && lst == FQVIT_ERR_TIMEOUT)) status = lst;
    if (status == FQVIT_ERR_TIMEOUT)
        return fail(FQVIT_ERR_TIMEOUT, "a kernel abandoned a bounded wait (results of that launch are invalid)");
    if (status == FQVIT_ERR_UNSUPPORTED)
        return fail(FQVIT_ERR_UNSUPPORTED,
                    "a kernel found its shared-memory layout different from the host's (that launch wrote no "
                    "output)");
    if (status == FQVIT_ERR_INVALID_ARG)
        return fail(FQVIT_ERR_INVALID_ARG,
                    "a Linear layer met a weight scale s_w[n] that is not positive and finite, or a multiplier "
                    "s_x s_w[n] / s_y outside (0, 1e30) (those channels hold zp_y)");
    return ok();
}

size_t fqvit_calibrate_workspace_size(int64_t rows, int32_t C, int32_t K)
{
    if (C < 1 || K < 0 || K > 7) return 0;
    return fqvit::calibrate_workspace_bytes(rows, C, K);
}

size_t fqvit_workspace_size(int32_t C, int32_t K) { return fqvit_calibrate_workspace_size(1, C, K); }

int fqvit_calibrate_ptf(const float *x, int64_t rows, int32_t C, int64_t ld_x, int32_t bits,
                        int32_t K, float *s, int32_t *zp, uint8_t *alpha, double *sse_opt,
                        void *workspace, size_t ws_bytes, void *stream)
{
    if (!x || !s || !zp || !alpha || !workspace) return fail(FQVIT_ERR_INVALID_ARG, "calibrate_ptf: NULL pointer");
    if (rows < 1 || C < 1 || C > 8192 || ld_x < C)
        return fail(FQVIT_ERR_INVALID_ARG, "calibrate_ptf: bad shape rows=%lld C=%d ld_x=%lld",
                    (long long)rows, C, (long long)ld_x);
    if (bits != 8) return fail(FQVIT_ERR_UNSUPPORTED, "calibrate_ptf: bits=%d (only 8)", bits);
    if (K < 0 || K > 7) return fail(FQVIT_ERR_UNSUPPORTED, "calibrate_ptf: K=%d (0..7)", K);
    if (!aligned(x, 4) || !aligned(s, 4) || !aligned(zp, 4) || !aligned(workspace, 8) ||
        (sse_opt && !aligned(sse_opt, 8)))
        return fail(FQVIT_ERR_INVALID_ARG, "calibrate_ptf: misaligned pointer");
    size_t need = fqvit::calibrate_workspace_bytes(rows, C, K);
    if (ws_bytes < need)
        return fail(FQVIT_ERR_INVALID_ARG, "calibrate_ptf: workspace %zu bytes, need %zu", ws_bytes, need);
    return cuda_status(fqvit::launch_calibrate(x, rows, C, ld_x, K, s, zp, alpha, sse_opt, workspace,
                                               as_stream(stream)),
                       "calibrate_ptf");
}

int fqvit_calibrate_minmax(const float *x, int64_t rows, int32_t C, int64_t ld_x, float *mnmx, void *workspace,
                           size_t ws_bytes, void *stream)
{
    if (!x || !mnmx || !workspace) return fail(FQVIT_ERR_INVALID_ARG, "calibrate_minmax: NULL pointer");
    if (rows < 1 || C < 1 || C > 8192 || ld_x < C)
        return fail(FQVIT_ERR_INVALID_ARG, "calibrate_minmax: bad shape rows=%lld C=%d ld_x=%lld", (long long)rows,
                    C, (long long)ld_x);
    if (!aligned(x, 4) || !aligned(mnmx, 4) || !aligned(workspace, 8))
        return fail(FQVIT_ERR_INVALID_ARG, "calibrate_minmax: misaligned pointer");
    size_t need = fqvit::calibrate_workspace_bytes(rows, C, 0);
    if (ws_bytes < need)
        return fail(FQVIT_ERR_INVALID_ARG, "calibrate_minmax: workspace %zu bytes, need %zu", ws_bytes, need);
    return cuda_status(fqvit::launch_calibrate_minmax(x, rows, C, ld_x, mnmx, workspace, as_stream(stream)),
                       "calibrate_minmax");
}

int fqvit_calibrate_sse_partial(const float *x, int64_t rows, int32_t C, int64_t ld_x, int32_t bits, int32_t K,
                                const float *mnmx, double *sse, void *workspace, size_t ws_bytes, void *stream)
{
    if (!x || !mnmx || !sse || !workspace) return fail(FQVIT_ERR_INVALID_ARG, "calibrate_sse_partial: NULL pointer");
    if (rows < 1 || C < 1 || C > 8192 || ld_x < C)
        return fail(FQVIT_ERR_INVALID_ARG, "calibrate_sse_partial: bad shape rows=%lld C=%d ld_x=%lld",
                    (long long)rows, C, (long long)ld_x);
    if (bits != 8) return fail(FQVIT_ERR_UNSUPPORTED, "calibrate_sse_partial: bits=%d (only 8)", bits);
    if (K < 0 || K > 7) return fail(FQVIT_ERR_UNSUPPORTED, "calibrate_sse_partial: K=%d (0..7)", K);
    if (!aligned(x, 4) || !aligned(mnmx, 4) || !aligned(sse, 8) || !aligned(workspace, 8))
        return fail(FQVIT_ERR_INVALID_ARG, "calibrate_sse_partial: misaligned pointer");
    if (ws_bytes < 64) return fail(FQVIT_ERR_INVALID_ARG, "calibrate_sse_partial: workspace %zu bytes, need 64", ws_bytes);
    return cuda_status(
        fqvit::launch_calibrate_sse_partial(x, rows, C, ld_x, K, mnmx, sse, workspace, as_stream(stream)),
        "calibrate_sse_partial");
}

int fqvit_calibrate_combine(const double *sse_parts, int32_t world, int32_t C, int32_t K, float mn, float mx,
                            float *s, int32_t *zp, uint8_t *alpha, double *sse_total)
{
    if (!sse_parts || !s || !zp || !alpha) return fail(FQVIT_ERR_INVALID_ARG, "calibrate_combine: NULL pointer");
    if (world < 1 || C < 1 || C > 8192) return fail(FQVIT_ERR_INVALID_ARG, "calibrate_combine: world=%d C=%d", world, C);
    if (K < 0 || K > 7) return fail(FQVIT_ERR_UNSUPPORTED, "calibrate_combine: K=%d (0..7)", K);
    if (!(mn <= mx) || !(mx - mn < 3.0e38f))
        return fail(FQVIT_ERR_INVALID_ARG, "calibrate_combine: range [%g, %g] is empty or not finite", (double)mn,
                    (double)mx);
    const int64_t n = (int64_t)C * (K + 1);
    for (int32_t c = 0; c < C; ++c) {
        int best = 0;
        double best_e = 0.0;
        for (int32_t a = 0; a <= K; ++a) {
            double t = 0.0;  // rank order, starting from zero: one rank gives its own sums back
            for (int32_t r = 0; r < world; ++r) t += sse_parts[r * n + (int64_t)c * (K + 1) + a];
            if (sse_total) sse_total[(int64_t)c * (K + 1) + a] = t;
            if (a == 0 || t < best_e) {
                best_e = t;
                best = a;
            }
        }
        alpha[c] = (uint8_t)best;
    }
    float s0;
    fqvit::calib_scale(mn, mx, K, s0, *s, *zp);
    return fail(FQVIT_OK, "");
}

int fqvit_ptf_quantize(const float *x, int64_t rows, int32_t C, int64_t ld_x, float s, int32_t zp,
                       const uint8_t *alpha, uint8_t *xq, int64_t ld_q, void *stream)
{
    if (!x || !alpha || !xq) return fail(FQVIT_ERR_INVALID_ARG, "ptf_quantize: NULL pointer");
    if (rows < 1 || C < 1 || C > 8192 || ld_x < C || ld_q < C)
        return fail(FQVIT_ERR_INVALID_ARG, "ptf_quantize: bad shape");
    if (!(s > 0.0f) || !(s < 3.0e38f)) return fail(FQVIT_ERR_INVALID_ARG, "ptf_quantize: s must be positive and finite");
    if (zp < 0 || zp > 255) return fail(FQVIT_ERR_INVALID_ARG, "ptf_quantize: zp=%d", zp);
    if (!aligned(x, 4)) return fail(FQVIT_ERR_INVALID_ARG, "ptf_quantize: misaligned x");
    return cuda_status(fqvit::launch_quantize(x, rows, C, ld_x, s, zp, alpha, xq, ld_q, as_stream(stream)),
                       "ptf_quantize");
}

int fqvit_ptf_layernorm(const uint8_t *xq, int64_t rows, int32_t C, int64_t ld_in, int32_t zp_in,
                        const uint8_t *alpha, const float *gamma, const float *beta, float s_out,
                        int32_t zp_out, uint8_t *yq, int64_t ld_out, int64_t *m1_opt, int64_t *m2_opt,
                        void *stream)
{
    if (!xq || !alpha || !gamma || !beta || !yq) return fail(FQVIT_ERR_INVALID_ARG, "ptf_layernorm: NULL pointer");
    if (rows < 1 || C < 1 || C > 8192 || ld_in < C || ld_out < C)
        return fail(FQVIT_ERR_INVALID_ARG, "ptf_layernorm: bad shape rows=%lld C=%d", (long long)rows, C);
    if (zp_in < 0 || zp_in > 255 || zp_out < 0 || zp_out > 255)
        return fail(FQVIT_ERR_INVALID_ARG, "ptf_layernorm: zero point outside 0..255");
    if (!(s_out > 0.0f) || !(s_out < 3.0e38f))
        return fail(FQVIT_ERR_INVALID_ARG, "ptf_layernorm: s_out must be positive and finite");
    if (!aligned(gamma, 4) || !aligned(beta, 4) || (m1_opt && !aligned(m1_opt, 8)) || (m2_opt && !aligned(m2_opt, 8)))
        return fail(FQVIT_ERR_INVALID_ARG, "ptf_layernorm: misaligned pointer");
    fqvit::LnArgs a{xq, rows, C, ld_in, zp_in, alpha, gamma, beta, s_out, zp_out, yq, ld_out, m1_opt, m2_opt};
    return cuda_status(fqvit::launch_layernorm(a, as_stream(stream)), "ptf_layernorm");
}

static int check_lis(const int8_t *logits, int64_t n_rows, int32_t L, int64_t ld_logit, float s_logit,
                     int32_t n_shift, const fqvit_relpos_bias *bias, const char *who)
{
    if (!logits) return fail(FQVIT_ERR_INVALID_ARG, "%s: NULL logits", who);
    if (n_rows < 1 || L < 1 || ld_logit < L) return fail(FQVIT_ERR_INVALID_ARG, "%s: bad shape", who);
    if (L > 1024) return fail(FQVIT_ERR_UNSUPPORTED, "%s: L=%d (at most 1024)", who, L);
    if (ld_logit % 4 != 0 || !aligned(logits, 4))
        return fail(FQVIT_ERR_INVALID_ARG, "%s: logits rows must be 4-byte aligned (ld %% 4 == 0)", who);
    if (n_shift != 15) return fail(FQVIT_ERR_UNSUPPORTED, "%s: n_shift=%d (only 15)", who, n_shift);
    if (!logit_scale_ok(s_logit))
        return fail(FQVIT_ERR_UNSUPPORTED, "%s: s_logit=%g outside [2^-7, 0.5]", who, (double)s_logit);
    if (bias) {
        if (!bias->table || bias->heads < 1 || bias->window < 1)
            return fail(FQVIT_ERR_INVALID_ARG, "%s: bad relative-position bias", who);
        if (bias->window * bias->window != L)
            return fail(FQVIT_ERR_INVALID_ARG, "%s: window^2 != L", who);
        if (n_rows % ((int64_t)bias->heads * L) != 0)
            return fail(FQVIT_ERR_INVALID_ARG, "%s: rows not a multiple of heads*L", who);
        if ((int64_t)bias->heads * (2 * bias->window - 1) * (2 * bias->window - 1) > 64 * 1024)
            return fail(FQVIT_ERR_UNSUPPORTED, "%s: bias table too large", who);
    }
    return FQVIT_OK;
}

int fqvit_lis_softmax(const int8_t *logits, int64_t n_rows, int32_t L, int64_t ld_logit, float s_logit,
                      int32_t n_shift, const fqvit_relpos_bias *bias_opt, uint8_t *codes, int64_t ld_codes,
                      uint64_t *rowsum_opt, void *stream)
{
    int rc = check_lis(logits, n_rows, L, ld_logit, s_logit, n_shift, bias_opt, "lis_softmax");
    if (rc) return rc;
    if (!codes) return fail(FQVIT_ERR_INVALID_ARG, "lis_softmax: NULL codes");
    if (ld_codes < (L + 1) / 2) return fail(FQVIT_ERR_INVALID_ARG, "lis_softmax: ld_codes < ceil(L/2)");
    if (rowsum_opt && !aligned(rowsum_opt, 8)) return fail(FQVIT_ERR_INVALID_ARG, "lis_softmax: misaligned rowsum");
    fqvit::LisArgs a{logits, n_rows, L, ld_logit, s_logit,
                     bias_opt ? bias_opt->table : nullptr, bias_opt ? bias_opt->heads : 1,
                     bias_opt ? bias_opt->window : 0, codes, ld_codes,
                     reinterpret_cast<uint64_t *>(rowsum_opt)};
    return cuda_status(fqvit::launch_lis_softmax(a, as_stream(stream)), "lis_softmax");
}

// acc == nullptr with need_acc false: the output is checked by the caller (8-bit path)
static int check_attnv(const int8_t *v, int64_t ld_v, int32_t zp_v, int64_t BH, int32_t L, int32_t d,
                       const int32_t *acc, int64_t ld_acc, const char *who, bool need_acc = true)
{
    if (!v || (need_acc && !acc)) return fail(FQVIT_ERR_INVALID_ARG, "%s: NULL pointer", who);
    if (BH < 1 || L < 1 || BH > 65535) return fail(FQVIT_ERR_INVALID_ARG, "%s: bad shape BH=%lld L=%d", who, (long long)BH, L);
    if (L > 1024) return fail(FQVIT_ERR_UNSUPPORTED, "%s: L=%d (at most 1024)", who, L);
    if (d != 32 && d != 64) return fail(FQVIT_ERR_UNSUPPORTED, "%s: d=%d (32 or 64)", who, d);
    if (ld_v < d || (need_acc && ld_acc < d)) return fail(FQVIT_ERR_INVALID_ARG, "%s: stride below d", who);
    if (zp_v < -255 || zp_v > 255) return fail(FQVIT_ERR_UNSUPPORTED, "%s: |zp_v| > 255", who);
    if (need_acc && !aligned(acc, 4)) return fail(FQVIT_ERR_INVALID_ARG, "%s: misaligned acc", who);
    return FQVIT_OK;
}

int fqvit_lis_attn_v(const uint8_t *codes, int64_t ld_codes, const int8_t *v, int64_t ld_v, int32_t zp_v,
                     int64_t BH, int32_t L, int32_t d, int32_t *acc, int64_t ld_acc, int32_t *range_flag_opt,
                     void *stream)
{
    int rc = check_attnv(v, ld_v, zp_v, BH, L, d, acc, ld_acc, "lis_attn_v");
    if (rc) return rc;
    if (!codes || ld_codes < (L + 1) / 2) return fail(FQVIT_ERR_INVALID_ARG, "lis_attn_v: bad codes");
    fqvit::AttnVArgs a{codes, ld_codes, v, ld_v, zp_v, BH, L, d, acc, ld_acc, range_flag_opt};
    return cuda_status(fqvit::launch_lis_attn_v(a, as_stream(stream)), "lis_attn_v");
}

int fqvit_lis_attention(const int8_t *logits, int64_t ld_logit, float s_logit, int32_t n_shift,
                        const fqvit_relpos_bias *bias_opt, const int8_t *v, int64_t ld_v, int32_t zp_v,
                        int64_t BH, int32_t L, int32_t d, int32_t *acc, int64_t ld_acc, uint8_t *codes_opt,
                        int64_t ld_codes, void *stream)
{
    int rc = check_attnv(v, ld_v, zp_v, BH, L, d, acc, ld_acc, "lis_attention");
    if (rc) return rc;
    rc = check_lis(logits, BH * L, L, ld_logit, s_logit, n_shift, bias_opt, "lis_attention");
    if (rc) return rc;
    if (codes_opt && ld_codes < (L + 1) / 2) return fail(FQVIT_ERR_INVALID_ARG, "lis_attention: ld_codes < ceil(L/2)");
    fqvit::LisArgs la{logits, BH * L, L, ld_logit, s_logit,
                      bias_opt ? bias_opt->table : nullptr, bias_opt ? bias_opt->heads : 1,
                      bias_opt ? bias_opt->window : 0, codes_opt, ld_codes, nullptr};
    fqvit::AttnVArgs a{nullptr, 0, v, ld_v, zp_v, BH, L, d, acc, ld_acc, nullptr};
    return cuda_status(fqvit::launch_lis_attention(la, a, as_stream(stream)), "lis_attention");
}

static int check_mask(const fqvit_window_mask *mask, const fqvit_relpos_bias *bias, int64_t n_rows, int32_t L,
                      const char *who)
{
    if (!mask) return FQVIT_OK;
    if (!mask->region || mask->n_windows < 1) return fail(FQVIT_ERR_INVALID_ARG, "%s: bad window mask", who);
    if (mask->mask_value < -32768 || mask->mask_value > 0)
        return fail(FQVIT_ERR_UNSUPPORTED, "%s: mask_value outside -32768..0", who);
    const int64_t heads = bias ? bias->heads : 1;
    if (n_rows % (heads * L * (int64_t)mask->n_windows) != 0)
        return fail(FQVIT_ERR_INVALID_ARG, "%s: rows not a multiple of heads*L*n_windows", who);
    return FQVIT_OK;
}

// The attention with its output requantized to 8 bits, with or without a window mask.
static int attention_q(const int8_t *logits, int64_t ld_logit, float s_logit, int32_t n_shift,
                       const fqvit_relpos_bias *bias_opt, const fqvit_window_mask *mask, const int8_t *v,
                       int64_t ld_v, int32_t zp_v, int64_t BH, int32_t L, int32_t d, float s_v, float s_out,
                       int32_t zp_out, uint8_t *out, int64_t ld_out, void *stream, const char *who)
{
    if (!out) return fail(FQVIT_ERR_INVALID_ARG, "%s: NULL output", who);
    if (ld_out < d) return fail(FQVIT_ERR_INVALID_ARG, "%s: ld_out < d", who);
    if (!(s_v > 0.0f) || !(s_v < 3.0e38f) || !(s_out > 0.0f) || !(s_out < 3.0e38f))
        return fail(FQVIT_ERR_INVALID_ARG, "%s: s_v and s_out must be positive and finite", who);
    if (zp_out < 0 || zp_out > 255) return fail(FQVIT_ERR_INVALID_ARG, "%s: zp_out outside 0..255", who);
    // the multiplier M = (s_v / s_out) / 2^15 as N2 / 2^N1 with 8 significant bits
    const float M = ldexpf(s_v / s_out, -15);
    if (!(M > 0.0f) || !(M < 1.0e30f)) return fail(FQVIT_ERR_UNSUPPORTED, "%s: s_v / s_out out of range", who);
    int n1 = 7 - ilogbf(M);
    if (n1 > 31) n1 = 31;
    const int n2 = (int)floorf(ldexpf(M, n1));
    int rc = check_attnv(v, ld_v, zp_v, BH, L, d, nullptr, 0, who, false);
    if (rc) return rc;
    rc = check_lis(logits, BH * L, L, ld_logit, s_logit, n_shift, bias_opt, who);
    if (rc) return rc;
    rc = check_mask(mask, bias_opt, BH * L, L, who);
    if (rc) return rc;
    fqvit::LisArgs la{logits, BH * L, L, ld_logit, s_logit,
                      bias_opt ? bias_opt->table : nullptr, bias_opt ? bias_opt->heads : 1,
                      bias_opt ? bias_opt->window : 0, nullptr, 0, nullptr};
    if (mask) {
        la.region = mask->region;
        la.n_windows = mask->n_windows;
        la.mask_value = mask->mask_value;
    }
    fqvit::AttnVArgs a{nullptr, 0, v, ld_v, zp_v, BH, L, d, nullptr, 0, nullptr};
    a.out8 = out;
    a.ld_out8 = ld_out;
    a.rq_n1 = n1 < -10 ? -10 : n1;
    a.rq_n2 = n2;
    a.rq_zp = zp_out;
    return cuda_status(fqvit::launch_lis_attention(la, a, as_stream(stream)), who);
}

int fqvit_lis_attention_q(const int8_t *logits, int64_t ld_logit, float s_logit, int32_t n_shift,
                          const fqvit_relpos_bias *bias_opt, const int8_t *v, int64_t ld_v, int32_t zp_v,
                          int64_t BH, int32_t L, int32_t d, float s_v, float s_out, int32_t zp_out, uint8_t *out,
                          int64_t ld_out, void *stream)
{
    return attention_q(logits, ld_logit, s_logit, n_shift, bias_opt, nullptr, v, ld_v, zp_v, BH, L, d, s_v, s_out,
                       zp_out, out, ld_out, stream, "lis_attention_q");
}

int fqvit_lis_attention_masked_q(const int8_t *logits, int64_t ld_logit, float s_logit, int32_t n_shift,
                                 const fqvit_relpos_bias *bias_opt, const fqvit_window_mask *mask, const int8_t *v,
                                 int64_t ld_v, int32_t zp_v, int64_t BH, int32_t L, int32_t d, float s_v,
                                 float s_out, int32_t zp_out, uint8_t *out, int64_t ld_out, void *stream)
{
    return attention_q(logits, ld_logit, s_logit, n_shift, bias_opt, mask, v, ld_v, zp_v, BH, L, d, s_v, s_out,
                       zp_out, out, ld_out, stream, "lis_attention_masked_q");
}

int fqvit_lis_softmax_masked(const int8_t *logits, int64_t n_rows, int32_t L, int64_t ld_logit, float s_logit,
                             int32_t n_shift, const fqvit_relpos_bias *bias_opt, const fqvit_window_mask *mask,
                             uint8_t *codes, int64_t ld_codes, uint64_t *rowsum_opt, void *stream)
{
    int rc = check_lis(logits, n_rows, L, ld_logit, s_logit, n_shift, bias_opt, "lis_softmax_masked");
    if (rc) return rc;
    rc = check_mask(mask, bias_opt, n_rows, L, "lis_softmax_masked");
    if (rc) return rc;
    if (!codes) return fail(FQVIT_ERR_INVALID_ARG, "lis_softmax_masked: NULL codes");
    if (ld_codes < (L + 1) / 2) return fail(FQVIT_ERR_INVALID_ARG, "lis_softmax_masked: ld_codes < ceil(L/2)");
    if (rowsum_opt && !aligned(rowsum_opt, 8))
        return fail(FQVIT_ERR_INVALID_ARG, "lis_softmax_masked: misaligned rowsum");
    fqvit::LisArgs a{logits, n_rows, L, ld_logit, s_logit,
                     bias_opt ? bias_opt->table : nullptr, bias_opt ? bias_opt->heads : 1,
                     bias_opt ? bias_opt->window : 0, codes, ld_codes,
                     reinterpret_cast<uint64_t *>(rowsum_opt)};
    if (mask) {
        a.region = mask->region;
        a.n_windows = mask->n_windows;
        a.mask_value = mask->mask_value;
    }
    return cuda_status(fqvit::launch_lis_softmax(a, as_stream(stream)), "lis_softmax_masked");
}

int fqvit_lis_attention_masked(const int8_t *logits, int64_t ld_logit, float s_logit, int32_t n_shift,
                               const fqvit_relpos_bias *bias_opt, const fqvit_window_mask *mask, const int8_t *v,
                               int64_t ld_v, int32_t zp_v, int64_t BH, int32_t L, int32_t d, int32_t *acc,
                               int64_t ld_acc, uint8_t *codes_opt, int64_t ld_codes, void *stream)
{
    int rc = check_attnv(v, ld_v, zp_v, BH, L, d, acc, ld_acc, "lis_attention_masked");
    if (rc) return rc;
    rc = check_lis(logits, BH * L, L, ld_logit, s_logit, n_shift, bias_opt, "lis_attention_masked");
    if (rc) return rc;
    rc = check_mask(mask, bias_opt, BH * L, L, "lis_attention_masked");
    if (rc) return rc;
    if (codes_opt && ld_codes < (L + 1) / 2)
        return fail(FQVIT_ERR_INVALID_ARG, "lis_attention_masked: ld_codes < ceil(L/2)");
    fqvit::LisArgs la{logits, BH * L, L, ld_logit, s_logit,
                      bias_opt ? bias_opt->table : nullptr, bias_opt ? bias_opt->heads : 1,
                      bias_opt ? bias_opt->window : 0, codes_opt, ld_codes, nullptr};
    if (mask) {
        la.region = mask->region;
        la.n_windows = mask->n_windows;
        la.mask_value = mask->mask_value;
    }
    fqvit::AttnVArgs a{nullptr, 0, v, ld_v, zp_v, BH, L, d, acc, ld_acc, nullptr};
    return cuda_status(fqvit::launch_lis_attention(la, a, as_stream(stream)), "lis_attention_masked");
}

// The logits' dyadic multiplier: M = (s_q s_k) / (sqrt(d) s_logit) in fp32 in this order,
// N1 = 7 - floor(log2 M) (at most 31), N2 = floor(M 2^N1).
static int qk_multiplier(float s_q, float s_k, float s_logit, int32_t d, int *n1, int *n2, const char *who)
{
    if (!(s_q > 0.0f) || !(s_q < 3.0e38f) || !(s_k > 0.0f) || !(s_k < 3.0e38f) || !(s_logit > 0.0f) ||
        !(s_logit < 3.0e38f))
        return fail(FQVIT_ERR_INVALID_ARG, "%s: s_q, s_k and s_logit must be positive and finite", who);
    const float a = s_q * s_k;
    const float r = sqrtf((float)d);
    const float c = r * s_logit;
    const float M = a / c;
    if (!(M > 0.0f) || !(M < 1.0e30f))
        return fail(FQVIT_ERR_UNSUPPORTED, "%s: s_q s_k / (sqrt(d) s_logit) out of range", who);
    int N1 = 7 - ilogbf(M);
    if (N1 > 31) N1 = 31;
    *n1 = N1;
    *n2 = (int)floorf(ldexpf(M, N1));
    return FQVIT_OK;
}

static int check_qk(const fqvit::QkArgs &a, const char *who)
{
    if (!a.q || !a.k || !a.logits) return fail(FQVIT_ERR_INVALID_ARG, "%s: NULL pointer", who);
    if (a.BH < 1 || a.L < 1 || a.d < 1)
        return fail(FQVIT_ERR_INVALID_ARG, "%s: bad shape BH=%lld L=%d d=%d", who, (long long)a.BH, a.L, a.d);
    if (a.ld_q < a.d || a.ld_k < a.d || a.ld_logit < a.L)
        return fail(FQVIT_ERR_INVALID_ARG, "%s: a row stride is below its row", who);
    if (a.zp_q < -128 || a.zp_q > 127 || a.zp_k < -128 || a.zp_k > 127 || a.zp_l < -128 || a.zp_l > 127)
        return fail(FQVIT_ERR_INVALID_ARG, "%s: zero points outside -128..127", who);
    if (a.L > 640 || a.d > 64 || a.d % 8 != 0)
        return fail(FQVIT_ERR_UNSUPPORTED, "%s: L=%d d=%d (L <= 640, d <= 64 a multiple of 8)", who, a.L, a.d);
    if (a.ld_q % 8 || a.ld_k % 8 || !aligned(a.q, 8) || !aligned(a.k, 8))
        return fail(FQVIT_ERR_INVALID_ARG, "%s: Q and K rows must be 8-byte aligned", who);
    if (a.ld_logit % 16 || !aligned(a.logits, 16))
        return fail(FQVIT_ERR_INVALID_ARG, "%s: logits rows must be 16-byte aligned", who);
    if (!fqvit::qk_logits_supported(a)) return fail(FQVIT_ERR_UNSUPPORTED, "%s: shape not supported", who);
    return FQVIT_OK;
}

int fqvit_qk_logits(const int8_t *q, int64_t ld_q, int32_t zp_q, const int8_t *k, int64_t ld_k, int32_t zp_k,
                    int64_t BH, int32_t L, int32_t d, float s_q, float s_k, float s_logit, int32_t zp_logit,
                    int8_t *logits, int64_t ld_logit, void *stream)
{
    fqvit::QkArgs a{q, ld_q, zp_q, k, ld_k, zp_k, BH, L, d, 0, 0, zp_logit, logits, ld_logit};
    int rc = qk_multiplier(s_q, s_k, s_logit, d, &a.n1, &a.n2, "qk_logits");
    if (rc) return rc;
    rc = check_qk(a, "qk_logits");
    if (rc) return rc;
    return cuda_status(fqvit::launch_qk_logits(a, as_stream(stream)), "qk_logits");
}

// Heads per group of the chained attention, a multiple of the unit the bias and the mask index
// by.  The library's choice is every head in one group, up to 1 GiB of logits: both kernels are
// issue-bound, so the launch tails of several groups cost more than keeping a group's logits in
// L2 saves (ViT-L/384, 512 heads: 0.204 ms in one group, 0.255 ms in groups of 147 that fit
// 48 MiB).
static int64_t qk_group_heads(int64_t BH, int32_t L, int64_t unit, int64_t requested)
{
    const int64_t row = (int64_t)L * (((int64_t)L + 15) / 16 * 16);
    int64_t g = requested > 0 ? requested : ((int64_t)1 << 30) / row;
    g = g / unit * unit;
    if (g < unit) g = unit;
    return g < BH ? g : BH;
}

size_t fqvit_qk_workspace_size(int64_t BH, int32_t L, int64_t group_heads)
{
    if (BH < 1 || L < 1) return 0;
    const int64_t g = qk_group_heads(BH, L, 1, group_heads);
    return (size_t)g * L * (((size_t)L + 15) / 16 * 16);
}

int fqvit_qk_lis_attention(const int8_t *q, int64_t ld_q, int32_t zp_q, const int8_t *k, int64_t ld_k,
                           int32_t zp_k, float s_q, float s_k, float s_logit, int32_t zp_logit, int32_t n_shift,
                           const fqvit_relpos_bias *bias_opt, const fqvit_window_mask *mask_opt, const int8_t *v,
                           int64_t ld_v, int32_t zp_v, int64_t BH, int32_t L, int32_t d, int32_t *acc,
                           int64_t ld_acc, int8_t *workspace, size_t workspace_bytes, int64_t group_heads,
                           void *stream)
{
    const char *who = "qk_lis_attention";
    const int64_t ld = ((int64_t)L + 15) / 16 * 16;
    fqvit::QkArgs qa{q, ld_q, zp_q, k, ld_k, zp_k, BH, L, d, 0, 0, zp_logit, workspace, ld};
    int rc = qk_multiplier(s_q, s_k, s_logit, d, &qa.n1, &qa.n2, who);
    if (rc) return rc;
    rc = check_qk(qa, who);
    if (rc) return rc;
    rc = check_attnv(v, ld_v, zp_v, BH, L, d, acc, ld_acc, who);
    if (rc) return rc;
    // the Log-Int-Softmax checks on a stand-in for the logits (the workspace, one group's rows)
    rc = check_lis(workspace, BH * L, L, ld, s_logit, n_shift, bias_opt, who);
    if (rc) return rc;
    rc = check_mask(mask_opt, bias_opt, BH * L, L, who);
    if (rc) return rc;
    const int64_t unit = (int64_t)(bias_opt ? bias_opt->heads : 1) * (mask_opt ? mask_opt->n_windows : 1);
    int64_t g = qk_group_heads(BH, L, unit, group_heads);
    const int64_t fit = (int64_t)(workspace_bytes / (size_t)(L * ld)) / unit * unit;
    if (fit < unit)
        return fail(FQVIT_ERR_INVALID_ARG, "%s: workspace of %zu bytes holds fewer than %lld heads", who,
                    workspace_bytes, (long long)unit);
    if (g > fit) g = fit;
    cudaStream_t st = as_stream(stream);
    for (int64_t h0 = 0; h0 < BH; h0 += g) {
        const int64_t n = BH - h0 < g ? BH - h0 : g;
        fqvit::QkArgs a = qa;
        a.q = q + h0 * L * ld_q;
        a.k = k + h0 * L * ld_k;
        a.BH = n;
        cudaError_t e = fqvit::launch_qk_logits(a, st);
        if (e != cudaSuccess) return cuda_status(e, who);
        fqvit::LisArgs la{workspace, n * L, L, ld, s_logit, bias_opt ? bias_opt->table : nullptr,
                          bias_opt ? bias_opt->heads : 1, bias_opt ? bias_opt->window : 0, nullptr, 0, nullptr};
        if (mask_opt) {
            la.region = mask_opt->region;
            la.n_windows = mask_opt->n_windows;
            la.mask_value = mask_opt->mask_value;
        }
        fqvit::AttnVArgs b{nullptr, 0, v + h0 * L * ld_v, ld_v, zp_v, n, L, d, acc + h0 * L * ld_acc, ld_acc, nullptr};
        e = fqvit::launch_lis_attention(la, b, st);
        if (e != cudaSuccess) return cuda_status(e, who);
    }
    return ok();
}

int fqvit_selftest_bounded_wait(void *stream)
{
    return cuda_status(fqvit::launch_bounded_wait_probe(as_stream(stream)), "selftest_bounded_wait");
}

// ---- MinMax Linear layers -------------------------------------------------

size_t fqvit_linear_workspace_size(int64_t M, int32_t K)
{
    if (M < 1 || K < 1) return 0;
    return fqvit::linear_workspace_bytes(M, K);
}

int fqvit_linear_pack_weight(const int8_t *w, int32_t N, int32_t K, int64_t ld_w, uint16_t *w_h, void *stream)
{
    const char *who = "linear_pack_weight";
    if (!w || !w_h) return fail(FQVIT_ERR_INVALID_ARG, "%s: NULL pointer", who);
    if (N < 1 || K < 1 || ld_w < K)
        return fail(FQVIT_ERR_INVALID_ARG, "%s: bad shape N=%d K=%d ld_w=%lld", who, N, K, (long long)ld_w);
    if (K % 8) return fail(FQVIT_ERR_UNSUPPORTED, "%s: K=%d (a multiple of 8)", who, K);
    if (ld_w % 8 || !aligned(w, 8) || !aligned(w_h, 16))
        return fail(FQVIT_ERR_INVALID_ARG, "%s: w rows must be 8-byte aligned and w_h 16-byte aligned", who);
    return cuda_status(fqvit::launch_linear_pack_weight(w, N, K, ld_w, w_h, as_stream(stream)), who);
}

int fqvit_linear_q(const uint8_t *x, int64_t M, int32_t K, int64_t ld_x, int32_t zp_x, float s_x,
                   const uint16_t *w_h, int32_t N, const float *s_w, const int32_t *bias_opt, float s_y,
                   int32_t zp_y, uint8_t *y, int64_t ld_y, int32_t *acc_opt, int64_t ld_acc, void *workspace,
                   size_t workspace_bytes, void *stream)
{
    const char *who = "linear_q";
    if (!x || !w_h || !s_w || !y || !workspace) return fail(FQVIT_ERR_INVALID_ARG, "%s: NULL pointer", who);
    if (M < 1 || K < 1 || N < 1 || ld_x < K || ld_y < N || (acc_opt && ld_acc < N))
        return fail(FQVIT_ERR_INVALID_ARG, "%s: bad shape M=%lld K=%d N=%d", who, (long long)M, K, N);
    if (zp_x < 0 || zp_x > 255 || zp_y < 0 || zp_y > 255)
        return fail(FQVIT_ERR_INVALID_ARG, "%s: zero points outside 0..255", who);
    if (!(s_x > 0.0f) || !(s_x < 3.0e38f) || !(s_y > 0.0f) || !(s_y < 3.0e38f))
        return fail(FQVIT_ERR_INVALID_ARG, "%s: s_x and s_y must be positive and finite", who);
    if (K % 8 || K > 16384 || N % 16 || N > 4096 || M > ((int64_t)1 << 31) - 1)
        return fail(FQVIT_ERR_UNSUPPORTED, "%s: K=%d N=%d M=%lld (K <= 16384 a multiple of 8, N <= 4096 a "
                    "multiple of 16, M < 2^31)", who, K, N, (long long)M);
    if (ld_x % 8 || !aligned(x, 8) || !aligned(w_h, 16) || ld_y % 16 || !aligned(y, 16) || !aligned(s_w, 4) ||
        !aligned(bias_opt, 4) || (acc_opt && (ld_acc % 4 || !aligned(acc_opt, 16))) || !aligned(workspace, 16))
        return fail(FQVIT_ERR_INVALID_ARG, "%s: misaligned pointer or row stride", who);
    if (workspace_bytes < fqvit_linear_workspace_size(M, K))
        return fail(FQVIT_ERR_INVALID_ARG, "%s: workspace of %zu bytes, %zu needed", who, workspace_bytes,
                    fqvit_linear_workspace_size(M, K));
    fqvit::LinearArgs a{x,    M,        ld_x, K,    zp_x,    s_x,    w_h,    N,
                        s_w,  bias_opt, s_y,  zp_y, y,       ld_y,   acc_opt, ld_acc,
                        static_cast<uint16_t *>(workspace)};
    if (!fqvit::linear_supported(a)) return fail(FQVIT_ERR_UNSUPPORTED, "%s: N=%d needs too much shared memory", who, N);
    return cuda_status(fqvit::launch_linear(a, as_stream(stream)), who);
}

static int heads_check(const char *who, int64_t B, int32_t H, int32_t L, int32_t d, int64_t ld_src,
                       int64_t min_src, const void *src, int64_t ld_dst, int64_t min_dst)
{
    if (!src) return fail(FQVIT_ERR_INVALID_ARG, "%s: NULL pointer", who);
    if (B < 1 || H < 1 || L < 1 || d < 1 || ld_src < min_src || ld_dst < min_dst)
        return fail(FQVIT_ERR_INVALID_ARG, "%s: bad shape B=%lld H=%d L=%d d=%d", who, (long long)B, H, L, d);
    if (d % 16) return fail(FQVIT_ERR_UNSUPPORTED, "%s: d=%d (a multiple of 16)", who, d);
    if (ld_src % 16 || ld_dst % 16 || !aligned(src, 16))
        return fail(FQVIT_ERR_INVALID_ARG, "%s: misaligned pointer or row stride", who);
    return FQVIT_OK;
}

int fqvit_split_qkv(const uint8_t *qkv, int64_t B, int32_t L, int32_t H, int32_t d, int64_t ld_qkv, int8_t *q,
                    int8_t *k, int8_t *v, int64_t ld_head, void *stream)
{
    const char *who = "split_qkv";
    int rc = heads_check(who, B, H, L, d, ld_qkv, 3 * (int64_t)H * d, qkv, ld_head, d);
    if (rc) return rc;
    if (!q || !k || !v) return fail(FQVIT_ERR_INVALID_ARG, "%s: NULL pointer", who);
    if (!aligned(q, 16) || !aligned(k, 16) || !aligned(v, 16))
        return fail(FQVIT_ERR_INVALID_ARG, "%s: misaligned pointer or row stride", who);
    fqvit::HeadsArgs a{qkv, nullptr, q, k, v, nullptr, B, H, L, d, ld_qkv, ld_head};
    return cuda_status(fqvit::launch_split_qkv(a, as_stream(stream)), who);
}

int fqvit_merge_heads(const uint8_t *heads, int64_t B, int32_t L, int32_t H, int32_t d, int64_t ld_head,
                      uint8_t *out, int64_t ld_out, void *stream)
{
    const char *who = "merge_heads";
    int rc = heads_check(who, B, H, L, d, ld_head, d, heads, ld_out, (int64_t)H * d);
    if (rc) return rc;
    if (!out) return fail(FQVIT_ERR_INVALID_ARG, "%s: NULL pointer", who);
    if (!aligned(out, 16)) return fail(FQVIT_ERR_INVALID_ARG, "%s: misaligned pointer or row stride", who);
    fqvit::HeadsArgs a{nullptr, heads, nullptr, nullptr, nullptr, out, B, H, L, d, ld_head, ld_out};
    return cuda_status(fqvit::launch_merge_heads(a, as_stream(stream)), who);
}

int fqvit_block_int(const fqvit_block_desc *b, void *stream)
{
    if (!b) return fail(FQVIT_ERR_INVALID_ARG, "block_int: NULL descriptor");
    int rc = fqvit_ptf_layernorm(b->xq, b->rows, b->C, b->C, b->zp_in, b->alpha, b->gamma, b->beta, b->s_out,
                                 b->zp_out, b->yq, b->C, nullptr, nullptr, stream);
    if (rc) return rc;
    return fqvit_lis_attention(b->logits, b->ld_logit, b->s_logit, 15, b->bias, b->v, b->d, b->zp_v, b->BH,
                               b->L, b->d, b->acc, b->d, nullptr, 0, stream);
}

}  // extern "C"
