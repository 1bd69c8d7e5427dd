/*
 * fqvit_oracle.c -- plain, slow CPU oracle for the FQ-ViT integer inference
 * path (PTF LayerNorm, Log-Int-Softmax attention and the MinMax Linear
 * layers of the block).
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the checker the CUDA library is
 * compared against.  Only tests, the package smoke check and the bench's CPU
 * baseline leg may load it; the product path never does.  It shares no code,
 * header, table or constant with the CUDA library.
 *
 * Every function follows the paper's equations in the paper's order, with
 * plain loops, IEEE fp32/fp64 arithmetic (build with -O2 -ffp-contract=off,
 * no fast-math) and 64-bit integers.  Where the paper leaves a rounding or
 * clipping rule open, the reading taken is stated beside the code.
 *
 * Parity status: every function below is pinned by tests under tests/
 * (worked example of Find_First_One, hand-computed i-exp points, closed-form
 * softmax rows, MinMax special cases of PTF, textbook LayerNorm agreement,
 * matmul form of the BitShift product, permutation-weight and unit-multiplier
 * closed forms of the Linear layer).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#ifdef _OPENMP
#include <omp.h>
#endif

#define OR_EXPORT __attribute__((visibility("default")))

/* ------------------------------------------------------------------ */
/* helpers                                                             */
/* ------------------------------------------------------------------ */

/* floor(v / 2^n) for n >= 0, written without relying on the behaviour of
 * >> on negative signed values. */
static int64_t floor_div_pow2(int64_t v, int n)
{
    int64_t d = (int64_t)1 << n;
    int64_t q = v / d; /* truncates toward zero */
    if ((v % d) != 0 && v < 0) q -= 1;
    return q;
}

static int64_t clamp_i64(int64_t v, int64_t lo, int64_t hi)
{
    return v < lo ? lo : (v > hi ? hi : v);
}

static float clamp_f32(float v, float lo, float hi)
{
    return v < lo ? lo : (v > hi ? hi : v);
}

OR_EXPORT int or_num_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

OR_EXPORT void or_set_num_threads(int n)
{
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
#else
    (void)n;
#endif
}

/* ------------------------------------------------------------------ */
/* Sec. 3.2, Eqs. 7-10: PTF calibration                                */
/* ------------------------------------------------------------------ */

/*
 * Layer-wise scale and zero point of PTF (Eqs. 8-9) and the per-channel
 * factor search (Eq. 10), for b = 8 bits.
 *
 *  mn, mx  : exact fp32 min / max over every calibration element (Eq. 4;
 *            the range is not widened to contain 0).
 *  s0      = fp32((mx - mn) / 255)       -- the MinMax scale of Eq. 5,
 *  s       = s0 / 2^K                    -- Eq. 8 (exact power-of-two),
 *  zp      = clip(rint(-mn / s0), 0, 255) -- Eq. 9 (2^K s == s0 exactly).
 *  Reading: if mx == mn the range is degenerate and (mx - mn) is taken as 1.
 *
 *  Eq. 10 is read with the quantizer of Eq. 7 inside the norm, i.e. with
 *  its clip and zero point: for alpha in 0..K and sa = 2^alpha * s,
 *      err_c(alpha) = sum_rows ( x - clip(rint(x/sa), -zp, 255-zp) * sa )^2
 *  where x/sa, rint, the product and the difference are fp32 (round to
 *  nearest even) and the square and the sum are fp64, summed in ascending
 *  row order.  alpha_c is the smallest alpha attaining the minimum.
 */
/* exact fp32 minimum and maximum over all elements */
OR_EXPORT int or_calibrate_minmax(const float *x, int64_t rows, int32_t C, int64_t ld, float *mn_out,
                                  float *mx_out)
{
    if (!x || rows < 1 || C < 1 || ld < C) return 1;
    float mn = x[0], mx = x[0];
    for (int64_t r = 0; r < rows; ++r)
        for (int32_t c = 0; c < C; ++c) {
            float v = x[r * ld + c];
            if (v < mn) mn = v;
            if (v > mx) mx = v;
        }
    *mn_out = mn;
    *mx_out = mx;
    return 0;
}

/* Eqs. 8-9 from the range: s0 = (max - min) / 255 is 2^K s, zp from s0 */
OR_EXPORT void or_calibrate_scale(float mn, float mx, int32_t K, float *s0_out, float *s_out,
                                  int32_t *zp_out)
{
    float range = mx - mn;
    if (range == 0.0f) range = 1.0f;
    float s0 = range / 255.0f;
    float t = -mn / s0;
    *s0_out = s0;
    *s_out = ldexpf(s0, -K);
    *zp_out = (int32_t)clamp_f32(rintf(t), 0.0f, 255.0f);
}

/* Eq. 10 for every channel and factor, rows summed in ascending order */
OR_EXPORT int or_calibrate_sse(const float *x, int64_t rows, int32_t C, int64_t ld, int32_t K,
                               float mn, float mx, double *sse /* C*(K+1) */)
{
    if (!x || !sse || rows < 1 || C < 1 || ld < C || K < 0 || K > 7) return 1;
    float s0, s;
    int32_t zp;
    or_calibrate_scale(mn, mx, K, &s0, &s, &zp);
#pragma omp parallel for schedule(static)
    for (int32_t c = 0; c < C; ++c) {
        for (int32_t a = 0; a <= K; ++a) {
            float sa = ldexpf(s0, a - K); /* 2^a * s, exact */
            double err = 0.0;
            for (int64_t r = 0; r < rows; ++r) {
                float v = x[r * ld + c];
                float q = rintf(v / sa);
                q = clamp_f32(q, (float)(-zp), (float)(255 - zp));
                float dq = q * sa;
                float d = v - dq;
                err += (double)d * (double)d;
            }
            sse[(int64_t)c * (K + 1) + a] = err;
        }
    }
    return 0;
}

OR_EXPORT int or_calibrate_ptf(const float *x, int64_t rows, int32_t C, int64_t ld,
                               int32_t K, float *s_out, int32_t *zp_out,
                               uint8_t *alpha, double *sse /* C*(K+1) or NULL */)
{
    if (!x || !alpha || rows < 1 || C < 1 || ld < C || K < 0 || K > 7) return 1;
    float mn, mx, s0;
    or_calibrate_minmax(x, rows, C, ld, &mn, &mx);
    or_calibrate_scale(mn, mx, K, &s0, s_out, zp_out);
    double *err = (double *)malloc(sizeof(double) * (size_t)C * (size_t)(K + 1));
    if (!err) return 1;
    or_calibrate_sse(x, rows, C, ld, K, mn, mx, err);
    for (int32_t c = 0; c < C; ++c) {
        const double *e = err + (int64_t)c * (K + 1);
        int best_a = 0;
        for (int32_t a = 1; a <= K; ++a)
            if (e[a] < e[best_a]) best_a = a;
        alpha[c] = (uint8_t)best_a;
    }
    if (sse) memcpy(sse, err, sizeof(double) * (size_t)C * (size_t)(K + 1));
    free(err);
    return 0;
}

/*
 * Eq. 7: X_Q = clip(rint(X / (2^alpha_c s)) + zp, 0, 255), written as
 * clip(rint(X / sa), -zp, 255 - zp) + zp (identical for integer zp).
 * The division is fp32, rint rounds half to even.
 */
OR_EXPORT int or_ptf_quantize(const float *x, int64_t rows, int32_t C, int64_t ld_x,
                              float s, int32_t zp, const uint8_t *alpha, uint8_t *xq,
                              int64_t ld_q)
{
    if (!x || !xq || !alpha || rows < 1 || C < 1) return 1;
#pragma omp parallel for schedule(static)
    for (int64_t r = 0; r < rows; ++r)
        for (int32_t c = 0; c < C; ++c) {
            float sa = ldexpf(s, alpha[c]);
            float q = rintf(x[r * ld_x + c] / sa);
            q = clamp_f32(q, (float)(-zp), (float)(255 - zp));
            xq[r * ld_q + c] = (uint8_t)((int32_t)q + zp);
        }
    return 0;
}

/* ------------------------------------------------------------------ */
/* Supplement, "Quantized Inference of LayerNorm": integer LayerNorm   */
/* ------------------------------------------------------------------ */

/*
 * Per row:
 *   Xh_c = (X_Q,c - zp) << alpha_c                     (Eq. 11; a left shift
 *                                                       of a negative value is
 *                                                       read as x * 2^alpha)
 *   M1 = sum Xh, M2 = sum Xh^2                          (int64)
 *   D  = C*M2 - M1^2, so sigma ~ (s/C) sqrt(D), mu = (s/C) M1.
 * The affine terms with s_in = s cancel:
 *   A = gamma * C / (s_out sqrt(D)),  B = beta/s_out - (gamma/s_out) M1/sqrt(D).
 * Evaluation order (fixed, no fused multiply-add, every operation fp32 and
 * correctly rounded; the paper does not fix the precision of these terms):
 *   sd = sqrtf((float)D); r = C / sd; t = (float)M1 / sd
 *   gs = gamma / s_out; bs = beta / s_out
 *   A = gs*r;  B = bs - gs*t
 * Readings where the paper is silent:
 *   - epsilon is dropped by the paper; for D == 0 (constant row) X - mu is
 *     exactly zero, so r = t = 0 (the epsilon -> 0 limit: output = beta).
 *   - N1 = b-1-floor(log2|A|) = 7 - ilogb(A), capped at 31; A == 0 gives
 *     N1 = 0, N2 = 0.  N2 = floor(|A| 2^N1).
 *   - Bq = rint(B * 2^N1) in fp32, saturated to +-2^62.
 *   - num = sign(A) N2 Xh + Bq; the outer rounding of num / 2^N1 rounds
 *     halves up; N1 < 0 multiplies by 2^-N1.  num is first clamped to
 *     +-2^40 and the left shift to 10 bits; both leave the final clip
 *     unchanged because |result| >= 512 saturates either way.
 *   - Y = clip(round(num / 2^N1) + zp_out, 0, 255).
 */
OR_EXPORT int or_ptf_layernorm(const uint8_t *xq, int64_t rows, int32_t C, int64_t ld_in,
                               int32_t zp_in, const uint8_t *alpha, const float *gamma,
                               const float *beta, float s_out, int32_t zp_out, uint8_t *y,
                               int64_t ld_out, int64_t *m1_out, int64_t *m2_out)
{
    if (!xq || !y || !alpha || !gamma || !beta || rows < 1 || C < 1) return 1;
#pragma omp parallel for schedule(static)
    for (int64_t r = 0; r < rows; ++r) {
        const uint8_t *xr = xq + r * ld_in;
        int64_t M1 = 0, M2 = 0;
        for (int32_t c = 0; c < C; ++c) {
            int64_t xh = ((int64_t)xr[c] - zp_in) * ((int64_t)1 << alpha[c]);
            M1 += xh;
            M2 += xh * xh;
        }
        if (m1_out) m1_out[r] = M1;
        if (m2_out) m2_out[r] = M2;
        int64_t D = (int64_t)C * M2 - M1 * M1;
        float rf = 0.0f, tf = 0.0f;
        if (D != 0) {
            float sd = sqrtf((float)D);
            rf = (float)C / sd;
            tf = (float)M1 / sd;
        }
        for (int32_t c = 0; c < C; ++c) {
            int64_t xh = ((int64_t)xr[c] - zp_in) * ((int64_t)1 << alpha[c]);
            float gs = gamma[c] / s_out;
            float bs = beta[c] / s_out;
            float A = gs * rf;
            float gt = gs * tf;
            float B = bs - gt;
            int N1;
            int64_t N2, sgn = 1;
            if (A == 0.0f) {
                N1 = 0;
                N2 = 0;
            } else {
                N1 = 7 - ilogbf(A);
                if (N1 > 31) N1 = 31;
                N2 = (int64_t)floorf(ldexpf(fabsf(A), N1));
                if (A < 0.0f) sgn = -1;
            }
            float bsc = ldexpf(B, N1);
            float bqf = clamp_f32(rintf(bsc), -4611686018427387904.0f, 4611686018427387904.0f);
            int64_t Bq = (int64_t)bqf;
            int64_t num = sgn * N2 * xh + Bq;
            num = clamp_i64(num, -((int64_t)1 << 40), (int64_t)1 << 40);
            int64_t R;
            if (N1 > 0)
                R = floor_div_pow2(num + ((int64_t)1 << (N1 - 1)), N1);
            else if (N1 == 0)
                R = num;
            else {
                int sh = -N1;
                if (sh > 10) sh = 10;
                R = num * ((int64_t)1 << sh);
            }
            y[r * ld_out + c] = (uint8_t)clamp_i64(R + zp_out, 0, 255);
        }
    }
    return 0;
}

/* ------------------------------------------------------------------ */
/* Supplement, Algorithm 1: integer-only exponential (i-exp)           */
/* ------------------------------------------------------------------ */

/*
 * Constants for logit scale s, computed in fp64:
 *   q_ln2 = floor(-ln2 / s)   (negative; the paper's sign convention)
 *   q_b   = floor(b / s)      with b = 1.353
 *   q_c   = floor(c / (a s^2)) with a = 0.3585, c = 0.344
 * (the polynomial L(p) = a (p + b)^2 + c of Eq. 31).
 */
static const double OR_LN2 = 0.693147180559945309417232121458176568;

OR_EXPORT void or_iexp_consts(float s, int64_t *q_ln2, int64_t *q_b, int64_t *q_c)
{
    double sd = (double)s;
    *q_ln2 = (int64_t)floor(-OR_LN2 / sd);
    *q_b = (int64_t)floor(1.353 / sd);
    *q_c = (int64_t)floor(0.344 / (0.3585 * (sd * sd)));
}

/*
 * i-exp of a non-positive integer q (Algorithm 1):
 *   q   <- max(q, n * q_ln2)
 *   z   =  floor(q / q_ln2)          (both <= 0: truncating division is floor)
 *   q_p =  q - z * q_ln2             (in (q_ln2, 0])
 *   q_L =  (q_p + q_b)^2 + q_c       (the listing's (q + q_b) is read as q_p)
 *   out =  q_L << (n - z)
 * n is not defined by the paper; it is the fixed-point headroom of the
 * output and the clamp bound on z.
 */
OR_EXPORT uint64_t or_iexp(int64_t q, int32_t n, int64_t q_ln2, int64_t q_b, int64_t q_c)
{
    int64_t lo = (int64_t)n * q_ln2;
    if (q < lo) q = lo;
    int64_t z = q / q_ln2;
    int64_t qp = q - z * q_ln2;
    int64_t qL = (qp + q_b) * (qp + q_b) + q_c;
    return (uint64_t)qL << (n - z);
}

/* ------------------------------------------------------------------ */
/* Supplement, Algorithm 2: I-Log2 and Log-Int-Softmax                 */
/* ------------------------------------------------------------------ */

/*
 * I-Log2(x): M = index of the most significant one bit (Find_First_One),
 * chi = bit (M-1) of x (0 when M == 0), result M + chi.
 */
OR_EXPORT int32_t or_ilog2(uint64_t x)
{
    if (x == 0) return 0;
    int32_t M = 0;
    while ((x >> M) > 1) ++M;
    int32_t chi = (M >= 1) ? (int32_t)((x >> (M - 1)) & 1u) : 0;
    return M + chi;
}

static int32_t relpos_index(int32_t i, int32_t j, int32_t w)
{
    int32_t yi = i / w, xi = i % w, yj = j / w, xj = j % w;
    return (yi - yj + w - 1) * (2 * w - 1) + (xi - xj + w - 1);
}

/*
 * Log-Int-Softmax of each row of int8 logits (Algorithm 2, Eqs. 16-17, 33):
 *   q~     = q - max(q)
 *   e_j    = i-exp(q~_j)
 *   q_rev  = round(sum(e) / e_j)   -- halves rounded up: (2S + e)/(2e)
 *   code_j = clip(I-Log2(q_rev), 0, 15)   (Attn_Q; the LIS output is 15-code)
 * Optional relative-position bias (Swin windows, not in the paper): added
 * to the int8 logit in integer arithmetic before the max.  Row r belongs
 * to head (r / L) % heads and query index r % L; the table is
 * [heads][(2w-1)^2] indexed by (dy + w-1)(2w-1) + (dx + w-1).
 * Optional shifted-window mask (Swin, not in the paper): region ids
 * [n_windows][L]; row r belongs to window (r / (L heads)) % n_windows, and
 * key j of query i gets mask_value (logit units) added when their region ids
 * in that window differ.  The i-exp clamp (Algorithm 1) bounds what a large
 * negative mask does.
 * codes: one byte per code, row stride ld_codes.  rowsum: S per row.
 */
OR_EXPORT int or_lis_softmax_masked(const int8_t *logits, int64_t n_rows, int32_t L, int64_t ld,
                                    float s, int32_t n, const int8_t *bias, int32_t heads,
                                    int32_t window, const uint8_t *region, int32_t n_windows,
                                    int32_t mask_value, uint8_t *codes, int64_t ld_codes,
                                    uint64_t *rowsum)
{
    if (!logits || !codes || n_rows < 1 || L < 1 || heads < 1) return 1;
    if (region && n_windows < 1) return 1;
    int64_t q_ln2, q_b, q_c;
    or_iexp_consts(s, &q_ln2, &q_b, &q_c);
    int32_t nb = (2 * window - 1) * (2 * window - 1);
#pragma omp parallel
    {
        int32_t *qv = (int32_t *)malloc(sizeof(int32_t) * (size_t)L);
        uint64_t *ev = (uint64_t *)malloc(sizeof(uint64_t) * (size_t)L);
#pragma omp for schedule(static)
        for (int64_t r = 0; r < n_rows; ++r) {
            const int8_t *row = logits + r * ld;
            int32_t i = (int32_t)(r % L);
            int32_t h = bias ? (int32_t)((r / L) % heads) : 0;
            const uint8_t *reg = region ? region + ((r / ((int64_t)L * heads)) % n_windows) * L : NULL;
            int32_t m = -2147483647;
            for (int32_t j = 0; j < L; ++j) {
                int32_t q = row[j];
                if (bias) q += bias[(int64_t)h * nb + relpos_index(i, j, window)];
                if (reg && reg[i] != reg[j]) q += mask_value;
                qv[j] = q;
                if (q > m) m = q;
            }
            uint64_t S = 0;
            for (int32_t j = 0; j < L; ++j) {
                ev[j] = or_iexp((int64_t)qv[j] - m, n, q_ln2, q_b, q_c);
                S += ev[j];
            }
            if (rowsum) rowsum[r] = S;
            for (int32_t j = 0; j < L; ++j) {
                uint64_t qrev = (2 * S + ev[j]) / (2 * ev[j]);
                int32_t code = or_ilog2(qrev);
                if (code > 15) code = 15;
                codes[r * ld_codes + j] = (uint8_t)code;
            }
        }
        free(qv);
        free(ev);
    }
    return 0;
}

OR_EXPORT int or_lis_softmax(const int8_t *logits, int64_t n_rows, int32_t L, int64_t ld,
                             float s, int32_t n, const int8_t *bias, int32_t heads,
                             int32_t window, uint8_t *codes, int64_t ld_codes,
                             uint64_t *rowsum)
{
    return or_lis_softmax_masked(logits, n_rows, L, ld, s, n, bias, heads, window, NULL, 1, 0, codes, ld_codes,
                                 rowsum);
}

/* ------------------------------------------------------------------ */
/* 8-bit requantization of the attention output                        */
/* ------------------------------------------------------------------ */

/*
 * The attention output acc (real value acc * s_v / 2^15, Eq. 15) quantized to
 * the next layer's 8-bit activation (Eq. 3: scale s_out, zero point zp_out),
 * with the dyadic multiplier of the supplement's LayerNorm output stage (the
 * requantization with A = M, B = 0):
 *   M  = (s_v / s_out) / 2^15        (one fp32 division, then an exact scaling)
 *   N1 = 7 - floor(log2 M)  (at most 31),   N2 = floor(M 2^N1)
 *   y  = clip(floor((N2 acc + 2^(N1-1)) / 2^N1) + zp_out, 0, 255)   for N1 > 0
 *   y  = clip(N2 acc 2^min(-N1, 10) + zp_out, 0, 255)                for N1 <= 0
 * The readings are those of or_ptf_layernorm: the division by 2^N1 rounds half
 * up (floor of the value plus one half), the result is clipped to 8 bits.
 * acc [rows][ld_acc] (d values per row), y [rows][ld_y].
 */
OR_EXPORT int or_attn_requant(const int32_t *acc, int64_t rows, int32_t d, int64_t ld_acc, float s_v, float s_out,
                              int32_t zp_out, uint8_t *y, int64_t ld_y)
{
    if (!acc || !y || rows < 1 || d < 1 || !(s_v > 0.0f) || !(s_out > 0.0f)) return 1;
    const float M = ldexpf(s_v / s_out, -15);
    if (!(M > 0.0f)) return 1;
    int N1 = 7 - ilogbf(M);
    if (N1 > 31) N1 = 31;
    const int64_t N2 = (int64_t)floorf(ldexpf(M, N1));
    for (int64_t r = 0; r < rows; ++r) {
        for (int32_t t = 0; t < d; ++t) {
            const int64_t num = N2 * (int64_t)acc[r * ld_acc + t];
            int64_t R;
            if (N1 > 0)
                R = floor_div_pow2(num + ((int64_t)1 << (N1 - 1)), N1);
            else if (N1 == 0)
                R = num;
            else {
                int sh = -N1;
                if (sh > 10) sh = 10;
                R = num * ((int64_t)1 << sh);
            }
            y[r * ld_y + t] = (uint8_t)clamp_i64(R + zp_out, 0, 255);
        }
    }
    return 0;
}

/* ------------------------------------------------------------------ */
/* The MatMul Q K^T and its 8-bit output quantizer (the logits)        */
/* ------------------------------------------------------------------ */

/*
 * Sec. 3 quantizes the MatMul modules with uniform MinMax, and Sec. 4.1 takes
 * activations asymmetric (a zero point): Q and K arrive as 8-bit codes with
 * zero points, and the product's output -- the logits fed to Log-Int-Softmax --
 * is quantized to 8 bits with the logit scale s_logit and zero point zp_l.
 *   P[bh][i][j] = sum_t (q[bh][i][t] - zp_q) (k[bh][j][t] - zp_k)     (int64)
 * P s_q s_k / sqrt(d) is the real logit.  Integer-only, the rescaling is the
 * dyadic multiplier of the supplement's LayerNorm output stage:
 *   M  = (s_q s_k) / (sqrt(d) s_logit)  in fp32, in this order:
 *        a = s_q s_k,  r = sqrtf(d),  c = r s_logit,  M = a / c
 *   N1 = 7 - floor(log2 M)  (at most 31),   N2 = floor(M 2^N1)
 *   logit = clip(floor((N2 P + 2^(N1-1)) / 2^N1) + zp_l, -128, 127)   N1 > 0
 *   logit = clip(N2 P 2^min(-N1, 10) + zp_l, -128, 127)                N1 <= 0
 * Logits are signed: the 8-bit code minus 128, zp_l likewise (the form the
 * Log-Int-Softmax functions take; the softmax only sees differences).
 * q [BH][L][ld_q], k [BH][L][ld_k] (d values per row), logits [BH*L][ld_logit]
 * (row i of head bh at bh*L + i, key j in byte j).
 */
OR_EXPORT int or_qk_logits(const int8_t *q, int64_t ld_q, int32_t zp_q, const int8_t *k, int64_t ld_k,
                           int32_t zp_k, int64_t BH, int32_t L, int32_t d, float s_q, float s_k,
                           float s_logit, int32_t zp_l, int8_t *logits, int64_t ld_logit)
{
    if (!q || !k || !logits || BH < 1 || L < 1 || d < 1 || ld_q < d || ld_k < d || ld_logit < L) return 1;
    if (!(s_q > 0.0f) || !(s_k > 0.0f) || !(s_logit > 0.0f)) return 1;
    const float a = s_q * s_k;
    const float r = sqrtf((float)d);
    const float c = r * s_logit;
    const float M = a / c;
    if (!(M > 0.0f) || !(M < INFINITY)) return 1;
    int N1 = 7 - ilogbf(M);
    if (N1 > 31) N1 = 31;
    const int64_t N2 = (int64_t)floorf(ldexpf(M, N1));
#ifdef _OPENMP
#pragma omp parallel for schedule(static)
#endif
    for (int64_t bh = 0; bh < BH; ++bh) {
        for (int32_t i = 0; i < L; ++i) {
            const int8_t *qi = q + (bh * L + i) * ld_q;
            for (int32_t j = 0; j < L; ++j) {
                const int8_t *kj = k + (bh * L + j) * ld_k;
                int64_t P = 0;
                for (int32_t t = 0; t < d; ++t) P += ((int64_t)qi[t] - zp_q) * ((int64_t)kj[t] - zp_k);
                const int64_t num = N2 * P;
                int64_t R;
                if (N1 > 0)
                    R = floor_div_pow2(num + ((int64_t)1 << (N1 - 1)), N1);
                else if (N1 == 0)
                    R = num;
                else {
                    int sh = -N1;
                    if (sh > 10) sh = 10;
                    R = num * ((int64_t)1 << sh);
                }
                logits[(bh * L + i) * ld_logit + j] = (int8_t)clamp_i64(R + zp_l, -128, 127);
            }
        }
    }
    return 0;
}

/* ------------------------------------------------------------------ */
/* Eq. 15 and the supplement's Attn.V: BitShift attention times values */
/* ------------------------------------------------------------------ */

/*
 * acc[bh][i][t] = sum_j (V[bh][j][t] - zp_v) << (15 - code[bh][i][j])
 * accumulated in int64 (a left shift of a negative value is read as a
 * multiplication by 2^(15-code)); the real value is acc * s_V / 2^15.
 * V is [BH][L][ld_v], codes [BH*L][ld_codes] (one byte per code),
 * acc [BH][L][ld_acc].  Returns 3 if any sum does not fit int32 (the
 * stored value is then saturated).
 */
OR_EXPORT int or_lis_attn_v(const uint8_t *codes, int64_t ld_codes, const int8_t *v,
                            int64_t ld_v, int32_t zp_v, int64_t BH, int32_t L, int32_t d,
                            int32_t *acc, int64_t ld_acc)
{
    if (!codes || !v || !acc || BH < 1 || L < 1 || d < 1) return 1;
    int overflow = 0;
#pragma omp parallel reduction(| : overflow)
    {
        int64_t *a = (int64_t *)malloc(sizeof(int64_t) * (size_t)d);
#pragma omp for schedule(static)
        for (int64_t bi = 0; bi < BH * (int64_t)L; ++bi) {
            int64_t bh = bi / L;
            const uint8_t *crow = codes + bi * ld_codes;
            const int8_t *vh = v + bh * (int64_t)L * ld_v;
            for (int32_t t = 0; t < d; ++t) a[t] = 0;
            for (int32_t j = 0; j < L; ++j) {
                int64_t w = (int64_t)1 << (15 - crow[j]);
                for (int32_t t = 0; t < d; ++t)
                    a[t] += ((int64_t)vh[(int64_t)j * ld_v + t] - zp_v) * w;
            }
            for (int32_t t = 0; t < d; ++t) {
                int64_t val = a[t];
                if (val > INT32_MAX || val < INT32_MIN) {
                    overflow = 1;
                    val = clamp_i64(val, INT32_MIN, INT32_MAX);
                }
                acc[bi * ld_acc + t] = (int32_t)val;
            }
        }
        free(a);
    }
    return overflow ? 3 : 0;
}

/* ------------------------------------------------------------------ */
/* MinMax Linear layer (Sec. 3, Sec. 4.1)                              */
/* ------------------------------------------------------------------ */

/*
 * A Linear layer of the fully quantized block.  Sec. 3 quantizes Linear
 * layers with uniform MinMax; Sec. 4.1 makes the weights symmetric and
 * channel-wise and the activations asymmetric and layer-wise:
 *   x  uint8 [M][ld_x]   real value (x - zp_x) s_x
 *   w  int8  [N][ld_w]   real value  w s_w[n]       (output channel n)
 *   b  int32 [N]         real value  b s_x s_w[n]   (NULL: no bias)
 * The integer product, in int64:
 *   acc[m][n] = sum_k (x[m][k] - zp_x) w[n][k] + b[n]
 * and the output quantizer, uniform MinMax with scale s_y and zero point
 * zp_y, applied with the dyadic multiplier of the supplement's LayerNorm
 * output stage, one per output channel:
 *   M_n = (s_x s_w[n]) / s_y   in fp32, in this order
 *   N1  = 7 - floor(log2 M_n)  (at most 31),   N2 = floor(M_n 2^N1)
 *   y   = clip(floor((N2 acc + 2^(N1-1)) / 2^N1) + zp_y, 0, 255)   N1 > 0
 *   y   = clip(N2 acc 2^min(-N1, 10) + zp_y, 0, 255)                N1 <= 0
 * y [M][ld_y]; acc_opt [M][ld_acc] (may be NULL) receives acc.
 * Returns 1 for invalid arguments (a scale that is not positive and finite,
 * or an M_n outside (0, 1e30)), 3 if an acc does not fit int32 (its stored
 * value is then saturated).
 */
OR_EXPORT int or_linear_q(const uint8_t *x, int64_t M, int32_t K, int64_t ld_x, int32_t zp_x, float s_x,
                          const int8_t *w, int32_t N, int64_t ld_w, const float *s_w, const int32_t *bias,
                          float s_y, int32_t zp_y, uint8_t *y, int64_t ld_y, int32_t *acc_opt, int64_t ld_acc)
{
    if (!x || !w || !s_w || !y || M < 1 || K < 1 || N < 1 || ld_x < K || ld_w < K || ld_y < N) return 1;
    if (acc_opt && ld_acc < N) return 1;
    if (zp_x < 0 || zp_x > 255 || zp_y < 0 || zp_y > 255) return 1;
    if (!(s_x > 0.0f) || !(s_x < INFINITY) || !(s_y > 0.0f) || !(s_y < INFINITY)) return 1;
    int32_t *n1 = (int32_t *)malloc(sizeof(int32_t) * (size_t)N);
    int64_t *n2 = (int64_t *)malloc(sizeof(int64_t) * (size_t)N);
    int bad = 0;
    for (int32_t n = 0; n < N; ++n) {
        const float a = s_x * s_w[n];
        const float Mn = a / s_y;
        if (!(s_w[n] > 0.0f) || !(Mn > 0.0f) || !(Mn < 1.0e30f)) {
            bad = 1;
            n1[n] = 0;
            n2[n] = 0;
            continue;
        }
        int e = 7 - ilogbf(Mn);
        if (e > 31) e = 31;
        n1[n] = e;
        n2[n] = (int64_t)floorf(ldexpf(Mn, e));
    }
    if (bad) {
        free(n1);
        free(n2);
        return 1;
    }
    int overflow = 0;
#ifdef _OPENMP
#pragma omp parallel for schedule(static) reduction(| : overflow)
#endif
    for (int64_t m = 0; m < M; ++m) {
        const uint8_t *xm = x + m * ld_x;
        for (int32_t n = 0; n < N; ++n) {
            const int8_t *wn = w + (int64_t)n * ld_w;
            int64_t s = 0;
            for (int32_t k = 0; k < K; ++k) s += ((int64_t)xm[k] - zp_x) * (int64_t)wn[k];
            if (bias) s += bias[n];
            if (s > INT32_MAX || s < INT32_MIN) {
                overflow = 1;
                s = clamp_i64(s, INT32_MIN, INT32_MAX);
            }
            if (acc_opt) acc_opt[m * ld_acc + n] = (int32_t)s;
            const int64_t num = n2[n] * s;
            int64_t R;
            if (n1[n] > 0)
                R = floor_div_pow2(num + ((int64_t)1 << (n1[n] - 1)), n1[n]);
            else if (n1[n] == 0)
                R = num;
            else {
                int sh = -n1[n];
                if (sh > 10) sh = 10;
                R = num * ((int64_t)1 << sh);
            }
            y[m * ld_y + n] = (uint8_t)clamp_i64(R + zp_y, 0, 255);
        }
    }
    free(n1);
    free(n2);
    return overflow ? 3 : 0;
}
