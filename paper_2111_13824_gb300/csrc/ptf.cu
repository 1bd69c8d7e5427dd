// ptf.cu -- Power-of-Two Factor calibration (Sec. 3.2, Eqs. 8-10) and the
// PTF quantizer (Eq. 7) on sm_103a.
//
// Calibration runs in four launches on the caller's stream (a calibration
// batch split by rows over several ranks runs the first and third per rank,
// with the range and the sums exchanged in between; see
// fqvit_calibrate_minmax / _sse_partial / _combine):
//   1. per-block min / max of the calibration batch (exact fp32 compares),
//   2. one block folds the partials into s, zp (Eqs. 8-9),
//   3. one thread per (channel, factor) sums the squared quantization error
//      of Eq. 10 over the rows, in ascending row order, in fp64 -- the order
//      fixes the rounding of the sum, so it is sequential per thread and the
//      parallelism comes from the C*(K+1) independent sums,
//   4. one thread per channel takes the smallest factor with the least error.
#include "fqvit_internal.cuh"

#include <cfloat>

namespace fqvit {

namespace {

constexpr int kMaxPartials = 1024;  // blocks of the min/max pass
constexpr int kWsHeader = 64;       // s0, zp, flags

__device__ __forceinline__ float pow2f(int e)  // 2^e for -126 <= e <= 127, exact
{
    return __int_as_float((e + 127) << 23);
}

__global__ void minmax_partial_kernel(const float *__restrict__ x, int64_t rows, int C,
                                      int64_t ld, float2 *__restrict__ part)
{
    float mn = FLT_MAX, mx = -FLT_MAX;
    for (int64_t r = blockIdx.x; r < rows; r += gridDim.x) {
        const float *xr = x + r * ld;
        for (int c = threadIdx.x; c < C; c += blockDim.x) {
            float v = __ldg(xr + c);
            mn = fminf(mn, v);
            mx = fmaxf(mx, v);
        }
    }
    __shared__ float smn[32], smx[32];
    for (int o = 16; o > 0; o >>= 1) {
        mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, o));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    }
    int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    if (l == 0) {
        smn[w] = mn;
        smx[w] = mx;
    }
    __syncthreads();
    if (w == 0) {
        int nw = blockDim.x >> 5;
        mn = l < nw ? smn[l] : FLT_MAX;
        mx = l < nw ? smx[l] : -FLT_MAX;
        for (int o = 16; o > 0; o >>= 1) {
            mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, o));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        }
        if (l == 0) part[blockIdx.x] = make_float2(mn, mx);
    }
}

// Eqs. 8-9: s0 = (max - min) / 255 is the MinMax scale 2^K s; zp from it.
__global__ void calib_finalize_kernel(const float2 *__restrict__ part, int nparts, int K,
                                      float *__restrict__ s_out, int32_t *__restrict__ zp_out,
                                      float *__restrict__ ws_s0, int32_t *__restrict__ ws_zp)
{
    float mn = FLT_MAX, mx = -FLT_MAX;
    for (int i = threadIdx.x; i < nparts; i += 32) {
        float2 p = part[i];
        mn = fminf(mn, p.x);
        mx = fmaxf(mx, p.y);
    }
    for (int o = 16; o > 0; o >>= 1) {
        mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, o));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    }
    if (threadIdx.x == 0) {
        float s0, s;
        int32_t zp;
        calib_scale(mn, mx, K, s0, s, zp);
        *s_out = s;
        *zp_out = zp;
        *ws_s0 = s0;
        *ws_zp = zp;
    }
}

// Folds the min / max partials of one shard into mnmx[2].
__global__ void minmax_final_kernel(const float2 *__restrict__ part, int nparts, float *__restrict__ mnmx)
{
    float mn = FLT_MAX, mx = -FLT_MAX;
    for (int i = threadIdx.x; i < nparts; i += 32) {
        float2 p = part[i];
        mn = fminf(mn, p.x);
        mx = fmaxf(mx, p.y);
    }
    for (int o = 16; o > 0; o >>= 1) {
        mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, o));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    }
    if (threadIdx.x == 0) {
        mnmx[0] = mn;
        mnmx[1] = mx;
    }
}

// s0 and zp of a given (global) range, for the Eq. 10 sums of one shard.
__global__ void calib_setscale_kernel(const float *__restrict__ mnmx, int K, float *__restrict__ ws_s0,
                                      int32_t *__restrict__ ws_zp)
{
    float s0, s;
    int32_t zp;
    calib_scale(mnmx[0], mnmx[1], K, s0, s, zp);
    *ws_s0 = s0;
    *ws_zp = zp;
}

// Eq. 10, one thread per (channel c, factor a): sum over rows of
// (x - clip(rint(x / (2^a s)), -zp, 255-zp) * 2^a s)^2 in fp64, ascending rows.
// x / (2^a s) is computed as (x / s0) * 2^(K-a): scaling a correctly rounded
// quotient by a power of two is the correctly rounded quotient by the scaled
// divisor (values small enough to lose bits round to 0 either way).
__global__ void calib_sse_kernel(const float *__restrict__ x, int64_t rows, int C, int64_t ld,
                                 int K, const float *__restrict__ ws_s0,
                                 const int32_t *__restrict__ ws_zp, double *__restrict__ sse)
{
    int c = blockIdx.x * blockDim.x + threadIdx.x;
    int a = blockIdx.y;
    if (c >= C) return;
    const float s0 = *ws_s0;
    const int zp = *ws_zp;
    const float up = pow2f(K - a);       // 1 / (2^(a-K))
    const float sa = __fmul_rn(s0, pow2f(a - K));  // 2^a s, exact
    const float lo = (float)(-zp), hi = (float)(255 - zp);
    double acc = 0.0;
    const float *xc = x + c;
    int64_t r = 0;
    for (; r + 4 <= rows; r += 4) {
        float v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) v[u] = __ldg(xc + (r + u) * ld);
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            float q = rintf(__fmul_rn(__fdiv_rn(v[u], s0), up));
            q = fminf(fmaxf(q, lo), hi);
            float d = __fsub_rn(v[u], __fmul_rn(q, sa));
            double dd = (double)d;
            acc = __dadd_rn(acc, __dmul_rn(dd, dd));
        }
    }
    for (; r < rows; ++r) {
        float v = __ldg(xc + r * ld);
        float q = rintf(__fmul_rn(__fdiv_rn(v, s0), up));
        q = fminf(fmaxf(q, lo), hi);
        float d = __fsub_rn(v, __fmul_rn(q, sa));
        double dd = (double)d;
        acc = __dadd_rn(acc, __dmul_rn(dd, dd));
    }
    sse[(int64_t)c * (K + 1) + a] = acc;
}

__global__ void calib_argmin_kernel(const double *__restrict__ sse, int C, int K,
                                    uint8_t *__restrict__ alpha)
{
    int c = blockIdx.x * blockDim.x + threadIdx.x;
    if (c >= C) return;
    const double *e = sse + (int64_t)c * (K + 1);
    double best = e[0];
    int ba = 0;
    for (int a = 1; a <= K; ++a)
        if (e[a] < best) {
            best = e[a];
            ba = a;
        }
    alpha[c] = (uint8_t)ba;
}

// Eq. 7.  x / (2^alpha s) = (x / s) * 2^-alpha by the same scaling argument.
__global__ void quantize_kernel(const float *__restrict__ x, int64_t rows, int C, int64_t ld_x,
                                float s, int zp, const uint8_t *__restrict__ alpha,
                                uint8_t *__restrict__ xq, int64_t ld_q)
{
    extern __shared__ float qsh[];  // 2^-alpha_c per channel
    for (int c = threadIdx.x; c < C; c += blockDim.x) qsh[c] = pow2f(-(int)alpha[c]);
    __syncthreads();
    const float lo = (float)(-zp), hi = (float)(255 - zp);
    for (int64_t r = blockIdx.x; r < rows; r += gridDim.x) {
        const float *xr = x + r * ld_x;
        uint8_t *qr = xq + r * ld_q;
        for (int c = threadIdx.x; c < C; c += blockDim.x) {
            float q = rintf(__fmul_rn(__fdiv_rn(__ldg(xr + c), s), qsh[c]));
            q = fminf(fmaxf(q, lo), hi);
            qr[c] = (uint8_t)((int)q + zp);
        }
    }
}

// blocks of the min / max pass
int minmax_blocks(int64_t rows)
{
    int nparts = (int)(rows < kMaxPartials ? rows : kMaxPartials);
    int nsm = sm_count();
    if (nparts > 4 * nsm) nparts = 4 * nsm;
    return nparts < 1 ? 1 : nparts;
}

}  // namespace

size_t calibrate_workspace_bytes(int64_t rows, int C, int K, bool sums)
{
    (void)rows;
    return (size_t)kWsHeader + sizeof(float2) * kMaxPartials + (sums ? sizeof(double) * (size_t)C * (K + 1) : 0);
}

cudaError_t launch_calibrate(const float *x, int64_t rows, int C, int64_t ld_x, int K, float *s,
                             int32_t *zp, uint8_t *alpha, double *sse, void *ws, cudaStream_t st)
{
    char *w = static_cast<char *>(ws);
    float *ws_s0 = reinterpret_cast<float *>(w);
    int32_t *ws_zp = reinterpret_cast<int32_t *>(w + 4);
    float2 *part = reinterpret_cast<float2 *>(w + kWsHeader);
    double *sse_buf = sse ? sse : reinterpret_cast<double *>(w + kWsHeader + sizeof(float2) * kMaxPartials);

    const int nparts = minmax_blocks(rows);
    minmax_partial_kernel<<<nparts, 256, 0, st>>>(x, rows, C, ld_x, part);
    calib_finalize_kernel<<<1, 32, 0, st>>>(part, nparts, K, s, zp, ws_s0, ws_zp);
    dim3 g((C + 31) / 32, K + 1);
    calib_sse_kernel<<<g, 32, 0, st>>>(x, rows, C, ld_x, K, ws_s0, ws_zp, sse_buf);
    calib_argmin_kernel<<<(C + 127) / 128, 128, 0, st>>>(sse_buf, C, K, alpha);
    return cudaGetLastError();
}

cudaError_t launch_calibrate_minmax(const float *x, int64_t rows, int C, int64_t ld_x, float *mnmx, void *ws,
                                    cudaStream_t st)
{
    float2 *part = reinterpret_cast<float2 *>(static_cast<char *>(ws) + kWsHeader);
    const int nparts = minmax_blocks(rows);
    minmax_partial_kernel<<<nparts, 256, 0, st>>>(x, rows, C, ld_x, part);
    minmax_final_kernel<<<1, 32, 0, st>>>(part, nparts, mnmx);
    return cudaGetLastError();
}

cudaError_t launch_calibrate_sse_partial(const float *x, int64_t rows, int C, int64_t ld_x, int K,
                                         const float *mnmx, double *sse, void *ws, cudaStream_t st)
{
    char *w = static_cast<char *>(ws);
    float *ws_s0 = reinterpret_cast<float *>(w);
    int32_t *ws_zp = reinterpret_cast<int32_t *>(w + 4);
    calib_setscale_kernel<<<1, 1, 0, st>>>(mnmx, K, ws_s0, ws_zp);
    dim3 g((C + 31) / 32, K + 1);
    calib_sse_kernel<<<g, 32, 0, st>>>(x, rows, C, ld_x, K, ws_s0, ws_zp, sse);
    return cudaGetLastError();
}

cudaError_t launch_quantize(const float *x, int64_t rows, int C, int64_t ld_x, float s, int32_t zp,
                            const uint8_t *alpha, uint8_t *xq, int64_t ld_q, cudaStream_t st)
{
    int nsm = sm_count();
    int64_t blocks = rows < (int64_t)nsm * 8 ? rows : (int64_t)nsm * 8;
    int threads = C >= 256 ? 256 : ((C + 31) / 32) * 32;
    quantize_kernel<<<(int)blocks, threads, sizeof(float) * C, st>>>(x, rows, C, ld_x, s, zp, alpha,
                                                                      xq, ld_q);
    return cudaGetLastError();
}

}  // namespace fqvit
