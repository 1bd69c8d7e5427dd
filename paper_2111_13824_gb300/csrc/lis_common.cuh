// lis_common.cuh -- device helpers shared by the Log-Int-Softmax kernels:
// the i-exp table (supplement Algorithm 1) and the division-free log2 code
// (Algorithm 2).  See lis.cu for the derivation of the code test.
#pragma once

#include <stdint.h>

#include <cmath>

namespace fqvit {
namespace lis {

// q~ in [-1335, 0]: int8 logits plus an int8 bias minus the maximum reach -510; with a window mask
// further, but e(q~) is constant below the clamp 15 q_ln2 >= -1335 (scales >= 2^-7), so indices past
// kLutSize - 1 read the last entry
constexpr int kLutSize = 1336;

struct IexpC {
    int q_ln2, q_b, q_c;
};

// e(-t) for t in [0, 287], n = 15
__device__ __forceinline__ uint32_t iexp_neg(int t, IexpC c)
{
    int q = -t;
    int lo = 15 * c.q_ln2;
    if (q < lo) q = lo;
    int z = q / c.q_ln2;
    int qp = q - z * c.q_ln2;
    int b = qp + c.q_b;
    uint32_t qL = (uint32_t)(b * b + c.q_c);
    return qL << (15 - z);
}

// Algorithm 1 constants of a scale, fp64 with one IEEE rounding per operation as in the
// oracle's definition; computed on the host once per launch (fp64 is slow on the device).
__host__ inline IexpC iexp_consts_host(float s)
{
    const double ln2 = 0.693147180559945309417232121458176568;
    const double sd = (double)s;
    IexpC c;
    c.q_ln2 = (int)floor(-ln2 / sd);
    c.q_b = (int)floor(1.353 / sd);
    c.q_c = (int)floor(0.344 / (0.3585 * (sd * sd)));
    return c;
}

__device__ __forceinline__ void build_lut(uint32_t *lut, IexpC c)
{
    for (int t = threadIdx.x; t < kLutSize; t += blockDim.x) lut[t] = iexp_neg(t, c);
}

struct RowSum {
    float hi, lo;  // 2S = hi + lo, hi = fp32(2S)
    int hibits;
};

__device__ __forceinline__ RowSum make_rowsum(unsigned long long S)
{
    unsigned long long s2 = 2ull * S;
    RowSum r;
    r.hi = __ull2float_rn(s2);
    r.lo = (float)(long long)(s2 - __float2ull_rn(r.hi));
    r.hibits = __float_as_int(r.hi);
    return r;
}

__device__ __forceinline__ uint32_t lis_code(uint32_t e, const RowSum &rs)
{
    float ef = __uint2float_rn(e);  // exact: e = q_L 2^(15-z), q_L < 2^16
    int k = (rs.hibits - __float_as_int(ef)) >> 23;
    if (k >= 16) return 15u;
    float Dk = (k == 1) ? 3.0f : __fsub_rn(__int_as_float(((k + 127) << 23) | 0x400000), 1.0f);
    float t = __fmaf_rn(ef, Dk, -rs.hi);
    return (uint32_t)(k - 1 + (t <= rs.lo ? 1 : 0));
}

// 8-bit requantization of an attention accumulator by the dyadic multiplier n2 / 2^n1 (n1 in
// [-10, 31]; the division rounds half up), plus the zero point, clipped to 0 .. 255
__device__ __forceinline__ uint32_t requant8(int acc, int n1, int n2, int zp)
{
    const long long num = (long long)n2 * acc;
    long long R = n1 > 0 ? (num + (1LL << (n1 - 1))) >> n1 : num * (1LL << -n1);
    R += zp;
    return (uint32_t)(R < 0 ? 0 : (R > 255 ? 255 : R));
}

__device__ __forceinline__ int relpos_idx(int i, int j, int w)
{
    int yi = i / w, xi = i - yi * w, yj = j / w, xj = j - yj * w;
    return (yi - yj + w - 1) * (2 * w - 1) + (xi - xj + w - 1);
}

}  // namespace lis
}  // namespace fqvit
