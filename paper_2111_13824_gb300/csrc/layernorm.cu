// layernorm.cu -- integer LayerNorm on PTF-quantized input (supplement,
// "Quantized Inference of LayerNorm": Eq. 11 shift, Eqs. 12-13 integer
// statistics, the A / B folding and the dyadic requantization of A).
//
// Per row: M1 = sum Xh and M2 = sum Xh^2 (Xh = (x - zp) << alpha_c), then the
// row terms r = C / sqrt(D), t = M1 / sqrt(D) with D = C M2 - M1^2 (fp32,
// correctly rounded), then each element is requantized; the row is read from
// HBM once and written once.  Two kernels: the staged kernel (C % 16 == 0,
// 16-byte aligned rows and strides: every shape of the models) and a generic
// one (any C, stride or alignment).
//
// Requantization.  With A = gs_c r and B = bs_c - gs_c t the paper's integer
// form is Y = round((sign(A) N2 Xh + Bq) / 2^N1) + zp_out with
// N1 = 7 - floor(log2|A|), N2 = floor(|A| 2^N1), Bq = rint(B 2^N1).  Two
// evaluations are used, chosen per row:
//   * fast: sign(A) N2 / 2^N1 is A with its fraction cut to 7 bits (a mask of
//     the fp32 bits), Bq / 2^N1 is B rounded to the grid 2^-N1 (adding and
//     subtracting 1.5 * 2^(23-N1)), and A_dy Xh + Bq/2^N1 + zp_out + 1/2 is
//     one fp32 FMA whose result, a multiple of 2^-N1 below 2^(24-N1), is
//     exact; its floor saturated to 0..255 is Y.  Valid when every channel of
//     the row has 0 <= N1 <= 14 and |B| 2^N1 < 2^22, which the row check
//     below guarantees from per-launch channel bounds.
//   * exact: the integer formula in int64, element by element.
#include "fqvit_internal.cuh"
#include "tc_common.cuh"

namespace fqvit {

namespace {

constexpr int kWarps = 8;  // warps (rows in flight) per block

struct LnShared {
    float gsmax;  // max |gamma/s_out| over channels
    float gsmin;  // min |gamma/s_out| over channels (0 if any is 0)
    float kappa;  // upper bound of max |beta/gamma| (fast-path check)
    int amax;     // max alpha
    int sumw;     // sum of 2^alpha over channels (staged kernel)
    int abort;    // a bounded wait of the block gave up (staged kernel)
};

__device__ __forceinline__ uint8_t ln_exact(float gs, float bs, float r, float t, int xh, int zp_out)
{
    float A = __fmul_rn(gs, r);
    float gt = __fmul_rn(gs, t);
    float B = __fsub_rn(bs, gt);
    int N1;
    long long N2;
    long long sgn = 1;
    if (A == 0.0f) {
        N1 = 0;
        N2 = 0;
    } else {
        N1 = 7 - ilogbf(A);
        if (N1 > 31) N1 = 31;
        N2 = (long long)floorf(ldexpf(fabsf(A), N1));
        if (A < 0.0f) sgn = -1;
    }
    float bsc = ldexpf(B, N1);
    float bqf = fminf(fmaxf(rintf(bsc), -4611686018427387904.0f), 4611686018427387904.0f);
    long long Bq = (long long)bqf;
    long long num = sgn * N2 * (long long)xh + Bq;
    const long long lim = 1LL << 40;
    num = num < -lim ? -lim : (num > lim ? lim : num);
    long long R;
    if (N1 > 0)
        R = (num + (1LL << (N1 - 1))) >> N1;  // arithmetic shift: floor
    else if (N1 == 0)
        R = num;
    else
        R = num * (1LL << (-N1 > 10 ? 10 : -N1));
    long long Y = R + zp_out;
    return (uint8_t)(Y < 0 ? 0 : (Y > 255 ? 255 : Y));
}

// per-launch channel constants of the generic kernel, computed by every block into shared memory
__device__ void ln_prologue(const LnArgs &a, float *gs_s, float *bs_s, uint8_t *al_s, LnShared &sh)
{
    if (threadIdx.x == 0) {
        sh.gsmax = 0.0f;
        sh.gsmin = __int_as_float(0x7F7FFFFF);
        sh.kappa = 0.0f;
        sh.amax = 0;
    }
    __syncthreads();
    float gmax = 0.0f, gmin = __int_as_float(0x7F7FFFFF), kap = 0.0f;
    int amax = 0;
    for (int c = threadIdx.x; c < a.C; c += blockDim.x) {
        float gs = __fdiv_rn(a.gamma[c], a.s_out);
        float bs = __fdiv_rn(a.beta[c], a.s_out);
        gs_s[c] = gs;
        bs_s[c] = bs;
        int al = a.alpha[c];
        al_s[c] = (uint8_t)al;
        amax = max(amax, al);
        float ag = fabsf(gs);
        gmax = fmaxf(gmax, ag);
        gmin = fminf(gmin, ag);
        if (ag > 0.0f) kap = fmaxf(kap, __fdiv_ru(fabsf(bs), ag));
    }
    // non-negative floats order like their bit patterns
    atomicMax(reinterpret_cast<int *>(&sh.gsmax), __float_as_int(gmax));
    atomicMin(reinterpret_cast<int *>(&sh.gsmin), __float_as_int(gmin));
    atomicMax(reinterpret_cast<int *>(&sh.kappa), __float_as_int(kap));
    atomicMax(&sh.amax, amax);
    __syncthreads();
}

// Row check for the fast path (all conditions conservative, see file comment):
//   N1 >= 0  <=>  |A| < 256       : gsmax r < 255
//   N1 <= 14 <=>  |A| >= 2^-7     : gsmin r >= 2^-7 (1 + 2^-10)
//   |B| 2^N1 < 2^22, with 2^N1 <= 2^8 / |A|: 2^8 (kappa + |t|) / r < 2^22
__device__ __forceinline__ bool ln_row_fast(const LnShared &sh, float r, float t)
{
    if (sh.amax > 5 || !(sh.gsmin > 0.0f) || r == 0.0f) return false;
    if (!(sh.gsmax * r < 255.0f)) return false;
    if (!(sh.gsmin * r >= 0.0078125f * 1.001f)) return false;
    return (sh.kappa + fabsf(t)) * 1.001f < 16384.0f * r;
}

// Generic path: any C, any stride or alignment; bytes, exact requantization.
__global__ void __launch_bounds__(kWarps * 32) ln_generic_kernel(LnArgs a)
{
    extern __shared__ __align__(16) unsigned char smem[];
    float *gs_s = reinterpret_cast<float *>(smem);
    float *bs_s = gs_s + a.C;
    uint8_t *al_s = reinterpret_cast<uint8_t *>(bs_s + a.C);
    __shared__ LnShared sh;
    ln_prologue(a, gs_s, bs_s, al_s, sh);
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    for (int64_t row = (int64_t)blockIdx.x * kWarps + warp; row < a.rows;
         row += (int64_t)gridDim.x * kWarps) {
        const uint8_t *src = a.xq + row * a.ld_in;
        long long m1 = 0, m2 = 0;
        for (int c = lane; c < a.C; c += 32) {
            long long xh = (long long)((int)src[c] - a.zp_in) << al_s[c];
            m1 += xh;
            m2 += xh * xh;
        }
        for (int o = 16; o > 0; o >>= 1) {
            m1 += __shfl_xor_sync(0xffffffffu, m1, o);
            m2 += __shfl_xor_sync(0xffffffffu, m2, o);
        }
        long long D = (long long)a.C * m2 - m1 * m1;
        float r = 0.0f, t = 0.0f;
        if (D != 0) {
            float sd = __fsqrt_rn(__ll2float_rn(D));
            r = __fdiv_rn((float)a.C, sd);
            t = __fdiv_rn(__ll2float_rn(m1), sd);
        }
        if (lane == 0) {
            if (a.m1) a.m1[row] = m1;
            if (a.m2) a.m2[row] = m2;
        }
        uint8_t *dst = a.yq + row * a.ld_out;
        for (int c = lane; c < a.C; c += 32) {
            int xh = ((int)src[c] - a.zp_in) << al_s[c];
            dst[c] = ln_exact(gs_s[c], bs_s[c], r, t, xh, a.zp_out);
        }
    }
}


// ---------------------------------------------------------------------------
// Staged kernel (C % 16 == 0, 16-byte aligned rows).  Each warp owns a two-stage ring in shared
// memory; the rows of its next group arrive by bulk copies (mbarrier complete_tx) while it works
// on the current group, so no registers hold data in flight.  A group is R rows per segment of S
// lanes (32 / S segments per warp).  The per-channel constants are read from shared memory once
// per 16-channel chunk and used for the group's R rows.
//
// Pass 1 (statistics, alpha <= 3 everywhere): for each byte x the value 2^23 + x is one byte
// permute (0x4B0000xx); Xh 2^-16 = fma(2^23 + x, 2^(a-16), -(2^23 + zp) 2^(a-16)) is exact, and
// fma(Xh 2^-16, Xh 2^-16, 2^-9) = 2^-9 + Xh^2 2^-32 lies in [2^-9, 2^-8), whose unit in the last
// place is 2^-32: the bit pattern minus 0x3B000000 is Xh^2 (two squares per pattern, at most
// 2 (255 * 8)^2 < 2^23).  M1 = sum x 2^a - zp sum 2^a from dp4a on the bytes and 2^a.  With
// larger alpha the squares are 64-bit integer products.
//
// Pass 2 (fast rows, conditions as ln_row_fast): with A'' = gs (r 2^16) = A 2^16 (exact
// scaling), A 2^16 cut to 8 significant bits (a mask) is N2 2^(16-N1), and the pattern of A''
// with its mantissa replaced by 0x400000 is M = 1.5 * 2^(23-N1), the constant whose unit in the
// last place is 2^-N1: (B + M) - M is B rounded to the grid 2^-N1 (ties to even, as rint).  Then
// y = fma(N2 2^(16-N1), Xh 2^-16, Bq 2^-N1 + zp_out + 1/2) is exact where it matters, and its
// floor saturated to 0..255 is one conversion.  The fp32 pairs use the packed f32x2 operations
// (two correctly rounded results per instruction, the same values as the scalar ones).  The
// product gs t is an fma with the addend +0: the code generator fuses a packed multiply and the
// packed add that uses it into one fma (the .rn modifiers notwithstanding), and B = bs - gs t,
// then rounded once instead of twice, can fall on the other side of a tie of B 2^N1.
namespace stg {

constexpr int kMaxWarps = 16;
constexpr int kStageThreads = kMaxWarps * 32;

__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c)
{
    float2 d;
    asm("{ .reg .b64 ra, rb, rc, rd;\n\t"
        "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\tmov.b64 rc, {%6, %7};\n\t"
        "fma.rn.f32x2 rd, ra, rb, rc;\n\tmov.b64 {%0, %1}, rd; }"
        : "=f"(d.x), "=f"(d.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
    return d;
}

__device__ __forceinline__ float2 mul2(float2 a, float2 b)
{
    float2 d;
    asm("{ .reg .b64 ra, rb, rd;\n\t"
        "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
        "mul.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd; }"
        : "=f"(d.x), "=f"(d.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return d;
}

__device__ __forceinline__ float2 add2(float2 a, float2 b)
{
    float2 d;
    asm("{ .reg .b64 ra, rb, rd;\n\t"
        "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
        "add.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd; }"
        : "=f"(d.x), "=f"(d.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return d;
}

// floor(y) saturated to 0 .. 255
__device__ __forceinline__ uint32_t floor_u8(float y)
{
    uint32_t r;
    asm("cvt.rmi.sat.u8.f32 %0, %1;" : "=r"(r) : "f"(y));
    return r;
}

__device__ __forceinline__ uint32_t byte_perm(uint32_t a, uint32_t b, uint32_t sel)
{
    uint32_t d;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
    return d;
}

// 2^23 + byte k of w, as an fp32 pattern
template <int K>
__device__ __forceinline__ float big_plus_byte(uint32_t w)
{
    return __uint_as_float(byte_perm(w, 0x4B000000u, 0x7540u | K));
}

__device__ __forceinline__ void expect_tx(uint64_t *b, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(tc::sa(b)), "r"(bytes) : "memory");
}

__device__ __forceinline__ void bulk_load(void *dst, const void *src, uint32_t bytes, uint64_t *bar)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(tc::sa(dst)),
        "l"(src), "r"(bytes), "r"(tc::sa(bar))
        : "memory");
}

__device__ __forceinline__ uint32_t u4_at(const uint4 &v, int q)
{
    return q == 0 ? v.x : q == 1 ? v.y : q == 2 ? v.z : v.w;
}

}  // namespace stg

// Channel constants of the staged kernel, in shared memory (float4 arrays indexed [q][chunk]:
// element k of entry (q, ch) is channel 16 ch + 4 q + k, so the lanes of a segment, reading
// consecutive chunks, read consecutive 16-byte words):
//   P = 2^(alpha-16), Q = -(2^23 + zp_in) 2^(alpha-16), G = gamma / s_out, Bs = beta / s_out,
//   W1 (bytes, [chunk]) = 2^alpha.
struct StageConsts {
    float4 *P, *Q, *G, *Bs;
    uint4 *W1;
};

__device__ __forceinline__ StageConsts stage_consts(unsigned char *smem, int nch)
{
    StageConsts k;
    k.P = reinterpret_cast<float4 *>(smem);
    k.Q = k.P + 4 * nch;
    k.G = k.Q + 4 * nch;
    k.Bs = k.G + 4 * nch;
    k.W1 = reinterpret_cast<uint4 *>(k.Bs + 4 * nch);
    return k;
}

// the parameters of channels c0 and c0 + blockDim.x (loaded before the rows' bulk copies are issued,
// so that they do not queue behind them)
struct ChLoad {
    float g0, b0, g1, b1;
    int al0, al1;
};

__device__ __forceinline__ ChLoad ch_load(const LnArgs &a, int c0)
{
    const int c1 = c0 + blockDim.x;
    const bool has0 = c0 < a.C, has1 = c1 < a.C;
    ChLoad l;
    l.g0 = has0 ? a.gamma[c0] : 1.0f;
    l.b0 = has0 ? a.beta[c0] : 0.0f;
    l.al0 = has0 ? a.alpha[c0] : 0;
    l.g1 = has1 ? a.gamma[c1] : 1.0f;
    l.b1 = has1 ? a.beta[c1] : 0.0f;
    l.al1 = has1 ? a.alpha[c1] : 0;
    return l;
}

__device__ void stage_prologue(const LnArgs &a, const StageConsts &k, LnShared &sh, const ChLoad &first)
{
    if (threadIdx.x == 0) {
        sh.gsmax = 0.0f;
        sh.gsmin = __int_as_float(0x7F7FFFFF);
        sh.kappa = 0.0f;
        sh.amax = 0;
        sh.sumw = 0;
        sh.abort = 0;
    }
    __syncthreads();
    const int nch = a.C >> 4;
    float gmax = 0.0f, gmin = __int_as_float(0x7F7FFFFF), kap = 0.0f;
    int amax = 0, sumw = 0;
    for (int c0 = threadIdx.x; c0 < a.C; c0 += 2 * blockDim.x) {
      // two channels per pass, their loads issued together
      const int c1 = c0 + blockDim.x;
      const bool has1 = c1 < a.C;
      const ChLoad l = c0 == (int)threadIdx.x ? first : ch_load(a, c0);
      const float g0 = l.g0, b0 = l.b0, g1 = l.g1, b1 = l.b1;
      const int al0 = l.al0, al1 = l.al1;
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        if (u == 1 && !has1) break;
        const int c = u ? c1 : c0;
        const float gs = __fdiv_rn(u ? g1 : g0, a.s_out);
        const float bs = __fdiv_rn(u ? b1 : b0, a.s_out);
        const int al = u ? al1 : al0;  // at most 7 (checked by the entry point)
        const int e = (c >> 4) + ((c >> 2) & 3) * nch, j = c & 3;
        const float p = __int_as_float((127 - 16 + al) << 23);
        reinterpret_cast<float *>(k.P + e)[j] = p;
        reinterpret_cast<float *>(k.Q + e)[j] = -(8388608.0f + (float)a.zp_in) * p;
        reinterpret_cast<float *>(k.G + e)[j] = gs;
        reinterpret_cast<float *>(k.Bs + e)[j] = bs;
        reinterpret_cast<uint8_t *>(k.W1)[c] = (uint8_t)(1u << al);
        amax = max(amax, al);
        sumw += 1 << al;
        const float ag = fabsf(gs);
        gmax = fmaxf(gmax, ag);
        gmin = fminf(gmin, ag);
        // |bs| / |gs| rounded to nearest, times 1 + 2^-20: above the exact ratio (a half unit in
        // the last place is 2^-24 of it), as the fast-row test needs
        if (ag > 0.0f) kap = fmaxf(kap, __fmul_ru(__fdiv_rn(fabsf(bs), ag), 1.00000095367431640625f));
      }
    }
    // warp reductions first (non-negative floats order like their bit patterns), then one shared
    // atomic per warp
    const uint32_t full = 0xffffffffu;
    const uint32_t wgmax = __reduce_max_sync(full, __float_as_uint(gmax));
    const uint32_t wgmin = __reduce_min_sync(full, __float_as_uint(gmin));
    const uint32_t wkap = __reduce_max_sync(full, __float_as_uint(kap));
    const int wamax = __reduce_max_sync(full, amax);
    const int wsum = __reduce_add_sync(full, sumw);
    if ((threadIdx.x & 31) == 0) {
        atomicMax(reinterpret_cast<unsigned int *>(&sh.gsmax), wgmax);
        atomicMin(reinterpret_cast<unsigned int *>(&sh.gsmin), wgmin);
        atomicMax(reinterpret_cast<unsigned int *>(&sh.kappa), wkap);
        atomicMax(&sh.amax, wamax);
        atomicAdd(&sh.sumw, wsum);
    }
    __syncthreads();
}

template <int S, int R>
__global__ void __launch_bounds__(stg::kStageThreads, 1) ln_stage_kernel(LnArgs a, int seg_stride)
{
    using namespace stg;
    extern __shared__ __align__(16) unsigned char smem[];
    __shared__ LnShared sh;
    __shared__ uint64_t bars[kMaxWarps][2];
    constexpr int SPW = 32 / S;  // segments per warp
    const int nch = a.C >> 4;
    const int C = a.C;
    const StageConsts K = stage_consts(smem, nch);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
    const int stage_bytes = SPW * seg_stride;
    {
        // the ring as the host laid it out must hold R rows per segment and fit the allocation
        uint32_t dyn;
        asm("mov.u32 %0, %%dynamic_smem_size;" : "=r"(dyn));
        if (seg_stride < R * C || seg_stride % 16 != 0 || nwarps > kMaxWarps ||
            (uint64_t)nch * 272 + (uint64_t)nwarps * 2 * stage_bytes > dyn) {
            if (threadIdx.x == 0) atomicCAS(&tc::g_status, 0, 2);
            return;
        }
    }
    unsigned char *ring = smem + (size_t)nch * 272 + (size_t)warp * 2 * stage_bytes;
    if (lane == 0) {
        tc::mbar_init(&bars[warp][0], 1);
        tc::mbar_init(&bars[warp][1], 1);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    pdl_release();
    pdl_wait();  // everything below reads or writes global memory

    const int seg = lane / S, sl = lane % S;
    constexpr int RPW = SPW * R;  // rows of a warp group
    const int cpl = (nch + S - 1) / S;
    const int64_t wg0 = (int64_t)blockIdx.x * nwarps + warp, wgs = (int64_t)gridDim.x * nwarps;
    // bulk copies of warp group wg into stage s (rows past the end are not copied)
    auto issue = [&](int64_t wg, int s) {
        const int64_t r0 = wg * RPW;
        if (r0 >= a.rows) return;
        const int nv = (int)(a.rows - r0 < RPW ? a.rows - r0 : RPW);
        uint64_t *bar = &bars[warp][s];
        if (lane == 0) expect_tx(bar, (uint32_t)nv * (uint32_t)C);
        __syncwarp();
        if (a.ld_in == C) {  // packed rows: a segment's rows are one contiguous copy
            for (int sg = lane; sg * R < nv; sg += 32) {
                const int cnt = nv - sg * R < R ? nv - sg * R : R;
                bulk_load(ring + s * stage_bytes + sg * seg_stride, a.xq + (r0 + (int64_t)sg * R) * C,
                          (uint32_t)(cnt * C), bar);
            }
        } else {
            for (int k = lane; k < nv; k += 32) {
                const int sg = k / R, j = k - sg * R;
                bulk_load(ring + s * stage_bytes + sg * seg_stride + j * C, a.xq + (r0 + k) * a.ld_in, (uint32_t)C,
                          bar);
            }
        }
    };

    const ChLoad first = ch_load(a, threadIdx.x);
    issue(wg0, 0);  // the first two groups arrive while the channel constants are derived
    issue(wg0 + wgs, 1);
    stage_prologue(a, K, sh, first);
    const bool fp_m2 = sh.amax <= 3;
    const int64_t zsum = (int64_t)a.zp_in * sh.sumw;
    const float2 zh = make_float2((float)a.zp_out + 0.5f, (float)a.zp_out + 0.5f);
    const float2 mag = make_float2(0.001953125f, 0.001953125f);  // 2^-9
    const float2 neg1 = make_float2(-1.0f, -1.0f);
    const float2 zero2 = make_float2(0.0f, 0.0f);  // fma(g, -t, +0) is the rounded product (+0 for a -0 product)

    int it = 0;
    for (int64_t wg = wg0; wg * RPW < a.rows; wg += wgs, ++it) {
        const int s = it & 1;
        if (it > 0) {
            tc::fence_async_smem();  // this warp's reads of stage s ^ 1 (last iteration) before the copies into it
            issue(wg + wgs, s ^ 1);
        }
        if (!tc::mbar_wait(&bars[warp][s], (uint32_t)(it >> 1) & 1u, (volatile int *)&sh.abort, false)) {
            // the copies of the other stage, if any, before the shared memory is released
            if ((wg + wgs) * RPW < a.rows)
                tc::mbar_wait(&bars[warp][s ^ 1], (uint32_t)((it + 1) >> 1) & 1u, (volatile int *)&sh.abort, false);
            return;
        }
        const unsigned char *sb = ring + s * stage_bytes + seg * seg_stride;
        const int64_t row0 = wg * RPW + (int64_t)seg * R;

        // ---- pass 1: M1 (dp4a on the raw bytes), M2
        uint32_t m1[R];
        unsigned long long m2[R];
        uint32_t m2f[R];
#pragma unroll
        for (int j = 0; j < R; ++j) m1[j] = 0, m2[j] = 0, m2f[j] = 0;
        int nck = 0;
        for (int i = 0; i < cpl; ++i) {
            const int ch = sl + S * i;
            if (ch >= nch) break;
            ++nck;
            const uint4 w1 = K.W1[ch];
            if (fp_m2) {
                float4 p[4], q[4];
#pragma unroll
                for (int qd = 0; qd < 4; ++qd) p[qd] = K.P[qd * nch + ch], q[qd] = K.Q[qd * nch + ch];
#pragma unroll
                for (int j = 0; j < R; ++j) {
                    const uint4 d = *reinterpret_cast<const uint4 *>(sb + j * C + 16 * ch);
                    m1[j] = __dp4a(d.x, w1.x, m1[j]);
                    m1[j] = __dp4a(d.y, w1.y, m1[j]);
                    m1[j] = __dp4a(d.z, w1.z, m1[j]);
                    m1[j] = __dp4a(d.w, w1.w, m1[j]);
#pragma unroll
                    for (int qd = 0; qd < 4; ++qd) {
                        const uint32_t w = u4_at(d, qd);
                        const float2 xa = fma2(make_float2(big_plus_byte<0>(w), big_plus_byte<1>(w)),
                                               make_float2(p[qd].x, p[qd].y), make_float2(q[qd].x, q[qd].y));
                        const float2 xb = fma2(make_float2(big_plus_byte<2>(w), big_plus_byte<3>(w)),
                                               make_float2(p[qd].z, p[qd].w), make_float2(q[qd].z, q[qd].w));
                        float2 v = fma2(xa, xa, mag);
                        v = fma2(xb, xb, v);
                        m2f[j] += __float_as_uint(v.x) + __float_as_uint(v.y);
                    }
                }
            } else {
#pragma unroll
                for (int j = 0; j < R; ++j) {
                    const uint4 d = *reinterpret_cast<const uint4 *>(sb + j * C + 16 * ch);
#pragma unroll
                    for (int qd = 0; qd < 4; ++qd) {
                        const uint32_t w = u4_at(d, qd), wa = u4_at(w1, qd);
                        m1[j] = __dp4a(w, wa, m1[j]);
#pragma unroll
                        for (int b = 0; b < 4; ++b) {
                            const int xh = ((int)((w >> (8 * b)) & 0xFF) - a.zp_in) * (int)((wa >> (8 * b)) & 0xFF);
                            m2[j] += (unsigned long long)((long long)xh * xh);
                        }
                    }
                }
            }
        }
        if (fp_m2) {
#pragma unroll
            for (int j = 0; j < R; ++j) m2[j] = m2f[j] - (uint32_t)nck * 8u * 0x3B000000u;
        }
        // ---- segment sums
        if (S == 32) {
#pragma unroll
            for (int j = 0; j < R; ++j) {
                m1[j] = __reduce_add_sync(0xffffffffu, m1[j]);
                const uint32_t p0 = __reduce_add_sync(0xffffffffu, (uint32_t)(m2[j] & 0xFFFF));
                const uint32_t p1 = __reduce_add_sync(0xffffffffu, (uint32_t)(m2[j] >> 16) & 0xFFFF);
                const uint32_t p2 = fp_m2 ? 0u : __reduce_add_sync(0xffffffffu, (uint32_t)(m2[j] >> 32));
                m2[j] = (unsigned long long)p0 + ((unsigned long long)p1 << 16) + ((unsigned long long)p2 << 32);
            }
        } else {
#pragma unroll
            for (int o = S / 2; o > 0; o >>= 1)
#pragma unroll
                for (int j = 0; j < R; ++j) {
                    m1[j] += __shfl_xor_sync(0xffffffffu, m1[j], o);
                    m2[j] += __shfl_xor_sync(0xffffffffu, m2[j], o);
                }
        }
        // ---- row terms: lane sl (< R) of the segment derives those of row sl, then broadcasts
        uint32_t m1o = m1[0];
        unsigned long long m2o = m2[0];
#pragma unroll
        for (int j = 1; j < R; ++j)
            if (sl == j) m1o = m1[j], m2o = m2[j];
        const long long M1 = (long long)m1o - zsum, M2 = (long long)m2o;
        float r = 0.0f, t = 0.0f;
        {
            const long long D = (long long)C * M2 - M1 * M1;
            if (D != 0) {
                const float sd = __fsqrt_rn(__ll2float_rn(D));
                r = __fdiv_rn((float)C, sd);
                t = __fdiv_rn(__ll2float_rn(M1), sd);
            }
        }
        if (sl < R && row0 + sl < a.rows) {
            if (a.m1) a.m1[row0 + sl] = M1;
            if (a.m2) a.m2[row0 + sl] = M2;
        }
        const bool fo = ln_row_fast(sh, r, t);
        float rj[R], tj[R];
        uint32_t fastm = 0;  // bit j: row j takes the fast evaluation
#pragma unroll
        for (int j = 0; j < R; ++j) {
            rj[j] = __shfl_sync(0xffffffffu, r, seg * S + j);
            tj[j] = __shfl_sync(0xffffffffu, t, seg * S + j);
            const bool fj = __shfl_sync(0xffffffffu, (int)fo, seg * S + j) != 0;
            if (fj && row0 + j < a.rows) fastm |= 1u << j;
        }

        // ---- pass 2: fast rows
        if (fastm) {
            for (int i = 0; i < cpl; ++i) {
                const int ch = sl + S * i;
                if (ch >= nch) break;
                uint4 d[R];
#pragma unroll
                for (int j = 0; j < R; ++j) d[j] = *reinterpret_cast<const uint4 *>(sb + j * C + 16 * ch);
                uint32_t o[R][4];
#pragma unroll
                for (int qd = 0; qd < 4; ++qd) {
                    const float4 p = K.P[qd * nch + ch], q = K.Q[qd * nch + ch];
                    const float4 g = K.G[qd * nch + ch], b = K.Bs[qd * nch + ch];
#pragma unroll
                    for (int j = 0; j < R; ++j) {  // every row (the other rows' bytes are not stored)
                        const uint32_t w = u4_at(d[j], qd);
                        const float2 ru = make_float2(rj[j] * 65536.0f, rj[j] * 65536.0f);
                        const float2 nt = make_float2(-tj[j], -tj[j]);
                        const float2 xa = fma2(make_float2(big_plus_byte<0>(w), big_plus_byte<1>(w)),
                                               make_float2(p.x, p.y), make_float2(q.x, q.y));
                        const float2 xb = fma2(make_float2(big_plus_byte<2>(w), big_plus_byte<3>(w)),
                                               make_float2(p.z, p.w), make_float2(q.z, q.w));
                        const float2 Aa = mul2(make_float2(g.x, g.y), ru), Ab = mul2(make_float2(g.z, g.w), ru);
                        const uint32_t a0 = __float_as_uint(Aa.x), a1 = __float_as_uint(Aa.y);
                        const uint32_t a2 = __float_as_uint(Ab.x), a3 = __float_as_uint(Ab.y);
                        const float2 na = make_float2(__uint_as_float((a0 & 0x7F800000u) | 0x80400000u),
                                                      __uint_as_float((a1 & 0x7F800000u) | 0x80400000u));
                        const float2 nb = make_float2(__uint_as_float((a2 & 0x7F800000u) | 0x80400000u),
                                                      __uint_as_float((a3 & 0x7F800000u) | 0x80400000u));
                        const float2 Ba = add2(make_float2(b.x, b.y), fma2(make_float2(g.x, g.y), nt, zero2));
                        const float2 Bb = add2(make_float2(b.z, b.w), fma2(make_float2(g.z, g.w), nt, zero2));
                        const float2 za = add2(add2(fma2(na, neg1, Ba), na), zh);
                        const float2 zb = add2(add2(fma2(nb, neg1, Bb), nb), zh);
                        const float2 ya = fma2(make_float2(__uint_as_float(a0 & 0xFFFF0000u), __uint_as_float(a1 & 0xFFFF0000u)),
                                               xa, za);
                        const float2 yb = fma2(make_float2(__uint_as_float(a2 & 0xFFFF0000u), __uint_as_float(a3 & 0xFFFF0000u)),
                                               xb, zb);
                        const uint32_t lo = byte_perm(floor_u8(ya.x), floor_u8(ya.y), 0x0040u);
                        const uint32_t hi = byte_perm(floor_u8(yb.x), floor_u8(yb.y), 0x0040u);
                        o[j][qd] = byte_perm(lo, hi, 0x5410u);
                    }
                }
#pragma unroll
                for (int j = 0; j < R; ++j)
                    if ((fastm >> j) & 1u)
                        __stcs(reinterpret_cast<uint4 *>(a.yq + (row0 + j) * a.ld_out) + ch,
                               make_uint4(o[j][0], o[j][1], o[j][2], o[j][3]));
            }
        }
        // ---- pass 2: the other rows, exact integer requantization element by element
#pragma unroll 1
        for (int j = 0; j < R; ++j) {
            if (((fastm >> j) & 1u) || row0 + j >= a.rows) continue;
            float rr = rj[0], tt = tj[0];  // row j's terms (selects: no indexed register arrays)
#pragma unroll
            for (int jj = 1; jj < R; ++jj)
                if (jj == j) rr = rj[jj], tt = tj[jj];
            for (int i = 0; i < cpl; ++i) {
                const int ch = sl + S * i;
                if (ch >= nch) break;
                const uint4 d = *reinterpret_cast<const uint4 *>(sb + j * C + 16 * ch);
                const uint4 w1 = K.W1[ch];
                uint32_t o[4];
#pragma unroll
                for (int qd = 0; qd < 4; ++qd) {
                    const float4 g = K.G[qd * nch + ch], b = K.Bs[qd * nch + ch];
                    const float gg[4] = {g.x, g.y, g.z, g.w}, bb[4] = {b.x, b.y, b.z, b.w};
                    const uint32_t w = u4_at(d, qd), wa = u4_at(w1, qd);
                    uint32_t y = 0;
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const int xh = ((int)((w >> (8 * e)) & 0xFF) - a.zp_in) * (int)((wa >> (8 * e)) & 0xFF);
                        y |= (uint32_t)ln_exact(gg[e], bb[e], rr, tt, xh, a.zp_out) << (8 * e);
                    }
                    o[qd] = y;
                }
                __stcs(reinterpret_cast<uint4 *>(a.yq + (row0 + j) * a.ld_out) + ch, make_uint4(o[0], o[1], o[2], o[3]));
            }
        }
        __syncwarp();
    }
}

}  // namespace

namespace {

// The staged kernel's shape for C = 16 nch and a segment width S, R rows per segment: the segment
// stride in the ring (R C rounded up to 128 bytes, plus 16 S bytes when segments share a
// quarter-warp, so that their 16-byte loads fall in distinct banks) and the warps per block that
// fit shared memory.  False when no warp fits.
struct StageShape {
    int seg_stride, warps, grid;
    size_t smem;
};

bool stage_shape(const LnArgs &a, int S, int R, StageShape &sh)
{
    const int nch = a.C / 16;
    const int spw = 32 / S;
    sh.seg_stride = (int)(((int64_t)R * a.C + 127) / 128 * 128) + (S < 8 ? 16 * S : 0);
    const size_t consts = (size_t)nch * 272;
    const size_t per_warp = (size_t)2 * spw * sh.seg_stride;
    const size_t budget = 232448 - 1024;  // the opt-in limit less the static arrays
    if (consts + per_warp > budget) return false;
    int warps = (int)((budget - consts) / per_warp);
    if (warps > stg::kMaxWarps) warps = stg::kMaxWarps;
    const int64_t groups = (a.rows + (int64_t)spw * R - 1) / ((int64_t)spw * R);
    const int nsm = sm_count();
    const int64_t want = (groups + nsm - 1) / nsm;  // warps per SM that cover the rows in one pass
    if (want < warps) warps = (int)(want < 1 ? 1 : want);
    sh.warps = warps;
    const int64_t blocks = (groups + warps - 1) / warps;
    sh.grid = (int)(blocks < nsm ? blocks : nsm);
    sh.smem = consts + (size_t)warps * per_warp;
    return true;
}

// segment width: the fewest idle lanes, then the widest
int stage_segment(int nch)
{
    int best = 32, bw = 1 << 30;
    for (int S = 32; S >= 1; S >>= 1) {
        const int w = S * ((nch + S - 1) / S) - nch;
        if (w < bw) bw = w, best = S;
    }
    return best;
}

// launches ln_stage_kernel<S, R> with the shape derived from the same R; cudaErrorNotSupported
// when no warp's ring fits shared memory
template <int S, int R>
cudaError_t stage_launch(const LnArgs &a, cudaStream_t st)
{
    StageShape sh;
    if (!stage_shape(a, S, R, sh)) return cudaErrorNotSupported;
    cudaError_t e = check_smem_fits((const void *)ln_stage_kernel<S, R>, sh.smem);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(ln_stage_kernel<S, R>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sh.smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(ln_stage_kernel<S, R>, dim3(sh.grid), dim3(32 * sh.warps), sh.smem, st, a, sh.seg_stride);
}

// Rows per segment: the most (4, 2, 1) whose warp groups still give at least half of the grid's
// warps one group each.  Fewer rows per segment amortize the channel constants and the row terms
// over fewer rows; too few groups leave warps idle.  Measured at full size (µs per launch, R = 4 /
// 2 / 1): DeiT-S (C = 384, 12608 rows) 9.7 / 6.7 / 9.6, ViT-B (C = 768, 12608 rows) 11.2 / 13.2 /
// 13.9, Swin-S (mean over its stages) 10.9 / 8.2 / 10.2.
template <int S>
cudaError_t stage_rows(const LnArgs &a, cudaStream_t st)
{
    const int64_t half = (int64_t)sm_count() * stg::kMaxWarps / 2;
    const int64_t spw = 32 / S;
    auto groups = [&](int64_t R) { return (a.rows + spw * R - 1) / (spw * R); };
    if (groups(4) >= half) return stage_launch<S, 4>(a, st);
    if (groups(2) >= half) return stage_launch<S, 2>(a, st);
    return stage_launch<S, 1>(a, st);
}

}  // namespace

cudaError_t read_clear_ln_status(int *status)
{
    int zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(status, tc::g_status, sizeof(int));
    if (e != cudaSuccess) return e;
    return cudaMemcpyToSymbol(tc::g_status, &zero, sizeof(int));
}

cudaError_t launch_layernorm(const LnArgs &a, cudaStream_t st)
{
    const bool staged = (a.C % 16 == 0) && (a.ld_in % 16 == 0) && (a.ld_out % 16 == 0) &&
                        ((uintptr_t)a.xq % 16 == 0) && ((uintptr_t)a.yq % 16 == 0);
    if (staged) {
        cudaError_t e;
        switch (stage_segment(a.C / 16)) {
        case 32: e = stage_rows<32>(a, st); break;
        case 16: e = stage_rows<16>(a, st); break;
        case 8: e = stage_rows<8>(a, st); break;
        case 4: e = stage_launch<4, 4>(a, st); break;
        case 2: e = stage_launch<2, 2>(a, st); break;
        default: e = stage_launch<1, 1>(a, st); break;
        }
        if (e != cudaErrorNotSupported) return e;
    }
    size_t smem = (size_t)a.C * (2 * sizeof(float) + 1);
    smem = (smem + 15) & ~(size_t)15;
    const int nsm = sm_count();
    const int64_t want = (a.rows + kWarps - 1) / kWarps;
    // Every block first derives the per-channel constants (three correctly rounded divisions per
    // channel), so the grid is the number of blocks that are resident at once: each block then
    // walks many rows.
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, ln_generic_kernel, kWarps * 32, smem) != cudaSuccess ||
        per_sm < 1)
        per_sm = 1;
    const int64_t cap = (int64_t)nsm * per_sm;
    const int blocks = (int)(want < cap ? want : cap);
    cudaFuncSetAttribute(ln_generic_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    ln_generic_kernel<<<blocks, kWarps * 32, smem, st>>>(a);
    return cudaGetLastError();
}

}  // namespace fqvit
