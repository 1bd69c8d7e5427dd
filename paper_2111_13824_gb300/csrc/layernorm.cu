// layernorm.cu -- integer LayerNorm on PTF-quantized input (supplement,
// "Quantized Inference of LayerNorm": Eq. 11 shift, Eqs. 12-13 integer
// statistics, the A / B folding and the dyadic requantization of A).
//
// One warp per token row.  Each lane holds CPL 16-byte chunks of the row in
// registers, so the row is read from HBM once: pass 1 forms M1 = sum Xh and
// M2 = sum Xh^2 (Xh = (x - zp) << alpha_c), a warp reduction gives the row
// terms r = C / sqrt(D), t = M1 / sqrt(D) (fp32, correctly rounded), pass 2
// requantizes each element and the row is written once.
//
// Requantization.  With A = gs_c r and B = bs_c - gs_c t the paper's integer
// form is Y = round((sign(A) N2 Xh + Bq) / 2^N1) + zp_out with
// N1 = 7 - floor(log2|A|), N2 = floor(|A| 2^N1), Bq = rint(B 2^N1).  Two
// evaluations are used, chosen per row (warp-uniform):
//   * fast: sign(A) N2 / 2^N1 is A with its fraction cut to 7 bits (a mask of
//     the fp32 bits), Bq / 2^N1 is B rounded to the grid 2^-N1 (adding and
//     subtracting 1.5 * 2^(23-N1)), and A_dy Xh + Bq/2^N1 + zp_out + 1/2 is
//     one fp32 FMA whose result, a multiple of 2^-N1 below 2^(24-N1), is
//     exact; its floor (an add rounded toward -inf) is Y.  Valid when every
//     channel of the row has 0 <= N1 <= 14 and |B| 2^N1 < 2^22, which the
//     row check below guarantees from per-launch channel bounds.
//   * exact: the integer formula in int64, element by element.
#include "fqvit_internal.cuh"

namespace fqvit {

namespace {

constexpr int kWarps = 8;  // warps (rows in flight) per block

struct LnShared {
    float gsmax;  // max |gamma/s_out| over channels
    float gsmin;  // min |gamma/s_out| over channels (0 if any is 0)
    float kappa;  // upper bound of max |beta/gamma| (fast-path check)
    int amax;     // max alpha
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

// fast path for one element (see the file comment); zh = zp_out + 0.5
__device__ __forceinline__ uint32_t ln_fast(float gs, float bs, float r, float t, int xh, float zh)
{
    float A = __fmul_rn(gs, r);
    int ab = __float_as_int(A);
    float Ady = __int_as_float(ab & (int)0xFFFF0000);
    float M = __int_as_float((ab & 0x7F800000) + ((16 << 23) | 0x400000));
    float B = __fsub_rn(bs, __fmul_rn(gs, t));
    float Bd = __fsub_rn(__fadd_rn(B, M), M);
    float Bz = __fadd_rn(Bd, zh);
    float xf = __fsub_rn(__int_as_float(xh + 0x4B400000), 12582912.0f);
    float y = __fmaf_rn(Ady, xf, Bz);
    y = fminf(fmaxf(y, 0.0f), 255.5f);
    return (uint32_t)__float_as_int(__fadd_rd(y, 12582912.0f)) & 0xFFu;
}

// Shared-memory position of channel c's constants: the four 16-byte units of each 16-channel chunk
// ch are permuted (unit q at q ^ ((ch >> 1) & 3)), so that eight lanes reading unit q of eight
// consecutive chunks touch eight different bank groups.  A permutation of 0 .. C-1 for C % 16 == 0;
// the vector path uses it, the generic path (any C) the identity.
__device__ __forceinline__ int ln_sidx(int c) { return (c & ~15) + ((((c >> 2) & 3) ^ ((c >> 5) & 3)) << 2) + (c & 3); }

// per-launch channel constants, computed by every block into shared memory (swizzled: ln_sidx)
__device__ void ln_prologue(const LnArgs &a, float *gs_s, float *bs_s, uint8_t *al_s, LnShared &sh, bool swz)
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
        const int sc = swz ? ln_sidx(c) : c;
        gs_s[sc] = gs;
        bs_s[sc] = bs;
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

// Vector path: C % 16 == 0, rows 16-byte aligned.  A segment of S lanes (a power of two) serves
// one row, so a warp carries 32 / S rows (short rows do not leave lanes idle); CPL = 16-byte
// chunks per lane, chunk sl + S i of the row for segment lane sl.
template <int S, int CPL>
__global__ void __launch_bounds__(kWarps * 32)
    ln_vec_kernel(LnArgs a)
{
    extern __shared__ __align__(16) unsigned char smem[];
    float *gs_s = reinterpret_cast<float *>(smem);
    float *bs_s = gs_s + a.C;
    uint8_t *al_s = reinterpret_cast<uint8_t *>(bs_s + a.C);
    __shared__ LnShared sh;
    pdl_release();
    pdl_wait();  // everything below reads or writes global memory
    ln_prologue(a, gs_s, bs_s, al_s, sh, true);

    constexpr int RPW = 32 / S;  // rows per warp
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int sl = lane & (S - 1), seg = lane / S;
    const int nch = a.C >> 4;
    const float zh = (float)a.zp_out + 0.5f;
    const float Cf = (float)a.C;

    // every lane of a warp runs every iteration (the segment reductions are warp shuffles);
    // rows past the end only skip their loads and stores
    const int64_t rstep = (int64_t)gridDim.x * kWarps * RPW;
    int64_t row = ((int64_t)blockIdx.x * kWarps + warp) * RPW + seg;
    // the row's 16-byte chunks, loaded one row ahead so that the HBM latency overlaps the work
    uint4 nv[CPL];
#pragma unroll
    for (int i = 0; i < CPL; ++i) {
        int ch = sl + S * i;
        nv[i] = (row < a.rows && ch < nch) ? __ldcs(reinterpret_cast<const uint4 *>(a.xq + row * a.ld_in) + ch)
                                           : make_uint4(0, 0, 0, 0);
    }
    for (; row - seg < a.rows; row += rstep) {  // warp-uniform: the warp's first row is in range
        const bool rv = row < a.rows;
        uint4 v[CPL];
#pragma unroll
        for (int i = 0; i < CPL; ++i) v[i] = nv[i];
        if (row + rstep < a.rows) {
            const uint4 *nsrc = reinterpret_cast<const uint4 *>(a.xq + (row + rstep) * a.ld_in);
#pragma unroll
            for (int i = 0; i < CPL; ++i) {
                int ch = sl + S * i;
                if (ch < nch) nv[i] = __ldcs(nsrc + ch);
            }
        }
        // pass 1: integer statistics
        int m1 = 0;
        unsigned long long m2 = 0;
#pragma unroll
        for (int i = 0; i < CPL; ++i) {
            int ch = sl + S * i;
            if (rv && ch < nch) {
                uint4 al4 = *reinterpret_cast<const uint4 *>(al_s + ch * 16);
                uint32_t w[4] = {v[i].x, v[i].y, v[i].z, v[i].w};
                uint32_t aw[4] = {al4.x, al4.y, al4.z, al4.w};
                unsigned int p2 = 0;  // <= 16 * (255 * 2^6)^2 < 2^32 for alpha <= 6
#pragma unroll
                for (int k = 0; k < 16; ++k) {
                    int x = (w[k >> 2] >> (8 * (k & 3))) & 0xFF;
                    int al = (aw[k >> 2] >> (8 * (k & 3))) & 0xFF;
                    int xh = (x - a.zp_in) << al;
                    m1 += xh;
                    if (sh.amax <= 6)
                        p2 += (unsigned int)(xh * xh);
                    else
                        m2 += (unsigned long long)((long long)xh * xh);
                }
                m2 += p2;
            }
        }
#pragma unroll
        for (int o = S / 2; o > 0; o >>= 1) {
            m1 += __shfl_xor_sync(0xffffffffu, m1, o);
            m2 += __shfl_xor_sync(0xffffffffu, m2, o);
        }
        if (!rv) continue;
        long long M1 = m1, M2 = (long long)m2;
        long long D = (long long)a.C * M2 - M1 * M1;
        float r = 0.0f, t = 0.0f;
        if (D != 0) {
            float sd = __fsqrt_rn(__ll2float_rn(D));
            r = __fdiv_rn(Cf, sd);
            t = __fdiv_rn(__ll2float_rn(M1), sd);
        }
        if (sl == 0) {
            if (a.m1) a.m1[row] = M1;
            if (a.m2) a.m2[row] = M2;
        }
        const bool fast = ln_row_fast(sh, r, t);  // one evaluation per row, chosen outside the loops
        uint4 *dst = reinterpret_cast<uint4 *>(a.yq + row * a.ld_out);
        // pass 2: requantization
        if (fast) {
#pragma unroll
            for (int i = 0; i < CPL; ++i) {
                int ch = sl + S * i;
                if (ch < nch) {
                    uint4 al4 = *reinterpret_cast<const uint4 *>(al_s + ch * 16);
                    uint32_t w[4] = {v[i].x, v[i].y, v[i].z, v[i].w};
                    uint32_t aw[4] = {al4.x, al4.y, al4.z, al4.w};
                    uint32_t o[4] = {0, 0, 0, 0};
                    const float4 *g4 = reinterpret_cast<const float4 *>(gs_s + ch * 16);
                    const float4 *b4 = reinterpret_cast<const float4 *>(bs_s + ch * 16);
                    const int qs = (ch >> 1) & 3;
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        float4 g = g4[q ^ qs], b = b4[q ^ qs];
                        float gg[4] = {g.x, g.y, g.z, g.w};
                        float bb[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            int x = (w[q] >> (8 * k)) & 0xFF;
                            int al = (aw[q] >> (8 * k)) & 0xFF;
                            int xh = (x - a.zp_in) << al;
                            o[q] |= ln_fast(gg[k], bb[k], r, t, xh, zh) << (8 * k);
                        }
                    }
                    __stcs(dst + ch, make_uint4(o[0], o[1], o[2], o[3]));
                }
            }
        } else {
#pragma unroll
            for (int i = 0; i < CPL; ++i) {
                int ch = sl + S * i;
                if (ch < nch) {
                    uint32_t o0 = 0, o1 = 0, o2 = 0, o3 = 0;
#pragma unroll 1
                    for (int k = 0; k < 16; ++k) {
                        const int c = ch * 16 + k;
                        const uint32_t wk = k < 8 ? (k < 4 ? v[i].x : v[i].y) : (k < 12 ? v[i].z : v[i].w);
                        int x = (wk >> (8 * (k & 3))) & 0xFF;
                        int xh = (x - a.zp_in) << al_s[c];
                        const int sc = ln_sidx(c);
                        const uint32_t y = (uint32_t)ln_exact(gs_s[sc], bs_s[sc], r, t, xh, a.zp_out) << (8 * (k & 3));
                        if (k < 4) o0 |= y; else if (k < 8) o1 |= y; else if (k < 12) o2 |= y; else o3 |= y;
                    }
                    __stcs(dst + ch, make_uint4(o0, o1, o2, o3));
                }
            }
        }
    }
}

// Generic path: any C, any stride or alignment; bytes, exact requantization.
__global__ void __launch_bounds__(kWarps * 32) ln_generic_kernel(LnArgs a)
{
    extern __shared__ __align__(16) unsigned char smem[];
    float *gs_s = reinterpret_cast<float *>(smem);
    float *bs_s = gs_s + a.C;
    uint8_t *al_s = reinterpret_cast<uint8_t *>(bs_s + a.C);
    __shared__ LnShared sh;
    ln_prologue(a, gs_s, bs_s, al_s, sh, false);
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

}  // namespace

cudaError_t launch_layernorm(const LnArgs &a, cudaStream_t st)
{
    size_t smem = (size_t)a.C * (2 * sizeof(float) + 1);
    smem = (smem + 15) & ~(size_t)15;
    const int nsm = sm_count();
    int64_t want = (a.rows + kWarps - 1) / kWarps;
    // Every block first derives the per-channel constants (three correctly rounded divisions per
    // channel), so the grid is the number of blocks that are resident at once: each block then
    // walks many rows.
    auto blocks_for = [&](const void *fn) -> int {
        int per_sm = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, kWarps * 32, smem) != cudaSuccess ||
            per_sm < 1)
            per_sm = 1;
        const int64_t cap = (int64_t)nsm * per_sm;
        return (int)(want < cap ? want : cap);
    };
    bool vec = (a.C % 16 == 0) && (a.ld_in % 16 == 0) && (a.ld_out % 16 == 0) &&
               ((uintptr_t)a.xq % 16 == 0) && ((uintptr_t)a.yq % 16 == 0) && a.C <= 4096;
    if (vec) {
        // segment width: the smallest power of two lanes holding the row's 16-byte chunks, at most 32
        const int nch = a.C / 16;
        int S = 1;
        while (S < nch && S < 32) S <<= 1;
        const int cpl = (nch + S - 1) / S;
        const int rpw = 32 / S;
        want = (a.rows + (int64_t)kWarps * rpw - 1) / ((int64_t)kWarps * rpw);
#define FQ_LN_LAUNCH(SS, N)                                                                      \
    {                                                                                           \
        cudaFuncSetAttribute(ln_vec_kernel<SS, N>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem); \
        return launch_pdl(ln_vec_kernel<SS, N>, dim3(blocks_for((const void *)ln_vec_kernel<SS, N>)), \
                          dim3(kWarps * 32), smem, st, a);                                      \
    }
        if (S < 32) {
            switch (S) {
            case 1: FQ_LN_LAUNCH(1, 1)
            case 2: FQ_LN_LAUNCH(2, 1)
            case 4: FQ_LN_LAUNCH(4, 1)
            case 8: FQ_LN_LAUNCH(8, 1)
            default: FQ_LN_LAUNCH(16, 1)
            }
        }
        switch (cpl) {
        case 1: FQ_LN_LAUNCH(32, 1)
        case 2: FQ_LN_LAUNCH(32, 2)
        case 3: FQ_LN_LAUNCH(32, 3)
        case 4: FQ_LN_LAUNCH(32, 4)
        case 5: FQ_LN_LAUNCH(32, 5)
        case 6: FQ_LN_LAUNCH(32, 6)
        case 7: FQ_LN_LAUNCH(32, 7)
        case 8: FQ_LN_LAUNCH(32, 8)
        default: break;
        }
#undef FQ_LN_LAUNCH
    }
    cudaFuncSetAttribute(ln_generic_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    ln_generic_kernel<<<blocks_for((const void *)ln_generic_kernel), kWarps * 32, smem, st>>>(a);
    return cudaGetLastError();
}

}  // namespace fqvit
