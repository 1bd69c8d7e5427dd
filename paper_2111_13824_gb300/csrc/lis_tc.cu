// lis_tc.cu -- fused Log-Int-Softmax + BitShift attention times values on
// the 5th-generation tensor cores (tcgen05) of sm_103a.
//
// Eq. 15 is a matrix product: acc = P (V - zp_V) with P[i][j] = 2^(15 - code_ij).
// Every P entry and every int8 value of V is exact in fp16, and for codes made
// by Log-Int-Softmax sum_j 2^-code_j <= 3 + L 2^-15 (2^-code < 1.5 / q_rev and
// q_rev >= S/e - 1/2), so with |V| <= 128 every partial sum of a row is an
// integer below 2^24: fp16 operands with fp32 accumulation give the integer
// result exactly.  The kernel therefore evaluates the shift-accumulate as
// tcgen05.mma.kind::f16 (M = 128 query rows, N = 64 = d, K = 16 keys per
// instruction) with the accumulator in tensor memory.
//
// One CTA per SM walks (head, 128-row tile) work items.  Roles:
//   warps 0-3 (thread = query row): the row maximum and i-exp row sum
//     (phase A), then per block of 64 keys the 4-bit codes written as fp16
//     operands 2^(15-code) into a 128B-swizzled K-major shared-memory tile,
//     and the block's V rows converted to fp16 (128B-swizzled, MN-major);
//     finally the epilogue reads the row's 64 accumulators from tensor memory.
//   warp 4, lane 0: bulk asynchronous copies of the tile's logits and the
//     head's V into shared memory, and the MMA issue.
// Ring of 3 operand stages, mbarrier hand-offs.  Every wait is bounded: after
// two seconds the kernel records a timeout status, drains what it issued and
// returns (the host reads the status with fqvit_sync_status).
#include "fqvit_internal.cuh"
#include "lis_common.cuh"

#include <cuda_fp16.h>

namespace fqvit {

__device__ int g_device_status = 0;

namespace {

using namespace lis;

constexpr int TM = 128;        // query rows per tile (MMA M)
constexpr int TKB = 64;        // keys per operand stage
constexpr int TSTAGES = 3;
constexpr int TD = 64;         // head dimension (MMA N)
constexpr int TMAXLD = 592;    // largest logit row stride handled here
constexpr int TCOPIES = 32;    // replicas of the i-exp table (one per lane)
constexpr int A_SLOT = TM * TKB * 2;
constexpr int B_SLOT = TKB * TD * 2;
constexpr unsigned long long kTimeoutNs = 2000000000ull;

struct TcParams {
    const int8_t *logits;
    int64_t ld;
    float s;
    const int8_t *v;
    int32_t *acc;
    int64_t BH;
    int L;
};

__device__ __forceinline__ uint32_t sa(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ uint64_t gtimer()
{
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ void mbar_init(uint64_t *b, uint32_t n)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(sa(b)), "r"(n) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t *b)
{
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(sa(b)) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t *b, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(sa(b)), "r"(bytes) : "memory");
}

__device__ __forceinline__ bool mbar_try(uint64_t *b, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
        : "=r"(ok)
        : "r"(sa(b)), "r"(parity)
        : "memory");
    return ok != 0;
}

// Bounded wait with exponential back-off (sleeping warps leave the issue slots
// to working ones); false on timeout or (honor_abort) when another role gave up.
__device__ __noinline__ bool mbar_wait(uint64_t *b, uint32_t parity, volatile int *abort_flag,
                                       bool honor_abort = true)
{
    if (mbar_try(b, parity)) return true;
    const uint64_t t0 = gtimer();
    uint32_t ns = 32;
    for (;;) {
        __nanosleep(ns);
        if (mbar_try(b, parity)) return true;
        if (ns < 1024) ns <<= 1;
        if (honor_abort && *abort_flag) return false;
        if (gtimer() - t0 > kTimeoutNs) {
            *abort_flag = 1;
            atomicExch(&g_device_status, 5);
            return false;
        }
    }
}

__device__ __forceinline__ void prefetch_l2(const void *src, uint32_t bytes)
{
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
}

__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes, uint64_t *b)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(sa(dst)),
        "l"(src), "r"(bytes), "r"(sa(b))
        : "memory");
}

__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// shared-memory matrix descriptor, 128-byte swizzle
__device__ __forceinline__ uint64_t smem_desc(uint32_t addr, uint32_t lbo, uint32_t sbo)
{
    uint64_t d = (uint64_t)((addr & 0x3FFFFu) >> 4);
    d |= (uint64_t)(lbo >> 4) << 16;
    d |= (uint64_t)(sbo >> 4) << 32;
    d |= 1ull << 46;  // descriptor version for tcgen05
    d |= 2ull << 61;  // SWIZZLE_128B
    return d;
}

// kind::f16 instruction descriptor: D f32, A/B f16, A K-major, B MN-major, N = 64, M = 128
constexpr uint32_t kIdesc = (1u << 4) | (1u << 16) | ((uint32_t)(TD >> 3) << 17) | ((uint32_t)(TM >> 4) << 24);

__device__ __forceinline__ void mma_f16(uint32_t dt, uint64_t ad, uint64_t bd, uint32_t accumulate)
{
    asm volatile(
        "{ .reg .pred p; setp.ne.b32 p, %4, 0; tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p; }" ::"r"(dt),
        "l"(ad), "l"(bd), "r"(kIdesc), "r"(accumulate)
        : "memory");
}

__device__ __forceinline__ void mma_commit(uint64_t *b)
{
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(sa(b))
                 : "memory");
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16])
{
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
}

__device__ __forceinline__ uint32_t fp16_operand(uint32_t code) { return (30u - code) << 10; }  // 2^(15-code)

// int8 x 2 (bytes b0, b1 of w ^ 0x80808080) -> half2 exact
__device__ __forceinline__ uint32_t i8x2_to_h2(uint32_t xw, uint32_t sel)
{
    uint32_t p = __byte_perm(xw, 0x64646464u, sel);  // 0x6400 | (v + 128): 1024 + v + 128
    __half2 h = *reinterpret_cast<__half2 *>(&p);
    h = __hsub2(h, __half2half2(__ushort_as_half((unsigned short)0x6480)));  // - 1152
    return *reinterpret_cast<uint32_t *>(&h);
}

struct TcShared {
    uint64_t lload, vload, full[TSTAGES], empty[TSTAGES], accfull, accempty, lfree, vfree, fin;
    uint32_t tmem;
    int abort_flag;
};

constexpr int TPARTS = 4;                      // threads per query row
constexpr int TSOFT = TM * TPARTS;             // softmax threads (16 warps)
constexpr int TPRODUCER_WARP = TSOFT / 32;     // warp 16: MMA issue
constexpr int TLOAD_WARP = TPRODUCER_WARP + 1; // warp 17: bulk copies of logits and V
constexpr int TTHREADS = (TLOAD_WARP + 1) * 32;
constexpr int TMAXKB = TMAXLD / TKB + 1;       // key blocks of the longest row

// fp16 exponent field (30 - code) of the operand 2^(15-code) for an i-exp
// value e of a row with 2S = hi + lo (G = bits of hi); see the file comment
// of lis.cu.  k = floor(log2(2S/e)) >= 1; codes above 15 clip to 15.
__device__ __forceinline__ uint32_t operand_exp(uint32_t e, int G, float hi, float lo)
{
    const float ef = __uint2float_rn(e);
    const int k = (G - __float_as_int(ef)) >> 23;
    const float Dk = fmaxf(__fsub_rn(__int_as_float((k << 23) + 0x3FC00000), 1.0f), 3.0f);
    const float t = __fmaf_rn(ef, Dk, -hi);
    uint32_t le;  // 0xFFFFFFFF when e D_k <= 2S
    asm("set.le.u32.f32 %0, %1, %2;" : "=r"(le) : "f"(t), "f"(lo));
    return (uint32_t)max(31 - k + (int)le, 15);
}

__device__ __forceinline__ uint32_t lds32(uint32_t a)
{
    uint32_t v;
    asm("ld.shared.b32 %0, [%1];" : "=r"(v) : "r"(a));
    return v;
}

// byte j of w, sign-extended
template <int J>
__device__ __forceinline__ int sbyte(uint32_t w)
{
    uint32_t y;
    asm("prmt.b32 %0, %1, 0, %2;" : "=r"(y) : "r"(w), "n"(J | ((J | 8) << 4) | ((J | 8) << 8) | ((J | 8) << 12)));
    return (int)y;
}

// i-exp value of byte J of w: table entry m - q of this lane
template <int J>
__device__ __forceinline__ uint32_t iexp_at(uint32_t lutq, uint32_t w)
{
    return lds32(lutq - 128u * (uint32_t)sbyte<J>(w));
}

template <int NKB>
__global__ void __launch_bounds__(TTHREADS, 1) lis_attn_tc_kernel(TcParams p)
{
    extern __shared__ unsigned char dsm_raw[];
    __shared__ TcShared sh;
    unsigned char *base = dsm_raw + ((1024u - (sa(dsm_raw) & 1023u)) & 1023u);
    unsigned char *As = base;
    unsigned char *Bs = As + TSTAGES * A_SLOT;
    int8_t *LG = (int8_t *)(Bs + TSTAGES * B_SLOT);
    int8_t *VS = LG + (size_t)TM * p.ld;
    uint32_t *LUT = (uint32_t *)(VS + (((size_t)p.L * TD + 15) & ~(size_t)15));

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    volatile int *abort_flag = &sh.abort_flag;
    if (tid == 0) {
        mbar_init(&sh.lload, 1);
        mbar_init(&sh.vload, 1);
        mbar_init(&sh.vfree, TSOFT);
        for (int s = 0; s < TSTAGES; ++s) {
            mbar_init(&sh.full[s], TSOFT);
            mbar_init(&sh.empty[s], 1);
        }
        mbar_init(&sh.accfull, 1);
        mbar_init(&sh.accempty, TM);
        mbar_init(&sh.lfree, TSOFT);
        mbar_init(&sh.fin, 1);
        sh.abort_flag = 0;
    }
    if (warp == TPRODUCER_WARP) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(sa(&sh.tmem)),
                     "r"(TD));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    {
        const IexpC c = iexp_consts(p.s);
        for (int i = tid; i < kLutSize * TCOPIES; i += blockDim.x) LUT[i] = iexp_neg(i / TCOPIES, c);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sh.tmem;

    const int L = p.L;
    const int tpb = (L + TM - 1) / TM;
    const int64_t ntiles = p.BH * tpb;

    if (tid < TSOFT) {
        // ---------------- softmax: thread = (query row r, 16-key quarter q of every 64-key block)
        const int r = tid >> 2, q = tid & 3;
        const int kk = tid >> 3, ci = tid & 7;  // V conversion: key kk of a block, values 8ci..8ci+7
        const uint32_t lut_lane = sa(LUT) + 4u * (uint32_t)lane;
        uint32_t g = 0;
        int it = 0;
        for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x, ++it) {
            const int64_t bh = tile / tpb;
            const int row = (int)(tile % tpb) * TM + r;
            const bool valid = row < L;
            if (!mbar_wait(&sh.lload, it & 1, abort_flag)) break;
            // the row's keys 64 kb + 16 q .. +15 of every block, from the staged tile
            const int8_t *lr = LG + (size_t)r * p.ld + 16 * q;
            uint4 w[NKB];
#pragma unroll
            for (int kb = 0; kb < NKB; ++kb) {
                const int k0 = kb * TKB + 16 * q;
                w[kb] = (valid && k0 < L) ? *reinterpret_cast<const uint4 *>(lr + kb * TKB)
                                          : make_uint4(0x80808080u, 0x80808080u, 0x80808080u, 0x80808080u);
                if (k0 < L && k0 + 16 > L) {  // keys at or past L: -128 (no effect on the max)
                    const int n = L - k0;
                    uint32_t ww[4] = {w[kb].x, w[kb].y, w[kb].z, w[kb].w};
#pragma unroll
                    for (int b = 0; b < 4; ++b) {
                        const int keep = n - 4 * b;
                        if (keep <= 0)
                            ww[b] = 0x80808080u;
                        else if (keep < 4)
                            ww[b] = (ww[b] & (0xFFFFFFFFu >> (32 - 8 * keep))) |
                                    (0x80808080u & ~(0xFFFFFFFFu >> (32 - 8 * keep)));
                    }
                    w[kb] = make_uint4(ww[0], ww[1], ww[2], ww[3]);
                }
            }
            fence_async_smem();
            mbar_arrive(&sh.lfree);  // the staged logits are in registers now: the next tile may load
            // phase A: row maximum and i-exp row sum
            uint32_t mx = 0x80808080u;
#pragma unroll
            for (int kb = 0; kb < NKB; ++kb)
                mx = __vmaxs4(mx, __vmaxs4(__vmaxs4(w[kb].x, w[kb].y), __vmaxs4(w[kb].z, w[kb].w)));
            int m = max(max(sbyte<0>(mx), sbyte<1>(mx)), max(sbyte<2>(mx), sbyte<3>(mx)));
            m = max(m, __shfl_xor_sync(0xffffffffu, m, 1));
            m = max(m, __shfl_xor_sync(0xffffffffu, m, 2));
            const uint32_t lutq = lut_lane + (uint32_t)(m * TCOPIES * 4);
            unsigned long long S = 0;
            if (valid) {
#pragma unroll
                for (int kb = 0; kb < NKB; ++kb) {
                    const int k0 = kb * TKB + 16 * q;
                    const uint32_t ww[4] = {w[kb].x, w[kb].y, w[kb].z, w[kb].w};
                    if (k0 + 16 <= L) {
#pragma unroll
                        for (int b = 0; b < 4; ++b) {
                            const uint32_t e0 = iexp_at<0>(lutq, ww[b]), e1 = iexp_at<1>(lutq, ww[b]);
                            const uint32_t e2 = iexp_at<2>(lutq, ww[b]), e3 = iexp_at<3>(lutq, ww[b]);
                            S += (unsigned long long)(e0 + e1) + (unsigned long long)(e2 + e3);  // each e < 2^31
                        }
                    } else if (k0 < L) {
                        const int n = L - k0;
#pragma unroll
                        for (int b = 0; b < 4; ++b) {
                            if (4 * b + 0 < n) S += iexp_at<0>(lutq, ww[b]);
                            if (4 * b + 1 < n) S += iexp_at<1>(lutq, ww[b]);
                            if (4 * b + 2 < n) S += iexp_at<2>(lutq, ww[b]);
                            if (4 * b + 3 < n) S += iexp_at<3>(lutq, ww[b]);
                        }
                    }
                }
            }
            S += __shfl_xor_sync(0xffffffffu, S, 1);
            S += __shfl_xor_sync(0xffffffffu, S, 2);
            const RowSum rs = make_rowsum(S);
            // phase B: the row's operands and the block's V, per 64-key block
            if (!mbar_wait(&sh.vload, it & 1, abort_flag)) break;
            bool stop = false;
#pragma unroll
            for (int kb = 0; kb < NKB; ++kb) {
                const int slot = (int)(g % TSTAGES);
                if (g >= TSTAGES && !mbar_wait(&sh.empty[slot], ((g / TSTAGES) - 1) & 1, abort_flag)) {
                    stop = true;
                    break;
                }
                const int k0 = kb * TKB + 16 * q;
                uint32_t o[8] = {0, 0, 0, 0, 0, 0, 0, 0};
                if (valid && k0 < L) {
                    const uint32_t ww[4] = {w[kb].x, w[kb].y, w[kb].z, w[kb].w};
                    uint32_t x[16];
#pragma unroll
                    for (int b = 0; b < 4; ++b) {
                        x[4 * b + 0] = operand_exp(iexp_at<0>(lutq, ww[b]), rs.hibits, rs.hi, rs.lo);
                        x[4 * b + 1] = operand_exp(iexp_at<1>(lutq, ww[b]), rs.hibits, rs.hi, rs.lo);
                        x[4 * b + 2] = operand_exp(iexp_at<2>(lutq, ww[b]), rs.hibits, rs.hi, rs.lo);
                        x[4 * b + 3] = operand_exp(iexp_at<3>(lutq, ww[b]), rs.hibits, rs.hi, rs.lo);
                    }
                    if (k0 + 16 > L) {  // keys at or past L get a zero operand
                        const int n = L - k0;
#pragma unroll
                        for (int j = 0; j < 16; ++j)
                            if (j >= n) x[j] = 0;
                    }
#pragma unroll
                    for (int b = 0; b < 8; ++b) o[b] = __byte_perm(x[2 * b], x[2 * b + 1], 0x5410) << 10;
                }
                unsigned char *arow = As + slot * A_SLOT + (r >> 3) * 1024 + (r & 7) * 128;
                *reinterpret_cast<uint4 *>(arow + (((2 * q) ^ (r & 7)) << 4)) = make_uint4(o[0], o[1], o[2], o[3]);
                *reinterpret_cast<uint4 *>(arow + (((2 * q + 1) ^ (r & 7)) << 4)) = make_uint4(o[4], o[5], o[6], o[7]);
                {
                    const int key = kb * TKB + kk;
                    uint4 v4 = make_uint4(0, 0, 0, 0);
                    if (key < L) {
                        const uint2 vw = *reinterpret_cast<const uint2 *>(VS + (size_t)key * TD + 8 * ci);
                        const uint32_t x0 = vw.x ^ 0x80808080u, x1 = vw.y ^ 0x80808080u;
                        v4.x = i8x2_to_h2(x0, 0x5140);
                        v4.y = i8x2_to_h2(x0, 0x7362);
                        v4.z = i8x2_to_h2(x1, 0x5140);
                        v4.w = i8x2_to_h2(x1, 0x7362);
                    }
                    *reinterpret_cast<uint4 *>(Bs + slot * B_SLOT + kk * 128 + ((ci ^ (kk & 7)) << 4)) = v4;
                }
                fence_async_smem();
                mbar_arrive(&sh.full[slot]);
                ++g;
            }
            if (stop || *abort_flag) break;
            fence_async_smem();
            mbar_arrive(&sh.vfree);  // the staged V of this tile is no longer read
            if (warp < 4) {
                // epilogue by warps 0-3 (tensor-memory lanes 32w..32w+31 = rows); the
                // other warps go on to the next tile meanwhile
                if (!mbar_wait(&sh.accfull, it & 1, abort_flag)) break;
                tc_fence_after();
                uint32_t v[4][16];
                const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
#pragma unroll
                for (int j = 0; j < 4; ++j) tmem_ld16(trow + 16 * j, v[j]);
                asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
                tc_fence_before();
                mbar_arrive(&sh.accempty);
                const int erow = (int)(tile % tpb) * TM + tid;
                if (erow < L) {
                    int4 *dst = reinterpret_cast<int4 *>(p.acc + ((size_t)bh * L + erow) * TD);
#pragma unroll
                    for (int j = 0; j < 4; ++j)
#pragma unroll
                        for (int c = 0; c < 4; ++c)
                            dst[4 * j + c] = make_int4(__float2int_rn(__uint_as_float(v[j][4 * c + 0])),
                                                       __float2int_rn(__uint_as_float(v[j][4 * c + 1])),
                                                       __float2int_rn(__uint_as_float(v[j][4 * c + 2])),
                                                       __float2int_rn(__uint_as_float(v[j][4 * c + 3])));
                }
            }
        }
    } else if (warp == TLOAD_WARP && lane == 0) {
        // ---------------- bulk copies: a tile's logits as soon as the previous tile's are in
        // registers, its V once the previous V is converted; L2 prefetch of the tile after
        int it = 0;
        int lloads = 0, vloads = 0;
        const uint32_t bv = (uint32_t)(L * TD);
        for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x, ++it) {
            const int64_t bh = tile / tpb;
            const int r0 = (int)(tile % tpb) * TM;
            if (it > 0 && !mbar_wait(&sh.lfree, (it - 1) & 1, abort_flag)) break;
            const uint32_t bl = (uint32_t)(min(TM, L - r0) * p.ld);
            mbar_expect_tx(&sh.lload, bl);
            bulk_g2s(LG, p.logits + ((size_t)bh * L + r0) * p.ld, bl, &sh.lload);
            ++lloads;
            const int64_t nxt = tile + gridDim.x;
            if (nxt < ntiles) {
                const int64_t bhn = nxt / tpb;
                const int r0n = (int)(nxt % tpb) * TM;
                prefetch_l2(p.logits + ((size_t)bhn * L + r0n) * p.ld, (uint32_t)(min(TM, L - r0n) * p.ld));
                if (bhn != bh) prefetch_l2(p.v + (size_t)bhn * L * TD, bv);
            }
            if (it > 0 && !mbar_wait(&sh.vfree, (it - 1) & 1, abort_flag)) break;
            mbar_expect_tx(&sh.vload, bv);
            bulk_g2s(VS, p.v + (size_t)bh * L * TD, bv, &sh.vload);
            ++vloads;
        }
        // drain: every copy issued has landed before the block exits
        if (lloads > 0) mbar_wait(&sh.lload, (lloads - 1) & 1, abort_flag, false);
        if (vloads > 0) mbar_wait(&sh.vload, (vloads - 1) & 1, abort_flag, false);
    } else if (warp == TPRODUCER_WARP && lane == 0) {
        // ---------------- MMA issue
        uint32_t g = 0;
        int it = 0;
        const int nkb = (L + TKB - 1) / TKB;
        for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x, ++it) {
            bool ok = true;
            for (int kb = 0; kb < nkb; ++kb, ++g) {
                const int slot = (int)(g % TSTAGES);
                if (!mbar_wait(&sh.full[slot], (g / TSTAGES) & 1, abort_flag)) {
                    ok = false;
                    break;
                }
                if (kb == 0 && it > 0 && !mbar_wait(&sh.accempty, (it - 1) & 1, abort_flag)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t a0 = sa(As + slot * A_SLOT), b0 = sa(Bs + slot * B_SLOT);
#pragma unroll
                for (int s = 0; s < TKB / 16; ++s)
                    mma_f16(tmem, smem_desc(a0 + 32 * s, 16, 1024), smem_desc(b0 + 2048 * s, 1024, 1024),
                            (kb | s) != 0);
                mma_commit(&sh.empty[slot]);
            }
            if (!ok) break;
            mma_commit(&sh.accfull);
        }
        // drain: every MMA issued by this thread has completed
        mma_commit(&sh.fin);
        mbar_wait(&sh.fin, 0, abort_flag, false);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == TPRODUCER_WARP)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TD));
}

size_t tc_smem_bytes(int L, int64_t ld)
{
    return 1024 + (size_t)TSTAGES * (A_SLOT + B_SLOT) + (size_t)TM * ld + (((size_t)L * TD + 15) & ~(size_t)15) +
           (size_t)kLutSize * TCOPIES * 4;
}

template <int NKB>
cudaError_t tc_launch(const TcParams &p, size_t smem, int grid, cudaStream_t st)
{
    cudaError_t e = cudaFuncSetAttribute(lis_attn_tc_kernel<NKB>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    lis_attn_tc_kernel<NKB><<<grid, TTHREADS, smem, st>>>(p);
    return cudaGetLastError();
}

}  // namespace

bool lis_attention_tc_eligible(const LisArgs &a, const AttnVArgs &b)
{
    return b.d == TD && a.bias == nullptr && a.codes == nullptr && b.zp_v == 0 && a.ld_logit <= TMAXLD &&
           a.ld_logit % 16 == 0 && b.ld_v == TD && b.ld_acc == TD && ((uintptr_t)a.logits % 16) == 0 &&
           ((uintptr_t)b.v % 16) == 0 && ((uintptr_t)b.acc % 16) == 0 && tc_smem_bytes(a.L, a.ld_logit) <= 232448;
}

cudaError_t launch_lis_attention_tc(const LisArgs &a, const AttnVArgs &b, cudaStream_t st)
{
    TcParams p{a.logits, a.ld_logit, a.s_logit, b.v, b.acc, b.BH, a.L};
    const size_t smem = tc_smem_bytes(a.L, a.ld_logit);
    const int64_t ntiles = b.BH * ((a.L + TM - 1) / TM);
    const int grid = (int)(ntiles < sm_count() ? ntiles : sm_count());
    switch ((a.L + TKB - 1) / TKB) {
    case 1: return tc_launch<1>(p, smem, grid, st);
    case 2: return tc_launch<2>(p, smem, grid, st);
    case 3: return tc_launch<3>(p, smem, grid, st);
    case 4: return tc_launch<4>(p, smem, grid, st);
    case 5: return tc_launch<5>(p, smem, grid, st);
    case 6: return tc_launch<6>(p, smem, grid, st);
    case 7: return tc_launch<7>(p, smem, grid, st);
    case 8: return tc_launch<8>(p, smem, grid, st);
    case 9: return tc_launch<9>(p, smem, grid, st);
    default: return tc_launch<10>(p, smem, grid, st);
    }
}

cudaError_t read_clear_device_status(int *status, cudaStream_t st)
{
    int zero = 0;
    cudaError_t e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return e;
    e = cudaMemcpyFromSymbol(status, g_device_status, sizeof(int));
    if (e != cudaSuccess) return e;
    return cudaMemcpyToSymbol(g_device_status, &zero, sizeof(int));
}

}  // namespace fqvit
