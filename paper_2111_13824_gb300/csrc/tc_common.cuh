// tc_common.cuh -- device helpers of the tcgen05 attention kernels: shared-memory
// addresses, mbarriers with bounded waits, tensor-memory loads and stores, MMA
// issue and descriptors, byte permutes, and the exact fp32 pieces of the
// Log-Int-Softmax code test (the derivation is in the file comment of lis.cu).
#pragma once

#include <cuda_fp16.h>
#include <stdint.h>

#include "lis_common.cuh"

namespace fqvit {
namespace tc {

using lis::RowSum;

constexpr unsigned long long kTimeoutNs = 2000000000ull;

// Status word of the kernels of one translation unit (0 ok, 5 a bounded wait
// timed out); each kernel file reads and clears its own copy on the host.
static __device__ int g_status = 0;

// kind::f16 instruction descriptor: D f32, A/B f16, A K-major, B MN-major, N = 64, M = 128
constexpr uint32_t kIdesc = (1u << 4) | (1u << 16) | ((uint32_t)(64 >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
// N = 16, B K-major (a block of ones, so its layout does not matter), M = 128
constexpr uint32_t kIdescOnes = (1u << 4) | ((uint32_t)(16 >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);

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

// try_wait that may suspend the thread until the phase completes, for at most ns nanoseconds
__device__ __forceinline__ bool mbar_try_for(uint64_t *b, uint32_t parity, uint32_t ns)
{
    uint32_t ok;
    asm volatile(
        "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3; selp.u32 %0, 1, 0, p; }"
        : "=r"(ok)
        : "r"(sa(b)), "r"(parity), "r"(ns)
        : "memory");
    return ok != 0;
}

// Bounded wait: the thread sleeps in the barrier (woken when the phase completes) in slices of
// at most 50 us; false on timeout or (honor_abort) when another role gave up.  (Sleeps growing
// to 256 ns between slices were tried: no gain for long rows, 5-8 % slower for short ones.)
static __device__ __noinline__ bool mbar_wait_slow(uint64_t *b, uint32_t parity, volatile int *abort_flag,
                                            bool honor_abort)
{
    if (mbar_try(b, parity)) return true;
    const uint64_t t0 = gtimer();
    for (;;) {
        if (mbar_try_for(b, parity, 50000)) return true;
        if (honor_abort && *abort_flag) return false;
        if (gtimer() - t0 > kTimeoutNs) {
            *abort_flag = 1;
            atomicExch(&g_status, 5);
            return false;
        }
        __nanosleep(64);
    }
}

// A completed phase costs one inline probe; the out-of-line wait (whose call makes the caller save and
// restore its live registers) runs only when the phase is still open.
__device__ __forceinline__ bool mbar_wait(uint64_t *b, uint32_t parity, volatile int *abort_flag,
                                          bool honor_abort = true)
{
    return mbar_try(b, parity) || mbar_wait_slow(b, parity, abort_flag, honor_abort);
}

__device__ __forceinline__ void prefetch_l2(const void *src, uint32_t bytes)
{
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
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

__device__ __forceinline__ void mma_commit(uint64_t *b)
{
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(sa(b))
                 : "memory");
}


// int8 x 2 (bytes b0, b1 of w ^ 0x80808080) -> half2 exact
__device__ __forceinline__ uint32_t i8x2_to_h2(uint32_t xw, uint32_t sel)
{
    uint32_t p = __byte_perm(xw, 0x64646464u, sel);  // 0x6400 | (v + 128): 1024 + v + 128
    __half2 h = *reinterpret_cast<__half2 *>(&p);
    h = __hsub2(h, __half2half2(__ushort_as_half((unsigned short)0x6480)));  // - 1152
    return *reinterpret_cast<uint32_t *>(&h);
}
// fp16 exponent field (30 - code) of the operand 2^(15-code) for an i-exp
// value ef (fp32) of a row with 2S = hi + lo (G = bits of hi); see the file comment
// of lis.cu.  k = floor(log2(2S/e)) >= 1; codes above 15 clip to 15.
__device__ __forceinline__ uint32_t operand_exp_f(float ef, int G, float hi, float lo)
{
    const int k = (G - __float_as_int(ef)) >> 23;
    const float Dk = fmaxf(__fsub_rn(__int_as_float((k << 23) + 0x3FC00000), 1.0f), 3.0f);
    const float t = __fmaf_rn(ef, Dk, -hi);
    uint32_t le;  // 0xFFFFFFFF when e D_k <= 2S
    asm("set.le.u32.f32 %0, %1, %2;" : "=r"(le) : "f"(t), "f"(lo));
    return (uint32_t)max(31 - k + (int)le, 15);
}

// the same for an integer i-exp value (exact in fp32: at most 16 significant bits)
__device__ __forceinline__ uint32_t operand_exp(uint32_t e, int G, float hi, float lo)
{
    return operand_exp_f(__uint2float_rn(e), G, hi, lo);
}


// 2S = hi + lo with hi = fp32(2S) rounded to nearest even and lo exact (|lo| < 2^19), from
// integer operations only (the same values as the fp32 conversions of make_rowsum)
__device__ __forceinline__ RowSum split_2s(unsigned long long S)
{
    const unsigned long long s2 = 2ull * S;
    RowSum rs;
    if (s2 < (1ull << 24)) {
        rs.hi = __uint2float_rn((uint32_t)s2);
        rs.lo = 0.0f;
    } else {
        const int p = 63 - __clzll((long long)s2);  // 24 .. 42
        const int sh = p - 23;
        unsigned long long mant = s2 >> sh;         // 2^23 .. 2^24 - 1
        const unsigned long long rem = s2 & ((1ull << sh) - 1), half = 1ull << (sh - 1);
        if (rem > half || (rem == half && (mant & 1ull))) ++mant;
        int e = p;
        if (mant == (1ull << 24)) {
            mant >>= 1;
            ++e;
        }
        rs.hi = __int_as_float(((127 + e) << 23) | (int)(mant & 0x7FFFFFull));
        const int lo = (int)((long long)s2 - (long long)(mant << (e - 23)));  // |lo| <= half < 2^19
        rs.lo = __fsub_rn(__int_as_float(lo + 0x4B400000), 12582912.0f);    // exact below 2^22
    }
    rs.hibits = __float_as_int(rs.hi);
    return rs;
}

// mbar_wait with one verdict for the whole warp (the callers go on to
// warp-collective tcgen05 instructions)
__device__ __forceinline__ bool mbar_wait_warp(uint64_t *b, uint32_t parity, volatile int *abort_flag)
{
    return __all_sync(0xFFFFFFFFu, mbar_wait(b, parity, abort_flag));
}

__device__ __forceinline__ uint32_t lds32(uint32_t a)
{
    uint32_t v;
    asm volatile("ld.shared.b32 %0, [%1];" : "=r"(v) : "r"(a) : "memory");
    return v;
}

// byte permute with the sign-replicate selector bit honoured
__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel)
{
    uint32_t y;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(y) : "r"(a), "r"(b), "r"(sel));
    return y;
}

// lane-wise maximum of two pairs of signed 16-bit integers
__device__ __forceinline__ uint32_t vmax16x2(uint32_t a, uint32_t b)
{
    uint32_t d;
    asm("max.s16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
    return d;
}

// byte j of w, sign-extended
template <int J>
__device__ __forceinline__ int sbyte(uint32_t w)
{
    uint32_t y;
    asm("prmt.b32 %0, %1, 0, %2;" : "=r"(y) : "r"(w), "n"(J | ((J | 8) << 4) | ((J | 8) << 8) | ((J | 8) << 12)));
    return (int)y;
}

// warp-collective (.sync.aligned): the whole warp, converged, writes its 32 lanes (2 columns)
__device__ __forceinline__ void tmem_st2(uint32_t taddr, uint32_t r0, uint32_t r1)
{
    __syncwarp();
    asm volatile("tcgen05.st.sync.aligned.32x32b.x2.b32 [%0], {%1,%2};" ::"r"(taddr), "r"(r0), "r"(r1) : "memory");
}

// warp-collective (.sync.aligned): the whole warp, converged, writes its 32 lanes (4 columns)
__device__ __forceinline__ void tmem_st4(uint32_t taddr, const uint32_t (&r)[4])
{
    __syncwarp();
    asm volatile("tcgen05.st.sync.aligned.32x32b.x4.b32 [%0], {%1,%2,%3,%4};" ::"r"(taddr), "r"(r[0]), "r"(r[1]),
                 "r"(r[2]), "r"(r[3])
                 : "memory");
}

// warp-collective (.sync.aligned): the whole warp, converged, writes its 32 lanes
__device__ __forceinline__ void tmem_st8(uint32_t taddr, const uint32_t (&r)[8])
{
    __syncwarp();
    asm volatile("tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"r"(taddr), "r"(r[0]),
                 "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7])
                 : "memory");
}

__device__ __forceinline__ void mma_f16_ta(uint32_t dt, uint32_t at, uint64_t bd, uint32_t accumulate,
                                           uint32_t idesc = kIdesc)
{
    asm volatile(
        "{ .reg .pred p; setp.ne.b32 p, %4, 0; tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p; }" ::"r"(dt),
        "r"(at), "l"(bd), "r"(idesc), "r"(accumulate)
        : "memory");
}

// D (tensor memory) (+)= A B with both operands in shared memory (descriptors)
__device__ __forceinline__ void mma_f16_ss(uint32_t dt, uint64_t ad, uint64_t bd, uint32_t idesc, bool accumulate)
{
    asm volatile(
        "{ .reg .pred p; setp.ne.b32 p, %4, 0; tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p; }" ::"r"(dt),
        "l"(ad), "l"(bd), "r"(idesc), "r"((uint32_t)accumulate)
        : "memory");
}

// shared-memory matrix descriptor without swizzle
__device__ __forceinline__ uint64_t smem_desc_plain(uint32_t addr, uint32_t lbo, uint32_t sbo)
{
    uint64_t d = (uint64_t)((addr & 0x3FFFFu) >> 4);
    d |= (uint64_t)(lbo >> 4) << 16;
    d |= (uint64_t)(sbo >> 4) << 32;
    d |= 1ull << 46;  // descriptor version for tcgen05
    return d;
}

__device__ __forceinline__ void tmem_ld1(uint32_t taddr, uint32_t &r)
{
    __syncwarp();
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x1.b32 {%0}, [%1];" : "=r"(r) : "r"(taddr));
}

__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes, uint64_t *b)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(sa(dst)),
        "l"(src), "r"(bytes), "r"(sa(b))
        : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t *b, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(sa(b)), "r"(bytes) : "memory");
}

// 32 bytes of int32 to global memory (32-byte aligned)
__device__ __forceinline__ void stg256(int32_t *p, const int (&v)[8])
{
    asm volatile("st.global.v8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"l"(p), "r"(v[0]), "r"(v[1]), "r"(v[2]),
                 "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7])
                 : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32])
{
    __syncwarp();
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
}

__device__ __forceinline__ void tmem_ld8(uint32_t taddr, uint32_t (&r)[8])
{
    __syncwarp();
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
                 : "r"(taddr));
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16])
{
    __syncwarp();
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
}

__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// minimum of two pairs of unsigned 16-bit integers
__device__ __forceinline__ uint32_t vmin16x2u(uint32_t a, uint32_t b)
{
    uint32_t d;
    asm("min.u16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
    return d;
}

// maximum of two pairs of unsigned 16-bit integers
__device__ __forceinline__ uint32_t vmax16x2u(uint32_t a, uint32_t b)
{
    uint32_t d;
    asm("max.u16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
    return d;
}

}  // namespace tc
}  // namespace fqvit
