// qk_tc.cu -- the MatMul Q K^T of attention with its 8-bit output quantizer, on
// the 5th-generation tensor cores (tcgen05) of sm_103a: int8 Q and K codes with
// zero points in, int8 logits out (the input of Log-Int-Softmax).
//
// P = (Q - zp_q)(K - zp_k)^T is exact on the tensor cores: every shifted code
// lies in -255 .. 255 (exact in fp16), every product below 2^16, and a sum of
// at most 64 of them below 2^22, exact in the fp32 accumulators.  The output
// quantizer is uniform MinMax (Sec. 3) applied with the dyadic multiplier of
// the supplement's LayerNorm output stage, M = s_q s_k / (sqrt(d) s_logit) as
// N2 / 2^N1:
//   logit = clip(floor((N2 P + 2^(N1-1)) / 2^N1) + zp_l, -128, 127).
// With |P| < 2^22 and N2 < 2^8, N2 P + 2^(N1-1) fits 31 bits, so the epilogue
// runs in 32-bit integers: the accumulator's bits plus 1.5 2^23 give P, one
// multiply-add, one arithmetic shift, and a saturating pack of four values.
//
// One CTA per SM walks (head, 128-row tile) work items, each CTA a contiguous
// range, so consecutive tiles share a head.  Per head, K -> fp16 in shared
// memory (B operand: keys x 64, K-major, 128-byte swizzle, d padded to 64 with
// zeros); per tile, the 128 query rows of Q likewise (A operand).  The keys go
// through the tensor cores in chunks of 128 (M = 128, N <= 128, K = 64) into four
// tensor-memory buffers, up to four chunks ahead of the epilogue.  Roles:
//   warps 0-15 (epilogue): convert the operands, then read each chunk back
//     (warp w: lanes 32 (w % 4) .., columns 32 (w / 4) ..), quantize it and
//     write the bytes into a staging buffer (or, for strides the tensor store
//     cannot take, into a shared-memory tile of the output that all of them
//     copy out with coalesced 16-byte stores);
//   warp 16, lane 0: the bulk copies of the next tile's Q and head's K and the
//     MMAs (a tcgen05.mma holds its issuing thread about 200 cycles, so it does
//     nothing else);
//   warp 17, lane 0: the tensor stores of the staging buffers.
// They meet only on mbarriers (chunk computed / read, staging written / read,
// operands converted), so no warp waits at a block barrier for another's MMA
// issue.  Every wait is bounded: after two seconds the kernel records a timeout
// status, drains what it issued and returns.
#include "fqvit_internal.cuh"
#include "tc_common.cuh"

#include <cmath>
#include <cstring>
#include <cuda.h>
#include <cuda_fp16.h>
#include <cudaTypedefs.h>

namespace fqvit {

namespace {

using namespace tc;

constexpr int QM = 128;          // query rows per tile (MMA M)
constexpr int QNC = 128;         // keys per chunk (MMA N of a full chunk)
constexpr int QNBUF = 4;         // tensor-memory buffers of a chunk (all 512 columns)
constexpr int QKD = 64;          // the MMA's reduction: d padded to 64
constexpr int QTHREADS = 512;    // epilogue threads (16 warps)
constexpr int QEPI_WARPS = QTHREADS / 32;
constexpr int QMMA_WARP = QEPI_WARPS;      // warp 16, lane 0: operand copies and MMAs
constexpr int QALL = QTHREADS + 64;        // + warp 17, lane 0: tensor stores
// Register bound of the launch: 18 warps put five on two of the four schedulers, whose register files
// (16384 each) then allow 96 per thread, the bound a block of 640 threads gets.
constexpr int QBOUND = 640;
constexpr int QMAXL = 640;       // keys of the longest row
constexpr int QROW = QKD * 2;    // bytes of an fp16 operand row
constexpr int QNST = 3;          // BULK: staging buffers of a chunk's output (128 x 128 bytes each)
constexpr int QST_BYTES = QM * QNC;

struct QkParams {
    const int8_t *q, *k;
    int64_t ld_q, ld_k;
    int zp_q, zp_k;
    int8_t *out;
    int64_t ld;
    int64_t BH;
    int L, d;
    int n1;       // N1 >= 1 (the host sends N1 <= 0 to the 64-bit epilogue)
    uint32_t c1;  // 2^(N1-1) + zp_l 2^N1 - N2 (0x4B400000): the constant of the multiply-add (mod 2^32)
    int n2;
    int zp_l;
};

struct QkShared {
    uint64_t sfull[QNBUF];   // the chunk in tensor-memory buffer b is computed (MMA commit)
    uint64_t sempty[QNBUF];  // every epilogue warp has read buffer b
    uint64_t stfull[QNST];   // every epilogue warp has written staging buffer s (BULK)
    uint64_t stfree[QNST];   // the tensor store of staging buffer s has read it (BULK)
    uint64_t opsready;       // the tile's Q (and a new head's K) are in the operand layout
    uint64_t fin, qload, kload;
    uint32_t tmem;
    int abort_flag;
};

__device__ __forceinline__ uint32_t pack_sat_s8(int hi, int lo, uint32_t c)
{
    uint32_t d;  // bits 31..16: c[15:0], 15..8: sat(hi), 7..0: sat(lo)
    asm("cvt.pack.sat.s8.s32.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(hi), "r"(lo), "r"(c));
    return d;
}

// eight int8 codes minus a zero point -> eight fp16 values (exact: -255 .. 255)
__device__ __forceinline__ uint4 codes_to_h8(uint2 w, __half2 z)
{
    const uint32_t x0 = w.x ^ 0x80808080u, x1 = w.y ^ 0x80808080u;
    uint32_t h[4] = {i8x2_to_h2(x0, 0x5140), i8x2_to_h2(x0, 0x7362), i8x2_to_h2(x1, 0x5140), i8x2_to_h2(x1, 0x7362)};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        __half2 t = __hsub2(*reinterpret_cast<const __half2 *>(&h[i]), z);
        h[i] = *reinterpret_cast<const uint32_t *>(&t);
    }
    return make_uint4(h[0], h[1], h[2], h[3]);
}

// The logit of one accumulator (an exact integer P in fp32, |P| < 2^22).
//   FOLD: (N2 P + 2^(N1-1) + zp_l 2^N1) >> N1 in 32 bits (the host checked that it fits)
//   else: the 64-bit formula, N1 of any sign
// (n2, c1, n1: the launch's constants, held in registers by the caller)
// Two accumulators plus 1.5 2^23 in one packed fp32 add (each sum exact: |P| < 2^22): the bit
// patterns 0x4B400000 + P of the FOLD form below
__device__ __forceinline__ void add_magic2(uint32_t a, uint32_t b, uint32_t &x, uint32_t &y)
{
    asm("{ .reg .b64 ra, rd;\n\t"
        "mov.b64 ra, {%2, %3};\n\t"
        "add.rn.f32x2 rd, ra, %4;\n\t"
        "mov.b64 {%0, %1}, rd; }"
        : "=r"(x), "=r"(y)
        : "r"(a), "r"(b), "l"(0x4B4000004B400000ull));
}

// The logit of an accumulator already in the form 0x4B400000 + P (FOLD): one multiply-add and a shift
__device__ __forceinline__ int logit_of_biased(uint32_t x, uint32_t n2, uint32_t c1, int n1)
{
    return (int)(x * n2 + c1) >> n1;
}

template <bool FOLD>
__device__ __forceinline__ int logit_of(uint32_t acc_bits, const QkParams &p, uint32_t n2, uint32_t c1, int n1)
{
    if (FOLD) {
        const uint32_t x = __float_as_uint(__fadd_rn(__uint_as_float(acc_bits), 12582912.0f));
        return (int)(x * n2 + c1) >> n1;
    } else {
        const int P = __float2int_rn(__uint_as_float(acc_bits));
        const long long num = (long long)p.n2 * P;
        long long R;
        if (p.n1 > 0)
            R = (num + (1ll << (p.n1 - 1))) >> p.n1;
        else
            R = num * (1ll << min(-p.n1, 10));
        R += p.zp_l;
        return (int)(R < -128 ? -128 : R > 127 ? 127 : R);
    }
}

// BULK: Q and K rows reach shared memory as int8 by bulk copies one tile (one head) ahead of
// their conversion (strides of at most 64 bytes, multiples of 16), and each chunk's 128 x 128
// output bytes leave through one of QNST staging buffers (128-byte swizzle) by a tensor store
// of the logits viewed as [BH][L][ld] (rows past L and bytes past ld clipped), so the drain of
// one chunk overlaps the work on the next.  Else each thread loads its codes from global
// memory as it converts them, and the tile's output is copied out from a shared-memory tile.
template <bool FOLD, bool BULK>
__global__ void __launch_bounds__(QBOUND, 1)
    qk_logits_tc_kernel(const __grid_constant__ QkParams p, const __grid_constant__ CUtensorMap tmap)
{
    extern __shared__ unsigned char dsm_raw[];
    __shared__ QkShared sh;
    unsigned char *base = dsm_raw + ((1024u - (sa(dsm_raw) & 1023u)) & 1023u);
    unsigned char *KS = base;                            // QMAXL x 128 B (keys, fp16, swizzled)
    unsigned char *QS = KS + QMAXL * QROW;               // QM x 128 B
    unsigned char *OS = QS + QM * QROW;                  // BULK: QNST x 16 KB staging; else QM x ld bytes
    unsigned char *KST = OS + (BULK ? (size_t)QNST * QST_BYTES : (size_t)QM * p.ld);  // BULK: L x ld_k int8
    unsigned char *QST = KST + (size_t)QMAXL * 64;       // BULK: QM x ld_q int8 of the next tile

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    volatile int *abort_flag = &sh.abort_flag;
    pdl_release();
    if (tid == 0) {
        for (int b = 0; b < QNBUF; ++b) {
            mbar_init(&sh.sfull[b], 1);
            mbar_init(&sh.sempty[b], QEPI_WARPS);
        }
        for (int s = 0; s < QNST; ++s) {
            mbar_init(&sh.stfull[s], QEPI_WARPS);
            mbar_init(&sh.stfree[s], 1);
        }
        mbar_init(&sh.opsready, QEPI_WARPS);
        mbar_init(&sh.fin, 1);
        mbar_init(&sh.qload, 1);
        mbar_init(&sh.kload, 1);
        sh.abort_flag = 0;
    }
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(sa(&sh.tmem)),
                     "r"(QNBUF * QNC));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    const int L = p.L, d = p.d;
    const int L16 = (L + 15) & ~15;                     // keys that go through the MMAs
    const int nch = (L + QNC - 1) / QNC;
    // bytes of each output row past the MMA'd keys (up to ld) stay zero for the whole launch
    for (int x = tid; !BULK && x < QM * (int)(p.ld - L16); x += QALL) {
        const int r = x / (int)(p.ld - L16), j = x - r * (int)(p.ld - L16);
        OS[(size_t)r * p.ld + L16 + j] = 0;
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sh.tmem;

    const int tpb = (L + QM - 1) / QM;
    const int64_t ntiles = p.BH * tpb;
    const int64_t t_begin = (int64_t)blockIdx.x * ntiles / gridDim.x;
    const int64_t t_end = (int64_t)(blockIdx.x + 1) * ntiles / gridDim.x;
    pdl_wait();  // the set-up above touched no global memory

    if (warp < QEPI_WARPS) {
        // ---------------- epilogue warps: operands in, accumulators out
        const __half2 zq2 = __half2half2(__int2half_rn(p.zp_q)), zk2 = __half2half2(__int2half_rn(p.zp_k));
        // the requantization's constants in registers (an integer multiply-add takes one constant-bank operand)
        uint32_t rn2 = (uint32_t)p.n2, rc1 = p.c1;
        int rn1 = p.n1;
        asm volatile("" : "+r"(rn2), "+r"(rc1), "+r"(rn1));
        const int qr = 32 * (warp & 3) + lane;  // tile row of this thread
        const int g = warp >> 2;                // 32-column group of a chunk
        uint32_t qph = 0, kph = 0;              // BULK: phases of the copy barriers waited for
        uint32_t gc = 0;                        // chunks are numbered across the CTA's tiles
        int cur_bh = -1;
        for (int64_t t = t_begin; t < t_end; ++t) {
            const int bh = (int)(t / tpb);
            const int r0 = (int)(t - (int64_t)bh * tpb) * QM;
            // ---- operands: K of a new head, the tile's Q rows (8 values = 16 bytes of fp16 per item).
            //      The MMAs of the previous tile, which read them, have completed: its last chunk was
            //      waited for below.
            bool bad = false;
            if (bh != cur_bh) {
                if (BULK) {
                    bad = !mbar_wait_warp(&sh.kload, kph & 1, abort_flag);
                    ++kph;
                }
                for (int x = tid; x < L16 * 8 && !bad; x += QTHREADS) {
                    const int key = x >> 3, c = x & 7;
                    uint4 h = make_uint4(0, 0, 0, 0);
                    if (key < L && 8 * c < d) {
                        const uint2 w = BULK ? *reinterpret_cast<const uint2 *>(KST + key * p.ld_k + 8 * c)
                                             : __ldg(reinterpret_cast<const uint2 *>(p.k + ((size_t)bh * L + key) * p.ld_k + 8 * c));
                        h = codes_to_h8(w, zk2);
                    }
                    *reinterpret_cast<uint4 *>(KS + key * QROW + ((c ^ (key & 7)) << 4)) = h;
                }
                cur_bh = bh;
            }
            if (BULK && !bad) {
                bad = !mbar_wait_warp(&sh.qload, qph & 1, abort_flag);
                ++qph;
            }
            for (int x = tid; x < QM * 8 && !bad; x += QTHREADS) {
                const int r = x >> 3, c = x & 7;
                uint4 h = make_uint4(0, 0, 0, 0);
                if (r0 + r < L && 8 * c < d) {
                    const uint2 w = BULK ? *reinterpret_cast<const uint2 *>(QST + r * p.ld_q + 8 * c)
                                         : __ldg(reinterpret_cast<const uint2 *>(p.q + ((size_t)bh * L + r0 + r) * p.ld_q + 8 * c));
                    h = codes_to_h8(w, zq2);
                }
                *reinterpret_cast<uint4 *>(QS + r * QROW + ((c ^ (r & 7)) << 4)) = h;
            }
            fence_async_smem();  // the operands are read by the MMAs (and the staging areas refilled)
            tc_fence_before();
            __syncwarp();
            if (!bad && lane == 0) mbar_arrive(&sh.opsready);
            // ---- chunks: read back, quantize, into the output staging (or tile)
            for (int c = 0; c < nch && !bad; ++c, ++gc) {
                const uint32_t b = gc % QNBUF, s = gc % QNST;
                bad = !mbar_wait_warp(&sh.sfull[b], (gc / QNBUF) & 1, abort_flag);
                // BULK: the store of chunk gc - QNST has read this staging buffer
                if (BULK && !bad && gc >= (uint32_t)QNST)
                    bad = !mbar_wait_warp(&sh.stfree[s], ((gc - QNST) / QNST) & 1, abort_flag);
                if (bad) break;
                tc_fence_after();
                const int col0 = c * QNC + 32 * g;  // first key of this warp's 32 columns
                // BULK: this chunk's staging buffer, 16-byte unit u of tile row qr at u ^ (qr % 8)
                unsigned char *srow = OS + (size_t)s * QST_BYTES + qr * QNC;
                if (BULK && col0 >= L16 && col0 < p.ld) {  // bytes past the keys, inside the row
                    *reinterpret_cast<uint4 *>(srow + (((2 * g) ^ (qr & 7)) << 4)) = make_uint4(0, 0, 0, 0);
                    *reinterpret_cast<uint4 *>(srow + (((2 * g + 1) ^ (qr & 7)) << 4)) = make_uint4(0, 0, 0, 0);
                }
                if (col0 < L16) {
                    uint32_t v[32];
                    tmem_ld32(tmem + ((uint32_t)(32 * (warp & 3)) << 16) + (uint32_t)(b * QNC + 32 * g), v);
                    tmem_wait_ld();
                    uint32_t w[8];
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        int l0, l1, l2, l3;
                        if (FOLD) {  // the magic additions two at a time
                            uint32_t x0, x1, x2, x3;
                            add_magic2(v[4 * i], v[4 * i + 1], x0, x1);
                            add_magic2(v[4 * i + 2], v[4 * i + 3], x2, x3);
                            l0 = logit_of_biased(x0, rn2, rc1, rn1);
                            l1 = logit_of_biased(x1, rn2, rc1, rn1);
                            l2 = logit_of_biased(x2, rn2, rc1, rn1);
                            l3 = logit_of_biased(x3, rn2, rc1, rn1);
                        } else {
                            l0 = logit_of<FOLD>(v[4 * i], p, rn2, rc1, rn1);
                            l1 = logit_of<FOLD>(v[4 * i + 1], p, rn2, rc1, rn1);
                            l2 = logit_of<FOLD>(v[4 * i + 2], p, rn2, rc1, rn1);
                            l3 = logit_of<FOLD>(v[4 * i + 3], p, rn2, rc1, rn1);
                        }
                        w[i] = pack_sat_s8(l1, l0, pack_sat_s8(l3, l2, 0u));
                    }
                    if (col0 + 32 > L) {  // keys at or past L: zero bytes (the last chunk only)
#pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            const int k0 = col0 + 4 * i;
                            if (k0 + 4 > L) w[i] &= k0 >= L ? 0u : (0xFFFFFFFFu >> (32 - 8 * (L - k0)));
                        }
                    }
                    if (BULK) {  // units past L16 hold zeros (w is masked past L) or lie past ld (clipped)
                        *reinterpret_cast<uint4 *>(srow + (((2 * g) ^ (qr & 7)) << 4)) = make_uint4(w[0], w[1], w[2], w[3]);
                        *reinterpret_cast<uint4 *>(srow + (((2 * g + 1) ^ (qr & 7)) << 4)) =
                            col0 + 16 < L16 ? make_uint4(w[4], w[5], w[6], w[7]) : make_uint4(0, 0, 0, 0);
                    } else {
                        unsigned char *dst = OS + (size_t)qr * p.ld + col0;
                        *reinterpret_cast<uint4 *>(dst) = make_uint4(w[0], w[1], w[2], w[3]);
                        if (col0 + 16 < L16) *reinterpret_cast<uint4 *>(dst + 16) = make_uint4(w[4], w[5], w[6], w[7]);
                    }
                }
                if (BULK) fence_async_smem();  // the staging bytes are read by the tensor store
                tc_fence_before();
                __syncwarp();
                if (lane == 0) {
                    mbar_arrive(&sh.sempty[b]);  // this warp's part of buffer b is read
                    if (BULK) mbar_arrive(&sh.stfull[s]);
                }
            }
            // ---- (without BULK) the tile's rows to global memory (contiguous there): 16 bytes per
            //      thread and step, each warp's stores one contiguous 512-byte run.  Every epilogue
            //      thread reaches this barrier, which also tells each of them whether any gave up; the
            //      next tile's chunks are computed only after every epilogue warp has arrived on
            //      opsready again, so after these copies.
            if (!BULK) {
                uint32_t any_bad;
                asm volatile(
                    "{ .reg .pred pb, pa; setp.ne.u32 pb, %1, 0; bar.red.or.pred pa, 1, %2, pb; selp.u32 %0, 1, 0, pa; }"
                    : "=r"(any_bad)
                    : "r"((uint32_t)bad), "n"(QTHREADS)
                    : "memory");
                if (any_bad) break;
                const int64_t bytes = (int64_t)min(QM, L - r0) * p.ld;
                int8_t *gdst = p.out + ((size_t)bh * L + r0) * p.ld;
                for (int64_t x = 16 * (int64_t)tid; x < bytes; x += 16 * QTHREADS)
                    *reinterpret_cast<uint4 *>(gdst + x) = *reinterpret_cast<const uint4 *>(OS + x);
            } else if (bad) {
                break;
            }
        }
    } else if (warp == QMMA_WARP) {
        // ---------------- warp 16, lane 0: the operand copies (BULK) and the MMAs
        if (lane == 0) {
            // instruction descriptor: D f32, A/B f16 K-major, M = 128, N = n
            auto idesc = [](int n) -> uint32_t {
                return (1u << 4) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(QM >> 4) << 24);
            };
            auto copy_q = [&](int64_t tt) {
                const int bq = (int)(tt / tpb), rq = (int)(tt - (int64_t)bq * tpb) * QM;
                const uint32_t bytes = (uint32_t)(min(QM, L - rq) * p.ld_q);
                mbar_expect_tx(&sh.qload, bytes);
                bulk_g2s(QST, p.q + ((size_t)bq * L + rq) * p.ld_q, bytes, &sh.qload);
            };
            auto copy_k = [&](int bk) {
                const uint32_t bytes = (uint32_t)(L * p.ld_k);
                mbar_expect_tx(&sh.kload, bytes);
                bulk_g2s(KST, p.k + (size_t)bk * L * p.ld_k, bytes, &sh.kload);
            };
            // a copy is issued only once the operands it replaces were converted (opsready), so at
            // most one is in flight on each barrier
            uint32_t qiss = 0, kiss = 0, issued = 0, gc = 0;
            if (BULK && t_begin < t_end) {
                copy_q(t_begin);
                copy_k((int)(t_begin / tpb));
                qiss = kiss = 1;
            }
            bool ok = true;
            for (int64_t t = t_begin; t < t_end && ok; ++t) {
                ok = mbar_wait(&sh.opsready, (uint32_t)(t - t_begin) & 1, abort_flag);
                if (!ok) break;
                tc_fence_after();
                if (BULK && t + 1 < t_end) {  // the staging areas were converted: the next tile's operands
                    copy_q(t + 1);
                    ++qiss;
                    if ((int)((t + 1) / tpb) != (int)(t / tpb)) {
                        copy_k((int)((t + 1) / tpb));
                        ++kiss;
                    }
                }
                for (int c = 0; c < nch; ++c, ++gc) {
                    const uint32_t b = gc % QNBUF;
                    // the epilogue warps have read buffer b's previous chunk
                    if (gc >= (uint32_t)QNBUF && !mbar_wait(&sh.sempty[b], ((gc - QNBUF) / QNBUF) & 1, abort_flag)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const int n = min(QNC, L16 - c * QNC);
                    const uint32_t a0 = sa(QS), b0 = sa(KS) + (uint32_t)(c * QNC * QROW);
#pragma unroll
                    for (int s = 0; s < QKD / 16; ++s)
                        mma_f16_ss(tmem + b * QNC, smem_desc(a0 + 32 * s, 16, 1024), smem_desc(b0 + 32 * s, 16, 1024),
                                   idesc(n), s != 0);
                    mma_commit(&sh.sfull[b]);
                    ++issued;
                }
            }
            // every copy and every MMA issued has completed before shared and tensor memory are released
            if (BULK && qiss > 0) mbar_wait(&sh.qload, (qiss - 1) & 1, abort_flag, false);
            if (BULK && kiss > 0) mbar_wait(&sh.kload, (kiss - 1) & 1, abort_flag, false);
            if (issued > 0) {
                mma_commit(&sh.fin);
                mbar_wait(&sh.fin, 0, abort_flag, false);
            }
        }
    } else if (BULK && lane == 0) {
        // ---------------- warp 17, lane 0: the tensor stores of the chunks' staging buffers
        uint32_t gc = 0;
        bool ok = true;
        for (int64_t t = t_begin; t < t_end && ok; ++t) {
            const int bh = (int)(t / tpb);
            const int r0 = (int)(t - (int64_t)bh * tpb) * QM;
            for (int c = 0; c < nch; ++c, ++gc) {
                const uint32_t s = gc % QNST;
                ok = mbar_wait(&sh.stfull[s], (gc / QNST) & 1, abort_flag);
                if (!ok) break;
                // chunk c of the tile: columns c 128 .., rows r0 .., head bh
                asm volatile(
                    "cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%1, %2, %3}], [%4];" ::"l"(&tmap),
                    "r"(c * QNC), "r"(r0), "r"(bh), "r"(sa(OS + (size_t)s * QST_BYTES))
                    : "memory");
                asm volatile("cp.async.bulk.commit_group;" ::: "memory");
                asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");  // the buffer has been read
                mbar_arrive(&sh.stfree[s]);
            }
        }
        asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");  // every store has completed
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(QNBUF * QNC));
}

size_t qk_smem_bytes(int64_t ld, bool bulk)
{
    return 1024 + (size_t)QMAXL * QROW + (size_t)QM * QROW +
           (bulk ? (size_t)QNST * QST_BYTES + (size_t)QMAXL * 64 + QM * 64 : (size_t)QM * ld);
}

constexpr size_t kQkStaticSmem = sizeof(QkShared) + 64;

template <bool FOLD, bool BULK>
cudaError_t qk_launch(const QkParams &p, const CUtensorMap &tm, size_t smem, int grid, cudaStream_t st)
{
    cudaError_t e = check_smem_fits((const void *)qk_logits_tc_kernel<FOLD, BULK>, smem);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(qk_logits_tc_kernel<FOLD, BULK>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(qk_logits_tc_kernel<FOLD, BULK>, dim3(grid), dim3(QALL), smem, st, p, tm);
}

// The logits as a 3-d tensor [BH][L][ld] of bytes for the tensor stores: boxes of 128 x 128 x 1,
// 128-byte swizzle.  False when the driver's encoder is unavailable or rejects the shape.
bool logits_tensor_map(CUtensorMap *tm, int8_t *out, int64_t BH, int L, int64_t ld)
{
    static PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
    static bool tried = false;
    if (!tried) {
        tried = true;
        void *fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    if (!encode) return false;
    const cuuint64_t dims[3] = {(cuuint64_t)ld, (cuuint64_t)L, (cuuint64_t)BH};
    const cuuint64_t strides[2] = {(cuuint64_t)ld, (cuuint64_t)ld * (cuuint64_t)L};
    const cuuint32_t box[3] = {(cuuint32_t)QNC, (cuuint32_t)QM, 1};
    const cuuint32_t estr[3] = {1, 1, 1};
    return encode(tm, CU_TENSOR_MAP_DATA_TYPE_UINT8, 3, out, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                  CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Bulk copies of the operands (16-byte aligned rows of at most 64 bytes) and tensor stores of the
// output (rows and row strides of at least one 128 x 128 box)
bool qk_bulk(const QkArgs &a)
{
    return a.ld_q % 16 == 0 && a.ld_k % 16 == 0 && a.ld_q <= 64 && a.ld_k <= 64 && ((uintptr_t)a.q % 16) == 0 &&
           ((uintptr_t)a.k % 16) == 0 && a.L >= QM && a.ld_logit >= QNC &&
           qk_smem_bytes(a.ld_logit, true) + kQkStaticSmem <= 232448;
}

}  // namespace

bool qk_logits_supported(const QkArgs &a)
{
    return a.L >= 1 && a.L <= QMAXL && a.d >= 1 && a.d <= QKD && a.d % 8 == 0 && a.ld_q % 8 == 0 &&
           a.ld_k % 8 == 0 && a.ld_logit % 16 == 0 && ((uintptr_t)a.q % 8) == 0 && ((uintptr_t)a.k % 8) == 0 &&
           ((uintptr_t)a.logits % 16) == 0 && qk_smem_bytes(a.ld_logit, false) + kQkStaticSmem <= 232448;
}

cudaError_t launch_qk_logits(const QkArgs &a, cudaStream_t st)
{
    QkParams p{};
    p.q = a.q;
    p.k = a.k;
    p.ld_q = a.ld_q;
    p.ld_k = a.ld_k;
    p.zp_q = a.zp_q;
    p.zp_k = a.zp_k;
    p.out = a.logits;
    p.ld = a.ld_logit;
    p.BH = a.BH;
    p.L = a.L;
    p.d = a.d;
    p.n1 = a.n1;
    p.n2 = a.n2;
    p.zp_l = a.zp_l;
    // 32-bit epilogue: N1 >= 1 and |N2 P| + 2^(N1-1) + |zp_l| 2^N1 < 2^31 for every P the codes allow
    const double pmax = (double)a.d * (128.0 + std::fabs((double)a.zp_q)) * (128.0 + std::fabs((double)a.zp_k));
    const bool fold = a.n1 >= 1 && a.n1 <= 31 &&
                      (double)a.n2 * pmax + std::ldexp(1.0, a.n1 - 1) + std::fabs((double)a.zp_l) * std::ldexp(1.0, a.n1) <
                          2147483648.0;
    if (fold)
        p.c1 = (uint32_t)((1ull << (a.n1 - 1)) + ((uint64_t)(int64_t)a.zp_l << a.n1) -
                          (uint64_t)a.n2 * 0x4B400000ull);
    CUtensorMap tm;
    memset(&tm, 0, sizeof(tm));
    const bool bulk = qk_bulk(a) && logits_tensor_map(&tm, a.logits, a.BH, a.L, a.ld_logit);
    const size_t smem = qk_smem_bytes(a.ld_logit, bulk);
    const int64_t ntiles = a.BH * ((a.L + QM - 1) / QM);
    const int grid = (int)(ntiles < sm_count() ? ntiles : sm_count());
    if (bulk)
        return fold ? qk_launch<true, true>(p, tm, smem, grid, st) : qk_launch<false, true>(p, tm, smem, grid, st);
    return fold ? qk_launch<true, false>(p, tm, smem, grid, st) : qk_launch<false, false>(p, tm, smem, grid, st);
}

cudaError_t read_clear_qk_status(int *status)
{
    int zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(status, g_status, sizeof(int));
    if (e != cudaSuccess) return e;
    return cudaMemcpyToSymbol(g_status, &zero, sizeof(int));
}

}  // namespace fqvit
