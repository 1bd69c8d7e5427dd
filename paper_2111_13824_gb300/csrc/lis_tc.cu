// lis_tc.cu -- fused Log-Int-Softmax + BitShift attention times values on
// the 5th-generation tensor cores (tcgen05) of sm_103a.
//
// Eq. 15 is a matrix product: acc = P (V - zp_V) with P[i][j] = 2^(15 - code_ij),
// computed as P V - zp_V (P 1).  Every P entry and every int8 value of V is exact
// in fp16, and for codes made by Log-Int-Softmax sum_j 2^-code_j <= 3 + L 2^-15
// (2^-code < 1.5 / q_rev and q_rev >= S/e - 1/2), so with |V| <= 128 every
// partial sum of P V is an integer below 2^24, and the row sums P 1 (a second,
// N = 16 product against a block of ones, only when zp_V != 0) stay below 2^17:
// fp16 operands with fp32 accumulation give the integers exactly, and
// zp_V (P 1) is subtracted in int32.  The kernel evaluates the products as
// tcgen05.mma.kind::f16 (M = 128 query rows, N = 64 = d, K = 16 keys per
// instruction) with the accumulators in tensor memory.
//
// One CTA per SM walks (head, 128-row tile) work items.  Roles:
//   warps 0-15 (four threads per query row; warp w serves rows 32 (w % 4) ..
//     and the keys 16 (w / 4) .. +15 of every block of 64 keys): the tile's
//     logits go from shared memory into registers, the row maximum and the
//     i-exp row sum are combined over the four threads of a row through
//     shared memory, the row's 256 possible operands are tabulated, and every
//     4-bit code is written, as the fp16 operand 2^(15-code) looked up in that
//     table, straight into tensor memory (the A operand: row = lane, K-major
//     pairs per column).  The same threads convert a head's V rows to fp16
//     (128B-swizzled, MN-major shared-memory tile, the B operand).
//   warps 16-19 (one per tensor-memory lane quarter): read each tile's
//     accumulators out of tensor memory as soon as its MMAs complete and store
//     the int32 rows (32-byte stores) while the softmax warps work on the next
//     tile; warp 16, lane 0 also issues the tile's MMAs (four per key block)
//     once every operand is written, warp 17, lane 0 the bulk copy of the next
//     tile's logits into shared memory, plus L2 prefetches.
// Every wait is bounded: after two seconds the kernel records a timeout
// status, drains what it issued and returns (the host reads the status with
// fqvit_sync_status).
#include "fqvit_internal.cuh"
#include "lis_common.cuh"
#include "tc_common.cuh"

#include <cmath>
#include <cuda_fp16.h>

namespace fqvit {

namespace {

using namespace lis;
using namespace tc;

constexpr int TM = 128;        // query rows per tile (MMA M)
constexpr int TKB = 64;        // keys per key block
constexpr int TD = 64;         // head dimension (MMA N)
constexpr int TCOPIES = 32;    // replicas of the i-exp table (one per lane)
constexpr int B_SLOT = TKB * TD * 2;

struct TcParams {
    const int8_t *logits;
    int64_t ld;
    float s;
    const int8_t *v;
    int32_t *acc;
    int64_t BH;
    int L;
    int zp;  // zero point of V (acc = sum_j 2^(15-code) (V - zp))
    IexpC ic;  // Algorithm 1 constants of the scale
    uint8_t *out8;  // when not null: 8-bit outputs (requant8 with n1, n2, zp8) instead of acc
    int64_t ld_out8;
    int n1, n2, zp8;
};

constexpr int TPARTS = 4;                         // threads per query row
constexpr int TSOFT = TM * TPARTS;                // softmax threads (16 warps)
constexpr int TEPI_WARP = TSOFT / 32;             // warps 16..19: accumulator read-out, one per lane quarter
constexpr int TMMA_WARP = TEPI_WARP;              //   warp 16 lane 0 also issues the MMAs
constexpr int TCOPY_WARP = TEPI_WARP + 1;         //   warp 17 lane 0 also copies the logits tiles
constexpr int TTHREADS = TSOFT + 128;
constexpr int TMAXKB = 10;                        // key blocks of the longest row (L <= 640)
constexpr int TA_COL = TD;                        // D: columns 0..63; A of key block kb: 64 + 32 kb ..
// row sums of P (only when zp_V != 0): 16 columns after A
__host__ __device__ constexpr int tr_col(int nkb) { return TA_COL + 32 * nkb; }
constexpr int SCR_THR = 0;                        // the logits tile doubles as threshold scratch: int32 [16][TM]
constexpr int SCR_BYTES = 16 * TM * 4;

// tensor-memory columns for NKB key blocks (a power of two >= 32)
__host__ __device__ constexpr int tmem_cols(int nkb)
{
    return tr_col(nkb) + 16 <= 128 ? 128 : tr_col(nkb) + 16 <= 256 ? 256 : 512;
}

struct TcShared {
    uint64_t lload, lfree, afull, mmadone, fin;
    IexpC c;
    uint32_t tmem;
    int abort_flag;
    int rising;  // some i-exp value exceeds the one before it (floored constants)
    int stop;    // set (never cleared) by a softmax thread whose wait gave up
    int ew_stop; // the same for the read-out warps
};

// Named barrier 1 over the TSOFT softmax threads.  Every softmax thread reaches every one of
// these barriers (the waits before them are bounded), so they end.  bar.sync is warp-aligned:
// lanes of a row-dependent branch meet first.
__device__ __forceinline__ void soft_bar()
{
    __syncwarp();
    asm volatile("bar.sync 1, %0;" ::"n"(TSOFT) : "memory");
}

// i-exp value of byte J of w: table entry m - q of this lane's replica (lutq points at entry m)
template <int J>
__device__ __forceinline__ uint32_t iexp_at(const uint32_t *lutq, uint32_t w)
{
    return lutq[-TCOPIES * sbyte<J>(w)];
}
// Named barrier 2 over the 128 read-out threads
__device__ __forceinline__ void epi_bar()
{
    __syncwarp();
    asm volatile("bar.sync 2, 128;" ::: "memory");
}

// Per tile (128 query rows of one head):
//   copy (warp 17, lane 0): logits tile -> shared memory (bulk copy) once the previous tile's
//               table is built, L2 prefetch of the tile after it (and of the next head's V)
//   softmax:    thread (row r, part q) takes keys 64 kb + 16 q .. +15 of every key block into
//               registers; the row maximum and the i-exp row sum are combined over the four parts
//               through shared memory.  The row's operands go into a table indexed by the raw
//               logit byte: word j of row r (OT[j][r], so that the 32 rows of a warp sit in 32
//               different banks) holds, in byte b, 4 (30 - code) for the logit byte 4 j + b.
//               Codes only depend on the row maximum, the row sum and the logit, so one table
//               serves the whole row.  Where the i-exp values never rise with the distance d to
//               the maximum, code(d) = #{k <= 15 : d >= delta_k} for the row's thresholds delta_k
//               (the first d with e(d) D_k <= 2S): the four parts find them by binary search,
//               histogram them into the table words and turn each word into its codes with a
//               byte prefix sum (a multiply by 0x01010101); the floored constants of a few scales
//               break the monotony, and those evaluate every entry.  Every logit then costs one
//               table load; two loads and one byte permute give the fp16 pair 2^(15-code) that
//               goes to tensor memory (A, K-major rows = lanes) once the previous tile's MMAs are
//               done.  V of a head -> fp16 in shared memory (B, MN-major) whenever the head
//               changes.
//   MMA (warp 16, lane 0): after all operands of the tile are written, 4 MMAs per key block,
//               one commit
//   read-out (warps 16-19): the tile's accumulators, while the softmax warps work on the next
// Each CTA takes a contiguous range of tiles, so that consecutive tiles share a head.
// SMALL_E: every i-exp value is below 2^28 (decided on the host from the scale), so 16 of them
// sum exactly in 32 bits
template <int NKB, bool SMALL_E>
__global__ void __launch_bounds__(TTHREADS, 1) lis_attn_tc_kernel(TcParams p)
{
    extern __shared__ unsigned char dsm_raw[];
    __shared__ TcShared sh;
    __shared__ __align__(16) uint32_t OT[64 * TM];              // operand table: word j of row r at [j][r]
    __shared__ float LUTF[256];                                 // fp32 of the i-exp values (exact: <= 16 bits)
    __shared__ __align__(128) uint32_t ONES[128];               // 16 x 16 fp16 ones: B of the row sums of P
    unsigned char *base = dsm_raw + ((1024u - (sa(dsm_raw) & 1023u)) & 1023u);
    unsigned char *Bs = base;                                   // NKB x 8 KB
    uint32_t *LUT = (uint32_t *)(Bs + NKB * B_SLOT);            // 256 x TCOPIES
    int *red_max = (int *)(LUT + 256 * TCOPIES);                // TPARTS x TM
    unsigned long long *red_sum = (unsigned long long *)(red_max + TPARTS * TM);
    unsigned char *LG = (unsigned char *)(red_sum + TPARTS * TM);  // TM x ld logits, then scratch
    int *thr = (int *)(LG + SCR_THR);                           // 16 x TM: delta_k of each row

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    volatile int *abort_flag = &sh.abort_flag;
    volatile int *stop_flag = &sh.stop;
    pdl_release();
    if (tid == 0) {
        mbar_init(&sh.lload, 1);
        mbar_init(&sh.lfree, TSOFT);
        mbar_init(&sh.afull, TSOFT);
        mbar_init(&sh.mmadone, 1);
        mbar_init(&sh.fin, 1);
        sh.abort_flag = 0;
        sh.rising = 0;
        sh.stop = 0;
        sh.ew_stop = 0;
        sh.c = p.ic;
    }
    if (warp == TMMA_WARP) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(sa(&sh.tmem)),
                     "r"(tmem_cols(NKB)));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    __syncthreads();
    {
        const IexpC c = sh.c;
        for (int i = tid; i < 256 * TCOPIES; i += blockDim.x) LUT[i] = iexp_neg(i / TCOPIES, c);
        for (int d = tid; d < 256; d += blockDim.x) LUTF[d] = __uint2float_rn(iexp_neg(d, c));
        for (int i = tid; i < 128; i += blockDim.x) ONES[i] = 0x3C003C00u;
        for (int d = tid; d < 255; d += blockDim.x)
            if (iexp_neg(d, c) < iexp_neg(d + 1, c)) sh.rising = 1;
    }
    fence_async_smem();  // ONES is read by the MMAs
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sh.tmem;
    pdl_wait();  // the set-up above touched no global memory

    const int L = p.L;
    const int tpb = (L + TM - 1) / TM;
    const int64_t ntiles = p.BH * tpb;
    const int64_t t_begin = (int64_t)blockIdx.x * ntiles / gridDim.x;
    const int ncta_tiles = (int)((int64_t)(blockIdx.x + 1) * ntiles / gridDim.x - t_begin);
    // (head, first row) of tile t_begin; every role steps it by one tile per iteration
    const int bh_begin = (int)(t_begin / tpb);
    const int r0_begin = (int)(t_begin - (int64_t)bh_begin * tpb) * TM;

    if (tid < TSOFT) {
        const int r = tid & (TM - 1), q = tid >> 7;   // warp (q, r / 32): lanes = rows = TMEM lanes
        const int kk = tid >> 3, ci = tid & 7;        // V conversion: key kk of a block, values 8 ci .. +7
        const uint32_t lut_lane = sa(LUT) + 4u * (uint32_t)lane;
        const uint32_t r4 = 4u * (uint32_t)r;
        const unsigned char *otb = reinterpret_cast<const unsigned char *>(OT);
        const uint32_t tlane = tmem + ((uint32_t)((warp & 3) * 32) << 16);
        const bool monotone = !sh.rising;            // codes never fall as d grows
        const int xs = (int)(int8_t)(uint8_t)(64 * q);  // part q's table words 16 q .. +15: logits xs .. xs + 63
        int npad = 0;  // keys at or past L inside this part's last partial block (summed as -128, then removed)
#pragma unroll
        for (int kb = 0; kb < NKB; ++kb) {
            const int k0 = kb * TKB + 16 * q;
            if (k0 < L && k0 + 16 > L) npad = k0 + 16 - L;
        }
        int it = 0;
        bool wait_bad = false;
        int conv_bh = -1;
        int bh = bh_begin;
        int r0 = r0_begin;
        for (; it < ncta_tiles; ++it, r0 = r0 + TM < L ? r0 + TM : (++bh, 0)) {
            const int row = r0 + r;
            const bool valid = row < L;
            const bool lbad = !mbar_wait_warp(&sh.lload, it & 1, abort_flag);
            const unsigned char *lr = LG + (size_t)r * p.ld + 16 * q;
            uint4 w[NKB];
#pragma unroll
            for (int kb = 0; kb < NKB; ++kb) {
                const int k0 = kb * TKB + 16 * q;
                w[kb] = (valid && k0 < L) ? *reinterpret_cast<const uint4 *>(lr + kb * TKB)
                                          : make_uint4(0x80808080u, 0x80808080u, 0x80808080u, 0x80808080u);
                if (valid && k0 < L && k0 + 16 > L) {  // keys at or past L: -128 (no effect on the max)
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
            // ---- row maximum over the four parts
            // signed 16-bit lanes: the high byte of the larger lane is the larger byte, so lanes of w
            // carry bytes 1 and 3 and lanes of w << 8 bytes 0 and 2
            uint32_t mo = 0x80008000u, me = 0x80008000u;
#pragma unroll
            for (int kb = 0; kb < NKB; ++kb) {
                mo = vmax16x2(vmax16x2(mo, w[kb].x), vmax16x2(w[kb].y, vmax16x2(w[kb].z, w[kb].w)));
                me = vmax16x2(vmax16x2(me, w[kb].x << 8), vmax16x2(w[kb].y << 8, vmax16x2(w[kb].z << 8, w[kb].w << 8)));
            }
            int m = max(max(sbyte<1>(mo), sbyte<3>(mo)), max(sbyte<1>(me), sbyte<3>(me)));
            red_max[q * TM + r] = m;
            if (lbad || wait_bad) *stop_flag = 1;
            soft_bar();
            if (*stop_flag) break;  // every softmax thread leaves here together
            m = max(max(red_max[r], red_max[TM + r]), max(red_max[2 * TM + r], red_max[3 * TM + r]));
            // ---- i-exp row sum over the four parts
            const uint32_t *lutq = LUT + lane + m * TCOPIES;
            unsigned long long S = 0;
            if (valid) {
#pragma unroll
                for (int kb = 0; kb < NKB; ++kb) {
                    if (kb * TKB + 16 * q < L) {
                        const uint32_t ww[4] = {w[kb].x, w[kb].y, w[kb].z, w[kb].w};
                        if (SMALL_E) {  // 16 values below 2^28: a 32-bit partial sum is exact
                            uint32_t a = 0;
#pragma unroll
                            for (int b = 0; b < 4; ++b) {
                                a += iexp_at<0>(lutq, ww[b]) + iexp_at<1>(lutq, ww[b]);
                                a += iexp_at<2>(lutq, ww[b]) + iexp_at<3>(lutq, ww[b]);
                            }
                            S += a;
                        } else {
#pragma unroll
                            for (int b = 0; b < 4; ++b) {
                                const uint32_t e0 = iexp_at<0>(lutq, ww[b]), e1 = iexp_at<1>(lutq, ww[b]);
                                const uint32_t e2 = iexp_at<2>(lutq, ww[b]), e3 = iexp_at<3>(lutq, ww[b]);
                                S += (unsigned long long)(e0 + e1) + (unsigned long long)(e2 + e3);  // e < 2^31
                            }
                        }
                    }
                }
                S -= (unsigned long long)npad * lutq[128 * TCOPIES];  // the padding bytes, -128 each
            }
            red_sum[q * TM + r] = S;
            // the table words of the previous tile are dead: clear this part's words for the histogram
            if (valid && monotone) {
#pragma unroll
                for (int i = 0; i < 16; ++i) OT[(16 * q + i) * TM + r] = 0u;
            }
            soft_bar();
            S = red_sum[r] + red_sum[TM + r] + red_sum[2 * TM + r] + red_sum[3 * TM + r];
            const RowSum rs = split_2s(S);
            // ---- this row's thresholds: part q finds delta_k for k = q + 1, q + 5, q + 9, q + 13,
            //      the four binary searches interleaved
            if (valid && monotone) {
                float Dk[4];
                int lo[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int k = q + 1 + 4 * i;
                    Dk[i] = k == 1 ? 3.0f : (float)(3 * (1 << (min(k, 15) - 1)) - 1);
                    lo[i] = 0;
                }
                // e(d) D_k <= 2S, exact: one rounding of an exact product minus hi, against lo
                auto hit = [&](int d, float D) -> bool { return __fmaf_rn(LUTF[d], D, -rs.hi) <= rs.lo; };
#pragma unroll
                for (int step = 128; step >= 1; step >>= 1)
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        if (!hit(lo[i] + step - 1, Dk[i])) lo[i] += step;
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int k = q + 1 + 4 * i;
                    if (lo[i] == 255 && !hit(255, Dk[i])) lo[i] = 256;
                    if (k <= 15) thr[(k - 1) * TM + r] = lo[i];
                }
            }
            soft_bar();
            // ---- this row's operand table
            if (valid) {
                if (monotone) {
                    // E(x) = 30 - code(x) = 15 + #{k : m - delta_k < x}.  Histogram of the thresholds
                    // m - delta_k over this part's logits (byte x - xs of the words), counting those
                    // below xs, then per word the exclusive byte prefix sum.
                    int n = 0;
#pragma unroll
                    for (int k = 0; k < 15; ++k) {
                        const int t = m - thr[k * TM + r] - xs;
                        n += t < 0 ? 1 : 0;
                        if ((unsigned)t < 64u) OT[(16 * q + (t >> 2)) * TM + r] += 1u << (8 * (t & 3));
                    }
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        uint32_t *wp = &OT[(16 * q + i) * TM + r];
                        const uint32_t h = *wp;
                        *wp = 0x3C3C3C3Cu + 4u * ((uint32_t)n * 0x01010101u + (h << 8) * 0x01010101u);
                        n += (int)((h * 0x01010101u) >> 24);
                    }
                } else {
                    auto E_at = [&](int x) -> uint32_t {
                        return operand_exp(lds32(lut_lane + (uint32_t)((m - x) * (TCOPIES * 4))), rs.hibits, rs.hi, rs.lo);
                    };
#pragma unroll 2
                    for (int i = 0; i < 16; ++i) {
                        const int j = q + 4 * i;
                        const int xlo = (int)(int8_t)(uint8_t)(4 * j);  // logits of word j: xlo .. xlo + 3
                        if (xlo > m) continue;                          // no key of this row reads it
                        const int hb = min(3, m - xlo);                 // bytes above hb exceed the maximum
                        const uint32_t E0 = E_at(xlo);
                        const uint32_t E1 = hb >= 1 ? E_at(xlo + 1) : E0;
                        const uint32_t E2 = hb >= 2 ? E_at(xlo + 2) : E1;
                        const uint32_t E3 = hb >= 3 ? E_at(xlo + 3) : E2;
                        OT[j * TM + r] = 4u * (E0 | (E1 << 8) | (E2 << 16) | (E3 << 24));
                    }
                }
            }
            soft_bar();
            mbar_arrive(&sh.lfree);  // the logits tile and its scratch are free: the next tile may load
            // the previous tile's MMAs have read A and B: they may be rewritten
            if (it > 0 && !mbar_wait_warp(&sh.mmadone, (it - 1) & 1, abort_flag)) {
                wait_bad = true;  // the next tile's first barrier ends the loop for all
                continue;
            }
            // ---- V of a new head -> fp16 B
            if (bh != conv_bh) {
#pragma unroll
                for (int kb = 0; kb < NKB; ++kb) {
                    const int key = kb * TKB + kk;
                    uint4 v4 = make_uint4(0, 0, 0, 0);
                    if (key < L) {
                        const uint2 vw = __ldg(reinterpret_cast<const uint2 *>(p.v + ((size_t)bh * L + key) * TD + 8 * ci));
                        const uint32_t x0 = vw.x ^ 0x80808080u, x1 = vw.y ^ 0x80808080u;
                        v4.x = i8x2_to_h2(x0, 0x5140);
                        v4.y = i8x2_to_h2(x0, 0x7362);
                        v4.z = i8x2_to_h2(x1, 0x5140);
                        v4.w = i8x2_to_h2(x1, 0x7362);
                    }
                    *reinterpret_cast<uint4 *>(Bs + kb * B_SLOT + kk * 128 + ((ci ^ (kk & 7)) << 4)) = v4;
                }
                conv_bh = bh;
            }
            // ---- operands of this row's keys -> tensor memory
#pragma unroll
            for (int kb = 0; kb < NKB; ++kb) {
                const int k0 = kb * TKB + 16 * q;
                uint32_t o[8] = {0, 0, 0, 0, 0, 0, 0, 0};
                if (valid && k0 < L) {
                    const uint32_t ww[4] = {w[kb].x, w[kb].y, w[kb].z, w[kb].w};
#pragma unroll
                    for (int b = 0; b < 4; ++b) {
                        const uint32_t v = ww[b];
                        // word (byte >> 2) of this row, then byte (byte & 3) of it into the high byte
                        // of each fp16 half; the low bytes copy the sign of a table byte (zero)
                        const uint32_t t0 = *reinterpret_cast<const uint32_t *>(otb + (((v << 7) & 0x7E00u) | r4));
                        const uint32_t t1 = *reinterpret_cast<const uint32_t *>(otb + (((v >> 1) & 0x7E00u) | r4));
                        const uint32_t t2 = *reinterpret_cast<const uint32_t *>(otb + (((v >> 9) & 0x7E00u) | r4));
                        const uint32_t t3 = *reinterpret_cast<const uint32_t *>(otb + (((v >> 17) & 0x7E00u) | r4));
                        o[2 * b] = prmt(t0, t1, ((v << 4) & 0x3030u) | 0x4808u);
                        o[2 * b + 1] = prmt(t2, t3, ((v >> 12) & 0x3030u) | 0x4808u);
                    }
                    if (k0 + 16 > L) {  // keys at or past L get a zero operand
                        const int n = L - k0;
#pragma unroll
                        for (int c = 0; c < 8; ++c) {
                            if (2 * c >= n)
                                o[c] = 0;
                            else if (2 * c + 1 == n)
                                o[c] &= 0xFFFFu;
                        }
                    }
                }
                tmem_st8(tlane + TA_COL + 32 * kb + 8 * q, o);
            }
            __syncwarp();
            asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
            tc_fence_before();
            fence_async_smem();
            mbar_arrive(&sh.afull);
        }
    } else {
        // ---------------- read-out warps (lane quarter eq), with the MMA issue and the logits copies
        const int eq = warp & 3;
        const uint32_t etl = tmem + ((uint32_t)(eq * 32) << 16);
        volatile int *ew_stop = &sh.ew_stop;
        const int nkb = (L + TKB - 1) / TKB;
        int bh = bh_begin;
        int r0 = r0_begin;
        if (warp == TCOPY_WARP && lane == 0) {
            prefetch_l2(p.v + (size_t)bh * L * TD, (uint32_t)(L * TD));
            const uint32_t bl = (uint32_t)(min(TM, L - r0) * p.ld);
            mbar_expect_tx(&sh.lload, bl);
            bulk_g2s(LG, p.logits + ((size_t)bh * L + r0) * p.ld, bl, &sh.lload);
        }
        for (int it = 0; it < ncta_tiles; ++it, r0 = r0 + TM < L ? r0 + TM : (++bh, 0)) {
            if (warp == TCOPY_WARP && lane == 0 && it + 1 < ncta_tiles) {
                // the next tile's logits as soon as this tile's table is built
                const int bhn = r0 + TM < L ? bh : bh + 1;
                const int r0n = r0 + TM < L ? r0 + TM : 0;
                if (mbar_wait(&sh.lfree, it & 1, abort_flag)) {
                    const uint32_t bl = (uint32_t)(min(TM, L - r0n) * p.ld);
                    mbar_expect_tx(&sh.lload, bl);
                    bulk_g2s(LG, p.logits + ((size_t)bhn * L + r0n) * p.ld, bl, &sh.lload);
                    if (bhn != bh) prefetch_l2(p.v + (size_t)bhn * L * TD, (uint32_t)(L * TD));
                    if (it + 2 < ncta_tiles) {
                        const int r0m = r0n + TM < L ? r0n + TM : 0;
                        const int bhm = r0n + TM < L ? bhn : bhn + 1;
                        prefetch_l2(p.logits + ((size_t)bhm * L + r0m) * p.ld, (uint32_t)(min(TM, L - r0m) * p.ld));
                    }
                }
            }
            if (warp == TMMA_WARP && lane == 0) {
                // this tile's MMAs once its operands are in place
                if (mbar_wait(&sh.afull, it & 1, abort_flag)) {
                    tc_fence_after();
                    const uint32_t b0 = sa(Bs);
                    const uint64_t ones = smem_desc_plain(sa(ONES), 128, 256);
                    if (p.zp == 0) {
                        for (int kb = 0; kb < nkb; ++kb)
#pragma unroll
                            for (int s = 0; s < TKB / 16; ++s)
                                mma_f16_ta(tmem, tmem + TA_COL + 32 * kb + 8 * s,
                                           smem_desc(b0 + kb * B_SLOT + 2048 * s, 1024, 1024), (kb | s) != 0);
                    } else {
                        for (int kb = 0; kb < nkb; ++kb)
#pragma unroll
                            for (int s = 0; s < TKB / 16; ++s) {
                                mma_f16_ta(tmem, tmem + TA_COL + 32 * kb + 8 * s,
                                           smem_desc(b0 + kb * B_SLOT + 2048 * s, 1024, 1024), (kb | s) != 0);
                                mma_f16_ta(tmem + tr_col(NKB), tmem + TA_COL + 32 * kb + 8 * s, ones,
                                           (kb | s) != 0, kIdescOnes);
                            }
                    }
                    mma_commit(&sh.mmadone);
                }
            }
            // this tile's accumulators: row 32 eq + lane of the tile, 64 columns in two halves
            const bool ok = mbar_wait_warp(&sh.mmadone, it & 1, abort_flag);
            if (ok) {
                tc_fence_after();
                const int row = r0 + 32 * eq + lane;
                int32_t *dst = p.out8 ? nullptr : p.acc + ((size_t)bh * L + row) * TD;
                // zp (sum_j 2^(15-code_j)), an exact integer below 2^24 times |zp| <= 255
                int zsum = 0;
                if (p.zp != 0) {
                    uint32_t rs;
                    tmem_ld1(etl + tr_col(NKB), rs);
                    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
                    zsum = p.zp * __float2int_rn(__uint_as_float(rs));
                }
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    uint32_t va[32];
                    tmem_ld32(etl + 32 * h, va);
                    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
                    if (row < L && p.out8) {  // 8-bit outputs: 32 bytes of this half of the row
                        uint32_t wq[8];
#pragma unroll
                        for (int c = 0; c < 8; ++c) {
                            wq[c] = 0;
#pragma unroll
                            for (int k = 0; k < 4; ++k)
                                wq[c] |= requant8(__float2int_rn(__uint_as_float(va[4 * c + k])) - zsum, p.n1, p.n2,
                                                  p.zp8) << (8 * k);
                        }
                        uint4 *d8 = reinterpret_cast<uint4 *>(p.out8 + ((size_t)bh * L + row) * p.ld_out8 + 32 * h);
                        d8[0] = make_uint4(wq[0], wq[1], wq[2], wq[3]);
                        d8[1] = make_uint4(wq[4], wq[5], wq[6], wq[7]);
                    } else if (row < L) {
#pragma unroll
                        for (int c = 0; c < 4; ++c) {
                            int v8[8];
#pragma unroll
                            for (int j = 0; j < 8; ++j)
                                v8[j] = __float2int_rn(__uint_as_float(va[8 * c + j])) - zsum;
                            stg256(dst + 32 * h + 8 * c, v8);
                        }
                    }
                }
            }
            tc_fence_before();
            if (!ok) *ew_stop = 1;
            epi_bar();  // all four quarters have read D: the next tile's MMAs may overwrite it
            if (*ew_stop) break;
        }
        if (warp == TCOPY_WARP && lane == 0) mbar_wait(&sh.lload, (ncta_tiles - 1) & 1, abort_flag, false);
        if (warp == TMMA_WARP && lane == 0) {  // every MMA issued has completed before tensor memory is freed
            mma_commit(&sh.fin);
            mbar_wait(&sh.fin, 0, abort_flag, false);
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == TMMA_WARP)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(tmem_cols(NKB)));
}

size_t tc_smem_bytes(int L, int64_t ld)
{
    const int nkb = (L + TKB - 1) / TKB;
    const size_t lg = (size_t)TM * ld > (size_t)SCR_BYTES ? (size_t)TM * ld : (size_t)SCR_BYTES;
    return 1024 + (size_t)nkb * B_SLOT + (size_t)256 * TCOPIES * 4 + (size_t)TPARTS * TM * (4 + 8) + lg;
}

// static shared memory of the kernel: the operand table, the fp32 i-exp table, the control block
constexpr size_t kTcStaticSmem = (size_t)64 * TM * 4 + 1024 + 512 + 256;

template <int NKB, bool SMALL_E>
cudaError_t tc_launch(const TcParams &p, size_t smem, int grid, cudaStream_t st)
{
    cudaError_t e = cudaFuncSetAttribute(lis_attn_tc_kernel<NKB, SMALL_E>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(lis_attn_tc_kernel<NKB, SMALL_E>, dim3(grid), dim3(TTHREADS), smem, st, p);
}

template <int NKB>
cudaError_t tc_launch_e(bool small_e, const TcParams &p, size_t smem, int grid, cudaStream_t st)
{
    return small_e ? tc_launch<NKB, true>(p, smem, grid, st) : tc_launch<NKB, false>(p, smem, grid, st);
}

// Whether every i-exp value of the scale is below 2^28: the largest is e(0) = (q_b^2 + q_c) 2^15.
bool small_iexp(const IexpC &c) { return ((double)c.q_b * c.q_b + c.q_c) * 32768.0 < 268435456.0; }

}  // namespace

bool lis_attention_tc_eligible(const LisArgs &a, const AttnVArgs &b)
{
    const bool out_ok = b.out8 ? (b.ld_out8 % 16 == 0 && ((uintptr_t)b.out8 % 16) == 0)
                               : (b.ld_acc == TD && ((uintptr_t)b.acc % 32) == 0);
    return b.d == TD && a.bias == nullptr && a.region == nullptr && a.codes == nullptr && a.L <= TMAXKB * TKB &&
           a.ld_logit % 16 == 0 && b.ld_v == TD && out_ok && ((uintptr_t)a.logits % 16) == 0 &&
           ((uintptr_t)b.v % 16) == 0 && tc_smem_bytes(a.L, a.ld_logit) + kTcStaticSmem <= 232448;
}

cudaError_t launch_lis_attention_tc(const LisArgs &a, const AttnVArgs &b, cudaStream_t st)
{
    if (lis_attention_tc_packed(a.L)) return launch_lis_attention_tc_packed(a, b, st);  // lis_tc_pack.cu
    TcParams p{a.logits, a.ld_logit, a.s_logit, b.v, b.acc, b.BH, a.L, b.zp_v, iexp_consts_host(a.s_logit),
               b.out8, b.ld_out8, b.rq_n1, b.rq_n2, b.rq_zp};
    const size_t smem = tc_smem_bytes(a.L, a.ld_logit);
    const int64_t ntiles = b.BH * ((a.L + TM - 1) / TM);
    const int grid = (int)(ntiles < sm_count() ? ntiles : sm_count());
    const bool se = small_iexp(p.ic);
    switch ((a.L + TKB - 1) / TKB) {
    case 1: return tc_launch_e<1>(se, p, smem, grid, st);
    case 2: return tc_launch_e<2>(se, p, smem, grid, st);
    case 3: return tc_launch_e<3>(se, p, smem, grid, st);
    case 4: return tc_launch_e<4>(se, p, smem, grid, st);
    case 5: return tc_launch_e<5>(se, p, smem, grid, st);
    case 6: return tc_launch_e<6>(se, p, smem, grid, st);
    case 7: return tc_launch_e<7>(se, p, smem, grid, st);
    case 8: return tc_launch_e<8>(se, p, smem, grid, st);
    case 9: return tc_launch_e<9>(se, p, smem, grid, st);
    default: return tc_launch_e<10>(se, p, smem, grid, st);
    }
}

cudaError_t read_clear_device_status(int *status, cudaStream_t st)
{
    int zero = 0;
    cudaError_t e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return e;
    e = cudaMemcpyFromSymbol(status, g_status, sizeof(int));
    if (e != cudaSuccess) return e;
    e = cudaMemcpyToSymbol(g_status, &zero, sizeof(int));
    if (e != cudaSuccess) return e;
    int wst = 0;
    e = read_clear_win_status(&wst);
    if (e != cudaSuccess) return e;
    if (*status == 0) *status = wst;
    int qst = 0;
    e = read_clear_qk_status(&qst);
    if (e != cudaSuccess) return e;
    if (*status == 0) *status = qst;
    int pst = 0;
    e = read_clear_tcp_status(&pst);
    if (*status == 0) *status = pst;
    return e;
}

}  // namespace fqvit
