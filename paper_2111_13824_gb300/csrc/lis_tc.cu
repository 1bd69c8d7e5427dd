// lis_tc.cu -- fused Log-Int-Softmax + BitShift attention times values on
// the 5th-generation tensor cores (tcgen05) of sm_103a, for rows of 65 .. 592
// keys (head dimension 64; the longest rows its shared-memory layout holds).
//
// Eq. 15 is a matrix product: acc = P (V - zp_V) with P[i][j] = 2^(15 - code_ij),
// computed as P V - zp_V (P 1).  Every P entry and every int8 value of V is exact
// in fp16, and for codes made by Log-Int-Softmax sum_j 2^-code_j <= 3 + L 2^-15
// (2^-code < 1.5 / q_rev and q_rev >= S/e - 1/2), so with |V| <= 128 every
// partial sum of P V is an integer below 2^24, and the row sums P 1 (a second,
// N = 16 product against a block of ones, only when zp_V != 0) stay below 2^17:
// fp16 operands with fp32 accumulation give the integers exactly, and
// zp_V (P 1) is subtracted in int32.  The products run as
// tcgen05.mma.kind::f16 (M = 128 query rows, N = 64 = d, K = 16 keys per
// instruction) with the operand P and the accumulators in tensor memory.
//
// One CTA per SM walks a contiguous range of 128-row tiles.  Without PACK a
// tile holds rows of one head (the last tile of a head is partly empty); with
// PACK (128 <= L <= 384) tile t holds rows 128 t .. 128 t + 127 of all BH L
// rows, so it may hold the end of one head and the start of the next: those
// run two sets of MMAs, one per head, against two V buffers into two
// accumulators.
//
// Roles:
//   warps 0-15, the softmax threads, four per query row (thread (r, q): warp
//     4 q + r / 32, lane r % 32, so that lanes are rows are tensor-memory
//     lanes; part q takes keys 64 kb + 16 q .. +15 of every 64-key block kb).
//     Per tile: the row's logits from the bulk-copied tile into registers, the
//     row maximum, then every logit byte becomes its distance d = m - q to the
//     maximum (four at once: a borrow-free 32-bit subtraction of the biased
//     bytes from the replicated maximum), the i-exp row sum from a table
//     indexed by d, the row's 15 code thresholds, the row's operand table (the
//     fp16 operand 2^(15 - code) of every d), and the operands of the row's
//     keys, looked up by d, straight into tensor memory.
//   warps 16-19, one per tensor-memory lane quarter: the accumulators of the
//     previous tile out of tensor memory into global memory, V of a new head
//     into the fp16 B operand in shared memory, the tile's MMAs (warp 16, lane
//     0) and the bulk copy of the next tile's logits (warp 17, lane 0).
//
// The combined table (64 KB at the absolute shared-memory address 64 K): line d
// (d = 0 .. 255) is 256 bytes.  Bytes 0 .. 127 hold the high byte 4 (30 - code)
// of the operand of distance d for the 128 rows of the tile, row r at byte
// 4 (r % 32) + r / 32, so that the 32 rows of a warp read 32 different banks;
// bytes 128 .. 255 hold 32 copies of the i-exp value e(d), copy c at byte
// 128 + 4 c (lane c reads its own copy: no bank conflicts for random d).  One
// byte permute turns a distance byte and a per-thread register into the full
// address 64 K | d << 8 | offset, so a table lookup costs one permute and one
// load.
//
// The operand table from thresholds: code(d) = #{k <= 15 : d >= delta_k} with
// delta_k the first d at which e(d) D_k <= 2S (D_1 = 3, D_k = 3 2^(k-1) - 1,
// an exact FMA test against 2S = hi + lo), where the i-exp values never rise
// with d.  The four parts of a row find its thresholds by binary search and
// add one, in byte r / 32 of the table word (line delta_k, lane r % 32), with a
// shared-memory atomic; then thread (lane l, warp g) turns lines 16 g .. 16 g +
// 15 of column l into codes by a running sum (four rows per word, counts
// below 16 per byte: no carries), the carry-in from the lines below taken from
// per-group totals counted at the same time.  The floored constants of a few
// scales make e(d) rise at band edges; those scales evaluate every entry
// directly with the code test.
//
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

constexpr int TM = 128;                    // query rows per tile (MMA M)
constexpr int TKB = 64;                    // keys per key block
constexpr int TD = 64;                     // head dimension (MMA N)
constexpr int TPARTS = 4;                  // threads per query row
constexpr int TSOFT = TM * TPARTS;         // softmax threads (16 warps)
constexpr int TEPI_WARP = TSOFT / 32;      // warps 16..19: read-out, one per lane quarter
constexpr int TMMA_WARP = TEPI_WARP;       //   warp 16 lane 0 also issues the MMAs
constexpr int TCOPY_WARP = TEPI_WARP + 1;  //   warp 17 lane 0 also copies the logits tiles
constexpr int TTHREADS = TSOFT + 128;
constexpr int TMAXKB = 10;                 // key blocks of the longest row
constexpr int kPackMaxBlocks = 6;          // PACK for 128 <= L <= 384

// Shared memory.  The kernel has no static shared memory, so its dynamic shared memory starts at
// the first address after the 1 KB the driver reserves (1024; the kernel checks it).  The combined
// table sits at the absolute address 64 K, so that one byte permute of a distance byte and a per-thread
// register holding (1 << 16 | byte offset) gives the full shared-memory address of a lookup (no add).
// Region A, from the start up to 64 K: the control area, then as many 2 KB B blocks (16 keys of V in
// fp16 each) as fit; region C, from 128 K on: the remaining B blocks, then the logits tile.
constexpr uint32_t kTabAbs = 0x10000;
constexpr uint32_t LUT_BYTE = 128;                    // i-exp copies in a table line
// control area (offsets from the start of dynamic shared memory)
constexpr uint32_t C_SH = 0;                          // TcShared
constexpr uint32_t C_ONES = 256;                      // 16 x 16 fp16 ones: B of the row sums of P
constexpr uint32_t C_LUTF = 1024;                     // fp32 of the i-exp values (exact: <= 16 bits)
constexpr uint32_t C_RMAX = 2048;                     // int [4][128]: row maxima of the parts
constexpr uint32_t C_RSUM = 4096;                     // u64 [4][128]: row sums of the parts
constexpr uint32_t C_GT = 8192;                       // u32 [32][20]: thresholds per (lane, 16-line group)
constexpr int GT_LD = 20;                             //   (row stride 20 words: 16-byte loads without conflicts)
constexpr uint32_t C_BK = C_GT + 32 * GT_LD * 4;      // u16 [1024] threshold buckets, or {hi, lo, hibits} [128]
                                                      //   of the rows (scales whose i-exp values rise)
constexpr uint32_t C_END = C_BK + 2048;
constexpr uint32_t kBlk = 16 * 64 * 2;                // one B block: 16 keys x 64 values, fp16
constexpr uint32_t kSmemOptin = 232448;               // dynamic shared memory a CTA may have

struct TcLayout {
    uint32_t tab;  // offset of the table (absolute kTabAbs)
    uint32_t bA;   // offset of the first B block of region A (1024-aligned address)
    int nA;        // B blocks in region A
    uint32_t bC;   // offset of region C (absolute 2 kTabAbs)
    uint32_t lg;   // offset of the logits tile
    uint32_t need; // dynamic bytes the layout spans
    bool fits;
};

// Layout for dynamic shared memory at absolute address base (a multiple of 1024), nblocks B blocks and a
// logits tile of lg_bytes
__host__ __device__ inline TcLayout tc_layout(uint32_t base, int nblocks, uint32_t lg_bytes)
{
    TcLayout l;
    l.fits = base + C_END <= kTabAbs;
    l.tab = kTabAbs - base;
    const uint32_t a0 = (base + C_END + 1023u) & ~1023u;
    const int navail = a0 < kTabAbs ? (int)((kTabAbs - a0) / kBlk) : 0;
    l.nA = navail < nblocks ? navail : nblocks;
    l.bA = a0 - base;
    l.bC = 2 * kTabAbs - base;
    l.lg = l.bC + (uint32_t)(nblocks - l.nA) * kBlk;
    l.need = l.lg + lg_bytes;
    l.fits = l.fits && l.need <= kSmemOptin;
    return l;
}

// Threshold buckets.  delta_k = #{d : e(d) > T} with T = 2S / D_k (i-exp values never rising with d).
// T is approximated by T' = fp32(fp32(2S) * fp32(1 / D_k)), within 2^-22 of T; the bucket of T' (its
// fp32 bits without the low 17, 64 buckets per octave) gives delta_k within [lo, lo + span]: lo counts
// the values above the bucket's upper edge (raised by 2^-20), lo + span those above its lower edge
// (lowered by 2^-20).  The exact test e(d) D_k <= 2S then settles the span by binary search (one probe
// at usual scales).  Buckets cover 16 octaves below e(0); above them delta_k = 0, below them (T under
// the smallest value e(0) 2^-15) delta_k = 256.
constexpr int BK_SHIFT = 17;
constexpr int BK_N = 1024;

// D_k and fp32 1 / D_k for k = 1 .. 15 (D_1 = 3, D_k = 3 2^(k-1) - 1)
__constant__ float kD[16] = {0.0f,    3.0f,    5.0f,    11.0f,   23.0f,   47.0f,    95.0f,    191.0f,
                             383.0f,  767.0f,  1535.0f, 3071.0f, 6143.0f, 12287.0f, 24575.0f, 49151.0f};
__constant__ float kRcpD[16] = {0.0f,          1.0f / 3.0f,     1.0f / 5.0f,     1.0f / 11.0f,
                                1.0f / 23.0f,  1.0f / 47.0f,    1.0f / 95.0f,    1.0f / 191.0f,
                                1.0f / 383.0f, 1.0f / 767.0f,   1.0f / 1535.0f,  1.0f / 3071.0f,
                                1.0f / 6143.0f, 1.0f / 12287.0f, 1.0f / 24575.0f, 1.0f / 49151.0f};

// tensor memory: D at 0 (PACK: the second head's D at 64), the operands P from ta_col on (8 columns
// per 16 keys), then the row sums of P (zp_V != 0), 16 columns
__host__ __device__ constexpr int ta_col(bool pack) { return pack ? 2 * TD : TD; }
__host__ __device__ constexpr int tr_col(int nkb, bool pack) { return ta_col(pack) + 32 * nkb; }
__host__ __device__ constexpr int tmem_cols(int nkb, bool pack)
{
    return tr_col(nkb, pack) + 16 <= 128 ? 128 : tr_col(nkb, pack) + 16 <= 256 ? 256 : 512;
}

struct TcParams {
    const int8_t *logits;
    int64_t ld;
    const int8_t *v;
    int32_t *acc;
    int64_t BH;
    int L;
    int zp;    // zero point of V (acc = sum_j 2^(15-code) (V - zp))
    IexpC ic;  // Algorithm 1 constants of the scale
    uint8_t *out8;  // when not null: 8-bit outputs (requant8 with n1, n2, zp8) instead of acc
    int64_t ld_out8;
    int n1, n2, zp8;
    uint32_t smem;  // dynamic shared memory of the launch
};

// A tile: rows g0 .. g0 + rows - 1 of the [BH * L] logit rows; the first nsplit belong to head h0,
// the rest (PACK only) to head h0 + 1.
struct TileInfo {
    int64_t g0;
    int rows, h0, nsplit;
};

template <bool PACK>
__device__ __forceinline__ TileInfo tile_info(int64_t t, int L, int64_t BH, int tpb)
{
    TileInfo ti;
    if (PACK) {
        ti.g0 = t * TM;
        ti.rows = (int)min((int64_t)TM, BH * L - ti.g0);
        ti.h0 = (int)(ti.g0 / L);
        ti.nsplit = (int)min((int64_t)ti.rows, (int64_t)(ti.h0 + 1) * L - ti.g0);
    } else {
        ti.h0 = (int)(t / tpb);
        const int r0 = (int)(t - (int64_t)ti.h0 * tpb) * TM;
        ti.g0 = (int64_t)ti.h0 * L + r0;
        ti.rows = min(TM, L - r0);
        ti.nsplit = ti.rows;
    }
    return ti;
}

// the tile after ti, without a division (PACK: a step of TM <= L rows crosses at most one head boundary)
template <bool PACK>
__device__ __forceinline__ TileInfo next_tile(TileInfo ti, int L, int64_t total)
{
    if (PACK) {
        ti.g0 += TM;
        if (ti.g0 >= (int64_t)(ti.h0 + 1) * L) ++ti.h0;
        ti.rows = (int)min((int64_t)TM, total - ti.g0);
        ti.nsplit = (int)min((int64_t)ti.rows, (int64_t)(ti.h0 + 1) * L - ti.g0);
    } else {
        int r0 = (int)(ti.g0 - (int64_t)ti.h0 * L) + TM;
        if (r0 >= L) {
            ++ti.h0;
            r0 = 0;
        }
        ti.g0 = (int64_t)ti.h0 * L + r0;
        ti.rows = min(TM, L - r0);
        ti.nsplit = ti.rows;
    }
    return ti;
}

struct TcShared {
    uint64_t lload, lfree, afull, mmadone, fin;
    TcLayout ly;
    IexpC c;
    uint32_t tmem;
    int bk0, bkmax;  // bucket number of table entry 0, and of the last entry
    int abort_flag;
    int rising;   // some i-exp value exceeds the one before it (floored constants)
    int stop;     // set (never cleared) by a softmax thread whose wait gave up
    int ew_stop;  // the same for the read-out warps
};

// Named barrier 1 over the TSOFT softmax threads.  Every softmax thread reaches every one of these
// barriers (the waits before them are bounded), so they end.  bar.sync is warp-aligned: lanes of a
// row-dependent branch meet first.
__device__ __forceinline__ void soft_bar()
{
    __syncwarp();
    asm volatile("bar.sync 1, %0;" ::"n"(TSOFT) : "memory");
}

// Named barrier 2 over the 128 read-out threads
__device__ __forceinline__ void epi_bar()
{
    __syncwarp();
    asm volatile("bar.sync 2, 128;" ::: "memory");
}

// byte J of the distance word v in bits 8..15, bytes 0 and 2 of the offset register o = (1 << 16) |
// offset in bits 0..7 and 16..23: the absolute table address kTabAbs | d << 8 | offset
template <int J>
__device__ __forceinline__ uint32_t tab_addr(uint32_t v, uint32_t o)
{
    uint32_t y;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(y) : "r"(v), "r"(o), "n"(0x7604 | (J << 4)));
    return y;
}

// shared-memory accesses at absolute addresses
// (volatile: the compiler keeps them between the barriers that order the table's writes and reads)
__device__ __forceinline__ uint32_t lds_u32(uint32_t a)
{
    uint32_t v;
    asm volatile("ld.shared.u32 %0, [%1];" : "=r"(v) : "r"(a));
    return v;
}
__device__ __forceinline__ uint32_t lds_u8(uint32_t a)
{
    uint32_t v;
    asm volatile("ld.shared.u8 %0, [%1];" : "=r"(v) : "r"(a));
    return v;
}
__device__ __forceinline__ void sts_u32(uint32_t a, uint32_t v) { asm volatile("st.shared.u32 [%0], %1;" ::"r"(a), "r"(v) : "memory"); }
__device__ __forceinline__ void sts_zero16(uint32_t a)
{
    asm volatile("st.shared.v4.u32 [%0], {%1, %1, %1, %1};" ::"r"(a), "r"(0u) : "memory");
}
__device__ __forceinline__ void red_add_u32(uint32_t a, uint32_t v)
{
    asm volatile("red.shared.add.u32 [%0], %1;" ::"r"(a), "r"(v) : "memory");
}

// the fp16 pair (high bytes b0 of t0 and b1 of t1; low bytes zero) for two keys
__device__ __forceinline__ uint32_t pack_ops(uint32_t t0, uint32_t t1)
{
    uint32_t y;
    asm("prmt.b32 %0, %1, %2, 0x4101;" : "=r"(y) : "r"(t0), "r"(t1));
    return y;
}

// Where the B blocks are: the first nA at offset bA of dynamic shared memory, the rest at bC
struct BlkMap {
    uint32_t bA, bC;
    int nA;
};

// Offset of B block blk (16 keys of one V buffer) in dynamic shared memory
__device__ __forceinline__ uint32_t blk_off(const BlkMap &bm, int blk)
{
    return blk < bm.nA ? bm.bA + (uint32_t)blk * kBlk : bm.bC + (uint32_t)(blk - bm.nA) * kBlk;
}

// V rows of one head (int8, L x 64) -> fp16 B (MN-major, 128-byte swizzled rows) in the B blocks
// blk0 .., rows of keys at or past L up to the last 16-key step zero.  The 128 read-out threads:
// thread t takes 16 values (16 (t % 4) ..) of keys t / 4, t / 4 + 32, ...
__device__ __forceinline__ void convert_v(const int8_t *vh, int L, int nkeys, unsigned char *dsm, const BlkMap &bm,
                                          int blk0, int t)
{
    const int c4 = t & 3;
    for (int j0 = t >> 2; j0 < nkeys; j0 += 8 * 32) {
        uint4 x[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int j = j0 + 32 * u;
            x[u] = (j < L) ? __ldg(reinterpret_cast<const uint4 *>(vh + (size_t)j * TD + 16 * c4))
                           : make_uint4(0x80808080u, 0x80808080u, 0x80808080u, 0x80808080u);
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int j = j0 + 32 * u;
            if (j >= nkeys) break;
            uint4 a = make_uint4(0, 0, 0, 0), b = make_uint4(0, 0, 0, 0);
            if (j < L) {
                const uint32_t x0 = x[u].x ^ 0x80808080u, x1 = x[u].y ^ 0x80808080u;
                const uint32_t x2 = x[u].z ^ 0x80808080u, x3 = x[u].w ^ 0x80808080u;
                a = make_uint4(i8x2_to_h2(x0, 0x5140), i8x2_to_h2(x0, 0x7362), i8x2_to_h2(x1, 0x5140),
                               i8x2_to_h2(x1, 0x7362));
                b = make_uint4(i8x2_to_h2(x2, 0x5140), i8x2_to_h2(x2, 0x7362), i8x2_to_h2(x3, 0x5140),
                               i8x2_to_h2(x3, 0x7362));
            }
            unsigned char *row = dsm + blk_off(bm, blk0 + (j >> 4)) + (uint32_t)(j & 15) * 128;
            *reinterpret_cast<uint4 *>(row + (((2 * c4) ^ (j & 7)) << 4)) = a;
            *reinterpret_cast<uint4 *>(row + (((2 * c4 + 1) ^ (j & 7)) << 4)) = b;
        }
    }
}

// One row of the accumulators (32 lanes = 32 rows of a lane quarter) out of tensor memory: columns
// dcol .. dcol + 63 of lane quarter etl, or, for lanes with use2, dcol2 .. (the second head's D).
__device__ __forceinline__ void read_out_row(const TcParams &p, uint32_t etl, uint32_t dcol, uint32_t dcol2,
                                             bool any2, bool use2, int64_t grow, bool ok_row, int zsum)
{
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        uint32_t va[32];
        tmem_ld32(etl + dcol + 32 * h, va);
        tmem_wait_ld();
        if (any2) {
            uint32_t vb[32];
            tmem_ld32(etl + dcol2 + 32 * h, vb);
            tmem_wait_ld();
            if (use2) {
#pragma unroll
                for (int c = 0; c < 32; ++c) va[c] = vb[c];
            }
        }
        if (!ok_row) continue;
        if (p.out8) {  // 8-bit outputs: 32 bytes of this half of the row
            uint32_t wq[8];
#pragma unroll
            for (int c = 0; c < 8; ++c) {
                wq[c] = 0;
#pragma unroll
                for (int k = 0; k < 4; ++k)
                    wq[c] |= requant8(__float2int_rn(__uint_as_float(va[4 * c + k])) - zsum, p.n1, p.n2, p.zp8)
                             << (8 * k);
            }
            uint4 *d8 = reinterpret_cast<uint4 *>(p.out8 + (size_t)grow * p.ld_out8 + 32 * h);
            d8[0] = make_uint4(wq[0], wq[1], wq[2], wq[3]);
            d8[1] = make_uint4(wq[4], wq[5], wq[6], wq[7]);
        } else {
            int32_t *dst = p.acc + (size_t)grow * TD + 32 * h;
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                int v8[8];
#pragma unroll
                for (int j = 0; j < 8; ++j) v8[j] = __float2int_rn(__uint_as_float(va[8 * c + j])) - zsum;
                stg256(dst + 8 * c, v8);
            }
        }
    }
}

// SMALL_E: every i-exp value is below 2^28 (decided on the host from the scale), so 16 of them sum
// exactly in 32 bits
template <int NKB, bool SMALL_E, bool PACK>
__global__ void __launch_bounds__(TTHREADS, 1) lis_attn_tc_kernel(TcParams p)
{
    extern __shared__ __align__(1024) unsigned char dsm[];
    TcShared &sh = *reinterpret_cast<TcShared *>(dsm + C_SH);
    uint32_t *ONES = reinterpret_cast<uint32_t *>(dsm + C_ONES);
    float *LUTF = reinterpret_cast<float *>(dsm + C_LUTF);
    int *red_max = reinterpret_cast<int *>(dsm + C_RMAX);
    unsigned long long *red_sum = reinterpret_cast<unsigned long long *>(dsm + C_RSUM);
    uint32_t *GT = reinterpret_cast<uint32_t *>(dsm + C_GT);
    uint16_t *BK = reinterpret_cast<uint16_t *>(dsm + C_BK);
    float *rs_hi = reinterpret_cast<float *>(dsm + C_BK);
    float *rs_lo = rs_hi + TM;
    int *rs_bits = reinterpret_cast<int *>(rs_lo + TM);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    volatile int *abort_flag = &sh.abort_flag;
    volatile int *stop_flag = &sh.stop;
    const int L = p.L;
    const int nsteps = (L + 15) >> 4;  // MMA K steps of 16 keys
    pdl_release();
    {
        // the layout for this CTA's shared-memory window; a window other than the expected one, or too
        // small, is reported (FQVIT_ERR_UNSUPPORTED) instead of run
        const TcLayout ly = tc_layout(sa(dsm), (PACK ? 2 : 1) * nsteps, (uint32_t)(TM * p.ld));
        if (!ly.fits || ly.need > p.smem || (sa(dsm) & 1023u) != 0) {
            if (tid == 0) atomicCAS(&g_status, 0, 2);
            return;
        }
        if (tid == 0) sh.ly = ly;
    }
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
                     "r"(tmem_cols(NKB, PACK)));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    __syncthreads();
    {
        // the 256 i-exp values once (the row-maximum exchange area is free until the first tile), then
        // their 32 copies per table line
        uint32_t *e_tmp = reinterpret_cast<uint32_t *>(red_max);
        const IexpC c = sh.c;
        for (int d = tid; d < 256; d += blockDim.x) {
            const uint32_t e = iexp_neg(d, c);
            e_tmp[d] = e;
            LUTF[d] = __uint2float_rn(e);
        }
        for (int i = tid; i < 128; i += blockDim.x) ONES[i] = 0x3C003C00u;
        __syncthreads();
        for (int i = tid; i < 256 * 32; i += blockDim.x)
            sts_u32(kTabAbs + (uint32_t)(i >> 5) * 256u + LUT_BYTE + 4u * (i & 31), e_tmp[i >> 5]);
        for (int d = tid; d < 255; d += blockDim.x)
            if (e_tmp[d] < e_tmp[d + 1]) sh.rising = 1;
    }
    if (tid == 0) {
        const int bkmax = (int)(__float_as_uint(LUTF[0] * (1.0f + 0x1p-20f)) >> BK_SHIFT);
        sh.bkmax = bkmax;
        sh.bk0 = bkmax - (BK_N - 1);
    }
    __syncthreads();  // the copies of the i-exp values read, rising, the bucket range
    if (!sh.rising) {
        // #{d : e(d) > x} by binary search (the values never rise with d)
        auto count_above = [&](float x) -> int {
            int lo = 0;
            for (int step = 128; step >= 1; step >>= 1)
                if (LUTF[lo + step - 1] > x) lo += step;
            if (lo == 255 && LUTF[255] > x) lo = 256;
            return lo;
        };
        for (int i = tid; i < BK_N; i += blockDim.x) {
            const uint32_t b = (uint32_t)(sh.bk0 + i);
            const float e_lo = __uint_as_float(b << BK_SHIFT) * (1.0f - 0x1p-20f);
            const float e_hi = __uint_as_float((b + 1) << BK_SHIFT) * (1.0f + 0x1p-20f);
            const int lo = count_above(e_hi), hi = count_above(e_lo);
            BK[i] = (uint16_t)(lo | (min(hi - lo, 127) << 9));  // 127: the search runs on to 256
        }
    }
    fence_async_smem();  // ONES is read by the MMAs
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sh.tmem;
    pdl_wait();  // the set-up above touched no global memory

    const int tpb = (L + TM - 1) / TM;
    const int64_t total = p.BH * L;
    const int64_t ntiles = PACK ? (total + TM - 1) / TM : p.BH * tpb;
    const int64_t t_begin = (int64_t)blockIdx.x * ntiles / gridDim.x;
    const int ncta_tiles = (int)((int64_t)(blockIdx.x + 1) * ntiles / gridDim.x - t_begin);
    constexpr int TA = ta_col(PACK);
    constexpr int TR = tr_col(NKB, PACK);

    if (tid < TSOFT) {
        const int k4 = warp & 3, q = warp >> 2;
        const int r = 32 * k4 + lane;                    // row of the tile = tensor-memory lane
        // offset registers of the table lookups (1 << 16 selects the table's 64 K page): this row's byte
        // in a line, and this lane's i-exp copy in a line
        const uint32_t rowb = 0x10000u | (4u * (uint32_t)lane + (uint32_t)k4);
        const uint32_t lutb = 0x10000u | (LUT_BYTE + 4u * (uint32_t)lane);
        const uint32_t tlane = tmem + ((uint32_t)(k4 * 32) << 16);
        const bool monotone = !sh.rising;  // codes never fall as d grows
        const uint32_t inc = 1u << (8 * k4);  // this row's byte of a table word
        // The last 64-key block holds R = 1 .. 64 keys (every other block holds 16 per part).  With R > 16
        // part q takes keys 16 q .. 16 q + 15 of it; with R <= 16 (one 16-key MMA step) the four parts
        // take 4 keys each, 4 q .. 4 q + 3, so that no part does a whole extra chunk for a few keys.
        const int R = L - (NKB - 1) * TKB;
        const bool quarter = R <= 16;
        const int last_keys = quarter ? min(4, max(0, R - 4 * q)) : min(16, max(0, R - 16 * q));
        // keys at or past L inside this part's last slice (summed as -128, then removed)
        const int npad = last_keys > 0 ? (quarter ? 4 : 16) - last_keys : 0;
        bool wait_bad = false;
        TileInfo ti = tile_info<PACK>(t_begin, L, p.BH, tpb);
        for (int it = 0; it < ncta_tiles; ++it, ti = next_tile<PACK>(ti, L, total)) {
            const bool valid = r < ti.rows;
            const bool lbad = !mbar_wait_warp(&sh.lload, it & 1, abort_flag);
            // ---- this part's logits into registers; keys at or past L become -128 (no effect on the
            //      maximum; their i-exp values are removed from the sum, their operands are zero)
            // (every part has 16 keys in each block but the last: L > 64 (NKB - 1))
            uint4 w[NKB];
#pragma unroll
            for (int kb = 0; kb < NKB; ++kb) w[kb] = make_uint4(0x80808080u, 0x80808080u, 0x80808080u, 0x80808080u);
            if (valid) {
                const unsigned char *lr = dsm + sh.ly.lg + (size_t)r * p.ld + 16 * q;
#pragma unroll
                for (int kb = 0; kb < NKB - 1; ++kb) w[kb] = *reinterpret_cast<const uint4 *>(lr + kb * TKB);
                if (quarter) {
                    if (last_keys > 0) {
                        uint32_t x = *reinterpret_cast<const uint32_t *>(lr - 16 * q + (NKB - 1) * TKB + 4 * q);
                        if (last_keys < 4)
                            x = (x & (0xFFFFFFFFu >> (32 - 8 * last_keys))) |
                                (0x80808080u & ~(0xFFFFFFFFu >> (32 - 8 * last_keys)));
                        w[NKB - 1].x = x;
                    }
                } else if (last_keys > 0) {
                    uint4 x = *reinterpret_cast<const uint4 *>(lr + (NKB - 1) * TKB);
                    if (last_keys < 16) {
                        uint32_t ww[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
                        for (int b = 0; b < 4; ++b) {
                            const int keep = last_keys - 4 * b;
                            if (keep <= 0)
                                ww[b] = 0x80808080u;
                            else if (keep < 4)
                                ww[b] = (ww[b] & (0xFFFFFFFFu >> (32 - 8 * keep))) |
                                        (0x80808080u & ~(0xFFFFFFFFu >> (32 - 8 * keep)));
                        }
                        x = make_uint4(ww[0], ww[1], ww[2], ww[3]);
                    }
                    w[NKB - 1] = x;
                }
            }
            mbar_arrive(&sh.lfree);  // the logits tile may be refilled
            // ---- row maximum: odd bytes as the high bytes of signed 16-bit lanes, even bytes biased
            //      to 0 .. 255 in unsigned 16-bit lanes
            uint32_t mo = 0x80008000u, me = 0u;
#pragma unroll
            for (int kb = 0; kb < NKB; ++kb) {
                const uint32_t ww[4] = {w[kb].x, w[kb].y, w[kb].z, w[kb].w};
#pragma unroll
                for (int b = 0; b < 4; ++b) {
                    mo = vmax16x2(mo, ww[b]);
                    me = vmax16x2u(me, (ww[b] ^ 0x00800080u) & 0x00FF00FFu);
                }
            }
            int m = max(max(sbyte<1>(mo), sbyte<3>(mo)), max((int)(me & 0xFFFFu), (int)(me >> 16)) - 128);
            red_max[q * TM + r] = m;
            if (lbad || wait_bad) *stop_flag = 1;
            soft_bar();  // A
            if (*stop_flag) break;  // every softmax thread leaves here together
            m = max(max(red_max[r], red_max[TM + r]), max(red_max[2 * TM + r], red_max[3 * TM + r]));
            // the previous tile's operand table is dead (every thread has passed its lookups): clear
            // its bytes and the group totals for this tile's thresholds
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const uint32_t c = (uint32_t)(tid + TSOFT * i);
                sts_zero16(kTabAbs + (c >> 3) * 256u + (c & 7u) * 16u);
            }
            GT[tid] = 0u;
            if (tid < 32 * GT_LD - TSOFT) GT[TSOFT + tid] = 0u;
            // ---- distances: byte d = m - q = (m + 128) - (q + 128), four per word, no borrows
            {
                const uint32_t mrep = (uint32_t)(m + 128) * 0x01010101u;
#pragma unroll
                for (int kb = 0; kb < NKB; ++kb) {
                    w[kb].x = mrep - (w[kb].x ^ 0x80808080u);
                    w[kb].y = mrep - (w[kb].y ^ 0x80808080u);
                    w[kb].z = mrep - (w[kb].z ^ 0x80808080u);
                    w[kb].w = mrep - (w[kb].w ^ 0x80808080u);
                }
            }
            // ---- i-exp row sum over the four parts
            unsigned long long S = 0;
            if (valid) {
                auto sum16 = [&](const uint4 &x) {
                    const uint32_t ww[4] = {x.x, x.y, x.z, x.w};
                    if (SMALL_E) {  // 16 values below 2^28: a 32-bit partial sum is exact
                        uint32_t a = 0;
#pragma unroll
                        for (int b = 0; b < 4; ++b) {
                            const uint32_t e0 = lds_u32(tab_addr<0>(ww[b], lutb));
                            const uint32_t e1 = lds_u32(tab_addr<1>(ww[b], lutb));
                            const uint32_t e2 = lds_u32(tab_addr<2>(ww[b], lutb));
                            const uint32_t e3 = lds_u32(tab_addr<3>(ww[b], lutb));
                            a += e0 + e1;
                            a += e2 + e3;
                        }
                        S += a;
                    } else {
#pragma unroll
                        for (int b = 0; b < 4; ++b) {
                            const uint32_t e0 = lds_u32(tab_addr<0>(ww[b], lutb));
                            const uint32_t e1 = lds_u32(tab_addr<1>(ww[b], lutb));
                            const uint32_t e2 = lds_u32(tab_addr<2>(ww[b], lutb));
                            const uint32_t e3 = lds_u32(tab_addr<3>(ww[b], lutb));
                            S += (unsigned long long)(e0 + e1) + (unsigned long long)(e2 + e3);  // e < 2^31
                        }
                    }
                };
#pragma unroll
                for (int kb = 0; kb < NKB - 1; ++kb) sum16(w[kb]);
                if (quarter) {
                    if (last_keys > 0) {
                        const uint32_t x = w[NKB - 1].x;
                        S += (unsigned long long)(lds_u32(tab_addr<0>(x, lutb)) + lds_u32(tab_addr<1>(x, lutb))) +
                             (unsigned long long)(lds_u32(tab_addr<2>(x, lutb)) + lds_u32(tab_addr<3>(x, lutb)));
                    }
                } else if (last_keys > 0) {
                    sum16(w[NKB - 1]);
                }
                // the padding bytes (-128, distance m + 128)
                S -= (unsigned long long)npad * lds_u32(((uint32_t)(m + 128) << 8) + lutb);
            }
            red_sum[q * TM + r] = S;
            soft_bar();  // B
            S = red_sum[r] + red_sum[TM + r] + red_sum[2 * TM + r] + red_sum[3 * TM + r];
            const RowSum rs = split_2s(S);
            if (monotone) {
                // ---- this row's thresholds: part q finds delta_k for k = q + 1, q + 5, q + 9, q + 13
                //      from the buckets and adds them to the table words
                if (valid) {
                    // e(d) D_k <= 2S, exact: one rounding of an exact product minus hi, against lo
                    auto hit = [&](int d, float D) -> bool { return __fmaf_rn(LUTF[d], D, -rs.hi) <= rs.lo; };
                    const int bk0 = sh.bk0, bkmax = sh.bkmax;
                    // the four searches run side by side (independent chains)
                    float D[4];
                    int lo[4], n[4];  // delta_k in [lo, lo + n]
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const int k = min(q + 1 + 4 * i, 15);
                        D[i] = kD[k];
                        const int b = (int)(__float_as_uint(rs.hi * kRcpD[k]) >> BK_SHIFT) - bk0;
                        if ((unsigned)b < (unsigned)BK_N) {
                            const uint32_t v = BK[b];
                            lo[i] = (int)(v & 511u);
                            n[i] = (int)(v >> 9);
                            if (n[i] == 127) n[i] = 256 - lo[i];
                        } else {
                            lo[i] = b < 0 ? 256 : 0;  // below the buckets: every value lies above T
                            n[i] = 0;
                        }
                    }
                    (void)bkmax;
                    // the first d in [lo, lo + n) that hits, else lo + n (binary search)
                    for (int step = 0; step < 9; ++step) {
                        bool more = false;
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            if (n[i] > 0) {
                                const int h = n[i] >> 1;
                                if (hit(lo[i] + h, D[i])) {
                                    n[i] = h;
                                } else {
                                    lo[i] += h + 1;
                                    n[i] -= h + 1;
                                }
                                more |= n[i] > 0;
                            }
                        }
                        if (!more) break;
                    }
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        if (q + 1 + 4 * i <= 15 && lo[i] < 256) {
                            red_add_u32(kTabAbs + ((uint32_t)lo[i] << 8) + 4u * (uint32_t)lane, inc);
                            red_add_u32(sa(&GT[lane * GT_LD + (lo[i] >> 4)]), inc);
                        }
                    }
                }
            } else if (q == 0) {
                rs_hi[r] = rs.hi;
                rs_lo[r] = rs.lo;
                rs_bits[r] = rs.hibits;
            }
            soft_bar();  // C
            // ---- the operand table: thread (lane, warp g) builds lines 16 g .. 16 g + 15 of column
            //      lane (rows lane, 32 + lane, 64 + lane, 96 + lane)
            {
                const int g = warp;
                if (monotone) {
                    uint32_t carry = 0;  // thresholds below line 16 g, per row byte
                    {
                        const uint4 *gt = reinterpret_cast<const uint4 *>(GT + lane * GT_LD);
                        const uint4 g0 = gt[0], g1 = gt[1], g2 = gt[2], g3 = gt[3];
                        const uint32_t gv[16] = {g0.x, g0.y, g0.z, g0.w, g1.x, g1.y, g1.z, g1.w,
                                                 g2.x, g2.y, g2.z, g2.w, g3.x, g3.y, g3.z, g3.w};
#pragma unroll
                        for (int j = 0; j < 15; ++j) carry += j < g ? gv[j] : 0u;
                    }
                    const uint32_t a0 = kTabAbs + (uint32_t)(16 * g) * 256u + 4u * (uint32_t)lane;
                    uint32_t h[16];  // the 16 loads first: the running sum then has no load in its chain
#pragma unroll
                    for (int i = 0; i < 16; ++i) h[i] = lds_u32(a0 + 256u * i);
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        carry += h[i];
                        sts_u32(a0 + 256u * i, 0x78787878u - 4u * carry);  // 4 (30 - code) per byte
                    }
                } else {
#pragma unroll 1
                    for (int i = 0; i < 16; ++i) {
                        const int d = 16 * g + i;
                        const float ef = LUTF[d];
                        uint32_t word = 0;
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            const int rr = 32 * k + lane;
                            const uint32_t E = operand_exp_f(ef, rs_bits[rr], rs_hi[rr], rs_lo[rr]);
                            word |= (4u * E) << (8 * k);
                        }
                        sts_u32(kTabAbs + (uint32_t)d * 256u + 4u * (uint32_t)lane, word);
                    }
                }
            }
            soft_bar();  // D
            // the previous tile's MMAs have read the operands in tensor memory: they may be rewritten
            if (it > 0 && !mbar_wait_warp(&sh.mmadone, (it - 1) & 1, abort_flag)) {
                wait_bad = true;  // the next tile's first barrier ends the loop for all
                continue;
            }
            // ---- operands of this row's keys -> tensor memory
            {
                auto ops16 = [&](const uint4 &x, uint32_t (&o)[8]) {
                    const uint32_t ww[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
                    for (int b = 0; b < 4; ++b) {
                        const uint32_t t0 = lds_u8(tab_addr<0>(ww[b], rowb));
                        const uint32_t t1 = lds_u8(tab_addr<1>(ww[b], rowb));
                        const uint32_t t2 = lds_u8(tab_addr<2>(ww[b], rowb));
                        const uint32_t t3 = lds_u8(tab_addr<3>(ww[b], rowb));
                        o[2 * b] = pack_ops(t0, t1);
                        o[2 * b + 1] = pack_ops(t2, t3);
                    }
                };
                // (rows past the tile's end take whatever their padding bytes give: their accumulator rows
                // are never read, and a row of D depends only on its own row of operands)
#pragma unroll
                for (int kb = 0; kb < NKB - 1; ++kb) {
                    uint32_t o[8];
                    ops16(w[kb], o);
                    tmem_st8(tlane + TA + 32 * kb + 8 * q, o);
                }
                if (quarter) {  // every part writes its 2 columns of the last MMA step (zeros past L)
                    const uint32_t x = w[NKB - 1].x;
                    uint32_t o0 = pack_ops(lds_u8(tab_addr<0>(x, rowb)), lds_u8(tab_addr<1>(x, rowb)));
                    uint32_t o1 = pack_ops(lds_u8(tab_addr<2>(x, rowb)), lds_u8(tab_addr<3>(x, rowb)));
                    if (last_keys < 4) {
                        o1 = last_keys <= 2 ? 0u : (o1 & 0xFFFFu);
                        if (last_keys < 2) o0 = last_keys == 1 ? (o0 & 0xFFFFu) : 0u;
                    }
                    tmem_st2(tlane + TA + 32 * (NKB - 1) + 2 * q, o0, o1);
                } else if (last_keys > 0) {  // warp-uniform
                    uint32_t o[8];
                    ops16(w[NKB - 1], o);
#pragma unroll
                    for (int c = 0; c < 8; ++c) {  // keys at or past L get a zero operand
                        if (2 * c >= last_keys)
                            o[c] = 0;
                        else if (2 * c + 1 == last_keys)
                            o[c] &= 0xFFFFu;
                    }
                    tmem_st8(tlane + TA + 32 * (NKB - 1) + 8 * q, o);
                }
            }
            __syncwarp();
            tmem_wait_st();
            tc_fence_before();
            mbar_arrive(&sh.afull);
        }
    } else {
        // ---------------- read-out warps (lane quarter eq), with V, the MMA issue and the logits copies
        const int eq = warp & 3;
        const int et = tid - TSOFT;  // 0 .. 127
        const uint32_t etl = tmem + ((uint32_t)(eq * 32) << 16);
        volatile int *ew_stop = &sh.ew_stop;
        int conv_hi = -1;  // the last head whose V went into its B buffer
        int ncopies = 0;
        auto blk0 = [&](int h) -> int { return PACK ? (h & 1) * nsteps : 0; };  // first B block of head h's V
        const BlkMap bm{sh.ly.bA, sh.ly.bC, sh.ly.nA};
        unsigned char *LG = dsm + sh.ly.lg;
        auto last_head = [](const TileInfo &t) { return t.nsplit < t.rows ? t.h0 + 1 : t.h0; };
        TileInfo ti = tile_info<PACK>(t_begin, L, p.BH, tpb);
        TileInfo tp = ti;  // the previous tile
        if (warp == TCOPY_WARP && lane == 0 && ncta_tiles > 0) {
            prefetch_l2(p.v + (size_t)ti.h0 * L * TD, (uint32_t)(L * TD));
            if (last_head(ti) != ti.h0) prefetch_l2(p.v + (size_t)last_head(ti) * L * TD, (uint32_t)(L * TD));
            const uint32_t bl = (uint32_t)(ti.rows * p.ld);
            mbar_expect_tx(&sh.lload, bl);
            bulk_g2s(LG, p.logits + (size_t)ti.g0 * p.ld, bl, &sh.lload);
            ++ncopies;
        }
        auto read_out = [&](const TileInfo &t) {
            const int i = 32 * eq + lane;  // row of the tile
            const bool any2 = PACK && t.nsplit < 32 * eq + 32 && t.nsplit < t.rows;
            const bool use2 = PACK && i >= t.nsplit;
            int zsum = 0;  // zp (sum_j 2^(15-code_j)), an exact integer below 2^24 times |zp| <= 255
            if (p.zp != 0) {
                uint32_t rsv;
                tmem_ld1(etl + TR, rsv);
                tmem_wait_ld();
                zsum = p.zp * __float2int_rn(__uint_as_float(rsv));
            }
            read_out_row(p, etl, 0, TD, any2, use2, t.g0 + i, i < t.rows, zsum);
        };
        int it = 0;
        for (; it < ncta_tiles; ++it) {
            if (it > 0) {
                tp = ti;
                ti = next_tile<PACK>(ti, L, total);
            }
            if (warp == TCOPY_WARP && lane == 0 && it + 1 < ncta_tiles) {
                // the next tile's logits as soon as every softmax thread holds this tile's
                const TileInfo tn = next_tile<PACK>(ti, L, total);
                if (mbar_wait(&sh.lfree, it & 1, abort_flag)) {
                    const uint32_t bl = (uint32_t)(tn.rows * p.ld);
                    mbar_expect_tx(&sh.lload, bl);
                    bulk_g2s(LG, p.logits + (size_t)tn.g0 * p.ld, bl, &sh.lload);
                    ++ncopies;
                    if (last_head(tn) != last_head(ti))
                        prefetch_l2(p.v + (size_t)last_head(tn) * L * TD, (uint32_t)(L * TD));
                    if (it + 2 < ncta_tiles) {
                        const TileInfo tm = next_tile<PACK>(tn, L, total);
                        prefetch_l2(p.logits + (size_t)tm.g0 * p.ld, (uint32_t)(tm.rows * p.ld));
                    }
                }
            }
            bool ok = true;
            if (it > 0) {  // the previous tile's accumulators; then D and the B buffers are free
                ok = mbar_wait_warp(&sh.mmadone, (it - 1) & 1, abort_flag);
                if (ok) {
                    tc_fence_after();
                    read_out(tp);
                }
            }
            // V of this tile's head(s) not yet in B
            if (ok) {
                for (int h = max(conv_hi + 1, ti.h0); h <= last_head(ti); ++h) {
                    convert_v(p.v + (size_t)h * L * TD, L, 16 * nsteps, dsm, bm, blk0(h), et);
                    conv_hi = h;
                }
            }
            fence_async_smem();
            tc_fence_before();
            if (!ok) *ew_stop = 1;
            epi_bar();  // D read, B written: this tile's MMAs may run
            if (*ew_stop) break;
            if (warp == TMMA_WARP && lane == 0) {
                if (mbar_wait(&sh.afull, it & 1, abort_flag)) {
                    tc_fence_after();
                    const uint64_t ones = smem_desc_plain(sa(ONES), 128, 256);
                    const int nh = (PACK && ti.nsplit < ti.rows) ? 2 : 1;
                    for (int hh = 0; hh < nh; ++hh) {
                        const int bb = blk0(ti.h0 + hh);
                        const uint32_t dcol = tmem + (uint32_t)(hh * TD);
                        // the blocks in order, region A's then region C's: a descriptor's address field
                        // (address / 16) grows by kBlk / 16 per block
                        uint64_t da = smem_desc(sa(dsm) + blk_off(bm, bb), 1024, 1024);
                        const uint64_t dc = smem_desc(sa(dsm) + bm.bC, 1024, 1024);
                        uint32_t at = tmem + TA;
                        for (int s = 0; s < nsteps; ++s) {
                            mma_f16_ta(dcol, at, da, s != 0);
                            at += 8;
                            da = (bb + s + 1 == bm.nA) ? dc : da + (kBlk >> 4);
                        }
                    }
                    if (p.zp != 0)
                        for (int s = 0; s < nsteps; ++s)
                            mma_f16_ta(tmem + TR, tmem + TA + 8 * s, ones, s != 0, kIdescOnes);
                    mma_commit(&sh.mmadone);
                } else {
                    *ew_stop = 1;
                }
            }
        }
        if (it == ncta_tiles && ncta_tiles > 0 && !*ew_stop) {  // the last tile's accumulators
            if (mbar_wait_warp(&sh.mmadone, (ncta_tiles - 1) & 1, abort_flag)) {
                tc_fence_after();
                read_out(ti);
            }
        }
        if (warp == TCOPY_WARP && lane == 0 && ncopies > 0)  // no copy may land after the CTA exits
            mbar_wait(&sh.lload, (ncopies - 1) & 1, abort_flag, false);
        if (warp == TMMA_WARP && lane == 0) {  // every MMA issued has completed before tensor memory is freed
            mma_commit(&sh.fin);
            mbar_wait(&sh.fin, 0, abort_flag, false);
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == TMMA_WARP)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(tmem_cols(NKB, PACK)));
}

// Dynamic shared memory of a launch: the layout's extent with the window at its expected start (1024:
// the kernel has no static shared memory), or 0 when it does not fit.
uint32_t tc_smem_bytes(int L, int64_t ld, bool pack)
{
    const TcLayout l = tc_layout(1024u, (pack ? 2 : 1) * ((L + 15) / 16), (uint32_t)(TM * ld));
    return l.fits ? l.need : 0u;
}

bool use_pack(int L) { return L >= TM && L <= kPackMaxBlocks * TKB; }

template <int NKB, bool SMALL_E, bool PACK>
cudaError_t tc_launch(const TcParams &p, size_t smem, int grid, cudaStream_t st)
{
    cudaError_t e = check_smem_fits((const void *)lis_attn_tc_kernel<NKB, SMALL_E, PACK>, smem);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(lis_attn_tc_kernel<NKB, SMALL_E, PACK>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(lis_attn_tc_kernel<NKB, SMALL_E, PACK>, dim3(grid), dim3(TTHREADS), smem, st, p);
}

template <int NKB>
cudaError_t tc_launch_e(bool small_e, bool pack, const TcParams &p, size_t smem, int grid, cudaStream_t st)
{
    if constexpr (NKB <= kPackMaxBlocks && NKB >= 2) {
        if (pack)
            return small_e ? tc_launch<NKB, true, true>(p, smem, grid, st)
                           : tc_launch<NKB, false, true>(p, smem, grid, st);
    }
    return small_e ? tc_launch<NKB, true, false>(p, smem, grid, st) : tc_launch<NKB, false, false>(p, smem, grid, st);
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
           ((uintptr_t)b.v % 16) == 0 && a.ld_logit <= 1024 && tc_smem_bytes(a.L, a.ld_logit, use_pack(a.L)) > 0;
}

cudaError_t launch_lis_attention_tc(const LisArgs &a, const AttnVArgs &b, cudaStream_t st)
{
    const bool pack = use_pack(a.L);
    const uint32_t smem = tc_smem_bytes(a.L, a.ld_logit, pack);
    TcParams p{a.logits, a.ld_logit, b.v, b.acc, b.BH, a.L, b.zp_v, iexp_consts_host(a.s_logit),
               b.out8, b.ld_out8, b.rq_n1, b.rq_n2, b.rq_zp, smem};
    const int64_t ntiles = pack ? (b.BH * a.L + TM - 1) / TM : b.BH * ((a.L + TM - 1) / TM);
    const int grid = (int)(ntiles < sm_count() ? ntiles : sm_count());
    const bool se = small_iexp(p.ic);
    switch ((a.L + TKB - 1) / TKB) {
    case 1: return tc_launch_e<1>(se, pack, p, smem, grid, st);
    case 2: return tc_launch_e<2>(se, pack, p, smem, grid, st);
    case 3: return tc_launch_e<3>(se, pack, p, smem, grid, st);
    case 4: return tc_launch_e<4>(se, pack, p, smem, grid, st);
    case 5: return tc_launch_e<5>(se, pack, p, smem, grid, st);
    case 6: return tc_launch_e<6>(se, pack, p, smem, grid, st);
    case 7: return tc_launch_e<7>(se, pack, p, smem, grid, st);
    case 8: return tc_launch_e<8>(se, pack, p, smem, grid, st);
    case 9: return tc_launch_e<9>(se, pack, p, smem, grid, st);
    default: return tc_launch_e<10>(se, pack, p, smem, grid, st);
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
    int lnst = 0;
    e = read_clear_ln_status(&lnst);
    if (*status == 0) *status = lnst;
    return e;
}

}  // namespace fqvit
