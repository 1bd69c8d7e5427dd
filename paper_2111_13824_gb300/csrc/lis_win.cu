// lis_win.cu -- fused Log-Int-Softmax + BitShift attention times values on the
// tcgen05 tensor cores for short rows: L <= 64 keys, as in windowed attention
// (7 x 7 windows: L = 49), with an optional relative-position bias.
//
// The product is the one of lis_tc.cu: acc = P (V - zp_V) with
// P[i][j] = 2^(15 - code_ij) exact in fp16 and fp32 accumulation exact for
// codes made by Log-Int-Softmax (Eq. 15, Algorithm 2).  A tile of the MMA
// (M = 128 rows) holds two heads: head slot h in {0, 1} owns tensor-memory
// lanes 64 h .. 64 h + 63 (query row i at lane 64 h + i) and keys
// 64 h .. 64 h + 63 of the K = 128 reduction.  A is block diagonal: a row's
// operands sit in its own slot's 32 tensor-memory columns (two keys per
// column) and the other slot's columns hold zeros, written once.  B holds the
// two heads' V rows as fp16 (rows = keys, 128-byte swizzled, MN-major), so
// one tile is 8 MMAs of K = 16.  With d = 32, B's columns 32 .. 63 are free:
// column 32 holds 1 for every key, which makes column 32 of D the row sum of
// P, and acc = P V - zp_V (P 1) needs no second product.
//
// A CTA runs up to four independent groups of 128 threads; thread r of a
// group serves query row r & 63 of head slot r >> 6, owns tensor-memory lane r
// of the group's 128 columns (D: 0..63, A: 64..127) and converts V's key row
// r & 63 of its slot.  Per tile a thread takes its row into registers, adds
// the bias, finds the maximum and the i-exp row sum, waits for the group's
// previous MMAs, stores their accumulators, writes its operands and its V row,
// and arrives on the group's mbarrier; the thread whose arrival count makes a
// multiple of 128 issues the tile's MMAs once all arrivals are in, so no
// thread waits for the group's slowest at a barrier.
//
// i-exp table: e(d) for the distance d = max - q~ in [0, ne), replicated for
// each of the 32 lanes (one 256-byte line per d: 32 copies of e, then 32 of
// fp32 e), so lookups are free of bank conflicts and a byte permute forms the
// address.  Distances past 15 |q_ln2| all give e(15 |q_ln2|) (the clamp of
// Algorithm 1), so d is clamped to ne - 1.
//
// Every wait is bounded (two seconds), after which the group stops, records a
// timeout status and the kernel drains what it issued.
#include "fqvit_internal.cuh"
#include "lis_common.cuh"
#include "tc_common.cuh"

#include <cstdlib>
#include <cstring>

namespace fqvit {

namespace {

using namespace lis;
using namespace tc;

constexpr int WMAXG = 4;                 // groups per CTA
constexpr int WB_BYTES = 128 * 128;      // B of a group: 128 keys x 64 fp16, 128B-swizzled (16 KB)
constexpr int WBIAS_ROW = 64;            // bytes per bias row (keys 0..63, 16-byte chunks swizzled)

struct WinParams {
    const int8_t *logits;
    int64_t ld;
    const int8_t *v;
    int64_t ld_v;
    int32_t *acc;
    int64_t ld_acc;
    const int8_t *bias;  // [heads][(2w-1)^2] or nullptr
    int heads;
    int window;
    int64_t BH;
    int L;
    int zp;
    IexpC ic;
    int ne;  // table entries: distances 0 .. ne - 1
    int ng;  // groups per CTA
    uint8_t *out8;  // when not null: 8-bit outputs (requant8 with n1, n2, zp8) instead of acc
    int64_t ld_out8;
    int n1, n2, zp8;
    const uint8_t *region;  // shifted-window mask: region ids [n_windows][L] (MASK variants)
    int n_windows;
    int mask_c;  // |mask value| clamped to 1024 (exact: see the kernel)
};

struct WinShared {
    uint64_t afull[WMAXG];    // a group's 128 threads wrote A and B and read D
    uint64_t mmadone[WMAXG];  // the group's MMAs completed
    uint32_t arrivals[WMAXG]; // arrivals so far: the one that makes a multiple of 128 issues the MMAs
    int issued[WMAXG];        // tiles whose MMAs were issued
    uint32_t tmem;
    int abort_flag;
};

__device__ __forceinline__ uint32_t win_tmem_cols(int ng) { return ng == 1 ? 128u : ng == 2 ? 256u : 512u; }

// the i-exp table line of the distance in the low (SEL = 0x5104) or high (0x5324) half of a
// pair word, for this lane: 256 d + 4 lane
template <uint32_t SEL>
__device__ __forceinline__ uint32_t lut_off(uint32_t dpair, uint32_t lane4)
{
    return prmt(dpair, lane4, SEL);
}

// fp16 exponent field (30 - code) of the operand 2^(15-code), as operand_exp_f with D_k read
// from a table (dk[k] = D_k for k = 1 .. 63; k <= 43 since 2S < 2^43 and e >= 1)
__device__ __forceinline__ uint32_t operand_exp_tab(float ef, int G, float hi, float lo, const float *dk)
{
    const int k = (G - __float_as_int(ef)) >> 23;
    const float t = __fmaf_rn(ef, dk[k], -hi);
    uint32_t le;  // 0xFFFFFFFF when e D_k <= 2S
    asm("set.le.u32.f32 %0, %1, %2;" : "=r"(le) : "f"(t), "f"(lo));
    return (uint32_t)max(31 - k + (int)le, 15);
}

// NQ: 16-key chunks of a row (L in 16 (NQ - 1) + 1 .. 16 NQ).  MASK (with BIAS): the shifted-window
// mask.  Logits then sit in the 16-bit lanes as v = q + bias + 1280 - (masked ? m_c : 0) with m_c the
// mask magnitude clamped to 1024: a key masked by more still lands below every unmasked key (the
// query's own key is never masked, v >= 1024) at a distance above 510 >= the table's last entry,
// which is the clamp 15 |q_ln2| of Algorithm 1 (the launch requires 15 |q_ln2| <= 510), so its
// i-exp value and the row maximum are those of the true mask.
template <int D, bool BIAS, bool SMALL_E, int NQ, bool MASK>
__global__ void __launch_bounds__(WMAXG * 128, 1) lis_attn_win_kernel(WinParams p)
{
    extern __shared__ __align__(16) unsigned char dsm_raw[];
    __shared__ WinShared sh;
    __shared__ uint32_t e_tmp[512];
    __shared__ float dk[64];
    __shared__ int koff[64], qbase[64];  // relative-position offsets (bias only)
    // the table first, at the fixed start of dynamic shared memory (lookups add no base), then
    // B (1024-byte aligned for the 128-byte swizzle) and the bias rows
    const unsigned char *LUTB = dsm_raw;                                      // ne x 256 B
    const uint32_t bs_off = (uint32_t)p.ne * 256u;
    unsigned char *Bs_all = dsm_raw + bs_off + ((1024u - ((sa(dsm_raw) + bs_off) & 1023u)) & 1023u);  // ng x 16 KB
    unsigned char *BR = Bs_all + p.ng * WB_BYTES;                             // heads x L x 64 B
    unsigned char *RG = BR + (BIAS ? (size_t)p.heads * p.L * WBIAS_ROW : 0);  // n_windows x 64 B region ids

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int g = tid >> 7, r = tid & 127;
    const int h = r >> 6, i = r & 63;
    const int L = p.L;
    volatile int *abort_flag = &sh.abort_flag;
    pdl_release();

    if (tid == 0) {
        for (int k = 0; k < p.ng; ++k) {
            mbar_init(&sh.afull[k], 128);
            mbar_init(&sh.mmadone[k], 1);
            sh.arrivals[k] = 0;
            sh.issued[k] = 0;
        }
        sh.abort_flag = 0;
    }
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(sa(&sh.tmem)),
                     "r"(win_tmem_cols(p.ng)));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    // set-up, phase 1: i-exp values, the D_k table, the raw bias table (into the B area, free
    // until phase 3) and the index offsets of the relative positions
    for (int d = tid; d < p.ne; d += blockDim.x) e_tmp[d] = iexp_neg(d, p.ic);
    for (int k = tid; k < 64; k += blockDim.x)  // D_1 = 3, D_k = 3 2^(k-1) - 1 (exact up to k = 24)
        dk[k] = k <= 1 ? 3.0f : __fsub_rn(__int_as_float(((k + 127) << 23) | 0x400000), 1.0f);
    const int nb = 2 * p.window - 1;
    pdl_wait();  // the first access to global memory follows
    if (BIAS) {
        for (int x = tid; x < p.heads * nb * nb; x += blockDim.x) Bs_all[x] = (unsigned char)p.bias[x];
        // entry of (query i, key j) = qbase[i] - koff[j]: (y_i - y_j + w - 1) nb + (x_i - x_j + w - 1)
        for (int j = tid; j < L; j += blockDim.x) {
            const int y = j / p.window, x = j - y * p.window;
            koff[j] = y * nb + x;
            qbase[j] = (y + p.window - 1) * nb + x + p.window - 1;
        }
    }
    __syncthreads();
    // phase 2: bias rows (byte j of row (head, query) = bias + 128 for keys j < L, 0 past L; the
    // 16-byte chunk c of a row sits at position c ^ ((query >> 1) & 3)) and the replicated table
    if (BIAS) {
        // thread: word wj (keys 4 wj .. +3) of rows tid / 16, + blockDim / 16, ...
        const int wj = tid & 15, rstep = blockDim.x >> 4;
        int kof[4];
#pragma unroll
        for (int b = 0; b < 4; ++b) kof[b] = 4 * wj + b < L ? koff[4 * wj + b] : -1;
        const int nrows = p.heads * L;
#pragma unroll 4
        for (int row = tid >> 4; row < nrows; row += rstep) {
            const int hh = row / L, qi = row - hh * L;
            const unsigned char *tab = Bs_all + hh * nb * nb + qbase[qi];
            uint32_t word = 0;
#pragma unroll
            for (int b = 0; b < 4; ++b)
                if (kof[b] >= 0) word |= (uint32_t)(((int)(int8_t)tab[-kof[b]] + 128) & 0xFF) << (8 * b);
            const int pc = (wj >> 2) ^ ((qi >> 1) & 3);
            *reinterpret_cast<uint32_t *>(BR + (size_t)row * WBIAS_ROW + 16 * pc + 4 * (wj & 3)) = word;
        }
    }
    for (int x = tid; x < p.ne * 16; x += blockDim.x) {  // 16 bytes: 4 copies of e (parts 0-7) or fp32 e
        const uint32_t e = e_tmp[x >> 4];
        const uint32_t w = (x & 8) ? __float_as_uint(__uint2float_rn(e)) : e;
        reinterpret_cast<uint4 *>(const_cast<unsigned char *>(LUTB))[x] = make_uint4(w, w, w, w);
    }
    __syncthreads();
    if (MASK)  // region ids, one 64-byte row per window (bytes past L: 0, never read as masked)
        for (int x = tid; x < p.n_windows * 64; x += blockDim.x) {
            const int wdx = x >> 6, j = x & 63;
            RG[x] = j < L ? p.region[(size_t)wdx * L + j] : 0;
        }
    // phase 3: B of every group: zeros, and (d = 32) fp16 1 in column 32 of every key row below L
    for (int x = tid; x < p.ng * WB_BYTES / 16; x += blockDim.x) {
        const int kk = (x >> 3) & 127, pos = x & 7, ci = pos ^ (kk & 7);
        uint4 z = make_uint4(0, 0, 0, 0);
        if (D == 32 && ci == 4 && (kk & 63) < L) z.x = 0x3C00u;
        *reinterpret_cast<uint4 *>(Bs_all + 16 * x) = z;
    }
    fence_async_smem();  // B is read by the MMAs
    tc_fence_before();
    __syncthreads();
    tc_fence_after();

    const uint32_t tmem = sh.tmem;
    const int ntiles = (int)((p.BH + 1) >> 1);  // BH <= 65535
    const int BH = (int)p.BH;
    const int gstride = (int)gridDim.x * p.ng;

    {
    const uint32_t tD = tmem + 128u * (uint32_t)g + ((uint32_t)((warp & 3) * 32) << 16);  // this warp's lanes
    const uint32_t tA = tD + 64u;
    unsigned char *Bg = Bs_all + g * WB_BYTES;
    const uint32_t lane4 = (uint32_t)lane << 2;
    const int nw = (L + 3) >> 2;   // words that hold keys (all but the last chunk's are full)
    uint32_t cm[4];                // byte masks of the last chunk's words: keys below L
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const int j0 = 16 * (NQ - 1) + 4 * k, n = L - j0;
        cm[k] = n >= 4 ? 0xFFFFFFFFu : n <= 0 ? 0u : (0xFFFFFFFFu >> (32 - 8 * n));
    }
    // A starts as zeros: the other slot's columns and the own slot's keys past the last
    // 16-key chunk are never written again (the first arrival on afull comes after this)
    {
        const uint32_t z[8] = {0, 0, 0, 0, 0, 0, 0, 0};
#pragma unroll
        for (int c = 0; c < 8; ++c) tmem_st8(tA + 8u * c, z);
        tmem_wait_st();
    }

    const uint32_t cap2 = (uint32_t)(p.ne - 1) * 0x10001u;
    const int qi = i < L ? i : L - 1;  // bias row of this thread (rows past L read the last one)
    const int sw = (qi >> 1) & 3;
    const int hstep = (int)((2 * (int64_t)gstride) % p.heads);  // head of the bias table: +2 gstride per tile

    auto load_row = [&](int t, uint4 (&w)[NQ]) {
        const int bh = 2 * t + h;
        const bool ok = t < ntiles && bh < BH && i < L;
        const int8_t *lr = p.logits + ((size_t)bh * L + i) * p.ld;
#pragma unroll
        for (int c = 0; c < NQ; ++c) w[c] = ok ? __ldg(reinterpret_cast<const uint4 *>(lr) + c) : make_uint4(0, 0, 0, 0);
    };

    // accumulators of tile t (rows of this thread): D columns 0 .. D-1 (and 32 = P 1 when D = 32)
    auto store_acc = [&](int t) {
        const int bh = 2 * t + h;
        const bool ok = bh < BH && i < L;
        int zsum = 0;
        if (D == 32 && p.zp != 0) {
            uint32_t x;
            tmem_ld1(tD + 32u, x);
            tmem_wait_ld();
            zsum = p.zp * __float2int_rn(__uint_as_float(x));
        }
#pragma unroll
        for (int c = 0; c < D / 8; ++c) {
            uint32_t va[8];
            tmem_ld8(tD + 8u * c, va);
            tmem_wait_ld();
            if (ok && p.out8) {  // 8 bytes of 8-bit outputs
                uint32_t lo = 0, hi = 0;
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    lo |= requant8(__float2int_rn(__uint_as_float(va[j])) - zsum, p.n1, p.n2, p.zp8) << (8 * j);
                    hi |= requant8(__float2int_rn(__uint_as_float(va[4 + j])) - zsum, p.n1, p.n2, p.zp8) << (8 * j);
                }
                *reinterpret_cast<uint2 *>(p.out8 + ((size_t)bh * L + i) * p.ld_out8 + 8 * c) = make_uint2(lo, hi);
            } else if (ok) {
                int v8[8];
#pragma unroll
                for (int j = 0; j < 8; ++j) v8[j] = __float2int_rn(__uint_as_float(va[j])) - zsum;
                stg256(p.acc + ((size_t)bh * L + i) * p.ld_acc + 8 * c, v8);
            }
        }
    };

    uint4 nw4[NQ];
    int t = (int)blockIdx.x * p.ng + g;
    int hh = BIAS ? (int)((2 * (int64_t)t + h) % p.heads) : 0;
    load_row(t, nw4);
    int it = 0;
    int prev = -1;
    bool stopped = false;
    for (; t < ntiles; t += gstride, ++it, hh = (hh + hstep >= p.heads ? hh + hstep - p.heads : hh + hstep)) {
        uint4 w[NQ];
#pragma unroll
        for (int c = 0; c < NQ; ++c) w[c] = nw4[c];
        load_row(t + gstride, nw4);  // the next tile's logits, in flight during this one

        const int bh = 2 * t + h;
        const bool valid = bh < BH && i < L;
        // ---- q + 128 per byte, keys past L zeroed (only the last chunk has any)
        uint32_t u[4 * NQ];
#pragma unroll
        for (int c = 0; c < NQ; ++c) {
            const uint32_t ww[4] = {w[c].x, w[c].y, w[c].z, w[c].w};
#pragma unroll
            for (int k = 0; k < 4; ++k) u[4 * c + k] = (ww[k] ^ 0x80808080u) & (c == NQ - 1 ? cm[k] : 0xFFFFFFFFu);
        }
        // ---- pairs of 16-bit lanes v = q + bias + 256 (0 for keys past L):
        //      vp[2j] holds keys (4j, 4j+2), vp[2j+1] keys (4j+1, 4j+3)
        uint32_t vp[8 * NQ];
        if (MASK) {
            const unsigned char *br = BR + ((size_t)hh * L + qi) * WBIAS_ROW;
            const unsigned char *rg = RG + (size_t)((bh / p.heads) % p.n_windows) * 64;
            const uint32_t rib = (uint32_t)rg[qi] * 0x01010101u;
#pragma unroll
            for (int c = 0; c < NQ; ++c) {
                const uint4 b4 = *reinterpret_cast<const uint4 *>(br + 16 * (c ^ sw));
                const uint4 r4 = *reinterpret_cast<const uint4 *>(rg + 16 * c);
                const uint32_t bb[4] = {b4.x, b4.y, b4.z, b4.w};
                const uint32_t rr[4] = {r4.x, r4.y, r4.z, r4.w};
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const int j = 4 * c + k;
                    // byte nonzero: the key's region differs from the query's (keys past L: never)
                    const uint32_t x = (rr[k] ^ rib) & (c == NQ - 1 ? cm[k] : 0xFFFFFFFFu);
                    const uint32_t me = ((prmt(x, 0u, 0x4240u) + 0x7FFF7FFFu) >> 15) & 0x00010001u;
                    const uint32_t mo = ((prmt(x, 0u, 0x4341u) + 0x7FFF7FFFu) >> 15) & 0x00010001u;
                    vp[2 * j] = prmt(u[j], 0u, 0x4240u) + prmt(bb[k], 0u, 0x4240u) + 0x04000400u - me * (uint32_t)p.mask_c;
                    vp[2 * j + 1] =
                        prmt(u[j], 0u, 0x4341u) + prmt(bb[k], 0u, 0x4341u) + 0x04000400u - mo * (uint32_t)p.mask_c;
                }
            }
        } else if (BIAS) {
            const unsigned char *br = BR + ((size_t)hh * L + qi) * WBIAS_ROW;
#pragma unroll
            for (int c = 0; c < NQ; ++c) {
                const uint4 b4 = *reinterpret_cast<const uint4 *>(br + 16 * (c ^ sw));
                const uint32_t bb[4] = {b4.x, b4.y, b4.z, b4.w};
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const int j = 4 * c + k;
                    vp[2 * j] = prmt(u[j], 0u, 0x4240u) + prmt(bb[k], 0u, 0x4240u);
                    vp[2 * j + 1] = prmt(u[j], 0u, 0x4341u) + prmt(bb[k], 0u, 0x4341u);
                }
            }
        } else {
#pragma unroll
            for (int j = 0; j < 4 * NQ; ++j) {
                vp[2 * j] = prmt(u[j], 0u, 0x4240u);
                vp[2 * j + 1] = prmt(u[j], 0u, 0x4341u);
            }
        }
        // ---- row maximum (keys past L are 0), then distances d = max - v clamped to the table
        uint32_t mx = vmax16x2u(vp[0], vp[1]);
#pragma unroll
        for (int k = 2; k < 8 * NQ; k += 2) mx = vmax16x2u(mx, vmax16x2u(vp[k], vp[k + 1]));
        const uint32_t m = max(mx & 0xFFFFu, mx >> 16);
        const uint32_t m2 = m * 0x10001u;
#pragma unroll
        for (int k = 0; k < 8 * NQ; ++k) vp[k] = vmin16x2u(m2 - vp[k], cap2);
        // ---- i-exp row sum over the words that hold keys (padding keys of the last word have
        //      d = max; they are taken out below)
        unsigned long long S = 0;
#pragma unroll
        for (int c = 0; c < NQ; ++c) {
            uint32_t a = 0;
            unsigned long long a64 = 0;
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                if (c < NQ - 1 || 4 * c + (k >> 1) < nw) {
                    const uint32_t dp = vp[8 * c + k];
                    const uint32_t e0 = *reinterpret_cast<const uint32_t *>(LUTB + lut_off<0x5104u>(dp, lane4));
                    const uint32_t e1 = *reinterpret_cast<const uint32_t *>(LUTB + lut_off<0x5324u>(dp, lane4));
                    if (SMALL_E)
                        a += e0 + e1;
                    else
                        a64 += (unsigned long long)e0 + e1;
                }
            }
            S += SMALL_E ? (unsigned long long)a : a64;
        }
        {
            const uint32_t mp = MASK ? m - 1024u : m;  // padding keys sit at v = 1024 (MASK) or 0
            const uint32_t dm = mp < (uint32_t)(p.ne - 1) ? mp : (uint32_t)(p.ne - 1);
            const uint32_t epad = *reinterpret_cast<const uint32_t *>(LUTB + ((dm << 8) | lane4));
            S -= (unsigned long long)(4 * nw - L) * epad;
        }
        const RowSum rs = split_2s(S);
        // V key row i of this slot (used after the operands: its latency hides behind them)
        uint4 vv[D / 16];
        {
            const int8_t *vr = p.v + ((size_t)bh * L + i) * p.ld_v;
#pragma unroll
            for (int c = 0; c < D / 16; ++c) vv[c] = valid ? __ldg(reinterpret_cast<const uint4 *>(vr) + c) : make_uint4(0, 0, 0, 0);
        }

        // ---- the previous tile's MMAs are done: its accumulators out, A and B free
        if (it > 0) {
            if (!mbar_wait_warp(&sh.mmadone[g], (it - 1) & 1, abort_flag)) {
                stopped = true;  // the abort flag is set: the other warps' waits end too
                break;
            }
            tc_fence_after();
            store_acc(prev);
        }
        // ---- operands 2^(15 - code) of this row's keys -> tensor memory (own slot), 16 keys at a
        //      time; chunks past NQ keep the zeros of the start
#pragma unroll
        for (int c = 0; c < NQ; ++c) {
            uint32_t o[8];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const int j = 4 * c + k;
                if (c == NQ - 1 && j >= nw) {
                    o[2 * k] = o[2 * k + 1] = 0u;
                    continue;
                }
                const uint32_t de = vp[2 * j], dod = vp[2 * j + 1];
                const float f0 = *reinterpret_cast<const float *>(LUTB + 128 + lut_off<0x5104u>(de, lane4));
                const float f2 = *reinterpret_cast<const float *>(LUTB + 128 + lut_off<0x5324u>(de, lane4));
                const float f1 = *reinterpret_cast<const float *>(LUTB + 128 + lut_off<0x5104u>(dod, lane4));
                const float f3 = *reinterpret_cast<const float *>(LUTB + 128 + lut_off<0x5324u>(dod, lane4));
                const uint32_t E0 = operand_exp_tab(f0, rs.hibits, rs.hi, rs.lo, dk);
                const uint32_t E1 = operand_exp_tab(f1, rs.hibits, rs.hi, rs.lo, dk);
                const uint32_t E2 = operand_exp_tab(f2, rs.hibits, rs.hi, rs.lo, dk);
                const uint32_t E3 = operand_exp_tab(f3, rs.hibits, rs.hi, rs.lo, dk);
                o[2 * k] = (E0 << 10) | (E1 << 26);
                o[2 * k + 1] = (E2 << 10) | (E3 << 26);
            }
            tmem_st8(tA + 32u * (uint32_t)h + 8u * c, o);
        }
        // ---- V key row i of this slot -> fp16 B (row 64 h + i, chunk ci at ci ^ (row & 7))
        if (valid) {
            const int kk = 64 * h + i;
            unsigned char *brow = Bg + kk * 128;
#pragma unroll
            for (int c = 0; c < D / 16; ++c) {
                const uint32_t x0 = vv[c].x ^ 0x80808080u, x1 = vv[c].y ^ 0x80808080u;
                const uint32_t x2 = vv[c].z ^ 0x80808080u, x3 = vv[c].w ^ 0x80808080u;
                uint4 lo, hi;
                lo.x = i8x2_to_h2(x0, 0x5140);
                lo.y = i8x2_to_h2(x0, 0x7362);
                lo.z = i8x2_to_h2(x1, 0x5140);
                lo.w = i8x2_to_h2(x1, 0x7362);
                hi.x = i8x2_to_h2(x2, 0x5140);
                hi.y = i8x2_to_h2(x2, 0x7362);
                hi.z = i8x2_to_h2(x3, 0x5140);
                hi.w = i8x2_to_h2(x3, 0x7362);
                *reinterpret_cast<uint4 *>(brow + (((2 * c) ^ (kk & 7)) << 4)) = lo;
                *reinterpret_cast<uint4 *>(brow + (((2 * c + 1) ^ (kk & 7)) << 4)) = hi;
            }
        }
        tmem_wait_st();
        fence_async_smem();
        tc_fence_before();
        mbar_arrive(&sh.afull[g]);  // A, B written and D read: the tile's MMAs may go
        if (atomicAdd(&sh.arrivals[g], 1u) % 128u == 127u) {
            // the last thread to count issues the tile's MMAs once every arrival is in
            if (mbar_wait(&sh.afull[g], (uint32_t)(it & 1), abort_flag)) {
                tc_fence_after();
                const uint32_t dcol = tmem + 128u * (uint32_t)g, acol = dcol + 64u;
                const uint32_t b0 = sa(Bg);
#pragma unroll
                for (int kb = 0; kb < 2; ++kb)
#pragma unroll
                    for (int s2 = 0; s2 < 4; ++s2)
                        mma_f16_ta(dcol, acol + 32u * kb + 8u * s2, smem_desc(b0 + kb * 8192 + 2048 * s2, 1024, 1024),
                                   (kb | s2) != 0);
                mma_commit(&sh.mmadone[g]);
                sh.issued[g] = it + 1;
            }
        }
        prev = t;
    }
    if (!stopped && it > 0) {
        if (mbar_wait_warp(&sh.mmadone[g], (it - 1) & 1, abort_flag)) {
            tc_fence_after();
            store_acc(prev);
        }
    }
    }
    // every MMA issued has completed before tensor memory is freed (after a timeout too)
    __syncthreads();
    if (tid < p.ng && sh.issued[tid] > 0) mbar_wait(&sh.mmadone[tid], (uint32_t)((sh.issued[tid] - 1) & 1), abort_flag, false);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(win_tmem_cols(p.ng)));
}

constexpr size_t kWinStaticSmem = 512 * 4 + 64 * 4 * 3 + sizeof(WinShared) + 256;
constexpr size_t kSmemLimit = 232448;

size_t win_smem_bytes(int ng, int ne, int heads, int L, bool bias, int mask_windows)
{
    return 1024 + (size_t)ng * WB_BYTES + (size_t)ne * 256 + (bias ? (size_t)heads * L * WBIAS_ROW : 0) +
           (size_t)mask_windows * 64;
}

// table entries: distances up to 255 (510 with a bias), and none past the clamp 15 |q_ln2|
int win_table_entries(const IexpC &c, bool bias)
{
    const int dmax = bias ? 510 : 255;
    const int clamp = 15 * -c.q_ln2;
    return (clamp < dmax ? clamp : dmax) + 1;
}

// groups per CTA that fit shared memory; the raw bias table (heads x (2w-1)^2 bytes) is
// staged in the groups' B area during the set-up
int win_groups(int ne, int heads, int L, int window, bool bias, int mask_windows)
{
    const size_t tab = bias ? (size_t)heads * (2 * window - 1) * (2 * window - 1) : 0;
    for (int ng = WMAXG; ng >= 1; --ng)
        if (win_smem_bytes(ng, ne, heads, L, bias, mask_windows) + kWinStaticSmem <= kSmemLimit &&
            tab <= (size_t)ng * WB_BYTES)
            return ng;
    return 0;
}

bool small_iexp_w(const IexpC &c) { return ((double)c.q_b * c.q_b + c.q_c) * 32768.0 < 268435456.0; }

template <int D, bool BIAS, bool SMALL_E, int NQ, bool MASK>
cudaError_t win_launch_q(const WinParams &p, size_t smem, int grid, cudaStream_t st)
{
    // the static arrays as compiled for this instantiation, not the estimate the group count used
    cudaError_t e = check_smem_fits((const void *)lis_attn_win_kernel<D, BIAS, SMALL_E, NQ, MASK>, smem);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(lis_attn_win_kernel<D, BIAS, SMALL_E, NQ, MASK>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(lis_attn_win_kernel<D, BIAS, SMALL_E, NQ, MASK>, dim3(grid), dim3(128 * p.ng), smem, st, p);
}

template <int D, bool BIAS, bool SMALL_E, bool MASK>
cudaError_t win_launch(const WinParams &p, size_t smem, int grid, cudaStream_t st)
{
    switch ((p.L + 15) >> 4) {
    case 1: return win_launch_q<D, BIAS, SMALL_E, 1, MASK>(p, smem, grid, st);
    case 2: return win_launch_q<D, BIAS, SMALL_E, 2, MASK>(p, smem, grid, st);
    case 3: return win_launch_q<D, BIAS, SMALL_E, 3, MASK>(p, smem, grid, st);
    default: return win_launch_q<D, BIAS, SMALL_E, 4, MASK>(p, smem, grid, st);
    }
}

// (bias, mask): (no, no), (yes, no), (yes, yes); a mask needs the bias (the eligibility checks)
template <int D>
cudaError_t win_launch_d(bool bias, bool mask, bool small_e, const WinParams &p, size_t smem, int grid,
                         cudaStream_t st)
{
    if (mask)
        return small_e ? win_launch<D, true, true, true>(p, smem, grid, st)
                       : win_launch<D, true, false, true>(p, smem, grid, st);
    if (bias)
        return small_e ? win_launch<D, true, true, false>(p, smem, grid, st)
                       : win_launch<D, true, false, false>(p, smem, grid, st);
    return small_e ? win_launch<D, false, true, false>(p, smem, grid, st)
                   : win_launch<D, false, false, false>(p, smem, grid, st);
}

}  // namespace

bool lis_attention_win_eligible(const LisArgs &a, const AttnVArgs &b)
{
    if (a.L > 64 || a.codes != nullptr || a.rowsum != nullptr) return false;
    if (!(b.d == 32 || (b.d == 64 && b.zp_v == 0))) return false;
    if (a.ld_logit % 16 != 0 || ((uintptr_t)a.logits % 16) != 0) return false;
    if (b.ld_v % 16 != 0 || ((uintptr_t)b.v % 16) != 0) return false;
    if (b.out8 ? (b.ld_out8 % 8 != 0 || ((uintptr_t)b.out8 % 8) != 0)
               : (b.ld_acc % 8 != 0 || ((uintptr_t)b.acc % 32) != 0))
        return false;
    const bool bias = a.bias != nullptr;
    const IexpC c = iexp_consts_host(a.s_logit);
    const int mwin = a.region ? a.n_windows : 0;
    // a mask needs the bias (the masked kernel variants) and the i-exp clamp inside the table
    if (a.region && (!bias || 15 * -c.q_ln2 > 510)) return false;
    return win_groups(win_table_entries(c, bias), a.heads, a.L, a.window, bias, mwin) > 0;
}

cudaError_t launch_lis_attention_win(const LisArgs &a, const AttnVArgs &b, cudaStream_t st)
{
    const bool bias = a.bias != nullptr;
    WinParams p{a.logits, a.ld_logit, b.v, b.ld_v, b.acc, b.ld_acc, a.bias, a.heads, a.window, b.BH, a.L, b.zp_v,
                iexp_consts_host(a.s_logit), 0, 0, b.out8, b.ld_out8, b.rq_n1, b.rq_n2, b.rq_zp,
                a.region, a.n_windows, a.mask_value < -1024 ? 1024 : -a.mask_value};
    const int mwin = a.region ? a.n_windows : 0;
    p.ne = win_table_entries(p.ic, bias);
    p.ng = win_groups(p.ne, a.heads, a.L, a.window, bias, mwin);
    const size_t smem = win_smem_bytes(p.ng, p.ne, a.heads, a.L, bias, mwin);
    const int64_t ntiles = (b.BH + 1) / 2;
    const int64_t want = (ntiles + p.ng - 1) / p.ng;
    const int grid = (int)(want < sm_count() ? want : sm_count());
    const bool se = small_iexp_w(p.ic);
    const bool mask = a.region != nullptr;
    return b.d == 32 ? win_launch_d<32>(bias, mask, se, p, smem, grid, st)
                     : win_launch_d<64>(bias, mask, se, p, smem, grid, st);
}

cudaError_t read_clear_win_status(int *status)
{
    int zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(status, g_status, sizeof(int));
    if (e != cudaSuccess) return e;
    return cudaMemcpyToSymbol(g_status, &zero, sizeof(int));
}

}  // namespace fqvit
