// lis.cu -- Log-Int-Softmax (supplement Algorithms 1-2, Eqs. 16-17, 33) and
// the BitShift attention times values (Eq. 15) on CUDA cores.
//
// i-exp.  For a logit scale s the values e(q~) for every q~ in [-287, 0]
// (int8 logits, plus an int8 relative-position bias) are tabulated in
// shared memory by each block.  For s in [2^-7, 1/2], q_L = (q_p + q_b)^2 + q_c
// is below 2^16, so e = q_L << (15 - z) fits 31 bits and is exact in fp32.
//
// Log2 code without a division.  I-Log2(x) >= k exactly when x >= T_k
// (T_1 = 2, T_k = 3 * 2^(k-2)), and round(S/e) >= T exactly when
// 2S >= (2T - 1) e.  With D_k = 2 T_k - 1 (3, 5, 11, 23, ..., 3 * 2^(k-1) - 1)
// the code is #{k <= 15 : e D_k <= 2S}.  Every D_k lies strictly between
// 2^k and 2^(k+1), so if 2S/e lies in [2^k, 2^(k+1)) the code is k - 1 or k
// and only the test e D_k <= 2S is left.  k = floor(log2(2S/e)) comes from
// the difference of the fp32 bit patterns of 2S (rounded) and e; rounding 2S
// can move k by one only where the remaining test is decided anyway.  The
// test itself is exact: with 2S = hi + lo (hi = fp32(2S), lo exact), the sign
// of fma(e, D_k, -hi) is the sign of e D_k - hi, and it is either exact or
// larger in magnitude than |lo|.
#include "fqvit_internal.cuh"
#include "lis_common.cuh"

#include <cstdlib>
#include <cstring>

namespace fqvit {

namespace {

using namespace lis;

// Codes of one row by one warp.  Lane owns keys 4*(lane + 32 i) .. +3.
// dst: packed nibbles (global or shared), written for bytes < ceil(L/2).
// reg: the window's region ids [L] when a shifted-window mask is given (else nullptr): key j of
// query qi gets mask_value where reg[j] != reg[qi]
template <int NW, bool BIAS>
__device__ void softmax_row(const int8_t *__restrict__ src, int L, const uint32_t *lut,
                            const int8_t *btab /* shared [(2w-1)^2] of this head */, int qi,
                            int w, uint8_t *dst, uint64_t *rowsum_dst, const uint8_t *reg, int mask_value)
{
    const int lane = threadIdx.x & 31;
    const int nwords = (L + 3) >> 2;
    const uint32_t *s32 = reinterpret_cast<const uint32_t *>(src);
    int val[NW][4];
    int m = -100000;
#pragma unroll
    for (int i = 0; i < NW; ++i) {
        int widx = lane + 32 * i;
        uint32_t word = widx < nwords ? __ldcs(s32 + widx) : 0u;
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            int key = 4 * widx + b;
            int q = (int)(int8_t)(word >> (8 * b));
            if (BIAS && key < L) q += btab[relpos_idx(qi, key, w)];
            if (reg && key < L && reg[key] != reg[qi]) q += mask_value;
            val[i][b] = q;
            if (key < L) m = max(m, q);
        }
    }
    m = __reduce_max_sync(0xffffffffu, m);
    unsigned long long S = 0;
    uint32_t e[NW][4];
#pragma unroll
    for (int i = 0; i < NW; ++i) {
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            int key = 4 * (lane + 32 * i) + b;
            uint32_t ev = key < L ? lut[min(m - val[i][b], kLutSize - 1)] : 0u;
            e[i][b] = ev;
            S += ev;
        }
    }
    for (int o = 16; o > 0; o >>= 1) S += __shfl_xor_sync(0xffffffffu, S, o);
    if (rowsum_dst && lane == 0) *rowsum_dst = (uint64_t)S;
    const RowSum rs = make_rowsum(S);
    const int nbytes = (L + 1) >> 1;
#pragma unroll
    for (int i = 0; i < NW; ++i) {
        int widx = lane + 32 * i;
        if (widx < nwords) {
            uint32_t packed = 0;
#pragma unroll
            for (int b = 0; b < 4; ++b) {
                int key = 4 * widx + b;
                uint32_t c = key < L ? lis_code(e[i][b], rs) : 0u;
                packed |= c << (4 * b);
            }
            int byte0 = 2 * widx;
            if (byte0 + 1 < nbytes) {
                dst[byte0] = (uint8_t)packed;
                dst[byte0 + 1] = (uint8_t)(packed >> 8);
            } else if (byte0 < nbytes) {
                dst[byte0] = (uint8_t)packed;
            }
        }
    }
}

template <int NW, bool BIAS>
__global__ void __launch_bounds__(256) lis_softmax_kernel(LisArgs a, IexpC ic)
{
    __shared__ uint32_t lut[kLutSize];
    extern __shared__ int8_t btab_all[];  // [heads][(2w-1)^2] when BIAS
    build_lut(lut, ic);
    const int nb = (2 * a.window - 1) * (2 * a.window - 1);
    if (BIAS)
        for (int i = threadIdx.x; i < a.heads * nb; i += blockDim.x) btab_all[i] = a.bias[i];
    __syncthreads();
    const int warp = threadIdx.x >> 5;
    const int nwarps = blockDim.x >> 5;
    for (int64_t row = (int64_t)blockIdx.x * nwarps + warp; row < a.n_rows;
         row += (int64_t)gridDim.x * nwarps) {
        const int qi = (int)(row % a.L);
        const int8_t *bt = nullptr;
        if (BIAS) bt = btab_all + (int)((row / a.L) % a.heads) * nb;
        const uint8_t *reg = a.region ? a.region + (row / ((int64_t)a.L * a.heads)) % a.n_windows * a.L : nullptr;
        softmax_row<NW, BIAS>(a.logits + row * a.ld_logit, a.L, lut, bt, qi, a.window,
                              a.codes + row * a.ld_codes, a.rowsum ? a.rowsum + row : nullptr, reg, a.mask_value);
    }
}

// BitShift accumulate for one (row, column group) over all keys.
// codes_row: packed nibbles; vs: V of the head in shared memory [L][d].
template <int CPT>
__device__ __forceinline__ void attnv_row(const uint8_t *codes_row, const int8_t *vs, int L,
                                          int d, int col0, int zp, int acc[CPT], long long &wsum)
{
#pragma unroll
    for (int k = 0; k < CPT; ++k) acc[k] = 0;
    wsum = 0;
    for (int j = 0; j < L; ++j) {
        uint32_t c = (codes_row[j >> 1] >> (4 * (j & 1))) & 0xF;
        int w = 1 << (15 - c);
        wsum += w;
        const int8_t *vr = vs + j * d + col0;
        if (CPT == 8) {
            uint2 p = *reinterpret_cast<const uint2 *>(vr);
            uint32_t pw[2] = {p.x, p.y};
#pragma unroll
            for (int k = 0; k < 8; ++k) acc[k] += ((int)(int8_t)(pw[k >> 2] >> (8 * (k & 3))) - zp) * w;
        } else {
            uint32_t p = *reinterpret_cast<const uint32_t *>(vr);
#pragma unroll
            for (int k = 0; k < CPT; ++k) acc[k] += ((int)(int8_t)(p >> (8 * k)) - zp) * w;
        }
    }
}

constexpr int kRowsPerBlock = 32;

// acc for 32 query rows of one head; 8 threads per row, d/8 columns each.
template <int CPT>
__global__ void __launch_bounds__(256) lis_attn_v_kernel(AttnVArgs a)
{
    extern __shared__ __align__(16) unsigned char sm[];
    int8_t *vs = reinterpret_cast<int8_t *>(sm);                       // [L][d]
    uint8_t *cs = reinterpret_cast<uint8_t *>(sm + ((a.L * a.d + 15) & ~15));  // [32][ldc]
    const int ldc = (a.L + 1) >> 1;
    const int64_t bh = blockIdx.y;
    const int row0 = blockIdx.x * kRowsPerBlock;
    const int8_t *vh = a.v + bh * (int64_t)a.L * a.ld_v;
    for (int i = threadIdx.x; i < a.L * a.d; i += blockDim.x) {
        int j = i / a.d, t = i - j * a.d;
        vs[i] = vh[(int64_t)j * a.ld_v + t];
    }
    for (int i = threadIdx.x; i < kRowsPerBlock * ldc; i += blockDim.x) {
        int r = i / ldc, b = i - r * ldc;
        int row = row0 + r;
        cs[i] = row < a.L ? a.codes[(bh * a.L + row) * a.ld_codes + b] : 0;
    }
    __syncthreads();
    const int r = threadIdx.x >> 3, g = threadIdx.x & 7;
    const int row = row0 + r;
    if (row >= a.L) return;
    int acc[CPT];
    long long wsum;
    attnv_row<CPT>(cs + r * ldc, vs, a.L, a.d, g * CPT, a.zp_v, acc, wsum);
    if (a.range_flag && wsum * (128 + (a.zp_v < 0 ? -a.zp_v : a.zp_v)) >= (1LL << 31)) *a.range_flag = 1;
    int32_t *dst = a.acc + (bh * a.L + row) * a.ld_acc + g * CPT;
#pragma unroll
    for (int k = 0; k < CPT; ++k) dst[k] = acc[k];
}

// Fused: codes of 32 rows into shared memory, then the accumulate.
template <int NW, bool BIAS, int CPT>
__global__ void __launch_bounds__(256) lis_attention_kernel(LisArgs la, AttnVArgs a, IexpC ic)
{
    extern __shared__ __align__(16) unsigned char sm[];
    __shared__ uint32_t lut[kLutSize];
    int8_t *vs = reinterpret_cast<int8_t *>(sm);
    size_t off = ((size_t)a.L * a.d + 15) & ~(size_t)15;
    uint8_t *cs = reinterpret_cast<uint8_t *>(sm + off);
    const int ldc = (a.L + 1) >> 1;
    off += ((size_t)kRowsPerBlock * ldc + 15) & ~(size_t)15;
    int8_t *btab_all = reinterpret_cast<int8_t *>(sm + off);
    const int nb = (2 * la.window - 1) * (2 * la.window - 1);

    build_lut(lut, ic);
    if (BIAS)
        for (int i = threadIdx.x; i < la.heads * nb; i += blockDim.x) btab_all[i] = la.bias[i];
    const int64_t bh = blockIdx.y;
    const int row0 = blockIdx.x * kRowsPerBlock;
    const int8_t *vh = a.v + bh * (int64_t)a.L * a.ld_v;
    for (int i = threadIdx.x; i < a.L * a.d; i += blockDim.x) {
        int j = i / a.d, t = i - j * a.d;
        vs[i] = vh[(int64_t)j * a.ld_v + t];
    }
    __syncthreads();
    const int warp = threadIdx.x >> 5;
    for (int r = warp; r < kRowsPerBlock; r += 8) {
        int row = row0 + r;
        if (row < a.L) {
            int64_t grow = bh * a.L + row;
            const int8_t *bt = BIAS ? btab_all + (int)(bh % la.heads) * nb : nullptr;
            const uint8_t *reg = la.region ? la.region + (bh / la.heads) % la.n_windows * a.L : nullptr;
            softmax_row<NW, BIAS>(la.logits + grow * la.ld_logit, a.L, lut, bt, row, la.window,
                                  cs + r * ldc, la.rowsum ? la.rowsum + grow : nullptr, reg, la.mask_value);
        }
    }
    __syncthreads();
    if (la.codes) {
        for (int i = threadIdx.x; i < kRowsPerBlock * ldc; i += blockDim.x) {
            int r = i / ldc, b = i - r * ldc;
            int row = row0 + r;
            if (row < a.L) la.codes[(bh * a.L + row) * la.ld_codes + b] = cs[i];
        }
    }
    const int r = threadIdx.x >> 3, g = threadIdx.x & 7;
    const int row = row0 + r;
    if (row >= a.L) return;
    int acc[CPT];
    long long wsum;
    attnv_row<CPT>(cs + r * ldc, vs, a.L, a.d, g * CPT, a.zp_v, acc, wsum);
    if (a.out8) {  // 8-bit output for the next layer instead of the accumulators
        uint8_t *d8 = a.out8 + (bh * a.L + row) * a.ld_out8 + g * CPT;
#pragma unroll
        for (int k = 0; k < CPT; ++k) d8[k] = (uint8_t)requant8(acc[k], a.rq_n1, a.rq_n2, a.rq_zp);
        return;
    }
    int32_t *dst = a.acc + (bh * a.L + row) * a.ld_acc + g * CPT;
#pragma unroll
    for (int k = 0; k < CPT; ++k) dst[k] = acc[k];
}

template <int NW, bool BIAS>
cudaError_t softmax_launch(const LisArgs &a, cudaStream_t st)
{
    int nsm = sm_count();
    int64_t want = (a.n_rows + 7) / 8;
    int64_t cap = (int64_t)nsm * 8;
    int blocks = (int)(want < cap ? want : cap);
    size_t smem = BIAS ? (size_t)a.heads * (2 * a.window - 1) * (2 * a.window - 1) : 0;
    if (smem > 48 * 1024)
        cudaFuncSetAttribute(lis_softmax_kernel<NW, BIAS>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
    lis_softmax_kernel<NW, BIAS><<<blocks, 256, smem, st>>>(a, iexp_consts_host(a.s_logit));
    return cudaGetLastError();
}

template <bool BIAS>
cudaError_t softmax_dispatch(const LisArgs &a, cudaStream_t st)
{
    int nw = ((a.L + 3) / 4 + 31) / 32;
    switch (nw) {
    case 1: return softmax_launch<1, BIAS>(a, st);
    case 2: return softmax_launch<2, BIAS>(a, st);
    case 3: return softmax_launch<3, BIAS>(a, st);
    case 4: return softmax_launch<4, BIAS>(a, st);
    case 5: return softmax_launch<5, BIAS>(a, st);
    case 6: return softmax_launch<6, BIAS>(a, st);
    case 7: return softmax_launch<7, BIAS>(a, st);
    default: return softmax_launch<8, BIAS>(a, st);
    }
}

template <int NW, bool BIAS>
cudaError_t fused_launch(const LisArgs &la, const AttnVArgs &a, cudaStream_t st)
{
    size_t smem = (((size_t)a.L * a.d + 15) & ~(size_t)15) +
                  (((size_t)kRowsPerBlock * ((a.L + 1) / 2) + 15) & ~(size_t)15) +
                  (BIAS ? (size_t)la.heads * (2 * la.window - 1) * (2 * la.window - 1) : 0);
    dim3 g((a.L + kRowsPerBlock - 1) / kRowsPerBlock, (unsigned)a.BH);
    if (a.d == 64) {
        cudaFuncSetAttribute(lis_attention_kernel<NW, BIAS, 8>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        lis_attention_kernel<NW, BIAS, 8><<<g, 256, smem, st>>>(la, a, iexp_consts_host(la.s_logit));
    } else {
        cudaFuncSetAttribute(lis_attention_kernel<NW, BIAS, 4>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        lis_attention_kernel<NW, BIAS, 4><<<g, 256, smem, st>>>(la, a, iexp_consts_host(la.s_logit));
    }
    return cudaGetLastError();
}

template <bool BIAS>
cudaError_t fused_dispatch(const LisArgs &la, const AttnVArgs &a, cudaStream_t st)
{
    int nw = ((a.L + 3) / 4 + 31) / 32;
    switch (nw) {
    case 1: return fused_launch<1, BIAS>(la, a, st);
    case 2: return fused_launch<2, BIAS>(la, a, st);
    case 3: return fused_launch<3, BIAS>(la, a, st);
    case 4: return fused_launch<4, BIAS>(la, a, st);
    case 5: return fused_launch<5, BIAS>(la, a, st);
    case 6: return fused_launch<6, BIAS>(la, a, st);
    case 7: return fused_launch<7, BIAS>(la, a, st);
    default: return fused_launch<8, BIAS>(la, a, st);
    }
}

}  // namespace

cudaError_t launch_lis_softmax(const LisArgs &a, cudaStream_t st)
{
    return a.bias ? softmax_dispatch<true>(a, st) : softmax_dispatch<false>(a, st);
}

cudaError_t launch_lis_attn_v(const AttnVArgs &a, cudaStream_t st)
{
    size_t smem = (((size_t)a.L * a.d + 15) & ~(size_t)15) + (size_t)kRowsPerBlock * ((a.L + 1) / 2);
    dim3 g((a.L + kRowsPerBlock - 1) / kRowsPerBlock, (unsigned)a.BH);
    if (a.d == 64) {
        cudaFuncSetAttribute(lis_attn_v_kernel<8>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        lis_attn_v_kernel<8><<<g, 256, smem, st>>>(a);
    } else {
        cudaFuncSetAttribute(lis_attn_v_kernel<4>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        lis_attn_v_kernel<4><<<g, 256, smem, st>>>(a);
    }
    return cudaGetLastError();
}

int attention_path_override()
{
    const char *e = getenv("FQVIT_ATTN_PATH");
    if (e && strcmp(e, "cuda_core") == 0) return 1;
    if (e && strcmp(e, "no_window") == 0) return 2;
    return 0;
}

cudaError_t launch_lis_attention(const LisArgs &la, const AttnVArgs &a, cudaStream_t st)
{
    const int path = attention_path_override();
    if (path == 0 && lis_attention_win_eligible(la, a)) return launch_lis_attention_win(la, a, st);
    if (path != 1 && lis_attention_tc_eligible(la, a)) return launch_lis_attention_tc(la, a, st);
    return la.bias ? fused_dispatch<true>(la, a, st) : fused_dispatch<false>(la, a, st);
}

}  // namespace fqvit
