// heads.cu -- the layout steps between the Linear layers and the attention core of a block: the
// QKV Linear's token-major output split into head-major Q, K and V codes, and the attention
// output's head-major rows merged back into token rows for the projection (Fig. 4 dataflow; the
// 8-bit codes are moved, not changed, except the shift to the signed form the attention kernels
// take).  Byte moves in 16-byte units, grid-stride, HBM-bound.
#include "fqvit_internal.cuh"

namespace fqvit {

namespace {

// qkv [B L][ld_qkv] uint8, part p (0 q, 1 k, 2 v) at columns p H d .. , head h at + h d;
// q/k/v [B H][L][ld_head] int8 = code - 128
__global__ void split_qkv_kernel(HeadsArgs a)
{
    pdl_release();
    pdl_wait();
    const int cpr = a.d >> 4;  // 16-byte chunks per head row
    const int64_t per_part = a.B * a.H * a.L * cpr;
    const int64_t total = 3 * per_part;
    for (int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; g < total; g += (int64_t)gridDim.x * blockDim.x) {
        const int p = (int)(g / per_part);
        int64_t r = g - p * per_part;
        const int c = (int)(r % cpr);
        r /= cpr;  // (b H + h) L + i
        const int i = (int)(r % a.L);
        const int64_t bh = r / a.L;
        const int h = (int)(bh % a.H);
        const int64_t b = bh / a.H;
        const uint4 v = *reinterpret_cast<const uint4 *>(a.src + (b * a.L + i) * a.ld_src +
                                                         ((int64_t)p * a.H + h) * a.d + 16 * c);
        int8_t *dst = p == 0 ? a.q : p == 1 ? a.k : a.v;
        *reinterpret_cast<uint4 *>(dst + r * a.ld_dst + 16 * c) =
            make_uint4(v.x ^ 0x80808080u, v.y ^ 0x80808080u, v.z ^ 0x80808080u, v.w ^ 0x80808080u);
    }
}

// src [B H][L][ld_src] uint8 -> dst [B L][ld_dst] uint8, head h at columns h d ..
__global__ void merge_heads_kernel(HeadsArgs a)
{
    pdl_release();
    pdl_wait();
    const int cpr = a.d >> 4;
    const int64_t total = a.B * a.H * a.L * cpr;
    for (int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; g < total; g += (int64_t)gridDim.x * blockDim.x) {
        const int c = (int)(g % cpr);
        int64_t r = g / cpr;  // token row (b L + i), head h: r = (b L + i) H + h
        const int h = (int)(r % a.H);
        r /= a.H;
        const int i = (int)(r % a.L);
        const int64_t b = r / a.L;
        const uint4 v = *reinterpret_cast<const uint4 *>(a.src_u8 + ((b * a.H + h) * a.L + i) * a.ld_src + 16 * c);
        *reinterpret_cast<uint4 *>(a.dst_u8 + r * a.ld_dst + (int64_t)h * a.d + 16 * c) = v;
    }
}

int heads_grid(int64_t chunks)
{
    const int64_t cap = (int64_t)sm_count() * 8;
    const int64_t want = (chunks + 255) / 256;
    return (int)(want < cap ? (want < 1 ? 1 : want) : cap);
}

}  // namespace

cudaError_t launch_split_qkv(const HeadsArgs &a, cudaStream_t st)
{
    const int64_t chunks = 3 * a.B * a.H * a.L * (a.d >> 4);
    return launch_pdl(split_qkv_kernel, dim3(heads_grid(chunks)), dim3(256), 0, st, a);
}

cudaError_t launch_merge_heads(const HeadsArgs &a, cudaStream_t st)
{
    const int64_t chunks = a.B * a.H * a.L * (a.d >> 4);
    return launch_pdl(merge_heads_kernel, dim3(heads_grid(chunks)), dim3(256), 0, st, a);
}

}  // namespace fqvit
