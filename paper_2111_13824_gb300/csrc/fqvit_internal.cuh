// fqvit_internal.cuh -- declarations shared by the host entry points
// (api.cu) and the kernel files.  Nothing here is part of the public ABI.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace fqvit {

// Number of SMs of the current device (cached per device).
int sm_count();

// Launch check of a kernel's shared memory: the compiled static size (as the runtime reports it,
// not an estimate) plus `dynamic` bytes within the device's opt-in limit per block.  Returns
// cudaErrorInvalidConfiguration when they do not fit, or the runtime's error.
cudaError_t check_smem_fits(const void *kernel, size_t dynamic);

// Programmatic dependent launch.  The step's kernels are launched with programmatic stream
// serialization: the next kernel's CTAs may start (and run their set-up: barriers, tensor
// memory, tables computed from arguments) while the previous kernel's last CTAs finish.  Every
// such kernel calls pdl_release() at entry and pdl_wait() before its first access to global
// memory (read or write): the wait returns once the previous grid has completed and its writes
// are visible, so the data dependencies of the stream stay as in a plain launch.  Without the
// launch attribute both are no-ops.
__device__ __forceinline__ void pdl_release() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

template <typename... Params, typename... Args>
cudaError_t launch_pdl(void (*kernel)(Params...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                       Args &&...args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args &&>(args)...);
}

// Sets the thread's fqvit_last_error message (empty for FQVIT_OK); returns code.
int record_error(int code, const char *msg);

// ---- PTF calibration / quantizer (ptf.cu) ---------------------------------
// Workspace of launch_calibrate; with sums == false the caller's sse buffer holds the error sums.
size_t calibrate_workspace_bytes(int64_t rows, int C, int K, bool sums = true);

// Eqs. 8-9 from the calibration range, shared by the device path and the host
// combine of sharded calibration: s0 = (mx - mn) / 255 (a zero range counts
// as 1) is 2^K s, zp = clip(rint(-mn / s0), 0, 255).  Every operation is a
// single IEEE round-to-nearest one, so host and device agree bit for bit.
__host__ __device__ inline void calib_scale(float mn, float mx, int K, float &s0, float &s, int32_t &zp)
{
    float range = mx - mn;
    if (range == 0.0f) range = 1.0f;
    s0 = range / 255.0f;
#ifdef __CUDA_ARCH__
    s = s0 * __int_as_float((127 - K) << 23);  // s0 / 2^K, exact
#else
    s = ldexpf(s0, -K);
#endif
    const float t = -mn / s0;
    zp = (int32_t)fminf(fmaxf(rintf(t), 0.0f), 255.0f);
}

// Per-rank stages of a calibration batch split by rows (sharded calibration):
// the shard's exact (min, max) into mnmx[2], and the shard's Eq. 10 sums for
// the global range mnmx[2] into sse[C][K+1].
cudaError_t launch_calibrate_minmax(const float *x, int64_t rows, int C, int64_t ld_x, float *mnmx, void *ws,
                                    cudaStream_t st);
cudaError_t launch_calibrate_sse_partial(const float *x, int64_t rows, int C, int64_t ld_x, int K,
                                         const float *mnmx, double *sse, void *ws, cudaStream_t st);
cudaError_t launch_calibrate(const float *x, int64_t rows, int C, int64_t ld_x, int K, float *s,
                             int32_t *zp, uint8_t *alpha, double *sse, void *ws,
                             cudaStream_t st);
cudaError_t launch_quantize(const float *x, int64_t rows, int C, int64_t ld_x, float s,
                            int32_t zp, const uint8_t *alpha, uint8_t *xq, int64_t ld_q,
                            cudaStream_t st);

// ---- integer LayerNorm (layernorm.cu) -------------------------------------
struct LnArgs {
    const uint8_t *xq;
    int64_t rows;
    int C;
    int64_t ld_in;
    int zp_in;
    const uint8_t *alpha;
    const float *gamma;
    const float *beta;
    float s_out;
    int zp_out;
    uint8_t *yq;
    int64_t ld_out;
    int64_t *m1;
    int64_t *m2;
};
cudaError_t launch_layernorm(const LnArgs &a, cudaStream_t st);

// ---- head split and merge of a block (heads.cu) ------------------------------
struct HeadsArgs {
    const uint8_t *src;      // split: the QKV Linear's output [B L][ld_src]
    const uint8_t *src_u8;   // merge: attention output [B H][L][ld_src]
    int8_t *q, *k, *v;       // split: [B H][L][ld_dst]
    uint8_t *dst_u8;         // merge: [B L][ld_dst]
    int64_t B;
    int H, L, d;
    int64_t ld_src, ld_dst;
};
cudaError_t launch_split_qkv(const HeadsArgs &a, cudaStream_t st);
cudaError_t launch_merge_heads(const HeadsArgs &a, cudaStream_t st);
// Reads and clears the LayerNorm kernels' status word (5: a bounded wait gave up).
cudaError_t read_clear_ln_status(int *status);

// ---- Log-Int-Softmax and BitShift attention (lis.cu) -----------------------
struct LisArgs {
    const int8_t *logits;
    int64_t n_rows;  // BH * L
    int L;
    int64_t ld_logit;
    float s_logit;
    const int8_t *bias;  // [heads][(2w-1)^2] or nullptr
    int heads;
    int window;
    uint8_t *codes;  // packed nibbles or nullptr
    int64_t ld_codes;
    uint64_t *rowsum;  // or nullptr
    // shifted-window mask: region ids [n_windows][L] or nullptr; mask_value (-32768 .. 0) is added
    // where a query's and a key's regions differ; window of row r: (r / (L heads)) % n_windows
    const uint8_t *region = nullptr;
    int n_windows = 1;
    int mask_value = 0;
};
cudaError_t launch_lis_softmax(const LisArgs &a, cudaStream_t st);

struct AttnVArgs {
    const uint8_t *codes;
    int64_t ld_codes;
    const int8_t *v;
    int64_t ld_v;
    int zp_v;
    int64_t BH;
    int L;
    int d;
    int32_t *acc;
    int64_t ld_acc;
    int32_t *range_flag;
    // 8-bit output instead of acc (fused attention only): y = clip(((n2 acc + 2^(n1-1)) >> n1)
    // + zp, 0, 255) for n1 > 0, clip(n2 acc 2^-n1 + zp, 0, 255) for -10 <= n1 <= 0
    uint8_t *out8 = nullptr;
    int64_t ld_out8 = 0;
    int rq_n1 = 0;
    int rq_n2 = 0;
    int rq_zp = 0;
};
cudaError_t launch_lis_attn_v(const AttnVArgs &a, cudaStream_t st);

// fused softmax + attn.V; codes written only when a.codes != nullptr
cudaError_t launch_lis_attention(const LisArgs &a, const AttnVArgs &b, cudaStream_t st);

// Q K^T with its 8-bit output quantizer on the tensor cores (qk_tc.cu):
// logit = clip(floor((n2 P + 2^(n1-1)) / 2^n1) + zp_l, -128, 127), P = (Q - zp_q)(K - zp_k)^T
struct QkArgs {
    const int8_t *q;
    int64_t ld_q;
    int zp_q;
    const int8_t *k;
    int64_t ld_k;
    int zp_k;
    int64_t BH;
    int L;
    int d;
    int n1, n2, zp_l;
    int8_t *logits;
    int64_t ld_logit;
};
bool qk_logits_supported(const QkArgs &a);
cudaError_t launch_qk_logits(const QkArgs &a, cudaStream_t st);
cudaError_t read_clear_qk_status(int *status);

// tensor-core (tcgen05) fused path for rows of 65 .. 592 keys (lis_tc.cu); rows of 128 .. 384 keys
// take tiles packed across heads
bool lis_attention_tc_eligible(const LisArgs &a, const AttnVArgs &b);
cudaError_t launch_lis_attention_tc(const LisArgs &a, const AttnVArgs &b, cudaStream_t st);

// tensor-core fused path for rows of at most 64 keys, two heads per MMA tile, with
// the optional relative-position bias (lis_win.cu)
bool lis_attention_win_eligible(const LisArgs &a, const AttnVArgs &b);
cudaError_t launch_lis_attention_win(const LisArgs &a, const AttnVArgs &b, cudaStream_t st);
cudaError_t read_clear_win_status(int *status);

// ---- MinMax Linear layer on the tensor cores (linear_tc.cu) ----------------
struct LinearArgs {
    const uint8_t *x;
    int64_t M, ld_x;
    int K, zp_x;
    float s_x;
    const uint16_t *w_h;  // fp16 [N][K]
    int N;
    const float *s_w;
    const int32_t *bias;  // may be NULL
    float s_y;
    int zp_y;
    uint8_t *y;
    int64_t ld_y;
    int32_t *acc;  // may be NULL
    int64_t ld_acc;
    uint16_t *xh;  // workspace: fp16 [M][K]
};
bool linear_supported(const LinearArgs &a);
cudaError_t launch_linear(const LinearArgs &a, cudaStream_t st);
// Workspace of launch_linear: the fp16 copy of x (M K 2 bytes, rounded up to 256) and 4096 int32 weight sums.
size_t linear_workspace_bytes(int64_t M, int K);
cudaError_t launch_linear_pack_weight(const int8_t *w, int N, int K, int64_t ld_w, uint16_t *w_h, cudaStream_t st);
cudaError_t read_clear_linear_status(int *status);
// one CTA whose wait on an mbarrier that nothing completes gives up (the bounded wait's timeout)
cudaError_t launch_bounded_wait_probe(cudaStream_t st);

// Synchronizes st, returns the device status word of the attention and LayerNorm kernels
// (0 ok, 5 a bounded wait timed out) and clears it; the Linear layers' word is read by
// read_clear_linear_status.
cudaError_t read_clear_device_status(int *status, cudaStream_t st);

// Attention implementation choice: 0 automatic, 1 CUDA cores only (FQVIT_ATTN_PATH=cuda_core),
// 2 no short-row kernel (FQVIT_ATTN_PATH=no_window: rows of at most 64 keys take the
// one-head-per-tile tensor-core kernel when it applies).
int attention_path_override();

}  // namespace fqvit
