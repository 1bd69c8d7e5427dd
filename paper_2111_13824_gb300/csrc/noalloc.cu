// noalloc.cu -- fqvit_calibrate_ptf_noalloc: PTF calibration for callers that
// cannot allocate device memory.
//
// fqvit_calibrate_ptf needs a caller-provided device workspace (per-block
// min / max partials and the per-channel error sums).  Some callers cannot
// obtain one: code that must not allocate device memory once it is running
// (real-time or certified inference with a fixed memory budget), and code
// whose device memory belongs to another allocator that will not hand out a
// separate buffer.  This entry point runs the same calibration kernels with
// their workspace in a fixed array of device memory that the library itself
// reserves when it is loaded, so the call allocates nothing.
//
// The array lives for as long as the library is loaded, on every GPU that
// loads it (kNoAllocScratchBytes each).  All calls share it and it keeps the
// contents of the last call; nothing in it has to start at zero (every byte a
// call reads was written earlier in the same call).  Two calls whose kernels
// overlap on the GPU -- on different streams, or from different host threads
// -- race on the array; serialise them.
#include "fqvit.h"
#include "fqvit_internal.cuh"

#include <mutex>

namespace {

// Room for the workspace of C * (K + 1) <= kNoAllocMaxSums error sums.
constexpr size_t kNoAllocScratchBytes = 160 * 1024;
constexpr int64_t kNoAllocMaxSums = 16384;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

// Device address of g_noalloc_scratch, resolved once per device with that
// device current.  (In host code the array's name is only a host-side handle.)
constexpr int kMaxDevices = 64;
void *g_scratch_addr[kMaxDevices] = {nullptr};
std::mutex g_scratch_mu;

cudaError_t scratch_for_current_device(void **out)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    if (g_scratch_addr[dev] == nullptr) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) return e;
        g_scratch_addr[dev] = p;
    }
    *out = g_scratch_addr[dev];
    return cudaSuccess;
}

}  // namespace

extern "C" {

int fqvit_calibrate_ptf_noalloc(const float *x, int64_t rows, int32_t C, int64_t ld_x, int32_t bits,
                                int32_t K, float *s, int32_t *zp, uint8_t *alpha, double *sse_opt,
                                void *stream)
{
    using fqvit::record_error;
    if (!x || !s || !zp || !alpha) return record_error(FQVIT_ERR_INVALID_ARG, "calibrate_ptf_noalloc: NULL pointer");
    if (rows < 1 || C < 1 || C > 8192 || ld_x < C)
        return record_error(FQVIT_ERR_INVALID_ARG, "calibrate_ptf_noalloc: bad shape");
    if (bits != 8) return record_error(FQVIT_ERR_UNSUPPORTED, "calibrate_ptf_noalloc: bits must be 8");
    if (K < 0 || K > 7) return record_error(FQVIT_ERR_UNSUPPORTED, "calibrate_ptf_noalloc: K must be 0..7");
    if ((int64_t)C * (K + 1) > kNoAllocMaxSums ||
        fqvit::calibrate_workspace_bytes(rows, C, K) > kNoAllocScratchBytes)
        return record_error(FQVIT_ERR_UNSUPPORTED,
                            "calibrate_ptf_noalloc: C*(K+1) exceeds 16384, the size of the library's fixed "
                            "scratch; use fqvit_calibrate_ptf with a workspace");
    if ((reinterpret_cast<uintptr_t>(x) % 4) || (reinterpret_cast<uintptr_t>(s) % 4) ||
        (reinterpret_cast<uintptr_t>(zp) % 4) || (sse_opt && (reinterpret_cast<uintptr_t>(sse_opt) % 8)))
        return record_error(FQVIT_ERR_INVALID_ARG, "calibrate_ptf_noalloc: misaligned pointer");
    void *ws = nullptr;
    cudaError_t e = scratch_for_current_device(&ws);
    if (e != cudaSuccess)
        return record_error(FQVIT_ERR_CUDA, "calibrate_ptf_noalloc: cannot resolve the scratch address");
    e = fqvit::launch_calibrate(x, rows, C, ld_x, K, s, zp, alpha, sse_opt, ws,
                                reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return record_error(FQVIT_ERR_CUDA, "calibrate_ptf_noalloc: launch failed");
    return record_error(FQVIT_OK, "");
}

}  // extern "C"
