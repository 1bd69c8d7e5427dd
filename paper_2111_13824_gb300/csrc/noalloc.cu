// noalloc.cu -- fqvit_calibrate_ptf_noalloc: PTF calibration for callers that
// cannot allocate device memory.
//
// fqvit_calibrate_ptf needs a caller-provided device workspace (per-block
// min / max partials and the per-channel error sums).  Some callers cannot
// obtain one: code that must not allocate device memory once it is running
// (real-time or certified inference with a fixed memory budget), and code
// whose device memory belongs to another allocator that will not hand out a
// separate buffer.  This entry point runs the same calibration kernels with
// their workspace in a fixed array of device memory that belongs to the
// library, so the call allocates nothing.
//
// The array is reserved on a GPU when the library's code is loaded there.
// With CUDA's default lazy module loading that happens on the first call on
// that GPU (the address lookup below loads the module), so that first call may
// take device memory and should be made at start-up, before the memory budget
// is fixed and before any stream capture (CUDA_MODULE_LOADING=EAGER reserves it
// when the context is created instead).  From then on the array stays until
// the process ends or the context is reset (kNoAllocScratchBytes per GPU).
// All calls share it and it keeps the contents of the last call; nothing in it
// has to start at zero (every byte a call reads was written earlier in the
// same call).  Two calls whose kernels overlap on the GPU -- on different
// streams, or from different host threads -- race on the array; serialise
// them.
#include "fqvit.h"
#include "fqvit_internal.cuh"

#include <cstdio>

namespace {

// Room for the workspace with C * (K + 1) <= kNoAllocMaxSums error sums kept in the array (the
// sums need no room when the caller passes sse_opt).
constexpr size_t kNoAllocScratchBytes = 160 * 1024;
constexpr int64_t kNoAllocMaxSums = 16384;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

// Device address of g_noalloc_scratch on the current device.  (In host code the array's name is
// only a host-side handle.)  Looked up on every call: it is cheap once the module is loaded, and
// an address kept from an earlier context would be stale after a reset.
cudaError_t scratch_for_current_device(void **out) { return cudaGetSymbolAddress(out, g_noalloc_scratch); }

int cuda_error(const char *what, cudaError_t e)
{
    char msg[256];
    std::snprintf(msg, sizeof msg, "calibrate_ptf_noalloc: %s: %s", what, cudaGetErrorString(e));
    return fqvit::record_error(FQVIT_ERR_CUDA, msg);
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
    // the error sums go to the array only when the caller passes no sse buffer
    if ((!sse_opt && (int64_t)C * (K + 1) > kNoAllocMaxSums) ||
        fqvit::calibrate_workspace_bytes(rows, C, K, sse_opt == nullptr) > kNoAllocScratchBytes)
        return record_error(FQVIT_ERR_UNSUPPORTED,
                            "calibrate_ptf_noalloc: C*(K+1) exceeds 16384, the error sums the library's fixed "
                            "scratch holds; pass sse_opt, or use fqvit_calibrate_ptf with a workspace");
    if ((reinterpret_cast<uintptr_t>(x) % 4) || (reinterpret_cast<uintptr_t>(s) % 4) ||
        (reinterpret_cast<uintptr_t>(zp) % 4) || (sse_opt && (reinterpret_cast<uintptr_t>(sse_opt) % 8)))
        return record_error(FQVIT_ERR_INVALID_ARG, "calibrate_ptf_noalloc: misaligned pointer");
    void *ws = nullptr;
    cudaError_t e = scratch_for_current_device(&ws);
    if (e != cudaSuccess) return cuda_error("cannot resolve the scratch address", e);
    e = fqvit::launch_calibrate(x, rows, C, ld_x, K, s, zp, alpha, sse_opt, ws,
                                reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_error("launch failed", e);
    return record_error(FQVIT_OK, "");
}

}  // extern "C"
