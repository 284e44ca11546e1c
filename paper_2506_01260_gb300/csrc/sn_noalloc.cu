// sn_noalloc.cu — sn_project_weight_noalloc: the bf16 weight projection with
// its scratch held in a fixed device array, for callers that cannot allocate
// device memory themselves.
//
// The projection needs scratch (fp32 partial sums of U^T W and the bf16
// A^T operand).  sn_project_weight takes that scratch from the caller; this
// entry point takes it from g_noalloc_scratch below instead.  The array is a
// file-scope __device__ object: every GPU that loads this library holds
// kNoallocScratchBytes of it until the process exits.  Host code cannot use
// the array's name as a device address, so the first call on each device
// (with that device current) looks the address up with cudaGetSymbolAddress;
// later calls in the same CUDA context reuse it.  The address belongs to the
// context it was looked up in, so it is cached together with that context and
// looked up again when the device's current context is a different one (after
// cudaDeviceReset, or under a caller's own non-primary context).
#include <cuda.h>
#include <mutex>

#include "sn_internal.cuh"

namespace {

constexpr size_t kNoallocScratchBytes = (size_t)32 << 20;   // 32 MiB
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoallocScratchBytes];

std::mutex g_noalloc_mu;
void *g_noalloc_ptr[kMaxDevices];
CUcontext g_noalloc_ctx[kMaxDevices];

typedef CUresult (*CtxGetCurrentFn)(CUcontext *);

// The driver's cuCtxGetCurrent, reached through the runtime (the library does
// not link the driver library itself).
CtxGetCurrentFn ctx_get_current()
{
    static CtxGetCurrentFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = (CtxGetCurrentFn)f;
    });
    return fn;
}

// Device address of the scratch array on the current device, in the current
// context (set-up on the first call per device and context).
sn_status noalloc_scratch(void **out)
{
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess)
        return SN_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices)
        return SN_ERR_UNSUPPORTED;
    CtxGetCurrentFn get = ctx_get_current();
    CUcontext ctx = nullptr;
    if (!get || get(&ctx) != CUDA_SUCCESS)
        return SN_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (!ctx || !g_noalloc_ptr[dev] || g_noalloc_ctx[dev] != ctx) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p)
            return SN_ERR_CUDA;
        // the lookup makes the device's primary context current if none was
        if (!ctx && (get(&ctx) != CUDA_SUCCESS || !ctx))
            return SN_ERR_CUDA;
        g_noalloc_ptr[dev] = p;
        g_noalloc_ctx[dev] = ctx;
    }
    *out = g_noalloc_ptr[dev];
    return SN_OK;
}

}  // namespace

extern "C" sn_status sn_project_weight_noalloc(sn_basis_t basis, sn_dtype dtype, const void *W,
                                                int64_t rows, int64_t cols, int64_t ld,
                                                void *W_out, sn_stream_t stream)
{
    if (dtype != SN_BF16)
        return SN_ERR_UNSUPPORTED;
    size_t need = 0;
    sn_status st = sn_project_weight_workspace(basis, dtype, cols, &need);
    if (st != SN_OK)
        return st;
    if (need > kNoallocScratchBytes)
        return SN_ERR_UNSUPPORTED;   // more scratch than the fixed array holds
    void *scratch = nullptr;
    if ((st = noalloc_scratch(&scratch)) != SN_OK)
        return st;
    // Every element of the scratch that the projection reads is written first
    // in the same call, so nothing needs clearing between calls.
    return sn_project_weight(basis, dtype, W, rows, cols, ld, W_out, scratch,
                             kNoallocScratchBytes, stream);
}
