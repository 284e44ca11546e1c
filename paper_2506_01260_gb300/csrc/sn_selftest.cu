// sn_selftest.cu — sn_selftest_wait_timeout: the bounded-wait rule exercised on
// purpose, so that failure detection can be tested on a GPU without a fault.
//
// One CTA of two warps sets up like the pipeline kernels (an mbarrier, an abort
// flag, 32 columns of tensor memory), then both warps wait for a phase of the
// barrier that no thread and no copy ever completes, with the same bounded wait
// (tc::warp_wait).  The first to pass the wait limit raises the CTA's abort
// flag and records SN_EBIT_TIMEOUT in the basis' error word; the other stops on
// the flag.  The CTA then frees its tensor memory and returns, leaving the
// context usable.
#include "sn_tc.cuh"

namespace {

__global__ void __launch_bounds__(64, 1) k_wait_timeout(unsigned int *err)
{
    using namespace sn::tc;
    __shared__ __align__(8) uint64_t bar;
    __shared__ uint32_t tmem_slot;
    __shared__ int abort_flag;
    const int warp = threadIdx.x >> 5;
    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&bar), 1);     // one arrival expected, none is ever made
        abort_flag = 0;
        mbar_fence_init();
    }
    if (warp == 0)
        tmem_alloc(smem_u32(&tmem_slot), 32);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;

    warp_wait(smem_u32(&bar), 0, &abort_flag, err);    // phase 0 never completes

    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, 32);
    }
}

}  // namespace

extern "C" sn_status sn_selftest_wait_timeout(sn_basis_t b, sn_stream_t stream)
{
    if (!b)
        return SN_ERR_INVALID_ARG;
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev != b->device)
        return SN_ERR_INVALID_ARG;
    k_wait_timeout<<<1, 64, 0, (cudaStream_t)stream>>>(b->err);
    sn::count_launch();
    return cudaGetLastError() == cudaSuccess ? SN_OK : SN_ERR_CUDA;
}
