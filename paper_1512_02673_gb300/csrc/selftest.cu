// Self-test of the bounded mbarrier wait used by the mat-vec and GEMM kernels:
// one warp waits on an mbarrier that nothing arrives at.  The wait must give
// up after `limit_ns` and report CM_ETIMEOUT through the status word, leaving
// the context usable.
#include "cm_internal.cuh"
#include "tma.cuh"

namespace {

__global__ void bounded_wait_kernel(int32_t *status, uint64_t limit_ns)
{
    __shared__ uint64_t bar;
    if (threadIdx.x == 0) cm_mbar_init(&bar, 1);   // expects one arrival that never comes
    cm_fence_mbar_init();
    __syncwarp();
    const bool ok = cm_mbar_wait(&bar, 0, limit_ns);
    if (__all_sync(0xffffffffu, !ok) && threadIdx.x == 0) *status = CM_ETIMEOUT;
}

}  // namespace

extern "C" cm_status cm_selftest_bounded_wait(int32_t *dev_status, uint64_t limit_ns,
                                              cm_stream_t stream)
{
    if (!dev_status || limit_ns == 0 || limit_ns > 2000000000ull) return CM_EINVAL;
    bounded_wait_kernel<<<1, 32, 0, (cudaStream_t)stream>>>(dev_status, limit_ns);
    return cudaGetLastError() == cudaSuccess ? CM_OK : CM_ECUDA;
}
