// A gradient step for callers that cannot allocate device memory.
//
// cm_gd_step needs a device workspace for the two stacked worker-result
// vectors and the residual z.  Some callers cannot provide one: a plug-in
// running inside a host application that owns all device memory through its
// own pool and forbids raw cudaMalloc, or a latency-critical loop that must
// not call the allocator (cudaMalloc and cudaFree can synchronize the
// device).  cm_gd_step_noalloc serves them from a fixed scratch array that
// lives in this library's device image: it calls no cudaMalloc, cudaFree or
// other allocating routine.
//
// The array holds CM_GD_STATIC_SCRATCH_BYTES bytes on every GPU that loads
// the library, until the process exits.  All calls on a device share it and
// it keeps the previous call's contents; no part of it has to start at zero,
// because each step writes every stacked result and every z entry before it
// reads them.  Two calls whose kernels overlap on the GPU (for example on two
// streams) race on the array and give undefined results.
#include <mutex>

#include "cm_internal.cuh"

static __device__ __align__(256) unsigned char g_gd_scratch[CM_GD_STATIC_SCRATCH_BYTES];

namespace {

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void *g_addr[kMaxDevices] = {nullptr};

// Device address of the scratch array on the current device.  In host code
// g_gd_scratch names a host-side stand-in, not device memory, so the address
// is looked up once per device (with that device current) and cached.
cudaError_t scratch_address(void **out)
{
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_addr[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_gd_scratch);
        if (e != cudaSuccess) return e;
        g_addr[dev] = p;
    }
    *out = g_addr[dev];
    return cudaSuccess;
}

}  // namespace

extern "C" cm_status cm_gd_step_noalloc(const cm_code *code_A, const float *A, int64_t lda,
                                        const float *PA, int64_t ldpa, const cm_code *code_AT,
                                        const float *AT, int64_t ldat, const float *PAT,
                                        int64_t ldpat, const float *y, float *x, float eta,
                                        uint32_t surv_A, uint32_t surv_AT, int32_t *dev_status,
                                        cm_stream_t stream)
{
    if (!code_A || !code_AT) return CM_EINVAL;
    if (cm_gd_workspace_bytes(code_A, code_AT) > (size_t)CM_GD_STATIC_SCRATCH_BYTES)
        return CM_ENOMEM;   // problem too large for the fixed scratch array
    void *ws = nullptr;
    if (scratch_address(&ws) != cudaSuccess || !ws) return CM_ECUDA;
    return cm_gd_step(code_A, A, lda, PA, ldpa, code_AT, AT, ldat, PAT, ldpat, y, x, eta, surv_A,
                      surv_AT, ws, (size_t)CM_GD_STATIC_SCRATCH_BYTES, dev_status, stream);
}
