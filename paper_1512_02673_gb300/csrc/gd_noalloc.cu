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

// In host code g_gd_scratch names a host-side stand-in, not device memory: the
// array's device address belongs to the module image loaded into one CUDA
// context, so it is looked up with cudaGetSymbolAddress (with the device
// current) and cached per device together with the unique ID of the context
// it came from.  A different current context on the device (after
// cudaDeviceReset, which replaces the primary context, or a context the caller
// created itself) has a different ID and gets a fresh lookup, never the old
// address.  Context IDs are never reused within a process.
using CtxGetCurrentFn = CUresult (*)(CUcontext *);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long *);

struct DriverFns {
    CtxGetCurrentFn get_current = nullptr;
    CtxGetIdFn get_id = nullptr;
};

const DriverFns &driver_fns()
{
    static DriverFns fns;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fns.get_current = reinterpret_cast<CtxGetCurrentFn>(p);
        p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fns.get_id = reinterpret_cast<CtxGetIdFn>(p);
    });
    return fns;
}

// Unique ID of the context current on this thread (false if there is none
// yet or the driver cannot tell; the caller then looks the address up afresh).
bool current_context_id(unsigned long long *id)
{
    const DriverFns &f = driver_fns();
    if (!f.get_current || !f.get_id) return false;
    CUcontext ctx = nullptr;
    if (f.get_current(&ctx) != CUDA_SUCCESS || !ctx) return false;
    return f.get_id(ctx, id) == CUDA_SUCCESS;
}

constexpr int kMaxDevices = 64;
struct CachedAddress {
    bool valid = false;
    unsigned long long ctx_id = 0;
    void *addr = nullptr;
};
std::mutex g_mu;
CachedAddress g_cache[kMaxDevices];

// Device address of the scratch array in the current device's current context.
cudaError_t scratch_address(void **out)
{
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_mu);
    CachedAddress &c = g_cache[dev];
    unsigned long long id = 0;
    if (c.valid && current_context_id(&id) && id == c.ctx_id) {
        *out = c.addr;
        return cudaSuccess;
    }
    // The lookup binds the device's context to this thread if none is yet,
    // so the context ID is read after it.
    void *p = nullptr;
    e = cudaGetSymbolAddress(&p, g_gd_scratch);
    if (e != cudaSuccess) return e;
    c.addr = p;
    c.valid = current_context_id(&c.ctx_id);
    *out = p;
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
