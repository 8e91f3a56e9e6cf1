// K5: coded GEMM on tcgen05 tensor cores (not built yet in this revision).
#include "cm_internal.cuh"

cudaError_t launch_coded_gemm(const CodeParams &, const uint16_t *, int64_t, const uint16_t *,
                              int64_t, const uint16_t *, int64_t, int, float *, int64_t,
                              cudaStream_t)
{
    return cudaErrorNotSupported;
}
