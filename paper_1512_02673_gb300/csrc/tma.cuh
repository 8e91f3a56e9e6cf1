// Tensor-memory-accelerator (TMA) and mbarrier helpers for sm_103a kernels:
// host-side tensor-map encoding through the driver entry point, device-side
// inline PTX for bulk tensor loads, transaction-counted mbarriers and
// bounded waits.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

// ---- host ---------------------------------------------------------------------------

// Encode a 2-D row-major tensor map: `height` rows of `width` elements with a
// row pitch of `pitch_bytes` (a multiple of 16), boxes of box_w x box_h
// elements.  Elements outside the tensor read as zero.  Returns false if the
// driver entry point is missing or rejects the description.
bool cm_make_tmap_2d(CUtensorMap *map, CUtensorMapDataType type, const void *base,
                     uint64_t width, uint64_t height, uint64_t pitch_bytes, uint32_t box_w,
                     uint32_t box_h, CUtensorMapSwizzle swizzle);

// Encode a 3-D tensor map: `depth` slabs of `height` rows of `width`
// elements; row pitch and slab pitch in bytes (multiples of 16); boxes of
// box_w x box_h x box_d elements, no swizzle, zero fill outside.
bool cm_make_tmap_3d(CUtensorMap *map, CUtensorMapDataType type, const void *base,
                     uint64_t width, uint64_t height, uint64_t depth, uint64_t pitch_bytes,
                     uint64_t slab_bytes, uint32_t box_w, uint32_t box_h, uint32_t box_d);

// ---- device -------------------------------------------------------------------------

__device__ __forceinline__ uint32_t cm_smem_u32(const void *p)
{
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void cm_mbar_init(uint64_t *bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;\n" ::"r"(cm_smem_u32(bar)), "r"(count));
}

// Make mbarrier initialisation visible to the async (TMA) proxy.
__device__ __forceinline__ void cm_fence_mbar_init()
{
    asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
}

__device__ __forceinline__ void cm_mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n" ::"r"(cm_smem_u32(bar)),
                 "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ void cm_mbar_arrive(uint64_t *bar)
{
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];\n" ::"r"(cm_smem_u32(bar)) : "memory");
}

__device__ __forceinline__ bool cm_mbar_try_wait(uint64_t *bar, uint32_t parity)
{
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}\n"
        : "=r"(done)
        : "r"(cm_smem_u32(bar)), "r"(parity)
        : "memory");
    return done != 0;
}

__device__ __forceinline__ uint64_t cm_globaltimer()
{
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;\n" : "=l"(t));
    return t;
}

// Wait for phase `parity` of an mbarrier to complete, giving up after about
// `limit_ns` nanoseconds of wall time.  Returns false on time-out.
__device__ __forceinline__ bool cm_mbar_wait(uint64_t *bar, uint32_t parity,
                                             uint64_t limit_ns = 2000000000ull)
{
    if (cm_mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = cm_globaltimer();
    for (uint32_t it = 1;; ++it) {
        if (cm_mbar_try_wait(bar, parity)) return true;
        if ((it & 255u) == 0 && cm_globaltimer() - t0 > limit_ns) return false;
    }
}

// 3-D TMA tile load global -> shared, completion counted on `bar`.
__device__ __forceinline__ void cm_tma_load_3d(void *smem_dst, const CUtensorMap *map, int32_t x,
                                               int32_t y, int32_t z, uint64_t *bar)
{
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes "
        "[%0], [%1, {%2, %3, %4}], [%5];\n" ::"r"(cm_smem_u32(smem_dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(cm_smem_u32(bar))
        : "memory");
}

// 2-D TMA tile load global -> shared, completion counted on `bar`.
// x = innermost (column) coordinate, y = row coordinate, in elements.
__device__ __forceinline__ void cm_tma_load_2d(void *smem_dst, const CUtensorMap *map, int32_t x,
                                               int32_t y, uint64_t *bar)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes "
        "[%0], [%1, {%2, %3}], [%4];\n" ::"r"(cm_smem_u32(smem_dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(cm_smem_u32(bar))
        : "memory");
}
