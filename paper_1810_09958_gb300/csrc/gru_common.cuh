// gru_common.cuh -- device helpers shared by the GRU recurrence kernels.
#pragma once
#include <cstdint>

#include <cuda_bf16.h>

#include "ptx.cuh"

namespace isam {

constexpr uint32_t kSiteGruStep = 0x201;  // bounded wait on the grid-wide step counter

__device__ __forceinline__ uint32_t ld_acquire_gpu(const uint32_t *p) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ void red_release_gpu_add(uint32_t *p, uint32_t v) {
    asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// Branch-free gate nonlinearities (a data-dependent branch in the gate code
// would split warps for the rest of the step): __expf and the approximate
// __fdividef, exact in the limits (exp overflow gives 0 and +-1).
__device__ __forceinline__ float sigmoidf_fast(float v) { return __fdividef(1.0f, 1.0f + __expf(-v)); }
// tanh(v) = 1 - 2 / (1 + e^{2v})
__device__ __forceinline__ float tanhf_fast(float v) { return 1.0f - __fdividef(2.0f, 1.0f + __expf(2.0f * v)); }

__device__ __forceinline__ uint16_t f32_to_bf16_rne(float f) {
    return __bfloat16_as_ushort(__float2bfloat16_rn(f));
}

// Spins (bounded) until the step counter reaches target.
__device__ __forceinline__ bool wait_counter(const uint32_t *counter, uint32_t target, const WaitCtx &w) {
    if (ld_acquire_gpu(counter) >= target) return true;
    const unsigned long long t0 = globaltimer();
    for (uint32_t i = 1;; ++i) {
        if (ld_acquire_gpu(counter) >= target) return true;
        if ((i & 15u) == 0u) {
            if (*w.abort_flag) return false;
            if (globaltimer() - t0 > w.timeout_ns) {
                report_timeout(w, kSiteGruStep);
                return false;
            }
        }
    }
}

}  // namespace isam
