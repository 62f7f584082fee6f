// gemm_common.cuh -- device helpers shared by the GEMM kernels.
#pragma once
#include "ptx.cuh"

namespace isam {

// Waits ignoring the abort flag (used only to let copies already issued land).
__device__ inline bool drain_wait(uint64_t *bar, uint32_t parity, unsigned long long timeout_ns) {
    const uint32_t a = smem_u32(bar);
    const unsigned long long t0 = globaltimer();
    while (!mbar_try_wait(a, parity)) {
        if (globaltimer() - t0 > timeout_ns) return false;
    }
    return true;
}

// bounded_wait by every lane of a warp, with a warp-uniform result.
template <bool cluster_scope = false>
__device__ __forceinline__ bool warp_wait(uint64_t *bar, uint32_t parity, const WaitCtx &w, uint32_t site) {
    const bool ok = bounded_wait<cluster_scope>(bar, parity, w, site);
    return __all_sync(0xffffffffu, ok) != 0;
}

}  // namespace isam
