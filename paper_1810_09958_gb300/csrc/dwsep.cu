// dwsep.cu -- separable depthwise convolution (placeholder until the fused kernel lands).
#include "internal.h"

namespace isam {
int dwsep_launch(int, int, int, int, int, const uint16_t *, const uint16_t *, const uint16_t *,
                 float *, DeviceState &, cudaStream_t) {
    return set_error(ISAM_ERR_UNSUPPORTED, "isam_dwsep_conv: not available in this build");
}
}  // namespace isam
