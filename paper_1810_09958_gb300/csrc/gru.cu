// gru.cu -- GRU forward (placeholder until the persistent recurrent kernel lands).
#include "internal.h"

namespace isam {
int gru_launch(int, int, int, const uint16_t *, const uint16_t *, const uint16_t *, const float *,
               const float *, float *, DeviceState &, cudaStream_t) {
    return set_error(ISAM_ERR_UNSUPPORTED, "isam_gru_forward: not available in this build");
}
}  // namespace isam
