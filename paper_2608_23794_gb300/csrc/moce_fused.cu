// Fused persistent forward kernel (pool -> gate -> mix in one launch).
#include "moce_internal.cuh"

namespace moce {

bool fused_supported(int, int, int, int, int) { return false; }

cudaError_t launch_fused(const uint16_t *, int, int, int, int, int, const int32_t *, const float *,
                         const int32_t *, int, const float *, const float *, const float *,
                         const float *, float, float, uint16_t *, const WsLayout &, unsigned char *,
                         cudaStream_t) {
    return cudaErrorNotSupported;
}

}  // namespace moce
