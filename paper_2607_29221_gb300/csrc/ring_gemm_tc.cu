// Tensor-core ring product (placeholder until the tcgen05 kernel lands).
#include "mosaic_internal.cuh"

namespace mosaic {

bool tc_available() { return false; }
bool mma_s8_available() { return false; }

mosaic_status ring_gemm_tc_planes(const uint16_t *, int64_t, int64_t, const uint16_t *, int64_t,
                                  int64_t, uint32_t *, int64_t, const uint32_t *, int64_t, int,
                                  int64_t, int64_t, int64_t, cudaStream_t) {
    return MOSAIC_ERR_UNSUPPORTED;
}

mosaic_status ring_gemm_mma_s8(const uint32_t *, int64_t, const uint32_t *, int64_t, uint32_t *,
                               int64_t, const uint32_t *, int64_t, int, int64_t, int64_t, int64_t,
                               cudaStream_t) {
    return MOSAIC_ERR_UNSUPPORTED;
}

}  // namespace mosaic
