// Unmask for callers that cannot allocate device memory.
//
// mosaic_unmask needs l * m words of scratch between its ring product
// (K + Q_d L^T) and its gather/decode pass, and takes them from a workspace the
// caller allocates.  Some callers have no way to do that: a plugin inside a
// host framework that owns every byte of device memory and exposes no
// allocator, a runtime with a fixed memory budget decided before the model
// loads, or a latency-critical serving loop that must never enter the CUDA
// allocator.  mosaic_unmask_noalloc serves them by taking its scratch from a
// fixed array compiled into this library instead.
//
// The array is a file-scope __device__ variable, so every GPU that loads the
// library holds it (16 MiB) until the process exits.  Host code cannot use the
// array's name as a device address (on the host it names a stand-in object),
// so every call looks the address up with cudaGetSymbolAddress on the current
// device (cheap once the module is loaded).  Nothing is cached: after a device
// or context reset the module reloads and the array may sit elsewhere.

#include "mosaic_internal.cuh"

namespace {

constexpr int64_t kScratchWords = (int64_t)1 << 22;   // 16 MiB of uint32: l * m <= 2^22

static __device__ __align__(256) uint32_t g_unmask_scratch[kScratchWords];

// Device address of the scratch array on the current device.
mosaic_status scratch_address(void **out) {
    void *addr = nullptr;
    if (cudaGetSymbolAddress(&addr, g_unmask_scratch) != cudaSuccess || addr == nullptr) return MOSAIC_ERR_CUDA;
    *out = addr;
    return MOSAIC_OK;
}

}  // namespace

extern "C" mosaic_status mosaic_unmask_noalloc(const mosaic_params *p, int64_t l, int64_t m,
                                               const uint32_t *Z, int64_t ldz, const uint32_t *K_tm,
                                               const uint32_t *L, const uint32_t *S_idx,
                                               const uint32_t *S_val, const float *s_w,
                                               const float *s_x, const float *bias, float *Y,
                                               uint32_t *Yhat, int64_t ldy, int variant,
                                               void *stream) {
    if (l < 0 || m < 1) return MOSAIC_ERR_SHAPE;
    // The fixed scratch holds l * m words; larger requests are refused before any work.
    if (l > kScratchWords / m) return MOSAIC_ERR_WORKSPACE;
    if (l == 0) return mosaic_unmask(p, l, m, Z, ldz, K_tm, L, S_idx, S_val, s_w, s_x, bias, Y, Yhat,
                                     ldy, variant, nullptr, 0, stream);
    void *ws = nullptr;
    const mosaic_status st = scratch_address(&ws);
    if (st != MOSAIC_OK) return st;
    // Every scratch word this call reads is written earlier in the same call,
    // so the array never needs clearing between calls.
    return mosaic_unmask(p, l, m, Z, ldz, K_tm, L, S_idx, S_val, s_w, s_x, bias, Y, Yhat, ldy, variant,
                         ws, (size_t)kScratchWords * sizeof(uint32_t), stream);
}
