// Float glue of a decoder layer that sits between the secure linear calls on
// the trusted side (Sec. 4.1: the non-linear parts stay with the client in
// plain arithmetic): RMSNorm and SiLU(gate) * up, each as one pass over HBM.
// These are model operations, not part of the masked product; they are fused
// here only because each is a chain of elementwise steps over 32-268 MB.
#include <math.h>

#include "mosaic_internal.cuh"

namespace mosaic {
namespace {

constexpr int kNormThreads = 256;

// One block per row: sum of squares in fp32 (each thread a strided partial,
// then a tree over the block), y = x * (1 / sqrt(mean + eps)).
__global__ void __launch_bounds__(kNormThreads) rmsnorm_kernel(const float *x, int64_t ldx, int64_t n, float eps,
                                                               float *y, int64_t ldy, int vec) {
    __shared__ float part[kNormThreads / 32];
    const int64_t row = blockIdx.x;
    const float *xr = x + row * ldx;
    float *yr = y + row * ldy;
    float ss = 0.0f;
    if (vec) {
        for (int64_t c = 4 * (int64_t)threadIdx.x; c < n; c += 4 * kNormThreads) {
            const float4 v = *reinterpret_cast<const float4 *>(xr + c);
            ss = fmaf(v.x, v.x, ss);
            ss = fmaf(v.y, v.y, ss);
            ss = fmaf(v.z, v.z, ss);
            ss = fmaf(v.w, v.w, ss);
        }
    } else {
        for (int64_t c = threadIdx.x; c < n; c += kNormThreads) ss = fmaf(xr[c], xr[c], ss);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
    if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = ss;
    __syncthreads();
    float tot = 0.0f;
#pragma unroll
    for (int w = 0; w < kNormThreads / 32; ++w) tot += part[w];
    const float inv = 1.0f / sqrtf(tot / (float)n + eps);
    if (vec) {
        for (int64_t c = 4 * (int64_t)threadIdx.x; c < n; c += 4 * kNormThreads) {
            const float4 v = *reinterpret_cast<const float4 *>(xr + c);
            *reinterpret_cast<float4 *>(yr + c) = make_float4(v.x * inv, v.y * inv, v.z * inv, v.w * inv);
        }
    } else {
        for (int64_t c = threadIdx.x; c < n; c += kNormThreads) yr[c] = xr[c] * inv;
    }
}

__device__ __forceinline__ float silu(float g) { return g / (1.0f + expf(-g)); }

// out[r][c] = silu(gu[r][c]) * gu[r][ffn + c]: block (x, r) covers columns
// [1024 x, 1024 x + 1024) of row r, four a thread.
__global__ void swiglu_kernel(const float *gu, int64_t ldg, int64_t ffn, float *out, int64_t ldo, int vec) {
    const int64_t r = blockIdx.y;
    const int64_t c = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) * 4;
    if (c >= ffn) return;
    const float *g = gu + r * ldg + c;
    const float *u = g + ffn;
    float *o = out + r * ldo + c;
    if (vec && c + 4 <= ffn) {
        const float4 a = *reinterpret_cast<const float4 *>(g);
        const float4 b = *reinterpret_cast<const float4 *>(u);
        *reinterpret_cast<float4 *>(o) = make_float4(silu(a.x) * b.x, silu(a.y) * b.y, silu(a.z) * b.z, silu(a.w) * b.w);
    } else {
        for (int k = 0; k < 4 && c + k < ffn; ++k) o[k] = silu(g[k]) * u[k];
    }
}

}  // namespace
}  // namespace mosaic

using namespace mosaic;

extern "C" {

mosaic_status mosaic_rmsnorm(const float *x, int64_t ldx, int64_t rows, int64_t n, float eps, float *y,
                             int64_t ldy, void *stream) {
    RoleScope role("glue");
    if (rows < 0 || n < 1 || ldx < n || ldy < n || rows > 0x7fffffff) return MOSAIC_ERR_SHAPE;
    if (!(eps >= 0.0f)) return MOSAIC_ERR_ARG;
    if (rows == 0) return MOSAIC_OK;
    if (!x || !y) return MOSAIC_ERR_ARG;
    const int vec = aligned16(x) && aligned16(y) && ldx % 4 == 0 && ldy % 4 == 0 && n % 4 == 0;
    cudaStream_t st = as_stream(stream);
    {
        KernelSpan span("rmsnorm", st);
        rmsnorm_kernel<<<(unsigned)rows, kNormThreads, 0, st>>>(x, ldx, n, eps, y, ldy, vec);
    }
    return launch_status();
}

mosaic_status mosaic_swiglu(const float *gu, int64_t ldg, int64_t rows, int64_t ffn, float *out, int64_t ldo,
                            void *stream) {
    RoleScope role("glue");
    if (rows < 0 || ffn < 1 || ldg < 2 * ffn || ldo < ffn || rows > 65535) return MOSAIC_ERR_SHAPE;
    if (rows == 0) return MOSAIC_OK;
    if (!gu || !out) return MOSAIC_ERR_ARG;
    const int vec = aligned16(gu) && aligned16(out) && ldg % 4 == 0 && ldo % 4 == 0 && ffn % 4 == 0;
    cudaStream_t st = as_stream(stream);
    const int64_t bx = (ffn + 1023) / 1024;
    if (bx > 0x7fffffff) return MOSAIC_ERR_SHAPE;
    {
        KernelSpan span("swiglu", st);
        swiglu_kernel<<<dim3((unsigned)bx, (unsigned)rows), 256, 0, st>>>(gu, ldg, ffn, out, ldo, vec);
    }
    return launch_status();
}

}  // extern "C"
