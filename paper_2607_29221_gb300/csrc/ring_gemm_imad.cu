// Ring product over Z_{2^32} on CUDA cores (one 32-bit multiply-add per
// ring MAC; the "native INT32 on the general-purpose pipeline" option of
// Sec. 5.2, kept as the comparison variant and used for the one-time
// chain products of Init W where operands arrive in either orientation).
//
// C[i][j] = (Cin ? Cin[i][j] : 0) + sgn * sum_k A(i, k) B(j, k)   (mod 2^32)
// with A(i, k) = A[i * sai + k * sak] and B(j, k) = B[j * sbj + k * sbk].
// 128 x 128 output tile per 256-thread CTA, 8 x 8 outputs per thread,
// BK = 16 staged through shared memory.
#include "mosaic_internal.cuh"

namespace mosaic {
namespace {

constexpr int BM = 128, BN = 128, BK = 16, NT = 256;

struct GemmArgs {
    const uint32_t *A;
    int64_t sai, sak;
    const uint32_t *B;
    int64_t sbj, sbk;
    uint32_t *C;
    int64_t ldc;
    const uint32_t *Cin;
    int64_t ldcin;
    int sgn;
    int64_t M, N, K;
};

// Loads a 128 x BK tile of X(r, k) = X[r * sr + k * sk] into S[k][r].
__device__ __forceinline__ void load_tile(uint32_t (*S)[BM + 4], const uint32_t *X, int64_t sr,
                                          int64_t sk, int64_t r0, int64_t k0, int64_t R, int64_t K) {
    const int tid = threadIdx.x;
    if (sk == 1) {
#pragma unroll
        for (int q = 0; q < (BM * BK) / NT; q++) {
            const int L = tid + NT * q;
            const int k = L % BK, r = L / BK;
            const int64_t gr = r0 + r, gk = k0 + k;
            S[k][r] = (gr < R && gk < K) ? X[gr * sr + gk] : 0u;
        }
    } else {
#pragma unroll
        for (int q = 0; q < (BM * BK) / NT; q++) {
            const int L = tid + NT * q;
            const int r = L % BM, k = L / BM;
            const int64_t gr = r0 + r, gk = k0 + k;
            S[k][r] = (gr < R && gk < K) ? X[gr * sr + gk * sk] : 0u;
        }
    }
}

__global__ void __launch_bounds__(NT) ring_gemm_imad_kernel(GemmArgs a) {
    __shared__ uint32_t As[BK][BM + 4];
    __shared__ uint32_t Bs[BK][BN + 4];
    const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
    const int64_t i0 = (int64_t)blockIdx.y * BM, j0 = (int64_t)blockIdx.x * BN;
    uint32_t acc[8][8];
#pragma unroll
    for (int p = 0; p < 8; p++)
#pragma unroll
        for (int q = 0; q < 8; q++) acc[p][q] = 0u;

    for (int64_t k0 = 0; k0 < a.K; k0 += BK) {
        load_tile(As, a.A, a.sai, a.sak, i0, k0, a.M, a.K);
        load_tile(Bs, a.B, a.sbj, a.sbk, j0, k0, a.N, a.K);
        __syncthreads();
#pragma unroll
        for (int k = 0; k < BK; k++) {
            uint32_t av[8], bv[8];
#pragma unroll
            for (int p = 0; p < 8; p++) av[p] = As[k][ty + 16 * p];
#pragma unroll
            for (int q = 0; q < 8; q++) bv[q] = Bs[k][tx + 16 * q];
#pragma unroll
            for (int p = 0; p < 8; p++)
#pragma unroll
                for (int q = 0; q < 8; q++) acc[p][q] += av[p] * bv[q];
        }
        __syncthreads();
    }
#pragma unroll
    for (int p = 0; p < 8; p++) {
        const int64_t i = i0 + ty + 16 * p;
        if (i >= a.M) continue;
#pragma unroll
        for (int q = 0; q < 8; q++) {
            const int64_t j = j0 + tx + 16 * q;
            if (j >= a.N) continue;
            uint32_t v = a.sgn >= 0 ? acc[p][q] : 0u - acc[p][q];
            if (a.Cin) v += a.Cin[i * a.ldcin + j];
            a.C[i * a.ldc + j] = v;
        }
    }
}

}  // namespace

mosaic_status ring_gemm_imad(const uint32_t *A, int64_t sai, int64_t sak, const uint32_t *B,
                             int64_t sbj, int64_t sbk, uint32_t *C, int64_t ldc,
                             const uint32_t *Cin, int64_t ldcin, int sgn, int64_t M, int64_t N,
                             int64_t K, cudaStream_t st) {
    if (M == 0 || N == 0) return MOSAIC_OK;
    GemmArgs a{A, sai, sak, B, sbj, sbk, C, ldc, Cin, ldcin, sgn, M, N, K};
    const int64_t gx = (N + BN - 1) / BN, gy = (M + BM - 1) / BM;
    if (gy > 65535) return MOSAIC_ERR_SHAPE;
    {
        KernelSpan span("ring_gemm_imad", st);
        ring_gemm_imad_kernel<<<dim3((unsigned)gx, (unsigned)gy), NT, 0, st>>>(a);
    }
    return launch_status();
}

}  // namespace mosaic
