// Freivalds integrity check of the server's answer (Sec. 3.2 box, Init W
// step 4 and Online step 4; appendix "Computational integrity"):
//   setup:  Ychk = a W'            (k check vectors, one-time per matrix)
//   online: a^T Y' == Ychk X'      per token, over Z_{2^32}
// The online products are skinny (k <= 16 rows) and go through the streaming
// ring product; the setup's column sums run here.
#include "mosaic_internal.cuh"

namespace mosaic {
namespace {

constexpr int kMaxK = 16;

// Y[v][c] += sum_{i in [i0, i1)} a[v][i] W[i][c] for one column c per thread
// (a warp reads 32 consecutive words of a row of W; a[v][i] is the same for
// the whole warp).  Partial sums of the row chunks meet with atomic adds,
// which wrap mod 2^32 like the sums themselves.
__global__ void colsum_kernel(const uint32_t *a, int k, const uint32_t *W, int64_t ldw, int64_t m,
                              int64_t ncols, int64_t rows_per_block, uint32_t *Y) {
    const int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t i0 = (int64_t)blockIdx.y * rows_per_block;
    const int64_t i1 = i0 + rows_per_block < m ? i0 + rows_per_block : m;
    if (c >= ncols) return;
    uint32_t acc[kMaxK];
#pragma unroll
    for (int v = 0; v < kMaxK; v++) acc[v] = 0u;
    for (int64_t i = i0; i < i1; i++) {
        const uint32_t w = W[i * ldw + c];
#pragma unroll
        for (int v = 0; v < kMaxK; v++)
            if (v < k) acc[v] += __ldg(a + (int64_t)v * m + i) * w;
    }
#pragma unroll
    for (int v = 0; v < kMaxK; v++)
        if (v < k) atomicAdd(Y + (int64_t)v * ncols + c, acc[v]);
}

__global__ void compare_kernel(const uint32_t *lhs, const uint32_t *rhs, int k, int64_t l, uint32_t *bad,
                               uint32_t *n_bad) {
    const int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (j >= l) return;
    uint32_t b = 0u;
    for (int v = 0; v < k; v++) b += lhs[(int64_t)v * l + j] != rhs[(int64_t)v * l + j] ? 1u : 0u;
    bad[j] = b;
    if (b) atomicAdd(n_bad, 1u);
}

// C (k x N) = A (k x K) B^T, B N x K: the streaming product when the operands
// qualify, else the CUDA-core one.
mosaic_status skinny_or_imad(const uint32_t *A, int64_t lda, const uint32_t *B, int64_t ldb, uint32_t *C,
                             int64_t k, int64_t N, int64_t K, cudaStream_t st) {
    if (skinny_ok(A, lda, B, ldb, k, K))
        return ring_gemm_skinny(A, lda, B, ldb, C, N, nullptr, 0, 1, k, N, K, st);
    return ring_gemm_imad(A, lda, 1, B, ldb, 1, C, N, nullptr, 0, 1, k, N, K, st);
}

}  // namespace

mosaic_status freivalds_colsum(const uint32_t *a, int k, const uint32_t *W, int64_t ldw, int64_t m,
                               int64_t ncols, uint32_t *Y, cudaStream_t st) {
    if (k < 1 || k > kMaxK) return MOSAIC_ERR_ARG;
    if (cudaMemsetAsync(Y, 0, sizeof(uint32_t) * (size_t)k * (size_t)ncols, st) != cudaSuccess)
        return MOSAIC_ERR_CUDA;
    if (m == 0 || ncols == 0) return MOSAIC_OK;
    // About four resident blocks per SM: split the rows so that the grid has
    // ~600 blocks, each summing at least 64 rows.
    const int64_t xblocks = (ncols + 255) / 256;
    int64_t yblocks = (608 + xblocks - 1) / xblocks;
    int64_t rows = (m + yblocks - 1) / yblocks;
    if (rows < 64) rows = 64;
    yblocks = (m + rows - 1) / rows;
    if (xblocks > 0x7fffffff || yblocks > 65535) return MOSAIC_ERR_SHAPE;
    {
        KernelSpan span("freivalds_colsum", st);
        colsum_kernel<<<dim3((unsigned)xblocks, (unsigned)yblocks), 256, 0, st>>>(a, k, W, ldw, m, ncols, rows, Y);
    }
    return launch_status();
}

mosaic_status freivalds_check(int k, const uint32_t *a, const uint32_t *Ychk, int64_t m, int64_t n_pad,
                              int64_t l, const uint32_t *Z, int64_t ldz, const uint32_t *Xp, int64_t ldx,
                              uint32_t *bad, uint32_t *n_bad, uint32_t *lhs, uint32_t *rhs, cudaStream_t st) {
    MOSAIC_TRY(skinny_or_imad(a, m, Z, ldz, lhs, k, l, m, st));
    MOSAIC_TRY(skinny_or_imad(Ychk, n_pad, Xp, ldx, rhs, k, l, n_pad, st));
    {
        KernelSpan span("freivalds_compare", st);
        compare_kernel<<<(unsigned)((l + 255) / 256), 256, 0, st>>>(lhs, rhs, k, l, bad, n_bad);
    }
    return launch_status();
}

}  // namespace mosaic
