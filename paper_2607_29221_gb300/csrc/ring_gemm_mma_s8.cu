// Ring product over Z_{2^32} on the legacy warp-level tensor path
// (mma.sync m16n8k32 s8 x s8 -> s32), kept to compare with the tcgen05 path.
//
// Sec. 5.2 ("Emulation approach") runs the limb products on INT8 tensor
// cores.  Here every operand is split into signed base-2^8 digits
// d_i = byte_i(a + 0x80808080) - 128 (int8 planes, a = sum_i d_i 2^(8i) mod
// 2^32); the 10 digit pairs with i + j <= 3 accumulate in int32 per shift
// group s = i + j (integer accumulation wraps mod 2^32, so there is no
// exactness limit on K), and the epilogue forms sum_s acc_s << 8s.
//
// CTA tile 64 x 64, 4 warps of 32 x 32, K staged 64 digits at a time (two
// cp.async stages; rows padded to 80 bytes so that the fragment loads of a
// warp hit 32 distinct banks).
#include "mosaic_internal.cuh"

namespace mosaic {
namespace {

constexpr int TM = 64, TN = 64, TK = 64;   // CTA tile; TK int8 digits per stage
constexpr int ROWB = 80;                   // bytes per staged row (64 + 16 pad)
constexpr int PLANE_B = TM * ROWB;         // one plane of one operand in a stage
constexpr int STAGE_B = 2 * 4 * PLANE_B;   // A and B, 4 planes each
constexpr int THREADS = 128;

// int8 digit planes: planes[d][row][c] = digit d of a[row][c], zeros for c >= cols.
__global__ void split_s8_kernel(const uint32_t *a, int64_t lda, int64_t rows, int64_t cols, int8_t *planes,
                                int64_t ldp, int64_t plane_stride) {
    const int64_t per_row = ldp / 4;
    const int64_t total = rows * per_row;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = i / per_row, c = (i - r * per_row) * 4;
        uint32_t w[4];
#pragma unroll
        for (int q = 0; q < 4; q++) w[q] = c + q < cols ? a[r * lda + c + q] + 0x80808080u : 0x80808080u;
#pragma unroll
        for (int d = 0; d < 4; d++) {
            // byte d of each word, minus 128 as int8 (= the byte with its top bit flipped)
            uint32_t packed = 0;
#pragma unroll
            for (int q = 0; q < 4; q++) packed |= (((w[q] >> (8 * d)) & 0xffu) ^ 0x80u) << (8 * q);
            *reinterpret_cast<uint32_t *>(planes + d * plane_stride + r * ldp + c) = packed;
        }
    }
}

__device__ __forceinline__ void mma_s8(int32_t (&c)[4], const uint32_t (&a)[4], const uint32_t (&b)[2]) {
    asm volatile(
        "mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+r"(c[0]), "+r"(c[1]), "+r"(c[2]), "+r"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}

struct S8Args {
    const int8_t *A;   // [4][M][ldp]
    const int8_t *B;   // [4][N][ldp]
    int64_t ldp, a_plane, b_plane;
    uint32_t *C;
    int64_t ldc;
    const uint32_t *Cin;
    int64_t ldcin;
    int sgn;
    int M, N, nk;      // nk = ldp / TK stages
};

__global__ void __launch_bounds__(THREADS) ring_gemm_s8_kernel(S8Args a) {
    extern __shared__ __align__(16) uint8_t sm8[];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int gid = lane >> 2, tig = lane & 3;
    const int64_t m0 = (int64_t)blockIdx.y * TM, n0 = (int64_t)blockIdx.x * TN;
    const int wm = (warp >> 1) * 32, wn = (warp & 1) * 32;

    // Stage s: A planes at s * STAGE_B + p * PLANE_B, B planes after them.
    auto load_stage = [&](int s, int kc) {
        const uint32_t base = (uint32_t)__cvta_generic_to_shared(sm8 + s * STAGE_B);
        // 2 operands x 4 planes x 64 rows x 4 chunks of 16 bytes = 2048 chunks
        for (int ch = tid; ch < 2048; ch += THREADS) {
            const int op = ch >> 10, p = (ch >> 8) & 3, r = (ch >> 2) & 63, c = ch & 3;
            const int64_t grow = (op ? n0 : m0) + r;
            const bool ok = grow < (op ? a.N : a.M);
            const int8_t *src = (op ? a.B + p * a.b_plane : a.A + p * a.a_plane) + (ok ? grow * a.ldp : 0) +
                                (int64_t)kc * TK + c * 16;
            const uint32_t dst = base + (uint32_t)((op * 4 + p) * PLANE_B + r * ROWB + c * 16);
            asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(ok ? 16 : 0)
                         : "memory");
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    };

    int32_t acc[4][2][4][4];
#pragma unroll
    for (int g = 0; g < 4; g++)
#pragma unroll
        for (int i = 0; i < 2; i++)
#pragma unroll
            for (int j = 0; j < 4; j++)
#pragma unroll
                for (int q = 0; q < 4; q++) acc[g][i][j][q] = 0;

    load_stage(0, 0);
    for (int kc = 0; kc < a.nk; kc++) {
        if (kc + 1 < a.nk) load_stage((kc + 1) & 1, kc + 1);
        else asm volatile("cp.async.commit_group;" ::: "memory");
        asm volatile("cp.async.wait_group 1;" ::: "memory");
        __syncthreads();
        const uint8_t *st = sm8 + (kc & 1) * STAGE_B;
#pragma unroll
        for (int k32 = 0; k32 < TK / 32; k32++) {
            uint32_t af[4][2][4], bf[4][4][2];
#pragma unroll
            for (int p = 0; p < 4; p++) {
                const uint8_t *pa = st + p * PLANE_B;
                const uint8_t *pb = st + (4 + p) * PLANE_B;
#pragma unroll
                for (int i = 0; i < 2; i++) {
                    const uint8_t *r0 = pa + (wm + i * 16 + gid) * ROWB + k32 * 32 + tig * 4;
                    af[p][i][0] = *reinterpret_cast<const uint32_t *>(r0);
                    af[p][i][1] = *reinterpret_cast<const uint32_t *>(r0 + 8 * ROWB);
                    af[p][i][2] = *reinterpret_cast<const uint32_t *>(r0 + 16);
                    af[p][i][3] = *reinterpret_cast<const uint32_t *>(r0 + 8 * ROWB + 16);
                }
#pragma unroll
                for (int j = 0; j < 4; j++) {
                    const uint8_t *c0 = pb + (wn + j * 8 + gid) * ROWB + k32 * 32 + tig * 4;
                    bf[p][j][0] = *reinterpret_cast<const uint32_t *>(c0);
                    bf[p][j][1] = *reinterpret_cast<const uint32_t *>(c0 + 16);
                }
            }
#pragma unroll
            for (int di = 0; di < 4; di++)
#pragma unroll
                for (int dj = 0; dj + di < 4; dj++)
#pragma unroll
                    for (int i = 0; i < 2; i++)
#pragma unroll
                        for (int j = 0; j < 4; j++) mma_s8(acc[di + dj][i][j], af[di][i], bf[dj][j]);
        }
        __syncthreads();
    }
    asm volatile("cp.async.wait_all;" ::: "memory");

    // C = Cin + sgn * sum_s acc_s << 8s (mod 2^32).
#pragma unroll
    for (int i = 0; i < 2; i++)
#pragma unroll
        for (int j = 0; j < 4; j++)
#pragma unroll
            for (int q = 0; q < 4; q++) {
                const int64_t row = m0 + wm + i * 16 + gid + (q >> 1) * 8;
                const int64_t col = n0 + wn + j * 8 + tig * 2 + (q & 1);
                if (row >= a.M || col >= a.N) continue;
                uint32_t v = 0;
#pragma unroll
                for (int g = 0; g < 4; g++) v += (uint32_t)acc[g][i][j][q] << (8 * g);
                if (a.sgn < 0) v = 0u - v;
                if (a.Cin) v += a.Cin[row * a.ldcin + col];
                a.C[row * a.ldc + col] = v;
            }
}

}  // namespace

bool mma_s8_available() {
    int dev = 0, major = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return false;
    if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess) return false;
    return major >= 8;
}

size_t ws_mma_s8(int64_t M, int64_t N, int64_t K) {
    const int64_t ldp = (K + TK - 1) / TK * TK;
    return 4 * (size_t)((M + N) * ldp) + 2 * 256;
}

mosaic_status ring_gemm_mma_s8(const uint32_t *A, int64_t lda, const uint32_t *B, int64_t ldb, uint32_t *C,
                               int64_t ldc, const uint32_t *Cin, int64_t ldcin, int sgn, int64_t M, int64_t N,
                               int64_t K, void *ws, size_t ws_bytes, cudaStream_t st) {
    if (M == 0 || N == 0) return MOSAIC_OK;
    if (!mma_s8_available()) return MOSAIC_ERR_UNSUPPORTED;
    if (M > (int64_t)INT32_MAX || N > (int64_t)INT32_MAX || (M + TM - 1) / TM > 65535) return MOSAIC_ERR_SHAPE;
    const int64_t ldp = (K + TK - 1) / TK * TK;
    if (ldp == 0) {
        const cudaError_t e = cudaMemset2DAsync(C, (size_t)ldc * 4, 0, (size_t)N * 4, (size_t)M, st);
        return e == cudaSuccess ? MOSAIC_OK : MOSAIC_ERR_CUDA;
    }
    if (!ws || ws_bytes < ws_mma_s8(M, N, K)) return MOSAIC_ERR_WORKSPACE;
    int8_t *Ap = reinterpret_cast<int8_t *>((reinterpret_cast<uintptr_t>(ws) + 255) & ~static_cast<uintptr_t>(255));
    int8_t *Bp = Ap + ((4 * M * ldp + 255) / 256) * 256;
    {
        KernelSpan span("split_s8", st);
        split_s8_kernel<<<grid_for(M * (ldp / 4), 256), 256, 0, st>>>(A, lda, M, K, Ap, ldp, M * ldp);
    }
    MOSAIC_TRY(launch_status());
    {
        KernelSpan span("split_s8", st);
        split_s8_kernel<<<grid_for(N * (ldp / 4), 256), 256, 0, st>>>(B, ldb, N, K, Bp, ldp, N * ldp);
    }
    MOSAIC_TRY(launch_status());
    static std::atomic<unsigned long long> attr_set{0};   // one bit per device ordinal
    if (!ensure_smem_limit(attr_set, ring_gemm_s8_kernel, 2 * STAGE_B)) return MOSAIC_ERR_CUDA;
    S8Args args{Ap, Bp, ldp, M * ldp, N * ldp, C, ldc, Cin, ldcin, sgn, (int)M, (int)N, (int)(ldp / TK)};
    const dim3 grid((unsigned)((N + TN - 1) / TN), (unsigned)((M + TM - 1) / TM));
    {
        KernelSpan span("ring_gemm_s8", st);
        ring_gemm_s8_kernel<<<grid, THREADS, 2 * STAGE_B, st>>>(args);
    }
    return launch_status();
}

}  // namespace mosaic
