// Ring product over Z_{2^32} for a few tokens: C = Cin + sgn * A B^T with A
// M x K (M <= 16 tokens), B N x K, both K-contiguous uint32, all sums wrapping
// mod 2^32 (the server product Y' = W' X' of Sec. 3 and the per-pass client
// compositions R^T C_d^T, R^T J_d^T, Q_d^T L^T of Eq. 5-7 when only a few
// tokens are in flight, e.g. one decode step).
//
// With M <= 16 every element of B is used M times, so the product is bound by
// streaming B from HBM once, 4 bytes per element, and the 10 digit-plane
// products of the tensor-core path (8 bytes of planes per element) would only
// double the traffic.  Each CTA is persistent (one per SM) and walks B tiles
// of BR rows:
//   warp 15     TMA producer: per stage one 2-D box {128 K, BR rows} of B and
//               one {128 K, MT rows} of A into shared memory; rows and K past
//               the ends are zero-filled by the copy engine
//   warps 0-14  consumers: warp w owns rows w*RW .. w*RW+RW-1 of the tile, lane
//               j the four K values 4j .. 4j+3 of every stage; it accumulates
//               RW x MT wrapping 32-bit dot-product pieces (integer multiply-add)
//               and, after the last stage of the tile, sums them across the
//               warp with a halving exchange (each step trades half of the
//               values with the partner lane) and writes C.
// Every wait is bounded; on expiry the kernel raises its error word, stops,
// lets its issued copies land (bounded) and returns.
#include "async_copy.cuh"
#include "mosaic_internal.cuh"

namespace mosaic {

__device__ uint32_t g_skinny_error = 0;

namespace {

constexpr int KC = 128;                     // K values per stage (512 bytes per row)
constexpr int CWARPS = 15;                  // consumer warps (16 warps in all: 128 registers a thread)
constexpr int THREADS = (CWARPS + 1) * 32;  // + one producer warp
constexpr int SMEM_BUDGET = 200 * 1024;

template <int MT, int RW>
struct SkCfg {
    static constexpr int BR = CWARPS * RW;     // B rows per tile
    static constexpr int B_BYTES = BR * KC * 4;
    static constexpr int A_BYTES = MT * KC * 4;
    static constexpr int STAGE = B_BYTES + A_BYTES;
    static constexpr int STAGES = SMEM_BUDGET / STAGE > 8 ? 8 : SMEM_BUDGET / STAGE;
    static constexpr int SMEM = STAGES * STAGE + 1024 + 2 * 8 * STAGES + 16;
    static_assert(STAGES >= 2, "");
    static_assert(BR <= 256 && MT <= 256, "TMA box rows");
};

struct SkArgs {
    uint32_t *C;
    int64_t ldc;
    const uint32_t *Cin;
    int64_t ldcin;
    int sgn;
    int M, N, nk, tiles;
};

__device__ __forceinline__ void raise_abort(volatile int *abort_flag) {
    *abort_flag = 1;
    atomicExch(&g_skinny_error, 1u);
}

template <int V>
struct Log2 {
    static constexpr int value = 1 + Log2<V / 2>::value;
};
template <>
struct Log2<1> {
    static constexpr int value = 0;
};

template <int MT, int RW>
__global__ void __launch_bounds__(THREADS, 1)
    ring_gemm_skinny_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                            SkArgs a) {
    using C = SkCfg<MT, RW>;
    constexpr int V = RW * MT;                 // partial sums per lane
    constexpr int H = Log2<V>::value < 5 ? Log2<V>::value : 5;   // halving exchanges
    constexpr int VL = V >> H;                 // sums a lane holds after them
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                ~static_cast<uintptr_t>(1023));
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + C::STAGES * C::STAGE);
    uint64_t *empty = full + C::STAGES;
    volatile int *abort_flag = reinterpret_cast<volatile int *>(empty + C::STAGES);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < C::STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], CWARPS);
        }
        *abort_flag = 0;
        mbar_init_fence();
    }
    __syncthreads();

    if (warp == CWARPS) {
        if (lane == 0) {
            uint32_t it = 0;
            bool ok = true;
            for (int tile = blockIdx.x; ok && tile < a.tiles; tile += gridDim.x) {
                for (int kc = 0; kc < a.nk; ++kc, ++it) {
                    const int s = (int)(it % C::STAGES);
                    const uint32_t ph = (it / C::STAGES) & 1u;
                    if (!mbar_wait(&empty[s], ph ^ 1u, abort_flag)) {
                        raise_abort(abort_flag);
                        ok = false;
                        break;
                    }
                    uint8_t *st = smem + s * C::STAGE;
                    mbar_expect_tx(&full[s], C::STAGE);
                    tma_load_2d(st, &tmB, &full[s], kc * KC, tile * C::BR);
                    tma_load_2d(st + C::B_BYTES, &tmA, &full[s], kc * KC, 0);
                }
            }
            // Let the last copy issued into every stage land before the CTA
            // exits (all of them have, unless a consumer gave up).
            const uint32_t first = it > (uint32_t)C::STAGES ? it - C::STAGES : 0;
            for (uint32_t q = first; q < it; ++q)
                if (!mbar_drain(&full[q % C::STAGES], (q / C::STAGES) & 1u)) atomicExch(&g_skinny_error, 1u);
        }
    } else {
        uint32_t it = 0;
        bool ok = true;
        const int r0 = warp * RW;
        for (int tile = blockIdx.x; ok && tile < a.tiles; tile += gridDim.x) {
            uint32_t acc[V];
#pragma unroll
            for (int v = 0; v < V; ++v) acc[v] = 0;
            for (int kc = 0; kc < a.nk; ++kc, ++it) {
                const int s = (int)(it % C::STAGES);
                if (!mbar_wait(&full[s], (it / C::STAGES) & 1u, abort_flag)) {
                    raise_abort(abort_flag);
                    ok = false;
                    break;
                }
                const uint4 *Bs = reinterpret_cast<const uint4 *>(smem + s * C::STAGE);
                const uint4 *As = reinterpret_cast<const uint4 *>(smem + s * C::STAGE + C::B_BYTES);
                uint4 b[RW];
#pragma unroll
                for (int r = 0; r < RW; ++r) b[r] = Bs[(r0 + r) * (KC / 4) + lane];
#pragma unroll
                for (int t = 0; t < MT; ++t) {
                    const uint4 x = As[t * (KC / 4) + lane];
#pragma unroll
                    for (int r = 0; r < RW; ++r)
                        acc[r * MT + t] += b[r].x * x.x + b[r].y * x.y + b[r].z * x.z + b[r].w * x.w;
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(&empty[s]);
            }
            if (!ok) break;
            // Sum the 32 lanes' pieces: H halving exchanges leave lane j with
            // the sums of values (j >> (5 - H)) * VL + i, i < VL; the lanes
            // that still share a value finish it with plain butterflies.
#pragma unroll
            for (int h = 0; h < H; ++h) {
                const int off = 16 >> h;
                const int half = V >> (h + 1);
                const bool upper = (lane & off) != 0;
#pragma unroll
                for (int i = 0; i < half; ++i) {
                    const uint32_t send = upper ? acc[i] : acc[half + i];
                    const uint32_t keep = upper ? acc[half + i] : acc[i];
                    acc[i] = keep + __shfl_xor_sync(0xffffffffu, send, off);
                }
            }
#pragma unroll
            for (int h = H; h < 5; ++h) {
#pragma unroll
                for (int i = 0; i < VL; ++i) acc[i] += __shfl_xor_sync(0xffffffffu, acc[i], 16 >> h);
            }
            if ((lane & ((1 << (5 - H)) - 1)) == 0) {
#pragma unroll
                for (int i = 0; i < VL; ++i) {
                    const int idx = (lane >> (5 - H)) * VL + i;
                    const int r = idx / MT, t = idx % MT;
                    const int64_t row = (int64_t)tile * C::BR + r0 + r;
                    if (t < a.M && row < a.N) {
                        uint32_t y = a.sgn < 0 ? 0u - acc[i] : acc[i];
                        if (a.Cin) y += a.Cin[(int64_t)t * a.ldcin + row];
                        a.C[(int64_t)t * a.ldc + row] = y;
                    }
                }
            }
        }
    }
}

// 2-D map over a K-contiguous uint32 matrix: {K, rows}, box {KC, box_rows}.
bool make_u32_map(CUtensorMap *map, const uint32_t *base, int64_t K, int64_t rows, int64_t ld, int box_rows) {
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)ld * 4};
    cuuint32_t box[2] = {(cuuint32_t)KC, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_UINT32, 2, const_cast<uint32_t *>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int MT, int RW>
mosaic_status launch_skinny(const uint32_t *A, int64_t lda, const uint32_t *B, int64_t ldb, uint32_t *Cm,
                            int64_t ldc, const uint32_t *Cin, int64_t ldcin, int sgn, int64_t M, int64_t N,
                            int64_t K, int sms, cudaStream_t st) {
    using C = SkCfg<MT, RW>;
    CUtensorMap ta, tb;
    if (!make_u32_map(&ta, A, K, M, lda, MT) || !make_u32_map(&tb, B, K, N, ldb, C::BR)) return MOSAIC_ERR_CUDA;
    static std::atomic<unsigned long long> attr_set{0};   // one bit per device ordinal
    if (!ensure_smem_limit(attr_set, ring_gemm_skinny_kernel<MT, RW>, C::SMEM)) return MOSAIC_ERR_CUDA;
    const int64_t tiles = (N + C::BR - 1) / C::BR;
    const int64_t nk = (K + KC - 1) / KC;
    if (tiles > 0x7fffffff || nk > 0x7fffffff) return MOSAIC_ERR_SHAPE;
    SkArgs args{Cm, ldc, Cin, ldcin, sgn, (int)M, (int)N, (int)nk, (int)tiles};
    const int grid = tiles < sms ? (int)tiles : sms;
    {
        KernelSpan span("ring_gemm_skinny", st);
        ring_gemm_skinny_kernel<MT, RW><<<grid, THREADS, C::SMEM, st>>>(ta, tb, args);
    }
    return launch_status();
}

template <int MT>
mosaic_status launch_rw(const uint32_t *A, int64_t lda, const uint32_t *B, int64_t ldb, uint32_t *Cm,
                        int64_t ldc, const uint32_t *Cin, int64_t ldcin, int sgn, int64_t M, int64_t N, int64_t K,
                        cudaStream_t st) {
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 1)
        return MOSAIC_ERR_CUDA;
    // 60-row tiles read the token slice of A half as often as 30-row tiles;
    // the smaller tiles are taken when they fill the last wave of the
    // persistent grid clearly better.
    auto eff = [&](int64_t br) {
        const int64_t t = (N + br - 1) / br, w = (t + sms - 1) / sms;
        return (double)t / (double)(w * sms);
    };
    if (eff(60) >= 0.85 || eff(60) >= eff(30))
        return launch_skinny<MT, 4>(A, lda, B, ldb, Cm, ldc, Cin, ldcin, sgn, M, N, K, sms, st);
    return launch_skinny<MT, 2>(A, lda, B, ldb, Cm, ldc, Cin, ldcin, sgn, M, N, K, sms, st);
}

}  // namespace

bool skinny_ok(const uint32_t *A, int64_t lda, const uint32_t *B, int64_t ldb, int64_t M, int64_t K) {
    return M >= 1 && M <= kSkinnyMaxM && K >= 1 && aligned16(A) && aligned16(B) && lda % 4 == 0 &&
           ldb % 4 == 0 && tc_available();
}

mosaic_status ring_gemm_skinny(const uint32_t *A, int64_t lda, const uint32_t *B, int64_t ldb, uint32_t *Cm,
                               int64_t ldc, const uint32_t *Cin, int64_t ldcin, int sgn, int64_t M, int64_t N,
                               int64_t K, cudaStream_t st) {
    if (N == 0) return MOSAIC_OK;
    if (!skinny_ok(A, lda, B, ldb, M, K) || N > (int64_t)INT32_MAX) return MOSAIC_ERR_SHAPE;
    if (M == 1) return launch_rw<1>(A, lda, B, ldb, Cm, ldc, Cin, ldcin, sgn, M, N, K, st);
    if (M == 2) return launch_rw<2>(A, lda, B, ldb, Cm, ldc, Cin, ldcin, sgn, M, N, K, st);
    if (M <= 4) return launch_rw<4>(A, lda, B, ldb, Cm, ldc, Cin, ldcin, sgn, M, N, K, st);
    if (M <= 8) return launch_rw<8>(A, lda, B, ldb, Cm, ldc, Cin, ldcin, sgn, M, N, K, st);
    return launch_rw<16>(A, lda, B, ldb, Cm, ldc, Cin, ldcin, sgn, M, N, K, st);
}

mosaic_status skinny_status() {
    uint32_t v = 0, zero = 0;
    if (cudaMemcpyFromSymbol(&v, g_skinny_error, sizeof v) != cudaSuccess) return MOSAIC_ERR_CUDA;
    if (v) {
        cudaMemcpyToSymbol(g_skinny_error, &zero, sizeof zero);
        return MOSAIC_ERR_TIMEOUT;
    }
    return MOSAIC_OK;
}

}  // namespace mosaic
