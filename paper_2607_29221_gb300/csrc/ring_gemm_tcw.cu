// Ring product over Z_{2^32} on the tensor cores for a few token rows
// (17 to 64), streaming the wide operand as uint32.
//
// C = A B^T with A: M x K (tokens, M <= 64) and B: N x K (masked weights,
// N in the thousands).  With so few tokens every element of B is used at most
// 64 times, so the product is bound by reading B (Sec. 5.2: decode at small
// batch is memory-bound).  The digit-plane product (ring_gemm_tc.cu) reads B
// as four bf16 planes, 8 bytes an element; this kernel reads the uint32 B,
// 4 bytes an element, and splits it into digits on the chip:
//   * 128 rows x 32 K of B land in shared memory by TMA (128-byte swizzle);
//   * converter warps split each element into its four signed base-2^8
//     digits d_i = byte_i(b + 0x80808080) - 128 as fp16 (exact for
//     |d| <= 128) and store them with tcgen05.st into a ring of tensor-memory
//     slots, from where the MMA reads its A operand: shared memory carries
//     only the TMA traffic and the small token operand;
//   * the tokens' digit planes (fp16 [4][M][Kp], split once per call) come by
//     TMA as one 3-D box {32 K, NT rows, 4 planes} per stage (64-byte swizzle);
//   * the product D (128 weight rows x tokens) = W_i [X_0; ...; X_{3-i}]^T
//     runs as ONE tcgen05.mma per weight digit i with N = (4 - i) NT, written
//     at column i NT of an accumulator set whose shift group s occupies
//     columns [s NT, (s + 1) NT): column block j of MMA i lands in group i + j,
//     so the 10 digit pairs with i + j <= 3 take 4 MMAs per 16 K;
//   * every 256 K (group 3 then holds 1024 products of at most 2^14, an exact
//     fp32 integer) the epilogue folds all four groups into int32 registers,
//     acc += g0 + 2^8 g1 + 2^16 g2 + 2^24 g3 mod 2^32, while the MMAs go on in
//     the other accumulator set (two sets when 8 NT columns leave room for
//     the digit slots);
//   * (weight tile, 256-K chunk) units are split evenly over a persistent
//     grid (stream-K); each CTA adds its partial tiles into C with red.add
//     (C is zeroed first), exact and order-free in Z_{2^32}.
// Warps: 0 TMA producer, 1 TMEM allocation + MMA issuer, 2..5 converters,
// 6..9 epilogue (warp w reaches TMEM lanes 32 (w % 4) .. + 31).  Every wait is
// bounded (about 2 s of %globaltimer): on expiry the kernel raises its device
// error word (read by tcw_status), stops, lets its own copies and products
// land (bounded), frees TMEM and returns.
#include <cuda.h>
#include <cuda_fp16.h>
#include <cudaTypedefs.h>

#include "async_copy.cuh"
#include "mosaic_internal.cuh"

namespace mosaic {

// Set when the kernel gave up a bounded wait.
__device__ uint32_t g_tcw_error = 0;

namespace {

constexpr int WR = 128;          // weight rows per tile (MMA M)
constexpr int KB = 32;           // K per stage
constexpr int CHUNK = 8;         // stages per drain: 256 K
constexpr uint32_t TMEM_COLS = 512;
constexpr int THREADS = 320;
constexpr int CONV_WARPS = 4;
constexpr int EPI_WARPS = 4;
constexpr int W_BOX = WR * KB * 4;          // 16 KB of uint32

template <int NT>
struct WCfg {
    static constexpr int X_PLANE = NT * KB * 2;            // one fp16 digit plane of the token box
    static constexpr int X_BOX = 4 * X_PLANE;
    static constexpr int STAGE = W_BOX + X_BOX;
    static constexpr int STAGES = NT <= 48 ? 6 : 5;
    static constexpr int NSETS = 8 * NT <= 384 ? 2 : 1;    // accumulator sets of 4 NT columns
    static constexpr int ACC_COLS = NSETS * 4 * NT;
    static constexpr int SLOTS_FIT = ((int)TMEM_COLS - ACC_COLS) / 64;
    static constexpr int SLOTS = SLOTS_FIT > 4 ? 4 : SLOTS_FIT;   // digit slots of 64 columns (4 planes x 32 K)
    static constexpr int SMEM = STAGES * STAGE + 1024 + 512;
    static_assert(NT % 16 == 0 && NT >= 16 && NT <= 64, "");
    static_assert(SLOTS >= 2, "at least two digit slots");
    static_assert(X_PLANE % 512 == 0, "token planes keep the 64-byte swizzle phase");
    // kind::f16 descriptor: D f32, A and B fp16, both K-major, N >> 3, M >> 4.
    __host__ __device__ static constexpr uint32_t idesc(int n) {
        return (1u << 4) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(WR >> 4) << 24);
    }
};

struct WArgs {
    uint32_t *C;
    int64_t ldc;
    int M, N, K;
    int tiles, nchunks;
};

__device__ __forceinline__ void raise_abort(volatile int *abort_flag) {
    *abort_flag = 1;
    atomicExch(&g_tcw_error, 1u);
}
__device__ __forceinline__ void fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// Shared-memory matrix descriptor: K-major, 64-byte swizzle, 8-row groups 512 B apart.
__device__ __forceinline__ uint64_t sdesc_sw64(uint32_t saddr) {
    uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);
    d |= (uint64_t)1 << 16;
    d |= (uint64_t)(512 >> 4) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)4 << 61;
    return d;
}
// D (TMEM) (+)= A (TMEM) x B (shared memory)^T.
__device__ __forceinline__ void umma_tmem_a(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc, uint32_t idesc,
                                            uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
        "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
__device__ __forceinline__ void umma_commit(uint64_t *bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                     smem_u32(bar))
                 : "memory");
}
// 16 columns of the warp's 32 lanes; the caller waits (tcgen05.wait::ld).
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t *v) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
          "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15])
        : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
// 16 columns of the warp's 32 lanes from registers.
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t *v) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
        "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};" ::"r"(taddr),
        "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]),
        "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15])
        : "memory");
}
__device__ __forceinline__ void tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// Digit i of two elements (already offset by 0x80808080) as two fp16 values
// (byte - 128) in one word: the bytes sit in the mantissas of 1024 + byte,
// and one packed subtraction of 1152 leaves byte - 128 (exact: every value
// involved is an integer below 2^11).
__device__ __forceinline__ uint32_t digit_pair_f16(uint32_t b0, uint32_t b1, int i) {
    const uint32_t t = __byte_perm(b0, b1, (uint32_t)i | ((uint32_t)(4 + i) << 8));
    const uint32_t h = (t & 0x00FF00FFu) | 0x64006400u;
    __half2 x = *reinterpret_cast<const __half2 *>(&h);
    const uint32_t c = 0xE480E480u;   // (-1152, -1152)
    x = __hadd2(x, *reinterpret_cast<const __half2 *>(&c));
    return *reinterpret_cast<uint32_t *>(&x);
}

// Exact fold of the four shift groups of one column into acc (mod 2^32).
// After 256 K: |g0| <= 2^22, |g1| <= 2^23, |g2| <= 3 2^22, |g3| <= 2^24.
// kM = 1.5 2^23: for an integer y with |y| <= 2^22, y + kM has the bits of
// kM + y, so fma(x, 2^-8, kM) - kM = round(x / 2^8) exactly and
// x - 2^8 round(x / 2^8) is exact with magnitude <= 2^7.
constexpr float kM = 12582912.0f;
__device__ __forceinline__ uint32_t fold4(float g0, float g1, float g2, float g3) {
    // g0 + 2^8 g1 = s01 + 2^16 h1, s01 = g0 + 2^8 (g1 - 2^8 h1) exact (|s01| < 2^24);
    // h1 << 16 is the bits of (g1 / 2^8 + kM) shifted by 16 (bits(kM) << 16 = 0 mod 2^32).
    const float t1 = __fmaf_rn(g1, 0.00390625f, kM);
    const float lo1 = __fmaf_rn(__fsub_rn(t1, kM), -256.0f, g1);
    const float s01 = __fmaf_rn(lo1, 256.0f, g0);
    // (g2 << 16) + (g3 << 24) = s23 << 16 mod 2^32, s23 = g2 + 2^8 (g3 mod+- 2^8) exact.
    const float lo3 = __fmaf_rn(__fsub_rn(__fmaf_rn(g3, 0.00390625f, kM), kM), -256.0f, g3);
    const float s23 = __fmaf_rn(lo3, 256.0f, g2);
    return (uint32_t)__float2int_rn(s01) + (__float_as_uint(t1) << 16) + ((uint32_t)__float2int_rn(s23) << 16);
}

template <int NT>
__global__ void __launch_bounds__(THREADS, 1)
    ring_gemm_tcw_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX,
                         WArgs a) {
    using C = WCfg<NT>;
    constexpr int S = C::STAGES, SL = C::SLOTS, NS = C::NSETS;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                ~static_cast<uintptr_t>(1023));
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + S * C::STAGE);
    uint64_t *empty = full + S;
    uint64_t *a_full = empty + S;
    uint64_t *a_empty = a_full + SL;
    uint64_t *acc_full = a_empty + SL;
    uint64_t *acc_empty = acc_full + NS;
    uint64_t *drain = acc_empty + NS;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(drain + 1);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nk = (a.K + KB - 1) / KB;
    // This CTA's units [u0, u1) of (tile, chunk), numbered tile-major.
    const int64_t U = (int64_t)a.tiles * a.nchunks;
    const int u0 = (int)(U * blockIdx.x / gridDim.x), u1 = (int)(U * (blockIdx.x + 1) / gridDim.x);
    const int tile0 = u0 / a.nchunks, c0 = u0 - tile0 * a.nchunks;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], CONV_WARPS + 1);
        }
        for (int b = 0; b < SL; ++b) {
            mbar_init(&a_full[b], CONV_WARPS);
            mbar_init(&a_empty[b], 1);
        }
        for (int s = 0; s < NS; ++s) {
            mbar_init(&acc_full[s], 1);
            mbar_init(&acc_empty[s], EPI_WARPS);
        }
        mbar_init(drain, 1);
        *abort_flag = 0;
        mbar_init_fence();
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                     "r"(TMEM_COLS)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    fence_before();
    __syncthreads();
    fence_after();
    const uint32_t tmem = *tmem_slot;
    const uint32_t slot_col = (uint32_t)C::ACC_COLS;   // first digit slot

    if (warp == 0) {
        // ---- TMA producer ----
        if (lane == 0) {
            int g = 0;   // stages issued
            int tile = tile0, c = c0;
            for (int u = u0; u < u1 && !*abort_flag; ++u) {
                const int kb1 = (c + 1) * CHUNK < nk ? (c + 1) * CHUNK : nk;
                bool ok = true;
                for (int kb = c * CHUNK; kb < kb1; ++kb, ++g) {
                    const int s = g % S, round = g / S;
                    if (round > 0 && !mbar_wait(&empty[s], (uint32_t)(round - 1) & 1u, abort_flag)) {
                        raise_abort(abort_flag);
                        ok = false;
                        break;
                    }
                    uint8_t *st = smem + s * C::STAGE;
                    mbar_expect_tx(&full[s], C::STAGE);
                    tma_load_2d(st, &tmW, &full[s], kb * KB, tile * WR);
                    tma_load_3d(st + W_BOX, &tmX, &full[s], kb * KB, 0, 0);
                }
                if (!ok) break;
                if (++c == a.nchunks) {
                    c = 0;
                    ++tile;
                }
            }
            if (*abort_flag) {
                // Let the copies this thread started land before the CTA exits.
                for (int q = g > S ? g - S : 0; q < g; ++q) mbar_drain(&full[q % S], (uint32_t)(q / S) & 1u);
            }
        }
    } else if (warp == 1) {
        // ---- MMA issuer ----
        if (lane == 0) {
            bool issued_any = false;
            int g = 0, cc = 0;   // stages consumed, chunks issued
            int c = c0;
            const uint64_t desc0 = sdesc_sw64(smem_u32(smem));
            for (int u = u0; u < u1 && !*abort_flag; ++u) {
                const int set = cc % NS, sround = cc / NS;
                if (sround > 0 && !mbar_wait(&acc_empty[set], (uint32_t)(sround - 1) & 1u, abort_flag)) {
                    raise_abort(abort_flag);
                    break;
                }
                fence_after();
                const uint32_t dset = tmem + (uint32_t)(set * 4 * NT);
                const int kb1 = (c + 1) * CHUNK < nk ? (c + 1) * CHUNK : nk;
                bool ok = true;
                for (int kb = c * CHUNK; kb < kb1; ++kb, ++g) {
                    const int s = g % S, b = g % SL;
                    if (!mbar_wait(&full[s], (uint32_t)(g / S) & 1u, abort_flag) ||
                        !mbar_wait(&a_full[b], (uint32_t)(g / SL) & 1u, abort_flag)) {
                        raise_abort(abort_flag);
                        ok = false;
                        break;
                    }
                    fence_after();
                    const uint64_t dx = desc0 + (uint64_t)((s * C::STAGE + W_BOX) >> 4);
                    const uint32_t aslot = tmem + slot_col + (uint32_t)(b * 64);
                    const bool first = kb == c * CHUNK;
#pragma unroll
                    for (int kk = 0; kk < KB / 16; ++kk) {
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            // Weight digit i against token digits 0 .. 3 - i: groups i .. 3.
                            umma_tmem_a(dset + (uint32_t)(i * NT), aslot + (uint32_t)(16 * i + 8 * kk),
                                        dx + (uint64_t)(2 * kk), C::idesc((4 - i) * NT),
                                        (first && kk == 0 && i == 0) ? 0u : 1u);
                        }
                    }
                    issued_any = true;
                    umma_commit(&empty[s]);
                    umma_commit(&a_empty[b]);
                }
                if (!ok) break;
                umma_commit(&acc_full[set]);
                ++cc;
                if (++c == a.nchunks) c = 0;
            }
            if (*abort_flag && issued_any) {
                umma_commit(drain);
                mbar_drain(drain, 0);
            }
        }
    } else if (warp < 2 + CONV_WARPS) {
        // ---- converters: row r of each weight box -> four fp16 digit columns in a TMEM slot ----
        const int q = warp & 3;
        const int r = q * 32 + lane;
        const uint32_t lane_base = tmem + ((uint32_t)(q * 32) << 16) + slot_col;
        int g = 0;
        int c = c0;
        bool ok = true;
        for (int u = u0; u < u1 && ok; ++u) {
            const int kb1 = (c + 1) * CHUNK < nk ? (c + 1) * CHUNK : nk;
            for (int kb = c * CHUNK; kb < kb1; ++kb, ++g) {
                const int s = g % S, b = g % SL;
                if (!mbar_wait(&full[s], (uint32_t)(g / S) & 1u, abort_flag)) {
                    raise_abort(abort_flag);
                    ok = false;
                    break;
                }
                // Row r of the box: 8 chunks of 16 bytes, chunk j stored at j ^ (r & 7).
                const uint32_t row_addr = smem_u32(smem + s * C::STAGE) + (uint32_t)r * 128u;
                uint32_t w[32];
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    const uint32_t addr = row_addr + (uint32_t)((j ^ (r & 7)) * 16);
                    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                                 : "=r"(w[4 * j]), "=r"(w[4 * j + 1]), "=r"(w[4 * j + 2]), "=r"(w[4 * j + 3])
                                 : "r"(addr)
                                 : "memory");
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(&empty[s]);
#pragma unroll
                for (int k = 0; k < 32; ++k) w[k] += 0x80808080u;
                if (g >= SL && !mbar_wait(&a_empty[b], (uint32_t)(g / SL - 1) & 1u, abort_flag)) {
                    raise_abort(abort_flag);
                    ok = false;
                    break;
                }
                fence_after();
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    uint32_t d[16];
#pragma unroll
                    for (int p = 0; p < 16; ++p) d[p] = digit_pair_f16(w[2 * p], w[2 * p + 1], i);
                    tmem_st16(lane_base + (uint32_t)(b * 64 + 16 * i), d);
                }
                tmem_st_wait();
                fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&a_full[b]);
            }
            if (++c == a.nchunks) c = 0;
        }
        tmem_st_wait();
    } else {
        // ---- epilogue: drain every chunk, add finished tile segments into C ----
        const int q = warp & 3;
        const int r = q * 32 + lane;
        const uint32_t lane_addr = tmem + ((uint32_t)(q * 32) << 16);
        uint32_t acc[NT];
#pragma unroll
        for (int t = 0; t < NT; ++t) acc[t] = 0u;
        int cc = 0;
        int tile = tile0, c = c0;
        for (int u = u0; u < u1; ++u) {
            const int set = cc % NS;
            if (!mbar_wait(&acc_full[set], (uint32_t)(cc / NS) & 1u, abort_flag)) {
                raise_abort(abort_flag);
                break;
            }
            fence_after();
            const uint32_t sa = lane_addr + (uint32_t)(set * 4 * NT);
#pragma unroll
            for (int p = 0; p < NT; p += 16) {
                uint32_t g0[16], g1[16], g2[16], g3[16];
                tmem_ld16(sa + 0 * NT + p, g0);
                tmem_ld16(sa + 1 * NT + p, g1);
                tmem_ld16(sa + 2 * NT + p, g2);
                tmem_ld16(sa + 3 * NT + p, g3);
                tmem_ld_wait();
#pragma unroll
                for (int j = 0; j < 16; ++j)
                    acc[p + j] += fold4(__uint_as_float(g0[j]), __uint_as_float(g1[j]), __uint_as_float(g2[j]),
                                        __uint_as_float(g3[j]));
            }
            fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&acc_empty[set]);
            ++cc;
            const bool tile_end = c == a.nchunks - 1 || u == u1 - 1;
            if (tile_end) {
                const int n = tile * WR + r;
                if (n < a.N) {
                    uint32_t *col = a.C + n;
#pragma unroll
                    for (int t = 0; t < NT; ++t)
                        if (t < a.M)
                            asm volatile("red.global.add.u32 [%0], %1;" ::"l"(col + (int64_t)t * a.ldc), "r"(acc[t])
                                         : "memory");
                }
#pragma unroll
                for (int t = 0; t < NT; ++t) acc[t] = 0u;
            }
            if (++c == a.nchunks) {
                c = 0;
                ++tile;
            }
        }
    }
    fence_before();
    __syncthreads();
    if (warp == 1) {
        fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TMEM_COLS) : "memory");
    }
}

// Digit planes of the token operand as fp16 bits: planes[d][r][c] = byte_d(a + 0x80808080) - 128.
__global__ void digit_split_f16_kernel(const uint32_t *a, int64_t lda, int64_t rows, int64_t cols,
                                       uint16_t *planes, int64_t ldp, int64_t plane_stride) {
    const int64_t total = rows * cols;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = i / cols, c = i - r * cols;
        const uint32_t b = a[r * lda + c] + 0x80808080u;
#pragma unroll
        for (int d = 0; d < 4; ++d)
            planes[d * plane_stride + r * ldp + c] =
                __half_as_ushort(__int2half_rn((int)((b >> (8 * d)) & 0xffu) - 128));
    }
}

bool make_w_map(CUtensorMap *map, const uint32_t *B, int64_t K, int64_t N, int64_t ldb) {
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)N};
    cuuint64_t strides[1] = {(cuuint64_t)ldb * 4};
    cuuint32_t box[2] = {(cuuint32_t)KB, (cuuint32_t)WR};
    cuuint32_t estr[2] = {1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_UINT32, 2, const_cast<uint32_t *>(B), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool make_x_map(CUtensorMap *map, const uint16_t *planes, int64_t K, int64_t M, int64_t ldp, int nt) {
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[3] = {(cuuint64_t)K, (cuuint64_t)M, 4};
    cuuint64_t strides[2] = {(cuuint64_t)ldp * 2, (cuuint64_t)(M * ldp) * 2};
    cuuint32_t box[3] = {(cuuint32_t)KB, (cuuint32_t)nt, 4};
    cuuint32_t estr[3] = {1, 1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 3, const_cast<uint16_t *>(planes), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int NT>
mosaic_status launch_tcw(const CUtensorMap &tw, const CUtensorMap &tx, const WArgs &args, int sms,
                         cudaStream_t st) {
    using C = WCfg<NT>;
    static std::atomic<unsigned long long> attr_set{0};
    if (!ensure_smem_limit(attr_set, ring_gemm_tcw_kernel<NT>, C::SMEM)) return MOSAIC_ERR_CUDA;
    const int64_t units = (int64_t)args.tiles * args.nchunks;
    const int64_t grid = units < sms ? units : sms;
    ring_gemm_tcw_kernel<NT><<<(unsigned)grid, THREADS, C::SMEM, st>>>(tw, tx, args);
    return launch_status();
}

}  // namespace

mosaic_status tcw_status() {
    uint32_t v = 0, zero = 0;
    if (cudaMemcpyFromSymbol(&v, g_tcw_error, sizeof v) != cudaSuccess) return MOSAIC_ERR_CUDA;
    if (v) {
        cudaMemcpyToSymbol(g_tcw_error, &zero, sizeof zero);
        return MOSAIC_ERR_TIMEOUT;
    }
    return MOSAIC_OK;
}

size_t tcw_ws_bytes(int64_t M, int64_t K) { return (size_t)(4 * M * ((K + 7) / 8 * 8)) * 2; }

bool tcw_ok(const uint32_t *A, int64_t lda, const uint32_t *B, int64_t ldb, int64_t M, int64_t N, int64_t K) {
    return M > kSkinnyMaxM && M <= kTcwMaxM && N >= 1 && K >= 1 && aligned16(A) && aligned16(B) && lda % 4 == 0 &&
           ldb % 4 == 0 && tc_available();
}

mosaic_status ring_gemm_tcw(const uint32_t *A, int64_t lda, const uint32_t *B, int64_t ldb, uint32_t *Cm,
                            int64_t ldc, int64_t M, int64_t N, int64_t K, uint16_t *Ap, cudaStream_t st) {
    if (M < 1 || M > kTcwMaxM || N < 1 || K < 1 || N > (int64_t)INT32_MAX || K > ((int64_t)1 << 20))
        return MOSAIC_ERR_SHAPE;
    if (!aligned16(Ap)) return MOSAIC_ERR_ALIGN;
    const int64_t Kp = (K + 7) / 8 * 8;
    digit_split_f16_kernel<<<grid_for(M * K, 256), 256, 0, st>>>(A, lda, M, K, Ap, Kp, M * Kp);
    MOSAIC_TRY(launch_status());
    if (cudaMemset2DAsync(Cm, (size_t)ldc * 4, 0, (size_t)N * 4, (size_t)M, st) != cudaSuccess)
        return MOSAIC_ERR_CUDA;
    const int nt = M <= 32 ? 32 : M <= 48 ? 48 : 64;
    CUtensorMap tw, tx;
    if (!make_w_map(&tw, B, K, N, ldb) || !make_x_map(&tx, Ap, K, M, Kp, nt)) return MOSAIC_ERR_CUDA;
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 1)
        return MOSAIC_ERR_CUDA;
    const int64_t tiles = (N + WR - 1) / WR, nk = (K + KB - 1) / KB, nchunks = (nk + CHUNK - 1) / CHUNK;
    if (tiles * nchunks > (int64_t)INT32_MAX) return MOSAIC_ERR_SHAPE;
    const WArgs args{Cm, ldc, (int)M, (int)N, (int)K, (int)tiles, (int)nchunks};
    if (nt == 32) return launch_tcw<32>(tw, tx, args, sms, st);
    if (nt == 48) return launch_tcw<48>(tw, tx, args, sms, st);
    return launch_tcw<64>(tw, tx, args, sms, st);
}

}  // namespace mosaic
