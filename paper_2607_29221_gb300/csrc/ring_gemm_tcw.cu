// Ring product over Z_{2^32} on the tensor cores for a few token rows
// (17 to 64), streaming the wide operand as uint32.
//
// C = A B^T with A: M x K (tokens, M <= 64) and B: N x K (masked weights,
// N in the thousands).  With so few tokens every element of B is used at most
// 64 times, so the product is bound by reading B (Sec. 5.2: decode at small
// batch is memory-bound).  The digit-plane product (ring_gemm_tc.cu) reads B
// as four bf16 planes, 8 bytes an element; this kernel reads the uint32 B,
// 4 bytes an element, and splits it into digits on the chip:
//   * a stage is 64 K: two boxes of 128 rows x 32 K of B land in shared
//     memory by TMA (128-byte swizzle), in a ring of their own that the
//     converters release as soon as they have read them;
//   * converter warps split each element into its four signed base-2^8
//     digits d_i = byte_i(b + 0x80808080) - 128 as fp16 (exact for
//     |d| <= 128) and store them with tcgen05.st into a ring of tensor-memory
//     slots, from where the MMA reads its A operand: shared memory carries
//     only the TMA traffic and the small token operand;
//   * the tokens' digit planes (fp16 [4][M][Kp], split once per call) come by
//     TMA as two 3-D boxes {32 K, NT rows, 4 planes} per stage (64-byte
//     swizzle) into a second ring; one barrier per stage, armed by a single
//     MMA commit, releases both the token boxes and the stage's digit slot;
//   * the product D (128 weight rows x tokens) = W_i [X_0; ...; X_{3-i}]^T
//     runs as ONE tcgen05.mma per weight digit i and 16 K with N = (4 - i) NT, written
//     at column i NT of an accumulator set whose shift group s occupies
//     columns [s NT, (s + 1) NT): column block j of MMA i lands in group i + j,
//     so the 10 digit pairs with i + j <= 3 take 4 MMAs per 16 K;
//   * every 256 K (group 3 then holds 1024 products of at most 2^14, an exact
//     fp32 integer) the epilogue folds all four groups into int32 registers,
//     acc += g0 + 2^8 g1 + 2^16 g2 + 2^24 g3 mod 2^32, while the MMAs go on in
//     the other accumulator set (two sets when 8 NT columns leave room for
//     four digit slots);
//   * (weight tile, 256-K chunk) units are split evenly over a persistent
//     grid (stream-K); each CTA adds its partial tiles into C with red.add
//     (C is zeroed first), exact and order-free in Z_{2^32}.
// Warps: 0 TMA producer, 1 TMEM allocation + MMA issuer, 2..9 converters
// (two groups of four, one warp per TMEM lane quarter; group j converts the
// j-th 32-K box of every stage), 10..13 epilogue (warp w reaches TMEM lanes
// 32 (w % 4) .. + 31).  Every wait is
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
constexpr int KB = 32;           // K per TMA box
constexpr int KS = 64;           // K per stage: two boxes
constexpr int CHUNK = 4;         // stages per drain: 256 K
constexpr uint32_t TMEM_COLS = 512;
constexpr int CONV_WARPS = 8;    // two groups of four (one warp per TMEM lane quarter)
constexpr int EPI_WARPS = 4;
constexpr int THREADS = 32 * (2 + CONV_WARPS + EPI_WARPS);
constexpr int W_BOX = WR * KB * 4;          // 16 KB of uint32
constexpr int SLOT_COLS = 4 * (KS / 2);     // a stage's digits: 4 planes x 32 columns (64 K of fp16 pairs)
constexpr int SLOTS = 2;                    // digit slots (stages) in TMEM

template <int NT>
struct WCfg {
    static constexpr int X_PLANE = NT * KB * 2;            // one fp16 digit plane of a token box
    static constexpr int X_BOX = 4 * X_PLANE;
    static constexpr int WST = NT == 64 ? 3 : 4;           // weight stages (2 boxes each) in the ring
    static constexpr int XST = NT == 64 ? 3 : 4;           // token stages (2 boxes each) in the ring
    static constexpr int NSETS = 8 * NT + SLOTS * SLOT_COLS <= (int)TMEM_COLS ? 2 : 1;   // accumulator sets
    static constexpr int ACC_COLS = NSETS * 4 * NT;
    static constexpr int SMEM = WST * 2 * W_BOX + XST * 2 * X_BOX + 1024 + 512;
    static_assert(SMEM <= 227 * 1024, "");
    static_assert(ACC_COLS + SLOTS * SLOT_COLS <= (int)TMEM_COLS, "");
    static_assert(NT % 16 == 0 && NT >= 16 && NT <= 64, "");
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
// 8 columns of the warp's 32 lanes; the caller waits (tcgen05.wait::ld).
__device__ __forceinline__ void tmem_ld8(uint32_t taddr, uint32_t *v) {
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
                 : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7])
                 : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
// 8 columns of the warp's 32 lanes from registers.
__device__ __forceinline__ void tmem_st8(uint32_t taddr, const uint32_t *v) {
    asm volatile("tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"r"(taddr),
                 "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7])
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
    constexpr int SW = C::WST, SX = C::XST, NS = C::NSETS;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                ~static_cast<uintptr_t>(1023));
    uint8_t *xring = smem + SW * 2 * W_BOX;
    uint64_t *w_full = reinterpret_cast<uint64_t *>(xring + SX * 2 * C::X_BOX);
    uint64_t *w_empty = w_full + SW;
    uint64_t *x_full = w_empty + SW;
    uint64_t *done = x_full + SX;       // stage s's MMAs complete: its token boxes and digit slot are free
    uint64_t *a_full = done + SX;
    uint64_t *acc_full = a_full + SLOTS;
    uint64_t *acc_empty = acc_full + NS;
    uint64_t *drain = acc_empty + NS;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(drain + 1);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nst = (a.K + KS - 1) / KS;   // stages of a tile
    // This CTA's units [u0, u1) of (tile, 256-K chunk), numbered tile-major.
    const int64_t U = (int64_t)a.tiles * a.nchunks;
    const int u0 = (int)(U * blockIdx.x / gridDim.x), u1 = (int)(U * (blockIdx.x + 1) / gridDim.x);
    const int tile0 = u0 / a.nchunks, c0 = u0 - tile0 * a.nchunks;

    if (threadIdx.x == 0) {
        for (int s = 0; s < SW; ++s) {
            mbar_init(&w_full[s], 1);
            mbar_init(&w_empty[s], CONV_WARPS);
        }
        for (int s = 0; s < SX; ++s) {
            mbar_init(&x_full[s], 1);
            mbar_init(&done[s], 1);
        }
        for (int b = 0; b < SLOTS; ++b) mbar_init(&a_full[b], CONV_WARPS);
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
        // ---- TMA producer: stage g = two W boxes and two token boxes of 32 K ----
        if (lane == 0) {
            int g = 0;   // stages issued
            int tile = tile0, c = c0;
            for (int u = u0; u < u1 && !*abort_flag; ++u) {
                const int ks1 = (c + 1) * CHUNK < nst ? (c + 1) * CHUNK : nst;
                bool ok = true;
                for (int ks = c * CHUNK; ks < ks1; ++ks, ++g) {
                    const int sw = g % SW, sx = g % SX;
                    if ((g >= SW && !mbar_wait(&w_empty[sw], (uint32_t)(g / SW - 1) & 1u, abort_flag)) ||
                        (g >= SX && !mbar_wait(&done[sx], (uint32_t)(g / SX - 1) & 1u, abort_flag))) {
                        raise_abort(abort_flag);
                        ok = false;
                        break;
                    }
                    uint8_t *ws = smem + sw * 2 * W_BOX;
                    mbar_expect_tx(&w_full[sw], 2 * W_BOX);
                    tma_load_2d(ws, &tmW, &w_full[sw], ks * KS, tile * WR);
                    tma_load_2d(ws + W_BOX, &tmW, &w_full[sw], ks * KS + KB, tile * WR);
                    uint8_t *xs = xring + sx * 2 * C::X_BOX;
                    mbar_expect_tx(&x_full[sx], 2 * C::X_BOX);
                    tma_load_3d(xs, &tmX, &x_full[sx], ks * KS, 0, 0);
                    tma_load_3d(xs + C::X_BOX, &tmX, &x_full[sx], ks * KS + KB, 0, 0);
                }
                if (!ok) break;
                if (++c == a.nchunks) {
                    c = 0;
                    ++tile;
                }
            }
            if (*abort_flag) {
                // Let the copies this thread started land before the CTA exits.
                for (int q = g > SW ? g - SW : 0; q < g; ++q) mbar_drain(&w_full[q % SW], (uint32_t)(q / SW) & 1u);
                for (int q = g > SX ? g - SX : 0; q < g; ++q) mbar_drain(&x_full[q % SX], (uint32_t)(q / SX) & 1u);
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
                const int ks1 = (c + 1) * CHUNK < nst ? (c + 1) * CHUNK : nst;
                bool ok = true;
                for (int ks = c * CHUNK; ks < ks1; ++ks, ++g) {
                    const int sx = g % SX, b = g % SLOTS;
                    if (!mbar_wait(&x_full[sx], (uint32_t)(g / SX) & 1u, abort_flag) ||
                        !mbar_wait(&a_full[b], (uint32_t)(g / SLOTS) & 1u, abort_flag)) {
                        raise_abort(abort_flag);
                        ok = false;
                        break;
                    }
                    fence_after();
                    const uint64_t dx = desc0 + (uint64_t)((SW * 2 * W_BOX + sx * 2 * C::X_BOX) >> 4);
                    const uint32_t aslot = tmem + slot_col + (uint32_t)(b * SLOT_COLS);
                    const bool first = ks == c * CHUNK;
#pragma unroll
                    for (int j = 0; j < 2; ++j) {
#pragma unroll
                        for (int kk = 0; kk < KB / 16; ++kk) {
#pragma unroll
                            for (int i = 0; i < 4; ++i) {
                                // Weight digit i against token digits 0 .. 3 - i: groups i .. 3.
                                umma_tmem_a(dset + (uint32_t)(i * NT), aslot + (uint32_t)(32 * i + 16 * j + 8 * kk),
                                            dx + (uint64_t)((j * C::X_BOX) >> 4) + (uint64_t)(2 * kk),
                                            C::idesc((4 - i) * NT), (first && j == 0 && kk == 0 && i == 0) ? 0u : 1u);
                            }
                        }
                    }
                    issued_any = true;
                    umma_commit(&done[sx]);
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
        // ---- converters: group j, row r of box j of each stage -> four fp16
        // digit planes of 16 words (32 K) in the stage's TMEM slot ----
        const int q = warp & 3, j = (warp - 2) >> 2;
        const int r = q * 32 + lane;
        const uint32_t lane_base = tmem + ((uint32_t)(q * 32) << 16) + slot_col + (uint32_t)(16 * j);
        int g = 0;
        int c = c0;
        bool ok = true;
        for (int u = u0; u < u1 && ok; ++u) {
            const int ks1 = (c + 1) * CHUNK < nst ? (c + 1) * CHUNK : nst;
            for (int ks = c * CHUNK; ks < ks1; ++ks, ++g) {
                const int sw = g % SW, b = g % SLOTS;
                if (!mbar_wait(&w_full[sw], (uint32_t)(g / SW) & 1u, abort_flag)) {
                    raise_abort(abort_flag);
                    ok = false;
                    break;
                }
                // Row r of box j: 8 chunks of 16 bytes, chunk i stored at i ^ (r & 7).
                const uint32_t row_addr = smem_u32(smem + (sw * 2 + j) * W_BOX) + (uint32_t)r * 128u;
                uint32_t w[32];
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const uint32_t addr = row_addr + (uint32_t)((i ^ (r & 7)) * 16);
                    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                                 : "=r"(w[4 * i]), "=r"(w[4 * i + 1]), "=r"(w[4 * i + 2]), "=r"(w[4 * i + 3])
                                 : "r"(addr)
                                 : "memory");
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(&w_empty[sw]);
#pragma unroll
                for (int k = 0; k < 32; ++k) w[k] += 0x80808080u;
                // The stage two back used this slot: its MMAs must be complete.
                if (g >= SLOTS && !mbar_wait(&done[(g - SLOTS) % SX], (uint32_t)((g - SLOTS) / SX) & 1u, abort_flag)) {
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
                    tmem_st8(lane_base + (uint32_t)(b * SLOT_COLS + 32 * i), d);
                    tmem_st8(lane_base + (uint32_t)(b * SLOT_COLS + 32 * i + 8), d + 8);
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
            for (int p = 0; p < NT; p += 8) {
                uint32_t g0[8], g1[8], g2[8], g3[8];
                tmem_ld8(sa + 0 * NT + p, g0);
                tmem_ld8(sa + 1 * NT + p, g1);
                tmem_ld8(sa + 2 * NT + p, g2);
                tmem_ld8(sa + 3 * NT + p, g3);
                tmem_ld_wait();
#pragma unroll
                for (int j = 0; j < 8; ++j)
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

// Digit planes of the token operand as fp16 bits, planes[d][r][c] =
// byte_d(a + 0x80808080) - 128, and C (rows x n, leading dimension ldc)
// zeroed for the red.add reduction, in one launch: block (x, r) covers
// columns [1024 x, 1024 x + 1024) of row r, four consecutive columns a
// thread (16-byte loads and stores where the row allows).
__device__ __forceinline__ uint16_t digit_f16(uint32_t b, int d) {
    return __half_as_ushort(__int2half_rn((int)((b >> (8 * d)) & 0xffu) - 128));
}
__global__ void split_f16_zero_kernel(const uint32_t *a, int64_t lda, int64_t cols, uint16_t *planes, int64_t ldp,
                                      int64_t plane_stride, uint32_t *C, int64_t ldc, int64_t n, int vec_a,
                                      int vec_c) {
    const int64_t r = blockIdx.y;
    const int64_t c = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) * 4;
    if (c < cols) {
        const uint32_t *ar = a + r * lda + c;
        uint16_t *pr = planes + r * ldp + c;
        if (vec_a && c + 4 <= cols) {
            const uint4 v = *reinterpret_cast<const uint4 *>(ar);
            const uint32_t b[4] = {v.x + 0x80808080u, v.y + 0x80808080u, v.z + 0x80808080u, v.w + 0x80808080u};
#pragma unroll
            for (int d = 0; d < 4; ++d)
                *reinterpret_cast<uint2 *>(pr + d * plane_stride) =
                    make_uint2((uint32_t)digit_f16(b[0], d) | ((uint32_t)digit_f16(b[1], d) << 16),
                               (uint32_t)digit_f16(b[2], d) | ((uint32_t)digit_f16(b[3], d) << 16));
        } else {
            for (int k = 0; k < 4 && c + k < cols; ++k) {
                const uint32_t b = ar[k] + 0x80808080u;
#pragma unroll
                for (int d = 0; d < 4; ++d) pr[d * plane_stride + k] = digit_f16(b, d);
            }
        }
    }
    if (c < n) {
        uint32_t *cr = C + r * ldc + c;
        if (vec_c && c + 4 <= n) {
            *reinterpret_cast<uint4 *>(cr) = make_uint4(0u, 0u, 0u, 0u);
        } else {
            for (int k = 0; k < 4 && c + k < n; ++k) cr[k] = 0u;
        }
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
    {
        KernelSpan span("ring_gemm_tcw", st);
        ring_gemm_tcw_kernel<NT><<<(unsigned)grid, THREADS, C::SMEM, st>>>(tw, tx, args);
    }
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
    {
        KernelSpan span("split_f16_zero", st);
        // Planes rows are Kp (a multiple of 8) fp16 apart, so their 8-byte stores are aligned.
        const int vec_a = aligned16(A) && lda % 4 == 0;
        const int vec_c = aligned16(Cm) && ldc % 4 == 0;
        const int64_t wide = K > N ? K : N;
        split_f16_zero_kernel<<<dim3((unsigned)((wide + 1023) / 1024), (unsigned)M), 256, 0, st>>>(
            A, lda, K, Ap, Kp, M * Kp, Cm, ldc, N, vec_a, vec_c);
    }
    MOSAIC_TRY(launch_status());
    const int nt = M <= 32 ? 32 : M <= 48 ? 48 : 64;
    CUtensorMap tw, tx;
    if (!make_w_map(&tw, B, K, N, ldb) || !make_x_map(&tx, Ap, K, M, Kp, nt)) return MOSAIC_ERR_CUDA;
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 1)
        return MOSAIC_ERR_CUDA;
    const int64_t tiles = (N + WR - 1) / WR, nst = (K + KS - 1) / KS, nchunks = (nst + CHUNK - 1) / CHUNK;
    if (tiles * nchunks > (int64_t)INT32_MAX) return MOSAIC_ERR_SHAPE;
    const WArgs args{Cm, ldc, (int)M, (int)N, (int)K, (int)tiles, (int)nchunks};
    if (nt == 32) return launch_tcw<32>(tw, tx, args, sms, st);
    if (nt == 48) return launch_tcw<48>(tw, tx, args, sms, st);
    return launch_tcw<64>(tw, tx, args, sms, st);
}

}  // namespace mosaic
