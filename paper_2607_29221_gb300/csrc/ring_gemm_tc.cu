// Ring product over Z_{2^32} on the 5th-generation tensor cores (tcgen05).
//
// Sec. 5.2 ("Emulation approach") emulates each 32-bit ring MAC with 8-bit
// limb products on INT8 tensor cores.  The INT8 tensor path (tcgen05
// kind::i8) does not exist on sm_103a, so this kernel re-designs the limb
// products for kind::f16 with bf16 operands:
//   * every operand a is split into SIGNED base-2^8 digits
//     d_i = byte_i(a + 0x80808080) - 128 in [-128, 127], so that
//     a = sum_i d_i 2^(8i) mod 2^32; each digit is an exact bf16 value;
//   * a b mod 2^32 = sum_{i+j<=3} 2^(8(i+j)) d_i e_j: only the 10 digit pairs
//     with i + j <= 3 survive mod 2^32, grouped into 4 shift groups
//     s = i + j (1, 2, 3, 4 products);
//   * each group accumulates in fp32 in tensor memory (TMEM); a product of
//     two digits is at most 2^14 in magnitude, so a group that has summed at
//     most 1024 products is still an exact integer (|sum| <= 2^24).  Every
//     CHUNK * BK = 256 values of K (group 3 then holds 1024 products) the
//     epilogue warps drain groups 2 and 3, every 512 values of K groups 0 and
//     1, into int32 registers: acc += g_s << 8s mod 2^32 (drain_01 and
//     drain_23 below convert the fp32 sums exactly).
//
// Pipeline (128 x BN output tiles, 10 warps):
//   warp 0      TMA producer: per stage one 3-D box {32 K, rows, 4 planes}
//               for A and one for B (64-byte swizzle), mbarrier complete_tx
//   warp 1      TMEM allocation (512 columns) and the single-thread MMA issuer
//               (12 tcgen05.mma per stage: 8 of 128 x 2BN x 16, 4 of 128 x BN x 16)
//   warps 2..9  epilogue: tcgen05.ld 32x32b, exact fp32 -> int32, shift-add (each lane
//               quarter of TMEM twice, half of the columns each)
// Every wait is bounded (about 2 s of %globaltimer); on expiry the kernel
// raises a device error word, stops issuing work, waits (bounded) for its
// own copies and products in flight, frees TMEM and returns.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "async_copy.cuh"
#include "mosaic_internal.cuh"

namespace mosaic {

__device__ uint32_t g_tc_error = 0;

namespace {

constexpr int BM = 128;
constexpr int BK = 32;          // bf16 K elements per stage = one 64-byte swizzled row
constexpr int STAGES = 3;
constexpr int CHUNK = 8;        // stages between drains: 256 K
constexpr uint32_t TMEM_COLS = 512;
constexpr int THREADS = 320;   // warp 0 TMA, warp 1 MMA, warps 2..9 epilogue
constexpr int EPI_WARPS = 8;
// Write-out slices: each epilogue warp moves its 32 rows 16 columns at a time
// through a [32][EPI_PITCH] block of shared memory (pitch 20 words: the
// row-per-lane 16-byte writes and the 8-rows-per-access 16-byte reads are
// both conflict-free).
constexpr int EPI_PITCH = 20;
constexpr int EPI_BYTES = EPI_WARPS * 32 * EPI_PITCH * 4;

// Drain conversions.  The fp32 group sums are integers with |x| <= 2^24 and
// the F2I unit converts 16 values per clock per SM while the tensor pipe
// idles, so each pair of groups is folded into ONE exact fp32 value first
// (FMA pipe).  kM = 1.5 * 2^23: for an integer y with |y| <= 2^22 the bits of
// y + kM are bits(kM) + y, so fma(x, 2^-8, kM) - kM is h = round(x / 2^8)
// exactly and fma(h, -2^8, x) = x - 2^8 h is exact (|x - 2^8 h| <= 2^7).
constexpr float kM = 12582912.0f;

// Groups 0 and 1 (|x0| <= 2^23, |x1| <= 2^24 after 512 K): with h =
// round(x1 / 2^8), x0 + 2^8 x1 = s + 2^16 h where s = x0 + 2^8 (x1 - 2^8 h)
// is exact (|s| < 2^24) and goes through F2I; h << 16 is the bits of
// x1 / 2^8 + kM shifted by 16, since bits(kM) << 16 = 0 mod 2^32.
__device__ __forceinline__ void drain_01(uint32_t *acc, const uint32_t *v0, const uint32_t *v1) {
#pragma unroll
    for (int cc = 0; cc < 32; ++cc) {
        const float x0 = __uint_as_float(v0[cc]), x1 = __uint_as_float(v1[cc]);
        const float t = __fmaf_rn(x1, 0.00390625f, kM);
        const float lo = __fmaf_rn(__fsub_rn(t, kM), -256.0f, x1);
        const float s = __fmaf_rn(lo, 256.0f, x0);
        acc[cc] += (uint32_t)__float2int_rn(s) + (__float_as_uint(t) << 16);
    }
}

// Groups 2 and 3 (|x2| <= 3 * 2^22, |x3| <= 2^24 after 256 K): (x2 << 16) +
// (x3 << 24) = s << 16 mod 2^32 with s = x2 + 2^8 (x3 - 2^8 round(x3 / 2^8)),
// exact (|s| < 2^24).
__device__ __forceinline__ void drain_23(uint32_t *acc, const uint32_t *v0, const uint32_t *v1) {
#pragma unroll
    for (int cc = 0; cc < 32; ++cc) {
        const float x3 = __uint_as_float(v1[cc]);
        const float lo3 = __fmaf_rn(__fsub_rn(__fmaf_rn(x3, 0.00390625f, kM), kM), -256.0f, x3);
        const float s = __fmaf_rn(lo3, 256.0f, __uint_as_float(v0[cc]));
        acc[cc] += (uint32_t)__float2int_rn(s) << 16;
    }
}

template <int BN>
struct Cfg {
    static constexpr int A_PLANE = BM * BK * 2;
    static constexpr int B_PLANE = BN * BK * 2;
    static constexpr int A_BYTES = 4 * A_PLANE;
    static constexpr int B_BYTES = 4 * B_PLANE;
    static constexpr int STAGE = A_BYTES + B_BYTES;
    static constexpr int SMEM = STAGES * STAGE + 1024 + 256 + EPI_BYTES;
    // kind::f16 instruction descriptors: D f32, A/B bf16, K-major, N >> 3, M >> 4;
    // IDESC2 has N = 2 BN (two consecutive B digit planes as one operand).
    static constexpr uint32_t IDESC = (1u << 4) | (1u << 7) | (1u << 10) |
                                      ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);
    static constexpr uint32_t IDESC2 = (1u << 4) | (1u << 7) | (1u << 10) |
                                       ((uint32_t)((2 * BN) >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);
    static_assert(2 * BN <= 256, "paired B planes must fit one MMA");
    static_assert(4 * BN <= (int)TMEM_COLS, "four shift groups must fit in TMEM");
    static_assert(BN % 32 == 0 && BN >= 32 && BN <= 128, "");
};

struct TcArgs {
    uint32_t *C;
    int64_t ldc;
    const uint32_t *Cin;   // plain mode only (stream-K mode prepares C instead)
    int64_t ldcin;
    int sgn;
    int M, N, K;
    int tiles_m, tiles_n;
    int split;             // 0: one CTA per tile; 1: stream-K over (tile, chunk) units
    int dp_tiles;          // split mode: tiles [0, dp_tiles) run whole, one per CTA
    // Columns [N1, N) go to a second output: C2[i][j - N1] (= Cin2 + ...).
    // N1 is a multiple of BN, so no tile straddles the two; N1 = N: one output.
    int N1;
    uint32_t *C2;
    int64_t ldc2;
    const uint32_t *Cin2;
    int64_t ldcin2;
    // Plain mode, first output: C = Cin - Csub + sgn * A B^T (Csub nullable).
    const uint32_t *Csub;
    int64_t ldcsub;
};

__device__ __forceinline__ void raise_abort(volatile int *abort_flag) {
    *abort_flag = 1;
    atomicExch(&g_tc_error, 1u);
}
__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// Shared-memory matrix descriptor: K-major, 64-byte swizzle; rows of 64 B,
// 8-row core groups 512 B apart (stride byte offset); descriptor version 1.
__device__ __forceinline__ uint64_t sdesc_sw64(uint32_t saddr) {
    uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);
    d |= (uint64_t)1 << 16;               // leading byte offset (unused for swizzled K-major)
    d |= (uint64_t)(512 >> 4) << 32;      // stride byte offset
    d |= (uint64_t)1 << 46;               // version
    d |= (uint64_t)4 << 61;               // SWIZZLE_64B
    return d;
}
__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                          uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
__device__ __forceinline__ void umma_commit(uint64_t *bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                     smem_u32(bar))
                 : "memory");
}
// 32 columns of TMEM for the warp's 32 lanes; the caller waits (tmem_wait).
__device__ __forceinline__ void tmem_ld32_nowait(uint32_t taddr, uint32_t *v) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
        "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),
          "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]),
          "=r"(v[14]), "=r"(v[15]), "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]),
          "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]), "=r"(v[25]),
          "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
        : "r"(taddr));
}
__device__ __forceinline__ void tmem_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

template <int BN>
__global__ void __launch_bounds__(THREADS, 1)
    ring_gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                        TcArgs a) {
    using C = Cfg<BN>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                ~static_cast<uintptr_t>(1023));
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + STAGES * C::STAGE);
    uint64_t *empty = full + STAGES;
    uint64_t *acc_full = empty + STAGES;
    uint64_t *acc_empty = acc_full + 1;
    uint64_t *drain = acc_empty + 1;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(drain + 1);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);
    const uint32_t epi_base = smem_u32(smem + STAGES * C::STAGE + 256);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nk = (a.K + BK - 1) / BK;
    const int nchunks = (nk + CHUNK - 1) / CHUNK;
    // Work of this CTA: units of (output tile, 256-wide K chunk), numbered
    // tile-major; tile t covers rows (t % tiles_m) * BM and columns
    // (t / tiles_m) * BN, so CTAs running side by side share B tiles.
    // Segment 0: whole tiles blockIdx.x + w * gridDim.x for every whole wave w
    // (dp_tiles = waves * gridDim.x; CTAs in step read the same B tiles at the
    // same K); segment 1: this CTA's even share of the remaining tiles' units
    // (stream-K).  Without split, segment 0 is every tile blockIdx.x + w *
    // gridDim.x (one tile when the grid covers them all).
    // Unit counts fit in 32 bits (tiles * nchunks < 2^31, checked by the host).
    int n0 = 0, s1b = 0, n1 = 0;
    const int tiles = a.tiles_m * a.tiles_n;
    if (a.split) {
        const int dp_units = a.dp_tiles * nchunks;
        n0 = (a.dp_tiles / (int)gridDim.x) * nchunks;
        const int64_t U = (int64_t)tiles * nchunks - dp_units;
        s1b = dp_units + (int)(U * blockIdx.x / gridDim.x);
        n1 = dp_units + (int)(U * (blockIdx.x + 1) / gridDim.x) - s1b;
    } else {
        n0 = ((tiles - (int)blockIdx.x + (int)gridDim.x - 1) / (int)gridDim.x) * nchunks;
    }
    const int n_units = n0 + n1;
    // Shift groups 0 and 1 gather 1 and 2 digit products per K value, so they
    // stay exact (|sum| <= 2^24) over two 256-wide chunks and are drained every
    // second chunk of a tile (and at the end of the tile or of a segment);
    // groups 2 and 3 are drained after every chunk.  `since` counts the chunks
    // accumulated in groups 0 and 1, including the current one.
    auto drains01 = [&](int k, int c, int since) {
        return since >= 2 || c == nchunks - 1 || k == n0 - 1 || k == n_units - 1;
    };
    // Walks this CTA's units in order without divisions: (tile, chunk c) of
    // unit k (segment 0: tiles blockIdx.x + w * gridDim.x; segment 1: units
    // s1b, s1b + 1, ...).
    struct UnitWalk {
        int k, tile, c;
    };
    const int s1_tile = s1b / nchunks;
    const int s1_c = (int)(s1b - s1_tile * nchunks);
    auto walk_init = [&](UnitWalk &w) {
        w.k = 0;
        w.tile = n0 > 0 ? (int)blockIdx.x : s1_tile;
        w.c = n0 > 0 ? 0 : s1_c;
    };
    auto walk_next = [&](UnitWalk &w) {
        if (++w.k == n0) {
            w.tile = s1_tile;
            w.c = s1_c;
        } else if (++w.c == nchunks) {
            w.c = 0;
            w.tile += w.k < n0 ? (int)gridDim.x : 1;
        }
    };

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(acc_full, 1);
        mbar_init(acc_empty, EPI_WARPS);
        mbar_init(drain, 1);
        *abort_flag = 0;
        mbar_init_fence();
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_u32(tmem_slot)),
                     "r"(TMEM_COLS)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        if (lane == 0) {
            int slot = 0;
            int s = 0;          // slot % STAGES
            uint32_t ph = 0;    // parity of the empty phase awaited for slot s (from the second round on)
            UnitWalk w;
            walk_init(w);
            for (; w.k < n_units && !*abort_flag; walk_next(w)) {
                const int m0 = (int)(w.tile % a.tiles_m) * BM, n0 = (int)(w.tile / a.tiles_m) * BN;
                const int c = w.c;
                const int ks1 = (c + 1) * CHUNK < nk ? (c + 1) * CHUNK : nk;
                bool ok = true;
                for (int ks = c * CHUNK; ks < ks1; ++ks, ++slot) {
                    if (slot >= STAGES && !mbar_wait(&empty[s], ph, abort_flag)) {
                        raise_abort(abort_flag);
                        ok = false;
                        break;
                    }
                    uint8_t *st = smem + s * C::STAGE;
                    mbar_expect_tx(&full[s], C::STAGE);
                    tma_load_3d(st, &tmA, &full[s], ks * BK, m0, 0);
                    tma_load_3d(st + C::A_BYTES, &tmB, &full[s], ks * BK, n0, 0);
                    if (++s == STAGES) {
                        s = 0;
                        if (slot >= STAGES) ph ^= 1u;   // slots [STAGES, 2 STAGES) wait parity 0, and so on
                    }
                }
                if (!ok) break;
            }
            if (*abort_flag) {
                // Let the copies this thread started land before the CTA exits.
                for (int q = slot > STAGES ? slot - STAGES : 0; q < slot; ++q) {
                    const unsigned long long t0 = gtime();
                    while (!mbar_try(&full[q % STAGES], (uint32_t)(q / STAGES) & 1) && gtime() - t0 < kWaitNs) {
                    }
                }
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            bool issued_any = false;
            uint32_t chunk_count = 0;
            int s = 0;          // shared-memory slot of the next stage
            uint32_t ph = 0;    // parity of its full barrier
            int since01 = 0;
            // Descriptors differ only in the start-address field (address >> 4).
            const uint64_t desc0 = sdesc_sw64(smem_u32(smem));
            constexpr uint64_t AP = C::A_PLANE >> 4, BP = C::B_PLANE >> 4;
            UnitWalk w;
            walk_init(w);
            for (; w.k < n_units && !*abort_flag; walk_next(w)) {
                const int k = w.k;
                const int c = w.c;
                const int ks0 = c * CHUNK, ks1 = (c + 1) * CHUNK < nk ? (c + 1) * CHUNK : nk;
                const uint32_t keep01 = since01 > 0 ? 1u : 0u;   // groups 0, 1 carry on
                if (drains01(k, c, ++since01)) since01 = 0;
                if (chunk_count > 0 && !mbar_wait(acc_empty, (uint32_t)(chunk_count - 1) & 1, abort_flag)) {
                    raise_abort(abort_flag);
                    break;
                }
                bool ok = true;
                for (int ks = ks0; ks < ks1; ++ks) {
                    if (!mbar_wait(&full[s], ph, abort_flag)) {
                        raise_abort(abort_flag);
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint64_t da = desc0 + (uint64_t)((s * C::STAGE) >> 4);
                    const uint64_t db = da + (uint64_t)(C::A_BYTES >> 4);
                    const bool first = ks == ks0;
                    // The 10 digit products d_i e_j (i + j <= 3) as 6 MMAs: B planes
                    // j and j + 1 are adjacent in shared memory and the shift
                    // groups i + j and i + j + 1 adjacent in TMEM, so one N = 2 BN
                    // product covers both.  A plane 0 goes first: its two paired
                    // products start all four groups of a chunk.
#pragma unroll
                    for (int kk = 0; kk < BK / 16; ++kk) {
                        const uint32_t z = (first && kk == 0) ? 0u : 1u;
                        const uint32_t z01 = (first && kk == 0) ? keep01 : 1u;
                        const uint64_t a0 = da + 2 * kk, b0 = db + 2 * kk;
                        umma_bf16(tmem + 0 * BN, a0, b0, C::IDESC2, z01);             // d0 e0, d0 e1
                        umma_bf16(tmem + 2 * BN, a0, b0 + 2 * BP, C::IDESC2, z);      // d0 e2, d0 e3
                        umma_bf16(tmem + 1 * BN, a0 + AP, b0, C::IDESC2, 1u);         // d1 e0, d1 e1
                        umma_bf16(tmem + 3 * BN, a0 + AP, b0 + 2 * BP, C::IDESC, 1u); // d1 e2
                        umma_bf16(tmem + 2 * BN, a0 + 2 * AP, b0, C::IDESC2, 1u);     // d2 e0, d2 e1
                        umma_bf16(tmem + 3 * BN, a0 + 3 * AP, b0, C::IDESC, 1u);      // d3 e0
                    }
                    issued_any = true;
                    umma_commit(&empty[s]);
                    if (++s == STAGES) {
                        s = 0;
                        ph ^= 1u;
                    }
                }
                if (!ok) break;
                umma_commit(acc_full);
                ++chunk_count;
            }
            if (*abort_flag && issued_any) {
                // Products in flight still read shared memory and write TMEM.
                umma_commit(drain);
                const unsigned long long t0 = gtime();
                while (!mbar_try(drain, 0) && gtime() - t0 < kWaitNs) {
                }
            }
        }
    } else {
        // Epilogue: warp w reads TMEM lanes 32 (w % 4) .. 32 (w % 4) + 31 and
        // columns [h HB, (h + 1) HB) of each group, h = (w - 2) / 4.
        constexpr int HB = BN / 2;
        const int q = warp & 3;
        const int h = (warp - 2) >> 2;
        const int row = q * 32 + lane;
        const uint32_t lane_addr = tmem + ((uint32_t)(q * 32) << 16) + h * HB;
        uint32_t acc[HB];
#pragma unroll
        for (int c = 0; c < HB; ++c) acc[c] = 0u;
        uint32_t chunk_count = 0;
        int since01 = 0;
        UnitWalk wk;
        walk_init(wk);
        for (; wk.k < n_units; walk_next(wk)) {
            const int k = wk.k, tile = wk.tile;
            const int c = wk.c;
            if (!mbar_wait(acc_full, (uint32_t)chunk_count & 1, abort_flag)) {
                raise_abort(abort_flag);
                break;
            }
            tc_fence_after();
            const bool d01 = drains01(k, c, ++since01);
            if (d01) since01 = 0;
            // Two groups are loaded before one wait.
#pragma unroll
            for (int c0 = 0; c0 < HB; c0 += 32) {
                uint32_t v0[32], v1[32];
                if (d01) {
                    tmem_ld32_nowait(lane_addr + 0 * BN + c0, v0);
                    tmem_ld32_nowait(lane_addr + 1 * BN + c0, v1);
                    tmem_wait();
                    drain_01(acc + c0, v0, v1);
                }
                tmem_ld32_nowait(lane_addr + 2 * BN + c0, v0);
                tmem_ld32_nowait(lane_addr + 3 * BN + c0, v1);
                tmem_wait();
                drain_23(acc + c0, v0, v1);
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(acc_empty);
            ++chunk_count;

            // Short products (no stream-K): one chunk before the tile is written,
            // pull this lane's row of the added / subtracted inputs into L2, so
            // that the write-out reads them from L2 instead of waiting on DRAM.
            if (!a.split && nchunks >= 2 && c == nchunks - 2) {
                const int tm0 = (int)(tile % a.tiles_m) * BM, ttn0 = (int)(tile / a.tiles_m) * BN;
                const bool sec = ttn0 >= a.N1;
                const int gr = tm0 + row;
                const int col = ttn0 - (sec ? a.N1 : 0) + h * HB;
                const uint32_t *pin = sec ? a.Cin2 : a.Cin;
                const int64_t ldp = sec ? a.ldcin2 : a.ldcin;
                const uint32_t *psub = sec ? nullptr : a.Csub;
                // Whole 64-column pieces only, so that every prefetched byte lies in the row.
                if (gr < a.M && col + HB <= (sec ? a.N - a.N1 : a.N1)) {
                    if (pin) {
                        const char *r0 = reinterpret_cast<const char *>(pin + (int64_t)gr * ldp + col);
                        asm volatile("prefetch.global.L2 [%0];" ::"l"(r0));
                        asm volatile("prefetch.global.L2 [%0];" ::"l"(r0 + 128));
                        asm volatile("prefetch.global.L2 [%0];" ::"l"(r0 + 4 * HB - 4));
                    }
                    if (psub) {
                        const char *r0 = reinterpret_cast<const char *>(psub + (int64_t)gr * a.ldcsub + col);
                        asm volatile("prefetch.global.L2 [%0];" ::"l"(r0));
                        asm volatile("prefetch.global.L2 [%0];" ::"l"(r0 + 128));
                        asm volatile("prefetch.global.L2 [%0];" ::"l"(r0 + 4 * HB - 4));
                    }
                }
            }

            if (c != nchunks - 1 && k != n0 - 1 && k != n_units - 1) continue;
            // End of this CTA's segment of the tile: write it out.
            const bool whole = k < n0 || ((s1b <= tile * nchunks) && (c == nchunks - 1));
            const int m0 = (int)(tile % a.tiles_m) * BM;
            const int tn0 = (int)(tile / a.tiles_m) * BN;
            const bool second = tn0 >= a.N1;
            const int n0 = tn0 - (second ? a.N1 : 0) + h * HB;
            const int nout = second ? a.N - a.N1 : a.N1;
            const int gm = m0 + row;
            uint32_t *const cbase = second ? a.C2 : a.C;
            const int64_t ldc_o = second ? a.ldc2 : a.ldc;
            const uint32_t *const cin0 = second ? a.Cin2 : a.Cin;
            const int64_t ldcin_o = second ? a.ldcin2 : a.ldcin;
            const uint32_t *const sub0 = second ? nullptr : a.Csub;
            if (a.sgn < 0) {
#pragma unroll
                for (int cc = 0; cc < HB; ++cc) acc[cc] = 0u - acc[cc];
            }
            // Other CTAs add into a split tile too: exact and order-free in Z_{2^32}.
            const bool atomic = a.split && !whole;
            // Plain mode: C = Cin - Csub + acc.  Stream-K mode, whole tile: C (prepared) += acc.
            const bool vecw = !atomic && (n0 + HB <= nout) && ((ldc_o & 3) == 0) &&
                              ((reinterpret_cast<uintptr_t>(cbase) & 15u) == 0) &&
                              (a.split || !cin0 || (((ldcin_o & 3) == 0) && ((reinterpret_cast<uintptr_t>(cin0) & 15u) == 0))) &&
                              (!sub0 || (((a.ldcsub & 3) == 0) && ((reinterpret_cast<uintptr_t>(sub0) & 15u) == 0)));
            if (vecw) {
                // Coalesced write-out: 16 columns of the warp's 32 rows go to its
                // slice block (one row per lane) and come back as 8 rows x 64
                // bytes per access, so C, Cin and Csub move in half lines
                // instead of 16 bytes of 32 rows per access.
                const uint32_t wb = epi_base + (uint32_t)((warp - 2) * 32 * EPI_PITCH * 4);
                const int pc = (lane >> 3) * 4;
#pragma unroll
                for (int s0 = 0; s0 < HB; s0 += 16) {
#pragma unroll
                    for (int cc = 0; cc < 16; cc += 4)
                        asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(
                                         wb + 4u * (uint32_t)(lane * EPI_PITCH + cc)),
                                     "r"(acc[s0 + cc]), "r"(acc[s0 + cc + 1]), "r"(acc[s0 + cc + 2]), "r"(acc[s0 + cc + 3])
                                     : "memory");
                    __syncwarp();
                    uint4 v[4], ib[4], sb[4];
#pragma unroll
                    for (int it = 0; it < 4; ++it) {
                        const int rl = it * 8 + (lane & 7);
                        const int gr = m0 + q * 32 + rl;
                        const int64_t col = n0 + s0 + pc;
                        asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                                     : "=r"(v[it].x), "=r"(v[it].y), "=r"(v[it].z), "=r"(v[it].w)
                                     : "r"(wb + 4u * (uint32_t)(rl * EPI_PITCH + pc))
                                     : "memory");
                        const uint32_t *bp = a.split ? cbase + (int64_t)gr * ldc_o + col
                                                     : (cin0 ? cin0 + (int64_t)gr * ldcin_o + col : nullptr);
                        const uint32_t *sp = sub0 ? sub0 + (int64_t)gr * a.ldcsub + col : nullptr;
                        ib[it] = (gr < a.M && bp) ? *reinterpret_cast<const uint4 *>(bp) : make_uint4(0, 0, 0, 0);
                        sb[it] = (gr < a.M && sp) ? *reinterpret_cast<const uint4 *>(sp) : make_uint4(0, 0, 0, 0);
                    }
                    __syncwarp();
#pragma unroll
                    for (int it = 0; it < 4; ++it) {
                        const int rl = it * 8 + (lane & 7);
                        const int gr = m0 + q * 32 + rl;
                        if (gr < a.M)
                            *reinterpret_cast<uint4 *>(cbase + (int64_t)gr * ldc_o + n0 + s0 + pc) =
                                make_uint4(v[it].x + ib[it].x - sb[it].x, v[it].y + ib[it].y - sb[it].y,
                                           v[it].z + ib[it].z - sb[it].z, v[it].w + ib[it].w - sb[it].w);
                    }
                }
            } else if (gm < a.M) {
                uint32_t *crow = cbase + (int64_t)gm * ldc_o;
                const uint32_t *cin = cin0 ? cin0 + (int64_t)gm * ldcin_o : nullptr;
                const uint32_t *sub = sub0 ? sub0 + (int64_t)gm * a.ldcsub : nullptr;
                if (atomic) {
#pragma unroll
                    for (int cc = 0; cc < HB; ++cc)
                        if (n0 + cc < nout) atomicAdd(crow + n0 + cc, acc[cc]);
                } else {
                    const uint32_t *base = a.split ? crow : cin;
#pragma unroll
                    for (int cc = 0; cc < HB; ++cc) {
                        const int gn = n0 + cc;
                        if (gn < nout) crow[gn] = acc[cc] + (base ? base[gn] : 0u) - (sub ? sub[gn] : 0u);
                    }
                }
            }
#pragma unroll
            for (int cc = 0; cc < HB; ++cc) acc[cc] = 0u;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TMEM_COLS)
                     : "memory");
    }
}

// 3-D map over bf16 digit planes: {K, rows, 4 planes}, box {BK, box_rows, 4}.
bool make_plane_map(CUtensorMap *map, const uint16_t *base, int64_t K, int64_t rows, int64_t ldp,
                    int64_t plane_stride, int box_rows) {
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[3] = {(cuuint64_t)K, (cuuint64_t)rows, 4};
    cuuint64_t strides[2] = {(cuuint64_t)ldp * 2, (cuuint64_t)plane_stride * 2};
    cuuint32_t box[3] = {(cuuint32_t)BK, (cuuint32_t)box_rows, 4};
    cuuint32_t estr[3] = {1, 1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<uint16_t *>(base), dims, strides, box,
              estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// C (and C2 for columns >= N1) = Cin + sgn * A B^T from digit planes.
struct TcOut {
    uint32_t *C;
    int64_t ldc;
    const uint32_t *Cin;
    int64_t ldcin;
    int64_t cols;
    const uint32_t *Csub = nullptr;   // first output only, plain mode
    int64_t ldcsub = 0;
};

// Prepares a stream-K output: its tiles are summed with atomic adds, so it
// starts as Cin (or 0).
cudaError_t prepare_split(const TcOut &o, int64_t M, cudaStream_t st) {
    if (o.cols == 0) return cudaSuccess;
    if (!o.Cin) return cudaMemset2DAsync(o.C, (size_t)o.ldc * 4, 0, (size_t)o.cols * 4, (size_t)M, st);
    if (o.Cin != o.C)
        return cudaMemcpy2DAsync(o.C, (size_t)o.ldc * 4, o.Cin, (size_t)o.ldcin * 4, (size_t)o.cols * 4,
                                 (size_t)M, cudaMemcpyDeviceToDevice, st);
    return cudaSuccess;
}

template <int BN>
mosaic_status launch_tc(const uint16_t *Ap, int64_t ldpa, int64_t a_plane, const uint16_t *Bp,
                        int64_t ldpb, int64_t b_plane, const TcOut &o1, const TcOut &o2, int sgn,
                        int64_t M, int64_t K, cudaStream_t st) {
    const int64_t N = o1.cols + o2.cols;
    uint32_t *Cm = o1.C;
    const uint32_t *Cin = o1.Cin;
    const int64_t ldc = o1.ldc, ldcin = o1.ldcin;
    using C = Cfg<BN>;
    CUtensorMap ta, tb;
    if (!make_plane_map(&ta, Ap, K, M, ldpa, a_plane, BM) || !make_plane_map(&tb, Bp, K, N, ldpb, b_plane, BN))
        return MOSAIC_ERR_CUDA;
    static std::atomic<unsigned long long> attr_set{0};   // one bit per device ordinal
    int dev = 0;
    if (!ensure_smem_limit(attr_set, ring_gemm_tc_kernel<BN>, C::SMEM, &dev)) return MOSAIC_ERR_CUDA;
    const int64_t tiles_m = (M + BM - 1) / BM, tiles_n = (N + BN - 1) / BN, tiles = tiles_m * tiles_n;
    const int64_t nk = (K + BK - 1) / BK, nchunks = (nk + CHUNK - 1) / CHUNK;
    if (tiles * nchunks > (int64_t)INT32_MAX) return MOSAIC_ERR_SHAPE;   // 32-bit unit numbers
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 1)
        return MOSAIC_ERR_CUDA;
    // Whole tiles on a persistent grid (at most one CTA per SM) unless the
    // last wave would leave more than 10% of the SMs idle; then the grid also
    // shares the remaining tiles' (tile, chunk) units evenly.  Short products
    // (fewer than 8 chunks, K < 2048) keep whole tiles only: there the
    // preparation of C and the split-tile atomics cost more than the idle SMs.
    const int64_t waves = (tiles + sms - 1) / sms;
    // A subtracted input is read in plain mode only (stream-K prepares C from Cin alone).
    const bool split = !o1.Csub && nchunks >= 8 && (double)tiles / (double)(waves * sms) < 0.9;
    TcArgs args{Cm, ldc, Cin, ldcin, sgn, (int)M, (int)N, (int)K, (int)tiles_m, (int)tiles_n, split ? 1 : 0,
                0, (int)o1.cols, o2.C, o2.ldc, o2.Cin, o2.ldcin, o1.Csub, o1.ldcsub};
    int64_t grid = tiles < sms ? tiles : sms;
    if (split) {
        if (prepare_split(o1, M, st) != cudaSuccess || prepare_split(o2, M, st) != cudaSuccess)
            return MOSAIC_ERR_CUDA;
        args.Cin = nullptr;
        args.Cin2 = nullptr;
        grid = tiles * nchunks < sms ? tiles * nchunks : sms;
        args.dp_tiles = (int)((tiles / grid) * grid);   // whole waves run as whole tiles
    }
    if (grid > 0x7fffffff) return MOSAIC_ERR_SHAPE;
    {
        KernelSpan span("ring_gemm_tc", st);
        ring_gemm_tc_kernel<BN><<<(unsigned)grid, THREADS, C::SMEM, st>>>(ta, tb, args);
    }
    return launch_status();
}

}  // namespace

bool tc_available() {
    int dev = 0, major = 0, minor = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return false;
    if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess) return false;
    if (cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess) return false;
    return major == 10 && minor == 3 && encode_fn() != nullptr;
}


mosaic_status ring_gemm_tc_planes(const uint16_t *Ap, int64_t ldpa, int64_t a_plane, const uint16_t *Bp,
                                  int64_t ldpb, int64_t b_plane, uint32_t *Cm, int64_t ldc,
                                  const uint32_t *Cin, int64_t ldcin, int sgn, int64_t M, int64_t N,
                                  int64_t K, cudaStream_t st) {
    if (M == 0 || N == 0) return MOSAIC_OK;
    if (M > (int64_t)INT32_MAX || N > (int64_t)INT32_MAX) return MOSAIC_ERR_SHAPE;
    if (K == 0) {
        // Empty product: C = Cin (or 0).
        cudaError_t e = !Cin ? cudaMemset2DAsync(Cm, (size_t)ldc * 4, 0, (size_t)N * 4, (size_t)M, st)
                       : Cin == Cm ? cudaSuccess
                                   : cudaMemcpy2DAsync(Cm, (size_t)ldc * 4, Cin, (size_t)ldcin * 4,
                                                       (size_t)N * 4, (size_t)M, cudaMemcpyDeviceToDevice, st);
        return e == cudaSuccess ? MOSAIC_OK : MOSAIC_ERR_CUDA;
    }
    const TcOut o1{Cm, ldc, Cin, ldcin, N}, none{nullptr, 0, nullptr, 0, 0};
    return launch_tc<128>(Ap, ldpa, a_plane, Bp, ldpb, b_plane, o1, none, sgn, M, K, st);
}

mosaic_status ring_gemm_tc_planes2(const uint16_t *Ap, int64_t ldpa, int64_t a_plane, const uint16_t *Bp,
                                   int64_t ldpb, int64_t b_plane, uint32_t *C1, int64_t ldc1,
                                   const uint32_t *Cin1, int64_t ldcin1, int64_t N1, uint32_t *C2, int64_t ldc2,
                                   const uint32_t *Cin2, int64_t ldcin2, int64_t N2, int64_t M, int64_t K,
                                   cudaStream_t st) {
    if (M == 0 || N1 + N2 == 0) return MOSAIC_OK;
    if (M > (int64_t)INT32_MAX || N1 + N2 > (int64_t)INT32_MAX || N1 % 128 != 0 || K == 0)
        return MOSAIC_ERR_SHAPE;
    const TcOut o1{C1, ldc1, Cin1, ldcin1, N1}, o2{C2, ldc2, Cin2, ldcin2, N2};
    return launch_tc<128>(Ap, ldpa, a_plane, Bp, ldpb, b_plane, o1, o2, 1, M, K, st);
}


mosaic_status ring_gemm_tc_planes_diff(const uint16_t *Ap, int64_t ldpa, int64_t a_plane, const uint16_t *Bp,
                                       int64_t ldpb, int64_t b_plane, uint32_t *Cm, int64_t ldc,
                                       const uint32_t *Cin, int64_t ldcin, const uint32_t *Csub, int64_t ldcsub,
                                       int sgn, int64_t M, int64_t N, int64_t K, cudaStream_t st) {
    if (M == 0 || N == 0) return MOSAIC_OK;
    if (M > (int64_t)INT32_MAX || N > (int64_t)INT32_MAX || K == 0 || !Cin || !Csub) return MOSAIC_ERR_SHAPE;
    TcOut o1{Cm, ldc, Cin, ldcin, N};
    o1.Csub = Csub;
    o1.ldcsub = ldcsub;
    const TcOut none{nullptr, 0, nullptr, 0, 0};
    return launch_tc<128>(Ap, ldpa, a_plane, Bp, ldpb, b_plane, o1, none, sgn, M, K, st);
}

mosaic_status device_status(cudaStream_t st) {
    if (cudaStreamSynchronize(st) != cudaSuccess) return MOSAIC_ERR_CUDA;
    uint32_t v = 0, zero = 0;
    if (cudaMemcpyFromSymbol(&v, g_tc_error, sizeof v) != cudaSuccess) return MOSAIC_ERR_CUDA;
    if (v) {
        cudaMemcpyToSymbol(g_tc_error, &zero, sizeof zero);
        return MOSAIC_ERR_TIMEOUT;
    }
    return MOSAIC_OK;
}

}  // namespace mosaic
