// Random Hadamard rotation R = H D fused with per-row quantisation and the
// mask-add (Sec. 4 "Random Hadamard rotation"; Pi_Sec-Linear box, Init W
// steps 1-2 and Online step 1; Approx-MatMul Online step 2).
//
// One row of n_pad = E * T fp32 values is held in registers by T threads
// (E consecutive elements each).  The butterfly stages run in the order
// h = 1, 2, ..., n_pad / 2 -- the same order as the plain radix-2 FWHT --
// so every output is rounded exactly like the textbook transform:
//   h <  E        inside a thread's registers,
//   E <= h < 32E  across lanes with warp shuffles,
//   h >= 32E      after one transpose through shared memory, again in
//                 registers (each thread then holds E / WN elements of each of
//                 the WN warp-sized segments).
// HBM traffic per row: read n floats (+ n mask words), write n_pad words
// (+ 4 bf16 digit planes when requested).
#include <cuda_bf16.h>
#include <math.h>

#include <atomic>

#include "async_copy.cuh"
#include "mosaic_internal.cuh"

namespace mosaic {

// Set when a streamed rotation gave up waiting for a row copy.
__device__ uint32_t g_fwht_error = 0;

namespace {

struct FwhtArgs {
    const float *x;
    int64_t ldx;
    int64_t rows;
    int64_t n;
    int64_t n_pad;
    const uint32_t *signs;
    int rotate;
    int mode;          // 0: write y (fp32); 1: encode
    float inv_sqrt;    // fl32(1 / sqrt(n_pad))
    float *y;
    int32_t qmax;
    const uint32_t *mask;
    int64_t ldm;
    uint32_t *out;
    int64_t ldo;
    float *scale;
    uint16_t *planes;  // [4][rows][n_pad]
    int vec_x;         // x rows 16-byte aligned
    int64_t ldy;       // mode 0: y row stride
    int split;         // rows are the halves of rows twice as long (the 65536-wide path)
};

__device__ __forceinline__ int pad_idx(int i) { return i + (i >> 5); }

// Signed base-2^8 digit i of a (b = a + 0x80808080; digit = byte_i(b) - 128)
// as an fp32 value, exactly: the byte is placed in the low mantissa bits of
// 2^23 (the float 2^23 + byte) and 2^23 + 128 is subtracted.  A digit in
// [-128, 127] has at most 8 significant bits, so its fp32 bits shifted right
// by 16 are its exact bf16 bits.
__device__ __forceinline__ uint32_t digit_f32_bits(uint32_t b, int i) {
    const uint32_t f = __byte_perm(b, 0x4B000000u, 0x7650u | (uint32_t)i);
    return __float_as_uint(__fadd_rn(__uint_as_float(f), -8388736.0f));
}
// bf16 bits of digit i of two ring elements, packed (first in the low half).
__device__ __forceinline__ uint32_t digit_pair_bf16(uint32_t b0, uint32_t b1, int i) {
    return __byte_perm(digit_f32_bits(b0, i), digit_f32_bits(b1, i), 0x7632u);
}

template <int CNT>
__device__ __forceinline__ void store_f32(float *p, const float *v) {
    if constexpr (CNT % 4 == 0) {
#pragma unroll
        for (int q = 0; q < CNT; q += 4) *reinterpret_cast<float4 *>(p + q) = make_float4(v[q], v[q + 1], v[q + 2], v[q + 3]);
    } else if constexpr (CNT == 2) {
        *reinterpret_cast<float2 *>(p) = make_float2(v[0], v[1]);
    } else {
#pragma unroll
        for (int q = 0; q < CNT; q++) p[q] = v[q];
    }
}

template <int CNT>
__device__ __forceinline__ void store_u32(uint32_t *p, const uint32_t *v) {
    if constexpr (CNT % 4 == 0) {
#pragma unroll
        for (int q = 0; q < CNT; q += 4) *reinterpret_cast<uint4 *>(p + q) = make_uint4(v[q], v[q + 1], v[q + 2], v[q + 3]);
    } else if constexpr (CNT == 2) {
        *reinterpret_cast<uint2 *>(p) = make_uint2(v[0], v[1]);
    } else {
#pragma unroll
        for (int q = 0; q < CNT; q++) p[q] = v[q];
    }
}

template <int CNT>
__device__ __forceinline__ void load_u32(const uint32_t *p, uint32_t *v) {
    if constexpr (CNT % 4 == 0) {
#pragma unroll
        for (int q = 0; q < CNT; q += 4) {
            uint4 t = *reinterpret_cast<const uint4 *>(p + q);
            v[q] = t.x; v[q + 1] = t.y; v[q + 2] = t.z; v[q + 3] = t.w;
        }
    } else if constexpr (CNT == 2) {
        uint2 t = *reinterpret_cast<const uint2 *>(p);
        v[0] = t.x; v[1] = t.y;
    } else {
#pragma unroll
        for (int q = 0; q < CNT; q++) v[q] = p[q];
    }
}

template <int CNT>
__device__ __forceinline__ void store_planes(uint16_t *p, int64_t plane_stride, const uint32_t *code) {
    if constexpr (CNT == 1) {
        const uint32_t b = code[0] + 0x80808080u;
#pragma unroll
        for (int d = 0; d < 4; d++) p[d * plane_stride] = (uint16_t)(digit_f32_bits(b, d) >> 16);
    } else {
        static_assert(CNT % 2 == 0, "digit planes are stored two elements at a time");
        uint32_t b[CNT];
#pragma unroll
        for (int q = 0; q < CNT; q++) b[q] = code[q] + 0x80808080u;
#pragma unroll
        for (int d = 0; d < 4; d++) {
            uint32_t w[CNT / 2];
#pragma unroll
            for (int q = 0; q < CNT / 2; q++) w[q] = digit_pair_bf16(b[2 * q], b[2 * q + 1], d);
            uint16_t *pd = p + d * plane_stride;
            if constexpr (CNT % 8 == 0) {
#pragma unroll
                for (int q = 0; q < CNT / 2; q += 4)
                    *reinterpret_cast<uint4 *>(pd + 2 * q) = make_uint4(w[q], w[q + 1], w[q + 2], w[q + 3]);
            } else if constexpr (CNT == 4) {
                *reinterpret_cast<uint2 *>(pd) = make_uint2(w[0], w[1]);
            } else {
                *reinterpret_cast<uint32_t *>(pd) = w[0];
            }
        }
    }
}

// A row held 32 values a thread, lane L of a warp holding elements 32 L + e
// (e = 0 .. 31) of the warp's block of 1024: the warp transposes its 32 x 32
// block through its own 4 KB of shared memory at `wb` (16-byte aligned):
// lane L's values go to words [32 L, 32 L + 32) with their 16-byte pieces
// XOR-permuted by L & 7, so the 16-byte stores and the 4-byte loads back are
// conflict-free.  On return lane L holds elements 32 e + L, and the warp has
// finished reading the block.  Lane L writes only its own 32 words, so the
// caller's last reads of them need no barrier.
__device__ __forceinline__ void warp_transpose32(float (&v)[32], uint32_t wb, int lane) {
    const uint32_t l = (uint32_t)lane;
#pragma unroll
    for (int q = 0; q < 8; ++q) {
        const uint32_t addr = wb + 4u * (32u * l + 4u * ((uint32_t)q ^ (l & 7u)));
        asm volatile("st.shared.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "f"(v[4 * q]), "f"(v[4 * q + 1]),
                     "f"(v[4 * q + 2]), "f"(v[4 * q + 3])
                     : "memory");
    }
    __syncwarp();
#pragma unroll
    for (int e = 0; e < 32; ++e) {
        const uint32_t addr = wb + 4u * (32u * (uint32_t)e + 4u * ((l >> 2) ^ ((uint32_t)e & 7u)) + (l & 3u));
        asm volatile("ld.shared.f32 %0, [%1];" : "=f"(v[e]) : "r"(addr) : "memory");
    }
    __syncwarp();
}
// Stages h = 32 .. 512 between the registers of the transposed block (v[e] =
// element 32 e + L).  Each pair, its order and its rounding are those of the
// shuffle form (lower p + q, upper p - q), so the results are identical; with
// the transpose, 40 shared-memory instructions replace 160 shuffles.
__device__ __forceinline__ void reg_stages32(float (&v)[32]) {
#pragma unroll
    for (int h = 1; h < 32; h <<= 1) {
#pragma unroll
        for (int i = 0; i < 32; i += 2 * h) {
#pragma unroll
            for (int j = i; j < i + h; j++) {
                const float p = v[j], q = v[j + h];
                v[j] = __fadd_rn(p, q);
                v[j + h] = __fsub_rn(p, q);
            }
        }
    }
}
__device__ __forceinline__ void warp_transpose_stages(float (&v)[32], uint32_t wb, int lane) {
    warp_transpose32(v, wb, lane);
    reg_stages32(v);
}

template <int E, int T>
struct Cfg {
    static constexpr int N = E * T;
    static constexpr int RPB = T >= 256 ? 1 : 256 / T;   // rows per block
    static constexpr int WN = T / 32;                     // warps per row
    static constexpr int CS = WN > 1 ? E / WN : E;        // run length per thread after phase 3
    static constexpr int RUNS = E / CS;                   // runs per thread
    static constexpr int SMEM_ROW = WN > 1 ? N + N / 32 : 0;
    static constexpr size_t SMEM = (size_t)RPB * SMEM_ROW * sizeof(float);
};

template <int E, int T>
__global__ void __launch_bounds__(T * Cfg<E, T>::RPB) fwht_kernel(FwhtArgs a) {
    using C = Cfg<E, T>;
    constexpr int N = C::N, WN = C::WN, CS = C::CS, RUNS = C::RUNS;
    static_assert(WN == 1 || E >= WN, "phase-3 layout needs E >= warps per row");
    extern __shared__ float smem[];
    __shared__ float red_max[C::RPB][WN];
    __shared__ int red_ok[C::RPB][WN];

    const int lt = threadIdx.x % T;
    const int rb = threadIdx.x / T;
    const int lane = threadIdx.x & 31;
    const int64_t row = (int64_t)blockIdx.x * C::RPB + rb;
    const bool active = row < a.rows;
    const int base = lt * E;

    float v[E];
    if (active) {
        // Split mode: row = 2 r + h is half h of the 2N-wide row r.
        const int64_t half = a.split ? (row & 1) : 0;
        const float *xr = a.split ? a.x + (row >> 1) * a.ldx + half * N : a.x + row * a.ldx;
        const int64_t nrow = a.split ? (a.n - half * N < 0 ? 0 : (a.n - half * N < N ? a.n - half * N : N)) : a.n;
        if (E % 4 == 0 && a.vec_x && base + E <= nrow) {
#pragma unroll
            for (int q = 0; q < E; q += 4) {
                float4 t = *reinterpret_cast<const float4 *>(xr + base + q);
                v[q] = t.x; v[q + 1] = t.y; v[q + 2] = t.z; v[q + 3] = t.w;
            }
        } else {
#pragma unroll
            for (int e = 0; e < E; e++) v[e] = (base + e < nrow) ? xr[base + e] : 0.0f;
        }
    } else {
#pragma unroll
        for (int e = 0; e < E; e++) v[e] = 0.0f;
    }
    // Element index of the run-th group of CS outputs this thread writes.
    auto out_elem = [&](int run) -> int {
        if constexpr (WN > 1) return run * 32 * E + lt * CS;
        else return base;
    };
    // The mask words this thread adds at the end are loaded now, so that their
    // latency overlaps the rotation (rows up to 16384 words: longer rows run
    // 1024-thread blocks whose register budget has no room for them).
    constexpr bool kPrefetch = N <= 16384;
    uint32_t mk_pre[kPrefetch ? E : 1];
    if constexpr (kPrefetch) {
        if (a.mode == 1 && a.mask && active) {
            const uint32_t *mr = a.mask + row * a.ldm;
#pragma unroll
            for (int run = 0; run < RUNS; run++) load_u32<CS>(mr + out_elem(run), mk_pre + run * CS);
        }
    }

    if (a.rotate) {
        if (a.signs) {
            const uint32_t w = a.signs[(a.split ? (row & 1) * (N / 32) : 0) + (base >> 5)] >> (base & 31);
#pragma unroll
            for (int e = 0; e < E; e++)
                if ((w >> e) & 1u) v[e] = -v[e];
        }
        // Phase 1: h = 1 .. E/2 in registers.
#pragma unroll
        for (int h = 1; h < E; h <<= 1) {
#pragma unroll
            for (int i = 0; i < E; i += 2 * h) {
#pragma unroll
                for (int j = i; j < i + h; j++) {
                    const float p = v[j], q = v[j + h];
                    v[j] = __fadd_rn(p, q);
                    v[j + h] = __fsub_rn(p, q);
                }
            }
        }
        // Phase 2: h = E .. 16E across lanes.  With 32 values a thread (and a
        // shared-memory row) the warp transposes its block in its own part of
        // the row buffer, words [1056 w, 1056 w + 1024), which is where its
        // phase-3 stores land, so no other warp touches them.  Otherwise: the
        // lower lane of a pair keeps v + o, the upper o - v, one fused
        // multiply-add by +-1 (the product is exact, so the single rounding is
        // that of the plain sum or difference).
        if constexpr (E == 32 && WN > 1) {
            warp_transpose_stages(
                v, (uint32_t)__cvta_generic_to_shared(smem + rb * C::SMEM_ROW + 1056 * (lt >> 5)), lane);
        } else {
#pragma unroll
            for (int hl = 1; hl < 32; hl <<= 1) {
                const float sgn = (lane & hl) ? -1.0f : 1.0f;
#pragma unroll
                for (int e = 0; e < E; e++) {
                    const float o = __shfl_xor_sync(0xffffffffu, v[e], hl);
                    v[e] = __fmaf_rn(v[e], sgn, o);
                }
            }
        }
    }

    // Phase 3: h = 32E .. N/2 after a transpose through shared memory.  The
    // transpose runs whether or not the row is rotated, so that the output
    // layout below is the same in both cases.
    if constexpr (WN > 1) {
        float *buf = smem + rb * C::SMEM_ROW;
        if (E == 32 && a.rotate) {
            // After the warp transpose v[e] is element 1024 w + 32 e + lane.
#pragma unroll
            for (int e = 0; e < E; e++) buf[pad_idx(1024 * (lt >> 5) + 32 * e + lane)] = v[e];
        } else {
#pragma unroll
            for (int e = 0; e < E; e++) buf[pad_idx(base + e)] = v[e];
        }
        __syncthreads();
#pragma unroll
        for (int j = 0; j < WN; j++)
#pragma unroll
            for (int u = 0; u < CS; u++) v[j * CS + u] = buf[pad_idx(j * 32 * E + lt * CS + u)];
        if (a.rotate) {
#pragma unroll
            for (int hj = 1; hj < WN; hj <<= 1) {
#pragma unroll
                for (int i = 0; i < WN; i += 2 * hj) {
#pragma unroll
                    for (int j = i; j < i + hj; j++) {
#pragma unroll
                        for (int u = 0; u < CS; u++) {
                            const float p = v[j * CS + u], q = v[(j + hj) * CS + u];
                            v[j * CS + u] = __fadd_rn(p, q);
                            v[(j + hj) * CS + u] = __fsub_rn(p, q);
                        }
                    }
                }
            }
        }
    }
    if (a.rotate) {
#pragma unroll
        for (int e = 0; e < E; e++) v[e] = __fmul_rn(v[e], a.inv_sqrt);
    }

    // Element index of v[run * CS + u].
    auto elem = [&](int run) -> int {
        if constexpr (WN > 1) return run * 32 * E + lt * CS;
        else return base;
    };
    (void)elem;

    if (a.mode == 0) {
        if (active) {
            float *yr = a.split ? a.y + (row >> 1) * a.ldy + (row & 1) * N : a.y + row * a.ldy;
#pragma unroll
            for (int run = 0; run < RUNS; run++) store_f32<CS>(yr + elem(run), v + run * CS);
        }
        return;
    }

    // Encode: per-row absmax (and finiteness) reduction.
    float mx = 0.0f;
    int ok = 1;
#pragma unroll
    for (int e = 0; e < E; e++) {
        ok &= isfinite(v[e]) ? 1 : 0;
        mx = fmaxf(mx, fabsf(v[e]));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        ok &= __shfl_xor_sync(0xffffffffu, ok, o);
    }
    if constexpr (WN > 1) {
        const int wr = lt >> 5;
        if (lane == 0) { red_max[rb][wr] = mx; red_ok[rb][wr] = ok; }
        __syncthreads();
#pragma unroll
        for (int w = 0; w < WN; w++) { mx = fmaxf(mx, red_max[rb][w]); ok &= red_ok[rb][w]; }
    }
    if (!active) return;
    const float s = ok ? __fdiv_rn(mx, (float)a.qmax) : __int_as_float(0x7fc00000);
    if (lt == 0) a.scale[row] = s;
    // code = clamp(rint(v / s), -qmax, qmax).  |v / s| <= qmax (1 + 2^-23)
    // < 2^22, where adding 1.5 * 2^23 rounds to the nearest integer (ties to
    // even) in the low mantissa bits, so the integer is read from the bits.
    const bool quant = ok && s != 0.0f;
    uint32_t code[E];
#pragma unroll
    for (int e = 0; e < E; e++) {
        const float t = __fadd_rn(__fdiv_rn(v[e], s), 12582912.0f);
        int32_t c = __float_as_int(t) - 0x4B400000;
        c = min(max(c, -a.qmax), a.qmax);
        code[e] = quant ? (uint32_t)c : 0u;
    }
    if (a.mask) {
        if constexpr (kPrefetch) {
#pragma unroll
            for (int e = 0; e < E; e++) code[e] += mk_pre[e];
        } else {
            const uint32_t *mr = a.mask + row * a.ldm;
#pragma unroll
            for (int run = 0; run < RUNS; run++) {
                uint32_t mk[CS];
                load_u32<CS>(mr + elem(run), mk);
#pragma unroll
                for (int u = 0; u < CS; u++) code[run * CS + u] += mk[u];
            }
        }
    }
    uint32_t *orow = a.out + row * a.ldo;
#pragma unroll
    for (int run = 0; run < RUNS; run++) store_u32<CS>(orow + elem(run), code + run * CS);
    if (a.planes) {
        const int64_t ps = a.rows * a.n_pad;
        uint16_t *prow = a.planes + row * a.n_pad;
#pragma unroll
        for (int run = 0; run < RUNS; run++) store_planes<CS>(prow + elem(run), ps, code + run * CS);
    }
}

template <int E, int T>
mosaic_status launch(const FwhtArgs &a, cudaStream_t st) {
    using C = Cfg<E, T>;
    static_assert(C::N >= 32, "");
    if (C::SMEM > 48 * 1024) {
        if (cudaFuncSetAttribute(fwht_kernel<E, T>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)C::SMEM) != cudaSuccess)
            return MOSAIC_ERR_CUDA;
    }
    const int64_t blocks = (a.rows + C::RPB - 1) / C::RPB;
    {
        KernelSpan span("fwht", st);
        fwht_kernel<E, T><<<(unsigned)blocks, T * C::RPB, C::SMEM, st>>>(a);
    }
    return launch_status();
}

// ---------------------------------------------------------------------------
// Encode of rows of 32768 whose length n is a multiple of 32 (the rotation
// alone runs rot_kernel below): a persistent grid (one block per SM) that
// fetches each block's NEXT input row by TMA while the current row is
// transformed and stored.  In the kernel above an SM
// holds a single row at a time (32 values per thread in registers, a 512- or
// 1024-thread block), so its loads, butterflies and stores never overlap.
// The row arrives as a 3-D tensor {32 values, chunks, rows} with the 128-byte
// swizzle: chunk c (thread c's 32 consecutive values) lies at bytes
// [128 c, 128 c + 128) with its 16-byte pieces XOR-permuted by c & 7, so each
// thread reads its own run with 8 conflict-free 16-byte loads.  The
// arithmetic (stage order, roundings) is that of fwht_kernel, line for line,
// so the results are identical.  The transpose runs in the input buffer
// (132 KB) and the encode reads the mask from global memory.  Every wait is
// bounded; on expiry the block raises g_fwht_error and stops.
// ---------------------------------------------------------------------------
template <int T>
struct StreamCfg {
    static constexpr int E = 32;
    static constexpr int N = E * T;
    static constexpr int WN = T / 32;
    static constexpr int CS = E / WN;
    static constexpr int RUNS = E / CS;
    static constexpr size_t XBUF = (size_t)(N + N / 32) * 4;        // input row, then its transpose
    static constexpr size_t SMEM = 1024 + XBUF + 64;
    static constexpr int BOX_CHUNKS = 256;                           // 32 KB per copy
    static constexpr int COPIES = N / 32 / BOX_CHUNKS;
};

template <int T>
__global__ void __launch_bounds__(T, 1) fwht_stream_kernel(const __grid_constant__ CUtensorMap tmx, FwhtArgs a) {
    using C = StreamCfg<T>;
    constexpr int E = C::E, N = C::N, WN = C::WN, CS = C::CS, RUNS = C::RUNS;
    extern __shared__ uint8_t raw[];
    uint8_t *base_ptr = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(raw) + 1023) & ~(uintptr_t)1023);
    float *xbuf = reinterpret_cast<float *>(base_ptr);
    float *tbuf = xbuf;
    uint64_t *bar_x = reinterpret_cast<uint64_t *>(base_ptr + C::XBUF);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(bar_x + 1);
    __shared__ float red_max[WN];
    __shared__ int red_ok[WN];

    const int lt = threadIdx.x, lane = lt & 31;
    const int base = lt * E;
    if (lt == 0) {
        mbar_init(bar_x, 1);
        *abort_flag = 0;
        mbar_init_fence();
    }
    __syncthreads();
    // Rows blockIdx.x, blockIdx.x + gridDim.x, ...
    auto issue_x = [&](int64_t row) {
        mbar_expect_tx(bar_x, (uint32_t)(N * 4));
#pragma unroll
        for (int c = 0; c < C::COPIES; ++c)
            tma_load_3d(reinterpret_cast<uint8_t *>(xbuf) + (size_t)c * C::BOX_CHUNKS * 128, &tmx, bar_x, 0,
                        c * C::BOX_CHUNKS, (int)row);
    };
    // The sign bits of this thread's 32 values are the same for every row.
    const uint32_t sign_w = (a.rotate && a.signs) ? a.signs[base >> 5] : 0u;
    int64_t row = blockIdx.x;
    if (lt == 0 && row < a.rows) issue_x(row);
    uint32_t ph = 0;
    for (; row < a.rows; row += gridDim.x, ph ^= 1u) {
        const int64_t next = row + gridDim.x;
        if (!mbar_wait(bar_x, ph, abort_flag)) {
            *abort_flag = 1;
            atomicExch(&g_fwht_error, 1u);
        }
        __syncthreads();
        if (*abort_flag) break;
        // The encode adds this row's mask words at the end: ask L2 for them now
        // (lane L: the warp's 128-byte line of run L).
        if (a.mode == 1 && a.mask)
            asm volatile("prefetch.global.L2 [%0];" ::"l"(a.mask + row * a.ldm + lane * 1024 + 32 * (lt >> 5)));
        // This thread's 32 values: chunk lt, 16-byte piece q at q ^ (lt & 7).
        float v[E];
        {
            const uint32_t rb = smem_u32(xbuf) + (uint32_t)lt * 128u;
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                const uint32_t addr = rb + (uint32_t)((q ^ (lt & 7)) * 16);
                asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
                             : "=f"(v[4 * q]), "=f"(v[4 * q + 1]), "=f"(v[4 * q + 2]), "=f"(v[4 * q + 3])
                             : "r"(addr)
                             : "memory");
            }
        }
        if (a.rotate) {
            if (a.signs) {
#pragma unroll
                for (int e = 0; e < E; e++)
                    if ((sign_w >> e) & 1u) v[e] = -v[e];
            }
#pragma unroll
            for (int h = 1; h < E; h <<= 1) {
#pragma unroll
                for (int i = 0; i < E; i += 2 * h) {
#pragma unroll
                    for (int j = i; j < i + h; j++) {
                        const float p = v[j], q = v[j + h];
                        v[j] = __fadd_rn(p, q);
                        v[j + h] = __fsub_rn(p, q);
                    }
                }
            }
            // Stages h = 32 .. 512 through this warp's 4 KB of the input
            // buffer, which only this warp has read.
            warp_transpose_stages(v, smem_u32(xbuf) + 4096u * (uint32_t)(lt >> 5), lane);
        }
        __syncthreads();   // every thread has read the input buffer
        if (a.rotate) {
            // v[e] is element 1024 w + 32 e + lane after the warp transpose.
#pragma unroll
            for (int e = 0; e < E; e++) tbuf[pad_idx(1024 * (lt >> 5) + 32 * e + lane)] = v[e];
        } else {
#pragma unroll
            for (int e = 0; e < E; e++) tbuf[pad_idx(base + e)] = v[e];
        }
        __syncthreads();
#pragma unroll
        for (int j = 0; j < WN; j++)
#pragma unroll
            for (int u = 0; u < CS; u++) v[j * CS + u] = tbuf[pad_idx(j * 32 * E + lt * CS + u)];
        // The transpose was done in the input buffer: fetch the next row now.
        __syncthreads();
        if (lt == 0 && next < a.rows && !*abort_flag) {
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            issue_x(next);
        }
        if (a.rotate) {
#pragma unroll
            for (int hj = 1; hj < WN; hj <<= 1) {
#pragma unroll
                for (int i = 0; i < WN; i += 2 * hj) {
#pragma unroll
                    for (int j = i; j < i + hj; j++) {
#pragma unroll
                        for (int u = 0; u < CS; u++) {
                            const float p = v[j * CS + u], q = v[(j + hj) * CS + u];
                            v[j * CS + u] = __fadd_rn(p, q);
                            v[(j + hj) * CS + u] = __fsub_rn(p, q);
                        }
                    }
                }
            }
#pragma unroll
            for (int e = 0; e < E; e++) v[e] = __fmul_rn(v[e], a.inv_sqrt);
        }
        auto elem = [&](int run) -> int { return run * 32 * E + lt * CS; };
        float mx = 0.0f;
        int ok = 1;
#pragma unroll
        for (int e = 0; e < E; e++) {
            ok &= isfinite(v[e]) ? 1 : 0;
            mx = fmaxf(mx, fabsf(v[e]));
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
            ok &= __shfl_xor_sync(0xffffffffu, ok, o);
        }
        if (lane == 0) {
            red_max[lt >> 5] = mx;
            red_ok[lt >> 5] = ok;
        }
        __syncthreads();
#pragma unroll
        for (int w = 0; w < WN; w++) {
            mx = fmaxf(mx, red_max[w]);
            ok &= red_ok[w];
        }
        const float s = ok ? __fdiv_rn(mx, (float)a.qmax) : __int_as_float(0x7fc00000);
        if (lt == 0) a.scale[row] = s;
        const bool quant = ok && s != 0.0f;
        uint32_t code[E];
#pragma unroll
        for (int e = 0; e < E; e++) {
            const float t = __fadd_rn(__fdiv_rn(v[e], s), 12582912.0f);
            int32_t c = __float_as_int(t) - 0x4B400000;
            c = min(max(c, -a.qmax), a.qmax);
            code[e] = quant ? (uint32_t)c : 0u;
        }
        if (a.mask) {
            const uint32_t *mr = a.mask + row * a.ldm;
#pragma unroll
            for (int run = 0; run < RUNS; run++) {
                uint32_t mk[CS];
                load_u32<CS>(mr + elem(run), mk);
#pragma unroll
                for (int u = 0; u < CS; u++) code[run * CS + u] += mk[u];
            }
        }
        uint32_t *orow = a.out + row * a.ldo;
#pragma unroll
        for (int run = 0; run < RUNS; run++) store_u32<CS>(orow + elem(run), code + run * CS);
        if (a.planes) {
            const int64_t ps = a.rows * a.n_pad;
            uint16_t *prow = a.planes + row * a.n_pad;
#pragma unroll
            for (int run = 0; run < RUNS; run++) store_planes<CS>(prow + elem(run), ps, code + run * CS);
        }
    }
    // After a normal exit every issued copy has been waited for; after an
    // expired wait, let the copies still in flight land (bounded) first.
    if (lt == 0 && *abort_flag) mbar_drain(bar_x, ph);
    __syncthreads();
}

// 3-D view {32 words, chunks, rows} of a row-major matrix with rows of `len`
// 4-byte words (len a multiple of 32) and row stride ld words.
bool make_chunk_map(CUtensorMap *map, const void *base, int64_t len, int64_t rows, int64_t ld, bool is_float) {
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[3] = {32, (cuuint64_t)(len / 32), (cuuint64_t)rows};
    cuuint64_t strides[2] = {128, (cuuint64_t)ld * 4};
    cuuint32_t box[3] = {32, 256, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    return fn(map, is_float ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_UINT32, 3,
              const_cast<void *>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
              CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int T>
mosaic_status launch_stream(const FwhtArgs &a, cudaStream_t st) {
    using C = StreamCfg<T>;
    CUtensorMap tmx;
    if (!make_chunk_map(&tmx, a.x, a.n, a.rows, a.ldx, true)) return MOSAIC_ERR_CUDA;
    static std::atomic<unsigned long long> attr_set{0};
    int dev = 0, sms = 0;
    if (!ensure_smem_limit(attr_set, fwht_stream_kernel<T>, C::SMEM, &dev) ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 1)
        return MOSAIC_ERR_CUDA;
    const int64_t grid = a.rows < sms ? a.rows : sms;
    {
        KernelSpan span("fwht_stream", st);
        fwht_stream_kernel<T><<<(unsigned)grid, T, C::SMEM, st>>>(tmx, a);
    }
    return launch_status();
}

// The streamed kernels take rows whose length is a multiple of 32 words with
// 16-byte aligned rows (x, and the mask when there is one); rows of 2^31 or
// more are left to the per-row kernel (32-bit row coordinates).
bool stream_ok(const FwhtArgs &a) {
    if (a.split || a.rows >= (int64_t)1 << 31) return false;
    if (a.n % 32 != 0 || !aligned16(a.x) || a.ldx % 4 != 0) return false;
    if (a.mode == 1 && a.mask && (!aligned16(a.mask) || a.ldm % 4 != 0)) return false;
    return encode_fn() != nullptr;
}

// ---------------------------------------------------------------------------
// Encode of rows of 16384 (length n a multiple of 32; the rotation alone runs
// rot_kernel below), two rows in flight per SM.  Each
// CTA (512 threads, 32 values a thread, at most 64 registers so that two CTAs
// share an SM) transforms one row at a time with the stage order and roundings
// of fwht_kernel, so the results are identical.  The row arrives by TMA in the
// CTA's input buffer (the 3-D {32 values, chunks, rows} view with the 128-byte
// swizzle: chunk c, thread c's 32 consecutive values, lies at bytes
// [128 c, 128 c + 128) with its 16-byte pieces XOR-permuted by c & 7, so each
// thread reads its run with 8 conflict-free 16-byte loads); the transpose
// reuses the buffer, and the next row's copy is issued as soon as the
// transpose has been read back.  One CTA cannot overlap its own butterflies
// with its stores, but the other CTA on the SM can.  The TMA wait is bounded
// (abort flag + g_fwht_error).
// ---------------------------------------------------------------------------
constexpr int kPairT = 512;                     // threads per CTA
constexpr int kPairE = 32;                      // values per thread
constexpr int kPairN = kPairT * kPairE;         // values per CTA: 16384
constexpr int kPairWN = kPairT / 32;            // warps: 16
constexpr int kPairCS = kPairE / kPairWN;       // run length after the transpose: 2
constexpr int kPairRuns = kPairE / kPairCS;     // runs: 16
constexpr size_t kPairXBUF = (size_t)(kPairN + kPairN / 32) * 4;   // padded transpose fits
constexpr size_t kPairSMEM = 1024 + kPairXBUF + 64;
constexpr int kPairBox = 256;                   // chunks of 32 values per TMA box (32 KB)

__global__ void __launch_bounds__(kPairT, 2) fwht_pair_kernel(const __grid_constant__ CUtensorMap tmx, FwhtArgs a) {
    constexpr int E = kPairE, N = kPairN, WN = kPairWN, CS = kPairCS, RUNS = kPairRuns;
    extern __shared__ uint8_t raw[];
    uint8_t *base_ptr = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(raw) + 1023) & ~(uintptr_t)1023);
    float *xbuf = reinterpret_cast<float *>(base_ptr);
    uint64_t *bar_x = reinterpret_cast<uint64_t *>(base_ptr + kPairXBUF);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(bar_x + 1);
    __shared__ float red_max[WN];
    __shared__ int red_ok[WN];

    const int lt = threadIdx.x, lane = lt & 31;
    const int base = lt * E;
    if (lt == 0) {
        mbar_init(bar_x, 1);
        *abort_flag = 0;
        mbar_init_fence();
    }
    __syncthreads();
    auto issue_x = [&](int64_t row) {
        mbar_expect_tx(bar_x, (uint32_t)(N * 4));
#pragma unroll
        for (int c = 0; c < N / 32 / kPairBox; ++c)
            tma_load_3d(reinterpret_cast<uint8_t *>(xbuf) + (size_t)c * kPairBox * 128, &tmx, bar_x, 0,
                        c * kPairBox, (int)row);
    };
    // The sign bits of this thread's 32 values are the same for every row.
    const uint32_t sign_w = (a.rotate && a.signs) ? a.signs[base >> 5] : 0u;
    int64_t row = blockIdx.x;
    if (lt == 0 && row < a.rows) issue_x(row);
    uint32_t ph = 0;
    for (; row < a.rows; row += gridDim.x, ph ^= 1u) {
        const int64_t next = row + gridDim.x;
        if (!mbar_wait(bar_x, ph, abort_flag)) {
            *abort_flag = 1;
            atomicExch(&g_fwht_error, 1u);
        }
        __syncthreads();
        if (*abort_flag) break;
        // The encode adds this row's mask words at the end: ask L2 for them now
        // (lane L: line L & 1 of the warp's 256 bytes of run L / 2).
        if (a.mode == 1 && a.mask)
            asm volatile("prefetch.global.L2 [%0];" ::"l"(a.mask + row * a.ldm + (lane >> 1) * 1024 + 64 * (lt >> 5) +
                                                       32 * (lane & 1)));
        float v[E];
        {
            const uint32_t rb = smem_u32(xbuf) + (uint32_t)lt * 128u;
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                const uint32_t addr = rb + (uint32_t)((q ^ (lt & 7)) * 16);
                asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
                             : "=f"(v[4 * q]), "=f"(v[4 * q + 1]), "=f"(v[4 * q + 2]), "=f"(v[4 * q + 3])
                             : "r"(addr)
                             : "memory");
            }
        }
        if (a.rotate) {
            if (a.signs) {
#pragma unroll
                for (int e = 0; e < E; e++)
                    if ((sign_w >> e) & 1u) v[e] = -v[e];
            }
#pragma unroll
            for (int h = 1; h < E; h <<= 1) {
#pragma unroll
                for (int i = 0; i < E; i += 2 * h) {
#pragma unroll
                    for (int j = i; j < i + h; j++) {
                        const float p = v[j], q = v[j + h];
                        v[j] = __fadd_rn(p, q);
                        v[j + h] = __fsub_rn(p, q);
                    }
                }
            }
            // Stages h = 32 .. 512 through this warp's 4 KB of the input
            // buffer, which only this warp has read.
            warp_transpose_stages(v, smem_u32(xbuf) + 4096u * (uint32_t)(lt >> 5), lane);
        }
        __syncthreads();   // every thread has read the input buffer
        if (a.rotate) {
            // v[e] is element 1024 w + 32 e + lane after the warp transpose.
#pragma unroll
            for (int e = 0; e < E; e++) xbuf[pad_idx(1024 * (lt >> 5) + 32 * e + lane)] = v[e];
        } else {
#pragma unroll
            for (int e = 0; e < E; e++) xbuf[pad_idx(base + e)] = v[e];
        }
        __syncthreads();
#pragma unroll
        for (int j = 0; j < WN; j++)
#pragma unroll
            for (int u = 0; u < CS; u++) v[j * CS + u] = xbuf[pad_idx(j * 32 * E + lt * CS + u)];
        __syncthreads();   // every thread has read the transpose
        if (lt == 0 && next < a.rows) {
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            issue_x(next);
        }
        if (a.rotate) {
#pragma unroll
            for (int hj = 1; hj < WN; hj <<= 1) {
#pragma unroll
                for (int i = 0; i < WN; i += 2 * hj) {
#pragma unroll
                    for (int j = i; j < i + hj; j++) {
#pragma unroll
                        for (int u = 0; u < CS; u++) {
                            const float p = v[j * CS + u], q = v[(j + hj) * CS + u];
                            v[j * CS + u] = __fadd_rn(p, q);
                            v[(j + hj) * CS + u] = __fsub_rn(p, q);
                        }
                    }
                }
            }
        }
        auto elem = [&](int run) -> int { return run * 32 * E + lt * CS; };
        if (a.rotate) {
#pragma unroll
            for (int e = 0; e < E; e++) v[e] = __fmul_rn(v[e], a.inv_sqrt);
        }
        if (a.mode == 0) {   // rotation alone (launched as rot_kernel; kept for direct use)
            float *yr = a.y + row * a.ldy;
#pragma unroll
            for (int run = 0; run < RUNS; run++) store_f32<CS>(yr + elem(run), v + run * CS);
            continue;
        }
        float mx = 0.0f;
        int ok = 1;
#pragma unroll
        for (int e = 0; e < E; e++) {
            ok &= isfinite(v[e]) ? 1 : 0;
            mx = fmaxf(mx, fabsf(v[e]));
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
            ok &= __shfl_xor_sync(0xffffffffu, ok, o);
        }
        if (lane == 0) {
            red_max[lt >> 5] = mx;
            red_ok[lt >> 5] = ok;
        }
        __syncthreads();
#pragma unroll
        for (int w = 0; w < WN; w++) {
            mx = fmaxf(mx, red_max[w]);
            ok &= red_ok[w];
        }
        const float s = ok ? __fdiv_rn(mx, (float)a.qmax) : __int_as_float(0x7fc00000);
        if (lt == 0) a.scale[row] = s;
        const bool quant = ok && s != 0.0f;
        uint32_t code[E];
#pragma unroll
        for (int e = 0; e < E; e++) {
            const float t = __fadd_rn(__fdiv_rn(v[e], s), 12582912.0f);
            int32_t c = __float_as_int(t) - 0x4B400000;
            c = min(max(c, -a.qmax), a.qmax);
            code[e] = quant ? (uint32_t)c : 0u;
        }
        if (a.mask) {
            const uint32_t *mr = a.mask + row * a.ldm;
#pragma unroll
            for (int run = 0; run < RUNS; run++) {
                uint32_t mk[CS];
                load_u32<CS>(mr + elem(run), mk);
#pragma unroll
                for (int u = 0; u < CS; u++) code[run * CS + u] += mk[u];
            }
        }
        uint32_t *orow = a.out + row * a.ldo;
#pragma unroll
        for (int run = 0; run < RUNS; run++) store_u32<CS>(orow + elem(run), code + run * CS);
        if (a.planes) {
            const int64_t ps = a.rows * a.n_pad;
            uint16_t *prow = a.planes + row * a.n_pad;
#pragma unroll
            for (int run = 0; run < RUNS; run++) store_planes<CS>(prow + elem(run), ps, code + run * CS);
        }
    }
    // After a normal exit every issued copy has been waited for; after an
    // expired wait, let the copy still in flight land (bounded) first.
    if (lt == 0 && *abort_flag) mbar_drain(bar_x, ph);
    __syncthreads();
}

mosaic_status launch_pair(const FwhtArgs &a, cudaStream_t st) {
    CUtensorMap tmx;
    if (!make_chunk_map(&tmx, a.x, a.n, a.rows, a.ldx, true)) return MOSAIC_ERR_CUDA;
    static std::atomic<unsigned long long> attr_set{0};
    int dev = 0, sms = 0, per_sm = 0;
    if (!ensure_smem_limit(attr_set, fwht_pair_kernel, kPairSMEM, &dev) ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 1 ||
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fwht_pair_kernel, kPairT, kPairSMEM) != cudaSuccess ||
        per_sm < 1)
        return MOSAIC_ERR_CUDA;
    // As many rows in flight as the GPU holds at once (two CTAs per SM), each
    // CTA walking rows with a stride of the grid.
    const int64_t slots = (int64_t)sms * per_sm;
    const int64_t grid = a.rows < slots ? a.rows : slots;
    {
        KernelSpan span("fwht_pair", st);
        fwht_pair_kernel<<<(unsigned)grid, kPairT, kPairSMEM, st>>>(tmx, a);
    }
    return launch_status();
}

// ---------------------------------------------------------------------------
// Rotation alone (mosaic_hadamard) of rows of 16384 and 32768 whose length n
// is a multiple of 32.  Without the encode's long per-row tail (quantise, mask
// words, digit planes) to hide it, the copy of a block's next row has to start
// early: these kernels refill the input buffer in two halves, each on its own
// barrier, the first as soon as every thread has read the row and the second
// once phase 2 is done, and run the exchange between warps for phase 3 in a
// buffer of its own (R, plus P for 32768).  Warps whose part of the input
// buffer is being refilled transpose their blocks for phase 2 in R instead.
// Rows arrive as for the kernels above (the 3-D {32 values, chunks, rows} view
// with the 128-byte swizzle); stage order and roundings are those of
// fwht_kernel, so the results are identical.  The TMA waits are bounded (abort
// flag + g_fwht_error).
//
// 16384 (two 512-thread CTAs per SM, 64 registers): phase 3 holds
// v[2 j + u] = element 1024 j + 512 u + t (t the thread), i.e. register
// 16 u + w of warp j, same lane, so the exchange runs through R (32 KB) in two
// rounds, one per half of the registers, and no thread holds more than 32
// values.
// 32768 (one 1024-thread CTA per SM): phase 3 holds v[j] = element
// 1024 j + t, register w of warp j, same lane; in round 0 every warp stores
// v[0..15] in R (64 KB) and warps 0-15 park v[16..31] in P (32 KB) before
// reading their 32 values from R; in round 1 warps 16-31 store v[16..31] in R
// and read theirs from R and P.
// ---------------------------------------------------------------------------
constexpr int kRotRowBox = 256;   // chunks of 32 values per TMA box (32 KB)

template <int T>
struct RotCfg {
    static_assert(T == 512 || T == 1024, "rows of 16384 or 32768");
    static constexpr int E = 32;
    static constexpr int N = E * T;
    static constexpr int WN = T / 32;
    static constexpr int BOXES = N / 32 / kRotRowBox;        // 2 or 4, half of them per half-row copy
    static constexpr size_t XBUF = (size_t)N * 4;            // the row as it lands
    static constexpr size_t RBUF = (size_t)N / 2 * 4;        // R: 16 registers x WN warps x 32 lanes
    static constexpr size_t PBUF = T == 1024 ? (size_t)N / 4 * 4 : 0;   // P: 16 registers x 16 warps x 32 lanes
    static constexpr size_t SMEM = 1024 + XBUF + RBUF + PBUF + 64;
};

template <int T>
__global__ void __launch_bounds__(T, T == 512 ? 2 : 1) rot_kernel(const __grid_constant__ CUtensorMap tmx, FwhtArgs a) {
    using C = RotCfg<T>;
    constexpr int E = C::E, N = C::N, WN = C::WN;
    extern __shared__ uint8_t raw[];
    uint8_t *base_ptr = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(raw) + 1023) & ~(uintptr_t)1023);
    float *xbuf = reinterpret_cast<float *>(base_ptr);
    float *rbuf = reinterpret_cast<float *>(base_ptr + C::XBUF);
    float *pbuf = reinterpret_cast<float *>(base_ptr + C::XBUF + C::RBUF);
    uint64_t *bar = reinterpret_cast<uint64_t *>(base_ptr + C::XBUF + C::RBUF + C::PBUF);   // one per half
    volatile int *abort_flag = reinterpret_cast<volatile int *>(bar + 2);

    const int lt = threadIdx.x, lane = lt & 31, w = lt >> 5;
    const int base = lt * E;
    if (lt == 0) {
        mbar_init(&bar[0], 1);
        mbar_init(&bar[1], 1);
        *abort_flag = 0;
        mbar_init_fence();
    }
    __syncthreads();
    // Half h of row `row`: boxes [h BOXES / 2, (h + 1) BOXES / 2).
    auto issue_half = [&](int64_t row, int h) {
        mbar_expect_tx(&bar[h], (uint32_t)(N * 2));
#pragma unroll
        for (int c = h * (C::BOXES / 2); c < (h + 1) * (C::BOXES / 2); ++c)
            tma_load_3d(reinterpret_cast<uint8_t *>(xbuf) + (size_t)c * kRotRowBox * 128, &tmx, &bar[h], 0,
                        c * kRotRowBox, (int)row);
    };
    // The sign bits of this thread's 32 values are the same for every row.
    const uint32_t sign_w = (a.rotate && a.signs) ? a.signs[base >> 5] : 0u;
    // This warp's 4 KB for its block transpose: R for the warps of the lower
    // half (refilled first), its own part of the upper half of the input
    // buffer for the others.
    const uint32_t wb = w < WN / 2 ? smem_u32(rbuf) + 4096u * (uint32_t)w : smem_u32(xbuf) + 4096u * (uint32_t)w;
    int64_t row = blockIdx.x;
    if (lt == 0 && row < a.rows) {
        issue_half(row, 0);
        issue_half(row, 1);
    }
    uint32_t ph = 0;
    for (; row < a.rows; row += gridDim.x, ph ^= 1u) {
        const int64_t next = row + gridDim.x;
        if (!mbar_wait(&bar[0], ph, abort_flag) || !mbar_wait(&bar[1], ph, abort_flag)) {
            *abort_flag = 1;
            atomicExch(&g_fwht_error, 1u);
        }
        __syncthreads();
        if (*abort_flag) break;
        // This thread's 32 values: chunk lt, 16-byte piece q at q ^ (lt & 7).
        float v[E];
        {
            const uint32_t rb = smem_u32(xbuf) + (uint32_t)lt * 128u;
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                const uint32_t addr = rb + (uint32_t)((q ^ (lt & 7)) * 16);
                asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
                             : "=f"(v[4 * q]), "=f"(v[4 * q + 1]), "=f"(v[4 * q + 2]), "=f"(v[4 * q + 3])
                             : "r"(addr)
                             : "memory");
            }
        }
        __syncthreads();   // every thread has read the row
        if (lt == 0 && next < a.rows) {
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            issue_half(next, 0);
        }
        if (a.rotate) {
            if (a.signs) {
#pragma unroll
                for (int e = 0; e < E; e++)
                    if ((sign_w >> e) & 1u) v[e] = -v[e];
            }
#pragma unroll
            for (int h = 1; h < E; h <<= 1) {
#pragma unroll
                for (int i = 0; i < E; i += 2 * h) {
#pragma unroll
                    for (int j = i; j < i + h; j++) {
                        const float p = v[j], q = v[j + h];
                        v[j] = __fadd_rn(p, q);
                        v[j + h] = __fsub_rn(p, q);
                    }
                }
            }
        }
        // v[e] becomes element 1024 w + 32 e + lane (with or without rotation,
        // so that the layout below is the same), then stages h = 32 .. 512.
        warp_transpose32(v, wb, lane);
        if (a.rotate) reg_stages32(v);
        __syncthreads();   // R and the upper half of the input buffer are free
        if (lt == 0 && next < a.rows) {
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            issue_half(next, 1);
        }
        if constexpr (T == 512) {
            float t[E];
            // R word (e * 16 + warp) * 32 + lane holds register 16 u + e in
            // round u; thread (w, lane) reads its 16 values of round u at e = w.
#pragma unroll
            for (int e = 0; e < 16; e++) rbuf[(e * 16 + w) * 32 + lane] = v[e];
            __syncthreads();
#pragma unroll
            for (int j = 0; j < WN; j++) t[2 * j] = rbuf[(w * 16 + j) * 32 + lane];
            __syncthreads();
#pragma unroll
            for (int e = 0; e < 16; e++) rbuf[(e * 16 + w) * 32 + lane] = v[16 + e];
            __syncthreads();
#pragma unroll
            for (int j = 0; j < WN; j++) t[2 * j + 1] = rbuf[(w * 16 + j) * 32 + lane];
#pragma unroll
            for (int e = 0; e < E; e++) v[e] = t[e];
        } else {
            // R word (e * 32 + warp) * 32 + lane holds register 16 r + e of
            // round r; P word (e * 16 + warp) * 32 + lane register 16 + e of
            // warps 0-15.
#pragma unroll
            for (int e = 0; e < 16; e++) rbuf[(e * 32 + w) * 32 + lane] = v[e];
            if (w < 16) {
#pragma unroll
                for (int e = 0; e < 16; e++) pbuf[(e * 16 + w) * 32 + lane] = v[16 + e];
            }
            __syncthreads();
            if (w < 16) {
#pragma unroll
                for (int j = 0; j < WN; j++) v[j] = rbuf[(w * 32 + j) * 32 + lane];
            }
            __syncthreads();
            if (w >= 16) {
#pragma unroll
                for (int e = 0; e < 16; e++) rbuf[(e * 32 + w) * 32 + lane] = v[16 + e];
            }
            __syncthreads();
            if (w >= 16) {
#pragma unroll
                for (int j = 0; j < 16; j++) v[j] = pbuf[((w - 16) * 16 + j) * 32 + lane];
#pragma unroll
                for (int j = 16; j < WN; j++) v[j] = rbuf[((w - 16) * 32 + j) * 32 + lane];
            }
        }
        // Phase 3 (h = 1024 .. N / 2): v[U j + u] is element 1024 j + 512 u + lt
        // (U = 2 for 16384; U = 1, u = 0 for 32768).
        constexpr int U = E / WN;
        if (a.rotate) {
#pragma unroll
            for (int hj = 1; hj < WN; hj <<= 1) {
#pragma unroll
                for (int i = 0; i < WN; i += 2 * hj) {
#pragma unroll
                    for (int j = i; j < i + hj; j++) {
#pragma unroll
                        for (int u = 0; u < U; u++) {
                            const float p = v[U * j + u], q = v[U * (j + hj) + u];
                            v[U * j + u] = __fadd_rn(p, q);
                            v[U * (j + hj) + u] = __fsub_rn(p, q);
                        }
                    }
                }
            }
#pragma unroll
            for (int e = 0; e < E; e++) v[e] = __fmul_rn(v[e], a.inv_sqrt);
        }
        // v[e] is element T e + lt.
        float *yr = a.y + row * a.ldy;
#pragma unroll
        for (int e = 0; e < E; e++) yr[T * e + lt] = v[e];
    }
    // After a normal exit every issued copy has been waited for; after an
    // expired wait, let the copies still in flight land (bounded) first.
    if (lt == 0 && *abort_flag) {
        mbar_drain(&bar[0], ph);
        mbar_drain(&bar[1], ph);
    }
    __syncthreads();
}

template <int T>
mosaic_status launch_rot(const FwhtArgs &a, cudaStream_t st) {
    using C = RotCfg<T>;
    CUtensorMap tmx;
    if (!make_chunk_map(&tmx, a.x, a.n, a.rows, a.ldx, true)) return MOSAIC_ERR_CUDA;
    static std::atomic<unsigned long long> attr_set{0};
    int dev = 0, sms = 0, per_sm = 0;
    if (!ensure_smem_limit(attr_set, rot_kernel<T>, C::SMEM, &dev) ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 1 ||
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, rot_kernel<T>, T, C::SMEM) != cudaSuccess ||
        per_sm < 1)
        return MOSAIC_ERR_CUDA;
    const int64_t slots = (int64_t)sms * per_sm;
    const int64_t grid = a.rows < slots ? a.rows : slots;
    {
        KernelSpan span("fwht_rot", st);
        rot_kernel<T><<<(unsigned)grid, T, C::SMEM, st>>>(tmx, a);
    }
    return launch_status();
}

// ---------------------------------------------------------------------------
// Rows of 65536: the first 15 stages (h = 1 .. 16384) run on the two halves
// as rows of 32768 (split mode, unscaled, into y or into `out` used as fp32
// scratch); the last stage h = 32768 pairs the halves elementwise here, then
// the scale 2^-8 = fl32(1 / sqrt(65536)) (exact), and for encode the row's
// absmax (atomic max of |v| bits: finite values order like their bits, and a
// non-finite value exceeds every finite one) and the quantisation.
// ---------------------------------------------------------------------------
constexpr int64_t kHalf = 32768;

__global__ void combine_kernel(float *y, int64_t ldy, int64_t rows, int rotate, uint32_t *amax) {
    const int64_t row = blockIdx.y;
    const int64_t k = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) * 4;
    float *lo = y + row * ldy + k, *hi = lo + kHalf;
    float4 a = *reinterpret_cast<const float4 *>(lo), b = *reinterpret_cast<const float4 *>(hi);
    float va[4] = {a.x, a.y, a.z, a.w}, vb[4] = {b.x, b.y, b.z, b.w};
    uint32_t m = 0u;
#pragma unroll
    for (int q = 0; q < 4; q++) {
        if (rotate) {
            const float p = va[q], r = vb[q];
            va[q] = __fmul_rn(__fadd_rn(p, r), 0.00390625f);
            vb[q] = __fmul_rn(__fsub_rn(p, r), 0.00390625f);
        }
        m = max(m, max(__float_as_uint(va[q]) & 0x7fffffffu, __float_as_uint(vb[q]) & 0x7fffffffu));
    }
    if (rotate) {
        *reinterpret_cast<float4 *>(lo) = make_float4(va[0], va[1], va[2], va[3]);
        *reinterpret_cast<float4 *>(hi) = make_float4(vb[0], vb[1], vb[2], vb[3]);
    }
    if (amax) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) m = max(m, __shfl_xor_sync(0xffffffffu, m, o));
        if ((threadIdx.x & 31) == 0) atomicMax(amax + row, m);
    }
}

// scale[row] (holding the absmax bits) becomes s = absmax / qmax, or NaN for a
// row with a non-finite value.
__global__ void scale_kernel(float *scale, int64_t rows, int32_t qmax) {
    const int64_t row = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (row >= rows) return;
    const uint32_t m = __float_as_uint(scale[row]);
    scale[row] = m >= 0x7f800000u ? __int_as_float(0x7fc00000) : __fdiv_rn(__uint_as_float(m), (float)qmax);
}

__global__ void quantize_kernel(uint32_t *out, int64_t ldo, const float *scale, int32_t qmax,
                                const uint32_t *mask, int64_t ldm, uint16_t *planes, int64_t rows) {
    const int64_t row = blockIdx.y;
    const int64_t k = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) * 4;
    const float s = scale[row];
    const bool quant = s == s && s != 0.0f;
    uint32_t *o = out + row * ldo + k;
    const uint4 bits = *reinterpret_cast<const uint4 *>(o);
    const uint32_t in[4] = {bits.x, bits.y, bits.z, bits.w};
    uint32_t code[4];
#pragma unroll
    for (int q = 0; q < 4; q++) {
        const float t = __fadd_rn(__fdiv_rn(__uint_as_float(in[q]), s), 12582912.0f);
        int32_t c = __float_as_int(t) - 0x4B400000;
        c = min(max(c, -qmax), qmax);
        code[q] = quant ? (uint32_t)c : 0u;
    }
    if (mask) {
        const uint4 mk = *reinterpret_cast<const uint4 *>(mask + row * ldm + k);
        code[0] += mk.x; code[1] += mk.y; code[2] += mk.z; code[3] += mk.w;
    }
    *reinterpret_cast<uint4 *>(o) = make_uint4(code[0], code[1], code[2], code[3]);
    if (planes) store_planes<4>(planes + row * 65536 + k, rows * 65536, code);
}

mosaic_status fwht65536(FwhtArgs a, cudaStream_t st) {
    const int64_t rows = a.rows;
    // Pass 1: stages h = 1 .. 16384 on the halves, unscaled, fp32 into y (mode
    // 0) or into `out` (mode 1).
    FwhtArgs h = a;
    h.split = 1;
    h.rows = 2 * rows;
    h.n_pad = kHalf;
    h.mode = 0;
    h.inv_sqrt = 1.0f;
    if (a.mode == 1) {
        h.y = reinterpret_cast<float *>(a.out);
        h.ldy = a.ldo;
    }
    {
        const mosaic_status rc = launch<32, 1024>(h, st);
        if (rc != MOSAIC_OK) return rc;
    }
    float *y = h.y;
    const int64_t ldy = h.ldy;
    const dim3 grid((unsigned)(kHalf / (256 * 4)), (unsigned)rows);
    if (rows > 65535) return MOSAIC_ERR_SHAPE;
    if (a.mode == 0) {
        {
            KernelSpan span("fwht_combine", st);
            combine_kernel<<<grid, 256, 0, st>>>(y, ldy, rows, a.rotate, nullptr);
        }
        return launch_status();
    }
    uint32_t *amax = reinterpret_cast<uint32_t *>(a.scale);
    if (cudaMemsetAsync(amax, 0, sizeof(uint32_t) * (size_t)rows, st) != cudaSuccess) return MOSAIC_ERR_CUDA;
    {
        KernelSpan span("fwht_combine", st);
        combine_kernel<<<grid, 256, 0, st>>>(y, ldy, rows, a.rotate, amax);
    }
    MOSAIC_TRY(launch_status());
    {
        KernelSpan span("fwht_scale", st);
        scale_kernel<<<(unsigned)((rows + 255) / 256), 256, 0, st>>>(a.scale, rows, a.qmax);
    }
    MOSAIC_TRY(launch_status());
    const dim3 g2((unsigned)(65536 / (256 * 4)), (unsigned)rows);
    {
        KernelSpan span("fwht_quantize", st);
        quantize_kernel<<<g2, 256, 0, st>>>(a.out, a.ldo, a.scale, a.qmax, a.mask, a.ldm, a.planes, rows);
    }
    return launch_status();
}

}  // namespace

mosaic_status fwht_encode(const float *x, int64_t ldx, int64_t rows, int64_t n, int64_t n_pad,
                          const uint32_t *sign_words, int rotate, int mode, float *y, int32_t qmax,
                          const uint32_t *mask, int64_t ldm, uint32_t *out, int64_t ldo, float *scale,
                          uint16_t *planes, cudaStream_t st) {
    if (rows == 0) return MOSAIC_OK;
    FwhtArgs a;
    a.x = x; a.ldx = ldx; a.rows = rows; a.n = n; a.n_pad = n_pad;
    a.signs = sign_words; a.rotate = rotate; a.mode = mode;
    a.inv_sqrt = (float)(1.0 / sqrt((double)n_pad));
    a.y = y; a.qmax = qmax; a.mask = mask; a.ldm = ldm; a.out = out; a.ldo = ldo;
    a.scale = scale; a.planes = planes;
    a.vec_x = aligned16(x) && (ldx % 4 == 0);
    a.ldy = n_pad;
    a.split = 0;
    if (n_pad == 65536) return fwht65536(a, st);
    switch (n_pad) {
        case 32: return launch<1, 32>(a, st);
        case 64: return launch<2, 32>(a, st);
        case 128: return launch<4, 32>(a, st);
        case 256: return launch<8, 32>(a, st);
        case 512: return launch<16, 32>(a, st);
        case 1024: return launch<16, 64>(a, st);
        case 2048: return launch<16, 128>(a, st);
        case 4096: return launch<16, 256>(a, st);
        case 8192: return launch<32, 256>(a, st);
        case 16384:
            if (!stream_ok(a)) return launch<32, 512>(a, st);
            return a.mode == 0 ? launch_rot<512>(a, st) : launch_pair(a, st);
        case 32768:
            if (!stream_ok(a)) return launch<32, 1024>(a, st);
            return a.mode == 0 ? launch_rot<1024>(a, st) : launch_stream<1024>(a, st);
        default: return MOSAIC_ERR_SHAPE;
    }
}

mosaic_status fwht_status() {
    uint32_t v = 0, zero = 0;
    if (cudaMemcpyFromSymbol(&v, g_fwht_error, sizeof v) != cudaSuccess) return MOSAIC_ERR_CUDA;
    if (v) {
        cudaMemcpyToSymbol(g_fwht_error, &zero, sizeof zero);
        return MOSAIC_ERR_TIMEOUT;
    }
    return MOSAIC_OK;
}

}  // namespace mosaic
