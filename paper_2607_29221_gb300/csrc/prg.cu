// Counter-mode ChaCha PRG and the samplers of the masks (Sec. 3.2 protocol
// box: uniform L, M_i, N_i, R; discrete Gaussian E_w, E_x with
// Pr[k] ~ exp(-k^2 / (2 sigma^2)) (Sec. 3.1); sparse S_i, T_i of Hamming
// weight t (Example 3.1)).
#include <math.h>

#include "mosaic_internal.cuh"

namespace mosaic {
namespace {

constexpr int kThreads = 256;

// One thread per 64-byte ChaCha block: 16 consecutive stream words.
// Stream id of a launch: sid, plus *sid_dev when given (read on the device,
// so that a captured graph draws a fresh stream on every replay).
__device__ __forceinline__ void stream_id(uint64_t sid, const uint64_t *sid_dev, uint32_t &lo, uint32_t &hi) {
    const uint64_t s = sid + (sid_dev ? *sid_dev : 0ull);
    lo = (uint32_t)s;
    hi = (uint32_t)(s >> 32);
}

// Uniform words of a rows x cols matrix in stream order (row-major), thread
// `first` of `stride` threads; with `planes`, also its tensor-core digit
// planes [4][rows][ldp] (bf16, plane stride `pstride`).
__device__ __forceinline__ void uniform_body(const Key &key, uint32_t tag, uint32_t sid_lo, uint32_t sid_hi,
                                             int rounds, int64_t cols, int64_t total, uint32_t *out, int64_t ldo,
                                             uint16_t *planes, int64_t ldp, int64_t pstride, int64_t first,
                                             int64_t stride) {
    const int64_t nblk = (total + 15) / 16;
    for (int64_t b = first; b < nblk; b += stride) {
        uint32_t w[16];
        chacha_block(key, (uint32_t)b, tag, sid_lo, sid_hi, rounds, w);
        int64_t word = b * 16;
        int64_t r = word / cols, c = word - r * cols;
#pragma unroll
        for (int i = 0; i < 16; i++) {
            if (word + i < total) {
                out[r * ldo + c] = w[i];
                if (planes) {
#pragma unroll
                    for (int d = 0; d < 4; d++) planes[d * pstride + r * ldp + c] = (uint16_t)digit_bits(w[i], d);
                }
                if (++c == cols) { c = 0; ++r; }
            }
        }
    }
}

__global__ void uniform_kernel(Key key, uint32_t tag, uint64_t sid, const uint64_t *sid_dev, int rounds,
                               int64_t cols, int64_t total, uint32_t *out, int64_t ldo) {
    uint32_t sid_lo, sid_hi;
    stream_id(sid, sid_dev, sid_lo, sid_hi);
    uniform_body(key, tag, sid_lo, sid_hi, rounds, cols, total, out, ldo, nullptr, 0, 0,
                 blockIdx.x * (int64_t)blockDim.x + threadIdx.x, (int64_t)gridDim.x * blockDim.x);
}

struct GaussTable {
    unsigned long long t[2 * kMaxGaussBound + 1];
    int n;        // 2B + 1
    int bound;    // B
};

// One thread per block: 8 samples, each from two consecutive words.  The
// sample is k = (number of table entries <= u) - B, capped at B, i.e. the
// smallest k_j with u < table[j] (table is non-decreasing).  The count is
// found by binary lifting over the sorted table: pos grows by each power of
// two (largest first) while the entry just below pos + step is still <= u.
// Samples [8 first, ...) of the Gaussian stream, `stride` threads; st = the
// table in shared memory (tab.n entries), top = largest power of two <= n.
// tab.n == 0 writes zeros (sigma = 0).
__device__ __forceinline__ void gaussian_body(const Key &key, uint32_t tag, uint32_t sid_lo, uint32_t sid_hi,
                                              int rounds, const unsigned long long *st, int n, int bound, int top,
                                              int64_t count, uint32_t *out, int64_t first, int64_t stride) {
    const int64_t nblk = (count + 7) / 8;
    for (int64_t b = first; b < nblk; b += stride) {
        uint32_t res[8];
        if (n == 0) {
#pragma unroll
            for (int i = 0; i < 8; i++) res[i] = 0u;
        } else {
            uint32_t w[16];
            chacha_block(key, (uint32_t)b, tag, sid_lo, sid_hi, rounds, w);
#pragma unroll
            for (int i = 0; i < 8; i++) {
                const unsigned long long u = (unsigned long long)w[2 * i] | ((unsigned long long)w[2 * i + 1] << 32);
                int cnt = 0;
                for (int step = top; step > 0; step >>= 1)
                    if (cnt + step <= n && st[cnt + step - 1] <= u) cnt += step;
                if (cnt > 2 * bound) cnt = 2 * bound;
                res[i] = (uint32_t)(cnt - bound);
            }
        }
        const int64_t e0 = b * 8;
        if (e0 + 8 <= count && ((reinterpret_cast<uintptr_t>(out + e0) & 15u) == 0)) {
            reinterpret_cast<uint4 *>(out + e0)[0] = make_uint4(res[0], res[1], res[2], res[3]);
            reinterpret_cast<uint4 *>(out + e0)[1] = make_uint4(res[4], res[5], res[6], res[7]);
        } else {
            for (int i = 0; i < 8; i++)
                if (e0 + i < count) out[e0 + i] = res[i];
        }
    }
}
__device__ __forceinline__ int pow2_floor(int n) {
    int top = 1;
    while (2 * top <= n) top *= 2;
    return top;
}

__global__ void gaussian_kernel(Key key, uint32_t tag, uint64_t sid, const uint64_t *sid_dev, int rounds,
                                GaussTable tab, int64_t count, uint32_t *out) {
    __shared__ unsigned long long st[2 * kMaxGaussBound + 1];
    uint32_t sid_lo, sid_hi;
    stream_id(sid, sid_dev, sid_lo, sid_hi);
    for (int i = threadIdx.x; i < tab.n; i += blockDim.x) st[i] = tab.t[i];
    __syncthreads();
    gaussian_body(key, tag, sid_lo, sid_hi, rounds, st, tab.n, tab.bound, pow2_floor(tab.n), count, out,
                  blockIdx.x * (int64_t)blockDim.x + threadIdx.x, (int64_t)gridDim.x * blockDim.x);
}

// One warp per sparse row; the row's window starts at block row * 4096.
// Each round the 32 lanes compute 32 consecutive ChaCha blocks (512 words),
// which are then consumed in stream order, 32 words at a time: a word's
// position is accepted if it is not in the row's bitmap and no lower lane of
// the batch drew the same position (warp match), which is exactly the
// sequential "skip repeats" rule; after the t-th accepted position the
// following words are values (zero words skipped).
constexpr int kSparseWarps = 4;

// Row j of the sparse matrix by one warp; sm_warp = the warp's 512 + bitmap_words words.
__device__ __forceinline__ void sparse_row(const Key &key, uint32_t tag, uint32_t sid_lo, uint32_t sid_hi,
                                           int rounds, int64_t j, uint32_t r, int t, uint32_t *idx, uint32_t *val,
                                           uint32_t *fail, int bitmap_words, uint32_t *sm_warp, bool lines = false) {
    const int lane = threadIdx.x & 31;
    uint32_t *words = sm_warp;
    uint32_t *bits = words + 512;
    for (int w = lane; w < bitmap_words; w += 32) bits[w] = 0u;
    __syncwarp();
    uint32_t *ri = idx + j * t;
    uint32_t *rv = val + j * t;
    const unsigned lt_mask = (1u << lane) - 1u;
    int got = 0, nv = 0;
    const uint32_t blk0 = (uint32_t)(j * (kSparseWindow / 16));
    for (int round = 0; round < kSparseWindow / 512 && nv < t; ++round) {
        uint32_t w16[16];
        chacha_block(key, blk0 + round * 32 + lane, tag, sid_lo, sid_hi, rounds, w16);
#pragma unroll
        for (int i = 0; i < 16; i++) words[lane * 16 + i] = w16[i];
        __syncwarp();
        for (int b = 0; b < 16 && nv < t; ++b) {
            const uint32_t w = words[b * 32 + lane];
            int val_start = 0;
            if (got < t) {
                const uint32_t p = (uint32_t)(((unsigned long long)w * r) >> 32);
                const bool taken = (bits[p >> 5] >> (p & 31)) & 1u;
                const unsigned same = __match_any_sync(0xffffffffu, p);
                const bool first = (__ffs(same) - 1) == lane;
                unsigned acc = __ballot_sync(0xffffffffu, !taken && first);
                const int need = t - got;
                val_start = 32;
                if (__popc(acc) >= need) {
                    unsigned m = acc;
                    for (int k = 1; k < need; ++k) m &= m - 1u;
                    const int last = __ffs(m) - 1;
                    acc &= last == 31 ? 0xffffffffu : ((2u << last) - 1u);
                    val_start = last + 1;
                }
                if ((acc >> lane) & 1u) {
                    ri[got + __popc(acc & lt_mask)] = lines ? pg_line(p) : p;
                    atomicOr(&bits[p >> 5], 1u << (p & 31));
                }
                got += __popc(acc);
                __syncwarp();
            }
            if (got >= t && val_start < 32) {
                unsigned accv = __ballot_sync(0xffffffffu, lane >= val_start && w != 0u);
                const int needv = t - nv;
                if (__popc(accv) > needv) {
                    unsigned m = accv;
                    for (int k = 0; k < needv; ++k) m &= m - 1u;
                    accv &= ~m;
                }
                if ((accv >> lane) & 1u) rv[nv + __popc(accv & lt_mask)] = w;
                nv += __popc(accv);
            }
        }
        __syncwarp();
    }
    if (nv < t) {
        for (int q = got + lane; q < t; q += 32) ri[q] = 0u;
        for (int q = nv + lane; q < t; q += 32) rv[q] = 0u;
        if (lane == 0 && fail) atomicExch(fail, 1u);
    }
}

__global__ void __launch_bounds__(kSparseWarps * 32)
    sparse_kernel(Key key, uint32_t tag, uint64_t sid, const uint64_t *sid_dev, int rounds, int64_t rows,
                  uint32_t r, int t, uint32_t *idx, uint32_t *val, uint32_t *fail, int bitmap_words) {
    extern __shared__ uint32_t sm[];
    uint32_t sid_lo, sid_hi;
    stream_id(sid, sid_dev, sid_lo, sid_hi);
    const int warp = threadIdx.x >> 5;
    const int64_t j = (int64_t)blockIdx.x * kSparseWarps + warp;
    if (j >= rows) return;
    sparse_row(key, tag, sid_lo, sid_hi, rounds, j, r, t, idx, val, fail, bitmap_words,
               sm + warp * (512 + bitmap_words));
}

// All draws of one Init X call in one launch (blocks of 128 threads, split
// by role so that the short draws run beside the long Gaussian one): R (and
// optionally its digit planes), the d - 1 sparse T lists, E_x.
struct InitxDraws {
    Key key;
    int rounds;
    uint64_t sid;
    const uint64_t *sid_dev;
    uint32_t tagR;
    int64_t r_cols, r_total;
    uint32_t *R;
    int64_t ldr;
    uint16_t *Rp;
    int64_t ldp, pstride;
    int nlev;
    uint32_t tagT[2], rT[2];
    int tT[2];
    int64_t rowsT;
    uint32_t *idx[2], *val[2];
    int bitmap_words;
    uint32_t tagE;
    int64_t ecount;
    uint32_t *E;
    GaussTable tab;
    int nbU, nbS, nbG;   // blocks per role (nbS per sparse level)
    int lines;           // lists hold pg_line(position)
};
constexpr int kDrawThreads = kSparseWarps * 32;

__global__ void __launch_bounds__(kDrawThreads) initx_draw_kernel(InitxDraws a) {
    extern __shared__ uint32_t sm[];
    uint32_t sid_lo, sid_hi;
    stream_id(a.sid, a.sid_dev, sid_lo, sid_hi);
    int blk = blockIdx.x;
    if (blk < a.nbU) {
        uniform_body(a.key, a.tagR, sid_lo, sid_hi, a.rounds, a.r_cols, a.r_total, a.R, a.ldr, a.Rp, a.ldp,
                     a.pstride, (int64_t)blk * kDrawThreads + threadIdx.x, (int64_t)a.nbU * kDrawThreads);
        return;
    }
    blk -= a.nbU;
    if (blk < a.nlev * a.nbS) {
        const int lv = blk / a.nbS;
        const int warp = threadIdx.x >> 5;
        const int64_t j = (int64_t)(blk - lv * a.nbS) * kSparseWarps + warp;
        if (j >= a.rowsT) return;
        sparse_row(a.key, a.tagT[lv], sid_lo, sid_hi, a.rounds, j, a.rT[lv], a.tT[lv], a.idx[lv], a.val[lv],
                   nullptr, a.bitmap_words, sm + warp * (512 + a.bitmap_words), a.lines != 0);
        return;
    }
    blk -= a.nlev * a.nbS;
    unsigned long long *st = reinterpret_cast<unsigned long long *>(sm);
    for (int i = threadIdx.x; i < a.tab.n; i += blockDim.x) st[i] = a.tab.t[i];
    __syncthreads();
    gaussian_body(a.key, a.tagE, sid_lo, sid_hi, a.rounds, st, a.tab.n, a.tab.bound,
                  a.tab.n ? pow2_floor(a.tab.n) : 0, a.ecount, a.E, (int64_t)blk * kDrawThreads + threadIdx.x,
                  (int64_t)a.nbG * kDrawThreads);
}

// Sampler grids: one thread per ChaCha block, up to 152 x 64 blocks.
int prg_blocks(int64_t items, int threads) {
    int64_t g = (items + threads - 1) / threads;
    if (g < 1) g = 1;
    if (g > 152 * 64) g = 152 * 64;
    return (int)g;
}

}  // namespace

int gaussian_table_host(float sigma, unsigned long long *table) {
    const int B = (int)ceil(12.0 * (double)sigma);
    const long double s = (long double)sigma;
    long double w[2 * kMaxGaussBound + 1];
    long double z = 0.0L;
    for (int k = -B; k <= B; k++) {
        w[k + B] = expl(-((long double)k * (long double)k) / (2.0L * s * s));
        z += w[k + B];
    }
    const long double two64 = 18446744073709551616.0L;
    long double acc = 0.0L;
    for (int j = 0; j < 2 * B + 1; j++) {
        acc += w[j];
        long double v = floorl(acc / z * two64);
        table[j] = v >= two64 ? ~0ull : (unsigned long long)v;
    }
    table[2 * B] = ~0ull;   // the full CDF saturates
    return B;
}

mosaic_status prg_uniform(const Key &key, uint32_t tag, uint64_t sid, int rounds, int64_t rows,
                          int64_t cols, uint32_t *out, int64_t ldo, cudaStream_t st, const uint64_t *sid_dev) {
    const int64_t total = rows * cols;
    if (total == 0) return MOSAIC_OK;
    const int64_t nblk = (total + 15) / 16;
    {
        KernelSpan span("prg_uniform", st);
        uniform_kernel<<<prg_blocks(nblk, kThreads), kThreads, 0, st>>>(
            key, tag, sid, sid_dev, rounds, cols, total, out, ldo);
    }
    return launch_status();
}

mosaic_status prg_gaussian(const Key &key, uint32_t tag, uint64_t sid, int rounds, float sigma,
                           int64_t count, uint32_t *out, cudaStream_t st, const uint64_t *sid_dev) {
    if (count == 0) return MOSAIC_OK;
    if (sigma == 0.0f) {
        return cudaMemsetAsync(out, 0, sizeof(uint32_t) * (size_t)count, st) == cudaSuccess
                   ? MOSAIC_OK : MOSAIC_ERR_CUDA;
    }
    GaussTable tab;
    tab.bound = gaussian_table_host(sigma, tab.t);
    tab.n = 2 * tab.bound + 1;
    const int64_t nblk = (count + 7) / 8;
    {
        KernelSpan span("prg_gaussian", st);
        gaussian_kernel<<<prg_blocks(nblk, kThreads), kThreads, 0, st>>>(
            key, tag, sid, sid_dev, rounds, tab, count, out);
    }
    return launch_status();
}

mosaic_status prg_initx(const Key &key, int rounds, uint64_t sid, const uint64_t *sid_dev, uint32_t tagR,
                        int64_t l, int64_t rd, uint32_t *R, uint16_t *Rp, int64_t Kp, int nlev, const uint32_t *tagT,
                        const uint32_t *rT, const uint32_t *tT, uint32_t *const *idx, uint32_t *const *val,
                        uint32_t tagE, float sigma, int64_t ecount, uint32_t *E, cudaStream_t st, bool lines) {
    if (l == 0) return MOSAIC_OK;
    if (nlev < 0 || nlev > 2) return MOSAIC_ERR_UNSUPPORTED;
    InitxDraws a{};
    a.key = key;
    a.rounds = rounds;
    a.sid = sid;
    a.sid_dev = sid_dev;
    a.tagR = tagR;
    a.r_cols = rd;
    a.r_total = l * rd;
    a.R = R;
    a.ldr = rd;
    a.Rp = Rp;
    a.ldp = Kp;
    a.pstride = l * Kp;
    a.nlev = nlev;
    a.rowsT = l;
    a.lines = lines ? 1 : 0;
    uint32_t rmax = 1;
    for (int i = 0; i < nlev; i++) {
        a.tagT[i] = tagT[i];
        a.rT[i] = rT[i];
        a.tT[i] = (int)tT[i];
        a.idx[i] = idx[i];
        a.val[i] = val[i];
        rmax = rT[i] > rmax ? rT[i] : rmax;
    }
    a.bitmap_words = (int)((rmax + 31) / 32);
    a.tagE = tagE;
    a.ecount = ecount;
    a.E = E;
    if (sigma != 0.0f) {
        a.tab.bound = gaussian_table_host(sigma, a.tab.t);
        a.tab.n = 2 * a.tab.bound + 1;
    } else {
        a.tab.bound = a.tab.n = 0;
    }
    const int64_t cap = 152 * 64;
    auto blocks = [&](int64_t threads_needed) {
        int64_t b = (threads_needed + kDrawThreads - 1) / kDrawThreads;
        return (int)(b < 1 ? 1 : b > cap ? cap : b);
    };
    a.nbU = blocks((a.r_total + 15) / 16);
    a.nbS = (int)((l + kSparseWarps - 1) / kSparseWarps);
    a.nbG = ecount > 0 ? blocks((ecount + 7) / 8) : 0;
    const int64_t grid = (int64_t)a.nbU + (int64_t)nlev * a.nbS + a.nbG;
    if (grid > 0x7fffffff) return MOSAIC_ERR_SHAPE;
    size_t smem = nlev > 0 ? (size_t)kSparseWarps * (512 + a.bitmap_words) * sizeof(uint32_t) : 0;
    const size_t tab_bytes = (size_t)(2 * kMaxGaussBound + 1) * sizeof(unsigned long long);
    if (smem < tab_bytes) smem = tab_bytes;
    if (smem > 48 * 1024 &&
        cudaFuncSetAttribute(initx_draw_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
            cudaSuccess)
        return MOSAIC_ERR_CUDA;
    {
        KernelSpan span("initx_draw", st);
        initx_draw_kernel<<<(unsigned)grid, kDrawThreads, smem, st>>>(a);
    }
    return launch_status();
}

mosaic_status prg_sparse(const Key &key, uint32_t tag, uint64_t sid, int rounds, int64_t rows,
                         uint32_t r, uint32_t t, uint32_t *idx, uint32_t *val, uint32_t *fail,
                         cudaStream_t st, const uint64_t *sid_dev) {
    if (rows == 0) return MOSAIC_OK;
    const int bitmap_words = (int)((r + 31) / 32);
    const size_t smem = (size_t)kSparseWarps * (512 + bitmap_words) * sizeof(uint32_t);
    if (smem > 48 * 1024 &&
        cudaFuncSetAttribute(sparse_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
            cudaSuccess)
        return MOSAIC_ERR_CUDA;
    {
        KernelSpan span("prg_sparse", st);
        sparse_kernel<<<(unsigned)((rows + kSparseWarps - 1) / kSparseWarps), kSparseWarps * 32, smem, st>>>(
            key, tag, sid, sid_dev, rounds, rows, r, (int)t, idx, val, fail, bitmap_words);
    }
    return launch_status();
}

}  // namespace mosaic

namespace mosaic {
namespace {
__global__ void add_u64_kernel(uint64_t *p, uint64_t delta) { *p += delta; }
}  // namespace

mosaic_status add_u64(uint64_t *p, uint64_t delta, cudaStream_t st) {
    add_u64_kernel<<<1, 1, 0, st>>>(p, delta);
    return launch_status();
}
}  // namespace mosaic
