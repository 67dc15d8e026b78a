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
__global__ void uniform_kernel(Key key, uint32_t tag, uint32_t sid_lo, uint32_t sid_hi, int rounds,
                               int64_t cols, int64_t total, uint32_t *out, int64_t ldo) {
    const int64_t nblk = (total + 15) / 16;
    for (int64_t b = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; b < nblk;
         b += (int64_t)gridDim.x * blockDim.x) {
        uint32_t w[16];
        chacha_block(key, (uint32_t)b, tag, sid_lo, sid_hi, rounds, w);
        int64_t word = b * 16;
        int64_t r = word / cols, c = word - r * cols;
#pragma unroll
        for (int i = 0; i < 16; i++) {
            if (word + i < total) {
                out[r * ldo + c] = w[i];
                if (++c == cols) { c = 0; ++r; }
            }
        }
    }
}

struct GaussTable {
    unsigned long long t[2 * kMaxGaussBound + 1];
    int n;        // 2B + 1
    int bound;    // B
};

// One thread per block: 8 samples, each from two consecutive words.  The
// sample is k = (number of table entries <= u) - B, capped at B, i.e. the
// smallest k_j with u < table[j] (table is non-decreasing).
__global__ void gaussian_kernel(Key key, uint32_t tag, uint32_t sid_lo, uint32_t sid_hi, int rounds,
                                GaussTable tab, int64_t count, uint32_t *out) {
    __shared__ unsigned long long st[2 * kMaxGaussBound + 1];
    for (int i = threadIdx.x; i < tab.n; i += blockDim.x) st[i] = tab.t[i];
    __syncthreads();
    const int64_t nblk = (count + 7) / 8;
    for (int64_t b = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; b < nblk;
         b += (int64_t)gridDim.x * blockDim.x) {
        uint32_t w[16];
        chacha_block(key, (uint32_t)b, tag, sid_lo, sid_hi, rounds, w);
        uint32_t res[8];
#pragma unroll
        for (int i = 0; i < 8; i++) {
            const unsigned long long u = (unsigned long long)w[2 * i] | ((unsigned long long)w[2 * i + 1] << 32);
            int cnt = 0;
            for (int j = 0; j < tab.n; j++) cnt += (st[j] <= u) ? 1 : 0;
            if (cnt > 2 * tab.bound) cnt = 2 * tab.bound;
            res[i] = (uint32_t)(cnt - tab.bound);
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

// One thread per sparse row; the row's window starts at block row * 4096.
__global__ void sparse_kernel(Key key, uint32_t tag, uint32_t sid_lo, uint32_t sid_hi, int rounds,
                              int64_t rows, uint32_t r, int t, uint32_t *idx, uint32_t *val,
                              uint32_t *fail) {
    const int64_t j = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    if (j >= rows) return;
    uint32_t *ri = idx + j * t;
    uint32_t *rv = val + j * t;
    int got = 0, nv = 0;
    const uint32_t blk0 = (uint32_t)(j * (kSparseWindow / 16));
    for (int bi = 0; bi < kSparseWindow / 16 && nv < t; bi++) {
        uint32_t w[16];
        chacha_block(key, blk0 + bi, tag, sid_lo, sid_hi, rounds, w);
#pragma unroll
        for (int i = 0; i < 16; i++) {
            if (got < t) {
                const uint32_t p = (uint32_t)(((unsigned long long)w[i] * r) >> 32);
                bool seen = false;
                for (int q = 0; q < got; q++) seen |= (ri[q] == p);
                if (!seen) ri[got++] = p;
            } else if (nv < t) {
                if (w[i] != 0u) rv[nv++] = w[i];
            }
        }
    }
    if (nv < t) {
        for (int q = got; q < t; q++) ri[q] = 0;
        for (int q = nv; q < t; q++) rv[q] = 0;
        if (fail) atomicExch(fail, 1u);
    }
}

int grid_for(int64_t items, int threads) {
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
                          int64_t cols, uint32_t *out, int64_t ldo, cudaStream_t st) {
    const int64_t total = rows * cols;
    if (total == 0) return MOSAIC_OK;
    const int64_t nblk = (total + 15) / 16;
    uniform_kernel<<<grid_for(nblk, kThreads), kThreads, 0, st>>>(
        key, tag, (uint32_t)sid, (uint32_t)(sid >> 32), rounds, cols, total, out, ldo);
    return launch_status();
}

mosaic_status prg_gaussian(const Key &key, uint32_t tag, uint64_t sid, int rounds, float sigma,
                           int64_t count, uint32_t *out, cudaStream_t st) {
    if (count == 0) return MOSAIC_OK;
    if (sigma == 0.0f) {
        return cudaMemsetAsync(out, 0, sizeof(uint32_t) * (size_t)count, st) == cudaSuccess
                   ? MOSAIC_OK : MOSAIC_ERR_CUDA;
    }
    GaussTable tab;
    tab.bound = gaussian_table_host(sigma, tab.t);
    tab.n = 2 * tab.bound + 1;
    const int64_t nblk = (count + 7) / 8;
    gaussian_kernel<<<grid_for(nblk, kThreads), kThreads, 0, st>>>(
        key, tag, (uint32_t)sid, (uint32_t)(sid >> 32), rounds, tab, count, out);
    return launch_status();
}

mosaic_status prg_sparse(const Key &key, uint32_t tag, uint64_t sid, int rounds, int64_t rows,
                         uint32_t r, uint32_t t, uint32_t *idx, uint32_t *val, uint32_t *fail,
                         cudaStream_t st) {
    if (rows == 0) return MOSAIC_OK;
    const int threads = 64;
    sparse_kernel<<<(unsigned)((rows + threads - 1) / threads), threads, 0, st>>>(
        key, tag, (uint32_t)sid, (uint32_t)(sid >> 32), rounds, rows, r, (int)t, idx, val, fail);
    return launch_status();
}

}  // namespace mosaic
