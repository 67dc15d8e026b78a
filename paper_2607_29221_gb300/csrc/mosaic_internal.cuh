// Internal declarations shared by the library's translation units.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

#include "../../include/mosaic.h"

namespace mosaic {

// Raises `kern`'s dynamic shared-memory limit to `bytes` on the current device,
// once per device ordinal (`done` holds one bit per ordinal).  Host threads may
// race on a first call: each may set the attribute (an idempotent runtime call)
// and the bit is published atomically.
template <typename Kernel>
inline bool ensure_smem_limit(std::atomic<unsigned long long> &done, Kernel kern, size_t bytes, int *dev_out = nullptr) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return false;
    if (dev_out) *dev_out = dev;
    const unsigned long long bit = 1ull << (dev & 63);
    if (done.load(std::memory_order_acquire) & bit) return true;
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes) != cudaSuccess)
        return false;
    done.fetch_or(bit, std::memory_order_acq_rel);
    return true;
}

constexpr int kSparseWindow = 65536;   // stream words reserved per sparse row
constexpr int kMaxGaussBound = 96;     // B = ceil(12 sigma) for sigma <= 8

// ChaCha quarter round and block (RFC 8439 Sec. 2.1-2.3).
__device__ __forceinline__ uint32_t rotl(uint32_t v, int c) { return __funnelshift_l(v, v, c); }

#define MOSAIC_QR(a, b, c, d)             \
    a += b; d ^= a; d = rotl(d, 16);      \
    c += d; b ^= c; b = rotl(b, 12);      \
    a += b; d ^= a; d = rotl(d, 8);       \
    c += d; b ^= c; b = rotl(b, 7);

struct Key {
    uint32_t k[8];
};

// Block `ctr` of stream (n0, n1, n2) -> 16 words in `o`.
__device__ __forceinline__ void chacha_block(const Key &key, uint32_t ctr, uint32_t n0, uint32_t n1,
                                             uint32_t n2, int rounds, uint32_t o[16]) {
    uint32_t x0 = 0x61707865u, x1 = 0x3320646eu, x2 = 0x79622d32u, x3 = 0x6b206574u;
    uint32_t x4 = key.k[0], x5 = key.k[1], x6 = key.k[2], x7 = key.k[3];
    uint32_t x8 = key.k[4], x9 = key.k[5], x10 = key.k[6], x11 = key.k[7];
    uint32_t x12 = ctr, x13 = n0, x14 = n1, x15 = n2;
    for (int r = 0; r < rounds; r += 2) {
        MOSAIC_QR(x0, x4, x8, x12);
        MOSAIC_QR(x1, x5, x9, x13);
        MOSAIC_QR(x2, x6, x10, x14);
        MOSAIC_QR(x3, x7, x11, x15);
        MOSAIC_QR(x0, x5, x10, x15);
        MOSAIC_QR(x1, x6, x11, x12);
        MOSAIC_QR(x2, x7, x8, x13);
        MOSAIC_QR(x3, x4, x9, x14);
    }
    o[0] = x0 + 0x61707865u; o[1] = x1 + 0x3320646eu; o[2] = x2 + 0x79622d32u; o[3] = x3 + 0x6b206574u;
    o[4] = x4 + key.k[0]; o[5] = x5 + key.k[1]; o[6] = x6 + key.k[2]; o[7] = x7 + key.k[3];
    o[8] = x8 + key.k[4]; o[9] = x9 + key.k[5]; o[10] = x10 + key.k[6]; o[11] = x11 + key.k[7];
    o[12] = x12 + ctr; o[13] = x13 + n0; o[14] = x14 + n1; o[15] = x15 + n2;
}

// Digit d of a as the bf16 bits of the signed value byte_d(a + 0x80808080) - 128
// (a = sum_d digit_d 2^(8d) mod 2^32); the tensor-core operands' digit planes.
__device__ __forceinline__ uint32_t digit_bits(uint32_t a, int d) {
    const int dig = (int)(((a + 0x80808080u) >> (8 * d)) & 0xffu) - 128;
    return __bfloat16_as_ushort(__float2bfloat16_rn((float)dig));
}

inline Key to_key(const mosaic_key *k) {
    Key r;
    for (int i = 0; i < 8; i++) r.k[i] = k->key[i];
    return r;
}

inline cudaStream_t as_stream(void *s) { return reinterpret_cast<cudaStream_t>(s); }

// Counts every kernel this library launches (read by mosaic_kernel_launches).
void count_launch();

inline mosaic_status launch_status() {
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return MOSAIC_ERR_CUDA;
    count_launch();
    return MOSAIC_OK;
}

// Optional per-kernel device timing (mosaic_kernel_timing).  A launcher opens
// a KernelSpan right before its launch and lets it close after; while timing
// is on and `st` is not being captured, the span brackets the launch with a
// CUDA event pair keyed by "<role>:<kernel>", the role being the entry point
// that made the call (set by a RoleScope there).
struct KernelSpan {
    KernelSpan(const char *kernel, cudaStream_t st);
    ~KernelSpan();
    KernelSpan(const KernelSpan &) = delete;
    KernelSpan &operator=(const KernelSpan &) = delete;
    void *slot_ = nullptr;
    cudaStream_t st_;
};
struct RoleScope {
    explicit RoleScope(const char *role);
    ~RoleScope();
    RoleScope(const RoleScope &) = delete;
    RoleScope &operator=(const RoleScope &) = delete;
    const char *prev_;
};

#define MOSAIC_TRY(expr)                        \
    do {                                        \
        mosaic_status _s = (expr);              \
        if (_s != MOSAIC_OK) return _s;         \
    } while (0)

inline bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
inline bool is_pow2(int64_t v) { return v > 0 && (v & (v - 1)) == 0; }
// Blocks for a grid-stride loop over `items`: enough to fill the GPU a few
// times over, at most 152 x 32.
inline int grid_for(int64_t items, int threads) {
    int64_t g = (items + threads - 1) / threads;
    if (g < 1) g = 1;
    if (g > 152 * 32) g = 152 * 32;
    return (int)g;
}

// ---- internal launchers (all enqueue on `st`, validate nothing beyond what they state) ----

// The samplers draw from stream id sid + (*sid_dev if sid_dev is given; read
// on the device when the kernel runs).
// Uniform words: out[i * ldo + j] = word (i * cols + j).
mosaic_status prg_uniform(const Key &key, uint32_t tag, uint64_t sid, int rounds, int64_t rows,
                          int64_t cols, uint32_t *out, int64_t ldo, cudaStream_t st,
                          const uint64_t *sid_dev = nullptr);
// Discrete Gaussian elements.
mosaic_status prg_gaussian(const Key &key, uint32_t tag, uint64_t sid, int rounds, float sigma,
                           int64_t count, uint32_t *out, cudaStream_t st, const uint64_t *sid_dev = nullptr);
// Sparse rows.
// All draws of an Init X call in one launch: R (l x rd, and its digit planes
// [4][l][Kp] when Rp is not null), nlev <= 2 sparse lists (l rows each) and
// the Gaussian E (ecount samples), each exactly as the single samplers draw it.
// With `lines`, the lists hold pg_line(position) instead of the position.
mosaic_status prg_initx(const Key &key, int rounds, uint64_t sid, const uint64_t *sid_dev, uint32_t tagR,
                        int64_t l, int64_t rd, uint32_t *R, uint16_t *Rp, int64_t Kp, int nlev, const uint32_t *tagT,
                        const uint32_t *rT, const uint32_t *tT, uint32_t *const *idx, uint32_t *const *val,
                        uint32_t tagE, float sigma, int64_t ecount, uint32_t *E, cudaStream_t st, bool lines = false);
mosaic_status prg_sparse(const Key &key, uint32_t tag, uint64_t sid, int rounds, int64_t rows,
                         uint32_t r, uint32_t t, uint32_t *idx, uint32_t *val, uint32_t *fail,
                         cudaStream_t st, const uint64_t *sid_dev = nullptr);
// *p += delta on the stream (advances a device-side pass counter).
mosaic_status add_u64(uint64_t *p, uint64_t delta, cudaStream_t st);
// Host-side Gaussian CDF table (long double), B = ceil(12 sigma); returns B.
int gaussian_table_host(float sigma, unsigned long long *table /* 2*kMaxGaussBound+1 */);

// FWHT / encode.
mosaic_status fwht_encode(const float *x, int64_t ldx, int64_t rows, int64_t n, int64_t n_pad,
                          const uint32_t *sign_words, int rotate, int mode /*0 hadamard,1 encode*/,
                          float *y, int32_t qmax, const uint32_t *mask, int64_t ldm, uint32_t *out,
                          int64_t ldo, float *scale, uint16_t *planes, cudaStream_t st);

// Reads and clears the streamed rotation's timeout word (after a stream sync).
mosaic_status fwht_status();

// Generic strided ring GEMM on CUDA cores:
// C[i*ldc + j] = (Cin ? Cin[i*ldcin + j] : 0) + sgn * sum_k A[i*sai + k*sak] * B[j*sbj + k*sbk]
mosaic_status ring_gemm_imad(const uint32_t *A, int64_t sai, int64_t sak, const uint32_t *B,
                             int64_t sbj, int64_t sbk, uint32_t *C, int64_t ldc,
                             const uint32_t *Cin, int64_t ldcin, int sgn, int64_t M, int64_t N,
                             int64_t K, cudaStream_t st);

// Digit planes.
mosaic_status digit_split(const uint32_t *a, int64_t lda, int64_t rows, int64_t cols,
                          uint16_t *planes, int64_t ldp, int64_t plane_stride, cudaStream_t st);

// Tensor-core ring GEMM from planes (NT, K-major planes); C = (Cin?) + sgn * A B^T.
mosaic_status ring_gemm_tc_planes(const uint16_t *Ap, int64_t ldpa, int64_t a_plane,
                                  const uint16_t *Bp, int64_t ldpb, int64_t b_plane, uint32_t *C,
                                  int64_t ldc, const uint32_t *Cin, int64_t ldcin, int sgn,
                                  int64_t M, int64_t N, int64_t K, cudaStream_t st);
// The same with two outputs side by side in B's rows: columns [0, N1) of the
// product go to C1 (+ Cin1), columns [N1, N1 + N2) to C2 (+ Cin2); N1 is a
// multiple of 128 and K > 0.
mosaic_status ring_gemm_tc_planes2(const uint16_t *Ap, int64_t ldpa, int64_t a_plane, const uint16_t *Bp,
                                   int64_t ldpb, int64_t b_plane, uint32_t *C1, int64_t ldc1,
                                   const uint32_t *Cin1, int64_t ldcin1, int64_t N1, uint32_t *C2, int64_t ldc2,
                                   const uint32_t *Cin2, int64_t ldcin2, int64_t N2, int64_t M, int64_t K,
                                   cudaStream_t st);
// C = Cin - Csub + sgn * A B^T from planes, one output (K > 0; never split
// into stream-K units).
mosaic_status ring_gemm_tc_planes_diff(const uint16_t *Ap, int64_t ldpa, int64_t a_plane, const uint16_t *Bp,
                                       int64_t ldpb, int64_t b_plane, uint32_t *C, int64_t ldc,
                                       const uint32_t *Cin, int64_t ldcin, const uint32_t *Csub, int64_t ldcsub,
                                       int sgn, int64_t M, int64_t N, int64_t K, cudaStream_t st);
// Legacy mma.sync s8 ring GEMM (NT, uint32 operands split into int8 digit
// planes in ws, at least ws_mma_s8(M, N, K) bytes).
size_t ws_mma_s8(int64_t M, int64_t N, int64_t K);
mosaic_status ring_gemm_mma_s8(const uint32_t *A, int64_t lda, const uint32_t *B, int64_t ldb,
                               uint32_t *C, int64_t ldc, const uint32_t *Cin, int64_t ldcin,
                               int sgn, int64_t M, int64_t N, int64_t K, void *ws, size_t ws_bytes,
                               cudaStream_t st);
bool tc_available();
mosaic_status device_status(cudaStream_t st);
bool mma_s8_available();

// Streaming ring GEMM for a few tokens (NT, uint32, K-contiguous):
// C = (Cin?) + sgn * A B^T with 1 <= M <= kSkinnyMaxM, each element of B read
// once through TMA.  skinny_ok() tells whether the operands qualify (16-byte
// aligned bases, row strides multiples of 4 words, a Blackwell device).
constexpr int64_t kSkinnyMaxM = 16;
bool skinny_ok(const uint32_t *A, int64_t lda, const uint32_t *B, int64_t ldb, int64_t M, int64_t K);
mosaic_status ring_gemm_skinny(const uint32_t *A, int64_t lda, const uint32_t *B, int64_t ldb,
                               uint32_t *C, int64_t ldc, const uint32_t *Cin, int64_t ldcin, int sgn,
                               int64_t M, int64_t N, int64_t K, cudaStream_t st);
// Reads and clears the streaming kernel's timeout word (after a stream sync).
mosaic_status skinny_status();

// Tensor-core ring GEMM for kSkinnyMaxM < M <= kTcwMaxM token rows that
// streams B as uint32 (4 bytes an element) and splits it into digits on the
// chip: C = A B^T (NT, uint32, K-contiguous).  Ap: tcw_ws_bytes(M, K) bytes of
// 16-byte aligned scratch for A's fp16 digit planes.  tcw_ok() tells whether
// the operands qualify (16-byte aligned bases, row strides multiples of 4
// words, a Blackwell device).
constexpr int64_t kTcwMaxM = 64;
size_t tcw_ws_bytes(int64_t M, int64_t K);
bool tcw_ok(const uint32_t *A, int64_t lda, const uint32_t *B, int64_t ldb, int64_t M, int64_t N, int64_t K);
mosaic_status ring_gemm_tcw(const uint32_t *A, int64_t lda, const uint32_t *B, int64_t ldb, uint32_t *C,
                            int64_t ldc, int64_t M, int64_t N, int64_t K, uint16_t *Ap, cudaStream_t st);
// Reads and clears that kernel's timeout word (after a stream sync).
mosaic_status tcw_status();

// Freivalds check: Y (k x ncols) = a (k x m) W (m x ncols, ldw), and the
// per-token comparison a^T Y' vs Ychk X' (lhs, rhs: k x l scratch each).
mosaic_status freivalds_colsum(const uint32_t *a, int k, const uint32_t *W, int64_t ldw, int64_t m,
                               int64_t ncols, uint32_t *Y, cudaStream_t st);
mosaic_status freivalds_check(int k, const uint32_t *a, const uint32_t *Ychk, int64_t m, int64_t n_pad,
                              int64_t l, const uint32_t *Z, int64_t ldz, const uint32_t *Xp, int64_t ldx,
                              uint32_t *bad, uint32_t *n_bad, uint32_t *lhs, uint32_t *rhs, cudaStream_t st);

// Sparse gathers.
// out[row][col] = a[row][col] - b[row][col] (b nullable) + sgn * sum_lev sum_q val * src[g][off_lev + idx]
// where (list entity, staged row g) = (row, col) if !list_is_col else (col, row).
struct SparseLevel {
    const uint32_t *idx;   // nlist x t
    const uint32_t *val;
    int t;
    int64_t off;           // offset of this level's segment (columns of src, or rows of P)
    uint32_t r;            // positions are < r; larger ones are skipped
    const uint32_t *tiled = nullptr;   // tile images of src's segment (build_tile_image), or null
    int lines = 0;                     // idx holds pg_line(position) (lists drawn for the tiled gather)
};
// Chunk permutation of line p in a staged tile of the tiled gather: rows
// 4c .. 4c+3 sit in 16-byte chunk c ^ pg_perm(p), an even number.
__host__ __device__ __forceinline__ uint32_t pg_perm(uint32_t p) { return ((p >> 2) & 3u) << 1; }
// Line offset of position p in a staged tile: 128-byte line p, the
// permutation bits in the 16-byte chunk field.
__host__ __device__ __forceinline__ uint32_t pg_line(uint32_t p) { return (p << 7) + (pg_perm(p) << 4); }
// True when the tiled gather takes lists of weight t over segments of r words
// staged in g_count rows (16-byte aligned lists assumed).
bool pgather_takes(int64_t g_count, uint32_t r, int t);
// Words of the tile images of a g_count x r segment (0 if the tiled gather
// does not take r); the images are built by build_tile_image.
size_t tile_image_words(int64_t g_count, uint32_t r);
mosaic_status build_tile_image(const uint32_t *src, int64_t lds, int64_t col0, uint32_t r, int64_t g_count,
                               uint32_t *img, cudaStream_t st);
mosaic_status gather_status();
// Launches a bounded wait that runs out after limit_ns (the self-test of the
// timeout path: reported by the next device status as MOSAIC_ERR_TIMEOUT).
mosaic_status wait_probe(unsigned long long limit_ns, cudaStream_t st);
// A caller's position list turned into the tiled gather's line offsets:
// dst[i] = pg_line(min(src[i], r - 1)) for count entries (a multiple of 4;
// both pointers 16-byte aligned).
struct LineCopy {
    const uint32_t *src;
    uint32_t *dst;
    int64_t count;
    uint32_t r;
};
// Before an unmask, in one launch: digit planes [4][l][Kp] of Q_d = columns
// [qcol, qcol + rd) of Z (when Qp is not null), the tile images of nimg <= 2
// segments Z[:, icol[k] .. + ir[k]) (tile_image_words(l, ir[k]) words each)
// and the line-offset copies of nlin <= 2 S lists.
mosaic_status unmask_prep(const uint32_t *Z, int64_t ldz, int64_t l, int64_t qcol, int64_t rd, uint16_t *Qp,
                          int64_t Kp, int nimg, const int64_t *icol, const uint32_t *ir, uint32_t *const *img,
                          int nlin, const LineCopy *lin, cudaStream_t st);
mosaic_status sparse_gather(const uint32_t *src, int64_t lds, int64_t seg_off, int64_t seg_len,
                            int64_t g_count, int64_t nlist, bool list_is_col, const SparseLevel *lev,
                            int nlev, const uint32_t *a, int64_t lda, const uint32_t *b, int64_t ldb,
                            int sgn, uint32_t *out, int64_t ldo, cudaStream_t st);
// The two Init X gathers of the same T lists in one launch per level:
// out[j][.] += sum_q val[j][q] * src[.][off + idx[j][q]] over g_count staged
// rows (tile images img[L]), and the same for (src2, g_count2, out2, img2[L]).
// Falls back to two sparse_gather calls when a job would not take the tiled
// gather.
mosaic_status sparse_gather_pair(const uint32_t *src, int64_t lds, int64_t g_count, uint32_t *out, int64_t ldo,
                                 const uint32_t *const *img, const uint32_t *src2, int64_t lds2, int64_t g_count2,
                                 uint32_t *out2, int64_t ldo2, const uint32_t *const *img2, int64_t nlist,
                                 const SparseLevel *lev, int nlev, cudaStream_t st);
// Unmask epilogue: list = output column j; staged rows = tokens k of Z.
// Y_hat = Y' - tmp - sum_i S_{i+1} Q_i, or tmp - sum_i S_{i+1} Q_i when
// `folded` (tmp already holds Y' - K - L Q_d), then decode.
mosaic_status unmask_decode(const uint32_t *Z, int64_t ldz, int64_t seg_off, int64_t seg_len,
                            int64_t l, int64_t m, const SparseLevel *lev, int nlev,
                            const uint32_t *tmp, int64_t ldt, const float *s_w, const float *s_x,
                            const float *bias, float *Y, uint32_t *Yhat, int64_t ldy,
                            cudaStream_t st, bool folded = false);
// out[j][c] = a[j][c] + sum_lev sum_q val[j][q] * P[(row_off_lev + idx[j][q]) * ldp + c]
mosaic_status sparse_rowgather(const uint32_t *P, int64_t ldp, const SparseLevel *lev, int nlev,
                               int64_t m, int64_t ncols, const uint32_t *a, int64_t lda,
                               uint32_t *out, int64_t ldo, cudaStream_t st);
// Elementwise and layout helpers.
mosaic_status add_u32(const uint32_t *a, int64_t lda, const uint32_t *b, int64_t ldb, uint32_t *out,
                      int64_t ldo, int64_t rows, int64_t cols, cudaStream_t st);
mosaic_status transpose_u32(const uint32_t *a, int64_t lda, int64_t rows, int64_t cols, uint32_t *out,
                            int64_t ldo, cudaStream_t st);

}  // namespace mosaic
