/*
 * mosaic.h -- C ABI of the GB300 masked ring-matmul library (libmosaic.so).
 *
 * The library computes the data-parallel hot path of MOSAIC's secure linear
 * layer: the random Hadamard rotation and fixed-point encoding of
 * Pi_Sec-Linear (Sec. 4 protocol box), the LWE/LPN masks of
 * Pi_Sec-Approx-MatMul (Sec. 3.2 protocol box, Init W and Init X), the
 * server's product over Z_{2^32} (Online step 3) and the client's unmask and
 * decode (Online step 5 and Pi_Sec-Linear Online step 3).
 *
 * Conventions shared by every entry point
 *  - Every matrix pointer is a DEVICE pointer owned by the caller; the
 *    library never allocates, frees or retains memory.  Scratch memory comes
 *    in `ws` (size from mosaic_workspace_bytes, for a 256-byte aligned ws as
 *    cudaMalloc returns; from a misaligned ws the bytes before its first
 *    256-byte boundary go unused) and must not overlap any other argument.
 *  - Every call is asynchronous on `stream` (a cudaStream_t passed as void*;
 *    NULL is the legacy default stream).  A status of MOSAIC_OK means the
 *    work was validated and enqueued; faults inside a kernel surface at the
 *    caller's next synchronisation as a CUDA error.
 *  - Matrices are row-major with an explicit leading dimension (elements).
 *    Activations are TOKEN-MAJOR: the paper's X (n x l) is stored as
 *    X_tm = X^T (l x n), and Y (m x l) as Y_tm (l x m).  Every ring product is
 *    "NT": C[i][j] = sum_k A[i][k] * B[j][k] mod 2^32.
 *  - Ring elements are uint32_t (kappa = 32: Z_{2^32}, two's complement for
 *    signed values).  Float inputs must be finite unless stated otherwise.
 *  - Host pointers (mosaic_params*, mosaic_key*) are read during the call
 *    only.
 *  - Errors are returned, never thrown or printed; no entry point exits.
 */
#ifndef MOSAIC_H
#define MOSAIC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    MOSAIC_OK = 0,
    MOSAIC_ERR_ARG = 1,          /* null pointer, bad enum, bad parameter value      */
    MOSAIC_ERR_SHAPE = 2,        /* size out of range, n_pad not a power of two, ... */
    MOSAIC_ERR_ALIGN = 3,        /* pointer or leading dimension misaligned          */
    MOSAIC_ERR_UNSUPPORTED = 4,  /* valid request this build does not implement      */
    MOSAIC_ERR_CUDA = 5,         /* a CUDA runtime call or launch failed             */
    MOSAIC_ERR_WORKSPACE = 6,    /* ws too small (see mosaic_workspace_bytes)        */
    MOSAIC_ERR_TIMEOUT = 7       /* a bounded device wait expired (read back by mosaic_device_status) */
} mosaic_status;

/* Protocol parameters (Example 3.1 defaults, lambda = 140).
 * d       nesting depth of the LWE + LPN mask, 1..3 (Sec. 3.2)
 * r[i-1]  rank r_i, i = 1..d (1536, 1024, 652); r_1 > r_2 > ... is not required
 * t[i-1]  Hamming weight t_i of each row of S_i and each column of T_i,
 *         i = 2..d (t[0] is unused; 80, 80); 1 <= t_i <= r_{i-1} / 2
 * sigma   Gaussian parameter of E_w, E_x: Pr[k] ~ exp(-k^2 / (2 sigma^2)),
 *         0 <= sigma <= 8 (0 disables the noise)
 * qbits   signed operand width b of Pi_Sec-Linear (16); the operand window is
 *         q_max = min(2^(b-1) - 1, floor(sqrt(2^31 / n_pad)))
 * rounds  ChaCha rounds of the PRG (20; 8 and 12 accepted)
 * kappa   ring width, must be 32                                           */
typedef struct {
    uint32_t kappa;
    uint32_t d;
    uint32_t r[3];
    uint32_t t[3];
    float sigma;
    uint32_t qbits;
    uint32_t rounds;
    /* 1: the activation mask nests like the weight mask (Sec. 3.2 box, Init X
     * 1b-1c: U_x = C_d R + sum_i C_i T_{i+1} + E_x, K = J_d R + sum_i J_i T_{i+1}).
     * 0: the paper's deployed variant (Sec. 5.2, "Protocol parameterization"):
     * the recursive LPN part of the activation mask is omitted, U_x = C_1 R + E_x
     * and K = J_1 R with R uniform r_1 x l; only J_1 is kept at Init W. */
    uint32_t act_nested;
} mosaic_params;

/* 256-bit PRG key (8 little-endian words). */
typedef struct {
    uint32_t key[8];
} mosaic_key;

/* Fills `p` with the Example 3.1 parameters (d = 3, r = 1536/1024/652,
 * t = 80/80, sigma = 0.5, b = 16, 20 rounds, kappa = 32, act_nested = 1). */
void mosaic_default_params(mosaic_params *p);

/* Number of kernels this library has launched in this process (all devices,
 * all threads; host-side counter, for benchmarking). */
uint64_t mosaic_kernel_launches(void);

/* Per-kernel device time, for measurement (not part of the method).
 * mosaic_kernel_timing(1) makes every later launch of this library on a
 * stream that is not being captured into a CUDA graph record a pair of CUDA
 * events around itself, on that stream; mosaic_kernel_timing(0) stops it.
 * Returns the previous setting.  Off by default (a launch then pays one atomic
 * load).  Timing adds two event records per launch, so time whole steps with
 * it off.
 * mosaic_kernel_times waits for every recorded pair, adds the durations to
 * per-key totals and writes up to `cap` of them to `out` (cap may be 0); the
 * key is "<role>:<kernel>", role naming the entry point that launched the
 * kernel (init_x, encode, ring_gemm, unmask, init_w, glue, ...).  With
 * `reset` the totals start again from zero after being written.  Returns the
 * number of keys, or -1 if an event could not be read (the records are
 * dropped).  Recorded pairs (and their events) stay held until this call
 * reads them. */
typedef struct {
    char name[64];
    uint64_t launches;
    double ms;
} mosaic_kernel_time;
int mosaic_kernel_timing(int enable);
int mosaic_kernel_times(mosaic_kernel_time *out, int cap, int reset);

/* Rate of the ChaCha20 integer mix (add, xor, rotate) on the current device,
 * in operations per second, for the draws' roofline (not part of the
 * method): one launch of 8 blocks of 256 threads per SM, each thread running
 * 2000 double rounds on 16 independent words, timed with CUDA events; waits
 * for the launch.  `scratch` is a device buffer of at least 8192 bytes per SM
 * (one word per thread is written there).  About 2 ms of GPU time. */
mosaic_status mosaic_int_mix_rate(uint32_t *scratch, size_t scratch_bytes, double *ops_per_second, void *stream);

/* Shared-memory read rate of the current device in bytes per second, for the
 * gathers' roofline (not part of the method), with the tiled gather's access:
 * two blocks of 512 threads and 64 KB per SM, each group of 8 lanes reading a
 * whole 128-byte line per 16-byte load instruction (four scattered lines per
 * warp access), 4000 x 8 volatile loads a thread, timed with CUDA events;
 * waits for the launch.  `scratch` is a device buffer of at least 4096 bytes
 * per SM.  About 1 ms of GPU time. */
mosaic_status mosaic_smem_read_rate(uint32_t *scratch, size_t scratch_bytes, double *bytes_per_second,
                                    void *stream);

/* Human-readable name of a status code (static string). */
const char *mosaic_status_string(mosaic_status s);

/* q_max for a rotation width n_pad (Sec. 4 straw-man paragraph: each entry of
 * W_hat X_hat is at most n q_max^2, and n q_max^2 <= 2^(kappa-1)).  Returns 0
 * if n_pad is not a power of two in [32, 65536] or qbits is outside [2, 16]. */
int32_t mosaic_qmax(int64_t n_pad, uint32_t qbits);

/* Writes the inversion table of the discrete Gaussian with parameter sigma
 * (Sec. 3.1: Pr[k] ~ exp(-k^2 / (2 sigma^2)) on [-B, B], B = ceil(12 sigma)):
 * table[j] = floor(2^64 CDF(j - B)) computed in long double, last entry
 * 2^64 - 1.  Host-only.  Returns B, or -1 if sigma is outside (0, 8] or
 * capacity < 2B + 1. */
int mosaic_gaussian_table(float sigma, uint64_t *table, int capacity);

/* ------------------------------------------------------------------------ */
/* PRG and samplers (Sec. 3.2 box: "C samples ...").  The generator is       */
/* ChaCha in counter mode (RFC 8439 block layout): stream (tag, stream_id)   */
/* uses nonce = (tag, stream_id low 32 bits, stream_id high 32 bits); word w */
/* of the stream is word w mod 16 of block floor(w / 16).                    */
/* Tags: kind in bits 0..7, level i in bits 8..15.                           */
/* ------------------------------------------------------------------------ */
enum {
    MOSAIC_TAG_M = 1,     /* public M_i        (stream_id: the chain id, n_pad by convention) */
    MOSAIC_TAG_N = 2,     /* public N_i                                                        */
    MOSAIC_TAG_L = 3,     /* secret L           (stream_id: matrix id)                         */
    MOSAIC_TAG_S = 4,     /* secret sparse S_i                                                  */
    MOSAIC_TAG_EW = 5,    /* weight noise E_w                                                   */
    MOSAIC_TAG_R = 6,     /* per-pass R         (stream_id: pass id)                            */
    MOSAIC_TAG_T = 7,     /* per-pass sparse T_i                                                */
    MOSAIC_TAG_EX = 8,    /* activation noise E_x                                               */
    MOSAIC_TAG_SIGN = 9,  /* rotation signs d   (stream_id: matrix id)                          */
    MOSAIC_TAG_CHECK = 10 /* Freivalds check vectors a (stream_id: matrix id)                   */
};

/* out[i * ldo + j] = stream word i * cols + j: uniform elements of Z_{2^32}.
 * rows, cols >= 0; rows * cols < 2^36; ldo >= cols. */
mosaic_status mosaic_prg_uniform(const mosaic_key *key, uint32_t tag, uint64_t stream_id,
                                 uint32_t rounds, int64_t rows, int64_t cols, uint32_t *out,
                                 int64_t ldo, void *stream);

/* out[e], e < count: discrete Gaussian ring elements (two's complement).
 * Element e reads u = word(2e) | word(2e+1) << 32 and returns the smallest
 * k in [-B, B] (B = ceil(12 sigma)) with u < floor(2^64 CDF(k)), else B.
 * sigma = 0 writes zeros.  count < 2^35. */
mosaic_status mosaic_prg_gaussian(const mosaic_key *key, uint32_t tag, uint64_t stream_id,
                                  uint32_t rounds, float sigma, int64_t count, uint32_t *out,
                                  void *stream);

/* rows sparse vectors over [0, r), exactly t nonzeros each (LPN noise of
 * Hamming weight t, Example 3.1).  Row j reads its own window of 65536
 * stream words starting at word j * 65536: positions p = (w * r) >> 32 in
 * draw order, repeats skipped, then the next nonzero words as values.
 * idx, val: rows x t row-major.  rows < 2^20, 1 <= t <= min(r/2, 1024).
 * `fail` (device, nullable) is set to 1 if a row exhausts its window
 * (probability below 2^-1000 within these limits). */
mosaic_status mosaic_prg_sparse(const mosaic_key *key, uint32_t tag, uint64_t stream_id,
                                uint32_t rounds, int64_t rows, uint32_t r, uint32_t t,
                                uint32_t *idx, uint32_t *val, uint32_t *fail, void *stream);

/* ------------------------------------------------------------------------ */
/* Rotation and encoding (Pi_Sec-Linear box; Sec. 4 "Random Hadamard        */
/* rotation").                                                               */
/* ------------------------------------------------------------------------ */

/* y = rows of H D x (Sec. 4: R = H D, H the normalised Walsh-Hadamard
 * matrix in Sylvester order, D = diag(d)).  Each row of x (length n, leading
 * dimension ldx) is zero-padded to n_pad, negated where bit c of
 * sign_words[c / 32] is set (sign_words: n_pad / 32 device words, NULL for
 * D = I), transformed by butterflies (a, b) -> (a + b, a - b) in fp32 with
 * stages h = 1, 2, ..., n_pad / 2 in that order, then multiplied by
 * fl32(1 / sqrt(n_pad)).  y: rows x n_pad (leading dimension n_pad); y must
 * not overlap x.  n_pad a power of two in [32, 65536], 1 <= n <= n_pad
 * (65536-wide rows run the first 15 stages on their halves, then the last
 * stage and the scale in a second pass over y; same rounding).
 * x, y 16-byte aligned; ldx a multiple of 4. */
mosaic_status mosaic_hadamard(const float *x, int64_t ldx, float *y, int64_t rows, int64_t n,
                              int64_t n_pad, const uint32_t *sign_words, void *stream);

/* Fused rotation + per-row quantisation + mask-add (Pi_Sec-Linear Online
 * step 1 for activation rows, Init W step 2 for weight rows; Approx-MatMul
 * Online step 2).  For each row: v = H D x as in mosaic_hadamard when
 * `rotate` is 1 (v = x zero-padded when 0); s = max|v| / qmax (fp32);
 * code = clamp(rint(v / s), -qmax, qmax) (IEEE division, ties to even),
 * 0 when s = 0; a row with a non-finite value gets s = NaN and code 0.
 * out[row][c] = code + mask[row][c] mod 2^32 (mask nullable: no add);
 * scale[row] = s.  `planes` (nullable) additionally receives the signed
 * base-2^8 digits of out as bf16 digit planes, layout [4][rows][n_pad]
 * (see mosaic_digit_split).  out: rows x ldo; mask: rows x ldm.
 * 1 <= qmax <= 32767.  Alignment as mosaic_hadamard; ldo, ldm multiples of 4. */
mosaic_status mosaic_encode(const float *x, int64_t ldx, int64_t rows, int64_t n, int64_t n_pad,
                            int32_t qmax, int rotate, const uint32_t *sign_words,
                            const uint32_t *mask, int64_t ldm, uint32_t *out, int64_t ldo,
                            float *scale, uint16_t *planes, void *stream);

/* Signed base-2^8 digit split of ring elements (Sec. 5.2 "Emulation
 * approach", re-designed with signed digits): with b = a + 0x80808080,
 * digit i is (int)((b >> 8i) & 0xff) - 128 in [-128, 127], so that
 * a = sum_i digit_i 2^(8i) mod 2^32.  Each digit is written exactly as a
 * bf16 value into planes[i][row][col] (layout [4][rows][cols], bf16 bits in
 * uint16_t).  cols a multiple of 8; lda a multiple of 4; 16-byte aligned. */
mosaic_status mosaic_digit_split(const uint32_t *a, int64_t lda, int64_t rows, int64_t cols,
                                 uint16_t *planes, void *stream);

/* ------------------------------------------------------------------------ */
/* Ring product (Approx-MatMul Online step 3; Sec. 5.2 emulation).           */
/* ------------------------------------------------------------------------ */
typedef enum {
    MOSAIC_GEMM_AUTO = 0,     /* fastest available variant for the shape                    */
    MOSAIC_GEMM_TC = 1,       /* tcgen05 kind::f16: 10 exact bf16 digit-pair products, TMEM  */
    MOSAIC_GEMM_MMA_S8 = 2,   /* legacy mma.sync s8 digit-pair products, int32 accumulators */
    MOSAIC_GEMM_IMAD = 3      /* CUDA-core 32-bit multiply-add                               */
} mosaic_gemm_variant;

/* 1 if this build implements `variant` on the current device (host-only
 * query of the build and of the device's compute capability), else 0. */
int mosaic_gemm_variant_available(int variant);

/* C[i][j] = sum_{k<K} A[i][k] B[j][k] mod 2^32, i < M, j < N.
 * A: M x K (lda), B: N x K (ldb), C: M x N (ldc); C must not overlap A or B.
 * M, N, K >= 0, K <= 2^20.  The TC and MMA_S8 variants split A and B into
 * digit planes in `ws` (mosaic_workspace_bytes(MOSAIC_OP_RING_GEMM, ...));
 * IMAD needs no workspace.  TC requires lda, ldb multiples of 4 and 16-byte
 * aligned A, B (MOSAIC_ERR_ALIGN otherwise; AUTO then runs IMAD).  With
 * 1 <= M <= MOSAIC_SKINNY_MAX_M (a few tokens, e.g. one decode step) and
 * K >= 1, TC and AUTO run a streaming CUDA-core kernel instead, which reads
 * each element of B once (4 bytes) and needs no workspace.  With
 * MOSAIC_SKINNY_MAX_M < M <= MOSAIC_STREAMW_MAX_M (a small decode batch) TC
 * and AUTO run a tensor-core kernel that also reads each element of B once as
 * uint32 and splits it into digits on the chip; it needs 8 M ceil8(K) bytes of
 * `ws` for A's digit planes.  Every path gives the same ring product. */
#define MOSAIC_SKINNY_MAX_M 16
#define MOSAIC_STREAMW_MAX_M 64
mosaic_status mosaic_ring_gemm(const uint32_t *A, int64_t lda, const uint32_t *B, int64_t ldb,
                               uint32_t *C, int64_t ldc, int64_t M, int64_t N, int64_t K,
                               int variant, void *ws, size_t ws_bytes, void *stream);

/* Same product from pre-split bf16 digit planes (layout [4][rows][K] with a
 * plane stride of rows_alloc * ldp elements, see mosaic_digit_split /
 * mosaic_encode).  A planes: M rows (plane stride a_plane), B planes: N rows
 * (plane stride b_plane); ldpa, ldpb leading dimensions in elements,
 * multiples of 8; 16-byte aligned.  Variant TC (or AUTO); the bf16 planes
 * feed only the tensor-core kernel (MOSAIC_ERR_UNSUPPORTED otherwise). */
mosaic_status mosaic_ring_gemm_planes(const uint16_t *A_planes, int64_t ldpa, int64_t a_plane,
                                      const uint16_t *B_planes, int64_t ldpb, int64_t b_plane,
                                      uint32_t *C, int64_t ldc, int64_t M, int64_t N, int64_t K,
                                      int variant, void *stream);

/* ------------------------------------------------------------------------ */
/* Masks (Sec. 3.2 protocol box).  Sr = r_1 + ... + r_d.                      */
/* ------------------------------------------------------------------------ */

/* Public chains for input width n_pad (Init W steps 1-3, 5): samples
 * M_i (r_i x r_{i-1}, element (a,b) = word a r_{i-1} + b of (M, level i))
 * and N_i (r_{i-1} x r_i, element (a,b) = word a r_i + b of (N, level i)),
 * r_0 = n_pad, from stream `chain_id`, and writes
 *   P  (Sr x n_pad): rows [P_1; P_2; ...; P_d], P_i = M_i ... M_1
 *   C  (n_pad x Sr): columns [C_1 | ... | C_d], C_i = N_1 ... N_i
 *   CT (Sr x n_pad): C transposed.
 * ws: mosaic_workspace_bytes(MOSAIC_OP_MASK_CHAINS, 0, n_pad, 0, p). */
mosaic_status mosaic_mask_chains(const mosaic_params *p, const mosaic_key *key,
                                 uint64_t chain_id, int64_t n_pad, uint32_t *P, uint32_t *C,
                                 uint32_t *CT, void *ws, size_t ws_bytes, void *stream);

/* Init W of Pi_Sec-Linear and Pi_Sec-Approx-MatMul for one weight matrix
 * W (m x n float, leading dimension ldw) with matrix id `matrix_id`:
 *   sign_words (n_pad/32)  d of R = H D           (stream (SIGN, matrix_id))
 *   W_hat, s_w (m)          rows of W R^T quantised (mosaic_encode)
 *   L (m x r_d)             uniform                 (stream (L, matrix_id))
 *   S_idx, S_val            S_{i+1}, i = 1..d-1: m x t_{i+1} each, stored
 *                           level after level        (stream (S, level i+1))
 *   E_w (m x n_pad)         Gaussian                (stream (EW, matrix_id))
 *   Wp ((m + Sr) x n_pad)   rows [0, m):   W' = W_hat + L P_d + sum S_{i+1} P_i + E_w
 *                           rows [m, m+Sr): a copy of P (server-side operand)
 *   J (m x Sr)              columns [J_1 | ... | J_d], J_i = (W_hat + E_w) C_i
 *                           (act_nested = 0: only J_1, columns [0, r_1), is
 *                           written; the others are left untouched)
 * Wp_planes (nullable): bf16 digit planes of Wp ([4][m + Sr][n_pad]).
 * ws: mosaic_workspace_bytes(MOSAIC_OP_MASK_WEIGHT, m, n_pad, 0, p). */
mosaic_status mosaic_mask_weight(const mosaic_params *p, const mosaic_key *key,
                                 uint64_t matrix_id, const float *W, int64_t ldw, int64_t m,
                                 int64_t n, int64_t n_pad, const uint32_t *P, const uint32_t *CT,
                                 uint32_t *sign_words, float *s_w, uint32_t *L, uint32_t *S_idx,
                                 uint32_t *S_val, uint32_t *Wp, uint16_t *Wp_planes, uint32_t *J,
                                 int variant, void *ws, size_t ws_bytes, void *stream);

/* Init X (per pass, independent of X): samples R^T (l x r_d, stream (R,
 * pass_id)), T_{i+1} (column k = sparse row k, stream (T, level i+1)) and
 * E_x^T (l x n_pad, stream (EX, pass_id)) and writes
 *   Ux_tm (l x n_pad) = (C_d R + sum_i C_i T_{i+1} + E_x)^T
 *   K_tm  (l x m)     = (J_d R + sum_i J_i T_{i+1})^T
 * from C (n_pad x Sr) and J (m x Sr).  With act_nested = 0: R^T is l x r_1
 * (same stream), no T is drawn, Ux_tm = (C_1 R + E_x)^T, K_tm = (J_1 R)^T.
 * ws: mosaic_workspace_bytes(MOSAIC_OP_MASK_ACTIVATION, m, n_pad, l, p). */
mosaic_status mosaic_mask_activation(const mosaic_params *p, const mosaic_key *key,
                                     uint64_t pass_id, int64_t m, int64_t n_pad, int64_t l,
                                     const uint32_t *C, const uint32_t *J, uint32_t *Ux_tm,
                                     uint32_t *K_tm, int variant, void *ws, size_t ws_bytes,
                                     void *stream);

/* Stationary operands of Init X, made once per weight matrix (after
 * mosaic_mask_weight) so that no pass re-splits or re-stages them.  The
 * buffer is opaque to the caller; it holds
 *  - the tensor-core digit planes [4][n_pad + m][Kp] bf16 (Kp = r rounded up
 *    to a multiple of 8, r = r_d, or r_1 with act_nested = 0): rows [0, n_pad)
 *    the C-factor block (C_d, or C_1), rows [n_pad, n_pad + m) the J-factor
 *    block (J_d, or J_1);
 *  - for each LPN level i of a nested activation mask, the segments C_i and
 *    J_i in the 32-row tile layout the sparse gathers stage with one bulk
 *    copy per tile.
 * Size: mosaic_workspace_bytes(MOSAIC_OP_ACTIVATION_PLANES, m, n_pad, 0, p).
 * 16-byte aligned device buffer. */
mosaic_status mosaic_prepare_activation(const mosaic_params *p, int64_t m, int64_t n_pad,
                                        const uint32_t *C, const uint32_t *J, uint16_t *cj_planes,
                                        void *stream);

/* mosaic_mask_activation with the planes of mosaic_prepare_activation (same
 * results; the two dense products R^T C^T and R^T J^T run as one tensor-core
 * product against the cached planes when l > MOSAIC_SKINNY_MAX_M). */
mosaic_status mosaic_mask_activation_planes(const mosaic_params *p, const mosaic_key *key,
                                            uint64_t pass_id, int64_t m, int64_t n_pad, int64_t l,
                                            const uint32_t *C, const uint32_t *J,
                                            const uint16_t *cj_planes, uint32_t *Ux_tm,
                                            uint32_t *K_tm, int variant, void *ws, size_t ws_bytes,
                                            void *stream);

/* General form of Init X: cj_planes as in mosaic_mask_activation_planes
 * (nullable: split per call), and the pass id is pass_id + *pass_dev when
 * pass_dev (a device word) is given -- read on the device when the samplers
 * run, so that a CUDA graph captured around this call (and around
 * mosaic_advance_pass) draws a fresh pass on every replay.  With pass_dev
 * NULL it is mosaic_mask_activation(_planes). */
mosaic_status mosaic_mask_activation_ex(const mosaic_params *p, const mosaic_key *key, uint64_t pass_id,
                                        const uint64_t *pass_dev, int64_t m, int64_t n_pad, int64_t l,
                                        const uint32_t *C, const uint32_t *J, const uint16_t *cj_planes,
                                        uint32_t *Ux_tm, uint32_t *K_tm, int variant, void *ws,
                                        size_t ws_bytes, void *stream);


/* Init X in two parts, for callers that overlap the draws with other work
 * (Sec. 3.2 box, Init X step 1a is the draws; 1b-1c the compositions).  Same
 * arguments and results as mosaic_mask_activation_ex, plus `phase`:
 *   MOSAIC_INITX_DRAWS    R (and its digit planes), the T lists into ws and
 *                         E_x into Ux_tm: one ALU-bound launch (ChaCha20);
 *   MOSAIC_INITX_COMPOSE  the tensor-core product and the LPN gathers that
 *                         turn them into U_x and K;
 *   MOSAIC_INITX_ALL      both (mosaic_mask_activation_ex).
 * A COMPOSE call must follow the DRAWS call of the same pass with the same
 * arguments (p, key, pass id, shapes, C, J, cj_planes, Ux_tm, K_tm, variant)
 * and the same workspace, untouched in between (the draws live there; make
 * the COMPOSE stream wait for the DRAWS stream).  Each phase alone validates
 * what the whole call validates. */
#define MOSAIC_INITX_DRAWS 1
#define MOSAIC_INITX_COMPOSE 2
#define MOSAIC_INITX_ALL 3
mosaic_status mosaic_mask_activation_phase(const mosaic_params *p, const mosaic_key *key, uint64_t pass_id,
                                           const uint64_t *pass_dev, int64_t m, int64_t n_pad, int64_t l,
                                           const uint32_t *C, const uint32_t *J, const uint16_t *cj_planes,
                                           uint32_t *Ux_tm, uint32_t *K_tm, int variant, void *ws,
                                           size_t ws_bytes, int phase, void *stream);

/* *pass_dev += delta, enqueued on `stream` (one-thread kernel). */
mosaic_status mosaic_advance_pass(uint64_t *pass_dev, uint64_t delta, void *stream);

/* One entry point for the three mask-generation roles of the protocol box
 * (Sec. 3.2, Pi_Sec-Approx-MatMul: Init W steps 1-3 and 5, Init X steps
 * 1a-1c; eq. weight-mask and eq. activation-mask).  The roles take different
 * operands -- the public chains are made once per input width, the weight
 * mask consumes a float matrix and yields seven client/server outputs, the
 * activation mask consumes the chains and J and yields U_x and K per pass --
 * so the role-specific buffers travel in one struct and `kind` selects the
 * role.  Each kind is exactly the role call named below (same validation,
 * same results, same workspace size); fields a kind does not name are
 * ignored.
 *
 *   kind                    stream_id    rows   l       fields used              same as
 *   MOSAIC_MASK_CHAINS      chain id     --     --      P, C, CT (outputs)       mosaic_mask_chains
 *   MOSAIC_MASK_WEIGHT      matrix id    m      --      W, ldw, n, P, CT (in);   mosaic_mask_weight
 *                                                       sign_words, s_w, L, S_idx,
 *                                                       S_val, Wp, Wp_planes
 *                                                       (nullable), J (out)
 *   MOSAIC_MASK_ACTIVATION  pass id      m      tokens  C, J, cj_planes          mosaic_mask_activation_ex
 *                                                       (nullable), pass_dev
 *                                                       (nullable) (in);
 *                                                       Ux_tm, K_tm (out)
 *
 * `variant` is used by WEIGHT and ACTIVATION.  Returns MOSAIC_ERR_ARG for an
 * unknown kind or a null `io`; otherwise the status of the role call.
 * ws: mosaic_workspace_bytes(MOSAIC_OP_MASK_CHAINS / _WEIGHT / _ACTIVATION, ...). */
typedef enum {
    MOSAIC_MASK_CHAINS = 1,
    MOSAIC_MASK_WEIGHT = 2,
    MOSAIC_MASK_ACTIVATION = 3
} mosaic_mask_kind;

typedef struct {
    const float *W;            /* WEIGHT: m x n float weights, leading dimension ldw */
    int64_t ldw;
    int64_t n;                 /* WEIGHT: columns of W (n <= n_pad)                  */
    uint32_t *P;               /* Sr x n_pad: CHAINS out, WEIGHT in                  */
    uint32_t *C;               /* n_pad x Sr: CHAINS out, ACTIVATION in              */
    uint32_t *CT;              /* Sr x n_pad: CHAINS out, WEIGHT in                  */
    uint32_t *sign_words;      /* WEIGHT out (n_pad / 32)                            */
    float *s_w;                /* WEIGHT out (m)                                     */
    uint32_t *L;               /* WEIGHT out (m x r_d)                               */
    uint32_t *S_idx;           /* WEIGHT out                                         */
    uint32_t *S_val;           /* WEIGHT out                                         */
    uint32_t *Wp;              /* WEIGHT out ((m + Sr) x n_pad)                      */
    uint16_t *Wp_planes;       /* WEIGHT out, nullable                               */
    uint32_t *J;               /* m x Sr: WEIGHT out, ACTIVATION in                  */
    const uint16_t *cj_planes; /* ACTIVATION in, nullable (mosaic_prepare_activation) */
    const uint64_t *pass_dev;  /* ACTIVATION in, nullable (device pass counter)      */
    uint32_t *Ux_tm;           /* ACTIVATION out (l x n_pad)                         */
    uint32_t *K_tm;            /* ACTIVATION out (l x m)                             */
} mosaic_mask_io;

mosaic_status mosaic_mask(int kind, const mosaic_params *p, const mosaic_key *key, uint64_t stream_id,
                          int64_t rows, int64_t n_pad, int64_t l, const mosaic_mask_io *io, int variant,
                          void *ws, size_t ws_bytes, void *stream);

/* ------------------------------------------------------------------------ */
/* Unmask and decode (Approx-MatMul Online step 5; Pi_Sec-Linear Online      */
/* step 3).                                                                  */
/* ------------------------------------------------------------------------ */

/* Z (l x ldz) is the server output X'_tm Wp^T: columns [0, m) hold Y'_tm,
 * columns [m, m + Sr) hold [Q_1 | ... | Q_d]_tm.  Computes
 *   Y_hat = Y' - K - L Q_d - sum_{i<d} S_{i+1} Q_i      (mod 2^32)
 *   Y[k][j] = ((float)(int32)Y_hat[k][j] * s_w[j]) * s_x[k] + bias[j]
 * (fp32, two roundings of the products, no fused multiply-add; bias
 * nullable).  Y: l x m fp32 (ldy); Yhat (nullable): l x m uint32 (ldy).
 * ws: mosaic_workspace_bytes(MOSAIC_OP_UNMASK, m, 0, l, p) bytes hold every
 * optional part (tensor-core digit planes of Q_d, tile images of the Q_i,
 * line-offset copies of the S lists); any size from 4 l m bytes (rounded up
 * to 256) works, parts that do not fit are skipped and the result is the
 * same; less returns MOSAIC_ERR_WORKSPACE. */
mosaic_status mosaic_unmask(const mosaic_params *p, int64_t l, int64_t m, const uint32_t *Z,
                            int64_t ldz, const uint32_t *K_tm, const uint32_t *L,
                            const uint32_t *S_idx, const uint32_t *S_val, const float *s_w,
                            const float *s_x, const float *bias, float *Y, uint32_t *Yhat,
                            int64_t ldy, int variant, void *ws, size_t ws_bytes, void *stream);

/* L (m x r_d) as tensor-core digit planes [4][m][Kp], Kp = r_d rounded up to a
 * multiple of 8, made once per weight matrix.  Size:
 * mosaic_workspace_bytes(MOSAIC_OP_UNMASK_PLANES, m, 0, 0, p); 16-byte aligned. */
mosaic_status mosaic_prepare_unmask(const mosaic_params *p, int64_t m, const uint32_t *L,
                                    uint16_t *L_planes, void *stream);

/* mosaic_unmask with the planes of mosaic_prepare_unmask (same results).
 * L_planes is required (MOSAIC_ERR_ARG when null, MOSAIC_ERR_ALIGN when not
 * 16-byte aligned). */
mosaic_status mosaic_unmask_planes(const mosaic_params *p, int64_t l, int64_t m, const uint32_t *Z,
                                   int64_t ldz, const uint32_t *K_tm, const uint32_t *L,
                                   const uint16_t *L_planes, const uint32_t *S_idx,
                                   const uint32_t *S_val, const float *s_w, const float *s_x,
                                   const float *bias, float *Y, uint32_t *Yhat, int64_t ldy,
                                   int variant, void *ws, size_t ws_bytes, void *stream);

/* Self-test of the timeout path: launches a kernel whose bounded wait on a
 * barrier phase that nothing completes gives up after limit_us microseconds
 * (1 .. 10^6) and raises a device error word, as a copy or product that
 * never arrives would; the next mosaic_device_status returns
 * MOSAIC_ERR_TIMEOUT (and clears the word).  No fault, no hang: the context
 * stays usable. */
mosaic_status mosaic_selftest_wait(int64_t limit_us, void *stream);

/* Synchronises `stream` and reports device-side failures of earlier calls:
 * MOSAIC_ERR_TIMEOUT if a tensor-core product, a streaming product or a tiled
 * gather gave up a bounded wait (the device error words are cleared by this
 * call), MOSAIC_ERR_CUDA if a CUDA error is pending, else MOSAIC_OK. */
mosaic_status mosaic_device_status(void *stream);

/* mosaic_unmask for callers that cannot allocate device memory (the paper
 * has no counterpart: this is a deployment convenience of this library).
 * Same arguments and results as mosaic_unmask, without `ws`/`ws_bytes`: the
 * l x m words of scratch come from a fixed 16 MiB array inside the library,
 * so it suits code that may not call cudaMalloc -- e.g. a plugin whose host
 * framework owns all device memory, or a serving loop with a fixed memory
 * budget.
 *  - Limit: l * m <= 2^22 (4,194,304); larger requests return
 *    MOSAIC_ERR_WORKSPACE and enqueue nothing.
 *  - Every GPU that loads the library holds the 16 MiB array until the
 *    process exits.
 *  - Every call looks up the array's device address (cudaGetSymbolAddress)
 *    on the current device; nothing is cached, so the entry point stays
 *    valid after cudaDeviceReset.  Make the first call on a device before
 *    any stream capture (it may load the module).
 *  - Speed: the array holds the l x m scratch first and then whichever
 *    optional parts of mosaic_unmask still fit (digit planes of Q_d, tile
 *    images of the Q_i, line-offset copies of the S lists).  Beyond small
 *    l x m the digit planes do not fit (they need about 8 (l + m) r_d bytes),
 *    so with MOSAIC_GEMM_TC / AUTO the Q_d L^T product runs on the CUDA cores
 *    (IMAD), several times slower than with a caller workspace; the results
 *    are the same.
 *  - All calls share the one array: calls whose GPU work overlaps (e.g. on two
 *    streams at once) race on it, so order them (same stream or events).
 *    Nothing in the array needs to start at zero: each call writes every
 *    scratch word before reading it.
 *  - It allocates and frees nothing. */
mosaic_status mosaic_unmask_noalloc(const mosaic_params *p, int64_t l, int64_t m,
                                    const uint32_t *Z, int64_t ldz, const uint32_t *K_tm,
                                    const uint32_t *L, const uint32_t *S_idx,
                                    const uint32_t *S_val, const float *s_w, const float *s_x,
                                    const float *bias, float *Y, uint32_t *Yhat, int64_t ldy,
                                    int variant, void *stream);

/* ------------------------------------------------------------------------ */
/* Float glue of a decoder layer (Sec. 4.1: the non-linear parts run on the   */
/* trusted side in plain arithmetic).  Model operations between the secure    */
/* linear calls, not part of the masked product; one pass over HBM each.     */
/* ------------------------------------------------------------------------ */
/* RMSNorm without a gain: y[r][c] = x[r][c] / sqrt(mean_c x[r][c]^2 + eps),
 * fp32, row-major (leading dimensions ldx, ldy >= n); y may equal x.  One
 * block per row, the sum of squares in fp32.  rows < 2^31. */
mosaic_status mosaic_rmsnorm(const float *x, int64_t ldx, int64_t rows, int64_t n, float eps, float *y,
                             int64_t ldy, void *stream);

/* SwiGLU gate: out[r][c] = silu(gu[r][c]) * gu[r][ffn + c] with
 * silu(g) = g / (1 + exp(-g)), fp32; gu is rows x 2 ffn (gate columns first,
 * leading dimension ldg >= 2 ffn), out rows x ffn (ldo >= ffn; must not
 * overlap gu).  rows <= 65535. */
mosaic_status mosaic_swiglu(const float *gu, int64_t ldg, int64_t rows, int64_t ffn, float *out, int64_t ldo,
                            void *stream);

/* ------------------------------------------------------------------------ */
/* Integrity check (Sec. 3.2 box, Init W step 4 and Online step 4; appendix  */
/* "Computational integrity": Freivalds' check).                             */
/* ------------------------------------------------------------------------ */
/* The box draws a with n entries and checks Y^chk X = a^T Y'; the shapes only
 * agree with a in Z_{2^32}^m and the masked input, so this library checks
 *     a^T Y' == (a^T W') X'   over Z_{2^32}
 * token by token, with k independent vectors a (an error e in Y' escapes one
 * vector with probability 2^-(32 - v), v = the number of trailing zero bits
 * of e, so k vectors bound it by 2^-k for the worst case e = 2^31).
 *
 * Setup (one-time per weight matrix): draws the k x m matrix a (row v = check
 * vector v) from stream (CHECK, matrix_id) and writes Ychk = a W' (k x n_pad)
 * from the masked weights W' (m x n_pad, leading dimension ldw; rows [0, m) of
 * the Wp operand of mosaic_mask_weight).  1 <= k <= 16.  Device buffers. */
mosaic_status mosaic_freivalds_setup(const mosaic_params *p, const mosaic_key *key,
                                     uint64_t matrix_id, int k, const uint32_t *Wm, int64_t ldw,
                                     int64_t m, int64_t n_pad, uint32_t *a, uint32_t *Ychk,
                                     void *stream);

/* Online check of one server answer: for every token j < l,
 *     lhs_v = sum_{i<m} a[v][i] Z[j][i]          (Y' = the first m columns of Z)
 *     rhs_v = sum_{c<n_pad} Ychk[v][c] Xp[j][c]  (X', leading dimension ldx)
 * bad[j] = number of vectors v with lhs_v != rhs_v, and *n_bad is increased by
 * the number of tokens with bad[j] != 0 (the caller zeroes it; read it after
 * the stream has been synchronised; a nonzero count means: abort).
 * ws: 2 k l words (mosaic_workspace_bytes(MOSAIC_OP_FREIVALDS_CHECK, k, 0, l, NULL)).
 * All pointers are device pointers; the products stream Z and X' once. */
mosaic_status mosaic_freivalds_check(int k, const uint32_t *a, const uint32_t *Ychk, int64_t m,
                                     int64_t n_pad, int64_t l, const uint32_t *Z, int64_t ldz,
                                     const uint32_t *Xp, int64_t ldx, uint32_t *bad,
                                     uint32_t *n_bad, void *ws, size_t ws_bytes, void *stream);

/* Workspace sizes. */
typedef enum {
    MOSAIC_OP_RING_GEMM = 1,        /* M = rows of A, n_pad = rows of B (N), l = K */
    MOSAIC_OP_MASK_CHAINS = 2,
    MOSAIC_OP_MASK_WEIGHT = 3,
    MOSAIC_OP_MASK_ACTIVATION = 4,
    MOSAIC_OP_UNMASK = 5,
    MOSAIC_OP_FREIVALDS_CHECK = 6,  /* m = k vectors, l = tokens */
    MOSAIC_OP_ACTIVATION_PLANES = 7,/* bytes of cj_planes for (m, n_pad)   */
    MOSAIC_OP_UNMASK_PLANES = 8     /* bytes of L_planes for m              */
} mosaic_op;

/* Bytes of `ws` the op needs for the given sizes and variant-independent
 * worst case (0 on invalid arguments).  Arguments unused by an op are
 * ignored. */
size_t mosaic_workspace_bytes(int op, int64_t m, int64_t n_pad, int64_t l,
                              const mosaic_params *p);

#ifdef __cplusplus
}
#endif

#endif /* MOSAIC_H */
