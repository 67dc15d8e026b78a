/*
 * MOSAIC oracle: a plain, slow, obviously correct CPU implementation of the
 * masked ring-matmul path (Pi_Sec-Approx-MatMul, Sec. 3.2 protocol box, and
 * Pi_Sec-Linear, Sec. 4 protocol box).
 *
 * TEST INFRASTRUCTURE.  Only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg may load this library.  It shares no code,
 * header, table or constant with the CUDA library; the two meet only through
 * the seeded inputs.
 *
 * Orientation follows the paper: W is m x n, X is n x l, Y = W X is m x l.
 * All ring arithmetic is uint32_t, i.e. exact in Z_{2^32} (kappa = 32,
 * Sec. 5.2 "Emulation approach": native 32-bit wraparound).
 *
 * Where the paper leaves a detail open (PRG, samplers, FWHT stage order,
 * rounding), the readings below are this build's definitions; each function
 * names the reading it takes.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#include <math.h>

/* ---------------------------------------------------------------------- */
/* PRG: ChaCha20 block function in counter mode (RFC 8439 Sec. 2.3).       */
/* The paper asks for masks "sampled" from uniform / Gaussian / sparse     */
/* distributions (Sec. 3.2 box, Init W step 1, Init X step 1a) without      */
/* naming a generator; a cryptographic counter-mode PRG is the reading.     */
/* ---------------------------------------------------------------------- */

static uint32_t rotl32(uint32_t v, int c) { return (v << c) | (v >> (32 - c)); }

static void quarter_round(uint32_t *x, int a, int b, int c, int d)
{
    x[a] += x[b]; x[d] ^= x[a]; x[d] = rotl32(x[d], 16);
    x[c] += x[d]; x[b] ^= x[c]; x[b] = rotl32(x[b], 12);
    x[a] += x[b]; x[d] ^= x[a]; x[d] = rotl32(x[d], 8);
    x[c] += x[d]; x[b] ^= x[c]; x[b] = rotl32(x[b], 7);
}

/* One 64-byte block: state = constants | key | counter | nonce, `rounds`
 * rounds (alternating column and diagonal rounds), then add the input state. */
void orc_chacha_block(const uint32_t key[8], uint32_t counter, const uint32_t nonce[3],
                      int rounds, uint32_t out[16])
{
    uint32_t s[16], x[16];
    s[0] = 0x61707865u; s[1] = 0x3320646eu; s[2] = 0x79622d32u; s[3] = 0x6b206574u;
    for (int i = 0; i < 8; i++) s[4 + i] = key[i];
    s[12] = counter;
    s[13] = nonce[0]; s[14] = nonce[1]; s[15] = nonce[2];
    memcpy(x, s, sizeof x);
    for (int r = 0; r < rounds; r += 2) {
        quarter_round(x, 0, 4, 8, 12);
        quarter_round(x, 1, 5, 9, 13);
        quarter_round(x, 2, 6, 10, 14);
        quarter_round(x, 3, 7, 11, 15);
        quarter_round(x, 0, 5, 10, 15);
        quarter_round(x, 1, 6, 11, 12);
        quarter_round(x, 2, 7, 8, 13);
        quarter_round(x, 3, 4, 9, 14);
    }
    for (int i = 0; i < 16; i++) out[i] = x[i] + s[i];
}

/* Word w of stream (tag, stream_id) is word w mod 16 of block floor(w/16),
 * with nonce = (tag, low 32 bits of stream_id, high 32 bits). */
void orc_prg_words(const uint32_t key[8], uint32_t tag, uint64_t stream_id, int rounds,
                   uint64_t first_word, int64_t count, uint32_t *out)
{
    uint32_t nonce[3] = { tag, (uint32_t)stream_id, (uint32_t)(stream_id >> 32) };
    uint32_t blk[16];
    uint64_t cur_block = UINT64_MAX;
    for (int64_t i = 0; i < count; i++) {
        uint64_t w = first_word + (uint64_t)i;
        uint64_t b = w / 16;
        if (b != cur_block) {
            orc_chacha_block(key, (uint32_t)b, nonce, rounds, blk);
            cur_block = b;
        }
        out[i] = blk[w % 16];
    }
}

/* Uniform ring elements (Sec. 3.2 box, "L <- Z^{m x r_d}" etc.): element
 * (i, j) of a rows x cols matrix is stream word i*cols + j. */
void orc_sample_uniform(const uint32_t key[8], uint32_t tag, uint64_t stream_id, int rounds,
                        int64_t rows, int64_t cols, uint32_t *out)
{
    orc_prg_words(key, tag, stream_id, rounds, 0, rows * cols, out);
}

/* Discrete Gaussian over Z_{2^32} with Pr[k] ~ exp(-k^2 / (2 sigma^2))
 * (Sec. 3.1, Thm 3.2 statement).  Inversion sampling: element e takes
 * u = word(2e) | word(2e+1) << 32 and returns the smallest k_j = j - B with
 * u < table[j]; if there is none it returns B.  table[j] = floor(2^64 CDF(k_j))
 * is passed in (the caller computes it to high precision).  The result is the
 * ring element k (two's complement). */
void orc_sample_gaussian(const uint32_t key[8], uint32_t tag, uint64_t stream_id, int rounds,
                         const uint64_t *table, int bound, int64_t count, uint32_t *out)
{
    uint32_t *w = (uint32_t *)malloc(sizeof(uint32_t) * 2 * (size_t)(count > 0 ? count : 1));
    orc_prg_words(key, tag, stream_id, rounds, 0, 2 * count, w);
    for (int64_t e = 0; e < count; e++) {
        uint64_t u = (uint64_t)w[2 * e] | ((uint64_t)w[2 * e + 1] << 32);
        int32_t k = bound;
        for (int j = 0; j <= 2 * bound; j++) {
            if (u < table[j]) { k = j - bound; break; }
        }
        out[e] = (uint32_t)k;
    }
    free(w);
}

/* Elements [first, first + count) of the same Gaussian stream (element e
 * still reads words 2e and 2e + 1), for sampled checks of large matrices. */
void orc_sample_gaussian_at(const uint32_t key[8], uint32_t tag, uint64_t stream_id, int rounds,
                            const uint64_t *table, int bound, int64_t first, int64_t count,
                            uint32_t *out)
{
    uint32_t *w = (uint32_t *)malloc(sizeof(uint32_t) * 2 * (size_t)(count > 0 ? count : 1));
    orc_prg_words(key, tag, stream_id, rounds, 2 * (uint64_t)first, 2 * count, w);
    for (int64_t e = 0; e < count; e++) {
        uint64_t u = (uint64_t)w[2 * e] | ((uint64_t)w[2 * e + 1] << 32);
        int32_t k = bound;
        for (int j = 0; j <= 2 * bound; j++) {
            if (u < table[j]) { k = j - bound; break; }
        }
        out[e] = (uint32_t)k;
    }
    free(w);
}

/* Sparse rows with exactly t nonzeros (LPN noise of Hamming weight t,
 * Example 3.1; S_i and T_i in the Sec. 3.2 box).  Row j draws from its own
 * window of 65536 stream words starting at word j * 65536: positions
 * p = (w * r) >> 32, skipping repeats, until t distinct positions; then
 * values = the next nonzero words.  Positions and values are kept in draw
 * order.  Returns 0, or -1 if some row exhausts its window. */
#define ORC_SPARSE_WINDOW 65536
int orc_sample_sparse(const uint32_t key[8], uint32_t tag, uint64_t stream_id, int rounds,
                      int64_t rows, uint32_t r, int t, uint32_t *idx, uint32_t *val)
{
    uint32_t *w = (uint32_t *)malloc(sizeof(uint32_t) * ORC_SPARSE_WINDOW);
    int status = 0;
    for (int64_t j = 0; j < rows && status == 0; j++) {
        orc_prg_words(key, tag, stream_id, rounds, (uint64_t)j * ORC_SPARSE_WINDOW,
                      ORC_SPARSE_WINDOW, w);
        int pos = 0, got = 0;
        while (got < t && pos < ORC_SPARSE_WINDOW) {
            uint32_t p = (uint32_t)(((uint64_t)w[pos++] * r) >> 32);
            int seen = 0;
            for (int q = 0; q < got; q++)
                if (idx[j * t + q] == p) { seen = 1; break; }
            if (!seen) idx[j * t + got++] = p;
        }
        int nv = 0;
        while (nv < t && pos < ORC_SPARSE_WINDOW) {
            uint32_t v = w[pos++];
            if (v != 0) val[j * t + nv++] = v;
        }
        if (got < t || nv < t) status = -1;
    }
    free(w);
    return status;
}

/* Row `row` alone of the sparse matrix above (same window, same rule). */
int orc_sample_sparse_row(const uint32_t key[8], uint32_t tag, uint64_t stream_id, int rounds,
                          int64_t row, uint32_t r, int t, uint32_t *idx, uint32_t *val)
{
    uint32_t *w = (uint32_t *)malloc(sizeof(uint32_t) * ORC_SPARSE_WINDOW);
    orc_prg_words(key, tag, stream_id, rounds, (uint64_t)row * ORC_SPARSE_WINDOW, ORC_SPARSE_WINDOW, w);
    int pos = 0, got = 0, nv = 0;
    while (got < t && pos < ORC_SPARSE_WINDOW) {
        uint32_t p = (uint32_t)(((uint64_t)w[pos++] * r) >> 32);
        int seen = 0;
        for (int q = 0; q < got; q++)
            if (idx[q] == p) { seen = 1; break; }
        if (!seen) idx[got++] = p;
    }
    while (nv < t && pos < ORC_SPARSE_WINDOW) {
        uint32_t v = w[pos++];
        if (v != 0) val[nv++] = v;
    }
    free(w);
    return (got < t || nv < t) ? -1 : 0;
}

/* ---------------------------------------------------------------------- */
/* Random Hadamard rotation R = H D (Sec. 4, "Random Hadamard rotation";    */
/* Pi_Sec-Linear box Init W step 1).  Each vector v of length n is          */
/* zero-padded to n_pad (a power of two), flipped by d (d_c = -1 where bit  */
/* c mod 32 of sign word c/32 is set), transformed by the unnormalised      */
/* Sylvester-order FWHT with stages h = 1, 2, 4, ..., n_pad/2 in that order, */
/* each pair (i, i+h) -> (a+b, a-b) in fp32, and finally multiplied by      */
/* fl32(1/sqrt(n_pad)) so that H is the normalised matrix (H H^T = I).       */
/* Rows of `x` are the vectors (rows of W, or columns of X taken as rows).  */
/* ---------------------------------------------------------------------- */
void orc_fwht_rows(const float *x, int64_t rows, int64_t n, int64_t ldx, int64_t n_pad,
                   const uint32_t *sign_words, float *y)
{
    const float inv = (float)(1.0 / sqrt((double)n_pad));
    float *v = (float *)malloc(sizeof(float) * (size_t)n_pad);
    for (int64_t row = 0; row < rows; row++) {
        for (int64_t c = 0; c < n_pad; c++) {
            float e = c < n ? x[row * ldx + c] : 0.0f;
            if (sign_words && ((sign_words[c / 32] >> (c % 32)) & 1u)) e = -e;
            v[c] = e;
        }
        for (int64_t h = 1; h < n_pad; h *= 2) {
            for (int64_t i = 0; i < n_pad; i += 2 * h) {
                for (int64_t j = i; j < i + h; j++) {
                    float a = v[j], b = v[j + h];
                    v[j] = a + b;
                    v[j + h] = a - b;
                }
            }
        }
        for (int64_t c = 0; c < n_pad; c++) y[row * n_pad + c] = v[c] * inv;
    }
    free(v);
}

/* Same transform in fp64 (used by the tests for orthogonality checks). */
void orc_fwht_rows_f64(const double *x, int64_t rows, int64_t n_pad,
                       const uint32_t *sign_words, double *y)
{
    const double inv = 1.0 / sqrt((double)n_pad);
    double *v = (double *)malloc(sizeof(double) * (size_t)n_pad);
    for (int64_t row = 0; row < rows; row++) {
        for (int64_t c = 0; c < n_pad; c++) {
            double e = x[row * n_pad + c];
            if (sign_words && ((sign_words[c / 32] >> (c % 32)) & 1u)) e = -e;
            v[c] = e;
        }
        for (int64_t h = 1; h < n_pad; h *= 2)
            for (int64_t i = 0; i < n_pad; i += 2 * h)
                for (int64_t j = i; j < i + h; j++) {
                    double a = v[j], b = v[j + h];
                    v[j] = a + b;
                    v[j + h] = a - b;
                }
        for (int64_t c = 0; c < n_pad; c++) y[row * n_pad + c] = v[c] * inv;
    }
    free(v);
}

/* ---------------------------------------------------------------------- */
/* Per-vector quantisation (Pi_Sec-Linear box, Init W step 2 and Online     */
/* step 1; Sec. 4 straw-man paragraph): s = ||v||_inf / q_max in fp32,      */
/* v_hat = round(v / s) with IEEE division and ties-to-even rounding,       */
/* clamped to [-q_max, q_max], embedded in Z_{2^32} as two's complement.    */
/* s = 0 gives the zero code.  A vector holding a non-finite value gets     */
/* scale NaN and the zero code.                                             */
/* ---------------------------------------------------------------------- */
void orc_encode_rows(const float *v, int64_t rows, int64_t n_pad, int32_t qmax,
                     uint32_t *code, float *scale)
{
    for (int64_t row = 0; row < rows; row++) {
        const float *x = v + row * n_pad;
        float absmax = 0.0f;
        int finite = 1;
        for (int64_t c = 0; c < n_pad; c++) {
            if (!isfinite(x[c])) finite = 0;
            float a = fabsf(x[c]);
            if (a > absmax) absmax = a;
        }
        float s = finite ? absmax / (float)qmax : NAN;
        scale[row] = s;
        for (int64_t c = 0; c < n_pad; c++) {
            int32_t q = 0;
            if (finite && s != 0.0f) {
                float f = rintf(x[c] / s);
                if (f > (float)qmax) f = (float)qmax;
                if (f < -(float)qmax) f = -(float)qmax;
                q = (int32_t)f;
            }
            code[row * n_pad + c] = (uint32_t)q;
        }
    }
}

/* ---------------------------------------------------------------------- */
/* Ring matrix product over Z_{2^32}: C = A B (A: M x K, B: K x N), the     */
/* naive triple loop with uint32 wraparound (Sec. 5.2: reduction to Z_{2^32} */
/* is native 32-bit overflow).  Rows of C are independent (OpenMP).         */
/* ---------------------------------------------------------------------- */
void orc_ring_matmul(const uint32_t *A, int64_t lda, const uint32_t *B, int64_t ldb,
                     uint32_t *C, int64_t ldc, int64_t M, int64_t N, int64_t K)
{
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t i = 0; i < M; i++) {
        uint32_t *c = C + i * ldc;
        for (int64_t j = 0; j < N; j++) c[j] = 0;
        for (int64_t k = 0; k < K; k++) {
            const uint32_t a = A[i * lda + k];
            const uint32_t *b = B + k * ldb;
            for (int64_t j = 0; j < N; j++) c[j] += a * b[j];
        }
    }
}

/* out = S Q, S (rows x r) row-sparse: row j holds t (position, value) pairs;
 * Q is r x l.  (S_{i+1} Q_i in the unmask step, Sec. 3.2 box step 5.) */
void orc_sparse_rows_matmul(const uint32_t *idx, const uint32_t *val, int64_t rows, int t,
                            const uint32_t *Q, int64_t ldq, int64_t l, uint32_t *out)
{
#pragma omp parallel for schedule(static)
    for (int64_t j = 0; j < rows; j++) {
        for (int64_t k = 0; k < l; k++) out[j * l + k] = 0;
        for (int q = 0; q < t; q++) {
            const uint32_t p = idx[j * t + q], v = val[j * t + q];
            for (int64_t k = 0; k < l; k++) out[j * l + k] += v * Q[p * ldq + k];
        }
    }
}

/* out = A T, A (rows x r) dense, T (r x l) column-sparse: column k holds t
 * (position, value) pairs.  (N_1..N_i T_{i+1} in U_x and J_i T_{i+1} in K,
 * Sec. 3.2 box Init X steps 1b-1c.) */
void orc_matmul_sparse_cols(const uint32_t *A, int64_t lda, int64_t rows,
                            const uint32_t *idx, const uint32_t *val, int64_t l, int t,
                            uint32_t *out)
{
#pragma omp parallel for schedule(static)
    for (int64_t j = 0; j < rows; j++) {
        for (int64_t k = 0; k < l; k++) {
            uint32_t acc = 0;
            for (int q = 0; q < t; q++)
                acc += A[j * lda + idx[k * t + q]] * val[k * t + q];
            out[j * l + k] = acc;
        }
    }
}

int orc_num_threads(void)
{
#ifdef _OPENMP
    extern int omp_get_max_threads(void);
    return omp_get_max_threads();
#else
    return 1;
#endif
}
