// extern "C" entry points of libmosaic.so: argument validation, workspace
// carving and the composition of kernels into the protocol steps of
// Pi_Sec-Approx-MatMul (Sec. 3.2 protocol box) and Pi_Sec-Linear (Sec. 4
// protocol box).  See include/mosaic.h for the contract of each call.
#include <math.h>
#include <string.h>

#include <atomic>

#include "mosaic_internal.cuh"

using namespace mosaic;

namespace mosaic {
static std::atomic<unsigned long long> g_launches{0};
void count_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }
}  // namespace mosaic

namespace {

constexpr size_t kAlign = 256;
size_t up(size_t v) { return (v + kAlign - 1) / kAlign * kAlign; }

// Bump allocator over the caller's workspace.
struct Carve {
    char *base;
    size_t cap, used;
    template <class T>
    T *take(size_t count) {
        const size_t bytes = up(count * sizeof(T));
        if (used + bytes > cap) return nullptr;
        T *p = reinterpret_cast<T *>(base + used);
        used += bytes;
        return p;
    }
};

// Carving starts at the first kAlign boundary inside ws, so every part is
// aligned (TMA operands, 16-byte vector accesses) even when the caller's
// buffer is not; its leading bytes then go unused.
Carve carve(void *ws, size_t bytes) {
    const size_t pad = (size_t)((kAlign - reinterpret_cast<uintptr_t>(ws) % kAlign) % kAlign);
    return Carve{static_cast<char *>(ws), bytes, pad < bytes ? pad : bytes};
}

bool rounds_ok(uint32_t r) { return r == 8 || r == 12 || r == 20; }

mosaic_status check_params(const mosaic_params *p) {
    if (!p) return MOSAIC_ERR_ARG;
    if (p->kappa != 32) return MOSAIC_ERR_UNSUPPORTED;
    if (p->d < 1 || p->d > 3) return MOSAIC_ERR_ARG;
    for (uint32_t i = 0; i < p->d; i++)
        if (p->r[i] < 2 || p->r[i] > 65536) return MOSAIC_ERR_ARG;
    for (uint32_t i = 1; i < p->d; i++) {
        const uint32_t t = p->t[i], r = p->r[i - 1];
        if (t < 1 || t > 1024 || t > r / 2) return MOSAIC_ERR_ARG;
    }
    if (!(p->sigma >= 0.0f && p->sigma <= 8.0f)) return MOSAIC_ERR_ARG;
    if (p->qbits < 2 || p->qbits > 16) return MOSAIC_ERR_ARG;
    if (!rounds_ok(p->rounds)) return MOSAIC_ERR_ARG;
    if (p->act_nested > 1) return MOSAIC_ERR_ARG;
    return MOSAIC_OK;
}

// Rank of the dense activation-mask factor R: r_d (nested) or r_1 (act_nested = 0).
int64_t r_act(const mosaic_params *p) { return p->act_nested ? p->r[p->d - 1] : p->r[0]; }
// Number of LPN levels in the activation mask.
uint32_t act_levels(const mosaic_params *p) { return p->act_nested ? p->d - 1 : 0; }

int64_t sum_r(const mosaic_params *p) {
    int64_t s = 0;
    for (uint32_t i = 0; i < p->d; i++) s += p->r[i];
    return s;
}
// Column / row offset of level i (1-based) inside the stacked chains.
int64_t off_r(const mosaic_params *p, uint32_t i) {
    int64_t s = 0;
    for (uint32_t q = 1; q < i; q++) s += p->r[q - 1];
    return s;
}
uint32_t tag_of(uint32_t kind, uint32_t level) { return kind | (level << 8); }
bool npad_ok(int64_t n_pad) { return is_pow2(n_pad) && n_pad >= 32 && n_pad <= 65536; }

// Bytes of digit planes a tensor-core product of an M x K by N x K pair needs.
size_t ws_gemm(int64_t M, int64_t N, int64_t K) {
    const int64_t Kp = (K + 7) / 8 * 8;
    const size_t bf16 = up(8 * (size_t)(M * Kp)) + up(8 * (size_t)(N * Kp));
    const size_t s8 = ws_mma_s8(M, N, K);   // int8 digit planes of the legacy variant
    return bf16 > s8 ? bf16 : s8;
}

// Ring product for the internal compositions (uint32 operands):
// C = (Cin ? Cin : 0) + sgn * A B^T with A(i, k) = A[i sai + k sak], B(j, k) = B[j sbj + k sbk].
// The tensor-core variant needs K-major operands with 16-byte aligned rows and
// room in `cv` for both operands' digit planes; otherwise the CUDA-core
// product runs.  The planes are dead once the product is enqueued (all work
// is ordered on `st`), so their workspace is handed back.
mosaic_status gemm_u32(int variant, Carve &cv, const uint32_t *A, int64_t sai, int64_t sak,
                       const uint32_t *B, int64_t sbj, int64_t sbk, uint32_t *C, int64_t ldc,
                       const uint32_t *Cin, int64_t ldcin, int sgn, int64_t M, int64_t N, int64_t K,
                       cudaStream_t st) {
    const bool want_tc = variant == MOSAIC_GEMM_TC || (variant == MOSAIC_GEMM_AUTO && tc_available());
    // A few tokens: stream B once at 4 bytes per element instead of its planes.
    if (want_tc && sak == 1 && sbk == 1 && skinny_ok(A, sai, B, sbj, M, K))
        return ring_gemm_skinny(A, sai, B, sbj, C, ldc, Cin, ldcin, sgn, M, N, K, st);
    const bool tc_ok = want_tc && sak == 1 && sbk == 1 && sai % 4 == 0 && sbj % 4 == 0 &&
                       aligned16(A) && aligned16(B) && K > 0 && cv.used + ws_gemm(M, N, K) <= cv.cap;
    if (!tc_ok) return ring_gemm_imad(A, sai, sak, B, sbj, sbk, C, ldc, Cin, ldcin, sgn, M, N, K, st);
    const int64_t Kp = (K + 7) / 8 * 8;
    const size_t mark = cv.used;
    uint16_t *Ap = cv.take<uint16_t>((size_t)(4 * M * Kp));
    uint16_t *Bp = cv.take<uint16_t>((size_t)(4 * N * Kp));
    MOSAIC_TRY(digit_split(A, sai, M, K, Ap, Kp, M * Kp, st));
    MOSAIC_TRY(digit_split(B, sbj, N, K, Bp, Kp, N * Kp, st));
    const mosaic_status s =
        ring_gemm_tc_planes(Ap, Kp, M * Kp, Bp, Kp, N * Kp, C, ldc, Cin, ldcin, sgn, M, N, K, st);
    cv.used = mark;
    return s;
}

size_t ws_chains(int64_t n_pad, const mosaic_params *p) {
    size_t s = 0;
    int64_t prev = n_pad;
    for (uint32_t i = 1; i <= p->d; i++) {
        const int64_t ri = p->r[i - 1];
        if (i >= 2) s += up(sizeof(uint32_t) * (size_t)(ri * prev)) * 2;   // M_i and N_i
        prev = ri;
    }
    return s;
}
int64_t sum_r(const mosaic_params *p);
// Minimum workspaces (CUDA-core products) and the extra room that lets the
// products run on the tensor cores.
size_t ws_weight_min(int64_t m, int64_t n_pad, const mosaic_params *) {
    return up(sizeof(uint32_t) * (size_t)(m * n_pad));
}
size_t ws_weight(int64_t m, int64_t n_pad, const mosaic_params *p) {
    return ws_weight_min(m, n_pad, p) + ws_gemm(m, sum_r(p), n_pad);
}
size_t ws_activation_min(int64_t l, const mosaic_params *p) {
    size_t s = up(sizeof(uint32_t) * (size_t)(l * r_act(p)));
    for (uint32_t i = 2; i <= act_levels(p) + 1; i++) s += 2 * up(sizeof(uint32_t) * (size_t)(l * p->t[i - 1]));
    return s;
}
int64_t kpad8(int64_t k) { return (k + 7) / 8 * 8; }
size_t ws_activation(int64_t m, int64_t n_pad, int64_t l, const mosaic_params *p) {
    // Room for the combined tensor-core product: planes of R^T and of [C; J].
    const size_t g = ws_gemm(l, n_pad + m, r_act(p));
    return ws_activation_min(l, p) + g;
}
// The activation planes buffer: digit planes of [C-factor; J-factor], then,
// for each LPN level i of a nested activation mask, the tile images of the
// segments C_i and J_i that the level's gathers stage (byte offsets; 0 where
// a level has none).
struct ActLayout {
    size_t c_img[2], j_img[2];
    size_t bytes;
};
ActLayout act_layout(int64_t m, int64_t n_pad, const mosaic_params *p) {
    ActLayout L{{0, 0}, {0, 0}, 0};
    size_t off = up(8 * (size_t)((n_pad + m) * kpad8(r_act(p))));
    for (uint32_t i = 1; i <= act_levels(p); i++) {
        const uint32_t ri = p->r[i - 1];
        const size_t wc = tile_image_words(n_pad, ri), wj = tile_image_words(m, ri);
        if (!wc || !wj) continue;
        L.c_img[i - 1] = off;
        off += up(4 * wc);
        L.j_img[i - 1] = off;
        off += up(4 * wj);
    }
    L.bytes = off;
    return L;
}
size_t activation_planes_bytes(int64_t m, int64_t n_pad, const mosaic_params *p) {
    return act_layout(m, n_pad, p).bytes;
}
size_t unmask_planes_bytes(int64_t m, const mosaic_params *p) {
    return 8 * (size_t)(m * kpad8(p->r[p->d - 1]));
}
size_t ws_unmask_min(int64_t m, int64_t l, const mosaic_params *) {
    return up(sizeof(uint32_t) * (size_t)(l * m));
}
// Tile images of the Q_i segments of Z for the unmask gathers (tokens are the
// staged rows); built per call when the workspace has room.
size_t unmask_images_bytes(int64_t l, const mosaic_params *p) {
    size_t s = 0;
    if (l <= 4) return 0;   // a few tokens take the single-pass gather, which stages rows directly
    for (uint32_t i = 1; i < p->d; i++) s += up(4 * tile_image_words(l, p->r[i - 1]));
    return s;
}
// Line-offset copies of the S lists for the levels that take the tiled gather.
size_t unmask_lines_bytes(int64_t m, int64_t l, const mosaic_params *p) {
    size_t s = 0;
    for (uint32_t i = 1; i < p->d; i++)
        if (pgather_takes(l, p->r[i - 1], (int)p->t[i])) s += up(4 * (size_t)(m * p->t[i]));
    return s;
}
size_t ws_unmask(int64_t m, int64_t l, const mosaic_params *p) {
    return ws_unmask_min(m, l, p) + ws_gemm(l, m, p->r[p->d - 1]) + unmask_images_bytes(l, p) +
           unmask_lines_bytes(m, l, p);
}

}  // namespace

extern "C" {

uint64_t mosaic_kernel_launches(void) { return mosaic::g_launches.load(std::memory_order_relaxed); }

void mosaic_default_params(mosaic_params *p) {
    if (!p) return;
    memset(p, 0, sizeof *p);
    p->kappa = 32;
    p->d = 3;
    p->r[0] = 1536; p->r[1] = 1024; p->r[2] = 652;
    p->t[0] = 0; p->t[1] = 80; p->t[2] = 80;
    p->sigma = 0.5f;
    p->qbits = 16;
    p->rounds = 20;
    p->act_nested = 1;
}

const char *mosaic_status_string(mosaic_status s) {
    switch (s) {
        case MOSAIC_OK: return "ok";
        case MOSAIC_ERR_ARG: return "invalid argument";
        case MOSAIC_ERR_SHAPE: return "invalid shape";
        case MOSAIC_ERR_ALIGN: return "misaligned pointer or leading dimension";
        case MOSAIC_ERR_UNSUPPORTED: return "unsupported by this build";
        case MOSAIC_ERR_CUDA: return "CUDA error";
        case MOSAIC_ERR_WORKSPACE: return "workspace too small";
        case MOSAIC_ERR_TIMEOUT: return "device wait timed out";
    }
    return "unknown status";
}

int32_t mosaic_qmax(int64_t n_pad, uint32_t qbits) {
    if (!npad_ok(n_pad) || qbits < 2 || qbits > 16) return 0;
    const int64_t cap = ((int64_t)1 << (qbits - 1)) - 1;
    const int64_t lim = ((int64_t)1 << 31) / n_pad;
    int64_t q = (int64_t)sqrt((double)lim);
    while (q * q > lim) q--;
    while ((q + 1) * (q + 1) <= lim) q++;
    return (int32_t)(q < cap ? q : cap);
}

int mosaic_gaussian_table(float sigma, uint64_t *table, int capacity) {
    if (!(sigma > 0.0f && sigma <= 8.0f) || !table) return -1;
    unsigned long long t[2 * kMaxGaussBound + 1];
    const int B = gaussian_table_host(sigma, t);
    if (capacity < 2 * B + 1) return -1;
    for (int i = 0; i < 2 * B + 1; i++) table[i] = t[i];
    return B;
}

mosaic_status mosaic_prg_uniform(const mosaic_key *key, uint32_t tag, uint64_t stream_id,
                                 uint32_t rounds, int64_t rows, int64_t cols, uint32_t *out,
                                 int64_t ldo, void *stream) {
    RoleScope role("prg");
    if (!key || !rounds_ok(rounds)) return MOSAIC_ERR_ARG;
    if (rows < 0 || cols < 0 || ldo < cols) return MOSAIC_ERR_SHAPE;
    if (rows * cols >= ((int64_t)1 << 36)) return MOSAIC_ERR_SHAPE;
    if (rows * cols == 0) return MOSAIC_OK;
    if (!out) return MOSAIC_ERR_ARG;
    return prg_uniform(to_key(key), tag, stream_id, (int)rounds, rows, cols, out, ldo,
                       as_stream(stream));
}

mosaic_status mosaic_prg_gaussian(const mosaic_key *key, uint32_t tag, uint64_t stream_id,
                                  uint32_t rounds, float sigma, int64_t count, uint32_t *out,
                                  void *stream) {
    RoleScope role("prg");
    if (!key || !rounds_ok(rounds)) return MOSAIC_ERR_ARG;
    if (!(sigma >= 0.0f && sigma <= 8.0f)) return MOSAIC_ERR_ARG;
    if (count < 0 || count >= ((int64_t)1 << 35)) return MOSAIC_ERR_SHAPE;
    if (count == 0) return MOSAIC_OK;
    if (!out) return MOSAIC_ERR_ARG;
    return prg_gaussian(to_key(key), tag, stream_id, (int)rounds, sigma, count, out,
                        as_stream(stream));
}

mosaic_status mosaic_prg_sparse(const mosaic_key *key, uint32_t tag, uint64_t stream_id,
                                uint32_t rounds, int64_t rows, uint32_t r, uint32_t t,
                                uint32_t *idx, uint32_t *val, uint32_t *fail, void *stream) {
    RoleScope role("prg");
    if (!key || !rounds_ok(rounds)) return MOSAIC_ERR_ARG;
    if (rows < 0 || rows >= ((int64_t)1 << 20)) return MOSAIC_ERR_SHAPE;
    if (t < 1 || t > 1024 || r < 2 || t > r / 2) return MOSAIC_ERR_ARG;
    if (rows == 0) return MOSAIC_OK;
    if (!idx || !val) return MOSAIC_ERR_ARG;
    return prg_sparse(to_key(key), tag, stream_id, (int)rounds, rows, r, t, idx, val, fail,
                      as_stream(stream));
}

mosaic_status mosaic_hadamard(const float *x, int64_t ldx, float *y, int64_t rows, int64_t n,
                              int64_t n_pad, const uint32_t *sign_words, void *stream) {
    RoleScope role("hadamard");
    if (!npad_ok(n_pad) || n < 1 || n > n_pad || rows < 0 || ldx < n) return MOSAIC_ERR_SHAPE;
    if (rows == 0) return MOSAIC_OK;
    if (!x || !y) return MOSAIC_ERR_ARG;
    if (!aligned16(y)) return MOSAIC_ERR_ALIGN;
    return fwht_encode(x, ldx, rows, n, n_pad, sign_words, 1, 0, y, 0, nullptr, 0, nullptr, 0,
                       nullptr, nullptr, as_stream(stream));
}

mosaic_status mosaic_encode(const float *x, int64_t ldx, int64_t rows, int64_t n, int64_t n_pad,
                            int32_t qmax, int rotate, const uint32_t *sign_words,
                            const uint32_t *mask, int64_t ldm, uint32_t *out, int64_t ldo,
                            float *scale, uint16_t *planes, void *stream) {
    RoleScope role("encode");
    if (!npad_ok(n_pad) || n < 1 || n > n_pad || rows < 0 || ldx < n || ldo < n_pad)
        return MOSAIC_ERR_SHAPE;
    if (mask && ldm < n_pad) return MOSAIC_ERR_SHAPE;
    if (qmax < 1 || qmax > 32767 || (rotate != 0 && rotate != 1)) return MOSAIC_ERR_ARG;
    if (rows == 0) return MOSAIC_OK;
    if (!x || !out || !scale) return MOSAIC_ERR_ARG;
    if (!aligned16(out) || ldo % 4 || (mask && (!aligned16(mask) || ldm % 4)) ||
        (planes && !aligned16(planes)))
        return MOSAIC_ERR_ALIGN;
    return fwht_encode(x, ldx, rows, n, n_pad, sign_words, rotate, 1, nullptr, qmax, mask, ldm, out,
                       ldo, scale, planes, as_stream(stream));
}

mosaic_status mosaic_digit_split(const uint32_t *a, int64_t lda, int64_t rows, int64_t cols,
                                 uint16_t *planes, void *stream) {
    RoleScope role("digit_split");
    if (rows < 0 || cols < 0 || cols % 8 || lda < cols) return MOSAIC_ERR_SHAPE;
    if (rows == 0 || cols == 0) return MOSAIC_OK;
    if (!a || !planes) return MOSAIC_ERR_ARG;
    if (!aligned16(a) || !aligned16(planes) || lda % 4) return MOSAIC_ERR_ALIGN;
    return digit_split(a, lda, rows, cols, planes, cols, rows * cols, as_stream(stream));
}

int mosaic_gemm_variant_available(int variant) {
    switch (variant) {
        case MOSAIC_GEMM_AUTO: return 1;
        case MOSAIC_GEMM_IMAD: return 1;
        case MOSAIC_GEMM_TC: return tc_available() ? 1 : 0;
        case MOSAIC_GEMM_MMA_S8: return mma_s8_available() ? 1 : 0;
    }
    return 0;
}

mosaic_status mosaic_ring_gemm(const uint32_t *A, int64_t lda, const uint32_t *B, int64_t ldb,
                               uint32_t *C, int64_t ldc, int64_t M, int64_t N, int64_t K,
                               int variant, void *ws, size_t ws_bytes, void *stream) {
    RoleScope role("ring_gemm");
    if (M < 0 || N < 0 || K < 0 || K > ((int64_t)1 << 20)) return MOSAIC_ERR_SHAPE;
    if (lda < K || ldb < K || ldc < N) return MOSAIC_ERR_SHAPE;
    if (variant < MOSAIC_GEMM_AUTO || variant > MOSAIC_GEMM_IMAD) return MOSAIC_ERR_ARG;
    if (M == 0 || N == 0) return MOSAIC_OK;
    if (!A || !B || !C) return MOSAIC_ERR_ARG;
    cudaStream_t st = as_stream(stream);
    if (K == 0)   // empty sums: C = 0 whatever the variant
        return cudaMemset2DAsync(C, (size_t)ldc * 4, 0, (size_t)N * 4, (size_t)M, st) == cudaSuccess
                   ? MOSAIC_OK
                   : MOSAIC_ERR_CUDA;
    const bool tc_layout = aligned16(A) && aligned16(B) && lda % 4 == 0 && ldb % 4 == 0;
    if (variant == MOSAIC_GEMM_IMAD || (variant == MOSAIC_GEMM_AUTO && (!tc_available() || !tc_layout)))
        return ring_gemm_imad(A, lda, 1, B, ldb, 1, C, ldc, nullptr, 0, 1, M, N, K, st);
    if (variant == MOSAIC_GEMM_MMA_S8)
        return ring_gemm_mma_s8(A, lda, B, ldb, C, ldc, nullptr, 0, 1, M, N, K, ws, ws_bytes, st);
    if (!tc_available()) return MOSAIC_ERR_UNSUPPORTED;
    // A few tokens: the streaming kernel reads B once, no planes needed.
    if (skinny_ok(A, lda, B, ldb, M, K))
        return ring_gemm_skinny(A, lda, B, ldb, C, ldc, nullptr, 0, 1, M, N, K, st);
    const int64_t Kp = (K + 7) / 8 * 8;
    if (!aligned16(A) || !aligned16(B) || lda % 4 || ldb % 4) return MOSAIC_ERR_ALIGN;
    Carve cv = carve(ws, ws_bytes);
    // Up to kTcwMaxM tokens: tensor cores, B read once as uint32 and split on the chip.
    if (tcw_ok(A, lda, B, ldb, M, N, K)) {
        uint16_t *Ap = cv.take<uint16_t>(tcw_ws_bytes(M, K) / 2);
        if (!Ap) return MOSAIC_ERR_WORKSPACE;
        return ring_gemm_tcw(A, lda, B, ldb, C, ldc, M, N, K, Ap, st);
    }
    // Tensor-core variant: split both operands into digit planes in ws.
    uint16_t *Ap = cv.take<uint16_t>((size_t)(4 * M * Kp));
    uint16_t *Bp = cv.take<uint16_t>((size_t)(4 * N * Kp));
    if (!Ap || !Bp) return MOSAIC_ERR_WORKSPACE;
    MOSAIC_TRY(digit_split(A, lda, M, K, Ap, Kp, M * Kp, st));
    MOSAIC_TRY(digit_split(B, ldb, N, K, Bp, Kp, N * Kp, st));
    return ring_gemm_tc_planes(Ap, Kp, M * Kp, Bp, Kp, N * Kp, C, ldc, nullptr, 0, 1, M, N, K, st);
}

mosaic_status mosaic_ring_gemm_planes(const uint16_t *A_planes, int64_t ldpa, int64_t a_plane,
                                      const uint16_t *B_planes, int64_t ldpb, int64_t b_plane,
                                      uint32_t *C, int64_t ldc, int64_t M, int64_t N, int64_t K,
                                      int variant, void *stream) {
    RoleScope role("ring_gemm");
    if (M < 0 || N < 0 || K < 0 || K > ((int64_t)1 << 20)) return MOSAIC_ERR_SHAPE;
    if (ldpa < K || ldpb < K || ldc < N || a_plane < M * ldpa || b_plane < N * ldpb)
        return MOSAIC_ERR_SHAPE;
    if (variant != MOSAIC_GEMM_TC && variant != MOSAIC_GEMM_AUTO) return MOSAIC_ERR_UNSUPPORTED;
    if (M == 0 || N == 0) return MOSAIC_OK;
    if (!A_planes || !B_planes || !C) return MOSAIC_ERR_ARG;
    if (!aligned16(A_planes) || !aligned16(B_planes) || ldpa % 8 || ldpb % 8 || a_plane % 8 ||
        b_plane % 8)
        return MOSAIC_ERR_ALIGN;
    if (!tc_available()) return MOSAIC_ERR_UNSUPPORTED;
    return ring_gemm_tc_planes(A_planes, ldpa, a_plane, B_planes, ldpb, b_plane, C, ldc, nullptr, 0,
                               1, M, N, K, as_stream(stream));
}

mosaic_status mosaic_selftest_wait(int64_t limit_us, void *stream) {
    if (limit_us < 1 || limit_us > 1000000) return MOSAIC_ERR_ARG;
    return wait_probe((unsigned long long)limit_us * 1000ull, as_stream(stream));
}

mosaic_status mosaic_device_status(void *stream) {
    const mosaic_status s = device_status(as_stream(stream));
    const mosaic_status s2 = skinny_status();
    const mosaic_status s3 = gather_status();
    const mosaic_status s4 = tcw_status();
    const mosaic_status s5 = fwht_status();
    if (s != MOSAIC_OK) return s;
    if (s2 != MOSAIC_OK) return s2;
    if (s3 != MOSAIC_OK) return s3;
    if (s4 != MOSAIC_OK) return s4;
    if (s5 != MOSAIC_OK) return s5;
    return cudaGetLastError() == cudaSuccess ? MOSAIC_OK : MOSAIC_ERR_CUDA;
}

size_t mosaic_workspace_bytes(int op, int64_t m, int64_t n_pad, int64_t l, const mosaic_params *p) {
    if (m < 0 || n_pad < 0 || l < 0) return 0;
    switch (op) {
        case MOSAIC_OP_RING_GEMM: return ws_gemm(m, n_pad, l);
        case MOSAIC_OP_MASK_CHAINS: return check_params(p) == MOSAIC_OK ? ws_chains(n_pad, p) : 0;
        case MOSAIC_OP_MASK_WEIGHT: return check_params(p) == MOSAIC_OK ? ws_weight(m, n_pad, p) : 0;
        case MOSAIC_OP_MASK_ACTIVATION:
            return check_params(p) == MOSAIC_OK ? ws_activation(m, n_pad, l, p) : 0;
        case MOSAIC_OP_UNMASK: return check_params(p) == MOSAIC_OK ? ws_unmask(m, l, p) : 0;
        case MOSAIC_OP_FREIVALDS_CHECK: return 2 * up(sizeof(uint32_t) * (size_t)(m * l));
        case MOSAIC_OP_ACTIVATION_PLANES:
            return check_params(p) == MOSAIC_OK ? activation_planes_bytes(m, n_pad, p) : 0;
        case MOSAIC_OP_UNMASK_PLANES: return check_params(p) == MOSAIC_OK ? unmask_planes_bytes(m, p) : 0;
    }
    return 0;
}

mosaic_status mosaic_mask_chains(const mosaic_params *p, const mosaic_key *key, uint64_t chain_id,
                                 int64_t n_pad, uint32_t *P, uint32_t *C, uint32_t *CT, void *ws,
                                 size_t ws_bytes, void *stream) {
    RoleScope role("init_w");
    MOSAIC_TRY(check_params(p));
    if (!key) return MOSAIC_ERR_ARG;
    if (!npad_ok(n_pad)) return MOSAIC_ERR_SHAPE;
    if (!P || !C || !CT) return MOSAIC_ERR_ARG;
    if (ws_bytes < ws_chains(n_pad, p)) return MOSAIC_ERR_WORKSPACE;
    cudaStream_t st = as_stream(stream);
    const Key k = to_key(key);
    const int R = (int)p->rounds;
    const int64_t Sr = sum_r(p);
    Carve cv = carve(ws, ws_bytes);
    // Level 1: M_1 (r_1 x n_pad) is P_1; N_1 (n_pad x r_1) is C_1.
    MOSAIC_TRY(prg_uniform(k, tag_of(MOSAIC_TAG_M, 1), chain_id, R, p->r[0], n_pad, P, n_pad, st));
    MOSAIC_TRY(prg_uniform(k, tag_of(MOSAIC_TAG_N, 1), chain_id, R, n_pad, p->r[0], C, Sr, st));
    for (uint32_t i = 2; i <= p->d; i++) {
        const int64_t ri = p->r[i - 1], rp = p->r[i - 2];
        const int64_t oi = off_r(p, i), op = off_r(p, i - 1);
        uint32_t *Mi = cv.take<uint32_t>((size_t)(ri * rp));
        uint32_t *Ni = cv.take<uint32_t>((size_t)(rp * ri));
        if (!Mi || !Ni) return MOSAIC_ERR_WORKSPACE;
        MOSAIC_TRY(prg_uniform(k, tag_of(MOSAIC_TAG_M, i), chain_id, R, ri, rp, Mi, rp, st));
        MOSAIC_TRY(prg_uniform(k, tag_of(MOSAIC_TAG_N, i), chain_id, R, rp, ri, Ni, ri, st));
        // P_i = M_i P_{i-1}:  C(a, c) = sum_b M_i[a][b] P_{i-1}[b][c]
        MOSAIC_TRY(ring_gemm_imad(Mi, rp, 1, P + op * n_pad, 1, n_pad, P + oi * n_pad, n_pad,
                                  nullptr, 0, 1, ri, n_pad, rp, st));
        // C_i = C_{i-1} N_i:  C(c, b) = sum_a C_{i-1}[c][a] N_i[a][b]
        MOSAIC_TRY(ring_gemm_imad(C + op, Sr, 1, Ni, 1, ri, C + oi, Sr, nullptr, 0, 1, n_pad, ri,
                                  rp, st));
    }
    return transpose_u32(C, Sr, n_pad, Sr, CT, n_pad, st);
}

mosaic_status mosaic_mask_weight(const mosaic_params *p, const mosaic_key *key, uint64_t matrix_id,
                                 const float *W, int64_t ldw, int64_t m, int64_t n, int64_t n_pad,
                                 const uint32_t *P, const uint32_t *CT, uint32_t *sign_words,
                                 float *s_w, uint32_t *L, uint32_t *S_idx, uint32_t *S_val,
                                 uint32_t *Wp, uint16_t *Wp_planes, uint32_t *J, int variant,
                                 void *ws, size_t ws_bytes, void *stream) {
    RoleScope role("init_w");
    MOSAIC_TRY(check_params(p));
    if (!key) return MOSAIC_ERR_ARG;
    if (!npad_ok(n_pad) || n < 1 || n > n_pad || m < 1 || ldw < n || m >= ((int64_t)1 << 20))
        return MOSAIC_ERR_SHAPE;
    if (!W || !P || !CT || !sign_words || !s_w || !L || !Wp || !J) return MOSAIC_ERR_ARG;
    if (p->d > 1 && (!S_idx || !S_val)) return MOSAIC_ERR_ARG;
    if (!aligned16(Wp) || (Wp_planes && !aligned16(Wp_planes))) return MOSAIC_ERR_ALIGN;
    if (ws_bytes < ws_weight_min(m, n_pad, p)) return MOSAIC_ERR_WORKSPACE;
    cudaStream_t st = as_stream(stream);
    const Key k = to_key(key);
    const int R = (int)p->rounds;
    const uint32_t d = p->d;
    const int64_t Sr = sum_r(p), rd = p->r[d - 1], od = off_r(p, d);
    Carve cv = carve(ws, ws_bytes);
    uint32_t *WE = cv.take<uint32_t>((size_t)(m * n_pad));
    if (!WE) return MOSAIC_ERR_WORKSPACE;

    // Pi_Sec-Linear Init W: d, then rows of W R^T quantised into W_hat (rows [0, m) of Wp).
    MOSAIC_TRY(prg_uniform(k, tag_of(MOSAIC_TAG_SIGN, 0), matrix_id, R, 1, n_pad / 32, sign_words,
                           n_pad / 32, st));
    const int32_t qmax = mosaic_qmax(n_pad, p->qbits);
    MOSAIC_TRY(fwht_encode(W, ldw, m, n, n_pad, sign_words, 1, 1, nullptr, qmax, nullptr, 0, Wp,
                           n_pad, s_w, nullptr, st));
    // E_w and W_hat + E_w.
    MOSAIC_TRY(prg_gaussian(k, tag_of(MOSAIC_TAG_EW, 0), matrix_id, R, p->sigma, m * n_pad, WE, st));
    MOSAIC_TRY(add_u32(Wp, n_pad, WE, n_pad, WE, n_pad, m, n_pad, st));
    // J_i = (W_hat + E_w) C_i for all i at once: J = WE CT^T (m x Sr); with
    // act_nested = 0 only J_1 (the first r_1 columns) is used and computed.
    const int64_t nJ = p->act_nested ? Sr : (int64_t)p->r[0];
    MOSAIC_TRY(gemm_u32(variant, cv, WE, n_pad, 1, CT, n_pad, 1, J, Sr, nullptr, 0, 1, m, nJ, n_pad, st));
    // L, S_{i+1}.
    MOSAIC_TRY(prg_uniform(k, tag_of(MOSAIC_TAG_L, 0), matrix_id, R, m, rd, L, rd, st));
    SparseLevel lev[2];
    int64_t soff = 0;
    for (uint32_t i = 1; i < d; i++) {
        const uint32_t t = p->t[i], ri = p->r[i - 1];
        MOSAIC_TRY(prg_sparse(k, tag_of(MOSAIC_TAG_S, i + 1), matrix_id, R, m, ri, t, S_idx + soff,
                              S_val + soff, nullptr, st));
        lev[i - 1] = SparseLevel{S_idx + soff, S_val + soff, (int)t, off_r(p, i), ri};
        soff += m * t;
    }
    // W' = (W_hat + E_w) + L P_d + sum_i S_{i+1} P_i.  With room in the
    // workspace (the J product's digit planes are released by now), L P_d
    // runs against P_d^T (K-major, so the tensor cores can take it) and the
    // sparse terms run on the tiled gather with the rows of P^T as its staged
    // rows; otherwise the product reads P_d strided and a plain row gather
    // reads P.
    {
        const size_t mark = cv.used;
        uint32_t *PdT = cv.take<uint32_t>((size_t)(n_pad * rd));
        if (PdT) {
            MOSAIC_TRY(transpose_u32(P + od * n_pad, n_pad, rd, n_pad, PdT, rd, st));
            MOSAIC_TRY(gemm_u32(variant, cv, L, rd, 1, PdT, rd, 1, Wp, n_pad, WE, n_pad, 1, m, n_pad, rd, st));
        } else {
            MOSAIC_TRY(gemm_u32(variant, cv, L, rd, 1, P + od * n_pad, 1, n_pad, Wp, n_pad, WE, n_pad, 1, m,
                                n_pad, rd, st));
        }
        cv.used = mark;
    }
    if (d > 1) {
        const size_t mark = cv.used;
        uint32_t *PT = cv.take<uint32_t>((size_t)(n_pad * od));   // rows [0, od) of P = P_1 .. P_{d-1}
        if (PT && od % 4 == 0) {
            MOSAIC_TRY(transpose_u32(P, n_pad, od, n_pad, PT, od, st));
            MOSAIC_TRY(sparse_gather(PT, od, 0, od, n_pad, m, false, lev, (int)d - 1, Wp, n_pad, nullptr, 0, 1,
                                     Wp, n_pad, st));
        } else {
            MOSAIC_TRY(sparse_rowgather(P, n_pad, lev, (int)d - 1, m, n_pad, Wp, n_pad, Wp, n_pad, st));
        }
        cv.used = mark;
    }
    // The server operand carries the public chains below W'.
    if (cudaMemcpyAsync(Wp + m * n_pad, P, sizeof(uint32_t) * (size_t)(Sr * n_pad),
                        cudaMemcpyDeviceToDevice, st) != cudaSuccess)
        return MOSAIC_ERR_CUDA;
    if (Wp_planes)
        MOSAIC_TRY(digit_split(Wp, n_pad, m + Sr, n_pad, Wp_planes, n_pad, (m + Sr) * n_pad, st));
    return MOSAIC_OK;
}

}  // extern "C"

namespace {

// Init X; `cj` (nullable) holds the digit planes of [C-factor; J-factor] made
// by mosaic_prepare_activation.
mosaic_status mask_activation_impl(const mosaic_params *p, const mosaic_key *key, uint64_t pass_id,
                                   const uint64_t *pass_dev, int64_t m, int64_t n_pad, int64_t l,
                                   const uint32_t *C, const uint32_t *J, const uint16_t *cj,
                                   uint32_t *Ux_tm, uint32_t *K_tm, int variant, void *ws,
                                   size_t ws_bytes, void *stream, int phase = MOSAIC_INITX_ALL) {
    RoleScope role("init_x");
    if (phase < 1 || phase > MOSAIC_INITX_ALL) return MOSAIC_ERR_ARG;
    MOSAIC_TRY(check_params(p));
    if (!key) return MOSAIC_ERR_ARG;
    if (!npad_ok(n_pad) || m < 1 || l < 0 || l >= ((int64_t)1 << 20)) return MOSAIC_ERR_SHAPE;
    if (l == 0) return MOSAIC_OK;
    if (!C || !J || !Ux_tm || !K_tm) return MOSAIC_ERR_ARG;
    if (ws_bytes < ws_activation_min(l, p)) return MOSAIC_ERR_WORKSPACE;
    cudaStream_t st = as_stream(stream);
    const Key k = to_key(key);
    const int R = (int)p->rounds;
    // Nested (Init X 1b-1c): dense factor R at rank r_d against C_d, J_d plus
    // d - 1 LPN levels.  act_nested = 0: R at rank r_1 against C_1, J_1 only.
    const uint32_t d = act_levels(p) + 1;
    const int64_t Sr = sum_r(p), rd = r_act(p), od = p->act_nested ? off_r(p, p->d) : 0;
    Carve cv = carve(ws, ws_bytes);
    uint32_t *Rt = cv.take<uint32_t>((size_t)(l * rd));
    if (!Rt) return MOSAIC_ERR_WORKSPACE;
    SparseLevel lev[2];
    uint32_t tagT[2] = {0, 0}, rT[2] = {0, 0}, tT[2] = {0, 0};
    uint32_t *ti[2] = {nullptr, nullptr}, *tv[2] = {nullptr, nullptr};
    for (uint32_t i = 1; i < d; i++) {
        const uint32_t t = p->t[i], ri = p->r[i - 1];
        ti[i - 1] = cv.take<uint32_t>((size_t)(l * t));
        tv[i - 1] = cv.take<uint32_t>((size_t)(l * t));
        if (!ti[i - 1] || !tv[i - 1]) return MOSAIC_ERR_WORKSPACE;
        tagT[i - 1] = tag_of(MOSAIC_TAG_T, i + 1);
        rT[i - 1] = ri;
        tT[i - 1] = t;
        lev[i - 1] = SparseLevel{ti[i - 1], tv[i - 1], (int)t, off_r(p, i), ri};
    }
    // U_x^T = E_x^T + R^T C_d^T + sum_i T_{i+1}^T C_i^T and
    // K^T = R^T J_d^T + sum_i T_{i+1}^T J_i^T: the two dense products share
    // R^T, so on the tensor cores they run as one product against the stacked
    // [C_d; J_d] (planes cached by mosaic_prepare_activation, or split here).
    const bool want_tc = variant == MOSAIC_GEMM_TC || (variant == MOSAIC_GEMM_AUTO && tc_available());
    const int64_t Kp = kpad8(rd), bplane = (n_pad + m) * Kp;
    const size_t need = up(8 * (size_t)(l * Kp)) + (cj ? 0 : up(8 * (size_t)bplane));
    const bool skinny = skinny_ok(Rt, rd, C + od, Sr, l, rd) && skinny_ok(Rt, rd, J + od, Sr, l, rd);
    const bool fused = want_tc && !skinny && n_pad % 128 == 0 && Sr % 4 == 0 && aligned16(C + od) &&
                       aligned16(J + od) && cv.used + need <= cv.cap;
    const size_t mark = cv.used;
    uint16_t *Rp = fused ? cv.take<uint16_t>((size_t)(4 * l * Kp)) : nullptr;
    // R (with its digit planes for the fused product), the T lists and E_x
    // (into U_x) in one launch.
    // The T lists only feed the gathers: when the tiled gather takes every
    // level, they are drawn as line offsets so that no pass rewrites them.
    bool lines = d > 1;
    for (uint32_t i = 1; i < d; i++)
        lines = lines && pgather_takes(n_pad, rT[i - 1], (int)tT[i - 1]) && pgather_takes(m, rT[i - 1], (int)tT[i - 1]);
    for (uint32_t i = 1; i < d; i++) lev[i - 1].lines = lines ? 1 : 0;
    if (phase & MOSAIC_INITX_DRAWS)
        MOSAIC_TRY(prg_initx(k, R, pass_id, pass_dev, tag_of(MOSAIC_TAG_R, 0), l, rd, Rt, Rp, Kp, (int)d - 1, tagT,
                             rT, tT, ti, tv, tag_of(MOSAIC_TAG_EX, 0), p->sigma, l * n_pad, Ux_tm, st, lines));
    if (!(phase & MOSAIC_INITX_COMPOSE)) return MOSAIC_OK;
    if (fused) {
        const uint16_t *B = cj;
        if (!B) {
            uint16_t *Bw = cv.take<uint16_t>((size_t)(4 * bplane));
            MOSAIC_TRY(digit_split(C + od, Sr, n_pad, rd, Bw, Kp, bplane, st));
            MOSAIC_TRY(digit_split(J + od, Sr, m, rd, Bw + n_pad * Kp, Kp, bplane, st));
            B = Bw;
        }
        MOSAIC_TRY(ring_gemm_tc_planes2(Rp, Kp, l * Kp, B, Kp, bplane, Ux_tm, n_pad, Ux_tm, n_pad, n_pad,
                                        K_tm, m, nullptr, 0, m, l, rd, st));
        cv.used = mark;
    } else {
        MOSAIC_TRY(gemm_u32(variant, cv, Rt, rd, 1, C + od, Sr, 1, Ux_tm, n_pad, Ux_tm, n_pad, 1, l,
                            n_pad, rd, st));
        MOSAIC_TRY(gemm_u32(variant, cv, Rt, rd, 1, J + od, Sr, 1, K_tm, m, nullptr, 0, 1, l, m, rd, st));
    }
    // With prepared planes the gathers stage C_i and J_i from their tile images.
    const ActLayout AL = act_layout(m, n_pad, p);
    auto image = [&](size_t off) -> const uint32_t * {
        return cj && off ? reinterpret_cast<const uint32_t *>(reinterpret_cast<const char *>(cj) + off) : nullptr;
    };
    if (d > 1) {
        // U_x += sum_i C_i T_{i+1} and K += sum_i J_i T_{i+1} read the same lists:
        // one launch per level serves both.
        const uint32_t *cimg[2] = {nullptr, nullptr}, *jimg[2] = {nullptr, nullptr};
        for (uint32_t i = 1; i < d; i++) {
            cimg[i - 1] = image(AL.c_img[i - 1]);
            jimg[i - 1] = image(AL.j_img[i - 1]);
        }
        MOSAIC_TRY(sparse_gather_pair(C, Sr, n_pad, Ux_tm, n_pad, cimg, J, Sr, m, K_tm, m, jimg, l, lev, (int)d - 1,
                                      st));
    }
    return MOSAIC_OK;
}

}  // namespace

extern "C" {

mosaic_status mosaic_mask_activation(const mosaic_params *p, const mosaic_key *key,
                                     uint64_t pass_id, int64_t m, int64_t n_pad, int64_t l,
                                     const uint32_t *C, const uint32_t *J, uint32_t *Ux_tm,
                                     uint32_t *K_tm, int variant, void *ws, size_t ws_bytes,
                                     void *stream) {
    return mask_activation_impl(p, key, pass_id, nullptr, m, n_pad, l, C, J, nullptr, Ux_tm, K_tm, variant,
                                ws, ws_bytes, stream);
}

mosaic_status mosaic_mask_activation_planes(const mosaic_params *p, const mosaic_key *key,
                                            uint64_t pass_id, int64_t m, int64_t n_pad, int64_t l,
                                            const uint32_t *C, const uint32_t *J,
                                            const uint16_t *cj_planes, uint32_t *Ux_tm,
                                            uint32_t *K_tm, int variant, void *ws, size_t ws_bytes,
                                            void *stream) {
    if (!cj_planes || !aligned16(cj_planes)) return MOSAIC_ERR_ARG;
    return mask_activation_impl(p, key, pass_id, nullptr, m, n_pad, l, C, J, cj_planes, Ux_tm, K_tm,
                                variant, ws, ws_bytes, stream);
}

mosaic_status mosaic_mask_activation_ex(const mosaic_params *p, const mosaic_key *key, uint64_t pass_id,
                                        const uint64_t *pass_dev, int64_t m, int64_t n_pad, int64_t l,
                                        const uint32_t *C, const uint32_t *J, const uint16_t *cj_planes,
                                        uint32_t *Ux_tm, uint32_t *K_tm, int variant, void *ws,
                                        size_t ws_bytes, void *stream) {
    if (cj_planes && !aligned16(cj_planes)) return MOSAIC_ERR_ALIGN;
    return mask_activation_impl(p, key, pass_id, pass_dev, m, n_pad, l, C, J, cj_planes, Ux_tm, K_tm,
                                variant, ws, ws_bytes, stream);
}

mosaic_status mosaic_mask_activation_phase(const mosaic_params *p, const mosaic_key *key, uint64_t pass_id,
                                           const uint64_t *pass_dev, int64_t m, int64_t n_pad, int64_t l,
                                           const uint32_t *C, const uint32_t *J, const uint16_t *cj_planes,
                                           uint32_t *Ux_tm, uint32_t *K_tm, int variant, void *ws,
                                           size_t ws_bytes, int phase, void *stream) {
    if (cj_planes && !aligned16(cj_planes)) return MOSAIC_ERR_ALIGN;
    return mask_activation_impl(p, key, pass_id, pass_dev, m, n_pad, l, C, J, cj_planes, Ux_tm, K_tm,
                                variant, ws, ws_bytes, stream, phase);
}

mosaic_status mosaic_mask(int kind, const mosaic_params *p, const mosaic_key *key, uint64_t stream_id,
                          int64_t rows, int64_t n_pad, int64_t l, const mosaic_mask_io *io, int variant,
                          void *ws, size_t ws_bytes, void *stream) {
    if (!io) return MOSAIC_ERR_ARG;
    switch (kind) {
    case MOSAIC_MASK_CHAINS:
        return mosaic_mask_chains(p, key, stream_id, n_pad, io->P, io->C, io->CT, ws, ws_bytes, stream);
    case MOSAIC_MASK_WEIGHT:
        return mosaic_mask_weight(p, key, stream_id, io->W, io->ldw, rows, io->n, n_pad, io->P, io->CT,
                                  io->sign_words, io->s_w, io->L, io->S_idx, io->S_val, io->Wp, io->Wp_planes,
                                  io->J, variant, ws, ws_bytes, stream);
    case MOSAIC_MASK_ACTIVATION:
        return mosaic_mask_activation_ex(p, key, stream_id, io->pass_dev, rows, n_pad, l, io->C, io->J,
                                         io->cj_planes, io->Ux_tm, io->K_tm, variant, ws, ws_bytes, stream);
    default:
        return MOSAIC_ERR_ARG;
    }
}

mosaic_status mosaic_advance_pass(uint64_t *pass_dev, uint64_t delta, void *stream) {
    if (!pass_dev) return MOSAIC_ERR_ARG;
    return add_u64(pass_dev, delta, as_stream(stream));
}

mosaic_status mosaic_prepare_activation(const mosaic_params *p, int64_t m, int64_t n_pad,
                                        const uint32_t *C, const uint32_t *J, uint16_t *cj_planes,
                                        void *stream) {
    RoleScope role("prepare");
    MOSAIC_TRY(check_params(p));
    if (!npad_ok(n_pad) || m < 1) return MOSAIC_ERR_SHAPE;
    if (!C || !J || !cj_planes) return MOSAIC_ERR_ARG;
    if (!aligned16(cj_planes)) return MOSAIC_ERR_ALIGN;
    const int64_t Sr = sum_r(p), rd = r_act(p), od = p->act_nested ? off_r(p, p->d) : 0;
    const int64_t Kp = kpad8(rd), bplane = (n_pad + m) * Kp;
    cudaStream_t st = as_stream(stream);
    MOSAIC_TRY(digit_split(C + od, Sr, n_pad, rd, cj_planes, Kp, bplane, st));
    MOSAIC_TRY(digit_split(J + od, Sr, m, rd, cj_planes + n_pad * Kp, Kp, bplane, st));
    const ActLayout L = act_layout(m, n_pad, p);
    char *base = reinterpret_cast<char *>(cj_planes);
    for (uint32_t i = 1; i <= act_levels(p); i++) {
        if (!L.c_img[i - 1]) continue;
        const uint32_t ri = p->r[i - 1];
        MOSAIC_TRY(build_tile_image(C, Sr, off_r(p, i), ri, n_pad,
                                    reinterpret_cast<uint32_t *>(base + L.c_img[i - 1]), st));
        MOSAIC_TRY(build_tile_image(J, Sr, off_r(p, i), ri, m, reinterpret_cast<uint32_t *>(base + L.j_img[i - 1]),
                                    st));
    }
    return MOSAIC_OK;
}

}  // extern "C"

namespace {

// Unmask + decode; `Lp` (nullable) holds L's digit planes from mosaic_prepare_unmask.
mosaic_status unmask_impl(const mosaic_params *p, int64_t l, int64_t m, const uint32_t *Z, int64_t ldz,
                          const uint32_t *K_tm, const uint32_t *L, const uint16_t *Lp, const uint32_t *S_idx,
                          const uint32_t *S_val, const float *s_w, const float *s_x, const float *bias,
                          float *Y, uint32_t *Yhat, int64_t ldy, int variant, void *ws, size_t ws_bytes,
                          void *stream) {
    RoleScope role("unmask");
    MOSAIC_TRY(check_params(p));
    const uint32_t d = p->d;
    const int64_t Sr = sum_r(p), rd = p->r[d - 1], od = off_r(p, d);
    if (l < 0 || m < 1 || ldz < m + Sr || ldy < m) return MOSAIC_ERR_SHAPE;
    if (l == 0) return MOSAIC_OK;
    if (!Z || !K_tm || !L || !s_w || !s_x || !Y) return MOSAIC_ERR_ARG;
    if (d > 1 && (!S_idx || !S_val)) return MOSAIC_ERR_ARG;
    if (ws_bytes < ws_unmask_min(m, l, p)) return MOSAIC_ERR_WORKSPACE;
    cudaStream_t st = as_stream(stream);
    Carve cv = carve(ws, ws_bytes);
    uint32_t *tmp = cv.take<uint32_t>((size_t)(l * m));
    if (!tmp) return MOSAIC_ERR_WORKSPACE;
    // tmp = K + Q_d L^T, or with the tensor-core product tmp = Y' - K - Q_d L^T
    // (token-major: Q_d^T is the column block [m + od, m + Sr) of Z).
    const uint32_t *Qd = Z + m + od;
    const bool want_tc = variant == MOSAIC_GEMM_TC || (variant == MOSAIC_GEMM_AUTO && tc_available());
    const int64_t Kp = kpad8(rd);
    const bool tc_planes = Lp && want_tc && !skinny_ok(Qd, ldz, L, rd, l, rd) && ldz % 4 == 0 && aligned16(Qd) &&
                           cv.used + up(8 * (size_t)(l * Kp)) <= cv.cap;
    uint16_t *Qp = tc_planes ? cv.take<uint16_t>((size_t)(4 * l * Kp)) : nullptr;
    SparseLevel lev[2];
    int64_t soff = 0;
    for (uint32_t i = 1; i < d; i++) {
        const uint32_t t = p->t[i], ri = p->r[i - 1];
        lev[i - 1] = SparseLevel{S_idx + soff, S_val + soff, (int)t, m + off_r(p, i), ri};
        soff += m * t;
    }
    // With room in the workspace, the gathers stage Q_i from tile images made
    // here, in the same launch that splits Q_d into digit planes.
    int nimg = 0;
    int64_t icol[2];
    uint32_t ir[2];
    uint32_t *img[2];
    if (d > 1 && unmask_images_bytes(l, p) && cv.used + unmask_images_bytes(l, p) <= cv.cap) {
        for (uint32_t i = 1; i < d; i++) {
            const uint32_t ri = p->r[i - 1];
            if (!tile_image_words(l, ri)) continue;
            img[nimg] = cv.take<uint32_t>(tile_image_words(l, ri));
            icol[nimg] = m + off_r(p, i);
            ir[nimg] = ri;
            lev[i - 1].tiled = img[nimg];
            ++nimg;
        }
    }
    // With room, the tiled gathers read line-offset copies of the S lists made
    // in the same launch, instead of converting every round.
    int nlin = 0;
    LineCopy lin[2];
    for (uint32_t i = 1; i < d; i++) {
        SparseLevel &lv = lev[i - 1];
        const size_t bytes = up(4 * (size_t)(m * lv.t));
        if (!pgather_takes(l, lv.r, lv.t) || !aligned16(lv.idx) || !aligned16(lv.val) ||
            !aligned16(cv.base + cv.used) || cv.used + bytes > cv.cap)
            continue;
        uint32_t *buf = cv.take<uint32_t>((size_t)(m * lv.t));
        lin[nlin++] = LineCopy{lv.idx, buf, m * lv.t, lv.r};
        lv.idx = buf;
        lv.lines = 1;
    }
    MOSAIC_TRY(unmask_prep(Z, ldz, l, m + od, rd, Qp, Kp, nimg, icol, ir, img, nlin, lin, st));
    if (Qp) {
        MOSAIC_TRY(ring_gemm_tc_planes_diff(Qp, Kp, l * Kp, Lp, Kp, m * Kp, tmp, m, Z, ldz, K_tm, m, -1, l, m, rd,
                                            st));
    } else {
        MOSAIC_TRY(gemm_u32(variant, cv, Qd, ldz, 1, L, rd, 1, tmp, m, K_tm, m, 1, l, m, rd, st));
    }
    // Y_hat = Y' - tmp - sum_i S_{i+1} Q_i (tmp - sum_i ... after the folded product), then decode.
    return unmask_decode(Z, ldz, m, od, l, m, lev, (int)d - 1, tmp, m, s_w, s_x, bias, Y, Yhat, ldy, st,
                         Qp != nullptr);
}

}  // namespace

extern "C" {

mosaic_status mosaic_unmask(const mosaic_params *p, int64_t l, int64_t m, const uint32_t *Z,
                            int64_t ldz, const uint32_t *K_tm, const uint32_t *L,
                            const uint32_t *S_idx, const uint32_t *S_val, const float *s_w,
                            const float *s_x, const float *bias, float *Y, uint32_t *Yhat,
                            int64_t ldy, int variant, void *ws, size_t ws_bytes, void *stream) {
    return unmask_impl(p, l, m, Z, ldz, K_tm, L, nullptr, S_idx, S_val, s_w, s_x, bias, Y, Yhat, ldy, variant,
                       ws, ws_bytes, stream);
}

mosaic_status mosaic_unmask_planes(const mosaic_params *p, int64_t l, int64_t m, const uint32_t *Z,
                                   int64_t ldz, const uint32_t *K_tm, const uint32_t *L,
                                   const uint16_t *L_planes, const uint32_t *S_idx, const uint32_t *S_val,
                                   const float *s_w, const float *s_x, const float *bias, float *Y,
                                   uint32_t *Yhat, int64_t ldy, int variant, void *ws, size_t ws_bytes,
                                   void *stream) {
    if (!L_planes) return MOSAIC_ERR_ARG;
    if (!aligned16(L_planes)) return MOSAIC_ERR_ALIGN;
    return unmask_impl(p, l, m, Z, ldz, K_tm, L, L_planes, S_idx, S_val, s_w, s_x, bias, Y, Yhat, ldy, variant,
                       ws, ws_bytes, stream);
}

mosaic_status mosaic_prepare_unmask(const mosaic_params *p, int64_t m, const uint32_t *L, uint16_t *L_planes,
                                    void *stream) {
    RoleScope role("prepare");
    MOSAIC_TRY(check_params(p));
    if (m < 1) return MOSAIC_ERR_SHAPE;
    if (!L || !L_planes) return MOSAIC_ERR_ARG;
    if (!aligned16(L_planes)) return MOSAIC_ERR_ALIGN;
    const int64_t rd = p->r[p->d - 1], Kp = kpad8(rd);
    return digit_split(L, rd, m, rd, L_planes, Kp, m * Kp, as_stream(stream));
}

mosaic_status mosaic_freivalds_setup(const mosaic_params *p, const mosaic_key *key, uint64_t matrix_id,
                                     int k, const uint32_t *Wm, int64_t ldw, int64_t m, int64_t n_pad,
                                     uint32_t *a, uint32_t *Ychk, void *stream) {
    RoleScope role("freivalds");
    MOSAIC_TRY(check_params(p));
    if (!key) return MOSAIC_ERR_ARG;
    if (k < 1 || k > 16) return MOSAIC_ERR_ARG;
    if (!npad_ok(n_pad) || m < 1 || ldw < n_pad) return MOSAIC_ERR_SHAPE;
    if (!Wm || !a || !Ychk) return MOSAIC_ERR_ARG;
    cudaStream_t st = as_stream(stream);
    MOSAIC_TRY(prg_uniform(to_key(key), tag_of(MOSAIC_TAG_CHECK, 0), matrix_id, (int)p->rounds, k, m, a, m, st));
    return freivalds_colsum(a, k, Wm, ldw, m, n_pad, Ychk, st);
}

mosaic_status mosaic_freivalds_check(int k, const uint32_t *a, const uint32_t *Ychk, int64_t m,
                                     int64_t n_pad, int64_t l, const uint32_t *Z, int64_t ldz,
                                     const uint32_t *Xp, int64_t ldx, uint32_t *bad, uint32_t *n_bad,
                                     void *ws, size_t ws_bytes, void *stream) {
    RoleScope role("freivalds");
    if (k < 1 || k > 16) return MOSAIC_ERR_ARG;
    if (m < 1 || n_pad < 1 || l < 0 || ldz < m || ldx < n_pad) return MOSAIC_ERR_SHAPE;
    if (l == 0) return MOSAIC_OK;
    if (!a || !Ychk || !Z || !Xp || !bad || !n_bad) return MOSAIC_ERR_ARG;
    Carve cv = carve(ws, ws_bytes);
    uint32_t *lhs = cv.take<uint32_t>((size_t)(k * l));
    uint32_t *rhs = cv.take<uint32_t>((size_t)(k * l));
    if (!lhs || !rhs) return MOSAIC_ERR_WORKSPACE;
    return freivalds_check(k, a, Ychk, m, n_pad, l, Z, ldz, Xp, ldx, bad, n_bad, lhs, rhs, as_stream(stream));
}

}  // extern "C"
