// Sparse (LPN) terms of the masks and of the unmask, and the decode epilogue
// (Sec. 3.2 protocol box: U_x and K in Init X steps 1b-1c, the unmask in
// Online step 5; Pi_Sec-Linear Online step 3 for the decode), plus small
// layout helpers.
//
// Every sparse term has the form  out[.][.] += sum_q val_q * src[g][p_q]:
// one side of the output indexes a sparse list (t positions p_q and values
// val_q) and the other side indexes a dense row g of `src` that the list
// gathers from.  A CTA stages TG rows g of src (only the segment the levels
// touch) in shared memory and each thread owns one list entity, so each
// gathered word comes from shared memory.
#include <cuda_bf16.h>

#include "async_copy.cuh"
#include "mosaic_internal.cuh"

namespace mosaic {

// Set when a tiled gather gave up waiting for its staging copy.
__device__ uint32_t g_gather_error = 0;

namespace {

constexpr int kMaxLev = 2;
constexpr int GW = 16;          // warps per CTA
constexpr int G_ENTS = 128;     // list entities per CTA
constexpr int kRing = 2;        // slots of the per-warp list ring

// One pass over one LPN level:
//   out[row][col] = a[row][col] - b[row][col] + sgn * sum_q val[e][q] * src[g][col0 + idx[e][q]]
// with (row, col) = (e, g) or, when the list indexes columns, (g, e); a, b
// nullable; positions must be < r (larger ones are clamped to r - 1, which
// keeps reads in bounds but gives an unspecified sum).  With `decode` the result
// Y_hat is also decoded: Y = ((float)(int32)Y_hat * s_w[col]) * s_x[row] + bias[col].
struct GatherArgs {
    const uint32_t *src;
    int64_t lds, col0;
    uint32_t r;
    int64_t segp;
    const uint32_t *idx, *val;
    int t;
    int64_t g_count, nlist;
    const uint32_t *a;
    int64_t lda;
    const uint32_t *b;
    int64_t ldb;
    int sgn;
    uint32_t *out;
    int64_t ldo;
    int decode;
    const float *s_w, *s_x, *bias;
    float *Y;
    int64_t ldy;
    int trusted;   // positions known to be < r (drawn by this library)
    const uint32_t *tiled;   // tile images of the level's segment (build_tile_image) or null
    int lines;               // positions are already line offsets (p << 7 | chunk bits), see pg_line
    // Tiled gather only: a second job on the same lists and segment columns.
    // Its units follow the first job's; they stage rows of src2 (tiled2)
    // and read a2 / write out2 (no b, no decode).
    int two;
    const uint32_t *src2, *tiled2, *a2;
    int64_t lds2, g_count2, lda2, ldo2;
    uint32_t *out2;
};

// Staged rows plus the per-warp list rings.
constexpr size_t gather_smem(int tg, int64_t segp) {
    return ((size_t)tg * (size_t)segp + 3) / 4 * 4 * sizeof(uint32_t) +
           (size_t)GW * kRing * (32 / tg) * 32 * sizeof(uint32_t);
}

// A CTA stages TG rows g of the level's segment of src (r words each) with a
// row stride segp = 1 (mod 32), so lane g of a warp reading word p of row g
// hits bank (g + p) mod 32: with TG = 32 the 32 lanes never conflict.  Each
// warp serves 32 / TG list entities; the TG lanes of an entity share its
// (position, value) loads (16-byte, prefetched 16 pairs at a time) and keep
// four independent partial sums.
template <int TG, bool LIST_IS_COL, bool CLAMP>
__global__ void __launch_bounds__(GW * 32) gather_kernel(GatherArgs a) {
    constexpr int EPW = 32 / TG;
    extern __shared__ uint32_t sg[];
    const int64_t g0 = (int64_t)blockIdx.y * TG;
    const int64_t rem = a.g_count - g0;
    const int gn = rem < TG ? (int)rem : TG;
    const int r = (int)a.r;
    for (int g = 0; g < gn; g++) {
        const uint32_t *srow = a.src + (g0 + g) * a.lds + a.col0;
        const uint32_t dst0 = (uint32_t)__cvta_generic_to_shared(sg + g * a.segp);
        for (int c = threadIdx.x; c < r; c += blockDim.x)
            asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(dst0 + 4u * c), "l"(srow + c)
                         : "memory");
    }
    asm volatile("cp.async.wait_all;" ::: "memory");
    __syncthreads();

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int h = lane / TG, g = lane % TG;
    const int64_t e_begin = (int64_t)blockIdx.x * G_ENTS;
    const int64_t e_end = e_begin + G_ENTS < a.nlist ? e_begin + G_ENTS : a.nlist;
    const uint32_t *row_g = sg + g * a.segp;
    // Positions of a well-formed list are < r; a malformed one is clamped to
    // r - 1 so that every shared-memory read stays inside the staged row.
    const uint32_t rlast = a.r ? a.r - 1 : 0;
    const int t = a.t;
    const bool vec = t > 0 && (t & 3) == 0 &&
                     ((reinterpret_cast<uintptr_t>(a.idx) | reinterpret_cast<uintptr_t>(a.val)) & 15u) == 0;
    const int stride = GW * EPW;
    const int64_t e_first = e_begin + warp * EPW + h;
    // Every lane of the warp runs the same number of entity iterations (the
    // warp's lanes serve entities e_first .. e_first + EPW - 1 of each sweep).
    const int n_ent = e_begin + warp * EPW < e_end
                          ? (int)((e_end - (e_begin + warp * EPW) + stride - 1) / stride) : 0;
    auto finish = [&](int64_t e, uint32_t sum) {
        if (e >= e_end || g >= gn) return;
        const int64_t row = LIST_IS_COL ? g0 + g : e;
        const int64_t col = LIST_IS_COL ? e : g0 + g;
        uint32_t res = a.sgn >= 0 ? sum : 0u - sum;
        if (a.a) res += a.a[row * a.lda + col];
        if (a.b) res -= a.b[row * a.ldb + col];
        if (a.out) a.out[row * a.ldo + col] = res;
        if (a.decode) {
            float y = __fmul_rn(__fmul_rn(__int2float_rn((int32_t)res), a.s_w[col]), a.s_x[row]);
            if (a.bias) y = __fadd_rn(y, a.bias[col]);
            a.Y[row * a.ldy + col] = y;
        }
    };
    if (t == 0) {
        for (int k = 0; k < n_ent; k++) finish(e_first + (int64_t)k * stride, 0u);
    } else if (vec) {
        // Rounds of 16 (position, value) pairs.  Lanes 0 .. 8 EPW - 1 copy the
        // warp's next round into a 2-slot shared-memory ring (cp.async,
        // zero-filled past the end of a list or of the entity range) while
        // the current round is gathered; the TG lanes of an entity read its
        // pairs from the ring with broadcast loads.
        const int R = (t + 15) >> 4;
        const int steps = n_ent * R;
        uint32_t *ring = sg + ((int64_t)TG * a.segp + 3) / 4 * 4 + warp * (kRing * 32 * EPW);
        // (ik, ir): entity iteration and round of the next step to issue.
        int ik = 0, ir = 0;
        auto issue = [&](int s) {
            const int k = ik, rr = ir;
            if (++ir == R) { ir = 0; ++ik; }
            if (lane < 8 * EPW && s < steps) {
                const int he = lane >> 3, part = lane & 7;
                const int64_t e = e_begin + warp * EPW + he + (int64_t)k * stride;
                const int q = rr * 16 + (part & 3) * 4;
                const bool ok = e < e_end && q < t;
                const uint32_t *src = (part < 4 ? a.idx : a.val) + (ok ? e * t + q : 0);
                const uint32_t dst =
                    (uint32_t)__cvta_generic_to_shared(ring + ((s % kRing) * EPW + he) * 32 + part * 4);
                asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src),
                             "r"(ok ? 16 : 0)
                             : "memory");
            }
            asm volatile("cp.async.commit_group;" ::: "memory");
        };
        for (int s = 0; s < kRing - 1; s++) issue(s);
        uint32_t s0 = 0u, s1 = 0u, s2 = 0u, s3 = 0u;
        int k = 0, rr = 0;
        for (int st = 0; st < steps; st++) {
            issue(st + kRing - 1);
            asm volatile("cp.async.wait_group %0;" ::"n"(kRing - 1) : "memory");
            __syncwarp();
            const uint4 *slot = reinterpret_cast<const uint4 *>(ring + ((st % kRing) * EPW + h) * 32);
#pragma unroll
            for (int u = 0; u < 4; u++) {
                const uint4 I = slot[u], V = slot[4 + u];
                s0 += V.x * row_g[CLAMP ? min(I.x, rlast) : I.x];
                s1 += V.y * row_g[CLAMP ? min(I.y, rlast) : I.y];
                s2 += V.z * row_g[CLAMP ? min(I.z, rlast) : I.z];
                s3 += V.w * row_g[CLAMP ? min(I.w, rlast) : I.w];
            }
            __syncwarp();
            if (rr == R - 1) {
                finish(e_first + (int64_t)k * stride, s0 + s1 + s2 + s3);
                s0 = s1 = s2 = s3 = 0u;
            }
            if (++rr == R) { rr = 0; ++k; }
        }
    } else {
        for (int k = 0; k < n_ent; k++) {
            const int64_t e = e_first + (int64_t)k * stride;
            uint32_t s0 = 0u;
            if (e < e_end) {
                const uint32_t *ip = a.idx + e * t;
                const uint32_t *vp = a.val + e * t;
                for (int q = 0; q < t; q++) s0 += vp[q] * row_g[min(ip[q], rlast)];
            }
            finish(e, s0);
        }
    }
}

// ---------------------------------------------------------------------------
// Persistent tiled gather (lists with t a multiple of 4 and 16-byte aligned,
// segments of up to kPgMaxR words).
//
// A tile is 32 rows g of the level's segment, staged TRANSPOSED: the 32 rows'
// words at position p form one 128-byte line (line p at byte 128 p), whose
// eight 16-byte chunks are XOR-permuted by f(p) = 2 ((p >> 2) & 3), an even
// number: rows 4c .. 4c+3 sit in chunk c ^ f(p).  A warp serves eight list
// entities at a time, four lanes each; lane i of an entity owns rows
// 8i .. 8i+7 (chunks 2i and 2i+1) and reads them at position p with two
// 16-byte loads.  The even entities of a warp read their even chunk first and
// the odd ones their odd chunk, and f(p) keeps a chunk's parity, so in each
// 16-byte access phase (two entities, eight lanes) the two entities' four
// chunks fall in distinct halves of the 32 banks whatever their positions:
// every load is conflict-free.  Each lane accumulates the two loads apart and
// puts the rows back in order when it writes the unit out.
// Staging: a warp loads 4 rows x 32 positions (four 128-byte segments, one
// 16-byte load a lane) and stores each word in its line.
// The (position, value) lists stream through a per-warp ring of two slots in
// rounds of 16 pairs (cp.async one round ahead, zero-filled past the end of a
// list).  A slot holds the round's positions then its values, quad q of
// entity e at word 32 q + 4 e, so one 16-byte load of quad q serves all eight
// entities from the 32 banks at once.  Lists already given as line addresses
// (`lines`: drawn that way, or converted once per call) are used as they
// are; otherwise, once a round has landed, each lane rewrites four positions
// into line addresses with the permutation bits in place (clamping positions
// of caller lists to r - 1), so that the gather loop needs one XOR per load.
// Work units are (tile, 128 entities), numbered tile-major and split evenly
// over a persistent grid, so a CTA stages each of its one or two tiles once;
// with a second job (`two`: another source and output on the same lists) its
// units follow the first job's.  Each unit's a - b operands are loaded when it
// starts and its outputs written when its last round is done (32-byte
// accesses where the output rows are the list entities and the layout
// allows; eight consecutive entities, 32 bytes, per output row otherwise).
// ---------------------------------------------------------------------------
constexpr int kPgRows = 32;
constexpr int kPgWarps = 16;
constexpr int kPgEPW = 8;                   // entities per warp
constexpr int kPgEnts = kPgEPW * kPgWarps;  // entities per unit
constexpr int kPgRing = 2;                  // ring slots per warp
constexpr int kPgSlot = 2 * 16 * kPgEPW;    // words per ring slot: 16 positions + 16 values per entity
constexpr uint32_t kPgMaxR = 1536;          // stage + rings + barrier + alignment within 227 KB

// Stage, rings, the staging barrier and abort flag (16 bytes), + 128 bytes
// to align the stage to a line.
size_t pgather_smem(uint32_t r) {
    return (size_t)((r + 31) / 32 * 32) * kPgRows * 4 + (size_t)kPgWarps * kPgRing * kPgSlot * 4 + 16 + 128;
}

__device__ __forceinline__ uint4 lds128(uint32_t addr) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "r"(addr)
                 : "memory");
    return v;
}
__device__ __forceinline__ void sts32(uint32_t addr, uint32_t v) {
    asm volatile("st.shared.u32 [%0], %1;" ::"r"(addr), "r"(v) : "memory");
}
__device__ __forceinline__ void sts128(uint32_t addr, uint4 v) {
    asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
                 : "memory");
}

constexpr int kPgStageBatch = 12;  // 16-byte loads a lane keeps in flight while staging

template <bool LIST_IS_COL, bool CLAMP>
__global__ void __launch_bounds__(kPgWarps * 32, 1)
    pgather_kernel(GatherArgs a, int units, int units0, int chunks, int vec_src, int vec_ab) {
    extern __shared__ __align__(16) uint32_t sm[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int grp = lane >> 2, li = lane & 3;
    const int r = (int)a.r, rp = (r + 31) / 32 * 32, t = a.t;
    const uint32_t sm_base = ((uint32_t)__cvta_generic_to_shared(sm) + 127u) & ~127u;
    const uint32_t ring_base = sm_base + 4u * (uint32_t)(rp * kPgRows + warp * (kPgRing * kPgSlot));
    // Staging barrier and abort flag after all rings.
    uint64_t *bar = reinterpret_cast<uint64_t *>(reinterpret_cast<char *>(sm) + (sm_base - smem_u32(sm)) +
                                                 4 * ((size_t)rp * kPgRows + (size_t)kPgWarps * kPgRing * kPgSlot));
    volatile int *abort_flag = reinterpret_cast<volatile int *>(bar + 1);
    uint32_t bar_phase = 0;
    if (a.tiled && threadIdx.x == 0) {
        mbar_init(bar, 1);
        *abort_flag = 0;
        mbar_init_fence();
    }
    const int u_begin = (int)((int64_t)units * blockIdx.x / gridDim.x);
    const int u_end = (int)((int64_t)units * (blockIdx.x + 1) / gridDim.x);
    const int R = (t + 15) >> 4;
    const int steps = (u_end - u_begin) * R;
    const uint32_t rlast = a.r - 1;
    // Byte offsets of this lane's two chunks in a line, in load order (before
    // the permutation): chunk 2 li + par first, par = 1 for the odd entities.
    const int par = grp & 1;
    const uint32_t chunk0 = 16u * (uint32_t)(2 * li + par);
    const uint32_t chunk1 = 16u * (uint32_t)(2 * li + (par ^ 1));

    // List rounds: lane (grp, li) copies quad li of round rr of entity
    // (chunk, warp, grp), positions and values, to slot words 32 li + 4 grp
    // and 128 + 32 li + 4 grp.
    const uint32_t st_idx = 4u * (uint32_t)(li * 32 + grp * 4);
    const uint32_t st_val = st_idx + 4u * 128u;
    int i_chunk = u_begin % chunks, i_rr = 0, i_s = 0;
    auto issue = [&]() {
        if (i_s < steps) {
            const int64_t e = (int64_t)i_chunk * kPgEnts + warp * kPgEPW + grp;
            const int q = i_rr * 16 + li * 4;
            const bool ok = e < a.nlist && q < t;
            const int64_t off = ok ? e * t + q : 0;
            const uint32_t dst = ring_base + 4u * (uint32_t)((i_s % kPgRing) * kPgSlot);
            asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst + st_idx), "l"(a.idx + off),
                         "r"(ok ? 16 : 0)
                         : "memory");
            asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst + st_val), "l"(a.val + off),
                         "r"(ok ? 16 : 0)
                         : "memory");
            if (++i_rr == R) {
                i_rr = 0;
                if (++i_chunk == chunks) i_chunk = 0;
            }
        }
        ++i_s;
        asm volatile("cp.async.commit_group;" ::: "memory");
    };

    // Transposed, permuted copy of rows tile*32 .. +31 (zeros past the ends).
    // Lane (gl, pq) of a warp loads words p .. p+3 (p = 32 b + 4 pq) of row
    // 4 j + gl and stores word p+k in line p+k, chunk j ^ f(p+k).  Each lane
    // keeps kPgStageBatch 16-byte loads in flight.
    // Tile images (a.tiled) hold exactly this layout: one bulk copy per 32 KB,
    // all threads wait (bounded) for the barrier.  Returns false if the copy
    // did not land in time (error word raised).
    auto stage_tiled = [&](const uint32_t *img, int64_t tile) -> bool {
        const uint32_t bytes = (uint32_t)rp * 128u;
        if (threadIdx.x == 0) {
            // The previous tile's shared-memory reads happen before these async writes.
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            mbar_expect_tx(bar, bytes);
            const char *src = reinterpret_cast<const char *>(img) + (size_t)tile * bytes;
            for (uint32_t off = 0; off < bytes; off += 32768u)
                bulk_load(sm_base + off, src + off, bytes - off < 32768u ? bytes - off : 32768u, bar);
        }
        const bool ok = mbar_wait(bar, bar_phase, abort_flag);
        if (!ok) {
            *abort_flag = 1;
            atomicExch(&g_gather_error, 1u);
        }
        bar_phase ^= 1u;
        return ok;
    };
    auto stage = [&](const uint32_t *src, int64_t lds, int64_t g_count, int64_t tile) {
        const int64_t g0 = tile * kPgRows;
        const int gl = lane >> 3, pq = lane & 7;
        const int total = 8 * (rp / 32);
        for (int it0 = warp; it0 < total; it0 += kPgWarps * kPgStageBatch) {
            uint4 w[kPgStageBatch];
#pragma unroll
            for (int j = 0; j < kPgStageBatch; j++) {
                const int it = it0 + j * kPgWarps;
                const int g = (it & 7) * 4 + gl;
                const int p = (it >> 3) * 32 + pq * 4;
                w[j] = make_uint4(0u, 0u, 0u, 0u);
                if (it < total && g0 + g < g_count && p < r) {
                    const uint32_t *srow = src + (g0 + g) * lds + a.col0;
                    if (vec_src && p + 4 <= r) {
                        w[j] = __ldg(reinterpret_cast<const uint4 *>(srow + p));
                    } else {
                        w[j].x = srow[p];
                        if (p + 1 < r) w[j].y = srow[p + 1];
                        if (p + 2 < r) w[j].z = srow[p + 2];
                        if (p + 3 < r) w[j].w = srow[p + 3];
                    }
                }
            }
#pragma unroll
            for (int j = 0; j < kPgStageBatch; j++) {
                const int it = it0 + j * kPgWarps;
                if (it < total) {
                    const int g = (it & 7) * 4 + gl;
                    const int p = (it >> 3) * 32 + pq * 4;
                    const uint32_t v[4] = {w[j].x, w[j].y, w[j].z, w[j].w};
#pragma unroll
                    for (int k = 0; k < 4; k++) {
                        const uint32_t pp = (uint32_t)(p + k);
                        sts32(sm_base + (pp << 7) + ((((uint32_t)g >> 2) ^ pg_perm(pp)) & 7u) * 16u +
                                  4u * (uint32_t)(g & 3),
                              v[k]);
                    }
                }
            }
        }
    };

#pragma unroll
    for (int j = 0; j < kPgRing - 1; j++) issue();
    int s = 0;
    // units0 (a multiple of chunks) is where the second job's units start.
    int64_t tile = (u_begin >= units0 ? u_begin - units0 : u_begin) / chunks;
    int chunk = u_begin % chunks;
    for (int u = u_begin; u < u_end; u++) {
        const bool j1 = u >= units0;   // the same for every thread
        if (u == units0) tile = 0;
        const int64_t g_count = j1 ? a.g_count2 : a.g_count;
        if (u == u_begin || chunk == 0) {   // a new tile: the same unit for every warp
            __syncthreads();
            const uint32_t *img = j1 ? a.tiled2 : a.tiled;
            if (img) {
                stage_tiled(img, tile);
            } else {
                stage(j1 ? a.src2 : a.src, j1 ? a.lds2 : a.lds, g_count, tile);
            }
            __syncthreads();
            if (img && *abort_flag) {
                // Let this CTA's copy land (bounded) before leaving.
                if (threadIdx.x == 0) mbar_drain(bar, bar_phase ^ 1u);
                break;
            }
        }
        const int64_t e = (int64_t)chunk * kPgEnts + warp * kPgEPW + grp;
        const int64_t g = tile * kPgRows + li * 8;
        const bool e_ok = e < a.nlist;
        // a - b of the unit's outputs: row e, columns g .. g+7 (or the transpose).
        const bool vec = vec_ab && !LIST_IS_COL && g + 8 <= g_count;
        const uint32_t *ja = j1 ? a.a2 : a.a;
        const int64_t jlda = j1 ? a.lda2 : a.lda;
        uint32_t ab[8] = {0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
        if (e_ok) {
            if (vec) {
#pragma unroll
                for (int h = 0; h < 2; h++) {
                    if (ja) {
                        const uint4 x = __ldg(reinterpret_cast<const uint4 *>(ja + e * jlda + g + 4 * h));
                        ab[4 * h] = x.x; ab[4 * h + 1] = x.y; ab[4 * h + 2] = x.z; ab[4 * h + 3] = x.w;
                    }
                    if (a.b) {
                        const uint4 x = __ldg(reinterpret_cast<const uint4 *>(a.b + e * a.ldb + g + 4 * h));
                        ab[4 * h] -= x.x; ab[4 * h + 1] -= x.y; ab[4 * h + 2] -= x.z; ab[4 * h + 3] -= x.w;
                    }
                }
            } else {
#pragma unroll
                for (int c = 0; c < 8; c++) {
                    if (g + c >= g_count) break;
                    const int64_t row = LIST_IS_COL ? g + c : e;
                    const int64_t col = LIST_IS_COL ? e : g + c;
                    uint32_t v = 0u;
                    if (ja) v += ja[row * jlda + col];
                    if (a.b) v -= a.b[row * a.ldb + col];
                    ab[c] = v;
                }
            }
        }
        // x*: the rows of the first load (chunk 2 li + par), y*: of the second.
        uint32_t x0 = 0u, x1 = 0u, x2 = 0u, x3 = 0u, y0 = 0u, y1 = 0u, y2 = 0u, y3 = 0u;
        for (int rr = 0; rr < R; rr++, s++) {
            issue();
            asm volatile("cp.async.wait_group %0;" ::"n"(kPgRing - 1) : "memory");
            __syncwarp();
            const uint32_t slot = ring_base + 4u * (uint32_t)((s % kPgRing) * kPgSlot);
            if (!a.lines) {
                // Positions 4 lane .. 4 lane + 3 of the round -> line offset | permutation bits.
                uint4 P = lds128(slot + 16u * (uint32_t)lane);
                if (CLAMP) {
                    P.x = min(P.x, rlast);
                    P.y = min(P.y, rlast);
                    P.z = min(P.z, rlast);
                    P.w = min(P.w, rlast);
                }
                sts128(slot + 16u * (uint32_t)lane, make_uint4(pg_line(P.x), pg_line(P.y), pg_line(P.z), pg_line(P.w)));
                __syncwarp();
            }
#pragma unroll
            for (int q = 0; q < 4; q++) {
                const uint4 I = lds128(slot + 4u * (uint32_t)(q * 32 + grp * 4));
                const uint4 V = lds128(slot + 4u * (uint32_t)(128 + q * 32 + grp * 4));
                const uint32_t pi[4] = {I.x, I.y, I.z, I.w};
                const uint32_t vi[4] = {V.x, V.y, V.z, V.w};
#pragma unroll
                for (int c = 0; c < 4; c++) {
                    const uint4 dx = lds128(sm_base + (pi[c] ^ chunk0));
                    const uint4 dy = lds128(sm_base + (pi[c] ^ chunk1));
                    x0 += vi[c] * dx.x;
                    x1 += vi[c] * dx.y;
                    x2 += vi[c] * dx.z;
                    x3 += vi[c] * dx.w;
                    y0 += vi[c] * dy.x;
                    y1 += vi[c] * dy.y;
                    y2 += vi[c] * dy.z;
                    y3 += vi[c] * dy.w;
                }
            }
            __syncwarp();
        }
        if (e_ok) {
            // Rows g .. g+3 come from the even chunk, g+4 .. g+7 from the odd one.
            const uint32_t acc[8] = {par ? y0 : x0, par ? y1 : x1, par ? y2 : x2, par ? y3 : x3,
                                     par ? x0 : y0, par ? x1 : y1, par ? x2 : y2, par ? x3 : y3};
            uint32_t res[8];
#pragma unroll
            for (int c = 0; c < 8; c++) res[c] = (a.sgn >= 0 ? acc[c] : 0u - acc[c]) + ab[c];
            uint32_t *jout = j1 ? a.out2 : a.out;
            const int64_t jldo = j1 ? a.ldo2 : a.ldo;
            if (vec && jout && !a.decode) {
                *reinterpret_cast<uint4 *>(jout + e * jldo + g) = make_uint4(res[0], res[1], res[2], res[3]);
                *reinterpret_cast<uint4 *>(jout + e * jldo + g + 4) = make_uint4(res[4], res[5], res[6], res[7]);
            } else {
#pragma unroll
                for (int c = 0; c < 8; c++) {
                    if (g + c >= g_count) break;
                    const int64_t row = LIST_IS_COL ? g + c : e;
                    const int64_t col = LIST_IS_COL ? e : g + c;
                    if (jout) jout[row * jldo + col] = res[c];
                    if (a.decode) {
                        float y = __fmul_rn(__fmul_rn(__int2float_rn((int32_t)res[c]), a.s_w[col]), a.s_x[row]);
                        if (a.bias) y = __fadd_rn(y, a.bias[col]);
                        a.Y[row * a.ldy + col] = y;
                    }
                }
            }
        }
        if (++chunk == chunks) {
            chunk = 0;
            ++tile;
        }
    }
    asm volatile("cp.async.wait_all;" ::: "memory");
}

template <bool LIST_IS_COL, bool CLAMP>
mosaic_status launch_pgather(const GatherArgs &a, cudaStream_t st) {
    const size_t smem = pgather_smem(a.r);
    auto kern = pgather_kernel<LIST_IS_COL, CLAMP>;
    static std::atomic<unsigned long long> attr_set{0};   // one bit per device ordinal
    int dev = 0, sms = 0, per_sm = 0;
    if (!ensure_smem_limit(attr_set, kern, 227 * 1024, &dev)) return MOSAIC_ERR_CUDA;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kPgWarps * 32, smem) != cudaSuccess ||
        per_sm < 1)
        return MOSAIC_ERR_CUDA;
    const int64_t tiles = (a.g_count + kPgRows - 1) / kPgRows;
    const int64_t tiles2 = a.two ? (a.g_count2 + kPgRows - 1) / kPgRows : 0;
    const int64_t chunks = (a.nlist + kPgEnts - 1) / kPgEnts;
    const int64_t units0 = tiles * chunks, units = (tiles + tiles2) * chunks;
    const int64_t slots = (int64_t)sms * per_sm;
    const int64_t grid = units < slots ? units : slots;
    if (units > 0x7fffffff) return MOSAIC_ERR_SHAPE;
    int vec_src = aligned16(a.src) && a.lds % 4 == 0 && a.col0 % 4 == 0;
    // 16-byte a / b / out accesses (rows = list entities only).
    int vec_ab = (!a.a || (aligned16(a.a) && a.lda % 4 == 0)) && (!a.b || (aligned16(a.b) && a.ldb % 4 == 0)) &&
                 (!a.out || (aligned16(a.out) && a.ldo % 4 == 0));
    if (a.two) {
        vec_src = vec_src && aligned16(a.src2) && a.lds2 % 4 == 0;
        vec_ab = vec_ab && (!a.a2 || (aligned16(a.a2) && a.lda2 % 4 == 0)) &&
                 (!a.out2 || (aligned16(a.out2) && a.ldo2 % 4 == 0));
    }
    {
        KernelSpan span("pgather", st);
        kern<<<(unsigned)grid, kPgWarps * 32, smem, st>>>(a, (int)units, (int)units0, (int)chunks, vec_src, vec_ab);
    }
    return launch_status();
}

// ---------------------------------------------------------------------------
// Few staged rows (g_count <= 4, e.g. the unmask of a decode step): one warp
// per list entity.  Each block stages the g_count rows of the level's segment
// once and its warps walk entities; the 32 lanes read an entity's (position,
// value) list with coalesced loads, each lane sums its share of the pairs for
// every staged row, and a butterfly sums the lanes.  The cost is one pass
// over the lists.
// ---------------------------------------------------------------------------
constexpr int kFewRows = 8;
constexpr int kFewWarps = 8;

template <bool LIST_IS_COL, bool CLAMP>
__global__ void __launch_bounds__(kFewWarps * 32) gather_few_kernel(GatherArgs a) {
    extern __shared__ uint32_t sf[];
    const int G = (int)a.g_count, r = (int)a.r, t = a.t;
    for (int i = threadIdx.x; i < G * r; i += blockDim.x) {
        const int g = i / r, p = i - g * r;
        sf[i] = a.src[(int64_t)g * a.lds + a.col0 + p];
    }
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rlast = a.r - 1;
    const int64_t stride = (int64_t)gridDim.x * kFewWarps;
    for (int64_t e = (int64_t)blockIdx.x * kFewWarps + warp; e < a.nlist; e += stride) {
        uint32_t acc[kFewRows];
#pragma unroll
        for (int k = 0; k < kFewRows; k++) acc[k] = 0u;
        const uint32_t *ip = a.idx + e * t;
        const uint32_t *vp = a.val + e * t;
        for (int q = lane; q < t; q += 32) {
            uint32_t p = ip[q];
            if (CLAMP) p = min(p, rlast);
            const uint32_t v = vp[q];
#pragma unroll
            for (int k = 0; k < kFewRows; k++)
                if (k < G) acc[k] += v * sf[k * r + p];
        }
#pragma unroll
        for (int k = 0; k < kFewRows; k++) {
            if (k >= G) break;
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) acc[k] += __shfl_xor_sync(0xffffffffu, acc[k], o);
        }
        // lane k finishes staged row k
        uint32_t mine = 0u;
#pragma unroll
        for (int k = 0; k < kFewRows; k++)
            if (lane == k) mine = acc[k];
        if (lane < G) {
            const int64_t row = LIST_IS_COL ? lane : e;
            const int64_t col = LIST_IS_COL ? e : lane;
            uint32_t res = a.sgn >= 0 ? mine : 0u - mine;
            if (a.a) res += a.a[row * a.lda + col];
            if (a.b) res -= a.b[row * a.ldb + col];
            if (a.out) a.out[row * a.ldo + col] = res;
            if (a.decode) {
                float y = __fmul_rn(__fmul_rn(__int2float_rn((int32_t)res), a.s_w[col]), a.s_x[row]);
                if (a.bias) y = __fadd_rn(y, a.bias[col]);
                a.Y[row * a.ldy + col] = y;
            }
        }
    }
}

template <bool LIST_IS_COL, bool CLAMP>
mosaic_status launch_few(const GatherArgs &a, cudaStream_t st) {
    const size_t smem = (size_t)a.g_count * a.r * sizeof(uint32_t);
    auto kern = gather_few_kernel<LIST_IS_COL, CLAMP>;
    static std::atomic<unsigned long long> attr_set{0};   // one bit per device ordinal
    int dev = 0, sms = 0;
    if (!ensure_smem_limit(attr_set, kern, 192 * 1024, &dev) ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return MOSAIC_ERR_CUDA;
    // Enough warps to stream the lists; every block stages the rows once.
    const int64_t need = (a.nlist + kFewWarps - 1) / kFewWarps;
    const int64_t cap = (int64_t)sms * 4;
    {
        KernelSpan span("gather_few", st);
        kern<<<(unsigned)(need < cap ? need : cap), kFewWarps * 32, smem, st>>>(a);
    }
    return launch_status();
}

template <int TG, bool LIST_IS_COL, bool CLAMP>
mosaic_status launch_gather(const GatherArgs &a, cudaStream_t st) {
    const size_t smem = gather_smem(TG, a.segp);
    if (smem > 48 * 1024 &&
        cudaFuncSetAttribute(gather_kernel<TG, LIST_IS_COL, CLAMP>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem) != cudaSuccess)
        return MOSAIC_ERR_CUDA;
    dim3 grid((unsigned)((a.nlist + G_ENTS - 1) / G_ENTS), (unsigned)((a.g_count + TG - 1) / TG));
    if (grid.y > 65535) return MOSAIC_ERR_SHAPE;
    {
        KernelSpan span("gather", st);
        gather_kernel<TG, LIST_IS_COL, CLAMP><<<grid, GW * 32, smem, st>>>(a);
    }
    return launch_status();
}

template <bool LIST_IS_COL, bool CLAMP>
mosaic_status dispatch_gather(GatherArgs a, cudaStream_t st) {
    // Up to 4 staged rows the lists dominate and one pass over them wins; from
    // about 8 rows on the tiled gather's line reads win despite its padding.
    if (a.t > 0 && a.r >= 1 && a.g_count <= 4 && a.g_count * (int64_t)a.r <= 48 * 1024 && !a.lines)
        return launch_few<LIST_IS_COL, CLAMP>(a, st);
    const bool lists_vec = a.t > 0 && (a.t & 3) == 0 &&
                           ((reinterpret_cast<uintptr_t>(a.idx) | reinterpret_cast<uintptr_t>(a.val)) & 15u) == 0;
    if (lists_vec && a.r >= 1 && a.r <= kPgMaxR) return launch_pgather<LIST_IS_COL, CLAMP>(a, st);
    if (a.lines) return MOSAIC_ERR_UNSUPPORTED;   // line-offset lists are for the tiled gather only
    a.segp = (int64_t)(a.r + 31) / 32 * 32 + 1;
    // The largest row tile with which two CTAs fit on an SM (one CTA stages
    // while the other gathers); else the largest that fits at all.
    const size_t two = 113 * 1024, one = 220 * 1024;
    for (size_t cap : {two, one}) {
        if (gather_smem(32, a.segp) <= cap) return launch_gather<32, LIST_IS_COL, CLAMP>(a, st);
        if (gather_smem(16, a.segp) <= cap) return launch_gather<16, LIST_IS_COL, CLAMP>(a, st);
        if (gather_smem(8, a.segp) <= cap) return launch_gather<8, LIST_IS_COL, CLAMP>(a, st);
        if (gather_smem(4, a.segp) <= cap) return launch_gather<4, LIST_IS_COL, CLAMP>(a, st);
    }
    if (gather_smem(2, a.segp) <= one) return launch_gather<2, LIST_IS_COL, CLAMP>(a, st);
    if (gather_smem(1, a.segp) <= one) return launch_gather<1, LIST_IS_COL, CLAMP>(a, st);
    return MOSAIC_ERR_SHAPE;
}

// Runs one pass per level: the first pass reads a and b, later passes
// accumulate into `out` (which then must not be null), the last pass decodes.
mosaic_status gather_levels(GatherArgs base, bool list_is_col, const SparseLevel *lev, int nlev,
                            uint32_t *scratch_out, int64_t ld_scratch, cudaStream_t st) {
    if (base.g_count == 0 || base.nlist == 0) return MOSAIC_OK;
    if (nlev > kMaxLev) return MOSAIC_ERR_UNSUPPORTED;
    const int passes = nlev > 0 ? nlev : 1;
    for (int L = 0; L < passes; L++) {
        GatherArgs g = base;
        const bool first = L == 0, last = L == passes - 1;
        if (nlev > 0) {
            g.col0 = lev[L].off; g.r = lev[L].r; g.idx = lev[L].idx; g.val = lev[L].val; g.t = lev[L].t;
            g.tiled = lev[L].tiled;
            g.lines = lev[L].lines;
        } else {
            g.col0 = 0; g.r = 0; g.idx = g.val = nullptr; g.t = 0; g.tiled = nullptr;
        }
        if (!first) {
            g.a = scratch_out; g.lda = ld_scratch; g.b = nullptr;
        }
        if (!last) {
            g.out = scratch_out; g.ldo = ld_scratch; g.decode = 0;
        }
        // Lists drawn by this library's sampler are in range by construction;
        // lists from callers are clamped per read.
        mosaic_status rc;
        if (base.trusted)
            rc = list_is_col ? dispatch_gather<true, false>(g, st) : dispatch_gather<false, false>(g, st);
        else
            rc = list_is_col ? dispatch_gather<true, true>(g, st) : dispatch_gather<false, true>(g, st);
        if (rc != MOSAIC_OK) return rc;
    }
    return MOSAIC_OK;
}

// One CTA per (output row j, column block): rows of P gathered by S_{i+1}.
__global__ void rowgather_kernel(const uint32_t *P, int64_t ldp, SparseLevel l0, SparseLevel l1,
                                 int nlev, int64_t ncols, const uint32_t *a, int64_t lda,
                                 uint32_t *out, int64_t ldo) {
    const int64_t j = blockIdx.y;
    const int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (c >= ncols) return;
    uint32_t acc = a ? a[j * lda + c] : 0u;
    for (int L = 0; L < nlev; L++) {
        const SparseLevel lv = L == 0 ? l0 : l1;
        const uint32_t *ip = lv.idx + j * lv.t;
        const uint32_t *vp = lv.val + j * lv.t;
        for (int q = 0; q < lv.t; q++) {
            const uint32_t pos = ip[q];
            if (pos < lv.r) acc += vp[q] * P[(lv.off + pos) * ldp + c];
        }
    }
    out[j * ldo + c] = acc;
}

__global__ void add_kernel(const uint32_t *a, int64_t lda, const uint32_t *b, int64_t ldb,
                           uint32_t *out, int64_t ldo, int64_t rows, int64_t cols) {
    const int64_t total = rows * cols;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = i / cols, c = i - r * cols;
        out[r * ldo + c] = a[r * lda + c] + b[r * ldb + c];
    }
}

__global__ void transpose_kernel(const uint32_t *a, int64_t lda, int64_t rows, int64_t cols,
                                 uint32_t *out, int64_t ldo) {
    __shared__ uint32_t tile[32][33];
    const int64_t r0 = (int64_t)blockIdx.y * 32, c0 = (int64_t)blockIdx.x * 32;
    for (int i = threadIdx.y; i < 32; i += blockDim.y) {
        const int64_t r = r0 + i, c = c0 + threadIdx.x;
        if (r < rows && c < cols) tile[i][threadIdx.x] = a[r * lda + c];
    }
    __syncthreads();
    for (int i = threadIdx.y; i < 32; i += blockDim.y) {
        const int64_t c = c0 + i, r = r0 + threadIdx.x;
        if (r < rows && c < cols) out[c * ldo + r] = tile[threadIdx.x][i];
    }
}


// 4 consecutive elements per thread: one 16-byte load (when aligned and in
// range) and one 8-byte store per plane; a ragged column tail goes element
// by element.  Columns at and beyond `cols` are not written.
__global__ void digit_split_kernel(const uint32_t *a, int64_t lda, int64_t rows, int64_t cols,
                                   uint16_t *planes, int64_t ldp, int64_t plane_stride, int vec) {
    const int64_t per_row = (cols + 3) / 4;
    const int64_t total = rows * per_row;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = i / per_row, c = (i - r * per_row) * 4;
        const uint32_t *src = a + r * lda + c;
        uint16_t *dst = planes + r * ldp + c;
        if (vec && c + 4 <= cols) {
            const uint4 x = *reinterpret_cast<const uint4 *>(src);
#pragma unroll
            for (int d = 0; d < 4; d++) {
                uint2 o;
                o.x = digit_bits(x.x, d) | (digit_bits(x.y, d) << 16);
                o.y = digit_bits(x.z, d) | (digit_bits(x.w, d) << 16);
                *reinterpret_cast<uint2 *>(dst + d * plane_stride) = o;
            }
        } else {
            for (int q = 0; q < 4 && c + q < cols; q++) {
                const uint32_t w = src[q];
#pragma unroll
                for (int d = 0; d < 4; d++) dst[d * plane_stride + q] = (uint16_t)digit_bits(w, d);
            }
        }
    }
}


// Tile images for the tiled gather: image t holds rows 32 t .. 32 t + 31 of
// the segment src[:, col0 .. col0 + r) exactly as pgather_kernel stages them
// (line p = the 32 rows' words at position p, 16-byte chunk c holding rows
// 4 (c ^ pg_perm(p)) .. + 3; zeros past the rows and positions), so that
// a whole tile is one contiguous copy.  Block (p-block, tile): 32 positions.
__device__ __forceinline__ void tile_image_block(const uint32_t *src, int64_t lds, int64_t col0, int r,
                                                 int64_t g_count, int rp, uint32_t *img, int64_t tile, int p0,
                                                 uint32_t (&t)[32][33]) {
    const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;   // 32 x 8 threads
    for (int k = ty; k < 32; k += 8) {
        const int64_t g = tile * 32 + k;
        const int p = p0 + tx;
        t[k][tx] = (g < g_count && p < r) ? src[g * lds + col0 + p] : 0u;
    }
    __syncthreads();
    const int c = tx >> 2, w = tx & 3;
    for (int k = ty; k < 32; k += 8) {
        const int p = p0 + k;
        const int g = ((c ^ (int)pg_perm((uint32_t)p)) << 2) | w;
        img[((size_t)tile * rp + p) * 32 + tx] = t[g][k];
    }
}
__global__ void tile_image_kernel(const uint32_t *src, int64_t lds, int64_t col0, int r, int64_t g_count, int rp,
                                  uint32_t *img) {
    __shared__ uint32_t t[32][33];
    tile_image_block(src, lds, col0, r, g_count, rp, img, blockIdx.y, blockIdx.x * 32, t);
}

// Before an unmask: the digit planes of Q_d (the A operand of Q_d L^T) and
// the tile images of the Q_i segments, in one launch of 256-thread blocks
// (the first nb_split blocks split, then one block per (image, tile, 32
// positions)).
struct UnmaskPrep {
    const uint32_t *Z;
    int64_t ldz, l;
    int64_t qcol, rd;          // Q_d = columns [qcol, qcol + rd)
    uint16_t *Qp;              // [4][l][Kp] or null
    int64_t Kp;
    int vec;
    int nb_split;
    int nimg;
    int64_t icol[2];
    int ir[2], irp[2], iblocks[2];
    uint32_t *img[2];
    // Line-offset copies of caller lists: dst[i] = pg_line(min(src[i], r - 1)).
    int nlin;
    const uint32_t *lsrc[2];
    uint32_t *ldst[2];
    int64_t lcount[2];   // entries, a multiple of 4
    uint32_t lr[2];
    int lblocks[2];
};

__device__ __forceinline__ void split4(const uint32_t *src, uint16_t *dst, int64_t plane_stride, int64_t c,
                                       int64_t cols, int vec) {
    if (vec && c + 4 <= cols) {
        const uint4 x = *reinterpret_cast<const uint4 *>(src);
#pragma unroll
        for (int d = 0; d < 4; d++) {
            uint2 o;
            o.x = digit_bits(x.x, d) | (digit_bits(x.y, d) << 16);
            o.y = digit_bits(x.z, d) | (digit_bits(x.w, d) << 16);
            *reinterpret_cast<uint2 *>(dst + d * plane_stride) = o;
        }
    } else {
        for (int q = 0; q < 4 && c + q < cols; q++) {
            const uint32_t w = src[q];
#pragma unroll
            for (int d = 0; d < 4; d++) dst[d * plane_stride + q] = (uint16_t)digit_bits(w, d);
        }
    }
}

__global__ void __launch_bounds__(256) unmask_prep_kernel(UnmaskPrep a) {
    __shared__ uint32_t t[32][33];
    int b = blockIdx.x;
    if (b < a.nb_split) {
        const int64_t per_row = (a.rd + 3) / 4, total = a.l * per_row;
        for (int64_t i = (int64_t)b * 256 + threadIdx.x; i < total; i += (int64_t)a.nb_split * 256) {
            const int64_t r = i / per_row, c = (i - r * per_row) * 4;
            split4(a.Z + r * a.ldz + a.qcol + c, a.Qp + r * a.Kp + c, a.l * a.Kp, c, a.rd, a.vec);
        }
        return;
    }
    b -= a.nb_split;
    for (int k = 0; k < a.nimg; k++) {
        if (b < a.iblocks[k]) {
            const int pb = a.irp[k] / 32;
            tile_image_block(a.Z, a.ldz, a.icol[k], a.ir[k], a.l, a.irp[k], a.img[k], b / pb, (b % pb) * 32, t);
            return;
        }
        b -= a.iblocks[k];
    }
    for (int k = 0; k < a.nlin; k++) {
        if (b < a.lblocks[k]) {
            const uint32_t rlast = a.lr[k] - 1;
            const int64_t quads = a.lcount[k] / 4;
            const uint4 *src = reinterpret_cast<const uint4 *>(a.lsrc[k]);
            uint4 *dst = reinterpret_cast<uint4 *>(a.ldst[k]);
            for (int64_t i = (int64_t)b * 256 + threadIdx.x; i < quads; i += (int64_t)a.lblocks[k] * 256) {
                const uint4 v = src[i];
                dst[i] = make_uint4(pg_line(min(v.x, rlast)), pg_line(min(v.y, rlast)), pg_line(min(v.z, rlast)),
                                    pg_line(min(v.w, rlast)));
            }
            return;
        }
        b -= a.lblocks[k];
    }
}

}  // namespace

bool pgather_takes(int64_t g_count, uint32_t r, int t) {
    return t > 0 && (t & 3) == 0 && r >= 1 && r <= kPgMaxR && g_count > 4;
}

size_t tile_image_words(int64_t g_count, uint32_t r) {
    if (r < 1 || r > kPgMaxR || g_count < 1) return 0;
    return (size_t)((g_count + kPgRows - 1) / kPgRows) * ((r + 31) / 32 * 32) * kPgRows;
}

mosaic_status build_tile_image(const uint32_t *src, int64_t lds, int64_t col0, uint32_t r, int64_t g_count,
                               uint32_t *img, cudaStream_t st) {
    if (!tile_image_words(g_count, r)) return MOSAIC_ERR_SHAPE;
    const int rp = (int)((r + 31) / 32 * 32);
    const int64_t tiles = (g_count + kPgRows - 1) / kPgRows;
    if (tiles > 65535) return MOSAIC_ERR_SHAPE;
    {
        KernelSpan span("tile_image", st);
        tile_image_kernel<<<dim3((unsigned)(rp / 32), (unsigned)tiles), 256, 0, st>>>(src, lds, col0, (int)r, g_count,
                                                                                      rp, img);
    }
    return launch_status();
}

mosaic_status unmask_prep(const uint32_t *Z, int64_t ldz, int64_t l, int64_t qcol, int64_t rd, uint16_t *Qp,
                          int64_t Kp, int nimg, const int64_t *icol, const uint32_t *ir, uint32_t *const *img,
                          int nlin, const LineCopy *lin, cudaStream_t st) {
    if (l == 0) return MOSAIC_OK;
    if (nimg < 0 || nimg > 2 || nlin < 0 || nlin > 2) return MOSAIC_ERR_UNSUPPORTED;
    UnmaskPrep a{};
    a.Z = Z;
    a.ldz = ldz;
    a.l = l;
    a.qcol = qcol;
    a.rd = rd;
    a.Qp = Qp;
    a.Kp = Kp;
    a.vec = (ldz % 4 == 0) && (qcol % 4 == 0) && (Kp % 4 == 0) && (reinterpret_cast<uintptr_t>(Z) & 15u) == 0 &&
            (reinterpret_cast<uintptr_t>(Qp) & 7u) == 0;
    int64_t grid = 0;
    if (Qp && rd > 0) {
        const int64_t items = l * ((rd + 3) / 4);
        a.nb_split = (int)((items + 255) / 256 < 152 * 8 ? (items + 255) / 256 : 152 * 8);
        grid += a.nb_split;
    }
    a.nimg = nimg;
    for (int k = 0; k < nimg; k++) {
        if (!tile_image_words(l, ir[k])) return MOSAIC_ERR_SHAPE;
        a.icol[k] = icol[k];
        a.ir[k] = (int)ir[k];
        a.irp[k] = (int)((ir[k] + 31) / 32 * 32);
        a.img[k] = img[k];
        const int64_t blocks = ((l + kPgRows - 1) / kPgRows) * (a.irp[k] / 32);
        if (blocks > 0x3fffffff) return MOSAIC_ERR_SHAPE;
        a.iblocks[k] = (int)blocks;
        grid += blocks;
    }
    a.nlin = nlin;
    for (int k = 0; k < nlin; k++) {
        if (lin[k].count % 4 != 0 || lin[k].r < 1 || !aligned16(lin[k].src) || !aligned16(lin[k].dst))
            return MOSAIC_ERR_UNSUPPORTED;
        a.lsrc[k] = lin[k].src;
        a.ldst[k] = lin[k].dst;
        a.lcount[k] = lin[k].count;
        a.lr[k] = lin[k].r;
        const int64_t quads = lin[k].count / 4;
        a.lblocks[k] = (int)((quads + 255) / 256 < 152 * 4 ? (quads + 255) / 256 : 152 * 4);
        grid += a.lblocks[k];
    }
    if (grid == 0) return MOSAIC_OK;
    if (grid > 0x7fffffff) return MOSAIC_ERR_SHAPE;
    {
        KernelSpan span("unmask_prep", st);
        unmask_prep_kernel<<<(unsigned)grid, 256, 0, st>>>(a);
    }
    return launch_status();
}

namespace {
// Self-test of the bounded waits: one thread waits on a barrier phase that
// nothing completes, gives up after limit_ns and raises the gather's error
// word exactly as a staging copy that never lands would.
__global__ void wait_probe_kernel(unsigned long long limit_ns) {
    __shared__ uint64_t bar;
    __shared__ int abort_flag;
    if (threadIdx.x != 0) return;
    mbar_init(&bar, 1);
    abort_flag = 0;
    mbar_init_fence();
    if (!mbar_wait(&bar, 0u, &abort_flag, limit_ns)) atomicExch(&g_gather_error, 1u);
}
}  // namespace

mosaic_status wait_probe(unsigned long long limit_ns, cudaStream_t st) {
    wait_probe_kernel<<<1, 32, 0, st>>>(limit_ns);
    return launch_status();
}

mosaic_status gather_status() {
    uint32_t v = 0, zero = 0;
    if (cudaMemcpyFromSymbol(&v, g_gather_error, sizeof v) != cudaSuccess) return MOSAIC_ERR_CUDA;
    if (v) {
        cudaMemcpyToSymbol(g_gather_error, &zero, sizeof zero);
        return MOSAIC_ERR_TIMEOUT;
    }
    return MOSAIC_OK;
}

mosaic_status sparse_gather(const uint32_t *src, int64_t lds, int64_t seg_off, int64_t seg_len,
                            int64_t g_count, int64_t nlist, bool list_is_col, const SparseLevel *lev,
                            int nlev, const uint32_t *a, int64_t lda, const uint32_t *b, int64_t ldb,
                            int sgn, uint32_t *out, int64_t ldo, cudaStream_t st) {
    (void)seg_off; (void)seg_len;
    GatherArgs g{};
    g.src = src; g.lds = lds; g.g_count = g_count; g.nlist = nlist;
    g.a = a; g.lda = lda; g.b = b; g.ldb = ldb; g.sgn = sgn; g.out = out; g.ldo = ldo;
    g.trusted = 1;   // the T lists of Init X come from prg_sparse
    // Later levels accumulate in place in `out`.
    return gather_levels(g, list_is_col, lev, nlev, out, ldo, st);
}

mosaic_status sparse_gather_pair(const uint32_t *src, int64_t lds, int64_t g_count, uint32_t *out, int64_t ldo,
                                 const uint32_t *const *img, const uint32_t *src2, int64_t lds2, int64_t g_count2,
                                 uint32_t *out2, int64_t ldo2, const uint32_t *const *img2, int64_t nlist,
                                 const SparseLevel *lev, int nlev, cudaStream_t st) {
    // Both jobs on the tiled gather, or two separate calls.
    bool pair = nlev > 0 && nlev <= kMaxLev;
    for (int L = 0; pair && L < nlev; L++) {
        const bool lists_vec = ((reinterpret_cast<uintptr_t>(lev[L].idx) | reinterpret_cast<uintptr_t>(lev[L].val)) &
                                15u) == 0;
        pair = lists_vec && pgather_takes(g_count, lev[L].r, lev[L].t) && pgather_takes(g_count2, lev[L].r, lev[L].t) &&
               (!img[L]) == (!img2[L]);
    }
    if (!pair) {
        SparseLevel l1[kMaxLev], l2[kMaxLev];
        for (int L = 0; L < nlev && L < kMaxLev; L++) {
            l1[L] = lev[L];
            l1[L].tiled = img[L];
            l2[L] = lev[L];
            l2[L].tiled = img2[L];
        }
        MOSAIC_TRY(sparse_gather(src, lds, 0, 0, g_count, nlist, false, l1, nlev, out, ldo, nullptr, 0, 1, out, ldo,
                                 st));
        return sparse_gather(src2, lds2, 0, 0, g_count2, nlist, false, l2, nlev, out2, ldo2, nullptr, 0, 1, out2,
                             ldo2, st);
    }
    if (g_count == 0 && g_count2 == 0) return MOSAIC_OK;
    if (nlist == 0) return MOSAIC_OK;
    for (int L = 0; L < nlev; L++) {
        GatherArgs g{};
        g.src = src; g.lds = lds; g.g_count = g_count; g.nlist = nlist;
        g.a = out; g.lda = ldo; g.sgn = 1; g.out = out; g.ldo = ldo;
        g.trusted = 1;   // the T lists of Init X come from prg_sparse
        g.col0 = lev[L].off; g.r = lev[L].r; g.idx = lev[L].idx; g.val = lev[L].val; g.t = lev[L].t;
        g.tiled = img[L];
        g.lines = lev[L].lines;
        g.two = 1;
        g.src2 = src2; g.lds2 = lds2; g.g_count2 = g_count2; g.tiled2 = img2[L];
        g.a2 = out2; g.lda2 = ldo2; g.out2 = out2; g.ldo2 = ldo2;
        MOSAIC_TRY((launch_pgather<false, false>(g, st)));
    }
    return MOSAIC_OK;
}

mosaic_status unmask_decode(const uint32_t *Z, int64_t ldz, int64_t seg_off, int64_t seg_len,
                            int64_t l, int64_t m, const SparseLevel *lev, int nlev,
                            const uint32_t *tmp, int64_t ldt, const float *s_w, const float *s_x,
                            const float *bias, float *Y, uint32_t *Yhat, int64_t ldy,
                            cudaStream_t st, bool folded) {
    (void)seg_off; (void)seg_len;
    GatherArgs g{};
    g.src = Z; g.lds = ldz; g.g_count = l; g.nlist = m;
    if (folded) {
        g.a = tmp; g.lda = ldt; g.b = nullptr; g.ldb = 0;
    } else {
        g.a = Z; g.lda = ldz; g.b = tmp; g.ldb = ldt;
    }
    g.sgn = -1; g.out = Yhat; g.ldo = ldy;
    g.decode = 1; g.s_w = s_w; g.s_x = s_x; g.bias = bias; g.Y = Y; g.ldy = ldy;
    // The partial Y_hat between levels lives in tmp (each element is read and
    // then overwritten by the same thread).
    return gather_levels(g, true, lev, nlev, const_cast<uint32_t *>(tmp), ldt, st);
}

mosaic_status sparse_rowgather(const uint32_t *P, int64_t ldp, const SparseLevel *lev, int nlev,
                               int64_t m, int64_t ncols, const uint32_t *a, int64_t lda,
                               uint32_t *out, int64_t ldo, cudaStream_t st) {
    if (m == 0 || ncols == 0) return MOSAIC_OK;
    if (nlev > kMaxLev) return MOSAIC_ERR_UNSUPPORTED;
    if (m > 65535) {
        // Split rows into launches of at most 65535 (grid.y limit).
        for (int64_t j0 = 0; j0 < m; j0 += 65535) {
            const int64_t mm = m - j0 < 65535 ? m - j0 : 65535;
            SparseLevel sub[kMaxLev];
            for (int i = 0; i < nlev; i++) {
                sub[i] = lev[i];
                sub[i].idx = lev[i].idx + j0 * lev[i].t;
                sub[i].val = lev[i].val + j0 * lev[i].t;
            }
            MOSAIC_TRY(sparse_rowgather(P, ldp, sub, nlev, mm, ncols, a ? a + j0 * lda : nullptr,
                                        lda, out + j0 * ldo, ldo, st));
        }
        return MOSAIC_OK;
    }
    SparseLevel l0 = nlev > 0 ? lev[0] : SparseLevel{nullptr, nullptr, 0, 0, 0};
    SparseLevel l1 = nlev > 1 ? lev[1] : SparseLevel{nullptr, nullptr, 0, 0, 0};
    dim3 grid((unsigned)((ncols + 255) / 256), (unsigned)m);
    {
        KernelSpan span("rowgather", st);
        rowgather_kernel<<<grid, 256, 0, st>>>(P, ldp, l0, l1, nlev, ncols, a, lda, out, ldo);
    }
    return launch_status();
}

mosaic_status add_u32(const uint32_t *a, int64_t lda, const uint32_t *b, int64_t ldb, uint32_t *out,
                      int64_t ldo, int64_t rows, int64_t cols, cudaStream_t st) {
    if (rows == 0 || cols == 0) return MOSAIC_OK;
    {
        KernelSpan span("ring_add", st);
        add_kernel<<<grid_for(rows * cols, 256), 256, 0, st>>>(a, lda, b, ldb, out, ldo, rows, cols);
    }
    return launch_status();
}

mosaic_status transpose_u32(const uint32_t *a, int64_t lda, int64_t rows, int64_t cols, uint32_t *out,
                            int64_t ldo, cudaStream_t st) {
    if (rows == 0 || cols == 0) return MOSAIC_OK;
    dim3 grid((unsigned)((cols + 31) / 32), (unsigned)((rows + 31) / 32));
    if (grid.y > 65535) return MOSAIC_ERR_SHAPE;
    {
        KernelSpan span("transpose", st);
        transpose_kernel<<<grid, dim3(32, 8), 0, st>>>(a, lda, rows, cols, out, ldo);
    }
    return launch_status();
}

mosaic_status digit_split(const uint32_t *a, int64_t lda, int64_t rows, int64_t cols,
                          uint16_t *planes, int64_t ldp, int64_t plane_stride, cudaStream_t st) {
    if (rows == 0 || cols == 0) return MOSAIC_OK;
    const int vec = (lda % 4 == 0) && (ldp % 4 == 0) && (plane_stride % 4 == 0) &&
                    (reinterpret_cast<uintptr_t>(a) & 15u) == 0 &&
                    (reinterpret_cast<uintptr_t>(planes) & 7u) == 0;
    {
        KernelSpan span("digit_split", st);
        digit_split_kernel<<<grid_for(rows * ((cols + 3) / 4), 256), 256, 0, st>>>(
            a, lda, rows, cols, planes, ldp, plane_stride, vec);
    }
    return launch_status();
}

}  // namespace mosaic
