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

#include "mosaic_internal.cuh"

namespace mosaic {
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

template <int TG, bool LIST_IS_COL, bool CLAMP>
mosaic_status launch_gather(const GatherArgs &a, cudaStream_t st) {
    const size_t smem = gather_smem(TG, a.segp);
    if (smem > 48 * 1024 &&
        cudaFuncSetAttribute(gather_kernel<TG, LIST_IS_COL, CLAMP>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem) != cudaSuccess)
        return MOSAIC_ERR_CUDA;
    dim3 grid((unsigned)((a.nlist + G_ENTS - 1) / G_ENTS), (unsigned)((a.g_count + TG - 1) / TG));
    if (grid.y > 65535) return MOSAIC_ERR_SHAPE;
    gather_kernel<TG, LIST_IS_COL, CLAMP><<<grid, GW * 32, smem, st>>>(a);
    return launch_status();
}

template <bool LIST_IS_COL, bool CLAMP>
mosaic_status dispatch_gather(GatherArgs a, cudaStream_t st) {
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
        } else {
            g.col0 = 0; g.r = 0; g.idx = g.val = nullptr; g.t = 0;
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

__device__ __forceinline__ uint32_t digit_bits(uint32_t a, int d) {
    const int dig = (int)(((a + 0x80808080u) >> (8 * d)) & 0xffu) - 128;
    return __bfloat16_as_ushort(__float2bfloat16_rn((float)dig));
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

int grid_for(int64_t items, int threads) {
    int64_t g = (items + threads - 1) / threads;
    if (g < 1) g = 1;
    if (g > 152 * 32) g = 152 * 32;
    return (int)g;
}

}  // namespace

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

mosaic_status unmask_decode(const uint32_t *Z, int64_t ldz, int64_t seg_off, int64_t seg_len,
                            int64_t l, int64_t m, const SparseLevel *lev, int nlev,
                            const uint32_t *tmp, int64_t ldt, const float *s_w, const float *s_x,
                            const float *bias, float *Y, uint32_t *Yhat, int64_t ldy,
                            cudaStream_t st) {
    (void)seg_off; (void)seg_len;
    GatherArgs g{};
    g.src = Z; g.lds = ldz; g.g_count = l; g.nlist = m;
    g.a = Z; g.lda = ldz; g.b = tmp; g.ldb = ldt; g.sgn = -1; g.out = Yhat; g.ldo = ldy;
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
    rowgather_kernel<<<grid, 256, 0, st>>>(P, ldp, l0, l1, nlev, ncols, a, lda, out, ldo);
    return launch_status();
}

mosaic_status add_u32(const uint32_t *a, int64_t lda, const uint32_t *b, int64_t ldb, uint32_t *out,
                      int64_t ldo, int64_t rows, int64_t cols, cudaStream_t st) {
    if (rows == 0 || cols == 0) return MOSAIC_OK;
    add_kernel<<<grid_for(rows * cols, 256), 256, 0, st>>>(a, lda, b, ldb, out, ldo, rows, cols);
    return launch_status();
}

mosaic_status transpose_u32(const uint32_t *a, int64_t lda, int64_t rows, int64_t cols, uint32_t *out,
                            int64_t ldo, cudaStream_t st) {
    if (rows == 0 || cols == 0) return MOSAIC_OK;
    dim3 grid((unsigned)((cols + 31) / 32), (unsigned)((rows + 31) / 32));
    if (grid.y > 65535) return MOSAIC_ERR_SHAPE;
    transpose_kernel<<<grid, dim3(32, 8), 0, st>>>(a, lda, rows, cols, out, ldo);
    return launch_status();
}

mosaic_status digit_split(const uint32_t *a, int64_t lda, int64_t rows, int64_t cols,
                          uint16_t *planes, int64_t ldp, int64_t plane_stride, cudaStream_t st) {
    if (rows == 0 || cols == 0) return MOSAIC_OK;
    const int vec = (lda % 4 == 0) && (ldp % 4 == 0) && (plane_stride % 4 == 0) &&
                    (reinterpret_cast<uintptr_t>(a) & 15u) == 0 &&
                    (reinterpret_cast<uintptr_t>(planes) & 7u) == 0;
    digit_split_kernel<<<grid_for(rows * ((cols + 3) / 4), 256), 256, 0, st>>>(
        a, lda, rows, cols, planes, ldp, plane_stride, vec);
    return launch_status();
}

}  // namespace mosaic
