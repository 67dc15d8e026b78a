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
constexpr int TE = 256;   // list entities per CTA (one per thread)

struct GatherArgs {
    const uint32_t *src;
    int64_t lds, seg_off, seg_len, g_count, nlist;
    SparseLevel lev[kMaxLev];
    int nlev;
    const uint32_t *a;
    int64_t lda;
    const uint32_t *b;
    int64_t ldb;
    int sgn;
    uint32_t *out;
    int64_t ldo;
    // decode (MODE 1)
    const float *s_w, *s_x, *bias;
    float *Y;
    int64_t ldy;
};

template <int TG, bool LIST_IS_COL, int MODE>
__global__ void __launch_bounds__(TE) gather_kernel(GatherArgs a) {
    extern __shared__ uint32_t sg[];
    const int64_t segp = a.seg_len + 1;   // +1 word per row: staged rows start in different banks
    const int64_t g0 = (int64_t)blockIdx.y * TG;
    const int64_t rem = a.g_count - g0;
    const int gn = rem < TG ? (int)rem : TG;
    for (int g = 0; g < gn; g++) {
        const uint32_t *srow = a.src + (g0 + g) * a.lds + a.seg_off;
        for (int64_t c = threadIdx.x; c < a.seg_len; c += blockDim.x) sg[g * segp + c] = srow[c];
    }
    __syncthreads();
    const int64_t e = (int64_t)blockIdx.x * TE + threadIdx.x;
    if (e >= a.nlist) return;
    uint32_t acc[TG];
#pragma unroll
    for (int g = 0; g < TG; g++) acc[g] = 0u;
    for (int L = 0; L < a.nlev; L++) {
        const SparseLevel lv = a.lev[L];
        const uint32_t *ip = lv.idx + e * lv.t;
        const uint32_t *vp = lv.val + e * lv.t;
        const int64_t off = lv.off - a.seg_off;
        for (int q = 0; q < lv.t; q++) {
            const uint32_t pos = ip[q];
            if (pos >= lv.r) continue;
            const uint32_t *col = sg + off + pos;
            const uint32_t v = vp[q];
#pragma unroll
            for (int g = 0; g < TG; g++) acc[g] += v * col[g * segp];
        }
    }
#pragma unroll
    for (int g = 0; g < TG; g++) {
        if (g >= gn) break;
        const int64_t row = LIST_IS_COL ? g0 + g : e;
        const int64_t colj = LIST_IS_COL ? e : g0 + g;
        uint32_t r = a.sgn >= 0 ? acc[g] : 0u - acc[g];
        if (a.a) r += a.a[row * a.lda + colj];
        if (a.b) r -= a.b[row * a.ldb + colj];
        if (MODE == 0) {
            a.out[row * a.ldo + colj] = r;
        } else {
            // Decode: Y[k][j] = ((float)(int32)Y_hat * s_w[j]) * s_x[k] + b[j].
            if (a.out) a.out[row * a.ldo + colj] = r;
            float y = __fmul_rn(__fmul_rn(__int2float_rn((int32_t)r), a.s_w[colj]), a.s_x[row]);
            if (a.bias) y = __fadd_rn(y, a.bias[colj]);
            a.Y[row * a.ldy + colj] = y;
        }
    }
}

template <int TG, bool LIST_IS_COL, int MODE>
mosaic_status launch_gather(const GatherArgs &a, cudaStream_t st) {
    const size_t smem = (size_t)TG * (size_t)(a.seg_len + 1) * sizeof(uint32_t);
    if (smem > 48 * 1024 &&
        cudaFuncSetAttribute(gather_kernel<TG, LIST_IS_COL, MODE>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
        return MOSAIC_ERR_CUDA;
    dim3 grid((unsigned)((a.nlist + TE - 1) / TE), (unsigned)((a.g_count + TG - 1) / TG));
    if (grid.y > 65535) return MOSAIC_ERR_SHAPE;
    gather_kernel<TG, LIST_IS_COL, MODE><<<grid, TE, smem, st>>>(a);
    return launch_status();
}

template <bool LIST_IS_COL, int MODE>
mosaic_status dispatch_gather(const GatherArgs &a, cudaStream_t st) {
    const size_t row_bytes = (size_t)(a.seg_len + 1) * sizeof(uint32_t);
    const size_t budget = 200 * 1024;
    if (row_bytes * 16 <= budget) return launch_gather<16, LIST_IS_COL, MODE>(a, st);
    if (row_bytes * 8 <= budget) return launch_gather<8, LIST_IS_COL, MODE>(a, st);
    if (row_bytes * 4 <= budget) return launch_gather<4, LIST_IS_COL, MODE>(a, st);
    if (row_bytes <= budget) return launch_gather<1, LIST_IS_COL, MODE>(a, st);
    return MOSAIC_ERR_SHAPE;
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

// 8 consecutive elements per thread -> one 16-byte store per plane.
__global__ void digit_split_kernel(const uint32_t *a, int64_t lda, int64_t rows, int64_t cols,
                                   uint16_t *planes, int64_t ldp, int64_t plane_stride) {
    const int64_t per_row = cols / 8;
    const int64_t total = rows * per_row;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = i / per_row, c = (i - r * per_row) * 8;
        const uint4 x0 = *reinterpret_cast<const uint4 *>(a + r * lda + c);
        const uint4 x1 = *reinterpret_cast<const uint4 *>(a + r * lda + c + 4);
        const uint32_t w[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
#pragma unroll
        for (int d = 0; d < 4; d++) {
            uint32_t h[8];
#pragma unroll
            for (int q = 0; q < 8; q++) {
                const int dig = (int)(((w[q] + 0x80808080u) >> (8 * d)) & 0xffu) - 128;
                h[q] = __bfloat16_as_ushort(__float2bfloat16_rn((float)dig));
            }
            uint4 o;
            o.x = h[0] | (h[1] << 16); o.y = h[2] | (h[3] << 16);
            o.z = h[4] | (h[5] << 16); o.w = h[6] | (h[7] << 16);
            *reinterpret_cast<uint4 *>(planes + d * plane_stride + r * ldp + c) = o;
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
    if (g_count == 0 || nlist == 0) return MOSAIC_OK;
    if (nlev > kMaxLev) return MOSAIC_ERR_UNSUPPORTED;
    GatherArgs g{};
    g.src = src; g.lds = lds; g.seg_off = seg_off; g.seg_len = seg_len; g.g_count = g_count;
    g.nlist = nlist; g.nlev = nlev;
    for (int i = 0; i < nlev; i++) g.lev[i] = lev[i];
    g.a = a; g.lda = lda; g.b = b; g.ldb = ldb; g.sgn = sgn; g.out = out; g.ldo = ldo;
    return list_is_col ? dispatch_gather<true, 0>(g, st) : dispatch_gather<false, 0>(g, st);
}

mosaic_status unmask_decode(const uint32_t *Z, int64_t ldz, int64_t seg_off, int64_t seg_len,
                            int64_t l, int64_t m, const SparseLevel *lev, int nlev,
                            const uint32_t *tmp, int64_t ldt, const float *s_w, const float *s_x,
                            const float *bias, float *Y, uint32_t *Yhat, int64_t ldy,
                            cudaStream_t st) {
    if (l == 0 || m == 0) return MOSAIC_OK;
    if (nlev > kMaxLev) return MOSAIC_ERR_UNSUPPORTED;
    GatherArgs g{};
    g.src = Z; g.lds = ldz; g.seg_off = seg_off; g.seg_len = seg_len; g.g_count = l; g.nlist = m;
    g.nlev = nlev;
    for (int i = 0; i < nlev; i++) g.lev[i] = lev[i];
    g.a = Z; g.lda = ldz; g.b = tmp; g.ldb = ldt; g.sgn = -1; g.out = Yhat; g.ldo = ldy;
    g.s_w = s_w; g.s_x = s_x; g.bias = bias; g.Y = Y; g.ldy = ldy;
    if (seg_len == 0) {
        // d = 1: no sparse level; stage nothing.
        g.seg_len = 0;
    }
    return dispatch_gather<true, 1>(g, st);
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
    digit_split_kernel<<<grid_for(rows * cols / 8, 256), 256, 0, st>>>(a, lda, rows, cols, planes,
                                                                        ldp, plane_stride);
    return launch_status();
}

}  // namespace mosaic
