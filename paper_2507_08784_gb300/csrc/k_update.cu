// K3 for the compressed steps of a truncated basis: the projected mean and the decompressed
// optimizer update without another pass over Mbar.  With U = (I - Y T Y^T) D and P = U[:, J]
// (the WY form of the truncated basis),
//   Rbar = P^T Mbar = D_J (Mbar[J, :] - Yt[J, :] Wbar),   Yt = Y T^T,  Wbar = Y^T Mbar,
// and Wbar comes out of K1's lambda epilogue; the selection's pr_kernel forms Rbar that way from
// the r rows J of Mbar and of Yt.  A CTA stages its TC columns of Rbar in shared memory, then
// streams X and the optimizer state once: Ghat = P Rbar (Alg. 3), MSGD (Eq. msgd) or Adam
// (Eq. adam).  Bytes per matrix element: X and the moments read and written (16 B MSGD, 24 B Adam);
// Mbar is touched only in the r selected rows.
#include "glr_internal.cuh"

namespace glr {

namespace {

constexpr int TU = 256;                // threads per CTA
constexpr int TC = 64;                 // oriented columns per CTA
constexpr int RCH = 64;                // oriented rows per CTA (X in its stored orientation)
constexpr int TCT = 16;                // oriented columns per CTA when X is read transposed

__device__ __forceinline__ float4 ld4(const float* p) { return *reinterpret_cast<const float4*>(p); }
__device__ __forceinline__ void st4(float* p, float4 v) { *reinterpret_cast<float4*>(p) = v; }

// The optimizer step with gradient estimates gh on four vectors of four consecutive elements,
// at offsets base + u * stride (u < 4, only where valid): every load is issued before the first
// arithmetic, so a thread keeps 8 (MSGD) or 12 (Adam) 16-byte loads in flight.
template <bool ADAM>
__device__ __forceinline__ void optimizer4x4(const UpdStreamGroup& g, const UpdStreamMat& M, const int64_t (&xi)[4],
                                             const bool (&ok)[4], const float (&gh)[4][4]) {
    float4 mo[4], x[4], vo[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        if (!ok[u]) continue;
        mo[u] = ld4(M.Mo + xi[u]);
        x[u] = ld4(M.X + xi[u]);
        if (ADAM) vo[u] = ld4(M.Vo + xi[u]);
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        if (!ok[u]) continue;
        float mv[4] = {mo[u].x, mo[u].y, mo[u].z, mo[u].w}, xv[4] = {x[u].x, x[u].y, x[u].z, x[u].w};
        float vv[4] = {0.f, 0.f, 0.f, 0.f};
        if (ADAM) { vv[0] = vo[u].x; vv[1] = vo[u].y; vv[2] = vo[u].z; vv[3] = vo[u].w; }
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            mv[e] = fmaf(g.beta1, mv[e], (1.0f - g.beta1) * gh[u][e]);
            if (ADAM) {
                vv[e] = fmaf(g.beta2, vv[e], (1.0f - g.beta2) * gh[u][e] * gh[u][e]);
                xv[e] -= g.lr * mv[e] / (sqrtf(vv[e]) + g.eps);
            } else {
                xv[e] -= g.lr * mv[e];
            }
        }
        st4(M.Mo + xi[u], make_float4(mv[0], mv[1], mv[2], mv[3]));
        st4(M.X + xi[u], make_float4(xv[0], xv[1], xv[2], xv[3]));
        if (ADAM) st4(M.Vo + xi[u], make_float4(vv[0], vv[1], vv[2], vv[3]));
    }
}
// rows a0 + u * astep (< mp), columns c..c+3 of a row-major m' x n' X
template <bool ADAM>
__device__ __forceinline__ void optimizer_rows(const UpdStreamGroup& g, const UpdStreamMat& M, int a0, int astep, int mp,
                                               int64_t ld, int c, const float (&gh)[4][4]) {
    int64_t xi[4];
    bool ok[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const int a = a0 + u * astep;
        ok[u] = a < mp;
        xi[u] = (int64_t)a * ld + c;
    }
    optimizer4x4<ADAM>(g, M, xi, ok, gh);
}
// X rows c0 + u * cstep (< cend), entries a..a+3 of a row-major n' x m' X
template <bool ADAM>
__device__ __forceinline__ void optimizer_cols(const UpdStreamGroup& g, const UpdStreamMat& M, int c0, int cstep,
                                               int cend, int64_t ld, int a, const float (&gh)[4][4]) {
    int64_t xi[4];
    bool ok[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const int c = c0 + u * cstep;
        ok[u] = c < cend;
        xi[u] = (int64_t)c * ld + a;
    }
    optimizer4x4<ADAM>(g, M, xi, ok, gh);
}

// RM: r rounded up to 4 or 8 or 16 (register arrays); r itself is the matrix's.  A CTA takes a
// tile of RCH rows x TC columns (X in its stored orientation) or all m' rows x TCT columns (X
// transposed); each thread issues the loads of four rows (or columns) before using them.
template <int RM, bool ADAM, bool TRANS>
__global__ void __launch_bounds__(TU, TRANS ? 1 : 3) update_stream_kernel(const __grid_constant__ UpdStreamGroup g) {
    __shared__ __align__(16) float Rs[RM * TC];             // Rbar[q][c0 + cc]
    int mi = 0;
    while (mi + 1 < g.nmat && blockIdx.x >= static_cast<unsigned>(g.mat[mi + 1].tile0)) ++mi;
    const UpdStreamMat& M = g.mat[mi];
    const int mp = M.mp, np = M.np, r = M.r, k = M.k;
    constexpr bool trans = TRANS;
    const int tcols = trans ? TCT : TC;
    const int ncol = (np + tcols - 1) / tcols;
    const int tile = blockIdx.x - M.tile0;
    const int c0 = (tile % ncol) * tcols, row0 = trans ? 0 : (tile / ncol) * RCH;
    const int tid = threadIdx.x;

    // ---- this CTA's columns of Rbar (formed by the selection) --------------------------------------
    for (int idx = tid; idx < RM * tcols; idx += TU) {
        const int q = idx / tcols, cc = idx % tcols, c = c0 + cc;
        Rs[q * TC + cc] = q < r && c < np ? M.Rbar[(int64_t)q * np + c] : 0.f;
    }
    __syncthreads();

    if constexpr (!TRANS) {
        // X is m' x n' row-major: a thread owns 4 columns of rows row0 + rl + 16 u, u < 4
        const int cq = tid & 15, rl = tid >> 4;
        const int c = c0 + 4 * cq;
        if (c >= np) return;                                 // n' % 4 == 0: the quad is whole
        const float* rs = Rs + 4 * cq;                       // Rbar[q][c..c+3] at rs + q TC
        const bool vec = (r % 4) == 0;                       // P rows are 16-byte aligned
        float gh[4][4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int a = row0 + rl + 16 * u;
            float pv[RM];
            const float* pa = M.P + (int64_t)(a < mp ? a : 0) * r;
            if (vec) {
#pragma unroll
                for (int q = 0; q < RM; q += 4) {
                    const float4 p4 = q < r ? __ldg(reinterpret_cast<const float4*>(pa + q)) : make_float4(0.f, 0.f, 0.f, 0.f);
                    pv[q] = p4.x; pv[q + 1] = p4.y; pv[q + 2] = p4.z; pv[q + 3] = p4.w;
                }
            } else {
#pragma unroll
                for (int q = 0; q < RM; ++q) pv[q] = q < r ? __ldg(pa + q) : 0.f;
            }
#pragma unroll
            for (int e = 0; e < 4; ++e) gh[u][e] = 0.f;
#pragma unroll
            for (int q = 0; q < RM; ++q) {
                const float4 rq = ld4(rs + q * TC);
                gh[u][0] = fmaf(pv[q], rq.x, gh[u][0]); gh[u][1] = fmaf(pv[q], rq.y, gh[u][1]);
                gh[u][2] = fmaf(pv[q], rq.z, gh[u][2]); gh[u][3] = fmaf(pv[q], rq.w, gh[u][3]);
            }
        }
        optimizer_rows<ADAM>(g, M, row0 + rl, 16, mp, (int64_t)np, c, gh);
    } else {
        // X is n' x m' row-major (m > n): a thread owns 4 rows a of the oriented layout (4
        // consecutive entries of an X row) and the columns lc + nl u, u < 4, of the tile
        const int A4 = mp >> 2;                              // m' % 4 == 0 for transposed matrices
        const int nl = TU / A4;
        const int a4 = tid % A4, lc = tid / A4;
        if (lc >= nl) return;
        float pr[4][RM];
#pragma unroll
        for (int e = 0; e < 4; ++e)
#pragma unroll
            for (int q = 0; q < RM; ++q) pr[e][q] = q < r ? __ldg(M.P + (int64_t)(4 * a4 + e) * r + q) : 0.f;
        for (int cb = lc; cb < TCT; cb += 4 * nl) {
            float gh[4][4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int cc = cb + u * nl;
                const bool ok = cc < TCT;
#pragma unroll
                for (int e = 0; e < 4; ++e) gh[u][e] = 0.f;
#pragma unroll
                for (int q = 0; q < RM; ++q) {
                    const float rv = ok ? Rs[q * TC + cc] : 0.f;
#pragma unroll
                    for (int e = 0; e < 4; ++e) gh[u][e] = fmaf(pr[e][q], rv, gh[u][e]);
                }
            }
            optimizer_cols<ADAM>(g, M, c0 + cb, nl, c0 + TCT < np ? c0 + TCT : np, (int64_t)mp, 4 * a4, gh);
        }
    }
}

template <int RM, bool TRANS>
cudaError_t launch_update_stream(const UpdStreamGroup& g, cudaStream_t st) {
    if (g.optimizer == GLR_ADAM) update_stream_kernel<RM, true, TRANS><<<g.total_tiles, TU, 0, st>>>(g);
    else update_stream_kernel<RM, false, TRANS><<<g.total_tiles, TU, 0, st>>>(g);
    return cudaGetLastError();
}

}  // namespace

int update_stream_tiles(int mp, int np, int transposed) {
    return transposed ? (np + TCT - 1) / TCT : ((np + TC - 1) / TC) * ((mp + RCH - 1) / RCH);
}

bool update_stream_eligible(int mp, int r, int transposed) {
    return r >= 1 && r <= 16 && (!transposed || (mp % 4 == 0 && mp / 4 <= TU / 2));
}

cudaError_t update_stream_group(const UpdStreamGroup& g, cudaStream_t st) {
    if (g.total_tiles <= 0) return cudaSuccess;
    int rmax = 0;
    for (int i = 0; i < g.nmat; ++i) {
        rmax = g.mat[i].r > rmax ? g.mat[i].r : rmax;
        if (g.mat[i].transposed != g.mat[0].transposed) return cudaErrorInvalidValue;   // one orientation per launch
    }
    const bool tr = g.mat[0].transposed != 0;
    if (rmax <= 4) return tr ? launch_update_stream<4, true>(g, st) : launch_update_stream<4, false>(g, st);
    if (rmax <= 8) return tr ? launch_update_stream<8, true>(g, st) : launch_update_stream<8, false>(g, st);
    if (rmax <= 16) return tr ? launch_update_stream<16, true>(g, st) : launch_update_stream<16, false>(g, st);
    return cudaErrorInvalidValue;
}

}  // namespace glr
