// Grouped block power iteration for the truncated-basis refresh (the Semi-Lazy SVD of Eq.
// SVD-P1 restricted to the top-k subspace): every refreshing matrix of a step advances together,
// one launch per stage.  One half-iteration is one pass over Mbar:
//   Z = (Mbar^T Q) S        (pow_t_kernel, column tiles of Mbar)        then S <- chol(Z^T Z)^-1
//   Q = (Mbar Z) S          (pow_n_kernel split-K partials, pow_r_kernel) then S <- chol(Q^T Q)^-1
// where S (k x k) is the inverse Cholesky factor that orthonormalises the previous iterate
// (CholeskyQR, Yamamoto et al. 2015), applied to the small output instead of the tall input:
// Mbar^T (Q S) = (Mbar^T Q) S.  The Gram matrices are summed from per-tile partials in a fixed
// order and factored in fp64 by one warp per matrix (pow_chol_kernel).  The final CholeskyQR2
// uses pow_apply_kernel; the Rayleigh-Ritz Gram H = Z^T Z comes out of pow_t_kernel the same way.
#include "glr_internal.cuh"

namespace glr {

namespace {

constexpr int TP = 256;                // threads per CTA
constexpr int PC = 64;                 // columns of Mbar per tile / split-K chunk, rows per row tile
constexpr int PR = 32;                 // rows of Mbar per staged block (pow_t_kernel)
constexpr int NCH = 512;               // columns per split-K chunk (pow_n_kernel)

// Gram partial of the 64 x KM block Zs (rows < nrows valid) into gout (KM x KM, row-major).
template <int KM>
__device__ __forceinline__ void gram_partial(const float* Zs, int nrows, float* gout) {
    for (int o = threadIdx.x; o < KM * KM; o += TP) {
        const int a = o / KM, b = o % KM;
        float s = 0.f;
        for (int c = 0; c < nrows; ++c) s = fmaf(Zs[c * KM + a], Zs[c * KM + b], s);
        gout[o] = s;
    }
}

// out (64 x KM block in smem, rows < nrows) <- in S (KM x KM in smem), into out (may alias
// nothing).  Thread (row = tid % 64, quarter) computes KM / 4 entries of its row.
template <int KM>
__device__ __forceinline__ void apply_S(const float* in, const float* S, float* out) {
    constexpr int KPT = KM / 4;
    const int row = threadIdx.x & 63, kq = threadIdx.x >> 6;
    float acc[KPT];
#pragma unroll
    for (int e = 0; e < KPT; ++e) acc[e] = 0.f;
    for (int l = 0; l < KM; ++l) {
        const float v = in[row * KM + l];
#pragma unroll
        for (int e = 0; e < KPT; ++e) acc[e] = fmaf(v, S[l * KM + kq * KPT + e], acc[e]);
    }
#pragma unroll
    for (int e = 0; e < KPT; ++e) out[row * KM + kq * KPT + e] = acc[e];
}

// Z[c][:] = (sum_a Mbar[a][c] Q[a][:]) (S if apply_s), for a tile of 64 columns; Gram partial of
// the tile's rows of Z into G[tile].
template <int KM>
__global__ void __launch_bounds__(TP) pow_t_kernel(const __grid_constant__ PowGroup g, int apply_s) {
    constexpr int KPT = KM / 4;
    __shared__ __align__(16) float As[PR][PC];
    __shared__ __align__(16) float Xs[PR * KM];
    __shared__ __align__(16) float Zs[PC * KM];
    __shared__ __align__(16) float Z2[PC * KM];
    __shared__ __align__(16) float Ss[KM * KM];
    int mi = 0;
    while (mi + 1 < g.nmat && blockIdx.x >= static_cast<unsigned>(g.mat[mi + 1].t0)) ++mi;
    const PowMat& M = g.mat[mi];
    if (!M.active) return;
    const int tile = blockIdx.x - M.t0, c0 = tile * PC;
    const int mp = M.mp, np = M.np, k = M.k;
    const int tid = threadIdx.x, cl = tid & 63, kq = tid >> 6;
    float acc[KPT];
#pragma unroll
    for (int e = 0; e < KPT; ++e) acc[e] = 0.f;
    // each thread stages two float4 of every 32 x 64 block of Mbar; the next block's loads are
    // issued before the current block is used
    constexpr int LPT = PR * PC / 4 / TP;                      // = 2 float4 of Mbar
    constexpr int XPT = PR * KM / TP;                          // = 2 or 4 entries of Q
    float4 nxt[2][LPT];                                        // two blocks in flight
    float xn[2][XPT];
    auto fetch = [&](int a0, int bufi) {
#pragma unroll
        for (int l = 0; l < LPT; ++l) {
            const int o = tid + l * TP, rr = o / (PC / 4), cc = 4 * (o % (PC / 4));
            const int a = a0 + rr, c = c0 + cc;
            nxt[bufi][l] = a < mp && c < np ? *reinterpret_cast<const float4*>(M.Mbar + (int64_t)a * np + c)   // n' % 4 == 0
                                            : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int l = 0; l < XPT; ++l) {
            const int o = tid + l * TP, rr = o / KM, q = o % KM, a = a0 + rr;
            xn[bufi][l] = a < mp && q < k ? M.Q[(int64_t)a * k + q] : 0.f;
        }
    };
    fetch(0, 0);
    if (PR < mp) fetch(PR, 1);
    for (int a0 = 0, bi = 0; a0 < mp; a0 += PR, bi ^= 1) {
        if (bi == 0) {
#pragma unroll
            for (int l = 0; l < LPT; ++l) {
                const int o = tid + l * TP, rr = o / (PC / 4), cc = 4 * (o % (PC / 4));
                *reinterpret_cast<float4*>(&As[rr][cc]) = nxt[0][l];
            }
#pragma unroll
            for (int l = 0; l < XPT; ++l) Xs[tid + l * TP] = xn[0][l];
        } else {
#pragma unroll
            for (int l = 0; l < LPT; ++l) {
                const int o = tid + l * TP, rr = o / (PC / 4), cc = 4 * (o % (PC / 4));
                *reinterpret_cast<float4*>(&As[rr][cc]) = nxt[1][l];
            }
#pragma unroll
            for (int l = 0; l < XPT; ++l) Xs[tid + l * TP] = xn[1][l];
        }
        __syncthreads();
        if (a0 + 2 * PR < mp) {
            if (bi == 0) fetch(a0 + 2 * PR, 0);
            else fetch(a0 + 2 * PR, 1);
        }
#pragma unroll 8
        for (int rr = 0; rr < PR; ++rr) {
            const float m = As[rr][cl];
#pragma unroll
            for (int e = 0; e < KPT; ++e) acc[e] = fmaf(m, Xs[rr * KM + kq * KPT + e], acc[e]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int e = 0; e < KPT; ++e) Zs[cl * KM + kq * KPT + e] = acc[e];
    for (int o = tid; o < KM * KM; o += TP) {
        const int a = o / KM, b = o % KM;
        Ss[o] = a < k && b < k ? M.S[a * k + b] : (a == b ? 1.f : 0.f);
    }
    __syncthreads();
    const float* Zo = Zs;
    if (apply_s) {
        apply_S<KM>(Zs, Ss, Z2);
        Zo = Z2;
    }
    __syncthreads();
    const int nrows = np - c0 < PC ? np - c0 : PC;
    for (int o = tid; o < nrows * KM; o += TP) {
        const int c = o / KM, q = o % KM;
        if (q < k) M.Z[(int64_t)(c0 + c) * k + q] = Zo[o];
    }
    gram_partial<KM>(Zo, nrows, M.G + (int64_t)tile * KM * KM);
}

// part[chunk][q][a] = sum over the chunk's NCH columns c of Mbar[a][c] Z[c][q], for one tile of
// 64 rows a: CTA (row tile, chunk), the chunk walked in 64-column blocks.
template <int KM>
__global__ void __launch_bounds__(TP) pow_n_kernel(const __grid_constant__ PowGroup g) {
    constexpr int KPT = KM / 4;
    __shared__ __align__(16) float As[PC][PC + 1];            // 64 rows x 64 columns
    __shared__ __align__(16) float Ys[PC * KM];
    int mi = 0;
    while (mi + 1 < g.nmat && blockIdx.x >= static_cast<unsigned>(g.mat[mi + 1].n0)) ++mi;
    const PowMat& M = g.mat[mi];
    if (!M.active) return;
    const int nrt = (M.mp + PC - 1) / PC;
    const int chunk = (blockIdx.x - M.n0) / nrt, rt = (blockIdx.x - M.n0) % nrt;
    const int a0 = rt * PC, cbeg = chunk * NCH;
    const int mp = M.mp, np = M.np, k = M.k;
    const int cend = cbeg + NCH < np ? cbeg + NCH : np;
    const int tid = threadIdx.x, al = tid & 63, kq = tid >> 6;
    constexpr int LPT = PC * PC / 4 / TP;                      // = 4 float4 of each 64 x 64 block
    constexpr int YPT = PC * KM / TP;                          // = 4 or 8 entries of Z
    float4 nxt[LPT];
    float yn[YPT];
    auto fetch = [&](int c0) {
#pragma unroll
        for (int l = 0; l < LPT; ++l) {
            const int o = tid + l * TP, rr = o / (PC / 4), cc = 4 * (o % (PC / 4));
            const int a = a0 + rr, c = c0 + cc;
            nxt[l] = a < mp && c < cend ? *reinterpret_cast<const float4*>(M.Mbar + (int64_t)a * np + c)
                                        : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int l = 0; l < YPT; ++l) {
            const int o = tid + l * TP, cc = o / KM, q = o % KM, c = c0 + cc;
            yn[l] = c < cend && q < k ? M.Z[(int64_t)c * k + q] : 0.f;
        }
    };
    float acc[KPT];
#pragma unroll
    for (int e = 0; e < KPT; ++e) acc[e] = 0.f;
    fetch(cbeg);
    for (int c0 = cbeg; c0 < cend; c0 += PC) {
        __syncthreads();
#pragma unroll
        for (int l = 0; l < LPT; ++l) {
            const int o = tid + l * TP, rr = o / (PC / 4), cc = 4 * (o % (PC / 4));
            As[rr][cc] = nxt[l].x; As[rr][cc + 1] = nxt[l].y; As[rr][cc + 2] = nxt[l].z; As[rr][cc + 3] = nxt[l].w;
        }
#pragma unroll
        for (int l = 0; l < YPT; ++l) Ys[tid + l * TP] = yn[l];
        __syncthreads();
        if (c0 + PC < cend) fetch(c0 + PC);
#pragma unroll 8
        for (int cc = 0; cc < PC; ++cc) {
            const float m = As[al][cc];
#pragma unroll
            for (int e = 0; e < KPT; ++e) acc[e] = fmaf(m, Ys[cc * KM + kq * KPT + e], acc[e]);
        }
    }
    const int a = a0 + al;
    float* part = M.part + (int64_t)chunk * KM * mp;
    if (a < mp)
#pragma unroll
        for (int e = 0; e < KPT; ++e) part[(int64_t)(kq * KPT + e) * mp + a] = acc[e];
}

// Q[a][:] = (sum over chunks of part[chunk][:][a]) S for a tile of 64 rows; Gram partial into G.
template <int KM>
__global__ void __launch_bounds__(TP) pow_r_kernel(const __grid_constant__ PowGroup g) {
    constexpr int KPT = KM / 4;
    __shared__ __align__(16) float Qs[PC * KM];
    __shared__ __align__(16) float Q2[PC * KM];
    __shared__ __align__(16) float Ss[KM * KM];
    int mi = 0;
    while (mi + 1 < g.nmat && blockIdx.x >= static_cast<unsigned>(g.mat[mi + 1].r0)) ++mi;
    const PowMat& M = g.mat[mi];
    if (!M.active) return;
    const int tile = blockIdx.x - M.r0, a0 = tile * PC;
    const int mp = M.mp, k = M.k, nch = M.nn;
    const int tid = threadIdx.x, al = tid & 63, kq = tid >> 6;
    const int a = a0 + al;
    float acc[KPT];
#pragma unroll
    for (int e = 0; e < KPT; ++e) acc[e] = 0.f;
    if (a < mp)
#pragma unroll 4
        for (int ch = 0; ch < nch; ++ch) {                      // fixed order over the chunks
            const float* p = M.part + (int64_t)ch * KM * mp + a;
#pragma unroll
            for (int e = 0; e < KPT; ++e) acc[e] += p[(int64_t)(kq * KPT + e) * mp];
        }
#pragma unroll
    for (int e = 0; e < KPT; ++e) Qs[al * KM + kq * KPT + e] = acc[e];
    for (int o = tid; o < KM * KM; o += TP) {
        const int r = o / KM, c = o % KM;
        Ss[o] = r < k && c < k ? M.S[r * k + c] : (r == c ? 1.f : 0.f);
    }
    __syncthreads();
    apply_S<KM>(Qs, Ss, Q2);
    __syncthreads();
    const int nrows = mp - a0 < PC ? mp - a0 : PC;
    for (int o = tid; o < nrows * KM; o += TP) {
        const int r = o / KM, q = o % KM;
        if (q < k) M.Q[(int64_t)(a0 + r) * k + q] = Q2[o];
    }
    gram_partial<KM>(Q2, nrows, M.G + (int64_t)tile * KM * KM);
}

// Q[a][:] <- Q[a][:] S for a tile of 64 rows (rows are independent: in place); Gram partial
// into G when gram.
template <int KM>
__global__ void __launch_bounds__(TP) pow_apply_kernel(const __grid_constant__ PowGroup g, int gram) {
    __shared__ __align__(16) float Qs[PC * KM];
    __shared__ __align__(16) float Q2[PC * KM];
    __shared__ __align__(16) float Ss[KM * KM];
    int mi = 0;
    while (mi + 1 < g.nmat && blockIdx.x >= static_cast<unsigned>(g.mat[mi + 1].r0)) ++mi;
    const PowMat& M = g.mat[mi];
    if (!M.active) return;
    const int tile = blockIdx.x - M.r0, a0 = tile * PC;
    const int mp = M.mp, k = M.k, tid = threadIdx.x;
    const int nrows = mp - a0 < PC ? mp - a0 : PC;
    for (int o = tid; o < PC * KM; o += TP) {
        const int r = o / KM, q = o % KM;
        Qs[o] = r < nrows && q < k ? M.Q[(int64_t)(a0 + r) * k + q] : 0.f;
    }
    for (int o = tid; o < KM * KM; o += TP) {
        const int r = o / KM, c = o % KM;
        Ss[o] = r < k && c < k ? M.S[r * k + c] : (r == c ? 1.f : 0.f);
    }
    __syncthreads();
    apply_S<KM>(Qs, Ss, Q2);
    __syncthreads();
    for (int o = tid; o < nrows * KM; o += TP) {
        const int r = o / KM, q = o % KM;
        if (q < k) M.Q[(int64_t)(a0 + r) * k + q] = Q2[o];
    }
    if (gram) gram_partial<KM>(Q2, nrows, M.G + (int64_t)tile * KM * KM);
}

// One warp per matrix: Gm = sum over the ntile partials (fp64 accumulation, tile order).
// mode 0: Gm = L L^T (fp32 Cholesky, retried with a growing diagonal shift on breakdown) and
// S = L^{-T}, so X S has orthonormal columns when Gm = X^T X; mode 1: the sum itself into H (the
// Rayleigh-Ritz Gram).
constexpr int TCH = 1024;              // threads of pow_chol_kernel

template <int KM>
__global__ void __launch_bounds__(TCH) pow_chol_kernel(const __grid_constant__ PowGroup g, int use_t_tiles, int mode) {
    __shared__ float Gs[KM][KM + 1];
    __shared__ float Ls[KM][KM + 1];
    __shared__ float Xi[KM][KM + 1];                           // L^{-1}, column c by lane c
    __shared__ double Gq[4][KM * KM];
    const PowMat& M = g.mat[blockIdx.x];
    if (!M.active) return;
    const int k = M.k, lane = threadIdx.x;
    const int nt = use_t_tiles ? M.nt : M.nr;
    // entry o of the sum over the nt partials: four threads take the tiles t = j (mod 4), each
    // with two accumulators, and the four slices are added in order
    for (int w = threadIdx.x; w < 4 * k * k; w += TCH) {
        const int o = w >> 2, j = w & 3, a = o / k, b = o % k;
        const float* p = M.G + a * KM + b;
        double s0 = 0.0, s1 = 0.0;
        int t = j;
        for (; t + 4 < nt; t += 8) {
            s0 += static_cast<double>(p[(int64_t)t * KM * KM]);
            s1 += static_cast<double>(p[(int64_t)(t + 4) * KM * KM]);
        }
        if (t < nt) s0 += static_cast<double>(p[(int64_t)t * KM * KM]);
        Gq[j][o] = s0 + s1;
    }
    __syncthreads();
    for (int o = threadIdx.x; o < k * k; o += TCH)
        Gs[o / k][o % k] = static_cast<float>((Gq[0][o] + Gq[1][o]) + (Gq[2][o] + Gq[3][o]));
    __syncthreads();
    if (threadIdx.x >= 32) return;                             // one warp factors
    if (mode == 1) {
        for (int o = lane; o < k * k; o += 32) M.H[o] = Gs[o / k][o % k];
        return;
    }
    float tr = 0.f;
    for (int i = 0; i < k; ++i) tr += Gs[i][i];
    if (lane == 0 && M.flag && (!(tr > 0.f) || !isfinite(tr))) atomicAdd(M.flag + 6, 1);   // degenerate block
    float shift = 0.f;
    for (int attempt = 0; attempt < 6; ++attempt) {
        for (int o = lane; o < k * k; o += 32) Ls[o / k][o % k] = Gs[o / k][o % k] + (o / k == o % k ? shift : 0.f);
        __syncwarp();
        bool ok = true;
        for (int j = 0; j < k && ok; ++j) {                    // right-looking, column j
            const float d = Ls[j][j];
            ok = d > 0.f;                                      // same value in every lane
            if (ok) {
                const float ljj = sqrtf(d);
                __syncwarp();
                for (int i = j + lane; i < k; i += 32) Ls[i][j] = i == j ? ljj : Ls[i][j] / ljj;
                __syncwarp();
                const int w = k - j - 1;
                for (int o = lane; o < w * w; o += 32) {
                    const int i = j + 1 + o / w, l = j + 1 + o % w;
                    if (l <= i) Ls[i][l] -= Ls[i][j] * Ls[l][j];
                }
                __syncwarp();
            }
        }
        if (ok) {
            if (lane < k) {                                    // column c = lane of L^{-1}
                const int c = lane;
                for (int i = 0; i < k; ++i) {
                    float v = i == c ? 1.f : 0.f;
                    for (int l = c; l < i; ++l) v -= Ls[i][l] * Xi[l][c];
                    Xi[i][c] = i < c ? 0.f : v / Ls[i][i];
                }
            }
            __syncwarp();
            for (int o = lane; o < k * k; o += 32) M.S[o] = Xi[o % k][o / k];   // S = L^{-T}
            if (attempt > 0 && lane == 0 && M.flag) atomicAdd(M.flag, 1);
            return;
        }
        shift = (shift == 0.f ? 1e-7f : shift * 100.f) * (tr > 0.f ? tr / k : 1.f);
        __syncwarp();
    }
    // no factorisation: leave S as identity and count it
    for (int o = lane; o < k * k; o += 32) M.S[o] = o / k == o % k ? 1.f : 0.f;
    if (lane == 0 && M.flag) { atomicAdd(M.flag, 1000); atomicAdd(M.flag + 6, 1); }
}

template <int KM>
cudaError_t pow_launch(const PowGroup& g, int stage, int arg, cudaStream_t st) {
    switch (stage) {
        case 0: pow_t_kernel<KM><<<g.tot_t, TP, 0, st>>>(g, arg); break;
        case 1: pow_n_kernel<KM><<<g.tot_n, TP, 0, st>>>(g); break;
        case 2: pow_r_kernel<KM><<<g.tot_r, TP, 0, st>>>(g); break;
        case 3: pow_apply_kernel<KM><<<g.tot_r, TP, 0, st>>>(g, arg); break;
        case 4: pow_chol_kernel<KM><<<g.nmat, TCH, 0, st>>>(g, arg, 0); break;
        case 5: pow_chol_kernel<KM><<<g.nmat, TCH, 0, st>>>(g, arg, 1); break;
        default: return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

}  // namespace

int pow_tile() { return PC; }
int pow_chunk() { return NCH; }

cudaError_t pow_stage(const PowGroup& g, int stage, int arg, cudaStream_t st) {
    if (g.nmat <= 0) return cudaSuccess;
    int kmax = 0;
    for (int i = 0; i < g.nmat; ++i) kmax = g.mat[i].k > kmax ? g.mat[i].k : kmax;
    if (kmax <= 16) return pow_launch<16>(g, stage, arg, st);
    if (kmax <= 32) return pow_launch<32>(g, stage, arg, st);
    return cudaErrorInvalidValue;
}

}  // namespace glr
