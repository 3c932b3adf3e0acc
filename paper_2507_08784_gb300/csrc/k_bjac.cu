// The paper-exact refresh (Eq. SVD-P1 with the full m' x m' basis) above m' = 1024: the
// eigen-decomposition H = Mbar Mbar^T = U diag(lambda) U^T by parallel block-cyclic two-sided
// Jacobi.
//
// H (n x n, n a multiple of 128) is cut into m = n / 64 blocks of 64 indices.  A round pairs the
// blocks by the circle method of a round-robin tournament (block 0 fixed, the others rotating one
// slot per round, so that every two blocks meet once in m - 1 rounds, one sweep), and the pairs
// of a round are stored next to each other: pair k holds rows and columns 128 k .. 128 k + 127.
// A round
//   1. takes each pair's 128 x 128 diagonal block S_k and forms J_k, one sweep of parallel cyclic
//      scalar Jacobi on S_k started from the identity (bjac_pair_kernel; the rotation formula
//      and circle ordering of the k x k eigen-solver), so that J_k stays close to the identity and
//      no reordering inside the pair is needed;
//   2. applies the block-diagonal J = diag(J_k): H <- J^T H J (each 128 x 128 pair block
//      J_i^T H_ij J_j, the upper ones formed and mirrored) and V <- V J, writing every 64-block
//      straight to its place in the next round's storage order;
// and a sweep ends with the off-diagonal norm, checked on the host against tol^2 of the total.
// V starts as the identity, so its columns follow H's storage order; at the end diag(H) and V
// are sorted by descending eigenvalue with the sign rule of the small solvers (sort_fix_basis).
//
// The block products are FFMA in fp32 (128 x 128 x 128 per product, 8 x 8 outputs a thread);
// the rotations keep H symmetric to rounding: an upper block and its mirror are written from the
// same registers and the diagonal pair blocks are symmetrised.
#include "glr_internal.cuh"

namespace glr {

namespace {

constexpr int BT = 256;            // threads of the block-product kernels
constexpr int KC = 32;             // K slice of a product
constexpr int LDS = 132;           // padded shared row (floats)

// storage position of block x in round rd of the tournament over m blocks, and the block at
// storage position p
__device__ __forceinline__ int position_of(int x, int m, int rd) {
    const int s = x == 0 ? 0 : 1 + ((x - 1 - rd) % (m - 1) + (m - 1)) % (m - 1);
    return s < m / 2 ? 2 * s : 2 * (m - 1 - s) + 1;
}
__device__ __forceinline__ int block_at(int p, int m, int rd) {
    const int s = (p & 1) ? m - 1 - (p >> 1) : (p >> 1);
    return s == 0 ? 0 : 1 + (s - 1 + rd) % (m - 1);
}
// where the data at storage position p of round rd goes for round rd + 1
__device__ __forceinline__ int dest_of(int p, int m, int rd) {
    return position_of(block_at(p, m, rd), m, (rd + 1) % (m - 1));
}

// acc (rows 4 ty + {0..3}, 64 + 4 ty + {0..3}; columns likewise with tx) += A B over K = 128,
// A[i][a] = A0[i lda + a] (a contiguous), B[a][j] = B0[a 128 + j] (j contiguous); As, Bs are
// KC x LDS slices in shared memory.
__device__ __forceinline__ void gemm128(const float* A0, int64_t lda, const float* B0, float (*As)[LDS],
                                        float (*Bs)[LDS], float (&acc)[8][8]) {
    const int t = threadIdx.x, tx = t & 15, ty = t >> 4;
    for (int kc = 0; kc < 128; kc += KC) {
        for (int e = t; e < 128 * KC; e += BT) {         // A: rows i, 32 consecutive a per row
            const int i = e / KC, a = e % KC;
            As[a][i] = A0[(int64_t)i * lda + kc + a];
        }
        for (int e = t; e < 128 * KC / 4; e += BT) {     // B: float4 along j
            const int a = e / 32, j4 = e % 32;
            *reinterpret_cast<float4*>(&Bs[a][4 * j4]) =
                *reinterpret_cast<const float4*>(B0 + (int64_t)(kc + a) * 128 + 4 * j4);
        }
        __syncthreads();
#pragma unroll 4
        for (int a = 0; a < KC; ++a) {
            const float4 a0 = *reinterpret_cast<const float4*>(&As[a][4 * ty]);
            const float4 a1 = *reinterpret_cast<const float4*>(&As[a][64 + 4 * ty]);
            const float4 b0 = *reinterpret_cast<const float4*>(&Bs[a][4 * tx]);
            const float4 b1 = *reinterpret_cast<const float4*>(&Bs[a][64 + 4 * tx]);
            const float av[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
            const float bv[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
            for (int u = 0; u < 8; ++u)
#pragma unroll
                for (int v = 0; v < 8; ++v) acc[u][v] = fmaf(av[u], bv[v], acc[u][v]);
        }
        __syncthreads();
    }
}
__device__ __forceinline__ int row_of(int u) { return (u < 4 ? 0 : 64) + 4 * (threadIdx.x >> 4) + (u & 3); }
__device__ __forceinline__ int col_of(int v) { return (v < 4 ? 0 : 64) + 4 * (threadIdx.x & 15) + (v & 3); }

// H2 <- (J^T H J) in the next round's order: one CTA per pair block (ki <= kj) of a matrix.
__global__ void __launch_bounds__(BT) bjac_apply_h_kernel(const __grid_constant__ BjacGroup g) {
    extern __shared__ float sm[];
    float (*As)[LDS] = reinterpret_cast<float (*)[LDS]>(sm);
    float (*Bs)[LDS] = reinterpret_cast<float (*)[LDS]>(sm + KC * LDS);
    float (*Xs)[LDS] = reinterpret_cast<float (*)[LDS]>(sm + 2 * KC * LDS);
    int mi = 0;
    while (mi + 1 < g.nmat && g.mat[mi + 1].tile0h <= (int)blockIdx.x) ++mi;
    const BjacMat& M = g.mat[mi];
    const int n = M.n, P = n / 128, m = n / 64;
    int e = blockIdx.x - M.tile0h, ki = 0;
    while (e >= P - ki) { e -= P - ki; ++ki; }
    const int kj = ki + e;
    float acc[8][8] = {};
    // X = H[pair ki, pair kj] J_kj
    gemm128(M.H + (int64_t)(128 * ki) * n + 128 * kj, n, M.J + (int64_t)kj * 16384, As, Bs, acc);
#pragma unroll
    for (int u = 0; u < 8; ++u)
#pragma unroll
        for (int v = 0; v < 8; ++v) Xs[row_of(u)][col_of(v)] = acc[u][v];
    __syncthreads();
    // out = J_ki^T X: A[i][a] = J_ki[a][i], read as the transposed slice below
    float out[8][8] = {};
    {
        const int t = threadIdx.x, tx = t & 15, ty = t >> 4;
        const float* Jk = M.J + (int64_t)ki * 16384;
        for (int kc = 0; kc < 128; kc += KC) {
            for (int q = t; q < 128 * KC / 4; q += BT) {
                const int a = q / 32, i4 = q % 32;
                *reinterpret_cast<float4*>(&As[a][4 * i4]) =
                    *reinterpret_cast<const float4*>(Jk + (int64_t)(kc + a) * 128 + 4 * i4);
            }
            __syncthreads();
#pragma unroll 4
            for (int a = 0; a < KC; ++a) {
                const float4 a0 = *reinterpret_cast<const float4*>(&As[a][4 * ty]);
                const float4 a1 = *reinterpret_cast<const float4*>(&As[a][64 + 4 * ty]);
                const float4 b0 = *reinterpret_cast<const float4*>(&Xs[kc + a][4 * tx]);
                const float4 b1 = *reinterpret_cast<const float4*>(&Xs[kc + a][64 + 4 * tx]);
                const float av[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
                const float bv[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
                for (int u = 0; u < 8; ++u)
#pragma unroll
                    for (int v = 0; v < 8; ++v) out[u][v] = fmaf(av[u], bv[v], out[u][v]);
            }
            __syncthreads();
        }
    }
#pragma unroll
    for (int u = 0; u < 8; ++u)
#pragma unroll
        for (int v = 0; v < 8; ++v) Xs[row_of(u)][col_of(v)] = out[u][v];
    __syncthreads();
    // rows of block 2 ki + (i >= 64) and columns of block 2 kj + (j >= 64), at their next places
    const int rd = M.round;
    const int r0 = 64 * dest_of(2 * ki, m, rd), r1 = 64 * dest_of(2 * ki + 1, m, rd);
    const int c0 = 64 * dest_of(2 * kj, m, rd), c1 = 64 * dest_of(2 * kj + 1, m, rd);
    for (int q = threadIdx.x; q < 128 * 128; q += BT) {
        const int i = q >> 7, j = q & 127;
        const int gi = (i < 64 ? r0 : r1) + (i & 63), gj = (j < 64 ? c0 : c1) + (j & 63);
        if (ki == kj) {
            M.H2[(int64_t)gi * n + gj] = 0.5f * (Xs[i][j] + Xs[j][i]);
        } else {
            M.H2[(int64_t)gi * n + gj] = Xs[i][j];
        }
    }
    if (ki != kj) {                                    // the mirror block, rows j, columns i
        for (int q = threadIdx.x; q < 128 * 128; q += BT) {
            const int j = q >> 7, i = q & 127;
            const int gi = (i < 64 ? r0 : r1) + (i & 63), gj = (j < 64 ? c0 : c1) + (j & 63);
            M.H2[(int64_t)gj * n + gi] = Xs[i][j];
        }
    }
}

// V2 <- V J in the next round's column order: one CTA per (128-row tile, pair).
__global__ void __launch_bounds__(BT) bjac_apply_v_kernel(const __grid_constant__ BjacGroup g) {
    extern __shared__ float sm[];
    float (*As)[LDS] = reinterpret_cast<float (*)[LDS]>(sm);
    float (*Bs)[LDS] = reinterpret_cast<float (*)[LDS]>(sm + KC * LDS);
    int mi = 0;
    while (mi + 1 < g.nmat && g.mat[mi + 1].tile0v <= (int)blockIdx.x) ++mi;
    const BjacMat& M = g.mat[mi];
    const int n = M.n, P = n / 128, m = n / 64;
    const int e = blockIdx.x - M.tile0v, rt = e / P, k = e % P;
    float acc[8][8] = {};
    gemm128(M.V + (int64_t)(128 * rt) * n + 128 * k, n, M.J + (int64_t)k * 16384, As, Bs, acc);
    const int c0 = 64 * dest_of(2 * k, m, M.round), c1 = 64 * dest_of(2 * k + 1, m, M.round);
#pragma unroll
    for (int u = 0; u < 8; ++u) {
        float* row = M.V2 + (int64_t)(128 * rt + row_of(u)) * n;
        const int tx = threadIdx.x & 15;
        *reinterpret_cast<float4*>(row + c0 + 4 * tx) = make_float4(acc[u][0], acc[u][1], acc[u][2], acc[u][3]);
        *reinterpret_cast<float4*>(row + c1 + 4 * tx) = make_float4(acc[u][4], acc[u][5], acc[u][6], acc[u][7]);
    }
}

// Per matrix, per CTA: the squared diagonal and off-diagonal sums of H (part[2 (mat G + cta)]).
__global__ void __launch_bounds__(256) bjac_norms_kernel(const __grid_constant__ BjacGroup g, float* part) {
    const BjacMat& M = g.mat[blockIdx.y];
    const int n = M.n;
    float d = 0.f, o = 0.f;
    for (int r = blockIdx.x; r < n; r += gridDim.x) {
        const float* row = M.H + (int64_t)r * n;
        for (int c = threadIdx.x; c < n; c += 256) {
            const float v = row[c];
            if (c == r) d += v * v; else o += v * v;
        }
    }
    __shared__ float red[2][8];
#pragma unroll
    for (int s = 16; s > 0; s >>= 1) {
        d += __shfl_xor_sync(0xffffffffu, d, s);
        o += __shfl_xor_sync(0xffffffffu, o, s);
    }
    if ((threadIdx.x & 31) == 0) { red[0][threadIdx.x >> 5] = d; red[1][threadIdx.x >> 5] = o; }
    __syncthreads();
    if (threadIdx.x == 0) {
        float sd = 0.f, so = 0.f;
        for (int w = 0; w < 8; ++w) { sd += red[0][w]; so += red[1][w]; }
        float* out = part + 2 * ((int64_t)blockIdx.y * gridDim.x + blockIdx.x);
        out[0] = sd; out[1] = so;
    }
}

// One sweep of parallel cyclic two-sided Jacobi on the 128 x 128 diagonal pair block S_k of H,
// from W = I: 127 rounds of 64 disjoint rotations (circle ordering; Golub & Van Loan sym.schur2),
// each round's rotations formed from the round's own 2 x 2 diagonal blocks, then S <- R^T S R and
// W <- W R in one barrier-separated phase.  S is packed (upper triangle by rows), W padded to 129
// columns; J_k = W is written row-major.  512 threads, two CTAs per SM.
constexpr int PT = 512;
constexpr int PN = 128, PH = 64, PLD = 129;
constexpr int kPairItems = PH * (PH + 1) / 2;                 // 2 x 2 blocks (bi <= bj) of a round
constexpr size_t kPairSmem = sizeof(float) * (PN * (PN + 1) / 2 + PN * PLD);

__device__ __forceinline__ int pcircle(int x) { return 1 + ((x % (PN - 1)) + (PN - 1)) % (PN - 1); }

__global__ void __launch_bounds__(PT, 2) bjac_pair_kernel(const __grid_constant__ BjacGroup g) {
    extern __shared__ float psm[];
    float* Ss = psm;                                   // packed upper triangle: (r, c >= r) at off[r] + c
    float* Ws = psm + PN * (PN + 1) / 2;               // W[a][j] at a PLD + j
    __shared__ int off[PN + 1];
    __shared__ int4 spq[PH];
    __shared__ float2 scs[PH];
    int mi = 0;
    while (mi + 1 < g.nmat && g.mat[mi + 1].tile0p <= (int)blockIdx.x) ++mi;
    const BjacMat& M = g.mat[mi];
    const int n = M.n, k = blockIdx.x - M.tile0p, t = threadIdx.x;
    const float* S0 = M.H + (int64_t)(PN * k) * (n + 1);
    for (int r = t; r <= PN; r += PT) off[r] = r * PN - r * (r + 1) / 2;
    __syncthreads();
    for (int e = t; e < PN * PN; e += PT) {
        const int r = e >> 7, c = e & 127;
        if (c >= r) Ss[off[r] + c] = S0[(int64_t)r * n + c];
        Ws[r * PLD + c] = r == c ? 1.f : 0.f;
    }
    // this thread's 2 x 2 blocks: block row i folded with block row PH - 1 - i (equal counts)
    constexpr int kItems = (kPairItems + PT - 1) / PT;
    int myblk[kItems];
#pragma unroll
    for (int u = 0; u < kItems; ++u) {
        const int e = t + u * PT;
        myblk[u] = -1;
        if (e < kPairItems) {
            const int fr = e / (PH + 1), tt = e - fr * (PH + 1);
            int bi, bj;
            if (tt < PH - fr) { bi = fr; bj = fr + tt; }
            else { bi = PH - 1 - fr; bj = bi + (tt - (PH - fr)); }
            myblk[u] = bi | (bj << 16);
        }
    }
    const int wa = t & (PN - 1), wj0 = t >> 7;         // W: row wa, rotations wj0, wj0 + 4, ...
    __syncthreads();
    for (int rd = 0; rd < PN - 1; ++rd) {
        if (t < PH) {
            int p = (t == 0) ? 0 : pcircle(rd + t);
            int q = (t == 0) ? pcircle(rd) : pcircle(rd - t);
            if (p > q) { const int tmp = p; p = q; q = tmp; }
            float c = 1.f, s = 0.f;
            const float hpq = Ss[off[p] + q], hpp = Ss[off[p] + p], hqq = Ss[off[q] + q];
            if (fabsf(hpq) > 1e-30f && fabsf(hpq) > 1e-9f * sqrtf(fabsf(hpp * hqq))) {
                const float theta = (hqq - hpp) / (2.f * hpq);
                float tt;
                if (fabsf(theta) > 1e15f) tt = 0.5f / theta;
                else tt = copysignf(1.f, theta) / (fabsf(theta) + sqrtf(theta * theta + 1.f));
                c = 1.f / sqrtf(tt * tt + 1.f);
                s = tt * c;
            }
            spq[t] = make_int4(p, q, off[p], off[q]);
            scs[t] = make_float2(c, s);
        }
        __syncthreads();
#pragma unroll
        for (int u = 0; u < kItems; ++u) {              // S <- R^T S R, 2 x 2 block by block
            if (myblk[u] < 0) continue;
            const int bi = myblk[u] & 0xFFFF, bj = myblk[u] >> 16;
            const float2 rci = scs[bi], rcj = scs[bj];
            const float ci = rci.x, si = rci.y, cj = rcj.x, sj = rcj.y;
            if (si == 0.f && sj == 0.f) continue;
            const int4 pi4 = spq[bi], pj4 = spq[bj];
            const int pi = pi4.x, qi = pi4.y, pj = pj4.x, qj = pj4.y;
            if (bi == bj) {
                const int i00 = pi4.z + pi, i01 = pi4.z + qi, i11 = pi4.w + qi;
                const float h00 = Ss[i00], h01 = Ss[i01], h11 = Ss[i11];
                const float a00 = ci * h00 - si * h01, a01 = ci * h01 - si * h11;
                const float a10 = si * h00 + ci * h01, a11 = si * h01 + ci * h11;
                Ss[i00] = cj * a00 - sj * a01;
                Ss[i11] = sj * a10 + cj * a11;
                Ss[i01] = 0.f;
                continue;
            }
            const int i00 = pi <= pj ? pi4.z + pj : pj4.z + pi;
            const int i01 = pi <= qj ? pi4.z + qj : pj4.w + pi;
            const int i10 = qi <= pj ? pi4.w + pj : pj4.z + qi;
            const int i11 = qi <= qj ? pi4.w + qj : pj4.w + qi;
            const float h00 = Ss[i00], h01 = Ss[i01], h10 = Ss[i10], h11 = Ss[i11];
            const float a00 = ci * h00 - si * h10, a01 = ci * h01 - si * h11;
            const float a10 = si * h00 + ci * h10, a11 = si * h01 + ci * h11;
            Ss[i00] = cj * a00 - sj * a01;
            Ss[i01] = sj * a00 + cj * a01;
            Ss[i10] = cj * a10 - sj * a11;
            Ss[i11] = sj * a10 + cj * a11;
        }
        float* wr = Ws + wa * PLD;                      // W <- W R
#pragma unroll 4
        for (int j = wj0; j < PH; j += PT / PN) {
            const float2 cs = scs[j];
            if (cs.y == 0.f) continue;
            const int4 pq = spq[j];
            const float vp = wr[pq.x], vq = wr[pq.y];
            wr[pq.x] = cs.x * vp - cs.y * vq;
            wr[pq.y] = cs.y * vp + cs.x * vq;
        }
        __syncthreads();
    }
    float* J = M.J + (int64_t)k * PN * PN;
    for (int e = t; e < PN * PN; e += PT) J[e] = Ws[(e >> 7) * PLD + (e & 127)];
}

__global__ void count_flag_kernel(int* flag, int v) { atomicAdd(flag, v); }

__global__ void bjac_eye_kernel(float* V, int n) {
    for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < (int64_t)n * n; q += (int64_t)gridDim.x * blockDim.x)
        V[q] = (q / n == q % n) ? 1.f : 0.f;
}
__global__ void bjac_diag_kernel(const float* H, int n, float* evals) {
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) evals[i] = H[(int64_t)i * n + i];
}

constexpr size_t kApplyHSmem = sizeof(float) * (2 * KC + 128) * LDS;
constexpr size_t kApplyVSmem = sizeof(float) * (2 * KC) * LDS;

}  // namespace

cudaError_t bjac_apply(BjacGroup& g, cudaStream_t st) {
    if (g.nmat <= 0) return cudaSuccess;
    g.tiles_h = g.tiles_v = 0;
    for (int i = 0; i < g.nmat; ++i) {
        BjacMat& M = g.mat[i];
        if (M.n < 256 || M.n % 128 || M.n > kBjacMaxN) return cudaErrorInvalidValue;
        const int P = M.n / 128;
        M.tile0h = g.tiles_h; g.tiles_h += P * (P + 1) / 2;
        M.tile0v = g.tiles_v; g.tiles_v += P * P;
    }
    cudaError_t e = cudaFuncSetAttribute(bjac_apply_h_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kApplyHSmem);
    if (e != cudaSuccess) return e;
    bjac_apply_h_kernel<<<g.tiles_h, BT, kApplyHSmem, st>>>(g);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    bjac_apply_v_kernel<<<g.tiles_v, BT, kApplyVSmem, st>>>(g);
    return cudaGetLastError();
}

cudaError_t bjac_pairs(BjacGroup& g, cudaStream_t st) {
    if (g.nmat <= 0) return cudaSuccess;
    int tiles = 0;
    for (int i = 0; i < g.nmat; ++i) {
        BjacMat& M = g.mat[i];
        if (M.n < 256 || M.n % 128 || M.n > kBjacMaxN) return cudaErrorInvalidValue;
        M.tile0p = tiles;
        tiles += M.n / 128;
    }
    cudaError_t e = cudaFuncSetAttribute(bjac_pair_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kPairSmem);
    if (e != cudaSuccess) return e;
    bjac_pair_kernel<<<tiles, PT, kPairSmem, st>>>(g);
    return cudaGetLastError();
}

cudaError_t bjac_norms(const BjacGroup& g, float* part, cudaStream_t st) {
    if (g.nmat <= 0) return cudaSuccess;
    bjac_norms_kernel<<<dim3(kBjacNormCtas, g.nmat), 256, 0, st>>>(g, part);
    return cudaGetLastError();
}

cudaError_t count_flag(int* flag, int v, cudaStream_t st) {
    count_flag_kernel<<<1, 1, 0, st>>>(flag, v);
    return cudaGetLastError();
}

cudaError_t bjac_eye(float* V, int n, cudaStream_t st) {
    bjac_eye_kernel<<<1024, 256, 0, st>>>(V, n);
    return cudaGetLastError();
}

cudaError_t bjac_diag(const float* H, int n, float* evals, cudaStream_t st) {
    bjac_diag_kernel<<<(n + 255) / 256, 256, 0, st>>>(H, n, evals);
    return cudaGetLastError();
}

}  // namespace glr
