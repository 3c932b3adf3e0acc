// Refresh kernels: the Semi-Lazy SVD step of Eq. SVD-P1 on the device.
//  * full basis: eigen-decomposition of H = Mbar Mbar^T by parallel cyclic Jacobi;
//  * truncated basis: block power iteration with CholeskyQR2, Rayleigh-Ritz (Jacobi on the
//    k x k projected Gram matrix) and the Householder reconstruction of the complement.
#include "glr_internal.cuh"

namespace glr {

namespace {

// ------------------------------------------------------------------------------------------
// Parallel cyclic two-sided Jacobi (one CTA).  Each round applies n/2 disjoint plane
// rotations chosen by the circle (round-robin) ordering: every rotation angle is computed
// from its own 2 x 2 diagonal block, then H <- J^T H J is applied block-wise (each 2 x 2
// block of H depends only on the rotations of its row pair and column pair, so the update
// is in place) and V <- V J.  Rotation formula: Golub & Van Loan, sym.schur2.
// ------------------------------------------------------------------------------------------
__device__ __forceinline__ int circle(int x, int nm1) { return 1 + ((x % nm1) + nm1) % nm1; }

__global__ void __launch_bounds__(1024) jacobi_kernel(float* Hg, int n, float* Vg, float* evals,
                                                      int* sweeps_out, int use_smem, int max_sweeps,
                                                      float tol) {
    extern __shared__ float sm[];
    const int npad = n + (n & 1), half = npad / 2, nm1 = npad - 1;
    const int tid = threadIdx.x, nth = blockDim.x;
    float* H = use_smem ? sm : Hg;
    float* V = use_smem ? sm + (size_t)n * n : Vg;
    float* cs = use_smem ? sm + 2 * (size_t)n * n : sm;
    float* sn = cs + half;
    int* pp = reinterpret_cast<int*>(sn + half);
    int* qq = pp + half;
    __shared__ float red_off[32], red_tot[32];
    __shared__ int done;
    if (use_smem)
        for (int e = tid; e < n * n; e += nth) H[e] = Hg[e];
    for (int e = tid; e < n * n; e += nth) V[e] = (e / n == e % n) ? 1.f : 0.f;
    __syncthreads();
    int sweep = 0;
    for (; sweep < max_sweeps; ++sweep) {
        float off = 0.f, tot = 0.f;
        for (int e = tid; e < n * n; e += nth) {
            const float h = H[e];
            tot += h * h;
            if (e / n != e % n) off += h * h;
        }
        for (int o = 16; o > 0; o >>= 1) {
            off += __shfl_xor_sync(0xffffffffu, off, o);
            tot += __shfl_xor_sync(0xffffffffu, tot, o);
        }
        if ((tid & 31) == 0) { red_off[tid >> 5] = off; red_tot[tid >> 5] = tot; }
        __syncthreads();
        if (tid == 0) {
            float o2 = 0.f, t2 = 0.f;
            for (int w = 0; w < (nth + 31) / 32; ++w) { o2 += red_off[w]; t2 += red_tot[w]; }
            done = (o2 <= tol * tol * t2) ? 1 : 0;
        }
        __syncthreads();
        if (done) break;
        for (int rd = 0; rd < nm1; ++rd) {
            for (int i = tid; i < half; i += nth) {
                int p = (i == 0) ? 0 : circle(rd + i, nm1);
                int q = (i == 0) ? circle(rd, nm1) : circle(rd - i, nm1);
                if (p > q) { const int tmp = p; p = q; q = tmp; }
                float c = 1.f, s = 0.f;
                if (q < n) {
                    const float hpq = H[(size_t)p * n + q];
                    const float hpp = H[(size_t)p * n + p], hqq = H[(size_t)q * n + q];
                    if (fabsf(hpq) > 1e-30f && fabsf(hpq) > 1e-9f * sqrtf(fabsf(hpp * hqq))) {
                        const float theta = (hqq - hpp) / (2.f * hpq);
                        float t;
                        if (fabsf(theta) > 1e15f) t = 0.5f / theta;
                        else t = copysignf(1.f, theta) / (fabsf(theta) + sqrtf(theta * theta + 1.f));
                        c = 1.f / sqrtf(t * t + 1.f);   // correctly rounded: keeps c^2 + s^2 = 1 tight
                        s = t * c;
                    }
                }
                cs[i] = c; sn[i] = s; pp[i] = p; qq[i] = q;
            }
            __syncthreads();
            for (int e = tid; e < half * half; e += nth) {
                const int bi = e / half, bj = e % half;
                const int pi = pp[bi], qi = qq[bi], pj = pp[bj], qj = qq[bj];
                const float ci = cs[bi], si = sn[bi], cj = cs[bj], sj = sn[bj];
                if (si == 0.f && sj == 0.f) continue;
                const bool vqi = qi < n, vqj = qj < n;
                float h00 = H[(size_t)pi * n + pj];
                float h01 = vqj ? H[(size_t)pi * n + qj] : 0.f;
                float h10 = vqi ? H[(size_t)qi * n + pj] : 0.f;
                float h11 = (vqi && vqj) ? H[(size_t)qi * n + qj] : 0.f;
                // rows: J_i^T
                const float a00 = ci * h00 - si * h10, a01 = ci * h01 - si * h11;
                const float a10 = si * h00 + ci * h10, a11 = si * h01 + ci * h11;
                // columns: J_j
                float n00 = cj * a00 - sj * a01, n01 = sj * a00 + cj * a01;
                float n10 = cj * a10 - sj * a11, n11 = sj * a10 + cj * a11;
                if (bi == bj && si != 0.f) { n01 = 0.f; n10 = 0.f; }
                H[(size_t)pi * n + pj] = n00;
                if (vqj) H[(size_t)pi * n + qj] = n01;
                if (vqi) H[(size_t)qi * n + pj] = n10;
                if (vqi && vqj) H[(size_t)qi * n + qj] = n11;
            }
            for (int e = tid; e < n * half; e += nth) {
                const int a = e / half, bj = e % half;
                const float sj = sn[bj];
                if (sj == 0.f) continue;
                const int pj = pp[bj], qj = qq[bj];
                const float cj = cs[bj];
                const float vp = V[(size_t)a * n + pj], vq = V[(size_t)a * n + qj];
                V[(size_t)a * n + pj] = cj * vp - sj * vq;
                V[(size_t)a * n + qj] = sj * vp + cj * vq;
            }
            __syncthreads();
        }
    }
    for (int i = tid; i < n; i += nth) evals[i] = H[(size_t)i * n + i];
    if (use_smem)
        for (int e = tid; e < n * n; e += nth) Vg[e] = V[e];
    if (tid == 0 && sweeps_out) *sweeps_out = sweep;
}

__device__ __forceinline__ uint32_t float_order(float f) {
    const uint32_t u = __float_as_uint(f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// argmax |column| (first index on ties) of one column, by one warp; returns the sign there.
__device__ float warp_column_sign(const float* A, int rows, int ld, int col) {
    const int lane = threadIdx.x & 31;
    float best = -1.f;
    int bidx = 0x7fffffff;
    for (int a = lane; a < rows; a += 32) {
        const float v = fabsf(A[(size_t)a * ld + col]);
        if (v > best) { best = v; bidx = a; }
    }
    for (int o = 16; o > 0; o >>= 1) {
        const float ob = __shfl_xor_sync(0xffffffffu, best, o);
        const int oi = __shfl_xor_sync(0xffffffffu, bidx, o);
        if (ob > best || (ob == best && oi < bidx)) { best = ob; bidx = oi; }
    }
    return (bidx < rows && A[(size_t)bidx * ld + col] < 0.f) ? -1.f : 1.f;
}

__device__ __forceinline__ void sort_fix_body(const float* evals, const float* V, int n, int ncols, float* Out,
                                              int ldo, float* evals_sorted, int npow2) {
    extern __shared__ unsigned long long keys[];
    const int tid = threadIdx.x;
    for (int i = tid; i < npow2; i += blockDim.x)
        keys[i] = (i < n) ? ((static_cast<unsigned long long>(float_order(evals[i])) << 32) |
                             (0xFFFFFFFFull - static_cast<unsigned long long>(i)))
                          : 0ull;
    __syncthreads();
    for (int size = 2; size <= npow2; size <<= 1)
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            for (int i = tid; i < npow2; i += blockDim.x) {
                const int partner = i ^ stride;
                if (partner > i) {
                    const bool desc = (i & size) == 0;
                    const unsigned long long x = keys[i], y = keys[partner];
                    if ((x < y) == desc) { keys[i] = y; keys[partner] = x; }
                }
            }
            __syncthreads();
        }
    const int warp = tid >> 5, lane = tid & 31, nw = blockDim.x >> 5;
    for (int c = warp; c < ncols; c += nw) {
        const int src = static_cast<int>(0xFFFFFFFFull - (keys[c] & 0xFFFFFFFFull));
        const float sg = warp_column_sign(V, n, n, src);
        // renormalise: thousands of plane rotations let the column norms drift by a few ulp each
        float ss = 0.f;
        for (int a = lane; a < n; a += 32) { const float v = V[(size_t)a * n + src]; ss = fmaf(v, v, ss); }
        for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
        const float scale = sg / sqrtf(ss);
        for (int a = lane; a < n; a += 32) Out[(size_t)a * ldo + c] = scale * V[(size_t)a * n + src];
        if (lane == 0 && evals_sorted) evals_sorted[c] = evals[src];
    }
}
__global__ void __launch_bounds__(1024) sort_fix_kernel(const float* evals, const float* V, int n, int ncols,
                                                        float* Out, int ldo, float* evals_sorted, int npow2) {
    sort_fix_body(evals, V, n, ncols, Out, ldo, evals_sorted, npow2);
}
__global__ void __launch_bounds__(1024) sort_fix_group_kernel(const __grid_constant__ FinishGroup g, int npow2) {
    const FinishMat& M = g.mat[blockIdx.x];
    sort_fix_body(M.evals, M.V, M.k, M.k, M.W, M.k, M.evals_sorted, npow2);
}

__global__ void fix_signs_group_kernel(const __grid_constant__ FinishGroup g) {
    const FinishMat& M = g.mat[blockIdx.y];
    const int col = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (col >= M.k) return;
    const float sg = warp_column_sign(M.Q, M.mp, M.k, col);
    if (sg < 0.f)
        for (int a = threadIdx.x & 31; a < M.mp; a += 32) M.Q[(size_t)a * M.k + col] = -M.Q[(size_t)a * M.k + col];
}
__global__ void fix_signs_kernel(float* A, int rows, int cols) {
    const int col = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (col >= cols) return;
    const float sg = warp_column_sign(A, rows, cols, col);
    if (sg < 0.f)
        for (int a = threadIdx.x & 31; a < rows; a += 32) A[(size_t)a * cols + col] = -A[(size_t)a * cols + col];
}

// Right-looking Cholesky (one CTA) with a diagonal shift retry on breakdown.
__global__ void __launch_bounds__(1024) cholesky_kernel(float* A, int n, float* orig, int* flag) {
    const int tid = threadIdx.x, nth = blockDim.x;
    __shared__ int fail;
    __shared__ float shift, trace;
    for (int e = tid; e < n * n; e += nth) orig[e] = A[e];
    if (tid == 0) {
        float tr = 0.f;
        for (int i = 0; i < n; ++i) tr += orig[(size_t)i * n + i];
        trace = tr;
        shift = 0.f;
    }
    __syncthreads();
    int attempt = 0;
    for (; attempt < 6; ++attempt) {
        if (attempt > 0) {
            for (int e = tid; e < n * n; e += nth) A[e] = orig[e] + ((e / n == e % n) ? shift : 0.f);
        }
        if (tid == 0) fail = 0;
        __syncthreads();
        const float thresh = 1e-12f * fmaxf(trace / n, 1e-30f);
        for (int j = 0; j < n; ++j) {
            const float d = A[(size_t)j * n + j];
            if (!(d > thresh)) { fail = 1; break; }      // uniform: every thread reads the same d
            const float ljj = sqrtf(d);
            __syncthreads();
            if (tid == 0) A[(size_t)j * n + j] = ljj;
            for (int i = j + 1 + tid; i < n; i += nth) A[(size_t)i * n + j] /= ljj;
            __syncthreads();
            const int rem = n - j - 1;
            for (int e = tid; e < rem * rem; e += nth) {
                const int i = j + 1 + e / rem, l = j + 1 + e % rem;
                if (l <= i) A[(size_t)i * n + l] -= A[(size_t)i * n + j] * A[(size_t)l * n + j];
            }
            __syncthreads();
        }
        __syncthreads();
        if (!fail) break;
        if (tid == 0) shift = (attempt == 0 ? 1e-7f : shift * 100.f) * fmaxf(trace / n, 1e-30f);
        __syncthreads();
    }
    for (int e = tid; e < n * n; e += nth)
        if (e % n > e / n) A[e] = 0.f;
    if (tid == 0 && flag) {
        *flag = attempt;
        // no factorisation after every shift, or a Gram matrix with no positive trace (a zero or
        // non-finite block): the refresh cannot orthonormalise it (flag + 6 counts these)
        if (attempt == 6 || !(trace > 0.f) || !isfinite(trace)) atomicAdd(flag + 6, 1);
    }
}

// Q <- Q L^{-T}: one warp per row, y_j = (x_j - sum_{l<j} y_l L_jl) / L_jj.
__global__ void trsm_kernel(float* Q, int rows, int n, const float* L) {
    const int warp = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (warp >= rows) return;
    float* y = Q + (size_t)warp * n;
    for (int j = 0; j < n; ++j) {
        float acc = 0.f;
        for (int l = lane; l < j; l += 32) acc = fmaf(y[l], L[(size_t)j * n + l], acc);
        for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
        const float val = (y[j] - acc) / L[(size_t)j * n + j];
        __syncwarp();
        if (lane == 0) y[j] = val;
        __syncwarp();
    }
}

__global__ void random_block_kernel(float* Q, int rows, int cols, uint64_t seed, uint32_t t) {
    const int nq = (cols + 3) / 4;
    const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= (int64_t)rows * nq) return;
    const int i = static_cast<int>(e / nq), q = static_cast<int>(e % nq);
    const float4 g = gauss4(seed, t, static_cast<uint32_t>(i), static_cast<uint32_t>(q), kTagPowerInit);
    const float gv[4] = {g.x, g.y, g.z, g.w};
    for (int v = 0; v < 4; ++v)
        if (q * 4 + v < cols) Q[(size_t)i * cols + q * 4 + v] = gv[v];
}

// Householder reconstruction, top block: modified LU of S - Q[:k, :k] with s_j = -sign of the
// current Schur-complement entry of Q (so every pivot has magnitude >= 1); then
// T Y1^T = Utilde S by forward substitution.  W (k x k scratch) ends holding L1\Utilde.
__device__ __forceinline__ void hh_top_body(const float* Q, int k, float* W, float* Y, float* T, float* s) {
    const int tid = threadIdx.x, nth = blockDim.x;
    for (int e = tid; e < k * k; e += nth) W[e] = -Q[e];   // rows 0..k-1 of Q (ld = k)
    __syncthreads();
    for (int j = 0; j < k; ++j) {
        const float qjj = -W[(size_t)j * k + j];
        const float sj = qjj >= 0.f ? -1.f : 1.f;
        __syncthreads();
        if (tid == 0) { W[(size_t)j * k + j] += sj; s[j] = sj; }
        __syncthreads();
        const float piv = W[(size_t)j * k + j];
        for (int i = j + 1 + tid; i < k; i += nth) W[(size_t)i * k + j] /= piv;
        __syncthreads();
        const int rem = k - j - 1;
        for (int e = tid; e < rem * rem; e += nth) {
            const int i = j + 1 + e / rem, l = j + 1 + e % rem;
            W[(size_t)i * k + l] -= W[(size_t)i * k + j] * W[(size_t)j * k + l];
        }
        __syncthreads();
    }
    for (int e = tid; e < k * k; e += nth) {
        const int i = e / k, l = e % k;
        Y[(size_t)i * k + l] = i > l ? W[e] : (i == l ? 1.f : 0.f);
    }
    // T row i: T[i][l] = Ut[i][l] s_l - sum_{c<l} T[i][c] Y1[l][c]  (T upper triangular)
    for (int i = tid; i < k; i += nth) {
        float* Ti = T + (size_t)i * k;
        for (int l = 0; l < k; ++l) {
            if (l < i) { Ti[l] = 0.f; continue; }
            float x = W[(size_t)i * k + l] * s[l];
            for (int c = i; c < l; ++c) x -= Ti[c] * W[(size_t)l * k + c];
            Ti[l] = x;
        }
    }
}

__global__ void __launch_bounds__(1024) hh_top_kernel(const float* Q, int k, float* W, float* Y, float* T,
                                                      float* s) {
    hh_top_body(Q, k, W, Y, T, s);
}
__global__ void __launch_bounds__(1024) hh_top_group_kernel(const __grid_constant__ FinishGroup g) {
    const FinishMat& M = g.mat[blockIdx.x];
    hh_top_body(M.Q, M.k, M.Wtop, M.Y, M.T, M.s);
}

// Rows a >= k: Y[a, :] Utilde = -Q[a, :], one warp per row (forward substitution).
__device__ __forceinline__ void hh_rows_body(const float* Q, int mp, int k, const float* W, float* Y, int warp) {
    const int lane = threadIdx.x & 31;
    const int a = k + warp;
    if (a >= mp) return;
    float* y = Y + (size_t)a * k;
    const float* qa = Q + (size_t)a * k;
    for (int l = 0; l < k; ++l) {
        float acc = 0.f;
        for (int c = lane; c < l; c += 32) acc = fmaf(y[c], W[(size_t)c * k + l], acc);
        for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
        const float val = (-qa[l] - acc) / W[(size_t)l * k + l];
        __syncwarp();
        if (lane == 0) y[l] = val;
        __syncwarp();
    }
}
__global__ void hh_rows_kernel(const float* Q, int mp, int k, const float* W, float* Y) {
    hh_rows_body(Q, mp, k, W, Y, blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5));
}
__global__ void hh_rows_group_kernel(const __grid_constant__ FinishGroup g) {
    const FinishMat& M = g.mat[blockIdx.y];
    hh_rows_body(M.Q, M.mp, M.k, M.Wtop, M.Y, blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5));
}

__global__ void wy_basis_kernel(int mp, int k, const float* Y, const float* Yt, const float* dsign, float* U) {
    const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= (int64_t)mp * mp) return;
    const int a = static_cast<int>(e / mp), j = static_cast<int>(e % mp);
    float v = (a == j) ? 1.f : 0.f;
    for (int c = 0; c < k; ++c) v = fmaf(-Y[(size_t)a * k + c], Yt[(size_t)j * k + c], v);
    if (j < k) v *= dsign[j];
    U[e] = v;
}

}  // namespace

cudaError_t jacobi_eig(float* H, int n, float* V, float* evals, int* sweeps, cudaStream_t st) {
    const int npad = n + (n & 1), half = npad / 2;
    const size_t pair_bytes = (size_t)half * 16;
    const size_t full = 2 * sizeof(float) * (size_t)n * n + pair_bytes;
    const int use_smem = full <= 200 * 1024 ? 1 : 0;
    const size_t smem = use_smem ? full : pair_bytes;
    {   // per device: set on every call (cheap next to the launch)
        const cudaError_t ea = cudaFuncSetAttribute(jacobi_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 210 * 1024);
        if (ea != cudaSuccess) return ea;
    }
    const float tol = 4.f * 5.96e-8f * sqrtf(static_cast<float>(n)) + 1e-7f;
    // one thread per 2 x 2 block update of a round, rounded to whole warps (at most 1024)
    const int work = n * half > half * half ? n * half : half * half;
    const int nth = work >= 1024 ? 1024 : ((work + 31) / 32) * 32;
    jacobi_kernel<<<1, nth, smem, st>>>(H, n, V, evals, sweeps, use_smem, 40, tol);
    return cudaGetLastError();
}

cudaError_t sort_fix_basis(const float* evals, const float* V, int n, int ncols, float* Out, int ldo,
                           float* evals_sorted, cudaStream_t st) {
    int npow2 = 1;
    while (npow2 < n) npow2 <<= 1;
    sort_fix_kernel<<<1, 1024, sizeof(unsigned long long) * npow2, st>>>(evals, V, n, ncols, Out, ldo,
                                                                         evals_sorted, npow2);
    return cudaGetLastError();
}

cudaError_t fix_column_signs(float* A, int rows, int cols, cudaStream_t st) {
    fix_signs_kernel<<<(cols + 7) / 8, 256, 0, st>>>(A, rows, cols);
    return cudaGetLastError();
}

cudaError_t finish_group(const FinishGroup& g, int stage, cudaStream_t st) {
    if (g.nmat <= 0) return cudaSuccess;
    int kmax = 0, rows_max = 0;
    for (int i = 0; i < g.nmat; ++i) {
        kmax = g.mat[i].k > kmax ? g.mat[i].k : kmax;
        rows_max = g.mat[i].mp - g.mat[i].k > rows_max ? g.mat[i].mp - g.mat[i].k : rows_max;
    }
    if (stage == 0) {                                   // sort the eigenpairs, normalise, fix signs
        int npow2 = 1;
        while (npow2 < kmax) npow2 <<= 1;
        sort_fix_group_kernel<<<g.nmat, 1024, sizeof(unsigned long long) * npow2, st>>>(g, npow2);
    } else if (stage == 1) {                            // column signs of Q
        fix_signs_group_kernel<<<dim3((kmax + 7) / 8, g.nmat), 256, 0, st>>>(g);
    } else if (stage == 2) {                            // Householder top block
        hh_top_group_kernel<<<g.nmat, 1024, 0, st>>>(g);
    } else {                                            // Householder rows below
        if (rows_max <= 0) return cudaSuccess;
        hh_rows_group_kernel<<<dim3((rows_max + 7) / 8, g.nmat), 256, 0, st>>>(g);
    }
    return cudaGetLastError();
}

namespace {
// Packed lower triangle: element (i, l), l <= i, at i (i + 1) / 2 + l.
__device__ __forceinline__ int tri(int i, int l) { return i * (i + 1) / 2 + l; }

// S = L^{-T} with L L^T = G (n x n symmetric positive definite, n <= 256): one CTA, the packed lower
// triangle in shared memory.  Right-looking Cholesky (a warp per row of the trailing update, lanes
// along the row); if a pivot is not positive a diagonal shift (1e-7, then x100, times the mean
// diagonal) is added and the factorisation restarts, at most six attempts, the attempts counted
// in *flag.  Then L^{-1} in place, column by column from the last: for j = n-1..0 the entries
// below the diagonal of column j are -(L^{-1}[i, j+1..i] . L[j+1..i, j]) / L_jj.  Each step first
// copies the column it reads into a contiguous array (a column of the packed triangle is strided
// by the row lengths, which would make the lanes' reads collide in the banks).  S (row-major
// n x n) is the transpose of L^{-1}.
// The Gram matrix is the sum of `nparts` partial matrices (leading dimension ld, spaced ld * ld
// apart).  Output: S = L^{-T} (row-major n x n), or with out_linv L^{-1} (row-major ld x ld, zero
// above the diagonal and outside n x n).
__device__ __forceinline__ void chol_inverse_body(const float* G, int nparts, int ld, int n, float* S, int out_linv,
                                                  int* flag) {
    extern __shared__ float L[];                       // n (n + 1) / 2 packed, then n + n temporaries
    float* col = L + n * (n + 1) / 2;
    float* tmp = col + n;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nw = blockDim.x >> 5;
    __shared__ int fail;
    __shared__ float shift, trace;
    if (warp == 0) {                                   // trace: a warp sum in a fixed order
        float tr = 0.f;
        for (int i = lane; i < n; i += 32) {
            float gi = 0.f;
            for (int p = 0; p < nparts; ++p) gi += G[(size_t)p * ld * ld + (size_t)i * ld + i];
            tr += gi;
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) tr += __shfl_xor_sync(0xffffffffu, tr, o);
        if (lane == 0) { trace = tr; shift = 0.f; }
    }
    __syncthreads();
    int attempt = 0;
    for (; attempt < 6; ++attempt) {
        for (int i = warp; i < n; i += nw)
            for (int l = lane; l <= i; l += 32) {
                float gil = 0.f;
                for (int p = 0; p < nparts; ++p) gil += G[(size_t)p * ld * ld + (size_t)i * ld + l];
                L[tri(i, l)] = gil + (l == i ? shift : 0.f);
            }
        if (tid == 0) fail = 0;
        __syncthreads();
        const float thresh = 1e-12f * fmaxf(trace / n, 1e-30f);
        for (int j = 0; j < n; ++j) {
            const float d = L[tri(j, j)];
            if (!(d > thresh)) { fail = 1; break; }      // uniform: every thread reads the same d
            const float ljj = sqrtf(d);
            __syncthreads();
            if (tid == 0) L[tri(j, j)] = ljj;
            for (int i = j + 1 + tid; i < n; i += blockDim.x) {
                const float v = L[tri(i, j)] / ljj;
                L[tri(i, j)] = v;
                col[i] = v;
            }
            __syncthreads();
            for (int i = j + 1 + warp; i < n; i += nw) {
                const float lij = col[i];
                for (int l = j + 1 + lane; l <= i; l += 32) L[tri(i, l)] -= lij * col[l];
            }
            __syncthreads();
        }
        __syncthreads();
        if (!fail) break;
        if (tid == 0) shift = (attempt == 0 ? 1e-7f : shift * 100.f) * fmaxf(trace / n, 1e-30f);
        __syncthreads();
    }
    if (tid == 0 && flag) {
        *flag = attempt;
        // no factorisation after every shift, or a Gram matrix with no positive trace (a zero or
        // non-finite block): the refresh cannot orthonormalise it (flag + 6 counts these)
        if (attempt == 6 || !(trace > 0.f) || !isfinite(trace)) atomicAdd(flag + 6, 1);
    }
    for (int j = n - 1; j >= 0; --j) {
        for (int l = j + 1 + tid; l < n; l += blockDim.x) col[l] = L[tri(l, j)];
        __syncthreads();
        for (int i = j + 1 + warp; i < n; i += nw) {
            float t = 0.f;
            for (int l = j + 1 + lane; l <= i; l += 32) t += L[tri(i, l)] * col[l];
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
            if (lane == 0) tmp[i] = t;
        }
        __syncthreads();
        const float ajj = 1.0f / L[tri(j, j)];
        for (int i = j + 1 + tid; i < n; i += blockDim.x) L[tri(i, j)] = -tmp[i] * ajj;
        if (tid == 0) L[tri(j, j)] = ajj;
        __syncthreads();
    }
    if (out_linv) {
        for (int e = tid; e < ld * ld; e += blockDim.x) {
            const int r = e / ld, c = e % ld;
            S[e] = (c <= r && r < n) ? L[tri(r, c)] : 0.f;
        }
        return;
    }
    for (int e = tid; e < n * n; e += blockDim.x) {
        const int r = e / n, c = e % n;
        S[e] = c >= r ? L[tri(c, r)] : 0.f;
    }
}

__global__ void __launch_bounds__(1024) chol_inverse_kernel(const float* G, int n, float* S, int* flag) {
    chol_inverse_body(G, 1, n, n, S, 0, flag);
}
// L^{-1} of the lower-triangular L = U^T, U the upper triangle of the n x n matrix at A (leading
// dimension lda): the inverse stage of chol_inverse_body alone.  Output row-major ld x ld.
__device__ __forceinline__ void tri_inverse_body(const float* A, int lda, int n, float* out, int ld) {
    extern __shared__ float L[];
    float* col = L + n * (n + 1) / 2;
    float* tmp = col + n;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nw = blockDim.x >> 5;
    for (int i = warp; i < n; i += nw)
        for (int l = lane; l <= i; l += 32) L[tri(i, l)] = A[(size_t)l * lda + i];
    __syncthreads();
    for (int j = n - 1; j >= 0; --j) {
        for (int l = j + 1 + tid; l < n; l += blockDim.x) col[l] = L[tri(l, j)];
        __syncthreads();
        for (int i = j + 1 + warp; i < n; i += nw) {
            float t = 0.f;
            for (int l = j + 1 + lane; l <= i; l += 32) t += L[tri(i, l)] * col[l];
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
            if (lane == 0) tmp[i] = t;
        }
        __syncthreads();
        const float ajj = 1.0f / L[tri(j, j)];
        for (int i = j + 1 + tid; i < n; i += blockDim.x) L[tri(i, j)] = -tmp[i] * ajj;
        if (tid == 0) L[tri(j, j)] = ajj;
        __syncthreads();
    }
    for (int e = tid; e < ld * ld; e += blockDim.x) {
        const int r = e / ld, c = e % ld;
        out[e] = (c <= r && r < n) ? L[tri(r, c)] : 0.f;
    }
}

__global__ void __launch_bounds__(1024) chol_group_kernel(const __grid_constant__ CholGroup g) {
    const CholMat& M = g.mat[blockIdx.x];
    if (M.tri_only) tri_inverse_body(M.part, M.n, M.n, M.out, M.ld);
    else chol_inverse_body(M.part, M.nparts, M.ld, M.n, M.out, 1, M.flag);
}
}  // namespace

cudaError_t chol_group(const CholGroup& g, cudaStream_t st) {
    if (g.nmat <= 0) return cudaSuccess;
    int nmax = 0;
    for (int i = 0; i < g.nmat; ++i) {
        if (g.mat[i].n < 1 || g.mat[i].n > 256 || g.mat[i].ld < g.mat[i].n) return cudaErrorInvalidValue;
        nmax = g.mat[i].n > nmax ? g.mat[i].n : nmax;
    }
    const size_t smem = sizeof(float) * ((size_t)nmax * (nmax + 1) / 2 + 2 * nmax);
    {   // per device: set on every call (cheap next to the launch)
        const cudaError_t ea = cudaFuncSetAttribute(chol_group_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                   (int)(sizeof(float) * (256 * 257 / 2 + 2 * 256)));
        if (ea != cudaSuccess) return ea;
    }
    chol_group_kernel<<<g.nmat, 1024, smem, st>>>(g);
    return cudaGetLastError();
}

cudaError_t chol_inverse(const float* G, int n, float* S, int* flag, cudaStream_t st) {
    if (n < 1 || n > 256) return cudaErrorInvalidValue;
    const size_t smem = sizeof(float) * ((size_t)n * (n + 1) / 2 + 2 * n);
    // the largest factor (n = 256) and its temporaries, below the per-CTA limit with the
    // kernel's few static bytes
    {   // per device: set on every call (cheap next to the launch)
        const cudaError_t ea = cudaFuncSetAttribute(chol_inverse_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                   (int)(sizeof(float) * (256 * 257 / 2 + 2 * 256)));
        if (ea != cudaSuccess) return ea;
    }
    chol_inverse_kernel<<<1, 1024, smem, st>>>(G, n, S, flag);
    return cudaGetLastError();
}

cudaError_t cholesky(float* A, int n, float* scratch, int* flag, cudaStream_t st) {
    cholesky_kernel<<<1, 1024, 0, st>>>(A, n, scratch, flag);
    return cudaGetLastError();
}

cudaError_t trsm_right_lt(float* Q, int rows, int n, const float* L, cudaStream_t st) {
    trsm_kernel<<<(rows + 7) / 8, 256, 0, st>>>(Q, rows, n, L);
    return cudaGetLastError();
}

cudaError_t random_block(float* Q, int rows, int cols, uint64_t seed, uint32_t t, cudaStream_t st) {
    const int64_t total = (int64_t)rows * ((cols + 3) / 4);
    random_block_kernel<<<(unsigned)((total + 255) / 256), 256, 0, st>>>(Q, rows, cols, seed, t);
    return cudaGetLastError();
}

cudaError_t householder_reconstruct(const float* Q, int mp, int k, float* Y, float* T, float* s,
                                    float* scratch, cudaStream_t st) {
    hh_top_kernel<<<1, 1024, 0, st>>>(Q, k, scratch, Y, T, s);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    if (mp > k) hh_rows_kernel<<<(mp - k + 7) / 8, 256, 0, st>>>(Q, mp, k, scratch, Y);
    return cudaGetLastError();
}

cudaError_t materialize_wy_basis(int mp, int k, const float* Y, const float* Yt, const float* dsign,
                                 float* U, cudaStream_t st) {
    const int64_t total = (int64_t)mp * mp;
    wy_basis_kernel<<<(unsigned)((total + 255) / 256), 256, 0, st>>>(mp, k, Y, Yt, dsign, U);
    return cudaGetLastError();
}

}  // namespace glr
