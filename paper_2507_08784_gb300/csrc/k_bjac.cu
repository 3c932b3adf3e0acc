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
//   2. applies the block-diagonal J = diag(J_k) on the tensor cores (tc_kernel<BjacMul>, k_tc.cu,
//      split TF32: A B + A_lo B + A B_lo): T^T = (H J)^T, then H <- T^T J = J^T H J (H symmetric)
//      and V <- V J, the last two writing every 64-block straight to its place in the next
//      round's storage order;
// and a sweep ends with the off-diagonal norm, checked on the host against tol^2 of the total.
// V starts as the identity, so its columns follow H's storage order; at the end diag(H) and V
// are sorted by descending eigenvalue with the sign rule of the small solvers (sort_fix_basis).
//
// Every product keeps its output's TF32 low part beside it (H_lo, T^T_lo, V_lo; J_lo from the
// pair sweep), so each operand enters the MMAs as hi + lo.
#include "glr_internal.cuh"

namespace glr {

namespace {

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
// columns; J_k^T is written row-major with its TF32 low part.  PT = 512 threads with two CTAs per
// SM when a launch has more pairs than SMs, else PT = 1024 (half the work per thread and round:
// each update's arithmetic is the same, so the results are too).
constexpr int PN = 128, PH = 64, PLD = 129;
constexpr int kPairItems = PH * (PH + 1) / 2;                 // 2 x 2 blocks (bi <= bj) of a round
constexpr size_t kPairSmem = sizeof(float) * (PN * (PN + 1) / 2 + PN * PLD);

__device__ __forceinline__ int pcircle(int x) { return 1 + ((x % (PN - 1)) + (PN - 1)) % (PN - 1); }

template <int PT>
__global__ void __launch_bounds__(PT, 1024 / PT) bjac_pair_kernel(const __grid_constant__ BjacGroup g) {
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
    // J_k^T (row c = column c of W) and its TF32 low part: the rotations' MMA operands
    float* Jt = M.J + (int64_t)k * PN * PN;
    float* Jl = M.Jlo + (int64_t)k * PN * PN;
    for (int e = t; e < PN * PN; e += PT) {
        const float v = Ws[(e & 127) * PLD + (e >> 7)];
        Jt[e] = v;
        Jl[e] = v - __uint_as_float(__float_as_uint(v) & 0xffffe000u);
    }
}

// Before the first round, per problem: H = the sum of nparts partial matrices (leading dimension
// ld; none when H is already formed), H's TF32 low part, V = I and V's low part 0.
__global__ void bjac_prep_kernel(const __grid_constant__ BjacPrepGroup g) {
    const BjacPrep& P = g.mat[blockIdx.y];
    const int n = P.n;
    for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < (int64_t)n * n; q += (int64_t)gridDim.x * blockDim.x) {
        const int r = (int)(q / n), c = (int)(q % n);
        float h;
        if (P.nparts > 0) {
            h = 0.f;
            for (int p = 0; p < P.nparts; ++p) h += P.part[(int64_t)p * P.ld * P.ld + (int64_t)r * P.ld + c];
            P.H[q] = h;
        } else {
            h = P.H[q];
        }
        P.Hlo[q] = h - __uint_as_float(__float_as_uint(h) & 0xffffe000u);
        P.V[q] = r == c ? 1.f : 0.f;
        P.Vlo[q] = 0.f;
    }
}

__global__ void count_flag_kernel(int* flag, int v) { atomicAdd(flag, v); }

__global__ void bjac_eye_kernel(float* V, int n) {
    for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < (int64_t)n * n; q += (int64_t)gridDim.x * blockDim.x)
        V[q] = (q / n == q % n) ? 1.f : 0.f;
}
__global__ void bjac_diag_kernel(const float* H, int n, float* evals) {
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) evals[i] = H[(int64_t)i * n + i];
}


}  // namespace

cudaError_t bjac_pairs(BjacGroup& g, cudaStream_t st) {
    if (g.nmat <= 0) return cudaSuccess;
    int tiles = 0;
    for (int i = 0; i < g.nmat; ++i) {
        BjacMat& M = g.mat[i];
        if (M.n < 256 || M.n % 128 || M.n > kBjacMaxN) return cudaErrorInvalidValue;
        M.tile0p = tiles;
        tiles += M.n / 128;
    }
    static int sms = 0;
    if (!sms) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    }
    if (tiles <= sms) {
        cudaError_t e = cudaFuncSetAttribute(bjac_pair_kernel<1024>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kPairSmem);
        if (e != cudaSuccess) return e;
        bjac_pair_kernel<1024><<<tiles, 1024, kPairSmem, st>>>(g);
    } else {
        cudaError_t e = cudaFuncSetAttribute(bjac_pair_kernel<512>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kPairSmem);
        if (e != cudaSuccess) return e;
        bjac_pair_kernel<512><<<tiles, 512, kPairSmem, st>>>(g);
    }
    return cudaGetLastError();
}

cudaError_t bjac_norms(const BjacGroup& g, float* part, cudaStream_t st) {
    if (g.nmat <= 0) return cudaSuccess;
    bjac_norms_kernel<<<dim3(kBjacNormCtas, g.nmat), 256, 0, st>>>(g, part);
    return cudaGetLastError();
}

cudaError_t bjac_prep(const BjacPrepGroup& g, cudaStream_t st) {
    if (g.nmat <= 0) return cudaSuccess;
    bjac_prep_kernel<<<dim3(64, g.nmat), 256, 0, st>>>(g);
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
