// The k x k Rayleigh-Ritz eigenproblems of a truncated refresh (Eq. SVD-P1 read as the top-k
// subspace of Mbar, see glr_refresh_host.cu): H = Q^T Mbar Mbar^T Q = W diag(lambda) W^T for every
// refreshing matrix, one CTA per matrix, all matrices in one launch.
//
// Parallel cyclic two-sided Jacobi (rotation formula: Golub & Van Loan, sym.schur2; circle
// ordering of the pairs): a round forms the n/2 rotations of disjoint index pairs from their own
// 2 x 2 diagonal blocks, then applies H <- J^T H J and W <- W J.  With the rotations fixed for the
// round, each 2 x 2 block of H (rows of pair i, columns of pair j) depends only on its own old
// entries and the two rotations, so the update is in place and needs one barrier.
//
// Storage: the upper triangle of H, packed by rows, in shared memory (n = 256: 129 KiB); W in
// tensor memory (128 lanes x 512 columns of 32 bits: row a of W in lane a mod 128, column
// (a / 128) n + j), read and written by tcgen05.ld / tcgen05.st from the warps of each lane
// quadrant.  A CTA of 1024 threads: the block updates of a round take half (half + 1) / 2
// 2 x 2 blocks, enumerated by folding block row i with block row half - 1 - i so that every
// thread has the same count.  A matrix stops at the start of the first sweep whose off-diagonal
// squared norm is within tol^2 of the total, or after max_sweeps sweeps.
#include "glr_internal.cuh"

namespace glr {

namespace {

constexpr int ET = 1024;
constexpr int kEigMaxN = 256;

__device__ __forceinline__ int circle(int x, int nm1) { return 1 + ((x % nm1) + nm1) % nm1; }

__device__ __forceinline__ void tm_st1(uint32_t ta, float a) {
    asm volatile("tcgen05.st.sync.aligned.32x32b.x1.b32 [%0], {%1};" ::"r"(ta), "r"(__float_as_uint(a)) : "memory");
}
__device__ __forceinline__ void tm_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void tm_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tm_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

__global__ void __launch_bounds__(ET, 1) eig_tmem_kernel(const __grid_constant__ EigGroup g) {
    extern __shared__ float Hs[];                      // packed upper triangle, n (n + 1) / 2
    __shared__ int off[kEigMaxN + 1];                  // Hs index of (r, c), r <= c: off[r] + c
    __shared__ int4 spq[kEigMaxN / 2];                 // the round's pairs: p, q, off[p], off[q] (q = n: no partner)
    __shared__ float2 scs[kEigMaxN / 2];               // and their rotations (c, s)
    __shared__ float red[2][ET / 32];
    __shared__ uint32_t tbase;
    __shared__ int s_stop;
    const EigMat& M = g.mat[blockIdx.x];
    const int n = M.n, t = threadIdx.x, warp = t >> 5, lane = t & 31;
    const int npad = n + (n & 1), half = npad / 2, nm1 = npad - 1;
    const int halves = (n + 127) / 128;
    uint32_t cols = 32;
    while (cols < (uint32_t)(halves * n)) cols <<= 1;
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                     ::"r"(static_cast<uint32_t>(__cvta_generic_to_shared(&tbase))), "r"(cols));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
        tm_fence_before();
    }
    for (int r = t; r <= n; r += ET) off[r] = r * n - r * (r + 1) / 2;
    __syncthreads();
    for (int r = warp; r < n; r += ET / 32)            // H (row-major n x n) -> packed upper triangle
        for (int c = r + lane; c < n; c += 32) {
            float v = 0.f;
            for (int p = 0; p < M.nparts; ++p) v += M.H[(size_t)p * M.ld * M.ld + (size_t)r * M.ld + c];
            Hs[off[r] + c] = v;
        }
    tm_fence_after();
    const uint32_t tmem = tbase;
    // this warp's lane quadrant: W rows a = h 128 + 32 qd + lane of every half h
    const int qd = warp & 3, w8 = warp >> 2;
    const uint32_t lanes = static_cast<uint32_t>(32 * qd) << 16;
    for (int h = 0; h < halves; ++h) {                 // W = I
        const int a = h * 128 + 32 * qd + lane;
        for (int j = w8; j < n; j += 8) tm_st1(tmem + lanes + (uint32_t)(h * n + j), a == j ? 1.f : 0.f);
    }
    tm_wait_st();
    __syncthreads();
    const int items = half * (half + 1) / 2;
    // this thread's 2 x 2 blocks (bi <= bj) of every round: block row i folded with block row
    // half - 1 - i so that the enumeration has rows of half + 1 entries
    constexpr int kItems = (kEigMaxN / 2) * (kEigMaxN / 2 + 1) / 2 / ET + 1;
    int myblk[kItems];
#pragma unroll
    for (int u = 0; u < kItems; ++u) {
        const int e = t + u * ET;
        myblk[u] = -1;
        if (e < items) {
            const int fr = e / (half + 1), tt = e - fr * (half + 1);
            int bi, bj;
            if (tt < half - fr) { bi = fr; bj = fr + tt; }
            else { bi = half - 1 - fr; bj = bi + (tt - (half - fr)); }
            myblk[u] = bi | (bj << 16);
        }
    }
    int sweep = 0;
    for (;;) {
        // convergence check at the start of a sweep
        float o = 0.f, d = 0.f;
        for (int r = warp; r < n; r += ET / 32) {
            for (int c = r + lane; c < n; c += 32) {
                const float v = Hs[off[r] + c];
                if (c == r) d += v * v; else o += v * v;
            }
        }
#pragma unroll
        for (int m = 16; m > 0; m >>= 1) {
            o += __shfl_xor_sync(0xffffffffu, o, m);
            d += __shfl_xor_sync(0xffffffffu, d, m);
        }
        if (lane == 0) { red[0][warp] = o; red[1][warp] = d; }
        __syncthreads();
        if (t == 0) {
            float o2 = 0.f, d2 = 0.f;
            for (int w = 0; w < ET / 32; ++w) { o2 += red[0][w]; d2 += red[1][w]; }
            o2 *= 2.f;                                   // each off-diagonal entry stands for two
            s_stop = (o2 <= M.tol * M.tol * (o2 + d2) || sweep >= g.max_sweeps) ? 1 : 0;
        }
        __syncthreads();
        if (s_stop) break;
        for (int rd = 0; rd < nm1; ++rd) {
            if (t < half) {                             // the round's rotations
                int p = (t == 0) ? 0 : circle(rd + t, nm1);
                int q = (t == 0) ? circle(rd, nm1) : circle(rd - t, nm1);
                if (p > q) { const int tmp = p; p = q; q = tmp; }
                float c = 1.f, s = 0.f;
                if (q < n) {
                    const float hpq = Hs[off[p] + q], hpp = Hs[off[p] + p], hqq = Hs[off[q] + q];
                    if (fabsf(hpq) > 1e-30f && fabsf(hpq) > 1e-9f * sqrtf(fabsf(hpp * hqq))) {
                        const float theta = (hqq - hpp) / (2.f * hpq);
                        float tt;
                        if (fabsf(theta) > 1e15f) tt = 0.5f / theta;
                        else tt = copysignf(1.f, theta) / (fabsf(theta) + sqrtf(theta * theta + 1.f));
                        c = 1.f / sqrtf(tt * tt + 1.f);
                        s = tt * c;
                    }
                }
                spq[t] = make_int4(p, q, off[p], q < n ? off[q] : 0);
                scs[t] = make_float2(c, s);
            }
            __syncthreads();
#pragma unroll
            for (int u = 0; u < kItems; ++u) {          // H <- J^T H J, 2 x 2 block by block (bi <= bj)
                if (myblk[u] < 0) continue;
                const int bi = myblk[u] & 0xFFFF, bj = myblk[u] >> 16;
                const float2 rci = scs[bi], rcj = scs[bj];
                const float ci = rci.x, si = rci.y, cj = rcj.x, sj = rcj.y;
                if (si == 0.f && sj == 0.f) continue;
                const int4 pi4 = spq[bi], pj4 = spq[bj];
                const int pi = pi4.x, qi = pi4.y, pj = pj4.x, qj = pj4.y;
                const bool vqi = qi < n, vqj = qj < n;
                if (bi == bj) {                          // diagonal block: the annihilated pair
                    const int i00 = pi4.z + pi, i01 = pi4.z + qi, i11 = pi4.w + qi;
                    const float h00 = Hs[i00], h01 = Hs[i01], h11 = Hs[i11];
                    const float a00 = ci * h00 - si * h01, a01 = ci * h01 - si * h11;
                    const float a10 = si * h00 + ci * h01, a11 = si * h01 + ci * h11;
                    Hs[i00] = cj * a00 - sj * a01;
                    Hs[i11] = sj * a10 + cj * a11;
                    Hs[i01] = 0.f;
                    continue;
                }
                // (x, y) of the symmetric matrix at the packed index of (min, max): offx + y or offy + x
                // (an index with no partner points at (pi, pj): it is neither read nor written)
                const int i00 = pi <= pj ? pi4.z + pj : pj4.z + pi;
                const int i01 = !vqj ? i00 : pi <= qj ? pi4.z + qj : pj4.w + pi;
                const int i10 = !vqi ? i00 : qi <= pj ? pi4.w + pj : pj4.z + qi;
                const int i11 = !(vqi && vqj) ? i00 : qi <= qj ? pi4.w + qj : pj4.w + qi;
                const float h00 = Hs[i00];
                const float h01 = vqj ? Hs[i01] : 0.f;
                const float h10 = vqi ? Hs[i10] : 0.f;
                const float h11 = (vqi && vqj) ? Hs[i11] : 0.f;
                const float a00 = ci * h00 - si * h10, a01 = ci * h01 - si * h11;
                const float a10 = si * h00 + ci * h10, a11 = si * h01 + ci * h11;
                Hs[i00] = cj * a00 - sj * a01;
                if (vqj) Hs[i01] = sj * a00 + cj * a01;
                if (vqi) Hs[i10] = cj * a10 - sj * a11;
                if (vqi && vqj) Hs[i11] = sj * a10 + cj * a11;
            }
            // W <- W J: the warps of each lane quadrant share the (pair, half) items, eight at a
            // time with all sixteen column loads in flight before one wait
            for (int h = 0; h < halves; ++h) {
                const uint32_t hb = tmem + lanes + (uint32_t)(h * n);
                for (int j0 = w8; j0 < half; j0 += 64) {
                    uint32_t ap[8], aq[8], up[8], uq[8];
                    bool act[8];
#pragma unroll
                    for (int b = 0; b < 8; ++b) {
                        const int j = j0 + 8 * b;
                        act[b] = j < half && scs[j].y != 0.f;   // warp-uniform
                        const int4 pq = spq[j < half ? j : 0];
                        ap[b] = hb + (uint32_t)pq.x;
                        aq[b] = hb + (uint32_t)pq.y;
                        if (act[b]) {
                            asm volatile("tcgen05.ld.sync.aligned.32x32b.x1.b32 {%0}, [%1];" : "=r"(up[b]) : "r"(ap[b]));
                            asm volatile("tcgen05.ld.sync.aligned.32x32b.x1.b32 {%0}, [%1];" : "=r"(uq[b]) : "r"(aq[b]));
                        }
                    }
                    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
                    for (int b = 0; b < 8; ++b) {
                        if (!act[b]) continue;
                        const float2 cs = scs[j0 + 8 * b];
                        const float vp = __uint_as_float(up[b]), vq = __uint_as_float(uq[b]);
                        tm_st1(ap[b], cs.x * vp - cs.y * vq);
                        tm_st1(aq[b], cs.y * vp + cs.x * vq);
                    }
                }
            }
            tm_wait_st();
            tm_fence_before();
            __syncthreads();                            // the rotations are rewritten next round
            tm_fence_after();
        }
        ++sweep;
    }
    // eigenvalues (diagonal), W to global memory (row-major n x n), sweeps
    for (int i = t; i < n; i += ET) M.evals[i] = Hs[off[i] + i];
    if (t == 0 && M.sweeps) *M.sweeps = sweep;
    for (int h = 0; h < halves; ++h) {
        const int a = h * 128 + 32 * qd + lane;
        for (int j = w8; j < n; j += 8) {
            uint32_t u;
            asm volatile("tcgen05.ld.sync.aligned.32x32b.x1.b32 {%0}, [%1];" : "=r"(u) : "r"(tmem + lanes + (uint32_t)(h * n + j)));
            asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
            if (a < n) M.V[(size_t)a * n + j] = __uint_as_float(u);
        }
    }
    tm_fence_before();
    __syncthreads();
    if (warp == 0) {
        tm_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(cols));
    }
}

}  // namespace

cudaError_t eig_tmem_group(const EigGroup& g, cudaStream_t st) {
    if (g.nmat <= 0) return cudaSuccess;
    int nmax = 0;
    for (int i = 0; i < g.nmat; ++i) {
        if (g.mat[i].n < 2 || g.mat[i].n > kEigMaxN || g.mat[i].ld < g.mat[i].n || g.mat[i].nparts < 1)
            return cudaErrorInvalidValue;
        nmax = g.mat[i].n > nmax ? g.mat[i].n : nmax;
    }
    const size_t smem = sizeof(float) * (size_t)nmax * (nmax + 1) / 2;
    {   // per device: set on every call (cheap next to the launch)
        const cudaError_t ea = cudaFuncSetAttribute(eig_tmem_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                   (int)(sizeof(float) * kEigMaxN * (kEigMaxN + 1) / 2));
        if (ea != cudaSuccess) return ea;
    }
    eig_tmem_kernel<<<g.nmat, ET, smem, st>>>(g);
    return cudaGetLastError();
}

}  // namespace glr
