// Full-basis refresh (Eq. SVD-P1, the paper-exact basis): the eigen-decomposition of the m' x m'
// Gram matrices H = Mbar Mbar^T of every refreshing matrix by parallel cyclic two-sided Jacobi,
// all matrices in one cooperative launch.  A round applies n/2 disjoint plane rotations chosen by
// the circle (round-robin) ordering — each angle from its own 2 x 2 diagonal block (Golub & Van
// Loan, sym.schur2) — then H <- J^T H J block-wise (each 2 x 2 block of H depends only on the
// rotations of its row and column pairs) and V <- V J.  The updates of a round are spread over
// every CTA of the grid, rounds separated by grid-wide barriers; a matrix stops at the start of
// the first sweep whose off-diagonal norm is within tol of the total.
//
// The grid barrier is an arrival counter and a generation word in global memory; a waiting CTA
// polls with short sleeps and gives up after about a second, counts the event in *err and
// returns, so a stuck barrier ends the kernel instead of hanging it.  The cooperative launch
// keeps every CTA resident, which is what makes the barrier safe to wait on.  Data written by one
// CTA and read by another (H, V, the norm partials) is read through L2 (__ldcg), so no stale L1
// line survives a barrier.
#include "glr_internal.cuh"

namespace glr {

namespace {

constexpr int JT = 256;                 // threads per CTA

__device__ __forceinline__ int circle(int x, int nm1) { return 1 + ((x % nm1) + nm1) % nm1; }

// All CTAs arrive; false when the wait timed out.  *count returns to 0 after every barrier.
__device__ bool grid_barrier(int* count, int* genp, int& gen) {
    __shared__ int s_ok;
    __syncthreads();
    if (threadIdx.x == 0) {
        int ok = 1;
        const int target = gen + 1;
        __threadfence();
        if (atomicAdd(count, 1) == static_cast<int>(gridDim.x) - 1) {
            atomicExch(count, 0);
            __threadfence();
            atomicExch(genp, target);
        } else {
            for (int spin = 0; *reinterpret_cast<volatile int*>(genp) != target; ++spin) {
                if (spin > 20000000) { ok = 0; break; }          // about a second of 32-64 ns sleeps
                __nanosleep(32);
            }
        }
        __threadfence();
        gen = target;
        s_ok = ok;
    }
    __syncthreads();
    return s_ok != 0;
}

// Each matrix runs its own sequence — a norm check, then its own n' - 1 rounds (n' = n rounded up
// to even), then the next check, ... — one stage per grid step, so what a matrix computes does not
// depend on the matrices it is grouped with.  In a round every CTA forms all of the round's
// rotations itself (from the current H, in shared memory) and applies its share of the 2 x 2
// block updates from the current H into the other H buffer (every block is written, rotated or
// not), so no CTA can see a diagonal block another CTA has already updated; V is updated in place
// (each entry by one thread).  A check's partial norms are written in one step and decided on at
// the start of the next, identically by every CTA.  One grid barrier per step.
enum : int { kCheck = 0, kRound = 1, kPending = 2, kDone = 3 };

__global__ void __launch_bounds__(JT) jacobi_group_kernel(const __grid_constant__ JacobiGroup g) {
    const int G = gridDim.x, b = blockIdx.x, t = threadIdx.x;
    const int64_t gtid = (int64_t)b * JT + t, gsz = (int64_t)G * JT;
    __shared__ int sstate[kGroupMax], sround[kGroupMax], ssweep[kGroupMax], sflip[kGroupMax];
    __shared__ float red[2][JT / 32];
    extern __shared__ float srot[];                     // per matrix at M.soff: cs, sn, pp, qq (half each)
    int gen = 0;
    bool ok = true;
    for (int mi = 0; mi < g.nmat; ++mi) {
        const JacobiMat& M = g.mat[mi];
        const int64_t nn = (int64_t)M.n * M.n;
        for (int64_t e = gtid; e < nn; e += gsz) M.V[e] = (e / M.n == e % M.n) ? 1.f : 0.f;
    }
    if (t < g.nmat) { sstate[t] = kCheck; sround[t] = 0; ssweep[t] = 0; sflip[t] = 0; }
    ok = grid_barrier(g.bar, g.bar + 1, gen);
    while (ok) {
        if (t < g.nmat && sstate[t] == kPending) {      // decide on last step's partials
            const JacobiMat& M = g.mat[t];
            float o2 = 0.f, t2 = 0.f;
            for (int c = 0; c < G; ++c) { o2 += __ldcg(g.part + (2 * t) * G + c); t2 += __ldcg(g.part + (2 * t + 1) * G + c); }
            if (o2 <= M.tol * M.tol * t2 || ssweep[t] >= g.max_sweeps) {
                sstate[t] = kDone;
                if (b == 0 && M.sweeps) *M.sweeps = ssweep[t];
            } else {
                sstate[t] = kRound;
                sround[t] = 0;
            }
        }
        __syncthreads();
        bool any = false;
        for (int mi = 0; mi < g.nmat; ++mi) any = any || sstate[mi] != kDone;
        if (!any) break;
        // norm checks, and every round's rotations (each matrix in its own shared slice)
        for (int mi = 0; mi < g.nmat; ++mi) {
            const JacobiMat& M = g.mat[mi];
            const int n = M.n;
            const float* Hc = sflip[mi] ? M.H2 : M.H;
            if (sstate[mi] == kCheck) {                 // off-diagonal and total squared norms, per CTA
                const int64_t nn = (int64_t)n * n;
                float off = 0.f, tot = 0.f;
                for (int64_t e = gtid; e < nn; e += gsz) {
                    const float h = __ldcg(Hc + e);
                    tot += h * h;
                    if (e / n != e % n) off += h * h;
                }
                for (int o = 16; o > 0; o >>= 1) {
                    off += __shfl_xor_sync(0xffffffffu, off, o);
                    tot += __shfl_xor_sync(0xffffffffu, tot, o);
                }
                if ((t & 31) == 0) { red[0][t >> 5] = off; red[1][t >> 5] = tot; }
                __syncthreads();
                if (t == 0) {
                    float o2 = 0.f, t2 = 0.f;
                    for (int w = 0; w < JT / 32; ++w) { o2 += red[0][w]; t2 += red[1][w]; }
                    g.part[(2 * mi) * G + b] = o2;
                    g.part[(2 * mi + 1) * G + b] = t2;
                }
                __syncthreads();
                continue;
            }
            if (sstate[mi] != kRound) continue;
            const int npad = n + (n & 1), half = npad / 2, nm1 = npad - 1, r = sround[mi];
            float* scs = srot + M.soff;
            float* ssn = scs + half;
            int* spp = reinterpret_cast<int*>(ssn + half);
            int* sqq = spp + half;
            for (int i = t; i < half; i += JT) {        // all of the round's rotations, in this CTA
                int p = (i == 0) ? 0 : circle(r + i, nm1);
                int q = (i == 0) ? circle(r, nm1) : circle(r - i, nm1);
                if (p > q) { const int tmp = p; p = q; q = tmp; }
                float c = 1.f, s = 0.f;
                if (q < n) {
                    const float hpq = __ldcg(Hc + (size_t)p * n + q);
                    const float hpp = __ldcg(Hc + (size_t)p * n + p), hqq = __ldcg(Hc + (size_t)q * n + q);
                    if (fabsf(hpq) > 1e-30f && fabsf(hpq) > 1e-9f * sqrtf(fabsf(hpp * hqq))) {
                        const float theta = (hqq - hpp) / (2.f * hpq);
                        float tt;
                        if (fabsf(theta) > 1e15f) tt = 0.5f / theta;
                        else tt = copysignf(1.f, theta) / (fabsf(theta) + sqrtf(theta * theta + 1.f));
                        c = 1.f / sqrtf(tt * tt + 1.f);
                        s = tt * c;
                    }
                }
                scs[i] = c; ssn[i] = s; spp[i] = p; sqq[i] = q;
            }
        }
        __syncthreads();
        // every round's updates
        for (int mi = 0; mi < g.nmat; ++mi) {
            if (sstate[mi] != kRound) continue;
            const JacobiMat& M = g.mat[mi];
            const int n = M.n, half = (n + (n & 1)) / 2;
            const float* Hc = sflip[mi] ? M.H2 : M.H;
            float* Hn = sflip[mi] ? M.H : M.H2;
            const float* scs = srot + M.soff;
            const float* ssn = scs + half;
            const int* spp = reinterpret_cast<const int*>(ssn + half);
            const int* sqq = spp + half;
            const int64_t hh = (int64_t)half * half;
            for (int64_t e = gtid; e < hh; e += gsz) {   // Hn = J^T Hc J, 2 x 2 block by block
                const int bi = static_cast<int>(e / half), bj = static_cast<int>(e % half);
                const float si = ssn[bi], sj = ssn[bj], ci = scs[bi], cj = scs[bj];
                const int pi = spp[bi], qi = sqq[bi], pj = spp[bj], qj = sqq[bj];
                const bool vqi = qi < n, vqj = qj < n;
                const float h00 = __ldcg(Hc + (size_t)pi * n + pj);
                const float h01 = vqj ? __ldcg(Hc + (size_t)pi * n + qj) : 0.f;
                const float h10 = vqi ? __ldcg(Hc + (size_t)qi * n + pj) : 0.f;
                const float h11 = (vqi && vqj) ? __ldcg(Hc + (size_t)qi * n + qj) : 0.f;
                float n00 = h00, n01 = h01, n10 = h10, n11 = h11;
                if (si != 0.f || sj != 0.f) {
                    const float a00 = ci * h00 - si * h10, a01 = ci * h01 - si * h11;
                    const float a10 = si * h00 + ci * h10, a11 = si * h01 + ci * h11;
                    n00 = cj * a00 - sj * a01; n01 = sj * a00 + cj * a01;
                    n10 = cj * a10 - sj * a11; n11 = sj * a10 + cj * a11;
                    if (bi == bj && si != 0.f) { n01 = 0.f; n10 = 0.f; }
                }
                Hn[(size_t)pi * n + pj] = n00;
                if (vqj) Hn[(size_t)pi * n + qj] = n01;
                if (vqi) Hn[(size_t)qi * n + pj] = n10;
                if (vqi && vqj) Hn[(size_t)qi * n + qj] = n11;
            }
            const int64_t nv = (int64_t)n * half;
            for (int64_t e = gtid; e < nv; e += gsz) {   // V <- V J, in place
                const int a = static_cast<int>(e / half), bj = static_cast<int>(e % half);
                const float sj = ssn[bj];
                if (sj == 0.f) continue;
                const int pj = spp[bj], qj = sqq[bj];
                const float cj = scs[bj];
                const float vp = __ldcg(M.V + (size_t)a * n + pj), vq = __ldcg(M.V + (size_t)a * n + qj);
                M.V[(size_t)a * n + pj] = cj * vp - sj * vq;
                M.V[(size_t)a * n + qj] = sj * vp + cj * vq;
            }
        }
        __syncthreads();                                 // the shared rotations are rewritten next step
        if (t < g.nmat) {                               // every CTA advances the same stages
            if (sstate[t] == kCheck) {
                sstate[t] = kPending;
            } else if (sstate[t] == kRound) {
                sflip[t] ^= 1;
                const int nm1 = g.mat[t].n + (g.mat[t].n & 1) - 1;
                if (++sround[t] == nm1) { sstate[t] = kCheck; ++ssweep[t]; }
            }
        }
        ok = grid_barrier(g.bar, g.bar + 1, gen);
    }
    if (!ok) {
        if (t == 0 && g.err) atomicAdd(g.err, 1);
        return;
    }
    for (int mi = 0; mi < g.nmat; ++mi) {
        const JacobiMat& M = g.mat[mi];
        const float* Hc = sflip[mi] ? M.H2 : M.H;
        for (int64_t i = gtid; i < M.n; i += gsz) M.evals[i] = __ldcg(Hc + (size_t)i * M.n + i);
    }
}

}  // namespace

int jacobi_group_grid() {
    static int grid = 0;
    if (!grid) {
        int dev = 0, sms = 0, per = 0, coop = 0;
        if (cudaGetDevice(&dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, dev) != cudaSuccess || !coop ||
            cudaFuncSetAttribute(jacobi_group_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kJacobiMaxSmem) != cudaSuccess ||
            cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per, jacobi_group_kernel, JT, kJacobiMaxSmem) != cudaSuccess || per < 1)
            return 0;
        grid = sms * (per < 2 ? per : 2);
    }
    return grid;
}

size_t jacobi_rot_floats(int n) { return 4 * (size_t)((n + (n & 1)) / 2); }

cudaError_t jacobi_group(const JacobiGroup& g, int grid, cudaStream_t st) {
    if (g.nmat <= 0) return cudaSuccess;
    if (grid <= 0 || grid > kJacobiMaxGrid) return cudaErrorInvalidValue;
    size_t smem = 0;
    for (int i = 0; i < g.nmat; ++i) {
        if (g.mat[i].soff != (int)smem) return cudaErrorInvalidValue;
        smem += jacobi_rot_floats(g.mat[i].n);
    }
    smem *= sizeof(float);
    if (smem > kJacobiMaxSmem) return cudaErrorInvalidValue;
    {   // per device: set on every call (cheap next to the launch)
        const cudaError_t ea = cudaFuncSetAttribute(jacobi_group_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kJacobiMaxSmem);
        if (ea != cudaSuccess) return ea;
    }
    cudaError_t e = cudaMemsetAsync(g.bar, 0, 2 * sizeof(int), st);    // arrivals and generation
    if (e != cudaSuccess) return e;
    void* args[] = {const_cast<JacobiGroup*>(&g)};
    return cudaLaunchCooperativeKernel(reinterpret_cast<const void*>(jacobi_group_kernel), dim3(grid), dim3(JT), args, smem, st);
}

}  // namespace glr
