// Streaming kernels of the GreedyLore step: the error-feedback compose pass (K1), the
// decompress + optimizer pass (K3), the deferred error materialisation, and a generic
// strided fp32 GEMM used by the small projections and the refresh.
#include "glr_internal.cuh"

namespace glr {

// ------------------------------------------------------------------------------------------
// Generic strided batched SGEMM: 64 x 64 output tile, K chunks of 16, 256 threads, 4 x 4
// outputs per thread.  Operand tiles are staged through shared memory with the load order
// chosen from the unit stride so global reads coalesce.
// ------------------------------------------------------------------------------------------
namespace {
constexpr int GB_M = 64, GB_N = 64, GB_K = 16;

__global__ void __launch_bounds__(256) gemm_f32_kernel(GemmDesc d, int kchunk) {
    __shared__ float As[GB_K][GB_M + 4];
    __shared__ float Bs[GB_K][GB_N + 4];
    const bool split = kchunk > 0;                  // blockIdx.z = K slice (batch == 1)
    const int z = split ? 0 : blockIdx.z;
    const float* A = d.A + z * d.sAz;
    const float* B = d.B + z * d.sBz;
    float* C = d.C + z * d.sCz;
    const int i0 = blockIdx.y * GB_M, j0 = blockIdx.x * GB_N;
    const int tid = threadIdx.x, tx = tid % 16, ty = tid / 16;
    float acc[4][4] = {};
    const bool a_i_unit = d.sAi == 1;
    const bool b_j_unit = d.sBj == 1;
    const int kbeg = split ? blockIdx.z * kchunk : 0;
    const int kend = split ? min(d.K, kbeg + kchunk) : d.K;
    for (int p0 = kbeg; p0 < kend; p0 += GB_K) {
        for (int e = tid; e < GB_M * GB_K; e += 256) {
            int ii, pp;
            if (a_i_unit) { ii = e % GB_M; pp = e / GB_M; } else { pp = e % GB_K; ii = e / GB_K; }
            const int gi = i0 + ii, gp = p0 + pp;
            As[pp][ii] = (gi < d.M && gp < kend) ? A[gi * d.sAi + gp * d.sAp] : 0.f;
        }
        for (int e = tid; e < GB_N * GB_K; e += 256) {
            int jj, pp;
            if (b_j_unit) { jj = e % GB_N; pp = e / GB_N; } else { pp = e % GB_K; jj = e / GB_K; }
            const int gj = j0 + jj, gp = p0 + pp;
            Bs[pp][jj] = (gj < d.N && gp < kend) ? B[gp * d.sBp + gj * d.sBj] : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int p = 0; p < GB_K; ++p) {
            float a[4], b[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) { a[u] = As[p][ty * 4 + u]; b[u] = Bs[p][tx * 4 + u]; }
#pragma unroll
            for (int u = 0; u < 4; ++u)
#pragma unroll
                for (int v = 0; v < 4; ++v) acc[u][v] = fmaf(a[u], b[v], acc[u][v]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const int gi = i0 + ty * 4 + u;
        if (gi >= d.M) continue;
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            const int gj = j0 + tx * 4 + v;
            if (gj >= d.N) continue;
            if (split) {
                d.ws[((int64_t)blockIdx.z * d.M + gi) * d.N + gj] = acc[u][v];
                continue;
            }
            float* c = C + gi * d.sCi + gj * d.sCj;
            const float val = d.alpha * acc[u][v];
            *c = d.beta == 0.f ? val : fmaf(d.beta, *c, val);
        }
    }
}

// C = alpha * sum_z ws[z] + beta * C, slices added in order.
__global__ void gemm_splitk_reduce(GemmDesc d, int splits) {
    const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= (int64_t)d.M * d.N) return;
    const int i = static_cast<int>(e / d.N), j = static_cast<int>(e % d.N);
    float acc = 0.f;
    for (int zz = 0; zz < splits; ++zz) acc += d.ws[(int64_t)zz * d.M * d.N + e];
    float* c = d.C + i * d.sCi + j * d.sCj;
    const float val = d.alpha * acc;
    *c = d.beta == 0.f ? val : fmaf(d.beta, *c, val);
}
}  // namespace

cudaError_t gemm_f32(const GemmDesc& d, cudaStream_t st) {
    if (d.M <= 0 || d.N <= 0 || d.batch <= 0) return cudaSuccess;
    const int tiles = ((d.N + GB_N - 1) / GB_N) * ((d.M + GB_M - 1) / GB_M);
    int splits = 1;
    if (d.batch == 1 && d.ws && tiles < 148 && d.K >= 512) {
        splits = d.K / 256;
        splits = splits < 296 / tiles ? splits : 296 / tiles;
        const int64_t fit = d.ws_floats / ((int64_t)d.M * d.N);
        splits = (int64_t)splits < fit ? splits : (int)fit;
    }
    if (splits > 1) {
        const int kchunk = ((d.K + splits - 1) / splits + GB_K - 1) / GB_K * GB_K;
        splits = (d.K + kchunk - 1) / kchunk;
        dim3 grid((d.N + GB_N - 1) / GB_N, (d.M + GB_M - 1) / GB_M, splits);
        gemm_f32_kernel<<<grid, 256, 0, st>>>(d, kchunk);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
        const int64_t total = (int64_t)d.M * d.N;
        gemm_splitk_reduce<<<(unsigned)((total + 255) / 256), 256, 0, st>>>(d, splits);
        return cudaGetLastError();
    }
    dim3 grid((d.N + GB_N - 1) / GB_N, (d.M + GB_M - 1) / GB_M, d.batch);
    gemm_f32_kernel<<<grid, 256, 0, st>>>(d, 0);
    return cudaGetLastError();
}

// ------------------------------------------------------------------------------------------
// K1 compose.  A 32 x 32 tile of the oriented m' x n' layout per CTA (32 x 8 threads, four
// rows per thread).  The tile's rows of Pprev (32 x r) stay in shared memory for all nodes;
// node i's columns of Rw_i (r x 32) and its G tile (transposed through shared memory when
// m > n) are staged per node.  The node sum is kept in registers.
// ------------------------------------------------------------------------------------------
namespace {
constexpr int CT = 32;

__global__ void __launch_bounds__(256) compose_kernel(ComposeArgs a) {
    extern __shared__ float sm[];
    float* Ps = sm;                       // CT x r
    float* Rs = Ps + CT * a.r;            // r x CT
    float* Gs = Rs + a.r * CT;            // CT x (CT + 1)
    const int a0 = blockIdx.y * CT, b0 = blockIdx.x * CT;
    const int tx = threadIdx.x, ty = threadIdx.y, tid = ty * CT + tx;
    const bool corr = !a.e_zero;
    if (corr) {
        for (int e = tid; e < CT * a.r; e += 256) {
            const int aa = e / a.r, q = e % a.r;
            Ps[e] = (a0 + aa < a.mp) ? a.Pprev[(int64_t)(a0 + aa) * a.r + q] : 0.f;
        }
    }
    float sum[4] = {0.f, 0.f, 0.f, 0.f};
    for (int i = 0; i < a.N; ++i) {
        const void* G = a.G[i];
        if (a.transposed) {       // G_i(a, b) = G_i[b * m' + a]: read along a
            for (int rr = ty; rr < CT; rr += 8) {
                const int b = b0 + rr, aa = a0 + tx;
                Gs[tx * (CT + 1) + rr] = (b < a.np && aa < a.mp) ? load_grad(G, (int64_t)b * a.mp + aa, a.grad_dtype) : 0.f;
            }
        } else {
            for (int rr = ty; rr < CT; rr += 8) {
                const int aa = a0 + rr, b = b0 + tx;
                Gs[rr * (CT + 1) + tx] = (aa < a.mp && b < a.np) ? load_grad(G, (int64_t)aa * a.np + b, a.grad_dtype) : 0.f;
            }
        }
        if (corr) {
            const float* Rw = a.Rw + (int64_t)i * a.r * a.np;
            for (int e = tid; e < a.r * CT; e += 256) {
                const int q = e / CT, bb = e % CT;
                Rs[e] = (b0 + bb < a.np) ? Rw[(int64_t)q * a.np + b0 + bb] : 0.f;
            }
        }
        __syncthreads();
        float* Bi = a.B + (int64_t)i * a.mp * a.np;
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int rr = ty + 8 * u, aa = a0 + rr, b = b0 + tx;
            if (aa >= a.mp || b >= a.np) continue;
            float mval = Gs[rr * (CT + 1) + tx];
            const int64_t idx = (int64_t)aa * a.np + b;
            if (corr) {
                float c = 0.f;
                for (int q = 0; q < a.r; ++q) c = fmaf(Ps[rr * a.r + q], Rs[q * CT + tx], c);
                mval += Bi[idx] - c;
            }
            if (a.write_B) Bi[idx] = mval;
            sum[u] += mval;
        }
        __syncthreads();
    }
    const float invN = 1.0f / static_cast<float>(a.N);
    bool bad = false;
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const int aa = a0 + ty + 8 * u, b = b0 + tx;
        if (aa < a.mp && b < a.np) {
            a.Mbar[(int64_t)aa * a.np + b] = sum[u] * invN;
            bad |= !isfinite(sum[u]);
        }
    }
    flag_nonfinite(bad, a.nonfinite);
}
}  // namespace

cudaError_t compose(const ComposeArgs& a, cudaStream_t st) {
    dim3 grid((a.np + CT - 1) / CT, (a.mp + CT - 1) / CT);
    const size_t smem = sizeof(float) * (2 * CT * a.r + CT * (CT + 1));
    {   // per device: set on every call (cheap next to the launch)
        const cudaError_t ea = cudaFuncSetAttribute(compose_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 160 * 1024);
        if (ea != cudaSuccess) return ea;
    }
    compose_kernel<<<grid, dim3(CT, 8), smem, st>>>(a);
    return cudaGetLastError();
}

// ------------------------------------------------------------------------------------------
// K3 decompress + optimizer.  Ghat for a 32 x 32 oriented tile is formed with coalesced reads
// into shared memory, then X / M / V are updated in X's own layout (transposed when m > n).
// ------------------------------------------------------------------------------------------
namespace {
__global__ void __launch_bounds__(256) update_kernel(UpdateArgs a) {
    extern __shared__ float sm[];
    float* Ps = sm;                       // CT x r
    float* Rs = Ps + CT * a.r;            // r x CT
    float* Gt = Rs + a.r * CT;            // CT x (CT + 1)
    const int a0 = blockIdx.y * CT, b0 = blockIdx.x * CT;
    const int tx = threadIdx.x, ty = threadIdx.y, tid = ty * CT + tx;
    if (a.compressed) {
        for (int e = tid; e < CT * a.r; e += 256) {
            const int aa = e / a.r, q = e % a.r;
            Ps[e] = (a0 + aa < a.mp) ? a.P[(int64_t)(a0 + aa) * a.r + q] : 0.f;
        }
        for (int e = tid; e < a.r * CT; e += 256) {
            const int q = e / CT, bb = e % CT;
            Rs[e] = (b0 + bb < a.np) ? a.Rbar[(int64_t)q * a.np + b0 + bb] : 0.f;
        }
        __syncthreads();
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const int rr = ty + 8 * u, aa = a0 + rr, b = b0 + tx;
        float g = 0.f;
        if (aa < a.mp && b < a.np) {
            if (a.compressed) {
                for (int q = 0; q < a.r; ++q) g = fmaf(Ps[rr * a.r + q], Rs[q * CT + tx], g);
            } else {
                g = a.Mbar[(int64_t)aa * a.np + b];
            }
        }
        Gt[rr * (CT + 1) + tx] = g;
    }
    __syncthreads();
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const int rr = ty + 8 * u;
        int64_t xi;
        float g;
        if (a.transposed) {   // X is n' x m' (m > n): X[b][a], contiguous along a
            const int b = b0 + rr, aa = a0 + tx;
            if (b >= a.np || aa >= a.mp) continue;
            xi = (int64_t)b * a.mp + aa;
            g = Gt[tx * (CT + 1) + rr];
        } else {
            const int aa = a0 + rr, b = b0 + tx;
            if (aa >= a.mp || b >= a.np) continue;
            xi = (int64_t)aa * a.np + b;
            g = Gt[rr * (CT + 1) + tx];
        }
        const float m1 = fmaf(a.beta1, a.Mo[xi], (1.0f - a.beta1) * g);
        a.Mo[xi] = m1;
        if (a.optimizer == GLR_ADAM) {
            const float v1 = fmaf(a.beta2, a.Vo[xi], (1.0f - a.beta2) * g * g);
            a.Vo[xi] = v1;
            a.X[xi] -= a.lr * m1 / (sqrtf(v1) + a.eps);
        } else {
            a.X[xi] -= a.lr * m1;
        }
    }
}

__global__ void __launch_bounds__(256) error_kernel(int mp, int np, int r, int e_zero, const float* B,
                                                    const float* Pprev, const float* Rw, float* E) {
    const int64_t idx = (int64_t)blockIdx.x * 256 + threadIdx.x;
    if (idx >= (int64_t)mp * np) return;
    if (e_zero) { E[idx] = 0.f; return; }
    const int aa = static_cast<int>(idx / np), b = static_cast<int>(idx % np);
    float c = 0.f;
    for (int q = 0; q < r; ++q) c = fmaf(Pprev[(int64_t)aa * r + q], Rw[(int64_t)q * np + b], c);
    E[idx] = B[idx] - c;
}
}  // namespace

cudaError_t update(const UpdateArgs& a, cudaStream_t st) {
    dim3 grid((a.np + CT - 1) / CT, (a.mp + CT - 1) / CT);
    const size_t smem = sizeof(float) * (2 * CT * a.r + CT * (CT + 1));
    {   // per device: set on every call (cheap next to the launch)
        const cudaError_t ea = cudaFuncSetAttribute(update_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 160 * 1024);
        if (ea != cudaSuccess) return ea;
    }
    update_kernel<<<grid, dim3(CT, 8), smem, st>>>(a);
    return cudaGetLastError();
}

cudaError_t materialize_error(int mp, int np, int r, int e_zero, const float* B, const float* Pprev,
                              const float* Rw, float* E, cudaStream_t st) {
    const int64_t total = (int64_t)mp * np;
    error_kernel<<<(unsigned)((total + 255) / 256), 256, 0, st>>>(mp, np, r, e_zero, B, Pprev, Rw, E);
    return cudaGetLastError();
}

}  // namespace glr

// ------------------------------------------------------------------------------------------
// Grouped fp32 products (the refresh's k-wide fp32 steps: Gram matrices, CholeskyQR's X L^{-T},
// the Rayleigh-Ritz rotation Q W, Yt = Y T^T): a 64 x 64 output tile per CTA of 256 threads, each
// thread a 4 x 4 block, K staged through shared memory 16 at a time; sums in a fixed order.
// ------------------------------------------------------------------------------------------
namespace glr {
namespace {

__global__ void __launch_bounds__(256) gemm_group_kernel(const __grid_constant__ GemmGroup g) {
    __shared__ float As[16][68], Bs[16][68];
    const int tile = blockIdx.x;
    int lo = 0, hi = g.nmat - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (g.mat[mid].tile0 <= tile) lo = mid; else hi = mid - 1;
    }
    const GemmMat& M = g.mat[lo];
    const int lt = tile - M.tile0, tn = (M.N + 63) / 64;
    const int i0 = (lt / tn) * 64, j0 = (lt % tn) * 64;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    float acc[4][4] = {};
    for (int p0 = 0; p0 < M.K; p0 += 16) {
        for (int e = threadIdx.x; e < 16 * 64; e += 256) {
            // consecutive threads along the operand's contiguous index
            const bool pa = M.sAp == 1;
            const int pp = pa ? (e & 15) : (e >> 6), ii = pa ? (e >> 4) : (e & 63);
            const int i = i0 + ii, p = p0 + pp;
            As[pp][ii] = (i < M.M && p < M.K) ? M.A[(int64_t)i * M.sAi + (int64_t)p * M.sAp] : 0.f;
            const bool jb = M.sBj == 1;
            const int jj = jb ? (e & 63) : (e >> 4), pq = jb ? (e >> 6) : (e & 15);
            const int j = j0 + jj, q = p0 + pq;
            Bs[pq][jj] = (j < M.N && q < M.K) ? M.B[(int64_t)q * M.sBp + (int64_t)j * M.sBj] : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int pp = 0; pp < 16; ++pp) {
            float a[4], b[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) { a[u] = As[pp][ty * 4 + u]; b[u] = Bs[pp][tx * 4 + u]; }
#pragma unroll
            for (int u = 0; u < 4; ++u)
#pragma unroll
                for (int v = 0; v < 4; ++v) acc[u][v] = fmaf(a[u], b[v], acc[u][v]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            const int i = i0 + ty * 4 + u, j = j0 + tx * 4 + v;
            if (i < M.M && j < M.N) M.C[(int64_t)i * M.sCi + (int64_t)j * M.sCj] = (M.alpha != 0.f ? M.alpha : 1.f) * acc[u][v];
        }
}

}  // namespace

cudaError_t gemm_group_f32(GemmGroup& g, cudaStream_t st) {
    g.total_tiles = 0;
    for (int i = 0; i < g.nmat; ++i) {
        GemmMat& M = g.mat[i];
        M.tile0 = g.total_tiles;
        g.total_tiles += ((M.M + 63) / 64) * ((M.N + 63) / 64);
    }
    if (g.total_tiles <= 0) return cudaSuccess;
    gemm_group_kernel<<<g.total_tiles, 256, 0, st>>>(g);
    return cudaGetLastError();
}

}  // namespace glr
