// The streaming passes of the first path when its rank-r products run as library GEMMs (large
// matrices: 2048 <= m' with r >= 32 and the like).  The products leave E_i = B_i - P_prev R_i in B
// and Ghat = P Rbar in a scratch already laid out like X, so both passes here are pure streams:
//   compose (Alg. 3, Eq. ef1): M_i = G_i + E_i, B_i <- M_i, Mbar = (1/N) sum_i M_i
//   update (Eq. msgd / Eq. adam): the optimizer on X with Ghat, element by element.
// Algorithmic bytes: compose N (gsize + 8) + 4 per matrix element (no B read after an error
// reset), update 16 (MSGD) or 24 (Adam) plus 4 for Ghat.
#include "glr_internal.cuh"

namespace glr {

namespace {

constexpr int TB = 256;                // threads per CTA
constexpr int TT = 64;                 // transposed compose: 64 x 64 oriented tile
constexpr int TP = TT + 1;             // its shared-memory pitch (2-way bank conflicts at most)

__device__ __forceinline__ float4 ld4(const float* p) { return *reinterpret_cast<const float4*>(p); }
__device__ __forceinline__ void st4(float* p, float4 v) { *reinterpret_cast<float4*>(p) = v; }
__device__ __forceinline__ float4 ldg4(const void* G, int64_t e, int dtype) {   // 4 gradient elements
    if (dtype == GLR_BF16) {
        const uint2 u = *reinterpret_cast<const uint2*>(static_cast<const __nv_bfloat16*>(G) + e);
        const float2 lo = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.x));
        const float2 hi = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.y));
        return make_float4(lo.x, lo.y, hi.x, hi.y);
    }
    return *reinterpret_cast<const float4*>(static_cast<const float*>(G) + e);
}

// G read in the oriented layout: quads of the flattened m' x n' array (m' n' % 4 == 0).  The
// nodes' loads of a quad are issued four nodes at a time before the adds.
__global__ void __launch_bounds__(TB) compose_rows_kernel(ComposeArgs a) {
    const int64_t nq = (int64_t)a.mp * a.np / 4;
    const int64_t plane = (int64_t)a.mp * a.np;
    const bool corr = !a.e_zero;
    const float invN = 1.0f / static_cast<float>(a.N);
    for (int64_t q = (int64_t)blockIdx.x * TB + threadIdx.x; q < nq; q += (int64_t)gridDim.x * TB) {
        const int64_t e = 4 * q;
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int i0 = 0; i0 < a.N; i0 += 4) {
            float4 g[4], b[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                if (i0 + u >= a.N) continue;
                g[u] = ldg4(a.G[i0 + u], e, a.grad_dtype);
                b[u] = corr ? ld4(a.B + (int64_t)(i0 + u) * plane + e) : make_float4(0.f, 0.f, 0.f, 0.f);
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                if (i0 + u >= a.N) continue;
                const float4 m = make_float4(g[u].x + b[u].x, g[u].y + b[u].y, g[u].z + b[u].z, g[u].w + b[u].w);
                if (a.write_B) st4(a.B + (int64_t)(i0 + u) * plane + e, m);
                acc.x += m.x; acc.y += m.y; acc.z += m.z; acc.w += m.w;
            }
        }
        st4(a.Mbar + e, make_float4(acc.x * invN, acc.y * invN, acc.z * invN, acc.w * invN));
        flag_nonfinite(!isfinite(acc.x) || !isfinite(acc.y) || !isfinite(acc.z) || !isfinite(acc.w), a.nonfinite);
    }
}

// G read transposed (m > n: G_i(a, b) = G_i[b m' + a]): one 64 x 64 oriented tile per CTA, node by
// node through a double-buffered shared tile.  Loads of G run along a (4 consecutive a per
// thread), the combine runs along b (B, Mbar rows); thread t owns rows a = t / 16 + 16 u and the
// columns 4 (t % 16) .. + 3 of the tile.  m' % 4 == 0 and n' % 4 == 0.
__global__ void __launch_bounds__(TB) compose_cols_kernel(ComposeArgs a) {
    __shared__ float Gs[2][TT * TP];                    // Gs[b * TP + a]
    const int a0 = blockIdx.y * TT, b0 = blockIdx.x * TT;
    const int t = threadIdx.x, lq = t % 16, lr = t / 16;
    const int64_t plane = (int64_t)a.mp * a.np;
    const bool corr = !a.e_zero;
    float4 acc[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) acc[u] = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int i = 0; i < a.N; ++i) {
        float* gs = Gs[i & 1];
#pragma unroll
        for (int u = 0; u < 4; ++u) {                       // G rows b (tile b = lr + 16 u), a quad lq
            const int bb = lr + 16 * u, b = b0 + bb, aa = a0 + 4 * lq;
            float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
            if (b < a.np && aa < a.mp) v = ldg4(a.G[i], (int64_t)b * a.mp + aa, a.grad_dtype);
            gs[bb * TP + 4 * lq] = v.x; gs[bb * TP + 4 * lq + 1] = v.y;
            gs[bb * TP + 4 * lq + 2] = v.z; gs[bb * TP + 4 * lq + 3] = v.w;
        }
        __syncthreads();                                    // the other buffer is free one node later
        float* Bi = a.B + (int64_t)i * plane;
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int ar = lr + 16 * u, aa = a0 + ar, bb = 4 * lq, b = b0 + bb;
            if (aa >= a.mp || b >= a.np) continue;
            const int64_t e = (int64_t)aa * a.np + b;
            float4 m = make_float4(gs[bb * TP + ar], gs[(bb + 1) * TP + ar], gs[(bb + 2) * TP + ar], gs[(bb + 3) * TP + ar]);
            if (corr) {
                const float4 x = ld4(Bi + e);
                m.x += x.x; m.y += x.y; m.z += x.z; m.w += x.w;
            }
            if (a.write_B) st4(Bi + e, m);
            acc[u].x += m.x; acc[u].y += m.y; acc[u].z += m.z; acc[u].w += m.w;
        }
    }
    const float invN = 1.0f / static_cast<float>(a.N);
    bool bad = false;
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const int aa = a0 + lr + 16 * u, b = b0 + 4 * lq;
        if (aa < a.mp && b < a.np) {
            st4(a.Mbar + (int64_t)aa * a.np + b,
                make_float4(acc[u].x * invN, acc[u].y * invN, acc[u].z * invN, acc[u].w * invN));
            bad |= !isfinite(acc[u].x) || !isfinite(acc[u].y) || !isfinite(acc[u].z) || !isfinite(acc[u].w);
        }
    }
    flag_nonfinite(bad, a.nonfinite);
}

// X, Mo (, Vo) and Ghat share X's layout: quads of the flattened m x n array (m n % 4 == 0).
template <bool ADAM>
__global__ void __launch_bounds__(TB) update_flat_kernel(UpdateArgs a) {
    const int64_t nq = (int64_t)a.mp * a.np / 4;
    for (int64_t q = (int64_t)blockIdx.x * TB + threadIdx.x; q < nq; q += (int64_t)gridDim.x * TB) {
        const int64_t e = 4 * q;
        const float4 g4 = ld4(a.Mbar + e), m4 = ld4(a.Mo + e), x4 = ld4(a.X + e);
        float4 v4 = make_float4(0.f, 0.f, 0.f, 0.f);
        if (ADAM) v4 = ld4(a.Vo + e);
        float g[4] = {g4.x, g4.y, g4.z, g4.w}, m[4] = {m4.x, m4.y, m4.z, m4.w};
        float x[4] = {x4.x, x4.y, x4.z, x4.w}, v[4] = {v4.x, v4.y, v4.z, v4.w};
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            m[c] = fmaf(a.beta1, m[c], (1.0f - a.beta1) * g[c]);
            if (ADAM) {
                v[c] = fmaf(a.beta2, v[c], (1.0f - a.beta2) * g[c] * g[c]);
                x[c] -= a.lr * m[c] / (sqrtf(v[c]) + a.eps);
            } else {
                x[c] -= a.lr * m[c];
            }
        }
        st4(a.Mo + e, make_float4(m[0], m[1], m[2], m[3]));
        st4(a.X + e, make_float4(x[0], x[1], x[2], x[3]));
        if (ADAM) st4(a.Vo + e, make_float4(v[0], v[1], v[2], v[3]));
    }
}

// The AMSGrad-type Adam of the convergence analysis (Appendix A): M and V are the EMAs of Ghat
// as in Eq. adam, the normaliser is one scalar, Vt = max(Vt, max over elements of V), and
// X -= lr M / sqrt(Vt + eps).  Ghat is read oriented (m' x n'); X, M, V are in X's layout
// (transposed when m > n).  The maximum is taken over non-negative floats, whose bit patterns
// order like their values, so an integer atomic max gives it exactly, in any order.
__global__ void __launch_bounds__(TB) amsgrad_moments_kernel(const float* Gh, int mp, int np, int transposed,
                                                             float* Mo, float* Vo, float b1, float b2,
                                                             unsigned* vmax_bits) {
    __shared__ unsigned red[TB / 32];
    const int64_t total = (int64_t)mp * np;
    const int xcols = transposed ? mp : np;
    unsigned local = 0u;
    for (int64_t e = (int64_t)blockIdx.x * TB + threadIdx.x; e < total; e += (int64_t)gridDim.x * TB) {
        const int xr = static_cast<int>(e / xcols), xc = static_cast<int>(e % xcols);
        const int a = transposed ? xc : xr, b = transposed ? xr : xc;
        const float g = Gh[(int64_t)a * np + b];
        const float m = fmaf(b1, Mo[e], (1.0f - b1) * g);
        const float v = fmaf(b2, Vo[e], (1.0f - b2) * g * g);
        Mo[e] = m;
        Vo[e] = v;
        local = max(local, __float_as_uint(v));
    }
    for (int o = 16; o > 0; o >>= 1) local = max(local, __shfl_xor_sync(0xffffffffu, local, o));
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = local;
    __syncthreads();
    if (threadIdx.x == 0) {
        unsigned mx = 0u;
        for (int w = 0; w < TB / 32; ++w) mx = max(mx, red[w]);
        atomicMax(vmax_bits, mx);
    }
}
__global__ void amsgrad_scalar_kernel(float* vt, const unsigned* vmax_bits) {
    vt[0] = fmaxf(vt[0], __uint_as_float(*vmax_bits));
}
__global__ void __launch_bounds__(TB) amsgrad_apply_kernel(float* X, const float* Mo, const float* vt, int64_t total,
                                                           float lr, float eps) {
    const float scale = lr / sqrtf(vt[0] + eps);
    for (int64_t e = (int64_t)blockIdx.x * TB + threadIdx.x; e < total; e += (int64_t)gridDim.x * TB)
        X[e] -= scale * Mo[e];
}

// Bias-corrected AdamW with decoupled weight decay (Loshchilov & Hutter): M, V as Eq. adam, then
// X -= lr (c1 M / (sqrt(c2 V) + eps) + wd X) with c1 = 1 / (1 - b1^s), c2 = 1 / (1 - b2^s) for
// optimizer step s (computed by the caller).  Ghat oriented, X / M / V in X's layout.
__global__ void __launch_bounds__(TB) adamw_kernel(const float* Gh, int mp, int np, int transposed, float* X,
                                                   float* Mo, float* Vo, float lr, float b1, float b2, float eps,
                                                   float wd, float c1, float c2) {
    const int64_t total = (int64_t)mp * np;
    const int xcols = transposed ? mp : np;
    for (int64_t e = (int64_t)blockIdx.x * TB + threadIdx.x; e < total; e += (int64_t)gridDim.x * TB) {
        const int xr = static_cast<int>(e / xcols), xc = static_cast<int>(e % xcols);
        const int a = transposed ? xc : xr, b = transposed ? xr : xc;
        const float g = Gh[(int64_t)a * np + b];
        const float m = fmaf(b1, Mo[e], (1.0f - b1) * g);
        const float v = fmaf(b2, Vo[e], (1.0f - b2) * g * g);
        Mo[e] = m;
        Vo[e] = v;
        const float x = X[e];
        X[e] = x - lr * (c1 * m / (sqrtf(c2 * v) + eps) + wd * x);
    }
}

// Algorithm 5's Adam-Update on the projected mean (r x n', any layout, e elements): M, V the EMAs
// of Eq. adam of Rbar, and Rh = M / (sqrt(V) + eps), the step direction in the subspace.
__global__ void __launch_bounds__(TB) galore_moments_kernel(const float* Rbar, int64_t total, float* Ms, float* Vs,
                                                            float* Rh, float b1, float b2, float eps) {
    for (int64_t e = (int64_t)blockIdx.x * TB + threadIdx.x; e < total; e += (int64_t)gridDim.x * TB) {
        const float g = Rbar[e];
        const float m = fmaf(b1, Ms[e], (1.0f - b1) * g);
        const float v = fmaf(b2, Vs[e], (1.0f - b2) * g * g);
        Ms[e] = m;
        Vs[e] = v;
        Rh[e] = m / (sqrtf(v) + eps);
    }
}
// X -= lr D with D oriented (m' x n'); X in its own layout (transposed when m > n).
__global__ void __launch_bounds__(TB) step_apply_kernel(const float* D, int mp, int np, int transposed, float* X,
                                                        float lr) {
    const int64_t total = (int64_t)mp * np;
    const int xcols = transposed ? mp : np;
    for (int64_t e = (int64_t)blockIdx.x * TB + threadIdx.x; e < total; e += (int64_t)gridDim.x * TB) {
        const int xr = static_cast<int>(e / xcols), xc = static_cast<int>(e % xcols);
        const int a = transposed ? xc : xr, b = transposed ? xr : xc;
        X[e] -= lr * D[(int64_t)a * np + b];
    }
}

int stream_grid(int64_t quads) {
    static int sms = 0;
    if (!sms) {
        int dev = 0;
        if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
            sms = 1;
    }
    const int64_t want = (quads + TB - 1) / TB, cap = (int64_t)sms * 8;
    return static_cast<int>(want < cap ? (want > 0 ? want : 1) : cap);
}

}  // namespace

cudaError_t compose_streamed(const ComposeArgs& a, cudaStream_t st) {
    if (a.mp % 4 || a.np % 4) return cudaErrorInvalidValue;
    if (a.transposed) {
        dim3 grid((a.np + TT - 1) / TT, (a.mp + TT - 1) / TT);
        compose_cols_kernel<<<grid, TB, 0, st>>>(a);
    } else {
        compose_rows_kernel<<<stream_grid((int64_t)a.mp * a.np / 4), TB, 0, st>>>(a);
    }
    return cudaGetLastError();
}

cudaError_t amsgrad_update(const float* Ghat, int mp, int np, int transposed, float* X, float* Mo, float* Vo,
                           float* vt, float lr, float beta1, float beta2, float eps, cudaStream_t st) {
    const int64_t total = (int64_t)mp * np;
    unsigned* bits = reinterpret_cast<unsigned*>(vt + 1);
    cudaError_t e = cudaMemsetAsync(bits, 0, sizeof(unsigned), st);
    if (e != cudaSuccess) return e;
    const int grid = stream_grid((total + 3) / 4);
    amsgrad_moments_kernel<<<grid, TB, 0, st>>>(Ghat, mp, np, transposed, Mo, Vo, beta1, beta2, bits);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    amsgrad_scalar_kernel<<<1, 1, 0, st>>>(vt, bits);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    amsgrad_apply_kernel<<<grid, TB, 0, st>>>(X, Mo, vt, total, lr, eps);
    return cudaGetLastError();
}

cudaError_t adamw_update(const float* Ghat, int mp, int np, int transposed, float* X, float* Mo, float* Vo, float lr,
                         float beta1, float beta2, float eps, float wd, float c1, float c2, cudaStream_t st) {
    const int64_t total = (int64_t)mp * np;
    adamw_kernel<<<stream_grid((total + 3) / 4), TB, 0, st>>>(Ghat, mp, np, transposed, X, Mo, Vo, lr, beta1, beta2,
                                                              eps, wd, c1, c2);
    return cudaGetLastError();
}

cudaError_t galore_moments(const float* Rbar, int64_t total, float* Ms, float* Vs, float* Rh, float beta1, float beta2,
                           float eps, cudaStream_t st) {
    galore_moments_kernel<<<stream_grid((total + 3) / 4), TB, 0, st>>>(Rbar, total, Ms, Vs, Rh, beta1, beta2, eps);
    return cudaGetLastError();
}

cudaError_t step_apply(const float* D, int mp, int np, int transposed, float* X, float lr, cudaStream_t st) {
    step_apply_kernel<<<stream_grid(((int64_t)mp * np + 3) / 4), TB, 0, st>>>(D, mp, np, transposed, X, lr);
    return cudaGetLastError();
}

cudaError_t update_streamed_flat(const UpdateArgs& a, cudaStream_t st) {
    // a.mp x a.np here is the element count of X in its own layout (a multiple of 4)
    const int64_t n = (int64_t)a.mp * a.np;
    if (n % 4) return cudaErrorInvalidValue;
    const int grid = stream_grid(n / 4);
    if (a.optimizer == GLR_ADAM) update_flat_kernel<true><<<grid, TB, 0, st>>>(a);
    else update_flat_kernel<false><<<grid, TB, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace glr
