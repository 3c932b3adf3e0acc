// Approx-Top-r (Algorithm 2) on the device: the bilinear forms lambda_j = u_j^T Mbar v_j with
// v_j generated in the GEMM epilogue (never stored), the fixed-order reduction, the arg-top-r
// of lambda-bar^2 (Eq. semi-lazy-svd-3) and the gather of P = U[:, J].
#include "glr_internal.cuh"

namespace glr {

namespace {
constexpr int LT = kLambdaTile;   // 64 rows (j) x 64 columns (b) per CTA
constexpr int LK = 16;

// C(j, b) = sum_p A(j, p) B(p, b) for a 64 x 64 tile; then for each row j the partial
// sum over the tile's columns of C'(j, b) v_j[b], with C' = C (dense) or Mbar - C (wy).
__global__ void __launch_bounds__(256) lambda_kernel(LambdaArgs a) {
    __shared__ float As[LK][LT + 4];
    __shared__ float Bs[LK][LT + 4];
    const int j0 = blockIdx.y * LT, b0 = blockIdx.x * LT;
    const int tid = threadIdx.x, tx = tid % 16, ty = tid / 16;
    // A(j, p): dense U^T -> U[p * m' + j] (unit stride along j); wy Yt -> Yt[j * K + p]
    const int64_t sAj = a.mode == 0 ? 1 : a.K;
    const int64_t sAp = a.mode == 0 ? a.mp : 1;
    float acc[4][4] = {};
    for (int p0 = 0; p0 < a.K; p0 += LK) {
        for (int e = tid; e < LT * LK; e += 256) {
            int jj, pp;
            if (a.mode == 0) { jj = e % LT; pp = e / LT; } else { pp = e % LK; jj = e / LK; }
            const int gj = j0 + jj, gp = p0 + pp;
            As[pp][jj] = (gj < a.mp && gp < a.K) ? a.A[gj * sAj + gp * sAp] : 0.f;
        }
        for (int e = tid; e < LT * LK; e += 256) {
            const int bb = e % LT, pp = e / LT;
            const int gb = b0 + bb, gp = p0 + pp;
            Bs[pp][bb] = (gb < a.np && gp < a.K) ? a.Bm[(int64_t)gp * a.np + gb] : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int p = 0; p < LK; ++p) {
            float x[4], y[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) { x[u] = As[p][ty * 4 + u]; y[u] = Bs[p][tx * 4 + u]; }
#pragma unroll
            for (int u = 0; u < 4; ++u)
#pragma unroll
                for (int v = 0; v < 4; ++v) acc[u][v] = fmaf(x[u], y[v], acc[u][v]);
        }
        __syncthreads();
    }
    const int bq = b0 + tx * 4;   // first column of this thread (a multiple of 4)
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const int j = j0 + ty * 4 + u;
        float s = 0.f;
        if (j < a.mp && bq < a.np) {
            const float4 g = gauss4_fast(a.seed, a.t, static_cast<uint32_t>(j), static_cast<uint32_t>(bq >> 2), kTagLambdaV);
            const float gv[4] = {g.x, g.y, g.z, g.w};
#pragma unroll
            for (int v = 0; v < 4; ++v) {
                const int b = bq + v;
                if (b < a.np) {
                    float c = acc[u][v];
                    if (a.mode == 1) {
                        c = a.Mbar[(int64_t)j * a.np + b] - c;
                        if (a.Csub) c -= a.Csub[(int64_t)j * a.np + b];
                    }
                    s = fmaf(c, gv[v], s);
                }
            }
        }
        // fixed-order reduction over the 16 column groups (lanes with equal ty share a half-warp)
#pragma unroll
        for (int off = 8; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
        if (tx == 0 && j < a.mp) a.part[(int64_t)blockIdx.x * a.mp + j] = s;
    }
}

// ---- the same partial sums for a dense basis on the tensor cores -----------------------------
// C = U^T Mbar by warp-level TF32 MMA (mma.sync m16n8k8) in the 3xTF32 form (x = hi + lo, hi the
// TF32 rounding of x, lo the TF32 truncation of x - hi; a b ~ a_hi b_hi + a_hi b_lo + a_lo b_hi),
// then part[tile][j] = sum over the tile's 64 columns b of C(j, b) v_j[b].  CTA tile 64 j x 64 b,
// K = m' in chunks of 32 staged in shared memory (row pitch 72: conflict-free fragment loads);
// 8 warps = 4 m-tiles x 2 column halves of 4 n-tiles each.
constexpr int LMK = 32;                 // K chunk
constexpr int LMP = 72;                 // shared row pitch (floats)

__device__ __forceinline__ void lm_split(float x, uint32_t& hi, uint32_t& lo) {
    hi = (__float_as_uint(x) + 0x1000u) & 0xffffe000u;
    lo = __float_as_uint(x - __uint_as_float(hi)) & 0xffffe000u;
}
__device__ __forceinline__ void lm_mma(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3, uint32_t b0,
                                       uint32_t b1) {
    asm volatile("mma.sync.aligned.m16n8k8.row.col.f32.tf32.tf32.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
                 "{%0,%1,%2,%3};\n"
                 : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
                 : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__global__ void __launch_bounds__(256) lambda_mma_kernel(LambdaArgs a) {
    __shared__ __align__(16) float As[LMK][LMP];             // U[p][j0 + jj]
    __shared__ __align__(16) float Bs[LMK][LMP];             // Mbar[p][b0 + bb]
    __shared__ float half_sum[2][LT];
    const int j0 = blockIdx.y * LT, b0 = blockIdx.x * LT;
    const int tid = threadIdx.x, w = tid >> 5, lane = tid & 31, g = lane >> 2, t = lane & 3;
    const int mt = w & 3, nh = w >> 2;                        // m-tile (16 rows j), column half
    const int mp = a.mp, np = a.np, K = a.K;
    constexpr int EPT = LMK * LT / 256;                       // 8 entries of each chunk per thread
    float na[EPT], nb[EPT];
    auto fetch = [&](int p0) {
#pragma unroll
        for (int l = 0; l < EPT; ++l) {
            const int e = tid + l * 256, pp = e / LT, cc = e % LT, gp = p0 + pp;
            na[l] = gp < K && j0 + cc < mp ? a.A[(int64_t)gp * mp + j0 + cc] : 0.f;
            nb[l] = gp < K && b0 + cc < np ? a.Bm[(int64_t)gp * np + b0 + cc] : 0.f;
        }
    };
    float acc[4][4];
#pragma unroll
    for (int nt = 0; nt < 4; ++nt)
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[nt][e] = 0.f;
    fetch(0);
    for (int p0 = 0; p0 < K; p0 += LMK) {
        __syncthreads();
#pragma unroll
        for (int l = 0; l < EPT; ++l) {
            const int e = tid + l * 256, pp = e / LT, cc = e % LT;
            As[pp][cc] = na[l];
            Bs[pp][cc] = nb[l];
        }
        __syncthreads();
        if (p0 + LMK < K) fetch(p0 + LMK);
#pragma unroll
        for (int k0 = 0; k0 < LMK; k0 += 8) {
            // A (16 j x 8 p): a0 (g, t), a1 (g + 8, t), a2 (g, t + 4), a3 (g + 8, t + 4)
            uint32_t ah[4], al[4];
            lm_split(As[k0 + t][mt * 16 + g], ah[0], al[0]);
            lm_split(As[k0 + t][mt * 16 + g + 8], ah[1], al[1]);
            lm_split(As[k0 + t + 4][mt * 16 + g], ah[2], al[2]);
            lm_split(As[k0 + t + 4][mt * 16 + g + 8], ah[3], al[3]);
#pragma unroll
            for (int nt = 0; nt < 4; ++nt) {
                // B (8 p x 8 b): b0 (t, g), b1 (t + 4, g)
                const int bc = nh * 32 + nt * 8 + g;
                uint32_t bh0, bl0, bh1, bl1;
                lm_split(Bs[k0 + t][bc], bh0, bl0);
                lm_split(Bs[k0 + t + 4][bc], bh1, bl1);
                lm_mma(acc[nt], al[0], al[1], al[2], al[3], bh0, bh1);
                lm_mma(acc[nt], ah[0], ah[1], ah[2], ah[3], bl0, bl1);
                lm_mma(acc[nt], ah[0], ah[1], ah[2], ah[3], bh0, bh1);
            }
        }
    }
    // C fragment: c0 (g, 2t), c1 (g, 2t + 1), c2 (g + 8, 2t), c3 (g + 8, 2t + 1) of each n-tile
    float s[2] = {0.f, 0.f};
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int j = j0 + mt * 16 + g + 8 * h;
        if (j < mp) {
#pragma unroll
            for (int nt = 0; nt < 4; ++nt) {
                const int bq = b0 + nh * 32 + nt * 8 + 4 * (t >> 1);   // the quad holding 2t, 2t + 1
                if (bq < np) {
                    const float4 v = gauss4_fast(a.seed, a.t, static_cast<uint32_t>(j), static_cast<uint32_t>(bq >> 2),
                                                 kTagLambdaV);
                    const bool upper = (t & 1) != 0;            // columns 2, 3 of the quad
                    const float v0 = upper ? v.z : v.x, v1 = upper ? v.w : v.y;
                    const int b = bq + 2 * (t & 1);
                    if (b < np) s[h] = fmaf(acc[nt][2 * h], v0, s[h]);
                    if (b + 1 < np) s[h] = fmaf(acc[nt][2 * h + 1], v1, s[h]);
                }
            }
        }
    }
#pragma unroll
    for (int h = 0; h < 2; ++h) {                             // the four lanes of a row, in order
        s[h] += __shfl_xor_sync(0xffffffffu, s[h], 1);
        s[h] += __shfl_xor_sync(0xffffffffu, s[h], 2);
        if (t == 0) half_sum[nh][mt * 16 + g + 8 * h] = s[h];
    }
    __syncthreads();
    for (int jj = tid; jj < LT; jj += 256) {
        const int j = j0 + jj;
        if (j < mp) a.part[(int64_t)blockIdx.x * mp + j] = half_sum[0][jj] + half_sum[1][jj];
    }
}
}  // namespace

cudaError_t lambda_partials(const LambdaArgs& a, cudaStream_t st) {
    dim3 grid(a.ntiles, (a.mp + LT - 1) / LT);
    if (a.mode == 0) lambda_mma_kernel<<<grid, 256, 0, st>>>(a);   // dense U: a dense contraction
    else lambda_kernel<<<grid, 256, 0, st>>>(a);
    return cudaGetLastError();
}

// ------------------------------------------------------------------------------------------
// Selection: one CTA.  lambda_j = d_j * sum_t part[j][t] (fixed order); keys
// (bits(lambda^2) << 32) | (~j) sorted descending by a bitonic network, so ties go to the
// lower index; the first r indices are then written in ascending order.
// ------------------------------------------------------------------------------------------
namespace {
__global__ void __launch_bounds__(1024) select_kernel(const float* part, int ntiles, int mp, int r,
                                                      const float* dsign, int k, float* lam,
                                                      int32_t* J, int npow2) {
    extern __shared__ unsigned long long keys[];
    const int tid = threadIdx.x;
    for (int j = tid; j < npow2; j += blockDim.x) {
        unsigned long long key = 0ull;
        if (j < mp) {
            float s = 0.f;
            for (int t = 0; t < ntiles; ++t) s += part[(int64_t)t * mp + j];   // coalesced over j
            if (dsign != nullptr && j < k) s *= dsign[j];
            lam[j] = s;
            const float sc = s * s;
            key = (static_cast<unsigned long long>(__float_as_uint(sc)) << 32) |
                  static_cast<unsigned long long>(0xFFFFFFFFu - static_cast<uint32_t>(j));
        }
        keys[j] = key;
    }
    __syncthreads();
    for (int size = 2; size <= npow2; size <<= 1) {
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
    }
    // ascending index order of the r winners: rank among the winners
    for (int q = tid; q < r; q += blockDim.x) {
        const uint32_t jq = 0xFFFFFFFFu - static_cast<uint32_t>(keys[q] & 0xFFFFFFFFull);
        int rank = 0;
        for (int w = 0; w < r; ++w) {
            const uint32_t jw = 0xFFFFFFFFu - static_cast<uint32_t>(keys[w] & 0xFFFFFFFFull);
            rank += jw < jq;
        }
        J[rank] = static_cast<int32_t>(jq);
    }
}

__global__ void build_P_kernel(int mode, int mp, int r, int k, const int32_t* J, const float* U,
                               const float* Y, const float* Yt, const float* dsign, float* P) {
    const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= (int64_t)mp * r) return;
    const int aa = static_cast<int>(e / r), q = static_cast<int>(e % r);
    const int j = J[q];
    if (mode == 0) { P[e] = U[(int64_t)aa * mp + j]; return; }
    // column j of (I - Y Yt^T), times d_j for the spectral columns j < k
    float v = (aa == j) ? 1.f : 0.f;
    const float* ya = Y + (int64_t)aa * k;
    const float* yj = Yt + (int64_t)j * k;
    for (int c = 0; c < k; ++c) v = fmaf(-ya[c], yj[c], v);
    if (j < k) v *= dsign[j];
    P[e] = v;
}
}  // namespace

// ------------------------------------------------------------------------------------------
// Grouped selection: lambda_reduce_kernel forms lambda-bar, select_group_kernel (one CTA per
// matrix) the arg-top-r J, and pr_kernel (one thread per output) P = U[:, J] and, for the
// matrices whose update streams X, Rbar = P^T Mbar from K1's Wbar.
// ------------------------------------------------------------------------------------------
namespace {
__device__ __forceinline__ unsigned long long shfl_xor_u64(unsigned long long v, int m) {
    const unsigned lo = __shfl_xor_sync(0xffffffffu, static_cast<unsigned>(v), m);
    const unsigned hi = __shfl_xor_sync(0xffffffffu, static_cast<unsigned>(v >> 32), m);
    return (static_cast<unsigned long long>(hi) << 32) | lo;
}

// Keys (lambda-bar_j^2 bits, ~j): distinct, larger score first and the lower index on ties.
__device__ __forceinline__ void select_top_r_block(const SelectMat& M, unsigned long long* keys) {
    const int tid = threadIdx.x, mp = M.mp, r = M.r, nth = blockDim.x;
    auto key_of = [&](int j) -> unsigned long long {
        return j < mp ? (static_cast<unsigned long long>(__float_as_uint(M.lam[j] * M.lam[j])) << 32) |
                            static_cast<unsigned long long>(0xFFFFFFFFu - static_cast<uint32_t>(j))
                      : 0ull;
    };
    auto index_of = [](unsigned long long key) { return static_cast<int32_t>(0xFFFFFFFFu - static_cast<uint32_t>(key)); };
    if (mp <= 1024 && r <= 32) {
        // each warp sorts its 32 keys (j = 32 w + lane) descending with a bitonic network and
        // keeps its r largest: the top r of all keys are among these candidates
        const int lane = tid & 31, w = tid >> 5, nw = (mp + 31) >> 5;
        unsigned long long key = key_of(tid);
#pragma unroll
        for (int size = 2; size <= 32; size <<= 1)
#pragma unroll
            for (int stride = size >> 1; stride > 0; stride >>= 1) {
                const unsigned long long other = shfl_xor_u64(key, stride);
                const bool keep_max = ((lane & stride) == 0) == ((lane & size) == 0 || size == 32);
                key = keep_max ? (key > other ? key : other) : (key < other ? key : other);
            }
        unsigned long long* cand = keys;                     // nw * r candidates
        __shared__ int32_t top[32];
        if (w < nw && lane < r) cand[w * r + lane] = key;
        __syncthreads();
        const int C = nw * r;
        if (tid < C) {
            const unsigned long long kc = cand[tid];
            int above = 0;
            for (int c = 0; c < C; ++c) above += cand[c] > kc;
            if (above < r) top[above] = index_of(kc);        // descending rank of a winner
        }
        __syncthreads();
        if (tid < r) {                                       // J in ascending index order
            const int32_t jq = top[tid];
            int pos = 0;
            for (int q = 0; q < r; ++q) pos += top[q] < jq;
            M.J[pos] = jq;
        }
        return;
    }
    int npow2 = 1;
    while (npow2 < mp) npow2 <<= 1;
    for (int j = tid; j < npow2; j += nth) keys[j] = key_of(j);
    __syncthreads();
    if (mp <= 1024) {
        // keys are distinct: j is among the r largest iff fewer than r keys exceed it
        __shared__ unsigned char win[1024];
        for (int j = tid; j < mp; j += nth) {
            const unsigned long long kj = keys[j];
            int above = 0;
            for (int w = 0; w < mp; ++w) above += keys[w] > kj;
            win[j] = above < r ? 1 : 0;
        }
        __syncthreads();
        for (int j = tid; j < mp; j += nth) {
            if (!win[j]) continue;
            int pos = 0;
            for (int w = 0; w < j; ++w) pos += win[w];
            M.J[pos] = j;
        }
    } else {
        for (int size = 2; size <= npow2; size <<= 1) {
            for (int stride = size >> 1; stride > 0; stride >>= 1) {
                for (int i = tid; i < npow2; i += nth) {
                    const int partner = i ^ stride;
                    if (partner > i) {
                        const bool desc = (i & size) == 0;
                        const unsigned long long x = keys[i], y = keys[partner];
                        if ((x < y) == desc) { keys[i] = y; keys[partner] = x; }
                    }
                }
                __syncthreads();
            }
        }
        for (int q = tid; q < r; q += nth) {
            const int32_t jq = index_of(keys[q]);
            int rank = 0;
            for (int w = 0; w < r; ++w) rank += index_of(keys[w]) < jq;
            M.J[rank] = jq;
        }
    }
}

__global__ void __launch_bounds__(1024) select_group_kernel(const __grid_constant__ SelectGroup g) {
    extern __shared__ unsigned long long keys[];
    const SelectMat& M = g.mat[blockIdx.x];
    if (M.do_select) select_top_r_block(M, keys);           // otherwise J was supplied
    if (!M.YtJ) return;
    // YtJ = Yt[J, :] (r x k) for the tcgen05 path's P and Rbar products
    __syncthreads();
    const int r = M.r, k = M.k;
    for (int e = threadIdx.x; e < r * k; e += blockDim.x) {
        const int q = e / k, c = e - q * k;
        M.YtJ[e] = M.Yt[(int64_t)M.J[q] * k + c];
    }

}

// Output o of the group: matrix i owns [out0, out0 + m' r) for P (row-major m' x r) and, when
// rbar is set, the next r n' for Rbar.
__global__ void __launch_bounds__(256) pr_kernel(const __grid_constant__ SelectGroup g) {
    const int64_t o = (int64_t)blockIdx.x * 256 + threadIdx.x;
    int mi = 0;
    while (mi + 1 < g.nmat && o >= g.mat[mi + 1].out0) ++mi;
    const SelectMat& M = g.mat[mi];
    int64_t local = o - M.out0;
    const int mp = M.mp, r = M.r, k = M.k;
    if (M.build_p && local < (int64_t)mp * r) {
        const int aa = static_cast<int>(local / r), q = static_cast<int>(local % r);
        const int j = M.J[q];
        if (M.mode == 0) { M.P[local] = M.U[(int64_t)aa * mp + j]; return; }
        // column j of (I - Y Yt^T), times d_j for the spectral columns j < k
        float v = (aa == j) ? 1.f : 0.f;
        const float* ya = M.Y + (int64_t)aa * k;
        const float* yj = M.Yt + (int64_t)j * k;
        for (int c = 0; c < k; ++c) v = fmaf(-ya[c], yj[c], v);
        if (j < k) v *= M.dsign[j];
        M.P[local] = v;
        return;
    }
    if (M.build_p) local -= (int64_t)mp * r;
    if (!M.rbar || local >= (int64_t)r * M.np) return;
    // Rbar = P^T Mbar = D_J (Mbar[J, :] - Yt[J, :] Wbar) with Wbar = Y^T Mbar (truncated basis)
    const int np = M.np;
    const int q = static_cast<int>(local / np), c = static_cast<int>(local % np);
    const int j = M.J[q];
    const float* ytj = M.Yt + (int64_t)j * k;
    const float* wc = M.Wbar + c;
    float v = M.Mbar[(int64_t)j * np + c];
    int kk = 0;
    for (; kk + 4 <= k; kk += 4) {                           // four independent loads per round
        const float w0 = wc[(int64_t)kk * np], w1 = wc[(int64_t)(kk + 1) * np];
        const float w2 = wc[(int64_t)(kk + 2) * np], w3 = wc[(int64_t)(kk + 3) * np];
        v = fmaf(-ytj[kk], w0, v); v = fmaf(-ytj[kk + 1], w1, v);
        v = fmaf(-ytj[kk + 2], w2, v); v = fmaf(-ytj[kk + 3], w3, v);
    }
    for (; kk < k; ++kk) v = fmaf(-ytj[kk], wc[(int64_t)kk * np], v);
    if (j < k) v *= M.dsign[j];                              // D = diag(d_0..d_{k-1}, 1, ..., 1)
    M.Rbar[local] = v;
}
}  // namespace

// lambda-bar_j = d_j * sum_t part[t][j]: block (x, matrix) covers 32 consecutive j (lanes)
// with its 32 warps taking every 32nd tile; the warp sums are added in warp order.
__global__ void __launch_bounds__(1024) lambda_reduce_kernel(const __grid_constant__ SelectGroup g) {
    const SelectMat& M = g.mat[blockIdx.y];
    if (!M.do_select) return;
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const int j = blockIdx.x * 32 + lane;
    if (blockIdx.x * 32 >= M.mp) return;
    __shared__ float red[32][33];
    float sum = 0.f;
    if (j < M.mp)
        for (int t = w; t < M.ntiles; t += 32) sum += M.part[(int64_t)t * M.mp + j];
    red[w][lane] = sum;
    __syncthreads();
    if (w == 0 && j < M.mp) {
        float tot = 0.f;
        for (int ww = 0; ww < 32; ++ww) tot += red[ww][lane];
        if (M.dsign != nullptr && j < M.k) tot *= M.dsign[j];
        M.lam[j] = tot;
    }
}

cudaError_t select_group(const SelectGroup& g, cudaStream_t st, int stages) {
    if (g.nmat <= 0) return cudaSuccess;
    int maxmp = 1;
    for (int i = 0; i < g.nmat; ++i) maxmp = g.mat[i].mp > maxmp ? g.mat[i].mp : maxmp;
    cudaError_t e = cudaSuccess;
    if (stages & 1) {
        lambda_reduce_kernel<<<dim3((maxmp + 31) / 32, g.nmat), 1024, 0, st>>>(g);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    if (!(stages & 2)) return cudaSuccess;
    int npow2 = 1;
    while (npow2 < maxmp) npow2 <<= 1;
    {   // per device: set on every call (cheap next to the launch)
        const cudaError_t ea = cudaFuncSetAttribute(select_group_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
        if (ea != cudaSuccess) return ea;
    }
    select_group_kernel<<<g.nmat, 1024, sizeof(unsigned long long) * npow2, st>>>(g);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    if (g.total_out <= 0) return cudaSuccess;              // every P formed by the caller
    pr_kernel<<<(unsigned)((g.total_out + 255) / 256), 256, 0, st>>>(g);
    return cudaGetLastError();
}

namespace {
__global__ void wy_gather_kernel(const float* Yt, const int32_t* J, int r, int k, float* YtJ) {
    const int e = blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= r * k) return;
    const int q = e / k, c = e % k;
    YtJ[e] = Yt[(int64_t)J[q] * k + c];
}
__global__ void wy_fix_kernel(float* P, const int32_t* J, const float* dsign, int mp, int r, int k) {
    const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= (int64_t)mp * r) return;
    const int a = static_cast<int>(e / r), q = static_cast<int>(e % r);
    const int j = J[q];
    float v = P[e] + (a == j ? 1.f : 0.f);
    if (j < k) v *= dsign[j];
    P[e] = v;
}
}  // namespace

cudaError_t wy_columns_gather(const float* Yt, const int32_t* J, int r, int k, float* YtJ, cudaStream_t st) {
    wy_gather_kernel<<<(r * k + 255) / 256, 256, 0, st>>>(Yt, J, r, k, YtJ);
    return cudaGetLastError();
}

cudaError_t wy_columns_fix(float* P, const int32_t* J, const float* dsign, int mp, int r, int k, cudaStream_t st) {
    const int64_t n = (int64_t)mp * r;
    wy_fix_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(P, J, dsign, mp, r, k);
    return cudaGetLastError();
}

cudaError_t select_top_r(const float* part, int ntiles, int mp, int r, const float* dsign, int k,
                         float* lam, int32_t* J, cudaStream_t st) {
    int npow2 = 1;
    while (npow2 < mp) npow2 <<= 1;
    const size_t smem = sizeof(unsigned long long) * npow2;
    {   // per device: set on every call (cheap next to the launch)
        const cudaError_t ea = cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
        if (ea != cudaSuccess) return ea;
    }
    select_kernel<<<1, 1024, smem, st>>>(part, ntiles, mp, r, dsign, k, lam, J, npow2);
    return cudaGetLastError();
}

cudaError_t build_P(int mode, int mp, int r, int k, const int32_t* J, const float* U, const float* Y,
                    const float* Yt, const float* dsign, float* P, cudaStream_t st) {
    const int64_t total = (int64_t)mp * r;
    build_P_kernel<<<(unsigned)((total + 255) / 256), 256, 0, st>>>(mode, mp, r, k, J, U, Y, Yt, dsign, P);
    return cudaGetLastError();
}

}  // namespace glr
