// Fused, grouped streaming kernels of the GreedyLore step.
//
// K1 (stream_group): one CTA per strip of BN columns of one matrix's oriented m' x n' layout,
// covering all m' rows.  For every node i the CTA stages the strip of B_i (the last step's
// composed gradient) and of G_i in shared memory with cp.async (B double-buffered across
// nodes), computes the deferred projection R_i = P_prev^T B_i for the strip (a reduction over
// the m' rows, which is why the whole strip is resident), forms
//     M_i = G_i + B_i - P_prev R_i            (Alg. 3 error-feedback line, Eq. ef1)
// writes B_i <- M_i, and accumulates the node sum in registers.  The epilogue writes
// Mbar = (1/N) sum_i M_i and, for a truncated basis, the strip's Approx-Top-r partial sums
//     part[strip][j] = sum_{b in strip} v_j[b] (Mbar - Yt (Y^T Mbar))[j, b]
// (Alg. 2 with U^T Mbar = Mbar - Yt W, W = Y^T Mbar over the strip; v_j from Philox in
// registers, never stored).  G and B are read once and B written once per step.
//
// K3 (update_group): per strip, Rbar = P^T Mbar (node average of R_i by linearity, Eq.
// 8zhb2we09), Ghat = P Rbar (Mbar at a refresh), then MSGD / Adam on X in its own layout
// (transposed back when m > n, Alg. 4).
//
// Thread layout: 512 threads; thread t owns column group cg = t % (BN/4) (4 columns) and
// the 4-row blocks starting at 4 * (t / (BN/4) + u * 512 / (BN/4)), u < 2.  Rank-r products
// are outer products of 128-bit shared-memory loads (P^T rows x R rows), so shared-memory
// traffic stays below the HBM time of the strip.
#include "glr_internal.cuh"

namespace glr {

namespace {

constexpr int NT = kFusedThreads;
constexpr int MAXB = 2;                 // 4x4 blocks per thread

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
    const unsigned s = static_cast<unsigned>(__cvta_generic_to_shared(smem));
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(s), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int Pending>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;\n" ::"n"(Pending) : "memory");
}

__host__ __device__ __forceinline__ size_t align16(size_t x) { return (x + 15) & ~size_t(15); }
__host__ __device__ __forceinline__ int up4(int x) { return (x + 3) & ~3; }
// Pitch of the transposed (r x m') copies: 16-byte rows, and rows q, q+1, ... start 4 banks
// apart so the scalar column reads of project_strip do not conflict.
__host__ __device__ __forceinline__ int tpitch(int mp) { return up4(mp) + 4; }

__device__ __forceinline__ float4 ld4(const float* p) { return *reinterpret_cast<const float4*>(p); }
__device__ __forceinline__ void st4(float* p, float4 v) { *reinterpret_cast<float4*>(p) = v; }
__device__ __forceinline__ float4 ld4(const __nv_bfloat16* p) {
    const uint2 u = *reinterpret_cast<const uint2*>(p);
    const __nv_bfloat162 lo = *reinterpret_cast<const __nv_bfloat162*>(&u.x);
    const __nv_bfloat162 hi = *reinterpret_cast<const __nv_bfloat162*>(&u.y);
    const float2 a = __bfloat1622float2(lo), b = __bfloat1622float2(hi);
    return make_float4(a.x, a.y, b.x, b.y);
}

// Stage rows [0, rows) x columns [c0, c0 + BN) of a row-major matrix (leading dim ld) into
// dst (pitch BN) with 16-byte cp.async; columns >= cols are zeroed.
template <typename T, int BN>
__device__ __forceinline__ void stage_cols(T* dst, const T* src, int ld, int rows, int c0, int cols) {
    constexpr int EPC = 16 / sizeof(T);
    constexpr int CPR = BN / EPC;
    static_assert(BN % EPC == 0, "strip width must be a multiple of 16 bytes");
    for (int c = threadIdx.x; c < rows * CPR; c += NT) {
        const int a = c / CPR, ch = c % CPR;
        const int col = c0 + ch * EPC;
        T* d = dst + a * BN + ch * EPC;
        if (col < cols) {
            cp_async16(d, src + (int64_t)a * ld + col);
        } else {
#pragma unroll
            for (int e = 0; e < EPC; ++e) d[e] = T(0.f);
        }
    }
}

// Stage rows [r0, r0 + BN) (each len elements, contiguous) into dst (pitch dpitch); rows
// >= nrows are zeroed.
template <typename T, int BN>
__device__ __forceinline__ void stage_rows(T* dst, int dpitch, const T* src, int len, int r0, int nrows) {
    constexpr int EPC = 16 / sizeof(T);
    const int cpr = len / EPC;
    for (int c = threadIdx.x; c < BN * cpr; c += NT) {
        const int rr = c / cpr, ch = c % cpr;
        T* d = dst + rr * dpitch + ch * EPC;
        if (r0 + rr < nrows) {
            cp_async16(d, src + (int64_t)(r0 + rr) * len + ch * EPC);
        } else {
#pragma unroll
            for (int e = 0; e < EPC; ++e) d[e] = T(0.f);
        }
    }
}

// Row slices of the strip reduction below: enough to give every thread a 1x4 output block.
template <int BN>
__host__ __device__ __forceinline__ int rsplits(int r) {
    const int blocks = r * (BN / 4);
    return blocks <= NT ? NT / blocks : 1;
}
template <int BN>
__host__ __device__ __forceinline__ int rpart_floats(int r) { return rsplits<BN>(r) * r * BN; }

// out[q][b] = sum_a P[a][q] S[a][b] (q < r, b < BN): P given transposed (Pt[q][a], pitch pt),
// S pitch BN.  1x4 output blocks (q, column group) are spread over the threads with the rows
// split into slices whose partial blocks are added in fixed order.  part: rpart_floats<BN>(r).
template <int BN>
__device__ __forceinline__ void project_strip(const float* S, const float* Pt, int pt, int mp, int r, float* part,
                                              float* out) {
    constexpr int CG = BN / 4;
    const int blocks = r * CG, splits = rsplits<BN>(r);
    const int tid = threadIdx.x;
    for (int t = tid; t < blocks * splits; t += NT) {
        const int blk = t % blocks, sp = t / blocks;
        const int q = blk / CG, cg = blk % CG;
        const int a0 = (mp * sp) / splits, a1 = (mp * (sp + 1)) / splits;
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int a = a0; a < a1; ++a) {
            const float p = Pt[q * pt + a];
            const float4 x = ld4(S + a * BN + 4 * cg);
            acc.x = fmaf(p, x.x, acc.x); acc.y = fmaf(p, x.y, acc.y);
            acc.z = fmaf(p, x.z, acc.z); acc.w = fmaf(p, x.w, acc.w);
        }
        st4(part + (sp * r + q) * BN + 4 * cg, acc);
    }
    __syncthreads();
    for (int o = tid; o < r * BN; o += NT) {
        float acc = 0.f;
        for (int sp = 0; sp < splits; ++sp) acc += part[sp * r * BN + o];
        out[o] = acc;
    }
    __syncthreads();
}

// c[i][j] = sum_q Pt[q][a0 + i] R[q][4 cg + j]   (Pt pitch pt, R pitch BN)
template <int BN>
__device__ __forceinline__ void outer_block(const float* Pt, int pt, const float* R, int r, int a0, int cg,
                                            float c[4][4]) {
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) c[i][j] = 0.f;
    for (int q = 0; q < r; ++q) {
        const float4 p = ld4(Pt + q * pt + a0);
        const float4 x = ld4(R + q * BN + 4 * cg);
        const float pv[4] = {p.x, p.y, p.z, p.w};
        const float xv[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int j = 0; j < 4; ++j) c[i][j] = fmaf(pv[i], xv[j], c[i][j]);
    }
}

// Copy a rows x cols row-major matrix to shared memory as its transpose (cols x tp),
// zero-padding each row from rows up to tp.
__device__ __forceinline__ void load_transposed(float* dst, int tp, const float* src, int rows, int cols) {
    for (int e = threadIdx.x; e < cols * tp; e += NT) {
        const int c = e / tp, a = e % tp;
        dst[e] = a < rows ? src[(int64_t)a * cols + c] : 0.f;
    }
}

__host__ __device__ __forceinline__ size_t gs_bytes_of(int mp, int BN, int gsize, int transposed) {
    const size_t strip_f = (size_t)mp * BN * 4;
    const size_t g = transposed ? (size_t)BN * (mp + 16 / gsize) * gsize : (size_t)mp * BN * gsize;
    return align16(strip_f > g ? strip_f : g);
}

struct StreamSmem {
    float *Bb0, *Bb1, *Pt, *Rs, *Rpart, *Ws;
    unsigned char* gs;
};

// Shared-memory carve-up of K1 (stream_smem_bytes adds up the same pieces).
template <int BN>
__device__ __forceinline__ StreamSmem carve_stream(unsigned char* smem, int mp, int r, int k, size_t gsb, int lam) {
    StreamSmem s;
    const size_t strip = (size_t)mp * BN;
    s.Bb0 = reinterpret_cast<float*>(smem);
    s.Bb1 = s.Bb0 + strip;
    s.gs = reinterpret_cast<unsigned char*>(s.Bb1 + strip);
    float* p = reinterpret_cast<float*>(s.gs + gsb);
    s.Pt = p;    p += align16((size_t)r * tpitch(mp) * 4) / 4;
    s.Rs = p;    p += align16((size_t)r * BN * 4) / 4;
    s.Rpart = p; p += align16((size_t)rpart_floats<BN>(lam ? (r > k ? r : k) : r) * 4) / 4;
    s.Ws = p;
    return s;
}

// ------------------------------------------------------------------------------------------
// K1
// ------------------------------------------------------------------------------------------
template <int BN, typename GT>
__global__ void __launch_bounds__(NT, 1) stream_kernel(const __grid_constant__ StreamGroup g) {
    extern __shared__ __align__(16) unsigned char smem[];
    int mi = 0;
    while (mi + 1 < g.nmat && blockIdx.x >= static_cast<unsigned>(g.mat[mi + 1].strip0)) ++mi;
    const StreamMat& M = g.mat[mi];
    const int s = blockIdx.x - M.strip0;
    const int b0 = s * BN;
    const int mp = M.mp, np = M.np, r = M.r, N = M.N;
    const int tid = threadIdx.x;
    constexpr int EPC = 16 / sizeof(GT);
    const int gpitch = mp + EPC;                      // transposed G strip pitch (elements)
    const StreamSmem sm = carve_stream<BN>(smem, mp, r, M.k, gs_bytes_of(mp, BN, sizeof(GT), M.transposed), M.lam);
    GT* Gs = reinterpret_cast<GT*>(sm.gs);
    const int pt = tpitch(mp);

    const bool corr = !M.e_zero;
    const GT* const* Gp = reinterpret_cast<const GT* const*>(g.G + M.g_off);
    auto stage_B = [&](int i, float* dst) {
        if (corr && i < N) stage_cols<float, BN>(dst, M.B + (int64_t)i * mp * np, np, mp, b0, np);
        cp_async_commit();
    };
    auto stage_G = [&](int i) {
        if (i < N) {
            if (M.transposed) stage_rows<GT, BN>(Gs, gpitch, Gp[i], mp, b0, np);
            else stage_cols<GT, BN>(Gs, Gp[i], np, mp, b0, np);
        }
        cp_async_commit();
    };
    if (corr) load_transposed(sm.Pt, pt, M.Pprev, mp, r);
    stage_B(0, sm.Bb0);
    stage_G(0);
    stage_B(1, sm.Bb1);

    constexpr int CG = BN / 4;
    constexpr int RPP = 4 * (NT / CG);                // rows per pass
    const int cg = tid % CG, rg = tid / CG;
    const int bcol = b0 + 4 * cg;
    const bool cvalid = bcol < np;                    // n' % 4 == 0: a column group is all in or all out
    float acc[MAXB][4][4];
#pragma unroll
    for (int u = 0; u < MAXB; ++u)
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int j = 0; j < 4; ++j) acc[u][i][j] = 0.f;

    for (int i = 0; i < N; ++i) {
        float* Bb = (i & 1) ? sm.Bb1 : sm.Bb0;
        cp_async_wait<2>();                 // B_i has landed (G_i and B_{i+1} may be in flight)
        __syncthreads();
        if (corr) project_strip<BN>(Bb, sm.Pt, pt, mp, r, sm.Rpart, sm.Rs);
        cp_async_wait<1>();                 // G_i has landed
        __syncthreads();
        float* Bi = M.B + (int64_t)i * mp * np;
#pragma unroll
        for (int u = 0; u < MAXB; ++u) {
            const int a0 = 4 * rg + u * RPP;
            if (a0 >= mp) continue;
            float c[4][4];
            if (corr) outer_block<BN>(sm.Pt, pt, sm.Rs, r, a0, cg, c);
            float gv[4][4];
            if (M.transposed) {
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const float4 x = ld4(Gs + (4 * cg + j) * gpitch + a0);
                    gv[0][j] = x.x; gv[1][j] = x.y; gv[2][j] = x.z; gv[3][j] = x.w;
                }
            } else {
#pragma unroll
                for (int ii = 0; ii < 4; ++ii) {
                    const float4 x = (a0 + ii < mp) ? ld4(Gs + (a0 + ii) * BN + 4 * cg) : make_float4(0.f, 0.f, 0.f, 0.f);
                    gv[ii][0] = x.x; gv[ii][1] = x.y; gv[ii][2] = x.z; gv[ii][3] = x.w;
                }
            }
#pragma unroll
            for (int ii = 0; ii < 4; ++ii) {
                const int a = a0 + ii;
                if (a >= mp) break;
                float m[4] = {gv[ii][0], gv[ii][1], gv[ii][2], gv[ii][3]};
                if (corr) {
                    const float4 bv = ld4(Bb + a * BN + 4 * cg);
                    m[0] += bv.x - c[ii][0]; m[1] += bv.y - c[ii][1];
                    m[2] += bv.z - c[ii][2]; m[3] += bv.w - c[ii][3];
                }
                if (M.write_B && cvalid) st4(Bi + (int64_t)a * np + bcol, make_float4(m[0], m[1], m[2], m[3]));
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[u][ii][j] += m[j];
            }
        }
        __syncthreads();                    // strip buffers free
        stage_G(i + 1);
        stage_B(i + 2, Bb);
    }
    cp_async_wait<0>();
    const float invN = 1.0f / static_cast<float>(N);
#pragma unroll
    for (int u = 0; u < MAXB; ++u)
#pragma unroll
        for (int ii = 0; ii < 4; ++ii)
#pragma unroll
            for (int j = 0; j < 4; ++j) acc[u][ii][j] *= invN;
#pragma unroll
    for (int u = 0; u < MAXB; ++u) {
        const int a0 = 4 * rg + u * RPP;
#pragma unroll
        for (int ii = 0; ii < 4; ++ii)
            if (a0 + ii < mp && cvalid)
                st4(M.Mbar + (int64_t)(a0 + ii) * np + bcol,
                    make_float4(acc[u][ii][0], acc[u][ii][1], acc[u][ii][2], acc[u][ii][3]));
    }
    if (!M.lam) return;

    // ---- truncated-basis Approx-Top-r partial sums for this strip ---------------------------
    const int k = M.k;
    float* Ms = reinterpret_cast<float*>(sm.gs);                  // m' x BN
    float* Yst = sm.Bb0;                                          // Y^T  (k x pt)
    float* Ytt = sm.Bb0 + align16((size_t)k * pt * 4) / 4;        // Yt^T (k x pt)
    __syncthreads();
#pragma unroll
    for (int u = 0; u < MAXB; ++u) {
        const int a0 = 4 * rg + u * RPP;
#pragma unroll
        for (int ii = 0; ii < 4; ++ii)
            if (a0 + ii < mp)
                st4(Ms + (a0 + ii) * BN + 4 * cg,
                    cvalid ? make_float4(acc[u][ii][0], acc[u][ii][1], acc[u][ii][2], acc[u][ii][3])
                           : make_float4(0.f, 0.f, 0.f, 0.f));
    }
    load_transposed(Yst, pt, M.Y, mp, k);
    load_transposed(Ytt, pt, M.Yt, mp, k);
    __syncthreads();
    project_strip<BN>(Ms, Yst, pt, mp, k, sm.Rpart, sm.Ws);     // W = Y^T Mbar_strip (k x BN)
    // every lane runs every block: the shuffles below need the whole warp
#pragma unroll
    for (int u = 0; u < MAXB; ++u) {
        const int a0 = 4 * rg + u * RPP;
        float rows[4] = {0.f, 0.f, 0.f, 0.f};
        if (a0 < mp && cvalid) {
            float c[4][4];
            outer_block<BN>(Ytt, pt, sm.Ws, k, a0, cg, c);
#pragma unroll
            for (int ii = 0; ii < 4; ++ii) {
                const int a = a0 + ii;
                if (a >= mp) break;
                const float4 m = ld4(Ms + a * BN + 4 * cg);
                const float4 v = gauss4(M.seed, M.t, static_cast<uint32_t>(a), static_cast<uint32_t>(bcol >> 2),
                                        kTagLambdaV);
                rows[ii] = (m.x - c[ii][0]) * v.x + (m.y - c[ii][1]) * v.y + (m.z - c[ii][2]) * v.z +
                           (m.w - c[ii][3]) * v.w;
            }
        }
#pragma unroll
        for (int ii = 0; ii < 4; ++ii) {
            float sum = rows[ii];
#pragma unroll
            for (int off = CG / 2; off > 0; off >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
            if (cg == 0 && a0 + ii < mp) M.part[(int64_t)s * mp + a0 + ii] = sum;
        }
    }
}

// ------------------------------------------------------------------------------------------
// K3
// ------------------------------------------------------------------------------------------
template <int BN>
__global__ void __launch_bounds__(NT, 1) update_kernel_fused(const __grid_constant__ UpdateGroup g) {
    extern __shared__ __align__(16) unsigned char smem[];
    int mi = 0;
    while (mi + 1 < g.nmat && blockIdx.x >= static_cast<unsigned>(g.mat[mi + 1].strip0)) ++mi;
    const UpdateMat& M = g.mat[mi];
    const int s = blockIdx.x - M.strip0;
    const int b0 = s * BN;
    const int mp = M.mp, np = M.np, r = M.r;
    const int tid = threadIdx.x;
    const int pt = tpitch(mp);
    float* Ms = reinterpret_cast<float*>(smem);                       // m' x BN
    float* Pt = Ms + align16((size_t)mp * BN * 4) / 4;                // r x pt (P transposed)
    float* Rs = Pt + align16((size_t)r * pt * 4) / 4;                 // r x BN
    float* Rpart = Rs + align16((size_t)r * BN * 4) / 4;
    stage_cols<float, BN>(Ms, M.Mbar, np, mp, b0, np);
    cp_async_commit();
    if (M.compressed) load_transposed(Pt, pt, M.P, mp, r);
    cp_async_wait<0>();
    __syncthreads();
    if (M.compressed) {
        project_strip<BN>(Ms, Pt, pt, mp, r, Rpart, Rs);
        for (int o = tid; o < r * BN; o += NT) {
            const int q = o / BN, b = o % BN;
            if (b0 + b < np) M.Rbar[(int64_t)q * np + b0 + b] = Rs[o];
        }
    }
    constexpr int CG = BN / 4;
    constexpr int RPP = 4 * (NT / CG);
    const int cg = tid % CG, rg = tid / CG;
    const int bcol = b0 + 4 * cg;
    if (bcol >= np) return;
    const float b1 = g.beta1, b2 = g.beta2, lr = g.lr, eps = g.eps;
    const bool adam = g.optimizer == GLR_ADAM;
#pragma unroll
    for (int u = 0; u < MAXB; ++u) {
        const int a0 = 4 * rg + u * RPP;
        if (a0 >= mp) break;
        float gh[4][4];
        if (M.compressed) {
            outer_block<BN>(Pt, pt, Rs, r, a0, cg, gh);
        } else {
#pragma unroll
            for (int ii = 0; ii < 4; ++ii) {
                const float4 x = a0 + ii < mp ? ld4(Ms + (a0 + ii) * BN + 4 * cg) : make_float4(0.f, 0.f, 0.f, 0.f);
                gh[ii][0] = x.x; gh[ii][1] = x.y; gh[ii][2] = x.z; gh[ii][3] = x.w;
            }
        }
        // four float4 vectors of X: rows a0..a0+3 (X[a][b], m <= n) or, when m > n, the
        // entries a0..a0+3 of the X rows b = bcol..bcol+3 (X[b][a]; m' % 4 == 0 there)
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            int64_t xi;
            float gv[4];
            if (M.transposed) {
                xi = (int64_t)(bcol + v) * mp + a0;
#pragma unroll
                for (int ii = 0; ii < 4; ++ii) gv[ii] = gh[ii][v];
            } else {
                if (a0 + v >= mp) continue;
                xi = (int64_t)(a0 + v) * np + bcol;
#pragma unroll
                for (int j = 0; j < 4; ++j) gv[j] = gh[v][j];
            }
            const float4 mo = ld4(M.Mo + xi), x = ld4(M.X + xi);
            float mv[4] = {mo.x, mo.y, mo.z, mo.w}, xv[4] = {x.x, x.y, x.z, x.w};
            float vv[4] = {0.f, 0.f, 0.f, 0.f};
            if (adam) {
                const float4 vo = ld4(M.Vo + xi);
                vv[0] = vo.x; vv[1] = vo.y; vv[2] = vo.z; vv[3] = vo.w;
            }
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                mv[e] = fmaf(b1, mv[e], (1.0f - b1) * gv[e]);
                if (adam) {
                    vv[e] = fmaf(b2, vv[e], (1.0f - b2) * gv[e] * gv[e]);
                    xv[e] -= lr * mv[e] / (sqrtf(vv[e]) + eps);
                } else {
                    xv[e] -= lr * mv[e];
                }
            }
            st4(M.Mo + xi, make_float4(mv[0], mv[1], mv[2], mv[3]));
            st4(M.X + xi, make_float4(xv[0], xv[1], xv[2], xv[3]));
            if (adam) st4(M.Vo + xi, make_float4(vv[0], vv[1], vv[2], vv[3]));
        }
    }
}

}  // namespace

size_t stream_smem_bytes(int mp, int r, int k, int BN, int gsize, int transposed, int lam) {
    const size_t strip = (size_t)mp * BN * 4;
    size_t bytes = 2 * strip + gs_bytes_of(mp, BN, gsize, transposed);
    bytes += align16((size_t)r * tpitch(mp) * 4) + align16((size_t)r * BN * 4);
    const int rk = lam ? (r > k ? r : k) : r;
    int rp = 0;
    switch (BN) {
        case 32: rp = rpart_floats<32>(rk); break;
        case 16: rp = rpart_floats<16>(rk); break;
        default: rp = rpart_floats<8>(rk); break;
    }
    bytes += align16((size_t)rp * 4);
    if (lam) {
        bytes += align16((size_t)k * BN * 4);
        // Y^T and Yt^T (k x tpitch(m') each) are staged in the two B buffers
        if (2 * align16((size_t)k * tpitch(mp) * 4) > 2 * strip) return ~size_t(0);
    }
    return bytes;
}

size_t update_smem_bytes(int mp, int r, int BN) {
    int rp = 0;
    switch (BN) {
        case 32: rp = rpart_floats<32>(r); break;
        case 16: rp = rpart_floats<16>(r); break;
        default: rp = rpart_floats<8>(r); break;
    }
    return align16((size_t)mp * BN * 4) + align16((size_t)r * tpitch(mp) * 4) + align16((size_t)r * BN * 4) +
           align16((size_t)rp * 4);
}

template <int BN, typename GT>
static cudaError_t launch_stream(const StreamGroup& g, size_t smem, cudaStream_t st) {
    static bool set = false;
    if (!set) {
        cudaError_t e = cudaFuncSetAttribute(stream_kernel<BN, GT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             227 * 1024);
        if (e != cudaSuccess) return e;
        set = true;
    }
    stream_kernel<BN, GT><<<g.total_strips, NT, smem, st>>>(g);
    return cudaGetLastError();
}

cudaError_t stream_group(const StreamGroup& g, size_t smem, cudaStream_t st) {
    if (g.total_strips <= 0) return cudaSuccess;
    const bool bf = g.grad_dtype == GLR_BF16;
    switch (g.BN) {
        case 32: return bf ? launch_stream<32, __nv_bfloat16>(g, smem, st) : launch_stream<32, float>(g, smem, st);
        case 16: return bf ? launch_stream<16, __nv_bfloat16>(g, smem, st) : launch_stream<16, float>(g, smem, st);
        case 8: return bf ? launch_stream<8, __nv_bfloat16>(g, smem, st) : launch_stream<8, float>(g, smem, st);
        default: return cudaErrorInvalidValue;
    }
}

template <int BN>
static cudaError_t launch_update(const UpdateGroup& g, size_t smem, cudaStream_t st) {
    static bool set = false;
    if (!set) {
        cudaError_t e = cudaFuncSetAttribute(update_kernel_fused<BN>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             227 * 1024);
        if (e != cudaSuccess) return e;
        set = true;
    }
    update_kernel_fused<BN><<<g.total_strips, NT, smem, st>>>(g);
    return cudaGetLastError();
}

cudaError_t update_group(const UpdateGroup& g, size_t smem, cudaStream_t st) {
    if (g.total_strips <= 0) return cudaSuccess;
    switch (g.BN) {
        case 32: return launch_update<32>(g, smem, st);
        case 16: return launch_update<16>(g, smem, st);
        case 8: return launch_update<8>(g, smem, st);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace glr
