// Fused, grouped streaming kernels of the GreedyLore step.
//
// K1 (stream_group): one CTA per strip of BN columns of one matrix's oriented m' x n' layout,
// covering all m' rows.  For every node i the CTA stages the strip of B_i (the last step's
// composed gradient) in shared memory with cp.async (two buffers: B_{i+1} is in flight while
// node i is processed), loads its G_i values straight into registers, computes
// the deferred projection R_i = P_prev^T B_i for the strip (a reduction over the m' rows,
// which is why the whole strip is resident), forms
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
// Thread layout: thread t owns column group cg = t % (BN/4) (4 columns) and the 4-row blocks
// starting at 4 * (t / (BN/4)) + u * (rows per pass).  Rank-r products are outer products of
// 128-bit shared-memory loads (P^T rows x R rows).
#include "glr_internal.cuh"

namespace glr {

namespace {

constexpr int NT = kFusedThreads;
constexpr int NTU = kUpdateThreads;

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
// Pitch of the transposed (r x m') copies: 16-byte rows covering m' rounded up to 16, and rows
// q, q+1, ... start 4 (or 20) banks apart so the scalar column reads do not conflict.
__host__ __device__ __forceinline__ int tpitch(int mp) { return transposed_pitch(mp); }

__device__ __forceinline__ float4 ld4(const float* p) { return *reinterpret_cast<const float4*>(p); }
__device__ __forceinline__ void st4(float* p, float4 v) { *reinterpret_cast<float4*>(p) = v; }
// Streaming global loads of 4 gradient values (read once per step).
__device__ __forceinline__ float4 ldg4(const float* p) { return __ldcs(reinterpret_cast<const float4*>(p)); }
__device__ __forceinline__ float4 ldg4(const __nv_bfloat16* p) {
    const uint2 u = __ldcs(reinterpret_cast<const uint2*>(p));
    const __nv_bfloat162 lo = *reinterpret_cast<const __nv_bfloat162*>(&u.x);
    const __nv_bfloat162 hi = *reinterpret_cast<const __nv_bfloat162*>(&u.y);
    const float2 a = __bfloat1622float2(lo), b = __bfloat1622float2(hi);
    return make_float4(a.x, a.y, b.x, b.y);
}

// Stage rows [0, rows) x columns [c0, c0 + BN) of a row-major fp32 matrix (leading dim ld)
// into dst (pitch BN) with 16-byte cp.async; columns >= cols are zeroed.
template <int BN, int NTH>
__device__ __forceinline__ void stage_cols(float* dst, const float* src, int ld, int rows, int c0, int cols) {
    constexpr int CPR = BN / 4;
    for (int c = threadIdx.x; c < rows * CPR; c += NTH) {
        const int a = c / CPR, ch = c % CPR;
        const int col = c0 + ch * 4;
        float* d = dst + a * BN + ch * 4;
        if (col < cols) cp_async16(d, src + (int64_t)a * ld + col);
        else st4(d, make_float4(0.f, 0.f, 0.f, 0.f));
    }
}

// Row slices of the strip reduction below: enough to give every thread a 1x4 output block.
template <int BN, int NTH>
__host__ __device__ __forceinline__ int rsplits(int r) {
    const int blocks = r * (BN / 4);
    return blocks <= NTH ? NTH / blocks : 1;
}
template <int BN, int NTH>
__host__ __device__ __forceinline__ int rpart_floats(int r) { return rsplits<BN, NTH>(r) * r * BN; }

// Work assignment of project_strip for one thread (computed once, outside the node loop):
// output block (q, column group cg) and the row slice [a0, a1) of split sp.
struct ProjSlot {
    int active, q, cg, sp, a0, a1;
};
template <int BN, int NTH>
__device__ __forceinline__ ProjSlot proj_slot(int mp, int r) {
    constexpr int CG = BN / 4;
    const int blocks = r * CG, splits = rsplits<BN, NTH>(r);
    ProjSlot s{};
    const int t = threadIdx.x;
    s.active = t < blocks * splits;           // blocks > NTH (splits 1) is handled by the caller
    const int blk = t % blocks;
    s.sp = t / blocks;
    s.q = blk / CG;
    s.cg = blk % CG;
    s.a0 = (mp * s.sp) / splits;
    s.a1 = (mp * (s.sp + 1)) / splits;
    return s;
}

// out[q][b] = sum_a P[a][q] S[a][b] (q < r, b < BN): P given transposed (Pt[q][a], pitch pt),
// S pitch BN.  1x4 output blocks (q, column group) are spread over the threads with the rows
// split into slices whose partial blocks are added in fixed order.  Requires r * BN / 4 <= NTH.
template <int BN, int NTH>
__device__ __forceinline__ void project_strip(const ProjSlot& ps, const float* S, const float* Pt, int pt, int r,
                                              float* part, float* out) {
    if (ps.active) {
        const float* pp = Pt + ps.q * pt + ps.a0;
        const float* sp = S + ps.a0 * BN + 4 * ps.cg;
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 4
        for (int n = ps.a1 - ps.a0; n > 0; --n) {
            const float p = *pp++;
            const float4 x = ld4(sp);
            sp += BN;
            acc.x = fmaf(p, x.x, acc.x); acc.y = fmaf(p, x.y, acc.y);
            acc.z = fmaf(p, x.z, acc.z); acc.w = fmaf(p, x.w, acc.w);
        }
        st4(part + (ps.sp * r + ps.q) * BN + 4 * ps.cg, acc);
    }
    __syncthreads();
    const int splits = rsplits<BN, NTH>(r);
    for (int o = threadIdx.x; o < r * BN; o += NTH) {
        const float* pq = part + o;
        float acc = 0.f;
        for (int n = splits; n > 0; --n, pq += r * BN) acc += *pq;
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
    const float* pp = Pt + a0;
    const float* rp = R + 4 * cg;
#pragma unroll 2
    for (int q = r; q > 0; --q, pp += pt, rp += BN) {
        const float4 p = ld4(pp);
        const float4 x = ld4(rp);
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
template <int NTH>
__device__ __forceinline__ void load_transposed(float* dst, int tp, const float* src, int rows, int cols) {
    for (int e = threadIdx.x; e < cols * tp; e += NTH) {
        const int c = e / tp, a = e % tp;
        dst[e] = a < rows ? src[(int64_t)a * cols + c] : 0.f;
    }
}

// Shared-memory carve-up of K1 (stream_smem_bytes adds up the same pieces).
struct StreamSmem {
    float* Bb;          // two m' x BN strip buffers, back to back
    float *Pt, *Rs, *Rpart, *Ws;
};
template <int BN>
__device__ __forceinline__ StreamSmem carve_stream(unsigned char* smem, int mp, int r, int k, int lam) {
    StreamSmem s;
    const size_t strip = (size_t)mp * BN;
    float* p = reinterpret_cast<float*>(smem);
    s.Bb = p;
    p += 2 * strip;
    s.Pt = p;    p += align16((size_t)r * tpitch(mp) * 4) / 4;
    s.Rs = p;    p += align16((size_t)r * BN * 4) / 4;
    s.Rpart = p; p += align16((size_t)rpart_floats<BN, NT>(lam ? (r > k ? r : k) : r) * 4) / 4;
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
    const StreamSmem sm = carve_stream<BN>(smem, mp, r, M.k, M.lam);
    const int pt = tpitch(mp);

    const bool corr = !M.e_zero;
    const GT* const* Gp = reinterpret_cast<const GT* const*>(g.G + M.g_off);
    auto stage_B = [&](int i) {
        if (corr && i < N) stage_cols<BN, NT>(sm.Bb + (size_t)(i & 1) * mp * BN, M.B + (int64_t)i * mp * np, np, mp, b0, np);
        cp_async_commit();
    };
    if (corr) load_transposed<NT>(sm.Pt, pt, M.Pprev, mp, r);
    const ProjSlot pslot = proj_slot<BN, NT>(mp, r);
    stage_B(0);

    constexpr int CG = BN / 4;
    const int cg = tid % CG;
    const int a0 = 4 * (tid / CG);                    // this thread's 4-row block (one pass covers m')
    const int bcol = b0 + 4 * cg;
    const bool mine = a0 < mp && bcol < np;           // n' % 4 == 0: a column group is all in or all out
    const int nrows = mine ? (mp - a0 < 4 ? mp - a0 : 4) : 0;
    float acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;

    for (int i = 0; i < N; ++i) {
        stage_B(i + 1);                      // buffer (i+1)&1 was released by node i-1
        cp_async_wait<1>();                  // B_i has landed (B_{i+1} may be in flight)
        __syncthreads();
        const float* Bb = sm.Bb + (size_t)(i & 1) * mp * BN;
        if (corr) project_strip<BN, NT>(pslot, Bb, sm.Pt, pt, r, sm.Rpart, sm.Rs);
        if (mine) {
                // G_i for this thread's block, straight to registers (32 warps per SM hide the latency)
            float gv[4][4];
            const GT* G = Gp[i];
            if (M.transposed) {
    #pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const float4 x = mine ? ldg4(G + (int64_t)(bcol + j) * mp + a0) : make_float4(0.f, 0.f, 0.f, 0.f);
                    gv[0][j] = x.x; gv[1][j] = x.y; gv[2][j] = x.z; gv[3][j] = x.w;
                }
            } else {
    #pragma unroll
                for (int ii = 0; ii < 4; ++ii) {
                    const float4 x = ii < nrows ? ldg4(G + (int64_t)(a0 + ii) * np + bcol) : make_float4(0.f, 0.f, 0.f, 0.f);
                    gv[ii][0] = x.x; gv[ii][1] = x.y; gv[ii][2] = x.z; gv[ii][3] = x.w;
                }
            }
            float c[4][4];
            if (corr) outer_block<BN>(sm.Pt, pt, sm.Rs, r, a0, cg, c);
            float* Bi = M.B + (int64_t)i * mp * np;
#pragma unroll
            for (int ii = 0; ii < 4; ++ii) {
                if (ii < nrows) {
                const int a = a0 + ii;
                float m[4] = {gv[ii][0], gv[ii][1], gv[ii][2], gv[ii][3]};
                if (corr) {
                    const float4 bv = ld4(Bb + a * BN + 4 * cg);
                    m[0] += bv.x - c[ii][0]; m[1] += bv.y - c[ii][1];
                    m[2] += bv.z - c[ii][2]; m[3] += bv.w - c[ii][3];
                }
                if (M.write_B)
                    st_stream4(Bi + (int64_t)a * np + bcol, m[0], m[1], m[2], m[3]);
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[ii][j] += m[j];
                }
            }
        }
        __syncthreads();                     // buffer i&1 free for node i+2
    }
    cp_async_wait<0>();
    const float invN = 1.0f / static_cast<float>(N);
#pragma unroll
    for (int ii = 0; ii < 4; ++ii)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[ii][j] *= invN;
    bool bad = false;
    if (mine)
#pragma unroll
        for (int ii = 0; ii < 4; ++ii)
            if (ii < nrows) {
                st4(M.Mbar + (int64_t)(a0 + ii) * np + bcol, make_float4(acc[ii][0], acc[ii][1], acc[ii][2], acc[ii][3]));
                bad |= !isfinite(acc[ii][0]) || !isfinite(acc[ii][1]) || !isfinite(acc[ii][2]) || !isfinite(acc[ii][3]);
            }
    flag_nonfinite(bad, M.nonfinite);
    if (!M.lam) return;

    // ---- truncated-basis Approx-Top-r partial sums for this strip ---------------------------
    // Y^T and Yt^T (k x tpitch(m') each, kept by the handle) are read through L1/L2.
    const int k = M.k;
    float* Ms = sm.Bb;                                            // m' x BN (node loop is over)
    if (a0 < mp)
#pragma unroll
        for (int ii = 0; ii < 4; ++ii)
            if (a0 + ii < mp)
                st4(Ms + (a0 + ii) * BN + 4 * cg, bcol < np ? make_float4(acc[ii][0], acc[ii][1], acc[ii][2], acc[ii][3])
                                                            : make_float4(0.f, 0.f, 0.f, 0.f));
    __syncthreads();
    project_strip<BN, NT>(proj_slot<BN, NT>(mp, k), Ms, M.YT, pt, k, sm.Rpart, sm.Ws);   // W = Y^T Mbar_strip (k x BN)
    float rows[4] = {0.f, 0.f, 0.f, 0.f};
    if (mine) {
        float c[4][4];
        outer_block<BN>(M.YtT, pt, sm.Ws, k, a0, cg, c);
#pragma unroll
        for (int ii = 0; ii < 4; ++ii) {
            if (ii < nrows) {
                const int a = a0 + ii;
                const float4 m = ld4(Ms + a * BN + 4 * cg);
                const float4 v = gauss4_fast(M.seed, M.t, static_cast<uint32_t>(a), static_cast<uint32_t>(bcol >> 2),
                                        kTagLambdaV);
                rows[ii] = (m.x - c[ii][0]) * v.x + (m.y - c[ii][1]) * v.y + (m.z - c[ii][2]) * v.z +
                           (m.w - c[ii][3]) * v.w;
            }
        }
    }
    // every lane takes part: the CG lanes of one row block reduce with shuffles
#pragma unroll
    for (int ii = 0; ii < 4; ++ii) {
        float sum = rows[ii];
#pragma unroll
        for (int off = CG / 2; off > 0; off >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
        if (cg == 0 && a0 + ii < mp) M.part[(int64_t)s * mp + a0 + ii] = sum;
    }
}

// ------------------------------------------------------------------------------------------
// K3
// ------------------------------------------------------------------------------------------
template <int BN>
__global__ void __launch_bounds__(NTU) update_kernel_fused(const __grid_constant__ UpdateGroup g) {
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
    stage_cols<BN, NTU>(Ms, M.Mbar, np, mp, b0, np);
    cp_async_commit();
    if (M.compressed) load_transposed<NTU>(Pt, pt, M.P, mp, r);
    cp_async_wait<0>();
    __syncthreads();
    if (M.compressed) {
        project_strip<BN, NTU>(proj_slot<BN, NTU>(mp, r), Ms, Pt, pt, r, Rpart, Rs);
        for (int o = tid; o < r * BN; o += NTU) {
            const int q = o / BN, b = o % BN;
            if (b0 + b < np) M.Rbar[(int64_t)q * np + b0 + b] = Rs[o];
        }
    }
    constexpr int CG = BN / 4;
    constexpr int RPP = 4 * (NTU / CG);
    const int cg = tid % CG, rg = tid / CG;
    const int bcol = b0 + 4 * cg;
    if (bcol >= np) return;
    const float b1 = g.beta1, b2 = g.beta2, lr = g.lr, eps = g.eps;
    const bool adam = g.optimizer == GLR_ADAM;
    for (int a0 = 4 * rg; a0 < mp; a0 += RPP) {
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

template <int BN, int NTH>
size_t rpart_bytes(int r) { return align16((size_t)rpart_floats<BN, NTH>(r) * 4); }

template <int NTH>
size_t rpart_bytes_bn(int BN, int r) {
    switch (BN) {
        case 32: return rpart_bytes<32, NTH>(r);
        case 16: return rpart_bytes<16, NTH>(r);
        case 8: return rpart_bytes<8, NTH>(r);
        default: return rpart_bytes<4, NTH>(r);
    }
}

}  // namespace

size_t stream_smem_bytes(int mp, int r, int k, int BN, int gsize, int transposed, int lam) {
    (void)gsize; (void)transposed;
    const size_t strip = (size_t)mp * BN * 4;
    size_t bytes = 2 * strip;
    bytes += align16((size_t)r * tpitch(mp) * 4) + align16((size_t)r * BN * 4);
    bytes += rpart_bytes_bn<NT>(BN, lam ? (r > k ? r : k) : r);
    if (lam) bytes += align16((size_t)k * BN * 4);
    return bytes;
}

namespace {
__global__ void transpose_pad_kernel(float* dst, int tp, const float* src, int rows, int cols) {
    const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= (int64_t)cols * tp) return;
    const int c = static_cast<int>(e / tp), a = static_cast<int>(e % tp);
    dst[e] = a < rows ? src[(int64_t)a * cols + c] : 0.f;
}
}  // namespace

cudaError_t transpose_pad(float* dst, int tp, const float* src, int rows, int cols, cudaStream_t st) {
    const int64_t total = (int64_t)cols * tp;
    transpose_pad_kernel<<<(unsigned)((total + 255) / 256), 256, 0, st>>>(dst, tp, src, rows, cols);
    return cudaGetLastError();
}

size_t update_smem_bytes(int mp, int r, int BN) {
    return align16((size_t)mp * BN * 4) + align16((size_t)r * tpitch(mp) * 4) + align16((size_t)r * BN * 4) +
           rpart_bytes_bn<NTU>(BN, r);
}

template <int BN, typename GT>
static cudaError_t launch_stream(const StreamGroup& g, size_t smem, cudaStream_t st) {
    {   // per device: set on every call (cheap next to the launch)
        const cudaError_t ea = cudaFuncSetAttribute(stream_kernel<BN, GT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             227 * 1024);
        if (ea != cudaSuccess) return ea;
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
        case 4: return bf ? launch_stream<4, __nv_bfloat16>(g, smem, st) : launch_stream<4, float>(g, smem, st);
        default: return cudaErrorInvalidValue;
    }
}

template <int BN>
static cudaError_t launch_update(const UpdateGroup& g, size_t smem, cudaStream_t st) {
    {   // per device: set on every call (cheap next to the launch)
        const cudaError_t ea = cudaFuncSetAttribute(update_kernel_fused<BN>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             227 * 1024);
        if (ea != cudaSuccess) return ea;
    }
    update_kernel_fused<BN><<<g.total_strips, NTU, smem, st>>>(g);
    return cudaGetLastError();
}

cudaError_t update_group(const UpdateGroup& g, size_t smem, cudaStream_t st) {
    if (g.total_strips <= 0) return cudaSuccess;
    switch (g.BN) {
        case 32: return launch_update<32>(g, smem, st);
        case 16: return launch_update<16>(g, smem, st);
        case 8: return launch_update<8>(g, smem, st);
        case 4: return launch_update<4>(g, smem, st);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace glr
