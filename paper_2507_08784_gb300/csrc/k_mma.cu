// K1 on the tensor cores: the fused compose pass of k_fused.cu with its two rank-r products
// done by warp-level TF32 MMA (mma.sync m16n8k8) in the 3xTF32 form (each fp32 operand x is
// split into x_hi = tf32(x) and x_lo = tf32(x - x_hi); a*b ~ a_hi b_hi + a_hi b_lo + a_lo b_hi,
// accumulated in fp32, which keeps fp32-level accuracy).  The products are tiny (K or N = r),
// so the tensor pipe is far from busy: the point is to replace ~4r FFMA (plus operand loads and
// index arithmetic) per node-element with a handful of MMA instructions per warp.
//
// Per CTA: one strip of 16 columns x all m' (<= 512) rows of one matrix; 16 warps.  A 3-slot
// cp.async ring holds node i's B and G strips while nodes i+1 and i+2 are in flight.
//   node i:  R_i^T (16 x r) = B_i,strip^T P_prev        K = m' split over the warps
//            C (m' x 16)    = P_prev R_i                 K = r
//            M_i = G_i + B_i - C;  B_i <- M_i;  acc += M_i
//   epilogue: Mbar, and for a truncated basis the Approx-Top-r partial sums of
//            (Mbar - Yt (Y^T Mbar)) v_j over the strip (the same two products with Y, Yt).
// Fragment layouts (PTX ISA, mma.m16n8k8 .tf32): with g = lane / 4, t = lane % 4,
//   A (16 x 8): a0 (g, t), a1 (g + 8, t), a2 (g, t + 4), a3 (g + 8, t + 4)
//   B (8 x 8):  b0 (t, g), b1 (t + 4, g)
//   C (16 x 8): c0 (g, 2t), c1 (g, 2t + 1), c2 (g + 8, 2t), c3 (g + 8, 2t + 1)
#include "glr_internal.cuh"

namespace glr {

namespace {

constexpr int T = kMmaThreads;         // 512 threads = 16 warps
constexpr int NW = T / 32;
constexpr int SW = 16;                 // strip width (columns)
constexpr int RP = SW + 8;             // pitch of R / W in shared memory: conflict-free B fragments

__device__ __forceinline__ uint32_t to_tf32(float x) {
    uint32_t r;
    asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x));
    return r;
}
__device__ __forceinline__ void split2(float x, uint32_t& hi, uint32_t& lo) {
    hi = to_tf32(x);
    lo = to_tf32(x - __uint_as_float(hi));
}
__device__ __forceinline__ void mma_tf32(float (&d)[4], const uint32_t (&a)[4], const uint32_t (&b)[2]) {
    asm volatile("mma.sync.aligned.m16n8k8.row.col.f32.tf32.tf32.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
                 "{%0,%1,%2,%3};\n"
                 : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
                 : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}
struct FragA { uint32_t hi[4], lo[4]; };
struct FragB { uint32_t hi[2], lo[2]; };
__device__ __forceinline__ FragA frag_a(float a0, float a1, float a2, float a3) {
    FragA f;
    split2(a0, f.hi[0], f.lo[0]); split2(a1, f.hi[1], f.lo[1]);
    split2(a2, f.hi[2], f.lo[2]); split2(a3, f.hi[3], f.lo[3]);
    return f;
}
__device__ __forceinline__ FragB frag_b(float b0, float b1) {
    FragB f;
    split2(b0, f.hi[0], f.lo[0]); split2(b1, f.hi[1], f.lo[1]);
    return f;
}
// d += a * b in 3xTF32 (small terms first)
__device__ __forceinline__ void mma3(float (&d)[4], const FragA& a, const FragB& b) {
    mma_tf32(d, a.lo, b.hi);
    mma_tf32(d, a.hi, b.lo);
    mma_tf32(d, a.hi, b.hi);
}

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
    const unsigned s = static_cast<unsigned>(__cvta_generic_to_shared(smem));
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(s), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int Pending>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;\n" ::"n"(Pending) : "memory");
}

__host__ __device__ __forceinline__ int up8(int x) { return (x + 7) & ~7; }
__host__ __device__ __forceinline__ int up16(int x) { return (x + 15) & ~15; }
// Pitch of the transposed r x m' copy of P: = 8 (mod 32) so the A-fragment loads hit 32 banks.
__host__ __device__ __forceinline__ int mma_pt(int mp) { return ((mp + 31) & ~31) + 8; }
__host__ __device__ __forceinline__ size_t a16(size_t x) { return (x + 15) & ~size_t(15); }

__device__ __forceinline__ float2 ldg2(const float* p) { return __ldcs(reinterpret_cast<const float2*>(p)); }
__device__ __forceinline__ float2 ldg2(const __nv_bfloat16* p) {
    const __nv_bfloat162 v = __ldcs(reinterpret_cast<const __nv_bfloat162*>(p));
    return __bfloat1622float2(v);
}
template <typename GT> __device__ __forceinline__ float ldg1(const GT* p);
template <> __device__ __forceinline__ float ldg1<float>(const float* p) { return __ldcs(p); }
template <> __device__ __forceinline__ float ldg1<__nv_bfloat16>(const __nv_bfloat16* p) {
    return __bfloat162float(__ldcs(p));
}

// Strips are 16 columns wide; a strip row is 64 bytes = four 16-byte chunks.  B strips are
// stored with chunk c of row a at position c ^ (2 * ((a >> 1) & 1)), which makes the A-fragment
// loads of the R^T product (rows k0 + t, t < 4, columns g and g + 8) hit 32 distinct banks.
__device__ __forceinline__ int sw_elem(int a, int c) {
    return a * SW + 4 * ((c >> 2) ^ (((a >> 1) & 1) << 1)) + (c & 3);
}

// R^T (16 x RQ) = S^T P: S the m' x 16 swizzled strip, P given transposed (Pt, RQ x pt, rows
// q >= r zero), K = m' split over the warps (warp w takes k-steps w, w + NW, ...).  The warp
// partials are added in warp order into out (RQ x RP).  Ends with __syncthreads.
template <bool GLOBAL_P>
__device__ __forceinline__ void rt_product(const float* S, const float* Pt, int pt, int mp16, int RQ, float* part,
                                           float* out) {
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
    const int nq = RQ / 8;             // 1..4 n-tiles over q
    float d[4][4];
#pragma unroll
    for (int j = 0; j < 4; ++j)
#pragma unroll
        for (int e = 0; e < 4; ++e) d[j][e] = 0.f;
    // A fragment addresses: rows k0 + t and k0 + t + 4 share the swizzle of row t (k0 % 8 == 0)
    const int swt = ((t >> 1) & 1) << 1;
    const int oa0 = t * SW + 4 * ((g >> 2) ^ swt) + (g & 3);          // (k0 + t, g)
    const int oa1 = t * SW + 4 * (((g >> 2) + 2) ^ swt) + (g & 3);    // (k0 + t, g + 8)
    const float* sk = S + (w * 8) * SW;
    const float* pk = Pt + g * pt + w * 8 + t;
    const int kstep = NW * 8;
    for (int k0 = w * 8; k0 < mp16; k0 += kstep, sk += kstep * SW, pk += kstep) {
        const FragA A = frag_a(sk[oa0], sk[oa1], sk[oa0 + 4 * SW], sk[oa1 + 4 * SW]);
#pragma unroll
        for (int nt = 0; nt < 4; ++nt) {
            if (nt < nq) {
                const float* prow = pk + nt * 8 * pt;
                const FragB B = GLOBAL_P ? frag_b(__ldg(prow), __ldg(prow + 4)) : frag_b(prow[0], prow[4]);
                mma3(d[nt], A, B);
            }
        }
    }
    float* mine = part + w * (RQ * SW) + (2 * t) * SW + g;
#pragma unroll
    for (int nt = 0; nt < 4; ++nt) {
        if (nt < nq) {
            float* m = mine + nt * 8 * SW;
            m[0] = d[nt][0];
            m[SW] = d[nt][1];
            m[8] = d[nt][2];
            m[SW + 8] = d[nt][3];
        }
    }
    __syncthreads();
    for (int o = threadIdx.x; o < RQ * SW; o += T) {
        const float* pp = part + o;
        float acc = 0.f;
#pragma unroll 4
        for (int ww = 0; ww < NW; ++ww, pp += RQ * SW) acc += *pp;
        out[(o / SW) * RP + (o % SW)] = acc;
    }
    __syncthreads();
}

// C fragments of P R for m-tile m0 (rows m0..m0+15) and the two 8-column tiles: c[nt][e],
// K = RQ (columns of P, zero beyond r).  R is RQ x RP.
template <bool GLOBAL_P>
__device__ __forceinline__ void c_product(const float* Pt, int pt, const float* R, int RQ, int m0, float (&c)[2][4]) {
    const int lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
#pragma unroll
    for (int nt = 0; nt < 2; ++nt)
#pragma unroll
        for (int e = 0; e < 4; ++e) c[nt][e] = 0.f;
    const float* p0 = Pt + t * pt + m0 + g;
    const float* rr = R + t * RP + g;
    for (int kq = 0; kq < RQ; kq += 8, p0 += 8 * pt, rr += 8 * RP) {
        const float* p1 = p0 + 4 * pt;
        const FragA A = GLOBAL_P ? frag_a(__ldg(p0), __ldg(p0 + 8), __ldg(p1), __ldg(p1 + 8))
                                 : frag_a(p0[0], p0[8], p1[0], p1[8]);
#pragma unroll
        for (int nt = 0; nt < 2; ++nt) {
            const FragB B = frag_b(rr[nt * 8], rr[4 * RP + nt * 8]);
            mma3(c[nt], A, B);
        }
    }
}

// Ring stage layout: [B strip: mp16 x 16 fp32, swizzled][G strip: mp16 x 16 (gradient dtype),
// or 16 x gpt when G is read transposed (m > n)].
__host__ __device__ __forceinline__ size_t stage_b_bytes(int mp16) { return (size_t)mp16 * SW * 4; }
__host__ __device__ __forceinline__ int g_tpitch(int mp16, int gsize) { return mp16 + 16 / gsize; }
__host__ __device__ __forceinline__ size_t stage_g_bytes(int mp16, int gsize, int transposed) {
    return a16(transposed ? (size_t)SW * g_tpitch(mp16, gsize) * gsize : (size_t)mp16 * SW * gsize);
}

template <typename GT>
__global__ void __launch_bounds__(T, 1) stream_mma_kernel(const __grid_constant__ StreamGroup g) {
    extern __shared__ __align__(16) unsigned char smem[];
    int mi = 0;
    while (mi + 1 < g.nmat && blockIdx.x >= static_cast<unsigned>(g.mat[mi + 1].strip0)) ++mi;
    const StreamMat& M = g.mat[mi];
    const int s = blockIdx.x - M.strip0;
    const int b0 = s * SW;
    const int mp = M.mp, np = M.np, r = M.r, N = M.N;
    const int mp16 = up16(mp), RQ = up8(r), pt = mma_pt(mp);
    const int tid = threadIdx.x, w = tid >> 5, lane = tid & 31, gg = lane >> 2, t = lane & 3;
    constexpr int GS = sizeof(GT);
    constexpr int EPC = 16 / GS;                      // gradient elements per 16-byte chunk
    const bool trans = M.transposed != 0;
    const int gpt = g_tpitch(mp16, GS);
    const size_t sb = stage_b_bytes(mp16), sg = stage_g_bytes(mp16, GS, trans), stage = sb + sg;
    unsigned char* ring = smem;
    float* Pt = reinterpret_cast<float*>(smem + 3 * stage);
    float* Rs = Pt + a16((size_t)RQ * pt * 4) / 4;
    float* Rpart = Rs + a16((size_t)32 * RP * 4) / 4;
    const bool corr = !M.e_zero;
    const GT* const* Gp = reinterpret_cast<const GT* const*>(g.G + M.g_off);

    // ---- per-thread staging plan (fixed for all nodes): up to 4 chunks of B and 4 of G -------
    int boff[4], bdst[4], goff[4], gdst[4];
    unsigned bmask = 0, gmask = 0;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const int c = tid + j * T;                    // B chunk: row a, 4 columns
        const int a = c >> 2, ch = c & 3, col = b0 + 4 * ch;
        boff[j] = a * np + col;
        bdst[j] = a * SW + 4 * (ch ^ (((a >> 1) & 1) << 1));
        if (c < mp * 4) {
            if (col < np) bmask |= 1u << j;
            else for (int st = 0; st < 3; ++st)       // columns past n': zero once in every slot
                *reinterpret_cast<float4*>(reinterpret_cast<float*>(ring + st * stage) + bdst[j]) =
                    make_float4(0.f, 0.f, 0.f, 0.f);
        }
        if (trans) {                                  // G rows b0 + bb, m' contiguous elements
            const int cpr = mp / EPC;
            const int bb = c / cpr, gch = c % cpr;
            goff[j] = (b0 + bb) * mp + gch * EPC;
            gdst[j] = bb * gpt + gch * EPC;
            if (c < SW * cpr) {
                if (b0 + bb < np) gmask |= 1u << j;
                else for (int st = 0; st < 3; ++st)
                    *reinterpret_cast<float4*>(reinterpret_cast<GT*>(ring + st * stage + sb) + gdst[j]) =
                        make_float4(0.f, 0.f, 0.f, 0.f);
            }
        } else {                                      // G rows a, SW columns
            constexpr int CPR = SW / EPC;
            const int ga = c / CPR, gch = c % CPR, gcol = b0 + gch * EPC;
            goff[j] = ga * np + gcol;
            gdst[j] = ga * SW + gch * EPC;
            if (c < mp * CPR) {
                if (gcol < np) gmask |= 1u << j;
                else for (int st = 0; st < 3; ++st)
                    *reinterpret_cast<float4*>(reinterpret_cast<GT*>(ring + st * stage + sb) + gdst[j]) =
                        make_float4(0.f, 0.f, 0.f, 0.f);
            }
        }
    }
    // rows mp..mp16 of every B strip and every (non-transposed) G strip stay zero
    for (int a = mp + (tid >> 4); a < mp16; a += T / SW) {
        const int c = tid & (SW - 1);
#pragma unroll
        for (int st = 0; st < 3; ++st) {
            reinterpret_cast<float*>(ring + st * stage)[a * SW + c] = 0.f;
            if (!trans) reinterpret_cast<GT*>(ring + st * stage + sb)[a * SW + c] = GT(0.f);
        }
    }
    if (corr)
        for (int q = 0; q < RQ; ++q)
            for (int a = tid; a < pt; a += T) Pt[q * pt + a] = (q < r && a < mp) ? M.Pprev[a * r + q] : 0.f;

    auto stage_node = [&](int i) {
        if (i < N) {
            unsigned char* base = ring + (size_t)(i % 3) * stage;
            if (corr) {
                float* dst = reinterpret_cast<float*>(base);
                const float* src = M.B + (int64_t)i * mp * np;
#pragma unroll
                for (int j = 0; j < 4; ++j)
                    if (bmask & (1u << j)) cp_async16(dst + bdst[j], src + boff[j]);
            }
            GT* dst = reinterpret_cast<GT*>(base + sb);
            const GT* src = Gp[i];
#pragma unroll
            for (int j = 0; j < 4; ++j)
                if (gmask & (1u << j)) cp_async16(dst + gdst[j], src + goff[j]);
        }
        cp_async_commit();
    };
    stage_node(0);
    stage_node(1);

    // ---- per-lane fragment geometry (fixed for all nodes) ------------------------------------
    const int ntiles_m = mp16 / 16;
    const int swz = ((gg >> 1) & 1) << 1;             // swizzle of rows m0 + gg (+8): m0 % 16 == 0
    int soff[2], goffc[2], colv[2];                  // per n-tile: swizzled column offset, G column, global column
#pragma unroll
    for (int nt = 0; nt < 2; ++nt) {
        const int bl = nt * 8 + 2 * t;
        soff[nt] = 4 * ((bl >> 2) ^ swz) + (bl & 3);
        goffc[nt] = trans ? bl * gpt : bl;
        colv[nt] = b0 + bl;
    }
    int rowoff[2][2];                                 // global row offsets a * n' of (u, h)
#pragma unroll
    for (int u = 0; u < 2; ++u)
#pragma unroll
        for (int h = 0; h < 2; ++h) rowoff[u][h] = ((w + u * NW) * 16 + gg + 8 * h) * np;

    float acc[2][2][4];
#pragma unroll
    for (int u = 0; u < 2; ++u)
#pragma unroll
        for (int nt = 0; nt < 2; ++nt)
#pragma unroll
            for (int e = 0; e < 4; ++e) acc[u][nt][e] = 0.f;

    for (int i = 0; i < N; ++i) {
        stage_node(i + 2);                 // ring slot (i+2)%3 was released by node i-1
        cp_async_wait<2>();                // node i has landed; nodes i+1, i+2 may be in flight
        __syncthreads();
        const unsigned char* base = ring + (size_t)(i % 3) * stage;
        const float* S = reinterpret_cast<const float*>(base);
        const GT* Gs = reinterpret_cast<const GT*>(base + sb);
        if (corr) rt_product<false>(S, Pt, pt, mp16, RQ, Rpart, Rs);
        float* Bi = M.B + (int64_t)i * mp * np;
#pragma unroll
        for (int u = 0; u < 2; ++u) {
            const int mt = w + u * NW;
            if (mt < ntiles_m) {
                const int m0 = mt * 16;
                float c[2][4];
                if (corr) c_product<false>(Pt, pt, Rs, RQ, m0, c);
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int a = m0 + gg + 8 * h;
                    if (a < mp) {
                        const float* Sa = S + a * SW;
                        const GT* Ga = trans ? Gs + a : Gs + a * SW;
                        float* Ba = Bi + rowoff[u][h];
#pragma unroll
                        for (int nt = 0; nt < 2; ++nt) {
                            if (colv[nt] < np) {
                                const GT* gp = Ga + goffc[nt];
                                float m0v = static_cast<float>(gp[0]);
                                float m1v = static_cast<float>(trans ? gp[gpt] : gp[1]);
                                if (corr) {
                                    const float2 bv = *reinterpret_cast<const float2*>(Sa + soff[nt]);
                                    m0v += bv.x - c[nt][2 * h];
                                    m1v += bv.y - c[nt][2 * h + 1];
                                }
                                if (M.write_B) __stcs(reinterpret_cast<float2*>(Ba + colv[nt]), make_float2(m0v, m1v));
                                acc[u][nt][2 * h] += m0v;
                                acc[u][nt][2 * h + 1] += m1v;
                            }
                        }
                    }
                }
            }
        }
        __syncthreads();
    }
    cp_async_wait<0>();
    const float invN = 1.0f / static_cast<float>(N);
#pragma unroll
    for (int u = 0; u < 2; ++u)
#pragma unroll
        for (int nt = 0; nt < 2; ++nt)
#pragma unroll
            for (int e = 0; e < 4; ++e) acc[u][nt][e] *= invN;
#pragma unroll
    for (int u = 0; u < 2; ++u) {
        const int mt = w + u * NW;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int a = mt * 16 + gg + 8 * h;
            if (mt < ntiles_m && a < mp)
#pragma unroll
                for (int nt = 0; nt < 2; ++nt)
                    if (colv[nt] < np)
                        *reinterpret_cast<float2*>(M.Mbar + rowoff[u][h] + colv[nt]) =
                            make_float2(acc[u][nt][2 * h], acc[u][nt][2 * h + 1]);
        }
    }
    if (!M.lam) return;

    // ---- truncated-basis Approx-Top-r partial sums: (Mbar - Yt (Y^T Mbar)) v_j ------------------
    const int k = M.k, KQ = up8(k), tp = transposed_pitch(mp);
    float* Ms = reinterpret_cast<float*>(ring);              // Mbar strip (swizzled, rows >= mp zero)
    float* Wp = reinterpret_cast<float*>(ring + stage);      // warp partials of W^T (ring slots 1-2)
    float* Ws = Rs;                                          // W = Y^T Mbar_strip (KQ x RP)
#pragma unroll
    for (int u = 0; u < 2; ++u) {
        const int mt = w + u * NW;
        if (mt < ntiles_m) {
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int a = mt * 16 + gg + 8 * h;
#pragma unroll
                for (int nt = 0; nt < 2; ++nt)
                    *reinterpret_cast<float2*>(Ms + a * SW + soff[nt]) =
                        colv[nt] < np && a < mp ? make_float2(acc[u][nt][2 * h], acc[u][nt][2 * h + 1])
                                                : make_float2(0.f, 0.f);
            }
        }
    }
    __syncthreads();
    rt_product<true>(Ms, M.YT, tp, mp16, KQ, Wp, Ws);        // W^T = Mbar_strip^T Y
    float rows[2][2] = {{0.f, 0.f}, {0.f, 0.f}};
#pragma unroll
    for (int u = 0; u < 2; ++u) {
        const int mt = w + u * NW;
        const int m0 = mt * 16;
        float c[2][4] = {};
        if (mt < ntiles_m) c_product<true>(M.YtT, tp, Ws, KQ, m0, c);
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int a = m0 + gg + 8 * h;
            // the 32 lanes draw the 32 distinct quads (row gg, quad lane & 3) of this row block;
            // each lane then fetches the two values of its own columns
            const float4 vq = gauss4(M.seed, M.t, static_cast<uint32_t>(a), static_cast<uint32_t>((b0 >> 2) + t),
                                     kTagLambdaV);
#pragma unroll
            for (int nt = 0; nt < 2; ++nt) {
                const int src = (lane & ~3) | (nt * 2 + (t >> 1));
                const float vx = __shfl_sync(0xffffffffu, vq.x, src), vy = __shfl_sync(0xffffffffu, vq.y, src);
                const float vz = __shfl_sync(0xffffffffu, vq.z, src), vw = __shfl_sync(0xffffffffu, vq.w, src);
                const bool hi = (t & 1) != 0;            // columns 2, 3 of the quad
                const float v0 = hi ? vz : vx, v1 = hi ? vw : vy;
                if (mt < ntiles_m && a < mp && colv[nt] < np) {
                    const float2 mv = *reinterpret_cast<const float2*>(Ms + a * SW + soff[nt]);
                    rows[u][h] += (mv.x - c[nt][2 * h]) * v0 + (mv.y - c[nt][2 * h + 1]) * v1;
                }
            }
        }
    }
    // the 4 lanes of a group (t = 0..3) hold one row's partial sums
#pragma unroll
    for (int u = 0; u < 2; ++u)
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            float v = rows[u][h];
            v += __shfl_xor_sync(0xffffffffu, v, 1);
            v += __shfl_xor_sync(0xffffffffu, v, 2);
            const int mt = w + u * NW;
            const int a = mt * 16 + gg + 8 * h;
            if (t == 0 && mt < ntiles_m && a < mp) M.part[(int64_t)s * mp + a] = v;
        }
}

}  // namespace

bool mma_stream_eligible(int mp, int np, int r, int k, int lam, int transposed, int gsize) {
    if (mp > kMmaMaxRows || r > 16 || (lam && (k > 32 || k % 8 != 0))) return false;
    if (np % 4 != 0 || (transposed && mp % 8 != 0)) return false;   // 16-byte chunks of G rows
    return mma_stream_smem_bytes(mp, r, k, lam, gsize, transposed) <= 227 * 1024;
}

size_t mma_stream_smem_bytes(int mp, int r, int k, int lam, int gsize, int transposed) {
    const int mp16 = up16(mp), RQ = up8(r), pt = mma_pt(mp), KQ = up8(k);
    const size_t stage = stage_b_bytes(mp16) + stage_g_bytes(mp16, gsize, transposed);
    if (lam && (size_t)NW * KQ * SW * 4 > 2 * stage) return ~size_t(0);   // W partials use ring slots 1-2
    return 3 * stage + a16((size_t)RQ * pt * 4) + a16((size_t)32 * RP * 4) + a16((size_t)NW * RQ * SW * 4);
}

template <typename GT>
static cudaError_t launch_mma(const StreamGroup& g, size_t smem, cudaStream_t st) {
    static bool set = false;
    if (!set) {
        cudaError_t e = cudaFuncSetAttribute(stream_mma_kernel<GT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             227 * 1024);
        if (e != cudaSuccess) return e;
        set = true;
    }
    stream_mma_kernel<GT><<<g.total_strips, T, smem, st>>>(g);
    return cudaGetLastError();
}

cudaError_t stream_group_mma(const StreamGroup& g, size_t smem, cudaStream_t st) {
    if (g.total_strips <= 0) return cudaSuccess;
    return g.grad_dtype == GLR_BF16 ? launch_mma<__nv_bfloat16>(g, smem, st) : launch_mma<float>(g, smem, st);
}

}  // namespace glr
