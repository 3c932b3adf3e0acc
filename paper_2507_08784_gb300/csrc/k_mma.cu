// K1 on the tensor cores: the fused compose pass with its two rank-r products done by warp-level
// TF32 MMA (mma.sync m16n8k8) in the 3xTF32 form (each fp32 operand x is split into x_hi and
// x_lo; a*b ~ a_hi b_hi + a_hi b_lo + a_lo b_hi, accumulated in fp32, which keeps fp32-level
// accuracy).  The products are tiny (K or N = r), so the tensor pipe is far from busy: the point
// is to replace ~2r FFMA (plus operand loads and index arithmetic) per node-element with a few
// MMA instructions per warp.
//
// Per CTA: one strip of 16 columns x all m' (<= 512) rows of one matrix; 16 warps.  A 3-slot
// ring holds node i's B and G strips while nodes i+1 and i+2 are in flight; after the last node
// the two free slots receive Y and Yt for the truncated-basis lambda epilogue.  The ring is
// filled by the Tensor Memory Accelerator (one thread issues a 2-D/3-D tile copy per operand and
// node, completion counted on a per-slot mbarrier) when G is read in its stored orientation, and
// by per-thread 16-byte cp.async otherwise (G read transposed, m > n).
//   node i:  R_i^T (16 x r) = B_i,strip^T P_prev        K = m' split over the warps
//            C (m' x 16)    = P_prev R_i                 K = r
//            M_i = G_i + (B_i - C);  B_i <- M_i;  acc += M_i
//   epilogue: Mbar, and for a truncated basis the Approx-Top-r partial sums of
//            (Mbar - Yt (Y^T Mbar)) v_j over the strip (the same two products with Y, Yt).
//
// Fragment layouts (PTX ISA, mma.m16n8k8 .tf32): with g = lane / 4, t = lane % 4,
//   A (16 x 8): a0 (g, t), a1 (g + 8, t), a2 (g, t + 4), a3 (g + 8, t + 4)
//   B (8 x 8):  b0 (t, g), b1 (t + 4, g)
//   C (16 x 8): c0 (g, 2t), c1 (g, 2t + 1), c2 (g + 8, 2t), c3 (g + 8, 2t + 1)
// Both products are computed transposed, with M = the strip's 16 columns, and their indices are
// relabelled so that one lane owns the same four elements of every operand.  With
// rho(t) = (t % 2) + 4 (t / 2), in each 8-row group the lane owns rows rho(t), rho(t) + 2 and
// strip columns 2g, 2g + 1:
//   e0 = (rho, 2g)   e1 = (rho, 2g + 1)   e2 = (rho + 2, 2g)   e3 = (rho + 2, 2g + 1).
//   R^T = B^T P   (M = columns, K = rows, N = q): M index m <-> column 2 (m % 8) + m / 8, K index
//                 t <-> row rho(t), t + 4 <-> rho(t) + 2.  A fragment = (e0, e1, e2, e3); B
//                 fragment P(rho, q), P(rho + 2, q).
//   C^T = R^T P^T (M = columns, K = q, N = rows): N index n <-> row prow(n) = rho(n / 2) +
//                 2 (n % 2), K index k <-> q = 2 (k % 4) + k / 4.  C fragment = (e0, e2, e1, e3);
//                 its A fragment is the R^T C fragment in the order (c0, c2, c1, c3); B fragment
//                 P(prow(g), 2t), P(prow(g), 2t + 1).
// Sums over K are order-free, so the relabelling changes nothing but the rounding order.  The
// row labels make the lane's 8-byte loads from the 64-byte-swizzled strips conflict-free.  B is
// read from shared memory once per node for both products, P's fragments are loaded once per
// strip into registers, and no operand is re-staged between the products.
#include <cuda.h>

#include "glr_internal.cuh"

namespace glr {

namespace {

constexpr int T = kMmaThreads;         // 512 threads = 16 warps
constexpr int NW = T / 32;
constexpr int SW = 16;                 // strip width (columns)
constexpr int GPW_MAX = 64 / NW;       // row groups per warp for r <= 8 (m' <= 512)

// x ~ hi + lo with hi = x rounded to the nearest TF32 value (ties away from zero: add half a unit
// of the 13 dropped mantissa bits, then clear them) and lo = the TF32 truncation of the exact
// remainder x - hi; |x - hi| <= 2^-11 |x|, so truncating it costs at most 2^-21 |x|.  Integer
// operations on the bit pattern; finite inputs below the largest binade.
__device__ __forceinline__ void split2(float x, uint32_t& hi, uint32_t& lo) {
    hi = (__float_as_uint(x) + 0x1000u) & 0xffffe000u;
    lo = __float_as_uint(x - __uint_as_float(hi)) & 0xffffe000u;
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

__device__ __forceinline__ void cp_async16(uint32_t saddr, const void* gmem) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(saddr), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int Pending>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;\n" ::"n"(Pending) : "memory");
}

// ---- Tensor Memory Accelerator and mbarrier ------------------------------------------------
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
// Waits for the phase of parity `parity` to complete, polling with short sleeps in between; after
// about a second (16 M polls of >= 64 ns) it gives up and returns false.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
    uint32_t ns = 16;
    for (int it = 0; it < 16000000; ++it) {
        uint32_t done;
        asm volatile("{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
                     : "=r"(done) : "r"(bar), "r"(parity) : "memory");
        if (done) return true;
        __nanosleep(ns);                   // back off (16 .. 64 ns) so waiting warps leave the issue slots
        ns = ns < 64 ? 2 * ns : 64;
    }
    return false;
}
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar) {
    asm volatile("cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
                 ::"r"(dst), "l"(map), "r"(x), "r"(y), "r"(bar) : "memory");
}
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* map, int x, int y, int z, uint32_t bar) {
    asm volatile("cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], [%5];"
                 ::"r"(dst), "l"(map), "r"(x), "r"(y), "r"(z), "r"(bar) : "memory");
}
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                 ::"r"(dst), "l"(src), "r"(bytes), "r"(bar) : "memory");
}

__host__ __device__ __forceinline__ int up8(int x) { return (x + 7) & ~7; }
__host__ __device__ __forceinline__ int up16(int x) { return (x + 15) & ~15; }
__host__ __device__ __forceinline__ size_t a16(size_t x) { return (x + 15) & ~size_t(15); }
__host__ __device__ __forceinline__ size_t a1k(size_t x) { return (x + 1023) & ~size_t(1023); }

// Strip layouts in shared memory (both staging paths write the same ones):
//   fp32 strips (B, and G when it is fp32): 64-byte rows, 16-byte chunk c of row a at position
//     c ^ ((a >> 1) & 3)  (the Tensor Memory Accelerator's 64-byte swizzle)
//   bf16 G strips: 32-byte rows, chunk c of row a at c ^ ((a >> 2) & 1)  (its 32-byte swizzle)
//   G read transposed (cp.async only): 16 rows (strip columns) of gpt elements.
__device__ __forceinline__ int sw64(int a, int c) { return a * SW + 4 * ((c >> 2) ^ ((a >> 1) & 3)) + (c & 3); }
__device__ __forceinline__ int sw32(int a, int c) { return a * SW + 8 * ((c >> 3) ^ ((a >> 2) & 1)) + (c & 7); }

// Tile copies: up8(m') rows in nbox boxes of box_rows rows (a box has at most 256 rows).
__host__ __device__ __forceinline__ int tma_nbox(int mp) { return (up8(mp) + 255) / 256; }
__host__ __device__ __forceinline__ int tma_box_rows(int mp) {
    const int nb = tma_nbox(mp);
    return up8((up8(mp) + nb - 1) / nb);
}
// Rows held by a slot, and the slot's B and G regions (TMA regions start on 1024-byte bounds).
__host__ __device__ __forceinline__ int slot_rows(int mp, bool tma) {
    return tma ? tma_nbox(mp) * tma_box_rows(mp) : up16(mp);
}
__host__ __device__ __forceinline__ int g_tpitch(int mp16, int gsize) { return mp16 + 16 / gsize; }
__host__ __device__ __forceinline__ size_t stage_b_bytes(int rows, bool tma) {
    return tma ? a1k((size_t)rows * SW * 4) : (size_t)rows * SW * 4;
}
__host__ __device__ __forceinline__ size_t stage_g_bytes(int mp, int rows, int gsize, int transposed, bool tma) {
    if (transposed) return a16((size_t)SW * g_tpitch(up16(mp), gsize) * gsize);
    return tma ? a1k((size_t)rows * SW * gsize) : (size_t)rows * SW * gsize;
}
// Warp partials of a 16 x (8 NT) product: one float4 per lane and n-tile; the pitch between
// warps is = 8 (mod 32) floats so the quarter-sums of the reduction hit distinct banks.
__host__ __device__ __forceinline__ int part_pitch(int NT) { return NT * 128 + 8; }
__host__ __device__ __forceinline__ bool lam_partials_in_slot(int KT, size_t stage) {
    return KT > 0 && (size_t)NW * part_pitch(KT) * 4 <= stage;
}

// tot[o] = sum over the NW warps of part[w][o], o < NT * 128, in a fixed order: four threads
// per output each add the warps w = q, q + 4, q + 8, ... in turn, then two xor-shuffles.
__device__ __forceinline__ void reduce_warps(const float* part, int pitch, int NT, float* tot) {
    const int nout = NT * 128;
    for (int base = 0; base < nout * 4; base += T) {
        const int idx = base + threadIdx.x, o = idx >> 2, q = idx & 3;
        float a = 0.f;
        if (o < nout) {
            const float* p = part + q * pitch + o;
#pragma unroll
            for (int ww = 0; ww < NW / 4; ++ww) a += p[4 * ww * pitch];
        }
        a += __shfl_xor_sync(0xffffffffu, a, 1);
        a += __shfl_xor_sync(0xffffffffu, a, 2);
        if (q == 0 && o < nout) tot[o] = a;
    }
}

template <typename GT> struct GradPair;
template <> struct GradPair<float> {
    // (row a, columns c, c + 1) of a 64-byte-swizzled fp32 strip, c even
    static __device__ __forceinline__ float2 row(const float* Gs, int a, int c) {
        return *reinterpret_cast<const float2*>(Gs + sw64(a, c));
    }
    // the same at a precomputed swizzled offset (Lane::sb0 / sb1 + kGroupStride j)
    static __device__ __forceinline__ float2 at(const float* Gs, int off, int, int) {
        return *reinterpret_cast<const float2*>(Gs + off);
    }
};
template <> struct GradPair<__nv_bfloat16> {
    static __device__ __forceinline__ float2 row(const __nv_bfloat16* Gs, int a, int c) {
        return __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(Gs + sw32(a, c)));
    }
    static __device__ __forceinline__ float2 at(const __nv_bfloat16* Gs, int, int offg, int) {
        return __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(Gs + offg));
    }
};

// ---- the pieces of a strip's work, shared by the kernels below ------------------------------
// Lane geometry (see the header): warp w, lane = 4 gg + t, rows rho and rho + 2 of each group,
// columns c2 and c2 + 1; prow is the row of the C^T = R^T P^T B fragment.
// The lane's rows in row group G8 = w + NW j are ra = 8 G8 + rho and rb = ra + 2; since 8 G8 is a
// multiple of 8 and rho + 2 < 8, the swizzle terms (ra >> 1) & 3 and (ra >> 2) & 1 depend on rho
// only, so a row's swizzled offset in a strip is a lane constant plus 128 G8 = 128 w + 2048 j:
// sb0 / sb1 for the 64-byte swizzle (B, fp32 G), sg0 / sg1 for the 32-byte one (bf16 G), in
// elements.
struct Lane {
    int tid, w, lane, gg, t, rho, prow, c2;
    int sb0, sb1, sg0, sg1;
};
__device__ __forceinline__ Lane lane_geometry() {
    Lane L;
    L.tid = threadIdx.x; L.w = L.tid >> 5; L.lane = L.tid & 31; L.gg = L.lane >> 2; L.t = L.lane & 3;
    L.rho = (L.t & 1) + 4 * (L.t >> 1);
    L.prow = ((L.gg >> 1) & 1) + 4 * (L.gg >> 2) + 2 * (L.gg & 1);
    L.c2 = 2 * L.gg;
    const int r0 = L.rho, r1 = L.rho + 2, base = 128 * L.w;
    L.sb0 = base + SW * r0 + 4 * ((L.c2 >> 2) ^ ((r0 >> 1) & 3)) + (L.c2 & 3);
    L.sb1 = base + SW * r1 + 4 * ((L.c2 >> 2) ^ ((r1 >> 1) & 3)) + (L.c2 & 3);
    L.sg0 = base + SW * r0 + 8 * ((L.c2 >> 3) ^ ((r0 >> 2) & 1)) + (L.c2 & 7);
    L.sg1 = base + SW * r1 + 8 * ((L.c2 >> 3) ^ ((r1 >> 2) & 1)) + (L.c2 & 7);
    return L;
}
constexpr int kGroupStride = 128 * NW;   // elements between a lane's rows in groups j and j + 1

// P_prev fragments of the lane's row groups (zero where E = 0, past m' or past r).
template <int NQ, int GPW>
__device__ __forceinline__ void load_pfrags(const float* P, int mp, int r, int ng, bool use, const Lane& L,
                                            FragB (&prt)[GPW][NQ], FragB (&pcb)[GPW][NQ]) {
#pragma unroll
    for (int j = 0; j < GPW; ++j) {
        const int G8 = L.w + NW * j;
        const int ra = 8 * G8 + L.rho, rc = 8 * G8 + L.prow;
        const bool u = use && G8 < ng;
#pragma unroll
        for (int nt = 0; nt < NQ; ++nt) {
            const int q = 8 * nt + L.gg, q0 = 8 * nt + 2 * L.t;
            prt[j][nt] = frag_b(u && q < r && ra < mp ? __ldg(P + ra * r + q) : 0.f,
                                u && q < r && ra + 2 < mp ? __ldg(P + (ra + 2) * r + q) : 0.f);
            pcb[j][nt] = frag_b(u && q0 < r && rc < mp ? __ldg(P + rc * r + q0) : 0.f,
                                u && q0 + 1 < r && rc < mp ? __ldg(P + rc * r + q0 + 1) : 0.f);
        }
    }
}

// One node on a strip resident in shared memory (S: B strip, Gs: G strip, transposed with pitch
// gpt when trans): warp partials of R_i^T = B_i^T P_prev, their reduction, and the combine
// M_i = G_i + (B_i - P_prev R_i) with B_i <- M_i (Bi: node i's B at the strip's first column)
// and acc += M_i.  Contains two barriers when corr, one otherwise; the caller's barrier before
// it made the strip readable.
template <typename GT, int NQ, int GPW>
__device__ __forceinline__ void compose_node(const float* S, const GT* Gs, bool trans, int gpt, bool corr,
                                             const FragB (&prt)[GPW][NQ], const FragB (&pcb)[GPW][NQ],
                                             float (&acc)[GPW][4], float* part, int pitch, float* tot, float* Bi,
                                             int mp, int np, int ng, bool write_B, bool colok, const Lane& L) {
    if (corr) {                            // warp partials of R_i^T = B_i^T P_prev
        // one accumulator per row group, so the groups' MMA chains run side by side
        float d[GPW][NQ][4];
#pragma unroll
        for (int j = 0; j < GPW; ++j)
#pragma unroll
            for (int nt = 0; nt < NQ; ++nt)
#pragma unroll
                for (int e = 0; e < 4; ++e) d[j][nt][e] = 0.f;
#pragma unroll
        for (int j = 0; j < GPW; ++j) {
            const int G8 = L.w + NW * j;
            if (G8 < ng) {
                const float2 x0 = *reinterpret_cast<const float2*>(S + L.sb0 + kGroupStride * j);
                const float2 x1 = *reinterpret_cast<const float2*>(S + L.sb1 + kGroupStride * j);
                const FragA A = frag_a(x0.x, x0.y, x1.x, x1.y);
#pragma unroll
                for (int nt = 0; nt < NQ; ++nt) mma3(d[j][nt], A, prt[j][nt]);
            }
        }
#pragma unroll
        for (int nt = 0; nt < NQ; ++nt) {
            float4 v = make_float4(d[0][nt][0], d[0][nt][1], d[0][nt][2], d[0][nt][3]);
#pragma unroll
            for (int j = 1; j < GPW; ++j) {
                v.x += d[j][nt][0]; v.y += d[j][nt][1]; v.z += d[j][nt][2]; v.w += d[j][nt][3];
            }
            *reinterpret_cast<float4*>(part + L.w * pitch + (nt * 32 + L.lane) * 4) = v;
        }
    }
    __syncthreads();
    FragA RA[NQ];
    if (corr) {
        reduce_warps(part, pitch, NQ, tot);
        __syncthreads();
#pragma unroll
        for (int nt = 0; nt < NQ; ++nt) {
            const float4 R = *reinterpret_cast<const float4*>(tot + (nt * 32 + L.lane) * 4);
            RA[nt] = frag_a(R.x, R.z, R.y, R.w);
        }
    }
    // the lane's element offsets from node i's strip base Bi (warp-uniform): its first row of
    // group 0 and column c2, the step to group j's rows (128 rows) and to row rb (2 rows); a node
    // holds fewer than 2^31 elements, so 32 bits suffice and the stores address uniform base +
    // lane offset
    const uint32_t orow = static_cast<uint32_t>((8 * L.w + L.rho) * np + L.c2);
    const uint32_t jstep = static_cast<uint32_t>(8 * NW * np), rstep = static_cast<uint32_t>(2 * np);
#pragma unroll
    for (int j = 0; j < GPW; ++j) {
        const int G8 = L.w + NW * j;
        if (G8 < ng) {
            const int ra = 8 * G8 + L.rho, rb = ra + 2;
            float c[4] = {0.f, 0.f, 0.f, 0.f};
            float2 x0 = make_float2(0.f, 0.f), x1 = make_float2(0.f, 0.f);
            if (corr) {
#pragma unroll
                for (int nt = 0; nt < NQ; ++nt) mma3(c, RA[nt], pcb[j][nt]);
                x0 = *reinterpret_cast<const float2*>(S + L.sb0 + kGroupStride * j);
                x1 = *reinterpret_cast<const float2*>(S + L.sb1 + kGroupStride * j);
            }
            float2 g0, g1;
            if (trans) {
                g0 = make_float2(static_cast<float>(Gs[L.c2 * gpt + ra]), static_cast<float>(Gs[(L.c2 + 1) * gpt + ra]));
                g1 = make_float2(static_cast<float>(Gs[L.c2 * gpt + rb]), static_cast<float>(Gs[(L.c2 + 1) * gpt + rb]));
            } else {
                g0 = GradPair<GT>::at(Gs, L.sb0 + kGroupStride * j, L.sg0 + kGroupStride * j, 0);
                g1 = GradPair<GT>::at(Gs, L.sb1 + kGroupStride * j, L.sg1 + kGroupStride * j, 0);
            }
            const float m0 = g0.x + (x0.x - c[0]);       // M = G + E, E = B - P_prev R
            const float m1 = g0.y + (x0.y - c[2]);
            const float m2 = g1.x + (x1.x - c[1]);
            const float m3 = g1.y + (x1.y - c[3]);
            if (write_B && colok) {
                const uint32_t oa = orow + j * jstep;
                if (ra < mp) st_stream2(Bi + oa, m0, m1);
                if (rb < mp) st_stream2(Bi + (oa + rstep), m2, m3);
            }
            acc[j][0] += m0; acc[j][1] += m1; acc[j][2] += m2; acc[j][3] += m3;
        }
    }
}

// acc <- acc / N, stored as the strip of Mbar (Mb: Mbar at the strip's first column).
template <int GPW>
__device__ __forceinline__ void store_mbar(float (&acc)[GPW][4], int N, float* Mb, int mp, int np, int ng, bool colok,
                                           const Lane& L, int* nonfinite) {
    const float invN = 1.0f / static_cast<float>(N);
    bool bad = false;
#pragma unroll
    for (int j = 0; j < GPW; ++j) {
        const int G8 = L.w + NW * j;
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[j][e] *= invN;
        const int ra = 8 * G8 + L.rho, rb = ra + 2;
        if (G8 < ng && colok) {
            if (ra < mp) {
                *reinterpret_cast<float2*>(Mb + (int64_t)ra * np) = make_float2(acc[j][0], acc[j][1]);
                bad |= !isfinite(acc[j][0]) || !isfinite(acc[j][1]);
            }
            if (rb < mp) {
                *reinterpret_cast<float2*>(Mb + (int64_t)rb * np) = make_float2(acc[j][2], acc[j][3]);
                bad |= !isfinite(acc[j][2]) || !isfinite(acc[j][3]);
            }
        }
    }
    flag_nonfinite(bad, nonfinite);
}

// Truncated-basis Approx-Top-r partial sums over the strip: (Mbar - Yt (Y^T Mbar)) v_j.
// v_j first: the 32 lanes draw the 32 quads (row, 4 columns) of a row group once each: lane
// (g, t) draws row rho + 2 (g % 2), quad g / 2 (no data needed, so it can run early).
template <int GPW>
__device__ __forceinline__ void lam_draw(float4 (&vq)[GPW], uint64_t seed, uint32_t t, int b0, int ng, const Lane& L) {
#pragma unroll
    for (int j = 0; j < GPW; ++j) {
        const int G8 = L.w + NW * j;
        if (G8 < ng)
            vq[j] = gauss4_fast(seed, t, static_cast<uint32_t>(8 * G8 + L.rho + 2 * (L.gg & 1)),
                           static_cast<uint32_t>((b0 >> 2) + (L.gg >> 1)), kTagLambdaV);
    }
}
// Warp partials of W^T = Mbar_strip^T Y (YF: Y in fragment order, KT n-tiles) into wpart.
template <int GPW>
__device__ __forceinline__ void lam_w_partials(const float* YF, int KT, const float (&acc)[GPW][4], float* wpart,
                                               int wpitch, int ng, const Lane& L) {
    float d[2][4][4];                                        // two accumulators per n-tile
#pragma unroll
    for (int h = 0; h < 2; ++h)
#pragma unroll
        for (int nt = 0; nt < 4; ++nt)
#pragma unroll
            for (int e = 0; e < 4; ++e) d[h][nt][e] = 0.f;
#pragma unroll
    for (int j = 0; j < GPW; ++j) {
        const int G8 = L.w + NW * j;
        if (G8 < ng) {
            const FragA A = frag_a(acc[j][0], acc[j][1], acc[j][2], acc[j][3]);
#pragma unroll
            for (int nt = 0; nt < 4; ++nt)
                if (nt < KT) {
                    const float2 y = *reinterpret_cast<const float2*>(YF + (G8 * KT + nt) * 64 + 2 * L.lane);
                    mma3(d[j & 1][nt], A, frag_b(y.x, y.y));
                }
        }
    }
#pragma unroll
    for (int nt = 0; nt < 4; ++nt)
        if (nt < KT)
            *reinterpret_cast<float4*>(wpart + L.w * wpitch + (nt * 32 + L.lane) * 4) =
                make_float4(d[0][nt][0] + d[1][nt][0], d[0][nt][1] + d[1][nt][1], d[0][nt][2] + d[1][nt][2],
                            d[0][nt][3] + d[1][nt][3]);
}
// With W^T reduced in tot: C = Yt W on the lane's elements (YtF: Yt in fragment order) and the
// row partial sums of (Mbar - C) v_j, written to part_row[a] (the strip's row of partials).
template <int GPW>
__device__ __forceinline__ void lam_finish(const float* YtF, int KT, const float* tot, const float (&acc)[GPW][4],
                                           const float4 (&vq)[GPW], float* part_row, int mp, int ng, bool colok,
                                           const Lane& L) {
    FragA WA[4];
#pragma unroll
    for (int nt = 0; nt < 4; ++nt)
        if (nt < KT) {
            const float4 W = *reinterpret_cast<const float4*>(tot + (nt * 32 + L.lane) * 4);
            WA[nt] = frag_a(W.x, W.z, W.y, W.w);
        }
    const bool odd = (L.gg & 1) != 0;
#pragma unroll
    for (int j = 0; j < GPW; ++j) {
        const int G8 = L.w + NW * j;                         // warp-uniform: shuffles below are safe
        if (G8 < ng) {
            float c[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
            for (int nt = 0; nt < 4; ++nt)
                if (nt < KT) {
                    const float2 y = *reinterpret_cast<const float2*>(YtF + (G8 * KT + nt) * 64 + 2 * L.lane);
                    mma3(c, WA[nt], frag_b(y.x, y.y));
                }
            const float d0 = acc[j][0] - c[0], d1 = acc[j][1] - c[2];
            const float d2 = acc[j][2] - c[1], d3 = acc[j][3] - c[3];
            // each lane keeps the half of its quad it needs and trades the other with lane g ^ 1
            const int ra = 8 * G8 + L.rho;
            const float4 v = vq[j];
            const float q0 = __shfl_xor_sync(0xffffffffu, odd ? v.x : v.z, 4);
            const float q1 = __shfl_xor_sync(0xffffffffu, odd ? v.y : v.w, 4);
            const float v0 = odd ? q0 : v.x, v1 = odd ? q1 : v.y;       // row rho
            const float v2 = odd ? v.z : q0, v3 = odd ? v.w : q1;       // row rho + 2
            float pa = colok ? d0 * v0 + d1 * v1 : 0.f;
            float pb = colok ? d2 * v2 + d3 * v3 : 0.f;
#pragma unroll
            for (int x = 4; x < 32; x <<= 1) {
                pa += __shfl_xor_sync(0xffffffffu, pa, x);
                pb += __shfl_xor_sync(0xffffffffu, pb, x);
            }
            if (L.gg == 0) {
                if (ra < mp) part_row[ra] = pa;
                if (ra + 2 < mp) part_row[ra + 2] = pb;
            }
        }
    }
}

// Base of the dynamic shared memory; tile copies with a 64-byte swizzle need 512-byte aligned
// destinations, so the TMA kernels align it by an offset within the shared window (pointer
// arithmetic keeps the shared address space).
template <bool ALIGN>
__device__ __forceinline__ unsigned char* smem_base() {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    unsigned char* p = smem_raw;
    if constexpr (ALIGN) p += (1024u - (static_cast<uint32_t>(__cvta_generic_to_shared(smem_raw)) & 1023u)) & 1023u;
    return p;
}

// ---- per-strip kernel: one CTA per strip ----------------------------------------------------
// NQ = ceil(r / 8) n-tiles over q; each warp owns up to GPW = GPW_MAX / NQ groups of 8 rows
// (group w + NW j), so m' <= 8 NW GPW.  TMA: tile copies (G in its stored orientation), else
// cp.async.  `maps` holds the tile-copy descriptors (unused without TMA).
template <typename GT, int NQ, bool TMA>
__device__ __forceinline__ void compose_strip(const StreamGroup& g, const TmaMaps* maps) {
    constexpr int GPW = GPW_MAX / NQ;
    unsigned char* smem = smem_base<TMA>();
    const Lane L = lane_geometry();
    const int tid = L.tid;
    int mi = 0;
    while (mi + 1 < g.nmat && blockIdx.x >= static_cast<unsigned>(g.mat[mi + 1].strip0)) ++mi;
    const StreamMat& M = g.mat[mi];
    const int s = blockIdx.x - M.strip0;
    const int b0 = s * SW;
    const int mp = M.mp, np = M.np, r = M.r, N = M.N;
    const int mp16 = up16(mp), ng = up8(mp) >> 3;
    constexpr int GS = sizeof(GT);
    constexpr int EPC = 16 / GS;                      // gradient elements per 16-byte chunk
    const bool trans = !TMA && M.transposed != 0;
    const int gpt = g_tpitch(mp16, GS);
    const int rows = slot_rows(mp, TMA);
    const size_t sb = stage_b_bytes(rows, TMA), sg = stage_g_bytes(mp, rows, GS, trans, TMA), stage = sb + sg;
    const int KT = M.lam ? up8(M.k) >> 3 : 0;        // n-tiles of the lambda epilogue
    // the epilogue's warp partials go to the last node's ring slot when they fit there
    const bool wslot = lam_partials_in_slot(KT, stage);
    const int pitch = part_pitch(wslot || NQ > KT ? NQ : KT);
    unsigned char* ring = smem;
    float* part = reinterpret_cast<float*>(smem + 3 * stage);
    float* tot = part + NW * pitch;                   // NQ * 128, and KT * 128 for the epilogue
    uint64_t* bars = reinterpret_cast<uint64_t*>(tot + (NQ > KT ? NQ : KT) * 128);
    const bool corr = !M.e_zero, write_B = M.write_B != 0;
    const GT* const* Gp = reinterpret_cast<const GT* const*>(g.G + M.g_off);
    // the matrix descriptor is indexed by a runtime value: read its pointers once
    float* const Bst = M.B;
    const float* const YFg = M.YF;
    const float* const YtFg = M.YtF;
    const bool colok = b0 + L.c2 < np;                // n' % 4 == 0: both columns or neither
    const uint32_t ring_s = static_cast<uint32_t>(__cvta_generic_to_shared(ring));
    // tile copies: full[3] (copy landed) then empty[3] (every warp is done with the slot)
    const uint32_t bars_s = static_cast<uint32_t>(__cvta_generic_to_shared(bars)), empty_s = bars_s + 24;
    int timed_out = 0;

    // ---- cp.async staging plan (fixed for all nodes): up to 4 chunks of B and 4 of G -----------
    int boff[4], bdst[4], goff[4], gdst[4];
    unsigned bmask = 0, gmask = 0;
    if constexpr (!TMA) {
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int c = tid + j * T;                // B chunk: row a, 4 columns
            const int a = c >> 2, ch = c & 3, col = b0 + 4 * ch;
            boff[j] = a * np + col;
            bdst[j] = a * SW + 4 * (ch ^ ((a >> 1) & 3));
            if (c < mp * 4) {
                if (col < np) bmask |= 1u << j;
                else for (int st = 0; st < 3; ++st)   // columns past n': zero once in every slot
                    *reinterpret_cast<float4*>(reinterpret_cast<float*>(ring + st * stage) + bdst[j]) =
                        make_float4(0.f, 0.f, 0.f, 0.f);
            }
            if (trans) {                              // G rows b0 + bb, m' contiguous elements
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
            } else {                                  // G rows a, SW columns
                constexpr int CPR = SW / EPC;
                const int ga = c / CPR, gch = c % CPR, gcol = b0 + gch * EPC;
                goff[j] = ga * np + gcol;
                gdst[j] = GS == 4 ? ga * SW + 4 * (gch ^ ((ga >> 1) & 3)) : ga * SW + 8 * (gch ^ ((ga >> 2) & 1));
                if (c < mp * CPR) {
                    if (gcol < np) gmask |= 1u << j;
                    else for (int st = 0; st < 3; ++st)
                        *reinterpret_cast<float4*>(reinterpret_cast<GT*>(ring + st * stage + sb) + gdst[j]) =
                            make_float4(0.f, 0.f, 0.f, 0.f);
                }
            }
        }
        // rows mp..mp16 of every B strip and every (non-transposed) G strip stay zero; transposed
        // matrices have m' % 8 == 0, so their row groups never reach past m'
        for (int a = mp + (tid >> 4); a < mp16; a += T / SW) {
            const int c = tid & (SW - 1);
#pragma unroll
            for (int st = 0; st < 3; ++st) {
                reinterpret_cast<float*>(ring + st * stage)[a * SW + c] = 0.f;
                if (!trans) reinterpret_cast<GT*>(ring + st * stage + sb)[a * SW + c] = GT(0.f);
            }
        }
    } else {
        if (tid == 0) {
#pragma unroll
            for (int st = 0; st < 3; ++st) {
                mbar_init(bars_s + 8 * st, 1);
                mbar_init(empty_s + 8 * st, NW);
            }
            asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        }
        __syncthreads();
    }

    // ring item j: node j's B (unless E = 0) and G strips; with the lambda epilogue, items N and
    // N + 1 are the fragment-ordered Y and Yt (up8(m') x 8 KT floats each).  With tile copies
    // thread 0 issues an item (rows past m' and columns past n' arrive as zeros); with cp.async
    // every thread issues its chunks and commits a group.
    const int nbox = tma_nbox(mp), brows = tma_box_rows(mp);
    auto stage_item = [&](int j) {
        const uint32_t base = ring_s + static_cast<uint32_t>((j % 3) * stage);
        if constexpr (TMA) {
            if (tid != 0 || j >= N + (KT ? 2 : 0)) return;
            const uint32_t bar = bars_s + 8 * (j % 3);
            // the slot's previous item (j - 3) must be released by every warp
            if (j >= 3 && !mbar_wait(empty_s + 8 * (j % 3), ((j / 3) - 1) & 1)) timed_out = 1;
            if (j < N) {
                const uint32_t gbytes = static_cast<uint32_t>(brows * SW * GS);
                mbar_expect_tx(bar, nbox * ((corr ? brows * SW * 4u : 0u) + gbytes));
                for (int b = 0; b < nbox; ++b) {
                    if (corr) tma_load_3d(base + b * brows * SW * 4, &maps->B[mi], b0, b * brows, j, bar);
                    tma_load_2d(base + static_cast<uint32_t>(sb) + b * gbytes, &maps->G[M.g_off + j], b0, b * brows,
                                bar);
                }
            } else {
                const uint32_t bytes = static_cast<uint32_t>(ng * KT * 256);   // 64 floats per (group, n-tile)
                mbar_expect_tx(bar, bytes);
                bulk_load(base, j == N ? YFg : YtFg, bytes, bar);
            }
        } else {
            if (j < N) {
                if (corr) {
                    const float* src = Bst + (int64_t)j * mp * np;
#pragma unroll
                    for (int q = 0; q < 4; ++q)
                        if (bmask & (1u << q)) cp_async16(base + 4u * bdst[q], src + boff[q]);
                }
                const GT* src = Gp[j];
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    if (gmask & (1u << q)) cp_async16(base + static_cast<uint32_t>(sb) + GS * gdst[q], src + goff[q]);
            } else if (j < N + 2 && KT) {
                const float* src = j == N ? YFg : YtFg;
                const int nch = ng * KT * 16;
                for (int c = tid; c < nch; c += T) cp_async16(base + 16u * c, src + 4 * c);
            }
            cp_async_commit();
        }
    };
    // item j has landed for this thread (tile copies: its slot's mbarrier completed item j's phase)
    auto await_item = [&](int j) {
        if constexpr (TMA) {
            if (!mbar_wait(bars_s + 8 * (j % 3), (j / 3) & 1)) timed_out = 1;
        }
    };
    stage_item(0);
    stage_item(1);

    FragB prt[GPW][NQ], pcb[GPW][NQ];
    load_pfrags<NQ, GPW>(M.Pprev, mp, r, ng, corr, L, prt, pcb);
    float acc[GPW][4];
#pragma unroll
    for (int j = 0; j < GPW; ++j)
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[j][e] = 0.f;

    for (int i = 0; i < N; ++i) {
        if constexpr (TMA) {
            stage_item(i + 2);             // thread 0, once node i - 1's slot is released
            await_item(i);
        } else {
            cp_async_wait<1>();            // node i has landed; item i + 1 may be in flight
            __syncthreads();               // ... for every thread; node i - 1 is finished
            stage_item(i + 2);             // into the slot node i - 1 used
        }
        const float* S = reinterpret_cast<const float*>(ring + (size_t)(i % 3) * stage);
        const GT* Gs = reinterpret_cast<const GT*>(ring + (size_t)(i % 3) * stage + sb);
        compose_node<GT, NQ, GPW>(S, Gs, trans, gpt, corr, prt, pcb, acc, part, pitch, tot,
                                  Bst + (int64_t)i * mp * np + b0, mp, np, ng, write_B, colok, L);
        if constexpr (TMA) {               // this warp is done with node i's slot
            __syncwarp();
            if (L.lane == 0) mbar_arrive(empty_s + 8 * (i % 3));
        }
    }
    if constexpr (!TMA) cp_async_wait<0>();
    store_mbar<GPW>(acc, N, M.Mbar + b0 + L.c2, mp, np, ng, colok, L, M.nonfinite);
    if (KT) {
        float4 vq[GPW];
        lam_draw<GPW>(vq, M.seed, M.t, b0, ng, L);
        await_item(N);
        await_item(N + 1);
        __syncthreads();                                     // Y, Yt landed for every thread
        const float* YF = reinterpret_cast<const float*>(ring + (size_t)(N % 3) * stage);
        const float* YtF = reinterpret_cast<const float*>(ring + (size_t)((N + 1) % 3) * stage);
        // the warp partials of W^T (in the slot of the last node, free once every thread is here)
        float* wpart = wslot ? reinterpret_cast<float*>(ring + (size_t)((N + 2) % 3) * stage) : part;
        const int wpitch = wslot ? part_pitch(KT) : pitch;
        lam_w_partials<GPW>(YF, KT, acc, wpart, wpitch, ng, L);
        __syncthreads();
        reduce_warps(wpart, wpitch, KT, tot);                // W^T = Mbar_strip^T Y
        __syncthreads();
        if (M.Wbar) {
            // W = Y^T Mbar for K3: tot[(nt 32 + lane) 4 + e] is W[8 nt + 2t + e % 2][b0 + 2g + e / 2]
            float* Wg = M.Wbar;
            const int k = M.k;
            for (int idx = tid; idx < KT * 128; idx += T) {
                const int ln = (idx >> 2) & 31, e = idx & 3;
                const int q = 8 * (idx >> 7) + 2 * (ln & 3) + (e & 1), col = b0 + 2 * (ln >> 2) + (e >> 1);
                if (q < k && col < np) Wg[(int64_t)q * np + col] = tot[idx];
            }
        }
        lam_finish<GPW>(YtF, KT, tot, acc, vq, M.part + (int64_t)s * mp, mp, ng, colok, L);
    }
    if (timed_out && g.err) atomicAdd(g.err, 1);
}

template <typename GT, int NQ>
__global__ void __launch_bounds__(T, 1) stream_mma_kernel(const __grid_constant__ StreamGroup g) {
    compose_strip<GT, NQ, false>(g, nullptr);
}
template <typename GT, int NQ>
__global__ void __launch_bounds__(T, 1) stream_tma_kernel(const __grid_constant__ StreamGroup g,
                                                          const __grid_constant__ TmaMaps maps) {
    compose_strip<GT, NQ, true>(g, &maps);
}
// dst = src (rows x cols, row-major, ld) in fragment order, up8(rows) x up8(cols) floats:
// block (group G8, n-tile nt) holds 64 floats, lane L = 4g + t's pair at 2L, 2L + 1.
//   form 0 (B fragment of X^T Y):  src(8 G8 + rho(t), 8 nt + g), src(8 G8 + rho(t) + 2, 8 nt + g)
//   form 1 (B fragment of W Y^T): src(8 G8 + prow(g), 8 nt + 2t), src(8 G8 + prow(g), 8 nt + 2t + 1)
// with rho(t) = (t % 2) + 4 (t / 2) and prow(g) = rho(g / 2) + 2 (g % 2).
__global__ void pack_frag_kernel(float* dst, const float* src, int rows, int cols, int ld, int form) {
    const int KT = up8(cols) >> 3;
    const int total = up8(rows) * KT * 8;
    for (int idx = blockIdx.x * blockDim.x + threadIdx.x; idx < total; idx += gridDim.x * blockDim.x) {
        const int blk = idx >> 6, L = (idx >> 1) & 31, e = idx & 1;
        const int G8 = blk / KT, nt = blk % KT, g = L >> 2, t = L & 3;
        int row, col;
        if (form == 0) { row = 8 * G8 + (t & 1) + 4 * (t >> 1) + 2 * e; col = 8 * nt + g; }
        else { row = 8 * G8 + ((g >> 1) & 1) + 4 * (g >> 2) + 2 * (g & 1); col = 8 * nt + 2 * t + e; }
        dst[idx] = row < rows && col < cols ? src[(int64_t)row * ld + col] : 0.f;
    }
}

}  // namespace

int mma_stream_nq(int r) { return (r + 7) / 8; }

bool mma_stream_eligible(int mp, int np, int r, int k, int lam, int transposed, int gsize) {
    const int NQ = mma_stream_nq(r), ng = up8(mp) / 8;
    if (NQ < 1 || NQ > 2 || (ng + NW - 1) / NW > GPW_MAX / NQ) return false;   // groups per warp
    if (lam && (k < 1 || k > 32)) return false;
    if (np % 4 != 0 || (transposed && mp % 8 != 0)) return false;      // 16-byte chunks of G rows
    return mma_stream_smem_bytes(mp, r, k, lam, gsize, transposed, 0) <= 227 * 1024;
}

bool mma_stream_tma_eligible(int mp, int np, int r, int k, int lam, int transposed, int gsize) {
    if (transposed || !mma_stream_eligible(mp, np, r, k, lam, transposed, gsize)) return false;
    if (((int64_t)np * gsize) % 16 != 0) return false;                 // row stride of a tile copy
    return mma_stream_smem_bytes(mp, r, k, lam, gsize, transposed, 1) <= 227 * 1024;
}

size_t mma_stream_smem_bytes(int mp, int r, int k, int lam, int gsize, int transposed, int tma) {
    const int NQ = mma_stream_nq(r), KT = lam ? up8(k) / 8 : 0;
    const int rows = slot_rows(mp, tma != 0);
    const size_t stage = stage_b_bytes(rows, tma != 0) + stage_g_bytes(mp, rows, gsize, transposed, tma != 0);
    if (lam && (size_t)up8(mp) * KT * 8 * 4 > stage) return ~size_t(0);   // Y, Yt use ring slots
    const int NT = NQ > KT ? NQ : KT;
    const int PT = lam_partials_in_slot(KT, stage) ? NQ : NT;
    const size_t bytes = 3 * stage + (size_t)NW * part_pitch(PT) * 4 + (size_t)NT * 128 * 4 + 3 * 8;
    return tma ? bytes + 24 + 1024 : bytes;            // empty barriers; room to align the base to 1024 bytes
}

int mma_tma_box_rows(int mp) { return tma_box_rows(mp); }

template <typename GT, int NQ>
static cudaError_t launch_mma(const StreamGroup& g, size_t smem, cudaStream_t st) {
    {   // per device: set on every call (cheap next to the launch)
        const cudaError_t ea = cudaFuncSetAttribute(stream_mma_kernel<GT, NQ>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             227 * 1024);
        if (ea != cudaSuccess) return ea;
    }
    stream_mma_kernel<GT, NQ><<<g.total_strips, T, smem, st>>>(g);
    return cudaGetLastError();
}
template <typename GT, int NQ>
static cudaError_t launch_tma(const StreamGroup& g, const TmaMaps& maps, size_t smem, cudaStream_t st) {
    {   // per device: set on every call (cheap next to the launch)
        const cudaError_t ea = cudaFuncSetAttribute(stream_tma_kernel<GT, NQ>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             227 * 1024);
        if (ea != cudaSuccess) return ea;
    }
    stream_tma_kernel<GT, NQ><<<g.total_strips, T, smem, st>>>(g, maps);
    return cudaGetLastError();
}

cudaError_t stream_group_mma(const StreamGroup& g, const TmaMaps* maps, size_t smem, cudaStream_t st) {
    if (g.total_strips <= 0) return cudaSuccess;
    const int NQ = mma_stream_nq(g.mat[0].r);
    for (int i = 1; i < g.nmat; ++i)
        if (mma_stream_nq(g.mat[i].r) != NQ) return cudaErrorInvalidValue;
    if (maps) {
        for (int i = 0; i < g.nmat; ++i)
            if (g.mat[i].transposed || g.mat[i].g_off + g.mat[i].N > kTmaGMax) return cudaErrorInvalidValue;
        if (g.grad_dtype == GLR_BF16)
            return NQ == 1 ? launch_tma<__nv_bfloat16, 1>(g, *maps, smem, st)
                           : launch_tma<__nv_bfloat16, 2>(g, *maps, smem, st);
        return NQ == 1 ? launch_tma<float, 1>(g, *maps, smem, st) : launch_tma<float, 2>(g, *maps, smem, st);
    }
    if (g.grad_dtype == GLR_BF16)
        return NQ == 1 ? launch_mma<__nv_bfloat16, 1>(g, smem, st) : launch_mma<__nv_bfloat16, 2>(g, smem, st);
    return NQ == 1 ? launch_mma<float, 1>(g, smem, st) : launch_mma<float, 2>(g, smem, st);
}

cudaError_t pack_frag(float* dst, const float* src, int rows, int cols, int ld, int form, cudaStream_t st) {
    const int total = up8(rows) * up8(cols);
    if (total <= 0) return cudaSuccess;
    pack_frag_kernel<<<(total + 255) / 256, 256, 0, st>>>(dst, src, rows, cols, ld, form);
    return cudaGetLastError();
}

}  // namespace glr
