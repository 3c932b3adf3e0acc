// The large-matrix path on the fifth-generation tensor cores (tcgen05): every rank-r and rank-k
// product of a GreedyLore step (Algorithm 3 with the truncated basis) as a TF32 tcgen05.mma with
// its accumulator in tensor memory, operands staged by the Tensor Memory Accelerator, and the
// step's elementwise work fused into the epilogues.  One kernel template (tc_kernel) runs every
// product; an "op" supplies the tile map, the tile copies, the MMAs and the epilogue:
//
//   PrevProj  R_w,i^T = (P_prev^T B_i)^T                 (the deferred error's projection)
//   Compose   M_i = G_i + B_i - P_prev R_w,i; B_i <- M_i; Mbar = (1/N) sum_i M_i   (Eq. ef1)
//   WBar      W^T = (Y^T Mbar)^T                          (U^T Mbar = D (Mbar - Yt W))
//   Lambda    partial sums of D (Mbar - Yt W)_j v_j over 64 columns (Algorithm 2)
//   PBuild    P = U[:, J] = (E_J - Y Yt[J, :]^T) D_J, and P^T
//   RBar      Rbar = P^T Mbar = D_J (Mbar[J, :] - Yt[J, :] W)   (the node average, Eq. 8zhb2we09)
//   Update    Ghat = P Rbar (or Mbar), then MSGD (Eq. msgd) / Adam (Eq. adam) on X  (K3)
//
// Layouts (oriented m' x n', m' <= n'): the node buffers B_i and Mbar are stored column-major
// (B_i^T, n' x m', m' contiguous) so that every contraction over m' reads a K-major operand; P
// is row-major m' x r with a transposed copy P^T (rpad x m'); R_w,i^T, W^T and Rbar^T are n' x
// rpad / kpad; Y, Yt are row-major m' x k and Y^T is kpad x m'.  Every MMA operand is K-major
// with the 128-byte swizzle: a 32-element (128-byte) K slice of 8-row groups, 1024 bytes per
// group.  kind::tf32 reads the top 19 bits of each fp32 operand (the low mantissa bits are
// dropped); operands this file writes for later products are rounded to the nearest TF32 value
// first.  Accumulation is fp32.
//
// Roles per CTA (352 threads, one CTA per SM, persistent over the tiles): warps 0-7 epilogue
// (warp w reads tensor-memory lanes 32 (w % 4) .. + 31; w / 4 picks a column half), warp 8
// issues the operand tile copies into a ring of shared-memory stages, warp 9 owns tensor memory
// and issues the MMAs, warp 10 copies the epilogue's element tiles into a second ring.  Stages
// are handed over on mbarriers (copy -> "full", MMA commit or epilogue -> "empty"); the
// accumulator (one or two buffers in tensor memory) on "tfull" (MMA commit) / "tempty" (the
// epilogue warps).  The epilogue writes its results into the data stage and stores them with
// tile copies.  Every wait polls with short sleeps and gives up after about a second: it then
// counts the event in the caller's error flag, raises the CTA's abort flag (every role leaves its
// loop), waits (bounded) for the copies already issued, frees tensor memory and returns.
#include <cuda.h>

#include <algorithm>

#include "glr_internal.cuh"

namespace glr {
namespace tc {

namespace {

// Epilogue warps per op (Op::kEpi); the three role warps follow them.
template <class Op> constexpr int threads_of() { return (Op::kEpi + 3) * 32; }
constexpr int kMaxStages = 8;
constexpr int kMaxDStages = 4;
constexpr uint32_t kTmemCols = 512;      // every op keeps more than half of shared memory, so one CTA per SM
constexpr size_t kSmemBudget = 220 * 1024;
constexpr size_t kMinSmem = 120 * 1024;  // above half of an SM's 228 KiB: one CTA, one allocation per SM

__device__ __forceinline__ uint32_t smem_u32(const void* p) { return static_cast<uint32_t>(__cvta_generic_to_shared(p)); }
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mbar_test(uint32_t bar, uint32_t parity) {
    uint32_t done;
    asm volatile("{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
                 : "=r"(done) : "r"(bar), "r"(parity) : "memory");
    return done != 0;
}
// Waits for phase `parity` of `bar`; false when the CTA aborted (now or already).  About a second
// of polling (16 M polls with sleeps of 16..64 ns) before giving up.
__device__ __forceinline__ bool wait_phase(uint32_t bar, uint32_t parity, volatile int* abort, int* err,
                                           int limit = 16000000) {
    uint32_t ns = 16;
    for (int it = 0; it < limit; ++it) {
        if (mbar_test(bar, parity)) return true;
        if ((it & 255) == 255 && *abort) return false;
        __nanosleep(ns);
        ns = ns < 64 ? 2 * ns : 64;
    }
    if (atomicExch(const_cast<int*>(abort), 1) == 0) atomicAdd(err, 1);
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
// Shared-memory matrix descriptor: K-major, 128-byte swizzle, 8-row groups 1024 bytes apart.
__device__ __forceinline__ uint64_t sdesc(uint32_t addr) {
    return static_cast<uint64_t>((addr >> 4) & 0x3FFFu) | (uint64_t(1) << 16) | (uint64_t(64) << 32) |
           (uint64_t(1) << 46) | (uint64_t(2) << 61);
}
// Instruction descriptor: kind::tf32, fp32 accumulator, both operands K-major, M = 128, N = n.
__device__ __forceinline__ uint32_t idesc(int n) {
    return (1u << 4) | (2u << 7) | (2u << 10) | (static_cast<uint32_t>(n >> 3) << 17) | (8u << 24);
}
__device__ __forceinline__ void mma(uint32_t d, uint64_t a, uint64_t b, uint32_t id, uint32_t acc) {
    asm volatile("{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\ntcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n}"
                 ::"r"(d), "l"(a), "l"(b), "r"(id), "r"(acc));
}
__device__ __forceinline__ void mma_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
// 16 consecutive accumulator columns of this thread's lane.
__device__ __forceinline__ void tmem_ld16(uint32_t ta, float (&v)[16]) {
    uint32_t u[16];
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
                 : "=r"(u[0]), "=r"(u[1]), "=r"(u[2]), "=r"(u[3]), "=r"(u[4]), "=r"(u[5]), "=r"(u[6]), "=r"(u[7]),
                   "=r"(u[8]), "=r"(u[9]), "=r"(u[10]), "=r"(u[11]), "=r"(u[12]), "=r"(u[13]), "=r"(u[14]), "=r"(u[15])
                 : "r"(ta));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int j = 0; j < 16; ++j) v[j] = __uint_as_float(u[j]);
}
// 8 consecutive accumulator columns of this thread's lane.
__device__ __forceinline__ void tmem_ld8(uint32_t ta, float (&v)[8]) {
    uint32_t u[8];
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                 : "=r"(u[0]), "=r"(u[1]), "=r"(u[2]), "=r"(u[3]), "=r"(u[4]), "=r"(u[5]), "=r"(u[6]), "=r"(u[7])
                 : "r"(ta));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int j = 0; j < 8; ++j) v[j] = __uint_as_float(u[j]);
}
// x rounded to the nearest TF32 value (ties away from zero), as an fp32 bit pattern.
__device__ __forceinline__ float rna_tf32(float x) {
    uint32_t u;
    asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(u) : "f"(x));
    return __uint_as_float(u);
}
__device__ __forceinline__ float grad_at(const void* G, int64_t e, int dtype) {
    if (dtype == GLR_BF16) return __bfloat162float(static_cast<const __nv_bfloat16*>(G)[e]);
    return static_cast<const float*>(G)[e];
}

// ------------------------------------------------------------------------------------------
// The pipeline.  An operand stage holds `na` A slices (128 rows x 32 K, 16 KiB each) and `nb`
// B slices (bn rows x 32 K each), every slice on a 1024-byte boundary.  A data stage holds the
// epilogue's element tiles (node gradients, error buffers, optimizer state), loaded by the data
// warp and, where the epilogue writes them back, stored from the same shared memory by tile
// copies once every epilogue thread has finished with the stage.
// ------------------------------------------------------------------------------------------
struct Tile {
    int mat;          // index into the group
    int lt;           // tile index within the matrix
    int nk;           // K slices of 32 (0: the epilogue runs without MMAs)
};

__device__ __forceinline__ Tile find_tile(const TcGroup& g, int tile) {
    int lo = 0, hi = g.nmat - 1;
    while (lo < hi) {                        // last matrix with tile0 <= tile
        const int mid = (lo + hi + 1) >> 1;
        if (g.mat[mid].tile0 <= tile) lo = mid; else hi = mid - 1;
    }
    Tile t;
    t.mat = lo;
    t.lt = tile - g.mat[lo].tile0;
    t.nk = 0;
    return t;
}

__device__ __forceinline__ void fence_proxy_async() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }
__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, int x, int y, uint32_t src) {
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];"
                 ::"l"(map), "r"(x), "r"(y), "r"(src) : "memory");
}
__device__ __forceinline__ void tma_store_3d(const CUtensorMap* map, int x, int y, int z, uint32_t src) {
    asm volatile("cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%1, %2, %3}], [%4];"
                 ::"l"(map), "r"(x), "r"(y), "r"(z), "r"(src) : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }

// The epilogue's side of the data ring.  acquire() waits for the next stage; release() marks this
// thread done with it: the last thread to finish (counted on the stage's "done" mbarrier, waited
// by thread 0 of the epilogue) lets `store` issue the tile copies back to global memory as one
// bulk group.  A stage goes back to the data warp once its group has read shared memory: with
// three or more stages the leader checks that one stage later (at most one group pending), so the
// copies of a stage overlap the work on the next; finish() drains the last one.
struct DataRing {
    uint8_t* base;
    uint32_t bytes;
    int n, s;
    uint32_t use;
    uint64_t *full, *empty, *done;
    volatile int* abort;
    int* err;
    int pend;                                         // stage whose group may still be reading (leader)
    // warp-uniform: every lane gets the stage, or none (the CTA aborted)
    __device__ __forceinline__ uint8_t* acquire() {
        const bool ok = wait_phase(smem_u32(&full[s]), use, abort, err);
        if (!__all_sync(0xffffffffu, ok)) return nullptr;
        return base + (size_t)s * bytes;
    }
    template <class Store>
    __device__ __forceinline__ void release(bool leader, Store store) {
        fence_proxy_async();                          // this thread's writes, before the copies read them
        mbar_arrive(smem_u32(&done[s]));
        if (leader) {
            if (wait_phase(smem_u32(&done[s]), use, abort, err)) store(smem_u32(base + (size_t)s * bytes));
            bulk_commit();                            // one group per stage (empty when nothing is stored)
            if (n < 3) {                              // two stages: hand this one back at once
                bulk_wait_read();
                mbar_arrive(smem_u32(&empty[s]));
            } else {
                if (pend >= 0) {
                    asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
                    mbar_arrive(smem_u32(&empty[pend]));
                }
                pend = s;
            }
        }
        if (++s == n) { s = 0; use ^= 1u; }
    }
    __device__ __forceinline__ void finish(bool leader) {
        if (!leader) return;
        bulk_wait_read();
        if (pend >= 0) mbar_arrive(smem_u32(&empty[pend]));
        pend = -1;
        asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");   // the stores are complete before the CTA ends
    }
};
struct NoStore { __device__ bool operator()(uint32_t) const { return false; } };

// Ops without epilogue data.
struct NoData {
    static constexpr int kEpi = 8;
    static __device__ __forceinline__ int ndata(const TcGroup&, const Tile&) { return 0; }
    static __device__ __forceinline__ uint32_t data_tx(const TcGroup&, const Tile&, int) { return 0; }
    static __device__ __forceinline__ void data_load(const TcGroup&, const Tile&, int, uint32_t, uint32_t) {}
};

template <class Op>
__global__ void __launch_bounds__(threads_of<Op>(), 1) tc_kernel(const __grid_constant__ TcGroup g) {
    constexpr int kEpiWarps = Op::kEpi;
    constexpr int kProdWarp = kEpiWarps, kMmaWarp = kEpiWarps + 1, kDataWarp = kEpiWarps + 2;
    extern __shared__ uint8_t dyn_smem[];
    uint8_t* ring = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(dyn_smem) + 1023) & ~uintptr_t(1023));
    __shared__ __align__(8) uint64_t full_bar[kMaxStages], empty_bar[kMaxStages], tfull_bar[2], tempty_bar[2];
    __shared__ __align__(8) uint64_t dfull_bar[kMaxDStages], dempty_bar[kMaxDStages], ddone_bar[kMaxDStages];
    __shared__ uint32_t tmem_base;
    __shared__ int abort_flag;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int S = g.stages, D = g.dstages;
    const uint32_t SB = g.stage_bytes, DB = g.dstage_bytes;
    uint8_t* dring = ring + (size_t)S * SB;
    const int nbuf = g.tbufs;
    volatile int* abort = &abort_flag;
    if (threadIdx.x == 0) {
        abort_flag = 0;
        for (int q = 0; q < S; ++q) { mbar_init(smem_u32(&full_bar[q]), 1); mbar_init(smem_u32(&empty_bar[q]), 1); }
        for (int q = 0; q < D; ++q) {
            mbar_init(smem_u32(&dfull_bar[q]), 1);
            mbar_init(smem_u32(&dempty_bar[q]), 1);
            mbar_init(smem_u32(&ddone_bar[q]), kEpiWarps * 32);
        }
        for (int b = 0; b < 2; ++b) { mbar_init(smem_u32(&tfull_bar[b]), 1); mbar_init(smem_u32(&tempty_bar[b]), kEpiWarps); }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == kMmaWarp) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                     ::"r"(smem_u32(&tmem_base)), "r"(kTmemCols));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    fence_before();
    __syncthreads();
    fence_after();
    const uint32_t tmem = tmem_base;
    const uint32_t buf_cols = kTmemCols / 2;

    if (warp == kProdWarp || warp == kDataWarp) {
        // operand copies (kProdWarp) or epilogue data copies (kDataWarp): the same loop over the
        // CTA's tiles on its own ring
        if (lane == 0) {
            const bool data = warp == kDataWarp;
            const int n = data ? D : S;
            const uint32_t bytes = data ? DB : SB;
            uint8_t* base = data ? dring : ring;
            uint64_t* fullb = data ? dfull_bar : full_bar;
            uint64_t* emptyb = data ? dempty_bar : empty_bar;
            int s = 0;
            uint32_t use = 0;                  // fills of stage s so far, as a phase bit
            uint32_t issued = 0, last_par = 0; // per stage (bit q): copies issued, parity of the last fill
            for (int tile = blockIdx.x; tile < g.total_tiles && !*abort; tile += gridDim.x) {
                Tile t = find_tile(g, tile);
                t.nk = Op::nk(g, t);
                const int cnt = data ? Op::ndata(g, t) : t.nk;
                for (int kc = 0; kc < cnt; ++kc) {
                    if (!wait_phase(smem_u32(&emptyb[s]), use ^ 1u, abort, g.err)) break;
                    const uint32_t st = smem_u32(base + (size_t)s * bytes);
                    const uint32_t fb = smem_u32(&fullb[s]);
                    if (data) {
                        mbar_expect_tx(fb, Op::data_tx(g, t, kc));
                        Op::data_load(g, t, kc, st, fb);
                    } else {
                        mbar_expect_tx(fb, Op::tx_bytes(g, t, kc));
                        Op::load(g, t, kc, st, fb);
                    }
                    issued |= 1u << s;
                    last_par = (last_par & ~(1u << s)) | (use << s);
                    if (++s == n) { s = 0; use ^= 1u; }
                }
            }
            if (*abort) {                      // let the copies already issued land before leaving
                for (int q = 0; q < n; ++q)
                    if (issued & (1u << q))
                        for (int it = 0; it < 4000000 && !mbar_test(smem_u32(&fullb[q]), (last_par >> q) & 1u); ++it)
                            __nanosleep(64);
            }
        }
    } else if (warp == kMmaWarp) {
        if (lane == 0) {
            int s = 0;
            uint32_t use = 0, tuse[2] = {0, 0};
            int b = 0;
            for (int tile = blockIdx.x; tile < g.total_tiles && !*abort; tile += gridDim.x) {
                Tile t = find_tile(g, tile);
                t.nk = Op::nk(g, t);
                if (!wait_phase(smem_u32(&tempty_bar[b]), tuse[b] ^ 1u, abort, g.err)) break;
                fence_after();
                const uint32_t dt = tmem + (uint32_t)b * buf_cols;
                bool ok = true;
                for (int kc = 0; kc < t.nk; ++kc) {
                    if (!wait_phase(smem_u32(&full_bar[s]), use, abort, g.err)) { ok = false; break; }
                    fence_after();
                    Op::mma(g, t, kc, smem_u32(ring + (size_t)s * SB), dt);
                    mma_commit(smem_u32(&empty_bar[s]));
                    if (++s == S) { s = 0; use ^= 1u; }
                }
                if (!ok) break;
                if (t.nk > 0) mma_commit(smem_u32(&tfull_bar[b]));
                else mbar_arrive(smem_u32(&tfull_bar[b]));
                tuse[b] ^= 1u;
                if (nbuf == 2) b ^= 1;
            }
        }
        __syncwarp();
    } else {
        uint32_t tuse[2] = {0, 0};
        int b = 0;
        DataRing dr{dring, DB, D, 0, 0u, dfull_bar, dempty_bar, ddone_bar, abort, g.err, -1};
        for (int tile = blockIdx.x; tile < g.total_tiles; tile += gridDim.x) {
            Tile t = find_tile(g, tile);
            t.nk = Op::nk(g, t);
            const bool ok = wait_phase(smem_u32(&tfull_bar[b]), tuse[b], abort, g.err);
            if (!__all_sync(0xffffffffu, ok)) break;       // warp-uniform, for the tensor-memory loads
            fence_after();
            if (!Op::epilogue(g, t, tmem + (uint32_t)b * buf_cols + ((uint32_t)(32 * (warp & 3)) << 16), warp, lane, dr))
                break;
            fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&tempty_bar[b]));
            tuse[b] ^= 1u;
            if (nbuf == 2) b ^= 1;
        }
        if (D > 0) dr.finish(warp == 0 && lane == 0);
    }
    fence_before();
    __syncthreads();
    if (warp == kMmaWarp) {
        fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols));
    }
}

// MMAs of one K slice: D (+)= A_slice B_slice^T, four k-steps of 8 (32 bytes) along the slice.
__device__ __forceinline__ void mma_slice(uint32_t d, uint32_t a, uint32_t b, int n, bool first) {
    const uint32_t id = idesc(n);
#pragma unroll
    for (int kk = 0; kk < 4; ++kk)
        mma(d, sdesc(a + 32 * kk), sdesc(b + 32 * kk), id, (first && kk == 0) ? 0u : 1u);
}

// ------------------------------------------------------------------------------------------
// PrevProj: tile = (128 columns c of n', node group).  D_i (128 x rpad) = B_i^T[c, :] P_prev^T^T
// over K = m'; the epilogue writes R_w,i^T[c][q] (rounded to TF32).  A = B_i^T slices (3-D map
// m' x n' x N), B = P_prev^T (rpad x m').
// ------------------------------------------------------------------------------------------
struct PrevProj : NoData {
    static __device__ __forceinline__ int nk(const TcGroup& g, const Tile& t) { return (g.mat[t.mat].mp + 31) / 32; }
    static __device__ __forceinline__ void decode(const TcMat& M, int lt, int& ct, int& i0, int& ni) {
        ct = lt / M.ng;
        i0 = (lt % M.ng) * M.na;
        ni = M.N - i0 < M.na ? M.N - i0 : M.na;
    }
    static __device__ __forceinline__ uint32_t tx_bytes(const TcGroup& g, const Tile& t, int) {
        const TcMat& M = g.mat[t.mat];
        int ct, i0, ni;
        decode(M, t.lt, ct, i0, ni);
        return (uint32_t)ni * 16384u + (uint32_t)M.rpad * 128u;
    }
    static __device__ __forceinline__ void load(const TcGroup& g, const Tile& t, int kc, uint32_t st, uint32_t bar) {
        const TcMat& M = g.mat[t.mat];
        int ct, i0, ni;
        decode(M, t.lt, ct, i0, ni);
        for (int a = 0; a < ni; ++a) tma_load_3d(st + a * 16384u, M.mA, kc * 32, ct * 128, i0 + a, bar);
        tma_load_2d(st + (uint32_t)M.na * 16384u, M.mB, kc * 32, 0, bar);
    }
    static __device__ __forceinline__ void mma(const TcGroup& g, const Tile& t, int kc, uint32_t st, uint32_t d) {
        const TcMat& M = g.mat[t.mat];
        int ct, i0, ni;
        decode(M, t.lt, ct, i0, ni);
        for (int a = 0; a < ni; ++a)
            mma_slice(d + (uint32_t)(a * M.rpad), st + a * 16384u, st + (uint32_t)M.na * 16384u, M.rpad, kc == 0);
    }
    static __device__ __forceinline__ bool epilogue(const TcGroup& g, const Tile& t, uint32_t tl, int warp, int lane, DataRing&) {
        const TcMat& M = g.mat[t.mat];
        int ct, i0, ni;
        decode(M, t.lt, ct, i0, ni);
        const int c = ct * 128 + 32 * (warp & 3) + lane;
        const int half = M.rpad / 2, q0 = (warp >> 2) * half;
        for (int a = 0; a < ni; ++a) {
            float* out = M.Rw + ((int64_t)(i0 + a) * M.np + c) * M.rpad;
            for (int q = q0; q < q0 + half; q += 16) {
                float v[16];
                tmem_ld16(tl + (uint32_t)(a * M.rpad + q), v);
                if (c < M.np) {
#pragma unroll
                    for (int j = 0; j < 16; j += 4)
                        *reinterpret_cast<float4*>(out + q + j) =
                            make_float4(rna_tf32(v[j]), rna_tf32(v[j + 1]), rna_tf32(v[j + 2]), rna_tf32(v[j + 3]));
                }
            }
        }
        return true;
    }
};

// ------------------------------------------------------------------------------------------
// Compose: tile = (128 rows a, 64 columns c).  D_i (128 x 64) = P_prev[a, :] R_w,i[:, c] (K = r)
// for every node; the epilogue forms M_i = G_i + B_i - D_i, writes B_i^T, and Mbar^T = mean_i M_i.
// A = P_prev (m' x r), B = R_w^T (3-D map rpad x n' x N).  Error reset (e_zero): no MMAs, M_i = G_i.
// Data stage of node i: B_i^T tile (64 columns x 128 rows fp32, 512 bytes a column, 32 KiB) and
// G_i's tile (bf16; 128 rows x 128 bytes with the 128-byte swizzle, or for m > n 64 columns x 256
// bytes), 16 KiB.  B_i^T is stored back from the stage.
// ------------------------------------------------------------------------------------------
struct Compose {
    static constexpr int kEpi = 16;
    static constexpr int BN = 64;
    static constexpr uint32_t kG = 32768;             // offset of the gradient tile in a data stage
    static __device__ __forceinline__ int nk(const TcGroup& g, const Tile& t) {
        const TcMat& M = g.mat[t.mat];
        return M.e_zero ? 0 : M.rpad / 32;
    }
    static __device__ __forceinline__ uint32_t tx_bytes(const TcGroup& g, const Tile& t, int) {
        return 16384u + (uint32_t)g.mat[t.mat].N * (BN * 128u);
    }
    static __device__ __forceinline__ void load(const TcGroup& g, const Tile& t, int kc, uint32_t st, uint32_t bar) {
        const TcMat& M = g.mat[t.mat];
        const int rt = t.lt / M.tn, ct = t.lt % M.tn;
        tma_load_2d(st, M.mA, kc * 32, rt * 128, bar);
        for (int i = 0; i < M.N; ++i) tma_load_3d(st + 16384u + i * (BN * 128u), M.mB, kc * 32, ct * BN, i, bar);
    }
    static __device__ __forceinline__ void mma(const TcGroup& g, const Tile& t, int kc, uint32_t st, uint32_t d) {
        const TcMat& M = g.mat[t.mat];
        for (int i = 0; i < M.N; ++i) mma_slice(d + (uint32_t)(i * BN), st, st + 16384u + i * (BN * 128u), BN, kc == 0);
    }
    static __device__ __forceinline__ int ndata(const TcGroup& g, const Tile& t) { return g.mat[t.mat].N; }
    static __device__ __forceinline__ uint32_t data_tx(const TcGroup& g, const Tile& t, int) {
        return (g.mat[t.mat].e_zero ? 0u : 32768u) + 16384u;
    }
    static __device__ __forceinline__ void data_load(const TcGroup& g, const Tile& t, int i, uint32_t st, uint32_t bar) {
        const TcMat& M = g.mat[t.mat];
        const int rt = t.lt / M.tn, ct = t.lt % M.tn;
        if (!M.e_zero) tma_load_3d(st, M.mD0, rt * 128, ct * BN, i, bar);
        if (M.transposed) tma_load_2d(st + kG, M.mD1 + i, rt * 128, ct * BN, bar);
        else tma_load_2d(st + kG, M.mD1 + i, ct * BN, rt * 128, bar);
    }
    static __device__ __forceinline__ bool epilogue(const TcGroup& g, const Tile& t, uint32_t tl, int warp, int lane,
                                                    DataRing& dr) {
        const TcMat& M = g.mat[t.mat];
        const int rt = t.lt / M.tn, ct = t.lt % M.tn;
        const int al = 32 * (warp & 3) + lane;            // row within the tile
        const int a = rt * 128 + al;
        const int cw = (warp >> 2) * 16;                  // this warp's 16 columns of the tile
        const int c0 = ct * BN + cw;
        const bool leader = warp == 0 && lane == 0;
        float acc[16];
#pragma unroll
        for (int j = 0; j < 16; ++j) acc[j] = 0.f;
        for (int i = 0; i < M.N; ++i) {
            uint8_t* sm = dr.acquire();
            if (!sm) return false;
            float* Bs = reinterpret_cast<float*>(sm) + al;    // B^T tile: column c at Bs[128 c]
            float m[16];
            if (!M.transposed) {
                const uint8_t* row = sm + kG + al * 128;
#pragma unroll
                for (int q = 0; q < 2; ++q) {
                    const uint4 u = *reinterpret_cast<const uint4*>(row + ((((cw >> 3) + q) ^ (al & 7)) << 4));
                    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
                    for (int h = 0; h < 4; ++h) {
                        const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[h]));
                        m[8 * q + 2 * h] = f.x;
                        m[8 * q + 2 * h + 1] = f.y;
                    }
                }
            } else {
                const __nv_bfloat16* col = reinterpret_cast<const __nv_bfloat16*>(sm + kG) + al;
#pragma unroll
                for (int j = 0; j < 16; ++j) m[j] = __bfloat162float(col[(cw + j) * 128]);
            }
            if (!M.e_zero) {
                float d[16];
                tmem_ld16(tl + (uint32_t)(i * BN + cw), d);
#pragma unroll
                for (int j = 0; j < 16; ++j) m[j] += Bs[(cw + j) * 128] - d[j];
            }
            if (M.write_B) {
#pragma unroll
                for (int j = 0; j < 16; ++j) Bs[(cw + j) * 128] = m[j];
            }
#pragma unroll
            for (int j = 0; j < 16; ++j) acc[j] += m[j];
            dr.release(leader, [&](uint32_t st) {
                if (!M.write_B) return false;
                tma_store_3d(M.mD0, rt * 128, ct * BN, i, st);
                return true;
            });
        }
        bool bad = false;
        if (a < M.mp) {
            const float invN = 1.0f / static_cast<float>(M.N);
#pragma unroll
            for (int j = 0; j < 16; ++j)
                if (c0 + j < M.np) {
                    const float v = acc[j] * invN;
                    bad |= !isfinite(v);
                    M.Mbar[(int64_t)(c0 + j) * M.mp + a] = v;
                }
            if (M.MbarRow) {                              // a refresh step: Mbar row-major as well
                float* row = M.MbarRow + (int64_t)a * M.np + c0;
#pragma unroll
                for (int j = 0; j < 16; j += 4)
                    if (c0 + j < M.np)
                        *reinterpret_cast<float4*>(row + j) =
                            make_float4(acc[j] * invN, acc[j + 1] * invN, acc[j + 2] * invN, acc[j + 3] * invN);
            }
        }
        flag_nonfinite(bad, M.nonfinite);
        return true;
    }
};

// ------------------------------------------------------------------------------------------
// WBar: tile = 256 columns c (two halves of 128).  D_h (128 x kpad) = Mbar^T[c, :] Y over
// K = m'; the epilogue writes W^T[c][q] (rounded to TF32).  A = Mbar^T (n' x m'), B = Y^T (kpad x m').
// ------------------------------------------------------------------------------------------
struct WBar : NoData {
    static __device__ __forceinline__ int nk(const TcGroup& g, const Tile& t) { return (g.mat[t.mat].mp + 31) / 32; }
    static __device__ __forceinline__ uint32_t tx_bytes(const TcGroup& g, const Tile& t, int) {
        return 2u * 16384u + (uint32_t)g.mat[t.mat].kpad * 128u;
    }
    static __device__ __forceinline__ void load(const TcGroup& g, const Tile& t, int kc, uint32_t st, uint32_t bar) {
        const TcMat& M = g.mat[t.mat];
        tma_load_2d(st, M.mA, kc * 32, t.lt * 256, bar);
        tma_load_2d(st + 16384u, M.mA, kc * 32, t.lt * 256 + 128, bar);
        tma_load_2d(st + 32768u, M.mB, kc * 32, 0, bar);
    }
    static __device__ __forceinline__ void mma(const TcGroup& g, const Tile& t, int kc, uint32_t st, uint32_t d) {
        const TcMat& M = g.mat[t.mat];
        mma_slice(d, st, st + 32768u, M.kpad, kc == 0);
        mma_slice(d + (uint32_t)M.kpad, st + 16384u, st + 32768u, M.kpad, kc == 0);
    }
    static __device__ __forceinline__ bool epilogue(const TcGroup& g, const Tile& t, uint32_t tl, int warp, int lane, DataRing&) {
        const TcMat& M = g.mat[t.mat];
        const int h = warp >> 2;
        const int c = t.lt * 256 + h * 128 + 32 * (warp & 3) + lane;
        float* out = M.W + (int64_t)c * M.kpad;
        for (int q = 0; q < M.kpad; q += 16) {
            float v[16];
            tmem_ld16(tl + (uint32_t)(h * M.kpad + q), v);
            if (c < M.np) {
#pragma unroll
                for (int j = 0; j < 16; j += 4)
                    *reinterpret_cast<float4*>(out + q + j) =
                        make_float4(rna_tf32(v[j]), rna_tf32(v[j + 1]), rna_tf32(v[j + 2]), rna_tf32(v[j + 3]));
            }
        }
        return true;
    }
};

// ------------------------------------------------------------------------------------------
// Lambda: tile = (128 rows j, 128 columns b).  D = Yt[j, :] W[:, b] (K = k); the epilogue adds
// (Mbar - D)(j, b) v_j[b] over each 32-column quarter into part[(4 ct + quarter) m' + j] (the
// signs D are applied when the partials are reduced).  A = Yt (m' x k), B = W^T (n' x kpad).  Data stage:
// the Mbar^T tile (128 columns x 128 rows fp32, 64 KiB).
// ------------------------------------------------------------------------------------------
struct Lambda {
    static constexpr int kEpi = 16;
    static __device__ __forceinline__ int nk(const TcGroup& g, const Tile& t) { return g.mat[t.mat].kpad / 32; }
    static __device__ __forceinline__ uint32_t tx_bytes(const TcGroup&, const Tile&, int) { return 2u * 16384u; }
    static __device__ __forceinline__ void load(const TcGroup& g, const Tile& t, int kc, uint32_t st, uint32_t bar) {
        const TcMat& M = g.mat[t.mat];
        const int rt = t.lt / M.tn, ct = t.lt % M.tn;
        tma_load_2d(st, M.mA, kc * 32, rt * 128, bar);
        tma_load_2d(st + 16384u, M.mB, kc * 32, ct * 128, bar);
    }
    static __device__ __forceinline__ void mma(const TcGroup&, const Tile&, int kc, uint32_t st, uint32_t d) {
        mma_slice(d, st, st + 16384u, 128, kc == 0);
    }
    static __device__ __forceinline__ int ndata(const TcGroup&, const Tile&) { return 1; }
    static __device__ __forceinline__ uint32_t data_tx(const TcGroup&, const Tile&, int) { return 65536u; }
    static __device__ __forceinline__ void data_load(const TcGroup& g, const Tile& t, int, uint32_t st, uint32_t bar) {
        const TcMat& M = g.mat[t.mat];
        const int rt = t.lt / M.tn, ct = t.lt % M.tn;
        tma_load_2d(st, M.mD0, rt * 128, ct * 128, bar);
    }
    static __device__ __forceinline__ bool epilogue(const TcGroup& g, const Tile& t, uint32_t tl, int warp, int lane,
                                                    DataRing& dr) {
        const TcMat& M = g.mat[t.mat];
        const int rt = t.lt / M.tn, ct = t.lt % M.tn;
        const int al = 32 * (warp & 3) + lane;
        const int j = rt * 128 + al;
        const int h = warp >> 2;                              // this warp's 32 columns
        const int b0 = ct * 128 + 32 * h;
        const uint8_t* sm = dr.acquire();
        if (!sm) return false;
        const float* Ms = reinterpret_cast<const float*>(sm) + al + (32 * h) * 128;   // column b0 + c at Ms[128 c]
        float acc = 0.f;
        for (int cc = 0; cc < 32; cc += 16) {
            float d[16];
            tmem_ld16(tl + (uint32_t)(32 * h + cc), d);
            if (j < M.mp) {
#pragma unroll
                for (int qq = 0; qq < 4; ++qq) {
                    const int b = b0 + cc + 4 * qq;
                    if (b >= M.np) break;
                    const float4 v = gauss4_fast(M.seed, M.t, (uint32_t)j, (uint32_t)(b >> 2), kTagLambdaV);
                    const float vv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        if (b + e < M.np) acc += (Ms[(cc + 4 * qq + e) * 128] - d[4 * qq + e]) * vv[e];
                }
            }
        }
        dr.release(warp == 0 && lane == 0, NoStore{});
        if (j < M.mp) M.part[(int64_t)(4 * ct + h) * M.mp + j] = acc;
        return true;
    }
};

// ------------------------------------------------------------------------------------------
// LambdaU (full basis): tile = (128 rows j, 256 columns b).  D = U^T[j, :] Mbar[:, b] (K = m',
// N = 256: each U^T slice serves 256 columns), and the epilogue adds D(j, b) v_j[b] over each
// warp's 64 columns into part[(4 ct + h) m' + j] (Algorithm 2's u_j^T Mbar v_j, the dense form of
// the scores).  A = U^T (m' x m', TF32), B = Mbar^T (n' x m') in two 128-row boxes.
// ------------------------------------------------------------------------------------------
struct LambdaU : NoData {
    static constexpr int kEpi = 16;
    static __device__ __forceinline__ int nk(const TcGroup& g, const Tile& t) { return (g.mat[t.mat].mp + 31) / 32; }
    static __device__ __forceinline__ uint32_t tx_bytes(const TcGroup&, const Tile&, int) { return 3u * 16384u; }
    static __device__ __forceinline__ void load(const TcGroup& g, const Tile& t, int kc, uint32_t st, uint32_t bar) {
        const TcMat& M = g.mat[t.mat];
        const int rt = t.lt / M.tn, ct = t.lt % M.tn;
        tma_load_2d(st, M.mA, kc * 32, rt * 128, bar);
        tma_load_2d(st + 16384u, M.mB, kc * 32, ct * 256, bar);
        tma_load_2d(st + 32768u, M.mB, kc * 32, ct * 256 + 128, bar);
    }
    static __device__ __forceinline__ void mma(const TcGroup&, const Tile&, int kc, uint32_t st, uint32_t d) {
        mma_slice(d, st, st + 16384u, 256, kc == 0);
    }
    static __device__ __forceinline__ bool epilogue(const TcGroup& g, const Tile& t, uint32_t tl, int warp, int lane,
                                                    DataRing&) {
        const TcMat& M = g.mat[t.mat];
        const int rt = t.lt / M.tn, ct = t.lt % M.tn;
        const int j = rt * 128 + 32 * (warp & 3) + lane;
        const int h = warp >> 2;                              // this warp's 64 columns
        const int b0 = ct * 256 + 64 * h;
        float acc = 0.f;
        for (int cc = 0; cc < 64; cc += 16) {
            float d[16];
            tmem_ld16(tl + (uint32_t)(64 * h + cc), d);
            if (j < M.mp) {
#pragma unroll
                for (int qq = 0; qq < 4; ++qq) {
                    const int b = b0 + cc + 4 * qq;
                    if (b >= M.np) break;
                    const float4 v = gauss4_fast(M.seed, M.t, (uint32_t)j, (uint32_t)(b >> 2), kTagLambdaV);
                    const float vv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        if (b + e < M.np) acc += d[4 * qq + e] * vv[e];
                }
            }
        }
        if (j < M.mp) M.part[(int64_t)(4 * ct + h) * M.mp + j] = acc;
        return true;
    }
};

// ------------------------------------------------------------------------------------------
// BjacMul (the blocked Jacobi of the full-basis refresh, k_bjac.cu): Y = X J_l over the 128
// columns of pair l, as three products per K slice (A B + A_lo B + A B_lo: the split TF32 form,
// about as accurate as fp32 FFMA); tile = (128-row block rt, pair l), K = 128.  Modes:
//   0: A = H rows, B = J_l^T:    D(i, c) = (H J)(i, 128 l + c), written to T^T (row 128 l + c)
//   1: A = T^T rows, B = J_l^T:  D(r, c) = (T^T J)(r, 128 l + c) = (J^T H J)(r, 128 l + c),
//      written transposed (the matrix is symmetric) at the next round's rows and columns
//   2: A = J_l^T, B = V rows:    D(c, r) = (V J)(r, 128 l + c), written to V' at row r and the
//      next round's column of 128 l + c
// With these orientations a warp's stores are 128 contiguous bytes.  Each output goes out with
// its TF32 low part x - trunc_tf32(x), the next product's second operand.
// ------------------------------------------------------------------------------------------
struct BjacMul : NoData {
    static constexpr int kEpi = 16;
    static __device__ __forceinline__ int nk(const TcGroup&, const Tile&) { return 4; }
    static __device__ __forceinline__ uint32_t tx_bytes(const TcGroup&, const Tile&, int) { return 4u * 16384u; }
    static __device__ __forceinline__ void load(const TcGroup& g, const Tile& t, int kc, uint32_t st, uint32_t bar) {
        const TcMat& M = g.mat[t.mat];
        const int P = M.mp / 128, rt = t.lt / P, l = t.lt % P;
        int ax, ay, bx, by;
        if (M.bjmode < 2) { ax = 128 * l + 32 * kc; ay = 128 * rt; bx = 32 * kc; by = 128 * l; }
        else { ax = 32 * kc; ay = 128 * l; bx = 128 * l + 32 * kc; by = 128 * rt; }
        tma_load_2d(st, M.mA, ax, ay, bar);
        tma_load_2d(st + 16384u, M.mA2, ax, ay, bar);
        tma_load_2d(st + 32768u, M.mB, bx, by, bar);
        tma_load_2d(st + 49152u, M.mB2, bx, by, bar);
    }
    static __device__ __forceinline__ void mma(const TcGroup&, const Tile&, int kc, uint32_t st, uint32_t d) {
        mma_slice(d, st, st + 32768u, 128, kc == 0);           // A B
        mma_slice(d, st + 16384u, st + 32768u, 128, false);    // A_lo B
        mma_slice(d, st, st + 49152u, 128, false);             // A B_lo
    }
    static __device__ __forceinline__ int dest(int x, int m, int rd) {
        return 64 * bjac_dest_of(x >> 6, m, rd) + (x & 63);
    }
    static __device__ __forceinline__ bool epilogue(const TcGroup& g, const Tile& t, uint32_t tl, int warp, int lane,
                                                    DataRing&) {
        const TcMat& M = g.mat[t.mat];
        const int n = M.mp, P = n / 128, m = n / 64, rt = t.lt / P, l = t.lt % P;
        const int row = 32 * (warp & 3) + lane, h = warp >> 2;
        // per-thread parts of the output index: a stride for the tile's columns, a fixed offset;
        // mode 1: a warp's 32 columns lie in one 64-block, whose next place is found once
        int64_t base = 0, step = 0;
        if (M.bjmode == 0) { base = (int64_t)(128 * l) * n + 128 * rt + row; step = n; }
        else if (M.bjmode == 1) {
            const int x0 = 128 * l + 32 * h;
            base = (int64_t)(64 * bjac_dest_of(x0 >> 6, m, M.bjround) + (x0 & 63)) * n + dest(128 * rt + row, m, M.bjround);
            step = n;
        } else { base = dest(128 * l + row, m, M.bjround); step = n; }
        for (int cc = 0; cc < 32; cc += 16) {
            float d[16];
            tmem_ld16(tl + (uint32_t)(32 * h + cc), d);
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                const int col = 32 * h + cc + e;
                const int64_t a = M.bjmode == 2 ? base + (int64_t)(128 * rt + col) * step
                                                : base + (int64_t)(cc + e + (M.bjmode == 0 ? 32 * h : 0)) * step;
                const float v = d[e];
                M.out[a] = v;
                M.out_lo[a] = v - __uint_as_float(__float_as_uint(v) & 0xffffe000u);
            }
        }
        return true;
    }
};

// ------------------------------------------------------------------------------------------
// PBuild: tile = 128 rows a.  D (128 x rpad) = Y[a, :] Yt[J, :]^T (K = k); the epilogue writes
// P(a, q) = d_{J_q} ([a == J_q] - D(a, q)) (rounded to TF32) and P^T.  A = Y (m' x k), B = YtJ
// (r x k, rows past r read as zeros).
// ------------------------------------------------------------------------------------------
struct PBuild : NoData {
    static __device__ __forceinline__ int nk(const TcGroup& g, const Tile& t) { return g.mat[t.mat].kpad / 32; }
    static __device__ __forceinline__ uint32_t tx_bytes(const TcGroup& g, const Tile& t, int) {
        return 16384u + (uint32_t)g.mat[t.mat].rpad * 128u;
    }
    static __device__ __forceinline__ void load(const TcGroup& g, const Tile& t, int kc, uint32_t st, uint32_t bar) {
        const TcMat& M = g.mat[t.mat];
        tma_load_2d(st, M.mA, kc * 32, t.lt * 128, bar);
        tma_load_2d(st + 16384u, M.mB, kc * 32, 0, bar);
    }
    static __device__ __forceinline__ void mma(const TcGroup& g, const Tile& t, int kc, uint32_t st, uint32_t d) {
        mma_slice(d, st, st + 16384u, g.mat[t.mat].rpad, kc == 0);
    }
    static __device__ __forceinline__ bool epilogue(const TcGroup& g, const Tile& t, uint32_t tl, int warp, int lane, DataRing&) {
        const TcMat& M = g.mat[t.mat];
        const int a = t.lt * 128 + 32 * (warp & 3) + lane;
        const int half = M.rpad / 2, q0 = (warp >> 2) * half;
        for (int q = q0; q < q0 + half; q += 16) {
            float d[16];
            tmem_ld16(tl + (uint32_t)q, d);
            if (a >= M.mp) continue;
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                const int qq = q + e;
                if (qq >= M.r) break;
                const int j = M.J[qq];
                float v = (a == j ? 1.f : 0.f) - d[e];
                if (j < M.k) v *= M.dsign[j];
                v = rna_tf32(v);
                M.Pout[(int64_t)a * M.r + qq] = v;
                M.PT[(int64_t)qq * M.mp + a] = v;
            }
        }
        return true;
    }
};

// ------------------------------------------------------------------------------------------
// RBar: tile = 128 columns b.  D (128 x 128) = Yt[J, :] W[:, b] (K = k, rows q >= r are zero);
// the epilogue writes Rbar^T(b, q) = d_{J_q} (Mbar(J_q, b) - D(q, b)) (rounded to TF32).  A = YtJ
// (r x k), B = W^T (n' x kpad).  Warp w: rows q = 32 (w % 4) + lane, columns 32 (w / 4) .. + 31;
// the 32 gathered Mbar(J_q, b) are loaded before any store so that they are all in flight.
// ------------------------------------------------------------------------------------------
struct RBar : NoData {
    static constexpr int kEpi = 16;
    static __device__ __forceinline__ int nk(const TcGroup& g, const Tile& t) { return g.mat[t.mat].kpad / 32; }
    static __device__ __forceinline__ uint32_t tx_bytes(const TcGroup&, const Tile&, int) { return 2u * 16384u; }
    static __device__ __forceinline__ void load(const TcGroup& g, const Tile& t, int kc, uint32_t st, uint32_t bar) {
        const TcMat& M = g.mat[t.mat];
        tma_load_2d(st, M.mA, kc * 32, 0, bar);
        tma_load_2d(st + 16384u, M.mB, kc * 32, t.lt * 128, bar);
    }
    static __device__ __forceinline__ void mma(const TcGroup&, const Tile&, int kc, uint32_t st, uint32_t d) {
        mma_slice(d, st, st + 16384u, 128, kc == 0);
    }
    static __device__ __forceinline__ bool epilogue(const TcGroup& g, const Tile& t, uint32_t tl, int warp, int lane, DataRing&) {
        const TcMat& M = g.mat[t.mat];
        const int q = 32 * (warp & 3) + lane;
        const int c0 = 32 * (warp >> 2);
        const int b0 = t.lt * 128 + c0;
        float d[32];
        tmem_ld16(tl + (uint32_t)c0, *reinterpret_cast<float(*)[16]>(d));
        tmem_ld16(tl + (uint32_t)(c0 + 16), *reinterpret_cast<float(*)[16]>(d + 16));
        if (q >= M.r) return true;
        const int j = M.J[q];
        const float dj = j < M.k ? M.dsign[j] : 1.f;
        const int nb = M.np - b0 < 32 ? M.np - b0 : 32;
        const float* col = M.Mbar + (int64_t)b0 * M.mp + j;     // Mbar(j, b0 + e) at col[e m']
        float mb[32];
#pragma unroll
        for (int e = 0; e < 32; ++e) mb[e] = e < nb ? __ldg(col + (int64_t)e * M.mp) : 0.f;
        float* out = M.RbarT + (int64_t)b0 * M.rpad + q;
#pragma unroll
        for (int e = 0; e < 32; ++e)
            if (e < nb) out[(int64_t)e * M.rpad] = rna_tf32(dj * (mb[e] - d[e]));
        return true;
    }
};

// ------------------------------------------------------------------------------------------
// Update (K3): tile = (128 rows a, 128 columns b).  Ghat = P[a, :] Rbar[:, b] (K = r), or Mbar
// when uncompressed (no MMAs); then the optimizer on X, Mo (, Vo) in X's layout (X(a, b) =
// X[a n' + b], or X[b m' + a] when m > n).  A = P (m' x r), B = Rbar^T (n' x rpad).  The tile's
// 128 columns pass through the data ring in four chunks of 32: X, Mo (, Vo) tiles of 128 x 32
// fp32 (16 KiB each; rows of 128 bytes with the 128-byte swizzle, or for m > n 32 columns of 512
// bytes), plus Mbar^T's tile when uncompressed; X, Mo, Vo are stored back from the stage.
// ------------------------------------------------------------------------------------------
struct Update {
    static constexpr int kEpi = 16;
    static __device__ __forceinline__ int nk(const TcGroup& g, const Tile& t) {
        const TcMat& M = g.mat[t.mat];
        return M.compressed ? M.rpad / 32 : 0;
    }
    static __device__ __forceinline__ uint32_t tx_bytes(const TcGroup&, const Tile&, int) { return 2u * 16384u; }
    static __device__ __forceinline__ void load(const TcGroup& g, const Tile& t, int kc, uint32_t st, uint32_t bar) {
        const TcMat& M = g.mat[t.mat];
        const int rt = t.lt / M.tn, ct = t.lt % M.tn;
        tma_load_2d(st, M.mA, kc * 32, rt * 128, bar);
        tma_load_2d(st + 16384u, M.mB, kc * 32, ct * 128, bar);
    }
    static __device__ __forceinline__ void mma(const TcGroup&, const Tile&, int kc, uint32_t st, uint32_t d) {
        mma_slice(d, st, st + 16384u, 128, kc == 0);
    }
    static __device__ __forceinline__ int ndata(const TcGroup&, const Tile&) { return 4; }
    static __device__ __forceinline__ uint32_t data_tx(const TcGroup& g, const Tile& t, int) {
        const TcMat& M = g.mat[t.mat];
        return 16384u * (2u + (g.optimizer != GLR_MSGD ? 1u : 0u) + (M.compressed ? 0u : 1u));
    }
    // x, y coordinates of chunk d in X's layout
    static __device__ __forceinline__ void xy(const TcMat& M, const Tile& t, int d, int& x, int& y) {
        const int rt = t.lt / M.tn, ct = t.lt % M.tn;
        if (M.transposed) { x = rt * 128; y = ct * 128 + 32 * d; }
        else { x = ct * 128 + 32 * d; y = rt * 128; }
    }
    static __device__ __forceinline__ void data_load(const TcGroup& g, const Tile& t, int d, uint32_t st, uint32_t bar) {
        const TcMat& M = g.mat[t.mat];
        int x, y;
        xy(M, t, d, x, y);
        tma_load_2d(st, M.mD0, x, y, bar);
        tma_load_2d(st + 16384u, M.mD1, x, y, bar);
        uint32_t off = 32768u;
        if (g.optimizer != GLR_MSGD) { tma_load_2d(st + off, M.mD2, x, y, bar); off += 16384u; }
        if (!M.compressed) {
            const int rt = t.lt / M.tn, ct = t.lt % M.tn;
            tma_load_2d(st + off, M.mD3, rt * 128, ct * 128 + 32 * d, bar);
        }
    }
    static __device__ __forceinline__ bool epilogue(const TcGroup& g, const Tile& t, uint32_t tl, int warp, int lane,
                                                    DataRing& dr) {
        const TcMat& M = g.mat[t.mat];
        const int al = 32 * (warp & 3) + lane;
        const int h = warp >> 2;                                  // this warp's 8 columns of each chunk
        const bool adam = g.optimizer != GLR_MSGD;
        const float lr = g.lr, b1 = g.beta1, b2 = g.beta2, eps = g.eps;
        const bool leader = warp == 0 && lane == 0;
        for (int d = 0; d < 4; ++d) {
            float gh[8];
            if (M.compressed) tmem_ld8(tl + (uint32_t)(32 * d + 8 * h), gh);
            uint8_t* sm = dr.acquire();
            if (!sm) return false;
            float* Xs = reinterpret_cast<float*>(sm);
            float* Ms = reinterpret_cast<float*>(sm + 16384);
            float* Vs = reinterpret_cast<float*>(sm + 32768);
            if (!M.compressed) {
                const float* Gs = reinterpret_cast<const float*>(sm + (adam ? 49152 : 32768)) + al;
#pragma unroll
                for (int e = 0; e < 8; ++e) gh[e] = Gs[(8 * h + e) * 128];
            }
            // this thread's 8 elements: row al, columns 8h .. 8h + 7 of the chunk; rows of 128 bytes
            // with the 128-byte swizzle are read as two 16-byte pieces (conflict-free), the columns
            // of 512 bytes (m > n) element by element (32 lanes, 32 consecutive floats)
            float x[8], mo[8], vo[8];
            int o[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                const int c = 8 * h + e;
                o[e] = M.transposed ? c * 128 + al : al * 32 + ((((c >> 2) ^ (al & 7)) << 2) | (c & 3));
            }
            if (M.transposed) {
#pragma unroll
                for (int e = 0; e < 8; ++e) { x[e] = Xs[o[e]]; mo[e] = Ms[o[e]]; if (adam) vo[e] = Vs[o[e]]; }
            } else {
#pragma unroll
                for (int p = 0; p < 2; ++p) {
                    const float4 a = *reinterpret_cast<const float4*>(Xs + o[4 * p]);
                    const float4 b = *reinterpret_cast<const float4*>(Ms + o[4 * p]);
                    x[4 * p] = a.x; x[4 * p + 1] = a.y; x[4 * p + 2] = a.z; x[4 * p + 3] = a.w;
                    mo[4 * p] = b.x; mo[4 * p + 1] = b.y; mo[4 * p + 2] = b.z; mo[4 * p + 3] = b.w;
                    if (adam) {
                        const float4 v = *reinterpret_cast<const float4*>(Vs + o[4 * p]);
                        vo[4 * p] = v.x; vo[4 * p + 1] = v.y; vo[4 * p + 2] = v.z; vo[4 * p + 3] = v.w;
                    }
                }
            }
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                const float gg = gh[e];
                mo[e] = b1 * mo[e] + (1.f - b1) * gg;
                if (adam) {
                    vo[e] = b2 * vo[e] + (1.f - b2) * gg * gg;
                    x[e] -= lr * mo[e] / (sqrtf(vo[e]) + eps);
                } else {
                    x[e] -= lr * mo[e];
                }
            }
            if (M.transposed) {
#pragma unroll
                for (int e = 0; e < 8; ++e) { Xs[o[e]] = x[e]; Ms[o[e]] = mo[e]; if (adam) Vs[o[e]] = vo[e]; }
            } else {
#pragma unroll
                for (int p = 0; p < 2; ++p) {
                    *reinterpret_cast<float4*>(Xs + o[4 * p]) = make_float4(x[4 * p], x[4 * p + 1], x[4 * p + 2], x[4 * p + 3]);
                    *reinterpret_cast<float4*>(Ms + o[4 * p]) =
                        make_float4(mo[4 * p], mo[4 * p + 1], mo[4 * p + 2], mo[4 * p + 3]);
                    if (adam)
                        *reinterpret_cast<float4*>(Vs + o[4 * p]) =
                            make_float4(vo[4 * p], vo[4 * p + 1], vo[4 * p + 2], vo[4 * p + 3]);
                }
            }
            dr.release(leader, [&](uint32_t st) {
                int x, y;
                xy(M, t, d, x, y);
                tma_store_2d(M.mD0, x, y, st);
                tma_store_2d(M.mD1, x, y, st + 16384u);
                if (adam) tma_store_2d(M.mD2, x, y, st + 32768u);
                return true;
            });
        }
        return true;
    }
};

// ------------------------------------------------------------------------------------------
// Refresh products.  PowT: tile = 256 rows c of n' (two halves of 128); D_h (128 x kpad) =
// Mbar^T[c, :] Q over K = m' (A = Mbar^T, B = Q^T TF32, kpad x m').  PowN: tile = 256 rows a of
// m'; D_h = Mbar[a, :] Z over K = n' (A = Mbar row-major, B = Z^T TF32, kpad x n'); with `split`
// the A slices of Mbar's low parts (Mbar - trunc_tf32(Mbar)) are multiplied too, so the product is
// exact to fp32 level for the TF32 value of B.  The epilogue writes out[row][q] (fp32, leading
// dimension ld_out, q < k) and outT[q][row] (TF32).
// ------------------------------------------------------------------------------------------
template <int kDir>
struct Pow : NoData {
    static __device__ __forceinline__ int nk(const TcGroup& g, const Tile& t) {
        const TcMat& M = g.mat[t.mat];
        return ((kDir == 0 ? M.mp : M.np) + 31) / 32;
    }
    static __device__ __forceinline__ uint32_t tx_bytes(const TcGroup& g, const Tile& t, int) {
        const TcMat& M = g.mat[t.mat];
        return (M.split ? 4u : 2u) * 16384u + (uint32_t)M.kpad * 128u;
    }
    static __device__ __forceinline__ void load(const TcGroup& g, const Tile& t, int kc, uint32_t st, uint32_t bar) {
        const TcMat& M = g.mat[t.mat];
        tma_load_2d(st, M.mA, kc * 32, t.lt * 256, bar);
        tma_load_2d(st + 16384u, M.mA, kc * 32, t.lt * 256 + 128, bar);
        uint32_t o = 32768u;
        if (M.split) {
            tma_load_2d(st + o, M.mA2, kc * 32, t.lt * 256, bar);
            tma_load_2d(st + o + 16384u, M.mA2, kc * 32, t.lt * 256 + 128, bar);
            o += 32768u;
        }
        tma_load_2d(st + o, M.mB, kc * 32, 0, bar);
    }
    static __device__ __forceinline__ void mma(const TcGroup& g, const Tile& t, int kc, uint32_t st, uint32_t d) {
        const TcMat& M = g.mat[t.mat];
        const uint32_t b = st + (M.split ? 65536u : 32768u);
        mma_slice(d, st, b, M.kpad, kc == 0);
        mma_slice(d + (uint32_t)M.kpad, st + 16384u, b, M.kpad, kc == 0);
        if (M.split) {
            mma_slice(d, st + 32768u, b, M.kpad, false);
            mma_slice(d + (uint32_t)M.kpad, st + 49152u, b, M.kpad, false);
        }
    }
    static __device__ __forceinline__ bool epilogue(const TcGroup& g, const Tile& t, uint32_t tl, int warp, int lane, DataRing&) {
        const TcMat& M = g.mat[t.mat];
        const int h = warp >> 2;
        const int c = t.lt * 256 + h * 128 + 32 * (warp & 3) + lane;
        for (int q = 0; q < M.kpad; q += 16) {
            float v[16];
            tmem_ld16(tl + (uint32_t)(h * M.kpad + q), v);
            if (c >= M.rows) continue;
#pragma unroll
            for (int j = 0; j < 16; j += 4)
                if (q + j < M.k)
                    *reinterpret_cast<float4*>(M.out + (int64_t)c * M.ld_out + q + j) =
                        make_float4(v[j], v[j + 1], v[j + 2], v[j + 3]);
#pragma unroll
            for (int j = 0; j < 16; ++j) M.outT[(int64_t)(q + j) * M.rows + c] = rna_tf32(v[j]);
        }
        return true;
    }
};
using PowT = Pow<0>;
using PowN = Pow<1>;

// ------------------------------------------------------------------------------------------
// Gram: tile = (matrix, chunk of kGramChunk rows).  D_h (128 x kpad) = X^T[h 128 .., rows] X over
// the chunk's rows (A = X^T slices of 128 rows, B = X^T with all kpad rows; X^T is TF32, kpad x
// rows).  The epilogue writes the chunk's partial Gram matrix out[chunk][l][l'] (kpad x kpad);
// the consumer sums the chunks in order.
// ------------------------------------------------------------------------------------------
struct Gram : NoData {
    static __device__ __forceinline__ int halves(const TcMat& M) { return (M.kpad + 127) / 128; }
    static __device__ __forceinline__ int nk(const TcGroup& g, const Tile& t) {
        const TcMat& M = g.mat[t.mat];
        const int r0 = t.lt * kGramChunk;
        const int len = M.rows - r0 < kGramChunk ? M.rows - r0 : kGramChunk;
        return (len + 31) / 32;
    }
    static __device__ __forceinline__ uint32_t tx_bytes(const TcGroup& g, const Tile& t, int) {
        const TcMat& M = g.mat[t.mat];
        return (uint32_t)halves(M) * 16384u + (uint32_t)M.kpad * 128u;
    }
    static __device__ __forceinline__ void load(const TcGroup& g, const Tile& t, int kc, uint32_t st, uint32_t bar) {
        const TcMat& M = g.mat[t.mat];
        const int x = t.lt * kGramChunk + kc * 32;
        for (int h = 0; h < halves(M); ++h) tma_load_2d(st + h * 16384u, M.mA, x, 128 * h, bar);
        tma_load_2d(st + 32768u, M.mB, x, 0, bar);
    }
    static __device__ __forceinline__ void mma(const TcGroup& g, const Tile& t, int kc, uint32_t st, uint32_t d) {
        const TcMat& M = g.mat[t.mat];
        for (int h = 0; h < halves(M); ++h)
            mma_slice(d + (uint32_t)(h * M.kpad), st + h * 16384u, st + 32768u, M.kpad, kc == 0);
    }
    static __device__ __forceinline__ bool epilogue(const TcGroup& g, const Tile& t, uint32_t tl, int warp, int lane, DataRing&) {
        const TcMat& M = g.mat[t.mat];
        const int h = warp >> 2;
        if (h >= halves(M)) return true;
        const int l = h * 128 + 32 * (warp & 3) + lane;
        float* out = M.out + ((int64_t)t.lt * M.kpad + l) * M.kpad;
        for (int q = 0; q < M.kpad; q += 16) {
            float v[16];
            tmem_ld16(tl + (uint32_t)(h * M.kpad + q), v);
            if (l >= M.kpad) continue;
#pragma unroll
            for (int j = 0; j < 16; j += 4)
                *reinterpret_cast<float4*>(out + q + j) = make_float4(v[j], v[j + 1], v[j + 2], v[j + 3]);
        }
        return true;
    }
};

// ------------------------------------------------------------------------------------------
// Apply: tile = 128 rows a.  D (128 x kpad) = X[a, :] Linv^T (K = kpad; A = X row-major rows x k,
// B = Linv row-major kpad x kpad, so that D = X L^{-T}); the epilogue writes X (in place: a tile
// reads only its own rows, all before the product completes) and X^T (TF32).  Warp w: lanes =
// rows, w / 4 picks a column half.
// ------------------------------------------------------------------------------------------
struct Apply : NoData {
    static __device__ __forceinline__ int nk(const TcGroup& g, const Tile& t) { return g.mat[t.mat].kpad / 32; }
    static __device__ __forceinline__ uint32_t tx_bytes(const TcGroup& g, const Tile& t, int) {
        return 16384u + (uint32_t)g.mat[t.mat].kpad * 128u;
    }
    static __device__ __forceinline__ void load(const TcGroup& g, const Tile& t, int kc, uint32_t st, uint32_t bar) {
        const TcMat& M = g.mat[t.mat];
        tma_load_2d(st, M.mA, kc * 32, t.lt * 128, bar);
        tma_load_2d(st + 16384u, M.mB, kc * 32, 0, bar);
    }
    static __device__ __forceinline__ void mma(const TcGroup& g, const Tile& t, int kc, uint32_t st, uint32_t d) {
        mma_slice(d, st, st + 16384u, g.mat[t.mat].kpad, kc == 0);
    }
    static __device__ __forceinline__ bool epilogue(const TcGroup& g, const Tile& t, uint32_t tl, int warp, int lane, DataRing&) {
        const TcMat& M = g.mat[t.mat];
        const int a = t.lt * 128 + 32 * (warp & 3) + lane;
        const int hw = M.kpad / 2, q0 = (warp >> 2) * hw;
        for (int q = q0; q < q0 + hw; q += 16) {
            float v[16];
            tmem_ld16(tl + (uint32_t)q, v);
            if (a >= M.rows) continue;
#pragma unroll
            for (int j = 0; j < 16; j += 4)
                if (q + j < M.k)
                    *reinterpret_cast<float4*>(M.out + (int64_t)a * M.ld_out + q + j) =
                        make_float4(v[j], v[j + 1], v[j + 2], v[j + 3]);
#pragma unroll
            for (int j = 0; j < 16; ++j) M.outT[(int64_t)(q + j) * M.rows + a] = rna_tf32(v[j]);
        }
        return true;
    }
};

// Stage bytes of an op for a group (the largest over its matrices).
template <class Op> size_t stage_bytes_of(const TcMat& M);
template <> size_t stage_bytes_of<PrevProj>(const TcMat& M) { return (size_t)M.na * 16384 + (size_t)M.rpad * 128; }
template <> size_t stage_bytes_of<Compose>(const TcMat& M) { return 16384 + (size_t)M.N * Compose::BN * 128; }
template <> size_t stage_bytes_of<WBar>(const TcMat& M) { return 2 * 16384 + (size_t)M.kpad * 128; }
template <> size_t stage_bytes_of<Lambda>(const TcMat&) { return 2 * 16384; }
template <> size_t stage_bytes_of<LambdaU>(const TcMat&) { return 3 * 16384; }
template <> size_t stage_bytes_of<BjacMul>(const TcMat&) { return 4 * 16384; }
template <> size_t stage_bytes_of<PBuild>(const TcMat& M) { return 16384 + (size_t)M.rpad * 128; }
template <> size_t stage_bytes_of<RBar>(const TcMat&) { return 2 * 16384; }
template <> size_t stage_bytes_of<Update>(const TcMat&) { return 2 * 16384; }
template <> size_t stage_bytes_of<PowT>(const TcMat& M) { return (M.split ? 4 : 2) * 16384 + (size_t)M.kpad * 128; }
template <> size_t stage_bytes_of<PowN>(const TcMat& M) { return (M.split ? 4 : 2) * 16384 + (size_t)M.kpad * 128; }
template <> size_t stage_bytes_of<Gram>(const TcMat& M) { return 2 * 16384 + (size_t)M.kpad * 128; }
template <> size_t stage_bytes_of<Apply>(const TcMat& M) { return 16384 + (size_t)M.kpad * 128; }

// Accumulator columns of one tile (two buffers when two fit in tensor memory).
template <class Op> int acc_cols_of(const TcMat& M);
template <> int acc_cols_of<PrevProj>(const TcMat& M) { return M.na * M.rpad; }
template <> int acc_cols_of<Compose>(const TcMat& M) { return M.N * Compose::BN; }
template <> int acc_cols_of<WBar>(const TcMat& M) { return 2 * M.kpad; }
template <> int acc_cols_of<Lambda>(const TcMat&) { return 128; }
template <> int acc_cols_of<LambdaU>(const TcMat&) { return 256; }
template <> int acc_cols_of<BjacMul>(const TcMat&) { return 128; }
template <> int acc_cols_of<PBuild>(const TcMat& M) { return M.rpad; }
template <> int acc_cols_of<RBar>(const TcMat&) { return 128; }
template <> int acc_cols_of<Update>(const TcMat&) { return 128; }
template <> int acc_cols_of<PowT>(const TcMat& M) { return 2 * M.kpad; }
template <> int acc_cols_of<PowN>(const TcMat& M) { return 2 * M.kpad; }
template <> int acc_cols_of<Gram>(const TcMat& M) { return ((M.kpad + 127) / 128) * M.kpad; }
template <> int acc_cols_of<Apply>(const TcMat& M) { return M.kpad; }

// Data-stage bytes of an op (0: no data ring).
template <class Op> size_t dstage_bytes_of(const TcGroup&, const TcMat&) { return 0; }
template <> size_t dstage_bytes_of<Compose>(const TcGroup&, const TcMat&) { return 49152; }
template <> size_t dstage_bytes_of<Lambda>(const TcGroup&, const TcMat&) { return 65536; }
template <> size_t dstage_bytes_of<Update>(const TcGroup& g, const TcMat& M) {
    return 16384 * (2 + (g.optimizer != GLR_MSGD ? 1 : 0) + (M.compressed ? 0 : 1));
}

int g_sms = 0;

template <class Op>
cudaError_t launch(TcGroup& g, cudaStream_t st) {
    if (g.nmat <= 0 || g.total_tiles <= 0) return cudaSuccess;
    size_t sb = 0, db = 0;
    int cols = 0;
    for (int i = 0; i < g.nmat; ++i) {
        sb = std::max(sb, stage_bytes_of<Op>(g.mat[i]));
        db = std::max(db, dstage_bytes_of<Op>(g, g.mat[i]));
        cols = std::max(cols, acc_cols_of<Op>(g.mat[i]));
    }
    if (cols > (int)kTmemCols) return cudaErrorInvalidValue;
    // without epilogue data: as many operand stages as fit; with it: two operand stages (one if
    // two leave no room for two data stages), then as many data stages as fit (at most four)
    int stages, dstages = 0;
    if (!db) {
        stages = std::min(static_cast<int>(kSmemBudget / sb), kMaxStages);
    } else {
        stages = kSmemBudget >= 2 * sb + 2 * db ? 2 : 1;
        dstages = std::min(static_cast<int>((kSmemBudget - stages * sb) / db), kMaxDStages);
        if (dstages < 1) return cudaErrorInvalidValue;
    }
    if (stages < 1) return cudaErrorInvalidValue;
    g.stages = stages;
    g.stage_bytes = static_cast<uint32_t>(sb);
    g.dstages = dstages;
    g.dstage_bytes = static_cast<uint32_t>(db);
    g.tbufs = 2 * cols <= (int)kTmemCols ? 2 : 1;
    size_t smem = (size_t)stages * sb + (size_t)dstages * db + 1024;
    if (smem < kMinSmem) smem = kMinSmem;
    if (!g_sms) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&g_sms, cudaDevAttrMultiProcessorCount, dev);
        if (g_sms <= 0) g_sms = 1;
    }
    cudaError_t e = cudaFuncSetAttribute(tc_kernel<Op>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int grid = std::min(g.total_tiles, g_sms);
    tc_kernel<Op><<<grid, threads_of<Op>(), smem, st>>>(g);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_prevproj(TcGroup& g, cudaStream_t st) { return launch<PrevProj>(g, st); }
cudaError_t launch_compose(TcGroup& g, cudaStream_t st) { return launch<Compose>(g, st); }
cudaError_t launch_wbar(TcGroup& g, cudaStream_t st) { return launch<WBar>(g, st); }
cudaError_t launch_lambda(TcGroup& g, cudaStream_t st) { return launch<Lambda>(g, st); }
cudaError_t launch_lambda_u(TcGroup& g, cudaStream_t st) { return launch<LambdaU>(g, st); }
cudaError_t launch_bjac(TcGroup& g, cudaStream_t st) { return launch<BjacMul>(g, st); }
cudaError_t launch_pbuild(TcGroup& g, cudaStream_t st) { return launch<PBuild>(g, st); }
cudaError_t launch_rbar(TcGroup& g, cudaStream_t st) { return launch<RBar>(g, st); }
cudaError_t launch_update(TcGroup& g, cudaStream_t st) { return launch<Update>(g, st); }
cudaError_t launch_powt(TcGroup& g, cudaStream_t st) { return launch<PowT>(g, st); }
cudaError_t launch_pown(TcGroup& g, cudaStream_t st) { return launch<PowN>(g, st); }
cudaError_t launch_gram(TcGroup& g, cudaStream_t st) { return launch<Gram>(g, st); }
cudaError_t launch_apply(TcGroup& g, cudaStream_t st) { return launch<Apply>(g, st); }

int compose_bn() { return Compose::BN; }

// ---- small helpers of the path ----------------------------------------------------------
namespace {
// dst (cols x ldd) = src^T rounded to TF32, src row-major rows x cols (leading dim lds); rows of
// dst past `rows` are left alone (zero from allocation).
// P = U[:, J] (m' x r, row-major) and P^T (r x m'), rounded to TF32: the projector of a full basis.
__global__ void gather_p_kernel(const float* __restrict__ U, int mp, const int32_t* __restrict__ J, int r,
                                float* __restrict__ P, float* __restrict__ PT) {
    const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= (int64_t)mp * r) return;
    const int q = (int)(e / mp), a = (int)(e % mp);
    const float v = rna_tf32(U[(int64_t)a * mp + J[q]]);
    P[(int64_t)a * r + q] = v;
    PT[(int64_t)q * mp + a] = v;
}

__global__ void transpose_round_kernel(float* dst, int ldd, const float* src, int rows, int cols, int lds) {
    __shared__ float tile[32][33];
    const int r0 = blockIdx.y * 32, c0 = blockIdx.x * 32;
    for (int y = threadIdx.y; y < 32; y += 8) {
        const int rr = r0 + y, cc = c0 + threadIdx.x;
        tile[y][threadIdx.x] = (rr < rows && cc < cols) ? src[(int64_t)rr * lds + cc] : 0.f;
    }
    __syncthreads();
    for (int y = threadIdx.y; y < 32; y += 8) {
        const int cc = c0 + y, rr = r0 + threadIdx.x;
        if (cc < cols && rr < rows) dst[(int64_t)cc * ldd + rr] = rna_tf32(tile[threadIdx.x][y]);
    }
}
__global__ void round_tf32_kernel(float* p, int64_t n) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        p[i] = rna_tf32(p[i]);
}
// E(a, b) = B^T[b][a] - sum_q P(a, q) Rw(q, b) (row-major m' x n'), Rw row-major r x n'.
__global__ void error_cm_kernel(const float* Bt, const float* P, const float* Rw, int mp, int np, int r, int e_zero,
                                float* E) {
    const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= (int64_t)mp * np) return;
    const int a = static_cast<int>(e / np), b = static_cast<int>(e % np);
    if (e_zero) { E[e] = 0.f; return; }            // an error reset: E = 0 whatever B holds
    float v = Bt[(int64_t)b * mp + a];
    for (int q = 0; q < r; ++q) v -= P[(int64_t)a * r + q] * Rw[(int64_t)q * np + b];
    E[e] = v;
}
}  // namespace

namespace {
// The bounded wait of the pipeline on an mbarrier that nothing arrives on: it gives up after
// `polls` polls, counts the event in *err (through the abort flag, as a stuck pipeline would)
// and the kernel returns.
__global__ void expire_kernel(int* err, int polls) {
    __shared__ __align__(8) uint64_t bar;
    __shared__ int abort_flag;
    if (threadIdx.x != 0) return;
    abort_flag = 0;
    mbar_init(smem_u32(&bar), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    wait_phase(smem_u32(&bar), 0, &abort_flag, err, polls);
}
}  // namespace

namespace {
// lo = x - (x truncated to TF32): what a TF32 product of x leaves out
__global__ void split_lo_kernel(const float4* src, float4* lo, int64_t n4) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += (int64_t)gridDim.x * blockDim.x) {
        const float4 v = src[i];
        auto l = [](float x) { return x - __uint_as_float(__float_as_uint(x) & 0xFFFFE000u); };
        lo[i] = make_float4(l(v.x), l(v.y), l(v.z), l(v.w));
    }
}
}  // namespace

cudaError_t split_lo(const float* src, float* lo, int64_t n, cudaStream_t st) {
    if (n % 4) return cudaErrorInvalidValue;
    split_lo_kernel<<<(unsigned)std::min<int64_t>((n / 4 + 255) / 256, 8 * 152), 256, 0, st>>>(
        reinterpret_cast<const float4*>(src), reinterpret_cast<float4*>(lo), n / 4);
    return cudaGetLastError();
}

cudaError_t expire_wait(int* err, int polls, cudaStream_t st) {
    expire_kernel<<<1, 32, 0, st>>>(err, polls);
    return cudaGetLastError();
}

cudaError_t gather_p(const float* U, int mp, const int32_t* J, int r, float* P, float* PT, cudaStream_t st) {
    const int64_t n = (int64_t)mp * r;
    gather_p_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(U, mp, J, r, P, PT);
    return cudaGetLastError();
}

cudaError_t transpose_round(float* dst, int ldd, const float* src, int rows, int cols, int lds, cudaStream_t st) {
    dim3 grid((cols + 31) / 32, (rows + 31) / 32), block(32, 8);
    transpose_round_kernel<<<grid, block, 0, st>>>(dst, ldd, src, rows, cols, lds);
    return cudaGetLastError();
}
cudaError_t round_tf32(float* p, int64_t n, cudaStream_t st) {
    round_tf32_kernel<<<(unsigned)std::min<int64_t>((n + 255) / 256, 4096), 256, 0, st>>>(p, n);
    return cudaGetLastError();
}
cudaError_t error_colmajor(const float* Bt, const float* P, const float* Rw, int mp, int np, int r, int e_zero,
                           float* E, cudaStream_t st) {
    const int64_t n = (int64_t)mp * np;
    error_cm_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(Bt, P, Rw, mp, np, r, e_zero, E);
    return cudaGetLastError();
}

}  // namespace tc
}  // namespace glr
