// Internal declarations shared by the CUDA translation units of libglr.so.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "glr.h"

namespace glr {

// ------------------------------------------------------------------------------------------
// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11) and Box-Muller: the random vectors
// v_j ~ N(0, I) of Eq. random-v.  Element (j, b) of the stacked m' x n' matrix uses counter
// (b / 4, j, t, tag) and key (seed lo, seed hi); the four output words give two Box-Muller
// pairs and v_j[b] = z_{b mod 4}.  Uniforms are (top 23 bits + 0.5) * 2^-23, exact in fp32.
// ------------------------------------------------------------------------------------------
constexpr uint32_t kTagLambdaV = 0x4C414D56u;   // v_j of Algorithm 2
constexpr uint32_t kTagPowerInit = 0x50574954u; // random start block of the power iteration

struct U32x4 { uint32_t x, y, z, w; };

__device__ __forceinline__ U32x4 philox4x32_10(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3,
                                               uint32_t k0, uint32_t k1) {
#pragma unroll
    for (int rnd = 0; rnd < 10; ++rnd) {
        if (rnd) { k0 += 0x9E3779B9u; k1 += 0xBB67AE85u; }
        const uint32_t hi0 = __umulhi(0xD2511F53u, c0), lo0 = 0xD2511F53u * c0;
        const uint32_t hi1 = __umulhi(0xCD9E8D57u, c2), lo1 = 0xCD9E8D57u * c2;
        const uint32_t n0 = hi1 ^ c1 ^ k0, n2 = hi0 ^ c3 ^ k1;
        c0 = n0; c1 = lo1; c2 = n2; c3 = lo0;
    }
    return {c0, c1, c2, c3};
}

// (top 23 bits + 1/2) 2^-23: exact in fp32, in [2^-24, 1 - 2^-24]
__device__ __forceinline__ float unit_open(uint32_t w) {
    return (static_cast<float>(w >> 9) + 0.5f) * 1.1920928955078125e-7f;  // 2^-23
}

// The four normals of quad q = b / 4 of row j.
__device__ __forceinline__ float4 gauss4(uint64_t seed, uint32_t t, uint32_t j, uint32_t q,
                                         uint32_t tag) {
    const U32x4 w = philox4x32_10(q, j, t, tag, static_cast<uint32_t>(seed),
                                  static_cast<uint32_t>(seed >> 32));
    float s0, c0, s1, c1;
    const float r0 = sqrtf(-2.0f * logf(unit_open(w.x)));
    const float r1 = sqrtf(-2.0f * logf(unit_open(w.z)));
    sincospif(2.0f * unit_open(w.y), &s0, &c0);
    sincospif(2.0f * unit_open(w.w), &s1, &c1);
    return make_float4(r0 * c0, r0 * s0, r1 * c1, r1 * s1);
}
// The same four normals with the hardware approximations of log, sin/cos and rsqrt: the draw for
// the v_j of the Approx-Top-r scores, where it runs once per element of every strip.  The
// approximate log has an absolute error of a few 1e-7 on [1/2, 2], so for u within ~1e-6 of 1
// -2 log u may come out as 0 or slightly negative; it is clamped to a tiny positive value
// (radius ~0 instead of at most ~1e-3), which keeps every normal finite.  Elsewhere the error is
// a few 1e-7 per normal.  cos/sin(2 pi u) are taken as -cos/-sin(pi (2u - 1)), whose argument
// lies in [-pi, pi), the range of the approximations' stated accuracy.
__device__ __forceinline__ float4 gauss4_fast(uint64_t seed, uint32_t t, uint32_t j, uint32_t q, uint32_t tag) {
    const U32x4 w = philox4x32_10(q, j, t, tag, static_cast<uint32_t>(seed),
                                  static_cast<uint32_t>(seed >> 32));
    constexpr float kPi = 3.14159265358979323846f;
    const float e0 = fmaxf(-2.0f * __logf(unit_open(w.x)), 1e-30f);
    const float e1 = fmaxf(-2.0f * __logf(unit_open(w.z)), 1e-30f);
    const float r0 = e0 * rsqrtf(e0), r1 = e1 * rsqrtf(e1);
    float s0, c0, s1, c1;
    __sincosf(kPi * fmaf(2.0f, unit_open(w.y), -1.0f), &s0, &c0);
    __sincosf(kPi * fmaf(2.0f, unit_open(w.w), -1.0f), &s1, &c1);
    return make_float4(-r0 * c0, -r0 * s0, -r1 * c1, -r1 * s1);
}

constexpr int kGroupMax = 32;          // matrices per grouped launch

// Streaming (evict-first) global stores of the error buffers.  Unlike the library's cache-hint
// store intrinsics these carry no memory clobber, which would make each store a compiler barrier
// and stop the shared-memory loads of the next rows from being scheduled across it; the kernels
// that use them never read the stored addresses back.
__device__ __forceinline__ void st_stream2(float* p, float a, float b) {
    asm("st.global.cs.v2.f32 [%0], {%1, %2};" ::"l"(p), "f"(a), "f"(b));
}
__device__ __forceinline__ void st_stream4(float* p, float a, float b, float c, float d) {
    asm("st.global.cs.v4.f32 [%0], {%1, %2, %3, %4};" ::"l"(p), "f"(a), "f"(b), "f"(c), "f"(d));
}

// A NaN or Inf in the node-mean gradient: one count per warp that holds any (flag may be null).
__device__ __forceinline__ void flag_nonfinite(bool bad, int* flag) {
    const unsigned m = __ballot_sync(__activemask(), bad);
    if (m && flag && static_cast<int>(threadIdx.x & 31) == __ffs(m) - 1) atomicAdd(flag, 1);
}

// ------------------------------------------------------------------------------------------
// Gradient element loads (fp32 or bf16, widened to fp32).
// ------------------------------------------------------------------------------------------
__device__ __forceinline__ float load_grad(const void* p, int64_t idx, int dtype) {
    if (dtype == GLR_BF16) return __bfloat162float(static_cast<const __nv_bfloat16*>(p)[idx]);
    return static_cast<const float*>(p)[idx];
}

// ------------------------------------------------------------------------------------------
// Launchers (all asynchronous on `st`; they return cudaGetLastError()).
// ------------------------------------------------------------------------------------------

// Strided, batched fp32 GEMM: for z < batch,
//   C_z(i, j) = alpha * sum_p A_z(i, p) B_z(p, j) + beta * C_z(i, j)
// with A_z(i, p) = A[z*sAz + i*sAi + p*sAp], B_z(p, j) = B[z*sBz + p*sBp + j*sBj],
// C_z(i, j) = C[z*sCz + i*sCi + j*sCj].  beta == 0 never reads C.  When few output tiles
// face a long K (the tall-skinny products of the refresh) and a workspace is given, K is split
// across CTAs whose partial tiles are summed afterwards in fixed order (no atomics).
struct GemmDesc {
    int M, N, K, batch;
    float alpha, beta;
    const float* A; int64_t sAz, sAi, sAp;
    const float* B; int64_t sBz, sBp, sBj;
    float* C;       int64_t sCz, sCi, sCj;
    float* ws = nullptr; int64_t ws_floats = 0;   // split-K workspace (optional)
};
constexpr int64_t kGemmWsFloats = int64_t(1) << 20;
cudaError_t gemm_f32(const GemmDesc& d, cudaStream_t st);

// K1 -- compose: for every node i and oriented element (a, b) of the m' x n' working layout
//   M_i(a, b) = G_i(a, b) + [!e_zero] (B_i(a, b) - sum_q Pprev(a, q) Rw_i(q, b))
//   B_i(a, b) = M_i(a, b)          (kept for the deferred error E_i = B_i - P P^T B_i)
//   Mbar(a, b) = (1/N) sum_i M_i(a, b)
// G_i is read in its caller layout (row-major m x n; transposed view when m > n).
struct ComposeArgs {
    const void* G[GLR_MAX_NODES];   // node gradients (device pointers)
    int grad_dtype;
    int transposed;         // 1: G_i(a, b) = G_i[b * m' + a]
    int mp, np, N, r;
    int e_zero;             // 1: E = 0 (skip B and the correction)
    int write_B;            // 0: warm-up steps, B is not needed
    float* B;               // N x m' x n'
    const float* Pprev;     // m' x r
    const float* Rw;        // N x r x n'  (Rw_i = Pprev^T B_i)
    float* Mbar;            // m' x n'
    int* nonfinite;         // counts warps that found a NaN / Inf in Mbar (may be null)
};
cudaError_t compose(const ComposeArgs& a, cudaStream_t st);

// Approx-Top-r partial sums: part[tb * m' + j] = sum_{b in tile tb} C(j, b) v_j[b] where
//   dense:  C = U^T Mbar                  (A(j, p) = U[p * m' + j], K = m')
//   wy:     C = Mbar - Yt Wbar            (A(j, c) = Yt[j * k + c], K = k)
struct LambdaArgs {
    int mode;               // 0 dense, 1 wy
    int mp, np, K;
    const float* A;         // U (dense) or Yt (wy)
    const float* Bm;        // Mbar (dense) or Wbar (wy)
    const float* Mbar;      // wy only
    const float* Csub;      // wy only, may be null: subtracted from Mbar as well (a precomputed Yt W)
    uint64_t seed; uint32_t t;
    float* part; int ntiles;
};
constexpr int kLambdaTile = 64;
cudaError_t lambda_partials(const LambdaArgs& a, cudaStream_t st);

// Reduce the partials in fixed order, apply the column signs d (k entries, may be null),
// pick J = the r largest lambda^2 (ties -> lower index), J ascending.
cudaError_t select_top_r(const float* part, int ntiles, int mp, int r, const float* dsign, int k,
                         float* lam, int32_t* J, cudaStream_t st);

// One CTA per matrix: lambda-bar from the partials (when do_select), J = arg-top-r, and
// P(:, q) = column J[q] of U (dense U, mode 0, or U = (I - Y Yt^T) D, mode 1).  r <= 1024.
struct SelectMat {
    const float* part; int ntiles;
    int mp, r, k, mode, do_select;
    const float* dsign; float* lam; int32_t* J;
    const float* U; const float* Y; const float* Yt; float* P;
    int rbar, np;                           // also form Rbar = P^T Mbar from Wbar (truncated basis)
    const float* Mbar; const float* Wbar; float* Rbar;
    int64_t out0;                           // first output of this matrix in pr_kernel
    int build_p;                            // 0: the caller forms P (wy_columns_*), pr_kernel skips it
    float* YtJ;                             // non-null: also gather YtJ = Yt[J, :] (r x k) after J
};
struct SelectGroup {
    int nmat;
    int64_t total_out;
    SelectMat mat[kGroupMax];
};
// stages: 1 = lambda-bar from the partials, 2 = arg-top-r, P and Rbar (3: both)
cudaError_t select_group(const SelectGroup& g, cudaStream_t st, int stages = 3);
// P = U[:, J] of a truncated basis U = (I - Y Yt^T) D formed around a library product:
// wy_columns_gather writes YtJ = Yt[J, :] (r x k); the caller forms P = -Y YtJ^T (m' x r);
// wy_columns_fix adds the identity columns e_{J_q} and scales column q by d_{J_q} (J_q < k).
cudaError_t wy_columns_gather(const float* Yt, const int32_t* J, int r, int k, float* YtJ, cudaStream_t st);
cudaError_t wy_columns_fix(float* P, const int32_t* J, const float* dsign, int mp, int r, int k, cudaStream_t st);

// P(:, q) = column J[q] of U: dense U (mode 0) or U = (I - Y Yt^T) D (mode 1).
cudaError_t build_P(int mode, int mp, int r, int k, const int32_t* J, const float* U,
                    const float* Y, const float* Yt, const float* dsign, float* P, cudaStream_t st);

// K3 -- decompress + optimizer: Ghat(a, b) = sum_q P(a, q) Rbar(q, b) (compressed) or
// Mbar(a, b), mapped back to X's layout (transposed when m > n), then MSGD / Adam.
struct UpdateArgs {
    int mp, np, r, transposed, compressed, optimizer;
    float lr, beta1, beta2, eps;
    const float* P; const float* Rbar; const float* Mbar;
    float* X; float* Mo; float* Vo;
};
cudaError_t update(const UpdateArgs& a, cudaStream_t st);
// The first path's streaming passes when its products run as library GEMMs (k_big.cu):
// compose_streamed takes B holding E_i (the correction already applied; r unused) and needs
// m' % 4 == n' % 4 == 0; update_streamed_flat takes Ghat in Mbar laid out like X (a.mp x a.np =
// X's element count as two factors) and runs the optimizer element by element.
cudaError_t compose_streamed(const ComposeArgs& a, cudaStream_t st);
cudaError_t update_streamed_flat(const UpdateArgs& a, cudaStream_t st);
// The AMSGrad-type optimizer step (k_big.cu): Ghat oriented m' x n', X / Mo / Vo in X's layout;
// vt[0] is the running scalar normaliser, vt[1] scratch for this step's maximum of V.
cudaError_t amsgrad_update(const float* Ghat, int mp, int np, int transposed, float* X, float* Mo, float* Vo,
                           float* vt, float lr, float beta1, float beta2, float eps, cudaStream_t st);
// Bias-corrected AdamW step (k_big.cu), same layouts; c1, c2 the bias corrections of this step.
cudaError_t adamw_update(const float* Ghat, int mp, int np, int transposed, float* X, float* Mo, float* Vo, float lr,
                         float beta1, float beta2, float eps, float wd, float c1, float c2, cudaStream_t st);
// Algorithm 5's subspace Adam (k_big.cu): Ms, Vs the EMAs of Rbar (total = r n' elements), Rh the
// step direction Ms / (sqrt(Vs) + eps); step_apply: X -= lr D, D oriented m' x n', X in its layout.
cudaError_t galore_moments(const float* Rbar, int64_t total, float* Ms, float* Vs, float* Rh, float beta1, float beta2,
                           float eps, cudaStream_t st);
cudaError_t step_apply(const float* D, int mp, int np, int transposed, float* X, float lr, cudaStream_t st);

// E_i = B_i - Pprev (Pprev^T B_i) given Rw_i = Pprev^T B_i  (or 0 when e_zero)
cudaError_t materialize_error(int mp, int np, int r, int e_zero, const float* B, const float* Pprev,
                              const float* Rw, float* E, cudaStream_t st);

// ---- refresh ------------------------------------------------------------------------------
// Cyclic two-sided Jacobi on the symmetric n x n matrix H (overwritten), one CTA:
// eigenvalues to evals, eigenvectors (columns) to V; the sweep count to *sweeps.
cudaError_t jacobi_eig(float* H, int n, float* V, float* evals, int* sweeps, cudaStream_t st);
// Sort eigenpairs by descending eigenvalue, write the first ncols vectors as columns of Out
// (rows x ncols, row-major, leading dim ldo), largest-|entry| of each column positive.
cudaError_t sort_fix_basis(const float* evals, const float* V, int n, int ncols, float* Out,
                           int ldo, float* evals_sorted, cudaStream_t st);
// Make the largest-|entry| of each column of A (rows x cols, row-major) positive.
cudaError_t fix_column_signs(float* A, int rows, int cols, cudaStream_t st);
// In-place Cholesky of the n x n SPD matrix A (lower factor in the lower triangle); if a
// pivot is not positive the diagonal is shifted and the factorisation restarted (*flag =
// number of restarts).  scratch: n*n floats.
cudaError_t cholesky(float* A, int n, float* scratch, int* flag, cudaStream_t st);
// S = L^{-T} for L L^T = G (n x n SPD, n <= 256), one CTA with the factor in shared memory; the
// same shifted retries as cholesky(), attempts counted in *flag.
cudaError_t chol_inverse(const float* G, int n, float* S, int* flag, cudaStream_t st);
// The same factor and inverse for several Gram matrices (one CTA each), each given as the sum of
// nparts partial matrices (leading dimension ld, ld * ld apart); writes L^{-1} row-major ld x ld.
struct CholMat { const float* part; int nparts, ld, n; float* out; int* flag; int tri_only; };   // tri_only: (U^T)^{-1} of the upper triangle of part (n x n)
struct CholGroup { int nmat; CholMat mat[64]; };
cudaError_t chol_group(const CholGroup& g, cudaStream_t st);
// The end of a truncated refresh for several matrices, one launch per stage: stage 0 sorts each
// eigenproblem's pairs by descending value and writes W (k x k, unit columns, signs fixed) and the
// sorted values; 1 fixes the column signs of Q (m' x k); 2 and 3 the Householder reconstruction
// (top block into Wtop, Y, T, s; then the rows below).
struct FinishMat {
    int mp, k;
    const float* evals; const float* V; float* W; float* evals_sorted;
    float* Q; float* Wtop; float* Y; float* T; float* s;
};
struct FinishGroup { int nmat; FinishMat mat[64]; };
cudaError_t finish_group(const FinishGroup& g, int stage, cudaStream_t st);
// C = A B in fp32 (FFMA) for several independent products, one launch: A(i, p) = A[i sAi + p sAp],
// B(p, j) = B[p sBp + j sBj], C(i, j) = C[i sCi + j sCj]; 64 x 64 output tiles.
struct GemmMat {
    int M, N, K;
    float alpha;                          // C = alpha A B (0 is read as 1)
    const float* A; int64_t sAi, sAp;
    const float* B; int64_t sBp, sBj;
    float* C; int64_t sCi, sCj;
    int tile0;
};
struct GemmGroup { int nmat, total_tiles; GemmMat mat[64]; };
cudaError_t gemm_group_f32(GemmGroup& g, cudaStream_t st);

// Full-basis refresh of several matrices at once (k_jacobi.cu): parallel cyclic Jacobi on each
// n x n Gram matrix H (n <= 1024; H and H2 are overwritten, the eigenvalues end in evals) with
// eigenvectors in V, spread over one cooperative grid.  part: 2 nmat grid floats; bar: two ints
// (zeroed by the launcher); err counts barrier waits that gave up; sweeps receives the sweeps
// each matrix took.  jacobi_group_grid() is 0 where cooperative launches are unavailable.
struct JacobiMat {
    int n; float tol;
    float* H; float* H2; float* V; float* evals;   // H2: a second n x n buffer (rounds alternate)
    int* sweeps;
    int soff;               // first float of this matrix's rotations in shared memory (see jacobi_rot_floats)
};
constexpr int kJacobiMaxGrid = 1024;
constexpr size_t kJacobiMaxSmem = 96 * 1024;     // the group's rotations; groups are split to fit
size_t jacobi_rot_floats(int n);
struct JacobiGroup {
    int nmat, max_sweeps;
    int* bar; int* err; float* part;
    JacobiMat mat[kGroupMax];
};
// The k x k Rayleigh-Ritz eigenproblems of truncated refreshes (k_eig.cu): one CTA per matrix,
// H (row-major, n <= 256, read only; summed from partial matrices) -> eigenvalues (unsorted) and eigenvectors V (row-major
// n x n, column j for evals[j]); sweeps done in *sweeps.
struct EigMat {
    int n; float tol;
    const float* H; int nparts, ld;       // H = the sum of nparts matrices (leading dimension ld, ld * ld apart)
    float* V; float* evals; int* sweeps;
};
constexpr int kEigGroupMax = 64;
struct EigGroup {
    int nmat, max_sweeps;
    EigMat mat[kEigGroupMax];
};
cudaError_t eig_tmem_group(const EigGroup& g, cudaStream_t st);

// The blocked Jacobi's round-robin tournament over m blocks of 64 indices (circle method: block 0
// fixed, the others one slot further each round; slots s and m - 1 - s pair up and are stored at
// positions 2 s, 2 s + 1): the storage position of block x in round rd, the block at position p,
// and where the data at position p of round rd goes for round rd + 1.
__host__ __device__ __forceinline__ int bjac_position_of(int x, int m, int rd) {
    const int s = x == 0 ? 0 : 1 + ((x - 1 - rd) % (m - 1) + (m - 1)) % (m - 1);
    return s < m / 2 ? 2 * s : 2 * (m - 1 - s) + 1;
}
__host__ __device__ __forceinline__ int bjac_block_at(int p, int m, int rd) {
    const int s = (p & 1) ? m - 1 - (p >> 1) : (p >> 1);
    return s == 0 ? 0 : 1 + (s - 1 + rd) % (m - 1);
}
__host__ __device__ __forceinline__ int bjac_dest_of(int p, int m, int rd) {
    return bjac_position_of(bjac_block_at(p, m, rd), m, (rd + 1) % (m - 1));
}

// Blocked Jacobi rounds of the full-basis refresh above m' = 1024 (k_bjac.cu; the rotations are
// tc_kernel<BjacMul> in k_tc.cu).  H: this round's n x n matrix in the round's storage order;
// J, Jlo: the round's n / 128 pair rotations as J_k^T (128 x 128 row-major each) and their TF32
// low parts.
constexpr int kBjacMaxN = 4096;
constexpr int kBjacGroupMax = 32;
constexpr int kBjacNormCtas = 64;
struct BjacMat {
    int n;
    const float* H;
    float* J; float* Jlo;
    int tile0p;
};
struct BjacGroup {
    int nmat;
    BjacMat mat[kBjacGroupMax];
};
// J_k^T of every pair of every matrix: one Jacobi sweep on H's 128 x 128 diagonal pair blocks
cudaError_t bjac_pairs(BjacGroup& g, cudaStream_t st);
// The start of a solve: H = sum of nparts partials (leading dimension ld; nparts = 0: H given),
// H_lo = H - trunc_tf32(H), V = I, V_lo = 0 (all n x n row-major)
struct BjacPrep {
    const float* part; int nparts, ld, n;
    float *H, *Hlo, *V, *Vlo;
};
struct BjacPrepGroup {
    int nmat;
    BjacPrep mat[kBjacGroupMax];
};
cudaError_t bjac_prep(const BjacPrepGroup& g, cudaStream_t st);
// part[2 (i kBjacNormCtas + c) + {0, 1}]: CTA c's squared diagonal / off-diagonal sums of H_i
cudaError_t bjac_norms(const BjacGroup& g, float* part, cudaStream_t st);
cudaError_t bjac_eye(float* V, int n, cudaStream_t st);
cudaError_t bjac_diag(const float* H, int n, float* evals, cudaStream_t st);
cudaError_t count_flag(int* flag, int v, cudaStream_t st);   // *flag += v on the device
int jacobi_group_grid();
cudaError_t jacobi_group(const JacobiGroup& g, int grid, cudaStream_t st);
// Q <- Q L^{-T} for the rows x n matrix Q (row-major) and lower-triangular L.
cudaError_t trsm_right_lt(float* Q, int rows, int n, const float* L, cudaStream_t st);
// Random Gaussian start block (rows x cols) from Philox with the power-iteration tag.
cudaError_t random_block(float* Q, int rows, int cols, uint64_t seed, uint32_t t, cudaStream_t st);
// Householder reconstruction (modified LU, Ballard et al. 2015) of orthonormal Q (mp x k):
// Y (mp x k unit lower trapezoidal), T (k x k upper), s (k signs) with (I - Y T Y^T)[:, :k]
// diag(s) = Q.  Work: scratch of k*k floats.
cudaError_t householder_reconstruct(const float* Q, int mp, int k, float* Y, float* T, float* s,
                                    float* scratch, cudaStream_t st);
// U = (I - Y Yt^T) D materialised (mp x mp).
cudaError_t materialize_wy_basis(int mp, int k, const float* Y, const float* Yt, const float* dsign,
                                 float* U, cudaStream_t st);

// ------------------------------------------------------------------------------------------
// Fused, grouped streaming kernels (one launch for every matrix of a group).  A CTA owns a
// strip of BN columns of one matrix's oriented m' x n' layout and all of its m' rows.
// ------------------------------------------------------------------------------------------
constexpr int kGroupPtrs = 512;        // node gradient pointers per grouped launch
constexpr int kFusedThreads = 1024;    // K1: one 4 x 4 block per thread, so m' <= 4096 * 4 / BN
constexpr int kUpdateThreads = 256;    // K3
constexpr int kMmaThreads = 512;       // K1 on the tensor cores (k_mma.cu)

struct StreamMat {
    int mp, np, N, r, k;
    int transposed, e_zero, write_B, lam;   // lam: truncated-basis lambda partials in the epilogue
    int g_off;                              // first gradient pointer of this matrix in StreamGroup::G
    int strip0, nstrips;                    // CTAs [strip0, strip0 + nstrips) work on this matrix
    float* B; const float* Pprev; float* Mbar;
    const float* YT; const float* YtT; float* part;   // Y^T, Yt^T (k x transposed_pitch(m')); part: nstrips x m'
    const float* YF; const float* YtF;                // Y, Yt in the tensor-core kernel's fragment order
    float* Wbar;                                      // tensor-core kernel: W = Y^T Mbar written here when set
    int* nonfinite;                                   // counts warps that found a NaN / Inf in Mbar
    uint64_t seed; uint32_t t;
};
struct StreamGroup {
    int nmat, grad_dtype, total_strips, BN;
    int* err;                               // bounded device waits that gave up are counted here
    StreamMat mat[kGroupMax];
    const void* G[kGroupPtrs];
};
// Tile-copy descriptors of the tensor-core K1 launch: B of each matrix (3-D: n' x m' x N) and
// each node gradient (2-D: n' x m'), boxes of 16 columns x mma_tma_box_rows(m') rows.  Passed
// by value as a kernel parameter (with StreamGroup under the 32 KiB parameter limit).
constexpr int kTmaGMax = 128;
struct TmaMaps {
    CUtensorMap B[kGroupMax];
    CUtensorMap G[kTmaGMax];
};
// K1 fused: per strip and node, R = Pprev^T B_i (deferred error), M_i = G_i + B_i - Pprev R,
// B_i <- M_i, Mbar; with lam = 1 also W = Y^T Mbar_strip and the lambda partial sums of
// (Mbar - Yt W) against v_j over the strip's columns.
cudaError_t stream_group(const StreamGroup& g, size_t smem_bytes, cudaStream_t st);
size_t stream_smem_bytes(int mp, int r, int k, int BN, int gsize, int transposed, int lam);
// Row pitch of the k x m' transposed copies (YT, YtT and the shared P^T of the FFMA kernel):
// 16-byte rows covering m' rounded up to 16; consecutive rows start 4 (or 20) banks apart.
__host__ __device__ __forceinline__ int transposed_pitch(int mp) { return ((mp + 15) & ~15) + 4; }
// K1 with its rank-r products on the tensor cores (3xTF32 mma.sync): strips of 16 columns,
// m' <= 512 for r <= 8 and m' <= 256 for r <= 16, truncated basis k <= 32.  One launch takes
// matrices of one mma_stream_nq(r) only.  With `maps` the ring is filled by tile copies (G read
// in its stored orientation, n' x gsize a multiple of 16 bytes), else by cp.async.
constexpr int kMmaStrip = 16;
int mma_stream_nq(int r);
bool mma_stream_eligible(int mp, int np, int r, int k, int lam, int transposed, int gsize);
bool mma_stream_tma_eligible(int mp, int np, int r, int k, int lam, int transposed, int gsize);
size_t mma_stream_smem_bytes(int mp, int r, int k, int lam, int gsize, int transposed, int tma);
int mma_tma_box_rows(int mp);
cudaError_t stream_group_mma(const StreamGroup& g, const TmaMaps* maps, size_t smem_bytes, cudaStream_t st);
// src (rows x cols, row-major, leading dimension ld) in the tensor-core kernel's fragment order
// (up8(rows) x up8(cols) floats, zero-padded); form 0 for Y, form 1 for Yt.
cudaError_t pack_frag(float* dst, const float* src, int rows, int cols, int ld, int form, cudaStream_t st);
// dst (cols x tp) = src^T for row-major src (rows x cols), entries a >= rows set to 0.
cudaError_t transpose_pad(float* dst, int tp, const float* src, int rows, int cols, cudaStream_t st);

struct UpdateMat {
    int mp, np, r, transposed, compressed;
    int strip0, nstrips;
    const float* P; float* Rbar; const float* Mbar;
    float* X; float* Mo; float* Vo;
};
struct UpdateGroup {
    int nmat, total_strips, BN, optimizer;
    float lr, beta1, beta2, eps;
    UpdateMat mat[kGroupMax];
};
// K3 fused: Rbar_strip = P^T Mbar_strip, Ghat = P Rbar (or Mbar), MSGD / Adam on X.
cudaError_t update_group(const UpdateGroup& g, size_t smem_bytes, cudaStream_t st);
size_t update_smem_bytes(int mp, int r, int BN);

// K3 for compressed steps of a truncated basis (k_update.cu): with Rbar formed by the selection
// (pr_kernel, from K1's Wbar), Ghat = P Rbar and MSGD / Adam streamed over X;
// update_stream_tiles() CTAs per matrix.
struct UpdStreamMat {
    int mp, np, r, k, transposed;
    int tile0, ntiles;                      // update_stream_kernel CTAs of this matrix
    const int32_t* J; const float* dsign; const float* Yt; const float* Wbar; const float* Mbar; const float* P;
    float* Rbar; float* X; float* Mo; float* Vo;
};
struct UpdStreamGroup {
    int nmat, total_tiles, optimizer;
    float lr, beta1, beta2, eps;
    UpdStreamMat mat[kGroupMax];
};
int update_stream_tiles(int mp, int np, int transposed);
bool update_stream_eligible(int mp, int r, int transposed);
cudaError_t update_stream_group(const UpdStreamGroup& g, cudaStream_t st);    // Ghat and the optimizer

// Grouped block power iteration of the truncated-basis refresh (k_power.cu), k <= 32.  Per
// matrix: t0/nt column tiles of pow_tile() columns (Mbar^T Q), n0 the first of nn x nr CTAs of
// the split-K product Mbar Z (nn chunks of pow_chunk() columns, nr row tiles of pow_tile() rows),
// r0/nr row tiles (reduction, apply).  part holds nn x KM x m' floats, G max(nt, nr) x KM x KM
// (KM = 16 for k <= 16, else 32); S, H are k x k.
struct PowMat {
    int mp, np, k, active;
    int t0, nt, n0, nn, r0, nr;
    const float* Mbar;
    float* Q; float* Z; float* part; float* G; float* S; float* H;
    int* flag;
};
struct PowGroup {
    int nmat, tot_t, tot_n, tot_r;
    PowMat mat[kGroupMax];
};
int pow_tile();
int pow_chunk();
// stage 0: Z = (Mbar^T Q) (S if arg) + Gram partials; 1: split-K partials of Mbar Z; 2: Q = (sum)
// S + Gram partials; 3: Q <- Q S (+ Gram partials if arg); 4: S <- chol(sum of Gram partials)^-T
// (arg: the partials of stage 0, else of stages 2/3); 5: H <- sum of the stage-0 partials.
cudaError_t pow_stage(const PowGroup& g, int stage, int arg, cudaStream_t st);

// ------------------------------------------------------------------------------------------
// The large-matrix path on the tcgen05 tensor cores (k_tc.cu).  Node buffers B_i and Mbar are
// column-major (B_i^T: n' x m'); P row-major m' x r with P^T (rpad x m'); R_w,i^T (n' x rpad per
// node), W^T (n' x kpad), Rbar^T (n' x rpad), Y^T (kpad x m'); rpad = r and kpad = k rounded up
// to 32.  Each launch takes up to kTcGroupMax matrices; a matrix's tiles are [tile0, tile0 +
// ntiles) of the launch.  Tensor maps live in device memory (one table per handle).
// ------------------------------------------------------------------------------------------
namespace tc {
constexpr int kTcGroupMax = 64;
constexpr int kTcGPtrs = 512;
struct TcMat {
    int mp, np, N, r, rpad, k, kpad;
    int transposed, gdtype, e_zero, write_B, compressed;
    int tile0, ntiles, tm, tn;            // this op's tiles of the matrix: tm x tn (or tn x ng node groups)
    int ng, na;                           // PrevProj: node groups of na nodes
    int g_off;                            // Compose: first gradient pointer in TcGroup::G
    const CUtensorMap* mA; const CUtensorMap* mB;      // the MMA operands
    const CUtensorMap* mD0; const CUtensorMap* mD1;    // epilogue data: Compose B^T, gradients (N maps);
    const CUtensorMap* mD2; const CUtensorMap* mD3;    // Update X, Mo, Vo, Mbar^T; Lambda Mbar^T
    float* B; float* Mbar; float* Rw; float* W; float* part;
    const int32_t* J; const float* dsign;
    float* Pout; float* PT; float* Rbar; float* RbarT;
    float* X; float* Mo; float* Vo;
    int* nonfinite;                                   // Compose: counts warps that found a NaN / Inf in Mbar
    uint64_t seed; uint32_t t;
    // refresh products (PowT, PowN, Gram, Apply): a second A operand (PowN split), the rows of the
    // operand they stream, their outputs (fp32, leading dimension ld_out) and TF32 transposes
    const CUtensorMap* mA2;
    int rows, ld_out, split, chunk;
    float* out; float* outT;
    float* MbarRow;                                   // Compose on a refresh step: Mbar row-major too
    // BjacMul (the blocked Jacobi's rotations): the second B operand (B's TF32 low parts; mA2 holds
    // A's), the output mode and the tournament round, the output's low parts
    const CUtensorMap* mB2;
    int bjmode, bjround;
    float* out_lo;
};
struct TcGroup {
    int nmat, total_tiles;
    int stages; uint32_t stage_bytes; int tbufs;     // set by the launcher: operand ring, accumulators
    int dstages; uint32_t dstage_bytes;              // ... and the epilogue's data ring
    int optimizer;                                   // Update: the optimizer of every matrix in the launch
    float lr, beta1, beta2, eps;
    int* err;                                        // bounded waits that gave up are counted here
    TcMat mat[kTcGroupMax];
    const void* G[kTcGPtrs];
};
cudaError_t launch_prevproj(TcGroup& g, cudaStream_t st);
cudaError_t launch_compose(TcGroup& g, cudaStream_t st);
cudaError_t launch_wbar(TcGroup& g, cudaStream_t st);
cudaError_t launch_lambda(TcGroup& g, cudaStream_t st);
cudaError_t launch_lambda_u(TcGroup& g, cudaStream_t st);   // full basis: the scores from U^T Mbar
// The blocked Jacobi's rotations in the split TF32 form (k_tc.cu, BjacMul; modes in k_tc.cu)
cudaError_t launch_bjac(TcGroup& g, cudaStream_t st);
cudaError_t launch_pbuild(TcGroup& g, cudaStream_t st);
cudaError_t launch_rbar(TcGroup& g, cudaStream_t st);
cudaError_t launch_update(TcGroup& g, cudaStream_t st);
// Truncated refresh products (k_tc.cu): PowT Z = Mbar^T Q, PowN Q = Mbar Z (TF32, or with the
// split A = A_hi + A_lo for fp32-level accuracy), Gram partial sums of X^T X over row chunks, Apply
// X <- X Linv^T.  Each writes its fp32 result and a TF32-rounded transpose.
cudaError_t launch_powt(TcGroup& g, cudaStream_t st);
cudaError_t launch_pown(TcGroup& g, cudaStream_t st);
cudaError_t launch_gram(TcGroup& g, cudaStream_t st);
cudaError_t launch_apply(TcGroup& g, cudaStream_t st);
constexpr int kGramChunk = 512;                  // rows per Gram partial
// Mlo = Mrow - trunc_tf32(Mrow), elementwise over n elements
cudaError_t split_lo(const float* src, float* lo, int64_t n, cudaStream_t st);
int compose_bn();
// dst (cols x ldd) = src^T rounded to TF32 (src row-major rows x cols, leading dimension lds)
cudaError_t transpose_round(float* dst, int ldd, const float* src, int rows, int cols, int lds, cudaStream_t st);
// P = U[:, J] (m' x r) and P^T (r x m') rounded to TF32, U row-major m' x m'
cudaError_t gather_p(const float* U, int mp, const int32_t* J, int r, float* P, float* PT, cudaStream_t st);
cudaError_t round_tf32(float* p, int64_t n, cudaStream_t st);
// One wait of the pipeline's bounded kind on an mbarrier that never completes, `polls` polls.
cudaError_t expire_wait(int* err, int polls, cudaStream_t st);
// E (row-major m' x n') = B^T - P Rw with B^T column-major (n' x m'), Rw row-major r x n'
cudaError_t error_colmajor(const float* Bt, const float* P, const float* Rw, int mp, int np, int r, int e_zero,
                           float* E, cudaStream_t st);
}  // namespace tc

// Message reported by glr_last_error(NULL) for entry points that have no handle.
void set_global_error(const char* msg);

}  // namespace glr
