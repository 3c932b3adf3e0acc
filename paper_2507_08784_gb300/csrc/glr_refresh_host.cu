// The Semi-Lazy SVD refresh of Eq. SVD-P1 on the host side: the order of the refresh kernels for
// a truncated basis (block power iteration with CholeskyQR, Rayleigh-Ritz, the Householder WY
// form; grouped across matrices through k_power.cu when k <= 32) and for the full basis (the
// cooperative Jacobi of all refreshing matrices, k_jacobi.cu).  Each handle's refresh runs on its
// own side stream.
#include "glr_host.cuh"

namespace glr {
namespace host {

// A (rows x k, row-major) <- A L^{-T} with L L^T = A^T A (CholeskyQR): the k x k factor and its
// inverse in one CTA, then one product into tmp; A and tmp trade places.
int cholqr(glr_handle* h, float*& A, float*& tmp, int rows, cudaStream_t st) {
    const int k = h->k;
    GLR_GEMM(h, gd(k, k, rows, A, 1, k, A, k, 1, h->gram, k, 1), st);
    if (k > 256) {                           // the factor does not fit one CTA's shared memory
        GLR_LAUNCH(h, 1, cholesky(h->gram, k, h->scratch, h->dflags + 0, st));
        GLR_LAUNCH(h, 1, trsm_right_lt(A, rows, k, h->gram, st));
        return GLR_OK;
    }
    GLR_LAUNCH(h, 1, chol_inverse(h->gram, k, h->scratch, h->dflags + 0, st));
    GLR_GEMM(h, gd(rows, k, k, A, k, 1, h->scratch, k, 1, tmp, k, 1), st);
    std::swap(A, tmp);
    return GLR_OK;
}

int wy_from_Q(glr_handle* h, cudaStream_t st) {
    const int mp = h->mp, k = h->k;
    GLR_LAUNCH(h, 2, householder_reconstruct(h->Q, mp, k, h->Y, h->T, h->dsign, h->scratch, st));
    // Yt = Y T^T
    GLR_GEMM(h, gd(mp, k, k, h->Y, k, 1, h->T, 1, k, h->Yt, k, 1), st);
    // transposed copies (k x tp, zero-padded) for the fused compose kernel's lambda epilogue
    GLR_LAUNCH(h, 1, transpose_pad(h->YT, transposed_pitch(mp), h->Y, mp, k, st));
    GLR_LAUNCH(h, 1, transpose_pad(h->YtT, transposed_pitch(mp), h->Yt, mp, k, st));
    if (h->mma) {
        GLR_LAUNCH(h, 1, pack_frag(h->YF, h->Y, mp, k, k, 0, st));
        GLR_LAUNCH(h, 1, pack_frag(h->YtF, h->Yt, mp, k, k, 1, st));
    }
    if (h->tcl) GLR_LAUNCH(h, 1, tc::transpose_round(h->YTk, mp, h->Y, mp, k, k, st));   // Y^T for the W products
    return GLR_OK;
}

// Rayleigh-Ritz after the k x k eigen-decomposition H = W diag W^T (eigenvalues in evals, W in
// Vk): Q <- Q W (columns by descending Ritz value, signs fixed), then the WY form.
int refresh_finish(glr_handle* h, cudaStream_t st) {
    const int mp = h->mp, k = h->k;
    GLR_LAUNCH(h, 1, sort_fix_basis(h->evals, h->Vk, k, k, h->gram, k, h->evals_sorted, st));
    GLR_GEMM(h, gd(mp, k, k, h->Q, k, 1, h->gram, k, 1, h->Qn, k, 1), st);
    GLR_LAUNCH(h, 1, fix_column_signs(h->Qn, mp, k, st));
    std::swap(h->Q, h->Qn);
    return wy_from_Q(h, st);
}

// End of a truncated refresh, with Q orthonormal and H = Q^T Mbar Mbar^T Q in Hk: the k x k
// Jacobi in one CTA, then refresh_finish.
int refresh_tail(glr_handle* h, cudaStream_t st) {
    GLR_LAUNCH(h, 1, jacobi_eig(h->Hk, h->k, h->Vk, h->evals, h->dflags + 1, st));
    return refresh_finish(h, st);
}

// Truncated refreshes of several matrices through the grouped block power iteration
// (k_power.cu): the same iteration as refresh_power (q power iterations, each half re-normalised by
// CholeskyQR, then CholeskyQR2 and the Rayleigh-Ritz Gram), one launch per stage for all of
// them on the first handle's side stream; the k x k tails run on each handle's own stream.
int refresh_grouped(std::vector<glr_handle*>& hs) {
    glr_handle* h0 = hs[0];
    cudaStream_t s0 = h0->rstream;
    for (glr_handle* h : hs) GLR_CK(h0, cudaStreamWaitEvent(s0, h->rfork, 0));
    {
        PhaseScope ps(h0, GLR_PH_REFRESH, s0);
        PowGroup g{};
        const int PC = pow_tile(), CH = pow_chunk();
        int q = h0->s.power_iters;
        for (glr_handle* h : hs) {
            if (h->refreshes == 0 && !h->basis_from_user)
                GLR_LAUNCH(h0, 1, random_block(h->Q, h->mp, h->k, h->s.seed, static_cast<uint32_t>(h->t), s0));
            PowMat& M = g.mat[g.nmat++];
            M.mp = h->mp; M.np = h->np; M.k = h->k; M.active = 1;
            M.t0 = g.tot_t; M.nt = (h->np + PC - 1) / PC; g.tot_t += M.nt;
            M.r0 = g.tot_r; M.nr = (h->mp + PC - 1) / PC; g.tot_r += M.nr;
            M.n0 = g.tot_n; M.nn = (h->np + CH - 1) / CH; g.tot_n += M.nn * M.nr;
            M.Mbar = h->Mbar; M.Q = h->Q; M.Z = h->Z; M.part = h->powpart; M.G = h->powG; M.S = h->powS;
            M.H = h->Hk; M.flag = h->dflags + 0;
            q = std::max(q, h->s.power_iters);
        }
        // a matrix with fewer power iterations than the group's maximum drops out early
        for (int it = 0; it < q; ++it) {
            for (int i = 0; i < g.nmat; ++i) g.mat[i].active = it < hs[i]->s.power_iters ? 1 : 0;
            GLR_LAUNCH(h0, 1, pow_stage(g, 0, it > 0 ? 1 : 0, s0));   // Z = (Mbar^T Q) S
            GLR_LAUNCH(h0, 1, pow_stage(g, 4, 1, s0));                // S = chol(Z^T Z)^-T
            GLR_LAUNCH(h0, 1, pow_stage(g, 1, 0, s0));                // partials of Mbar Z
            GLR_LAUNCH(h0, 1, pow_stage(g, 2, 0, s0));                // Q = (Mbar Z) S
            GLR_LAUNCH(h0, 1, pow_stage(g, 4, 0, s0));                // S = chol(Q^T Q)^-T
        }
        for (int i = 0; i < g.nmat; ++i) g.mat[i].active = 1;
        GLR_LAUNCH(h0, 1, pow_stage(g, 3, 1, s0));                    // CholeskyQR2: Q <- Q S ...
        GLR_LAUNCH(h0, 1, pow_stage(g, 4, 0, s0));
        GLR_LAUNCH(h0, 1, pow_stage(g, 3, 0, s0));                    // ... twice: orthonormal
        GLR_LAUNCH(h0, 1, pow_stage(g, 0, 0, s0));                    // Rayleigh-Ritz: Z = Mbar^T Q
        GLR_LAUNCH(h0, 1, pow_stage(g, 5, 1, s0));                    // H = Z^T Z
    }
    GLR_CK(h0, cudaEventRecord(h0->rpow, s0));
    for (glr_handle* h : hs) {
        if (h != h0) GLR_CK(h, cudaStreamWaitEvent(h->rstream, h0->rpow, 0));
        PhaseScope ps(h, GLR_PH_REFRESH, h->rstream);
        g_ws = h->gemm_ws;
        const int rc = refresh_tail(h, h->rstream);
        g_ws = nullptr;
        if (rc != GLR_OK) return rc;
    }
    return GLR_OK;
}

// Full-basis refreshes of several matrices: H = Mbar Mbar^T on each handle's side stream, one
// cooperative Jacobi launch for all of them on the first handle's side stream (k_jacobi.cu), then
// each handle sorts its eigenvectors by descending eigenvalue and fixes their signs on its own.
int refresh_exact_grouped(std::vector<glr_handle*>& hs) {
    {   // above m' = 1024: the blocked solver (tcgen05 path only)
        std::vector<glr_handle*> big, small;
        for (glr_handle* h : hs) (h->mp > kMaxFullBasis ? big : small).push_back(h);
        if (!big.empty()) {
            std::stable_sort(big.begin(), big.end(), [](const glr_handle* a, const glr_handle* b) { return a->mp < b->mp; });
            const int rc = refresh_exact_blocked(big);
            if (rc != GLR_OK) return rc;
        }
        if (small.empty()) return GLR_OK;
        hs.swap(small);
    }
    const int grid = jacobi_group_grid();
    for (size_t c0 = 0, c1 = 0; c0 < hs.size(); c0 = c1) {
        // a group: at most kGroupMax matrices whose rotations fit the kernel's shared memory
        size_t rot = 0;
        for (c1 = c0; c1 < hs.size() && c1 - c0 < (size_t)kGroupMax; ++c1) {
            const size_t add = jacobi_rot_floats(hs[c1]->mp) * sizeof(float);
            if (c1 > c0 && rot + add > kJacobiMaxSmem) break;
            rot += add;
        }
        glr_handle* h0 = hs[c0];
        cudaStream_t s0 = h0->rstream;
        for (size_t i = c0; i < c1; ++i) {
            glr_handle* h = hs[i];
            PhaseScope ps(h, GLR_PH_REFRESH, h->rstream);
            const int mp = h->mp, np = h->np;
            GLR_GEMM(h, gd(mp, mp, np, h->Mbar, np, 1, h->Mbar, 1, np, h->Hbuf, mp, 1), h->rstream);
            if (!grid) {                                         // no cooperative launch: one CTA each
                GLR_LAUNCH(h, 1, jacobi_eig(h->Hbuf, mp, h->Vbuf, h->evals, h->dflags + 1, h->rstream));
                GLR_LAUNCH(h, 1, sort_fix_basis(h->evals, h->Vbuf, mp, mp, h->U, mp, h->evals_sorted, h->rstream));
                continue;
            }
            GLR_CK(h, cudaEventRecord(h->rpow, h->rstream));
            if (h != h0) GLR_CK(h0, cudaStreamWaitEvent(s0, h->rpow, 0));
        }
        if (!grid) continue;
        JacobiGroup g{};
        size_t soff = 0;
        g.max_sweeps = 40;
        g.bar = h0->dflags + 4; g.err = h0->dflags + 2; g.part = h0->jpart;
        for (size_t i = c0; i < c1; ++i) {
            glr_handle* h = hs[i];
            JacobiMat& M = g.mat[g.nmat++];
            const int n = h->mp;
            M.n = n; M.tol = 4.f * 5.96e-8f * sqrtf(static_cast<float>(n)) + 1e-7f;
            M.H = h->Hbuf; M.H2 = h->jwork; M.V = h->Vbuf; M.evals = h->evals;
            M.sweeps = h->dflags + 1;
            M.soff = (int)soff;
            soff += jacobi_rot_floats(n);
        }
        {
            PhaseScope ps(h0, GLR_PH_REFRESH, s0);
            GLR_LAUNCH(h0, 1, jacobi_group(g, grid, s0));
        }
        GLR_CK(h0, cudaEventRecord(h0->rpow, s0));
        for (size_t i = c0; i < c1; ++i) {
            glr_handle* h = hs[i];
            if (h != h0) GLR_CK(h, cudaStreamWaitEvent(h->rstream, h0->rpow, 0));
            PhaseScope ps(h, GLR_PH_REFRESH, h->rstream);
            GLR_LAUNCH(h, 1, sort_fix_basis(h->evals, h->Vbuf, h->mp, h->mp, h->U, h->mp, h->evals_sorted, h->rstream));
        }
    }
    return GLR_OK;
}

// The blocked Jacobi (k_bjac.cu) for a set of symmetric n x n problems, n a multiple of 128 from
// 256 to 4096: the full basis's m' x m' eigenproblem, or a truncated refresh's k x k Rayleigh-Ritz
// problem.  Each problem lives in its handle's buffers (H in Hbuf with its low part in Hlo, T^T in
// jwork / Ttlo, V in Vbuf / Vbuf2 with Vlo / V2lo, the rotations in bjJ / bjJlo) and the kMapBj*
// tensor maps over them; bjac_prep has set H, H_lo, V = I, V_lo = 0.  The problems of one size run
// together, one sweep at a time, each sweep opened by the norm check (per-CTA partials summed on
// the host in a fixed order, so that the decision does not depend on the grouping); a round is the
// pair sweeps (J_k^T and its low part), then the three split-TF32 products of tc_kernel<BjacMul>:
// T^T = (H J)^T, H <- T^T J, V' <- V J.  A problem that has not converged after kBjacMaxSweeps
// sweeps keeps its last V and counts a numeric failure (GLR_ENUMERIC from glr_get_stats).
constexpr int kBjacMaxSweeps = 30;

struct BjItem {
    glr_handle* h;
    int n, vpar, rd;
    bool done;
    const float* V() const { return vpar ? h->Vbuf2 : h->Vbuf; }
};

int bjac_run(std::vector<BjItem>& all, glr_handle* h0, cudaStream_t s0) {
    std::stable_sort(all.begin(), all.end(), [](const BjItem& a, const BjItem& b) { return a.n < b.n; });
    std::vector<float> part;
    static thread_local tc::TcGroup tg;
    for (size_t a0 = 0; a0 < all.size();) {
        size_t a1 = a0;                                         // the problems of one size
        while (a1 < all.size() && all[a1].n == all[a0].n) ++a1;
        const int n = all[a0].n, m = n / 64, P = n / 128;
        const double tol = 4.0 * 5.96e-8 * std::sqrt((double)n) + 1e-7;
        for (int sweep = 0;; ++sweep) {
            std::vector<BjItem*> act;
            for (size_t i = a0; i < a1; ++i)
                if (!all[i].done) act.push_back(&all[i]);
            for (size_t c0 = 0; c0 < act.size(); c0 += kBjacGroupMax) {
                BjacGroup g{};
                for (size_t c = c0; c < act.size() && c < c0 + kBjacGroupMax; ++c) {
                    BjacMat& M = g.mat[g.nmat++];
                    M.n = n; M.H = act[c]->h->Hbuf;
                }
                GLR_LAUNCH(h0, 1, bjac_norms(g, h0->bjpart, s0));
                part.resize((size_t)2 * kBjacNormCtas * g.nmat);
                GLR_CK(h0, cudaMemcpyAsync(part.data(), h0->bjpart, sizeof(float) * part.size(), cudaMemcpyDeviceToHost, s0));
                GLR_CK(h0, cudaStreamSynchronize(s0));
                for (int i = 0; i < g.nmat; ++i) {
                    double d = 0.0, o = 0.0;
                    for (int c = 0; c < kBjacNormCtas; ++c) {
                        d += part[2 * ((size_t)i * kBjacNormCtas + c)];
                        o += part[2 * ((size_t)i * kBjacNormCtas + c) + 1];
                    }
                    BjItem* S = act[c0 + i];
                    if (o <= tol * tol * (o + d)) S->done = true;
                    else if (sweep == kBjacMaxSweeps) {
                        S->done = true;
                        S->h->numeric_failures_host++;
                    }
                    if (S->done) S->h->bj_sweeps = sweep;
                }
            }
            act.erase(std::remove_if(act.begin(), act.end(), [](BjItem* S) { return S->done; }), act.end());
            if (act.empty()) break;
            for (int round = 0; round < m - 1; ++round) {
                for (size_t c0 = 0; c0 < act.size(); c0 += kBjacGroupMax) {
                    BjacGroup g{};
                    for (size_t c = c0; c < act.size() && c < c0 + kBjacGroupMax; ++c) {
                        BjacMat& M = g.mat[g.nmat++];
                        M.n = n; M.H = act[c]->h->Hbuf; M.J = act[c]->h->bjJ; M.Jlo = act[c]->h->bjJlo;
                    }
                    GLR_LAUNCH(h0, 1, bjac_pairs(g, s0));
                }
                for (int mode = 0; mode < 3; ++mode) {
                    for (size_t c0 = 0; c0 < act.size(); c0 += tc::kTcGroupMax) {
                        tg.nmat = 0; tg.total_tiles = 0; tg.err = h0->dflags + 2;
                        for (size_t c = c0; c < act.size() && c < c0 + tc::kTcGroupMax; ++c) {
                            const BjItem* S = act[c];
                            glr_handle* h = S->h;
                            tc::TcMat M{};
                            M.mp = n; M.ntiles = P * P; M.tile0 = tg.total_tiles; M.bjmode = mode; M.bjround = S->rd;
                            const int vin = S->vpar ? kMapBjV1 : kMapBjV0;
                            if (mode == 0) {
                                M.mA = tcl_map(h, kMapBjH); M.mA2 = tcl_map(h, kMapBjHlo);
                                M.mB = tcl_map(h, kMapBjJ); M.mB2 = tcl_map(h, kMapBjJlo);
                                M.out = h->jwork; M.out_lo = h->Ttlo;
                            } else if (mode == 1) {
                                M.mA = tcl_map(h, kMapBjT); M.mA2 = tcl_map(h, kMapBjTlo);
                                M.mB = tcl_map(h, kMapBjJ); M.mB2 = tcl_map(h, kMapBjJlo);
                                M.out = h->Hbuf; M.out_lo = h->Hlo;
                            } else {
                                M.mA = tcl_map(h, kMapBjJ); M.mA2 = tcl_map(h, kMapBjJlo);
                                M.mB = tcl_map(h, vin); M.mB2 = tcl_map(h, vin + 1);
                                M.out = S->vpar ? h->Vbuf : h->Vbuf2; M.out_lo = S->vpar ? h->Vlo : h->V2lo;
                            }
                            tg.total_tiles += M.ntiles;
                            tg.mat[tg.nmat++] = M;
                        }
                        GLR_LAUNCH(h0, 1, tc::launch_bjac(tg, s0));
                    }
                }
                for (BjItem* S : act) {
                    S->vpar ^= 1;
                    S->rd = (S->rd + 1) % (m - 1);
                }
            }
        }
        a0 = a1;
    }
    for (BjItem& S : all) {
        glr_handle* h = S.h;
        GLR_CK(h, cudaMemcpyAsync(h->dflags + 1, &h->bj_sweeps, sizeof(int), cudaMemcpyHostToDevice, s0));
        if (h->numeric_failures_host) {
            GLR_LAUNCH(h, 1, count_flag(h->dflags + 6, h->numeric_failures_host, s0));
            h->numeric_failures_host = 0;
        }
    }
    return GLR_OK;
}

// bjac_prep over the items (in groups); part(h) gives a problem's partials and their count and
// leading dimension (count 0: H is already in Hbuf).
template <class Parts>
int bjac_prepare(const std::vector<BjItem>& items, glr_handle* h0, cudaStream_t s0, Parts parts) {
    for (size_t c0 = 0; c0 < items.size(); c0 += kBjacGroupMax) {
        BjacPrepGroup g{};
        for (size_t c = c0; c < items.size() && c < c0 + kBjacGroupMax; ++c) {
            glr_handle* h = items[c].h;
            BjacPrep& P = g.mat[g.nmat++];
            P.n = items[c].n; P.H = h->Hbuf; P.Hlo = h->Hlo; P.V = h->Vbuf; P.Vlo = h->Vlo;
            parts(h, P);
        }
        GLR_LAUNCH(h0, 1, bjac_prep(g, s0));
    }
    return GLR_OK;
}

// Full-basis refreshes above m' = 1024, all on the first handle's side stream: H = Mbar Mbar^T by
// the grouped FFMA product (Mbar is column-major on the tcgen05 path), the blocked Jacobi, then
// each handle's sorted, sign-fixed U and its TF32 transpose.
int refresh_exact_blocked(std::vector<glr_handle*>& hs) {
    glr_handle* h0 = hs[0];
    cudaStream_t s0 = h0->rstream;
    for (glr_handle* h : hs) {
        if (h == h0) continue;
        GLR_CK(h, cudaEventRecord(h->rpow, h->rstream));
        GLR_CK(h0, cudaStreamWaitEvent(s0, h->rpow, 0));
    }
    PhaseScope ps(h0, GLR_PH_REFRESH, s0);
    {   // H = Mbar Mbar^T (Mbar^T is n' x m' row-major)
        GemmGroup gg{};
        auto flush = [&]() -> int {
            if (gg.nmat) GLR_LAUNCH(h0, 1, gemm_group_f32(gg, s0));
            gg.nmat = 0;
            return GLR_OK;
        };
        for (glr_handle* h : hs) {
            GemmMat& G = gg.mat[gg.nmat++];
            G = GemmMat{};
            G.M = h->mp; G.N = h->mp; G.K = h->np; G.alpha = 1.f;
            G.A = h->Mbar; G.sAi = 1; G.sAp = h->mp;
            G.B = h->Mbar; G.sBp = h->mp; G.sBj = 1;
            G.C = h->Hbuf; G.sCi = h->mp; G.sCj = 1;
            if (gg.nmat == 64 && flush() != GLR_OK) return GLR_ECUDA;
        }
        if (flush() != GLR_OK) return GLR_ECUDA;
    }
    std::vector<BjItem> items;
    for (glr_handle* h : hs) items.push_back(BjItem{h, h->mp, 0, 0, false});
    int rc = bjac_prepare(items, h0, s0, [](glr_handle*, BjacPrep& P) { P.nparts = 0; });
    if (rc == GLR_OK) rc = bjac_run(items, h0, s0);
    if (rc != GLR_OK) return rc;
    for (const BjItem& S : items) {
        glr_handle* h = S.h;
        const int n = h->mp;
        GLR_LAUNCH(h, 1, bjac_diag(h->Hbuf, n, h->evals, s0));
        GLR_LAUNCH(h, 1, sort_fix_basis(h->evals, S.V(), n, n, h->U, n, h->evals_sorted, s0));
        GLR_LAUNCH(h, 1, tc::transpose_round(h->UT, n, h->U, n, n, n, s0));
    }
    GLR_CK(h0, cudaEventRecord(h0->rpow, s0));
    for (glr_handle* h : hs)
        if (h != h0) GLR_CK(h, cudaStreamWaitEvent(h->rstream, h0->rpow, 0));
    return GLR_OK;
}

// The power-iteration part of a truncated refresh (Eq. SVD-P1 read as the top-k subspace of
// Mbar): q block power iterations from the previous basis (a seeded Gaussian block at the first
// refresh), each half re-orthonormalised by CholeskyQR, CholeskyQR2 at the end, then the
// Rayleigh-Ritz matrix H = Z^T Z = Q^T Mbar Mbar^T Q in Hk.
int refresh_power(glr_handle* h, cudaStream_t st) {
    const int mp = h->mp, np = h->np, k = h->k;
    if (h->refreshes == 0 && !h->basis_from_user)
        GLR_LAUNCH(h, 1, random_block(h->Q, mp, k, h->s.seed, static_cast<uint32_t>(h->t), st));
    int rc;
    // Mbar(a, b) at a * sa + b * sb: row-major, or column-major on the tcgen05 path
    const int64_t sa = h->tcl ? 1 : np, sb = h->tcl ? mp : 1;
    for (int it = 0; it < h->s.power_iters; ++it) {
        // Z = Mbar^T Q (n' x k) and Q = Mbar Z (m' x k), each re-orthonormalised by CholeskyQR
        // (one pass keeps the block well conditioned; the span is what the iteration needs)
        GLR_GEMM(h, gd(np, k, mp, h->Mbar, sb, sa, h->Q, k, 1, h->Z, k, 1), st);
        if ((rc = cholqr(h, h->Z, h->Zn, np, st)) != GLR_OK) return rc;
        GLR_GEMM(h, gd(mp, k, np, h->Mbar, sa, sb, h->Z, k, 1, h->Q, k, 1), st);
        if ((rc = cholqr(h, h->Q, h->Qn, mp, st)) != GLR_OK) return rc;
    }
    if ((rc = cholqr(h, h->Q, h->Qn, mp, st)) != GLR_OK) return rc;   // CholeskyQR2: orthonormal to rounding
    // Rayleigh-Ritz: Z = Mbar^T Q, H = Z^T Z = Q^T Mbar Mbar^T Q
    GLR_GEMM(h, gd(np, k, mp, h->Mbar, sb, sa, h->Q, k, 1, h->Z, k, 1), st);
    GLR_GEMM(h, gd(k, k, np, h->Z, 1, k, h->Z, k, 1, h->Hk, k, 1), st);
    return GLR_OK;
}

// Truncated refreshes of several matrices with large k: each handle's power iteration on its
// own side stream, then the k x k Rayleigh-Ritz eigen-decompositions of all of them in one
// cooperative Jacobi launch (k_jacobi.cu: every CTA of the grid works on every matrix, where the
// one-CTA Jacobi of refresh_tail would take k x k rotations in a single SM), then each handle's
// finish on its own stream.  Without cooperative launches, refresh_tail per handle.
int refresh_trunc_grouped(std::vector<glr_handle*>& hs) {
    for (glr_handle* h : hs) {
        PhaseScope ps(h, GLR_PH_REFRESH, h->rstream);
        g_ws = h->gemm_ws;
        const int rc = refresh_power(h, h->rstream);
        g_ws = nullptr;
        if (rc != GLR_OK) return rc;
    }
    // k <= 256: every matrix's eigenproblem in one launch, one CTA each (k_eig.cu)
    bool small = true;
    for (glr_handle* h : hs) small = small && h->k <= 256;
    if (small) {
        for (size_t c0 = 0; c0 < hs.size(); c0 += kEigGroupMax) {
            const size_t c1 = std::min(hs.size(), c0 + (size_t)kEigGroupMax);
            glr_handle* h0 = hs[c0];
            cudaStream_t s0 = h0->rstream;
            EigGroup g{};
            g.max_sweeps = 40;
            for (size_t i = c0; i < c1; ++i) {
                glr_handle* h = hs[i];
                if (h != h0) {
                    GLR_CK(h, cudaEventRecord(h->rpow, h->rstream));
                    GLR_CK(h0, cudaStreamWaitEvent(s0, h->rpow, 0));
                }
                EigMat& M = g.mat[g.nmat++];
                const int n = h->k;
                M.n = n; M.tol = 4.f * 5.96e-8f * sqrtf(static_cast<float>(n)) + 1e-7f;
                M.H = h->Hk; M.nparts = 1; M.ld = n; M.V = h->Vk; M.evals = h->evals; M.sweeps = h->dflags + 1;
            }
            {
                PhaseScope ps(h0, GLR_PH_REFRESH, s0);
                GLR_LAUNCH(h0, 1, eig_tmem_group(g, s0));
            }
            GLR_CK(h0, cudaEventRecord(h0->rpow, s0));
            for (size_t i = c0; i < c1; ++i) {
                glr_handle* h = hs[i];
                if (h != h0) GLR_CK(h, cudaStreamWaitEvent(h->rstream, h0->rpow, 0));
                PhaseScope ps(h, GLR_PH_REFRESH, h->rstream);
                g_ws = h->gemm_ws;
                const int rc = refresh_finish(h, h->rstream);
                g_ws = nullptr;
                if (rc != GLR_OK) return rc;
            }
        }
        return GLR_OK;
    }
    const int grid = jacobi_group_grid();
    if (!grid) {
        for (glr_handle* h : hs) {
            PhaseScope ps(h, GLR_PH_REFRESH, h->rstream);
            g_ws = h->gemm_ws;
            const int rc = refresh_tail(h, h->rstream);
            g_ws = nullptr;
            if (rc != GLR_OK) return rc;
        }
        return GLR_OK;
    }
    for (size_t c0 = 0, c1 = 0; c0 < hs.size(); c0 = c1) {
        size_t rot = 0;
        for (c1 = c0; c1 < hs.size() && c1 - c0 < (size_t)kGroupMax; ++c1) {
            const size_t add = jacobi_rot_floats(hs[c1]->k) * sizeof(float);
            if (c1 > c0 && rot + add > kJacobiMaxSmem) break;
            rot += add;
        }
        glr_handle* h0 = hs[c0];
        cudaStream_t s0 = h0->rstream;
        JacobiGroup g{};
        size_t soff = 0;
        g.max_sweeps = 40;
        g.bar = h0->dflags + 4; g.err = h0->dflags + 2; g.part = h0->jpart;
        for (size_t i = c0; i < c1; ++i) {
            glr_handle* h = hs[i];
            if (h != h0) {
                GLR_CK(h, cudaEventRecord(h->rpow, h->rstream));
                GLR_CK(h0, cudaStreamWaitEvent(s0, h->rpow, 0));
            }
            JacobiMat& M = g.mat[g.nmat++];
            const int n = h->k;
            M.n = n; M.tol = 4.f * 5.96e-8f * sqrtf(static_cast<float>(n)) + 1e-7f;
            M.H = h->Hk; M.H2 = h->scratch; M.V = h->Vk; M.evals = h->evals;
            M.sweeps = h->dflags + 1;
            M.soff = (int)soff;
            soff += jacobi_rot_floats(n);
        }
        {
            PhaseScope ps(h0, GLR_PH_REFRESH, s0);
            GLR_LAUNCH(h0, 1, jacobi_group(g, grid, s0));
        }
        GLR_CK(h0, cudaEventRecord(h0->rpow, s0));
        for (size_t i = c0; i < c1; ++i) {
            glr_handle* h = hs[i];
            if (h != h0) GLR_CK(h, cudaStreamWaitEvent(h->rstream, h0->rpow, 0));
            PhaseScope ps(h, GLR_PH_REFRESH, h->rstream);
            g_ws = h->gemm_ws;
            const int rc = refresh_finish(h, h->rstream);
            g_ws = nullptr;
            if (rc != GLR_OK) return rc;
        }
    }
    return GLR_OK;
}


// ---- the tcgen05 path's refresh: every stage one grouped launch for all refreshing matrices ----
namespace {

tc::TcMat refresh_mat(const glr_handle* h) {
    tc::TcMat M{};
    M.mp = h->mp; M.np = h->np; M.N = h->N; M.r = h->r; M.rpad = h->rpad; M.k = h->k; M.kpad = h->kpad;
    M.transposed = h->transposed; M.gdtype = h->s.grad_dtype;
    return M;
}

// One op over the handles for which fill(h, M) returns true, kTcGroupMax matrices per launch, on st.
template <class Fill>
int refresh_op(std::vector<glr_handle*>& hs, cudaError_t (*launch)(tc::TcGroup&, cudaStream_t), cudaStream_t st,
               Fill fill) {
    static thread_local tc::TcGroup g;
    size_t i = 0;
    while (i < hs.size()) {
        g.nmat = 0; g.total_tiles = 0; g.err = nullptr;
        glr_handle* h0 = nullptr;
        for (; i < hs.size() && g.nmat < tc::kTcGroupMax; ++i) {
            glr_handle* h = hs[i];
            tc::TcMat M = refresh_mat(h);
            if (!fill(h, M)) continue;
            if (!h0) { h0 = h; g.err = h->dflags + 2; }
            M.tile0 = g.total_tiles;
            g.total_tiles += M.ntiles;
            g.mat[g.nmat++] = M;
        }
        if (h0 && g.total_tiles > 0) {
            PhaseScope ps(h0, GLR_PH_REFRESH, st);
            GLR_LAUNCH(h0, 1, launch(g, st));
        }
    }
    return GLR_OK;
}

int cdiv(int a, int b) { return (a + b - 1) / b; }

// One grouped fp32 product per handle (fill describes it), 64 per launch.
template <class Fill>
int fp32_products(std::vector<glr_handle*>& hs, cudaStream_t st, Fill fill) {
    for (size_t c0 = 0; c0 < hs.size(); c0 += 64) {
        GemmGroup gg{};
        for (size_t i = c0; i < hs.size() && i < c0 + 64; ++i) fill(hs[i], gg.mat[gg.nmat++]);
        PhaseScope ps(hs[c0], GLR_PH_REFRESH, st);
        GLR_LAUNCH(hs[c0], 1, gemm_group_f32(gg, st));
    }
    return GLR_OK;
}

// X^T X (Gram partials over row chunks), its factor L^{-1}, then X <- X L^{-T} (and X^T): the
// CholeskyQR of X = Z (n' rows) or Q (m' rows) in TF32 products.
int cholqr_tc(std::vector<glr_handle*>& hs, bool zside, cudaStream_t st, const std::vector<int>& active) {
    std::vector<glr_handle*> act;
    for (size_t i = 0; i < hs.size(); ++i) if (active[i]) act.push_back(hs[i]);
    int rc = refresh_op(act, tc::launch_gram, st, [zside](glr_handle* h, tc::TcMat& M) {
        M.rows = zside ? h->np : h->mp;
        M.mA = tcl_map(h, zside ? kMapZTtA : kMapQTtA); M.mB = tcl_map(h, zside ? kMapZTtB : kMapQTtB);
        M.out = h->gpart; M.ntiles = cdiv(M.rows, tc::kGramChunk);
        return true;
    });
    if (rc != GLR_OK) return rc;
    for (size_t c0 = 0; c0 < act.size(); c0 += 64) {
        CholGroup cg{};
        for (size_t i = c0; i < act.size() && i < c0 + 64; ++i) {
            glr_handle* h = act[i];
            CholMat& C = cg.mat[cg.nmat++];
            C.part = h->gpart; C.nparts = cdiv(zside ? h->np : h->mp, tc::kGramChunk); C.ld = h->kpad; C.n = h->k;
            C.out = h->Linv; C.flag = h->dflags + 0;
        }
        PhaseScope ps(act[c0], GLR_PH_REFRESH, st);
        GLR_LAUNCH(act[c0], 1, chol_group(cg, st));
    }
    return refresh_op(act, tc::launch_apply, st, [zside](glr_handle* h, tc::TcMat& M) {
        M.rows = zside ? h->np : h->mp;
        M.mA = tcl_map(h, zside ? kMapZA : (h->Q == h->Qbuf0 ? kMapQA : kMapQA1)); M.mB = tcl_map(h, kMapLinv);
        M.out = zside ? h->Z : h->Q; M.outT = zside ? h->ZTt : h->QTt; M.ld_out = h->k;
        M.ntiles = cdiv(M.rows, 128);
        return true;
    });
}

}  // namespace

// Truncated refreshes on the tcgen05 path (k <= 256; Mbar column-major, plus the row-major copy
// the compose pass wrote on this step).  q block power iterations from the previous basis (a
// seeded Gaussian block at the first refresh): Z = Mbar^T Q and Q = Mbar Z as TF32 tcgen05
// products, each re-orthonormalised by a TF32 CholeskyQR (the span is what the iteration needs);
// the last Q = Mbar Z multiplies Mbar's TF32 low parts too, so the subspace it spans is exact to
// fp32 level for the iterate it is applied to.  Then CholeskyQR2 in fp32 (orthonormal to
// rounding), the Rayleigh-Ritz matrix H = (Mbar^T Q)^T (Mbar^T Q), the k x k eigenproblems
// (k_eig.cu) and each handle's finish (sort, signs, Householder WY form).
int refresh_tcl_grouped(std::vector<glr_handle*>& hs) {
    glr_handle* h0 = hs[0];
    cudaStream_t s0 = h0->rstream;
    int rc;
    for (glr_handle* h : hs) GLR_CK(h0, cudaStreamWaitEvent(s0, h->rfork, 0));
    int q = 0;
    for (glr_handle* h : hs) {
        PhaseScope ps(h, GLR_PH_REFRESH, s0);
        if (h->refreshes == 0 && !h->basis_from_user)
            GLR_LAUNCH(h, 1, random_block(h->Q, h->mp, h->k, h->s.seed, static_cast<uint32_t>(h->t), s0));
        GLR_LAUNCH(h, 1, tc::transpose_round(h->QTt, h->mp, h->Q, h->mp, h->k, h->k, s0));
        q = std::max(q, h->s.power_iters);
    }
    std::vector<int> active(hs.size(), 1);
    for (int it = 0; it < q; ++it) {
        for (size_t i = 0; i < hs.size(); ++i) active[i] = it < hs[i]->s.power_iters ? 1 : 0;
        auto is_active = [&](glr_handle* h) {
            for (size_t i = 0; i < hs.size(); ++i) if (hs[i] == h) return active[i] != 0;
            return false;
        };
        // Z = Mbar^T Q
        rc = refresh_op(hs, tc::launch_powt, s0, [&](glr_handle* h, tc::TcMat& M) {
            if (!is_active(h)) return false;
            M.rows = h->np; M.mA = tcl_map(h, kMapMbarT); M.mB = tcl_map(h, kMapQTtB);
            M.out = h->Z; M.outT = h->ZTt; M.ld_out = h->k; M.ntiles = cdiv(h->np, 256);
            return true;
        });
        if (rc != GLR_OK) return rc;
        if ((rc = cholqr_tc(hs, true, s0, active)) != GLR_OK) return rc;
        // Q = Mbar Z; a handle's last iteration with Mbar's low parts
        for (size_t i = 0; i < hs.size(); ++i) {
            glr_handle* h = hs[i];
            if (!active[i] || it != h->s.power_iters - 1) continue;
            PhaseScope ps(h, GLR_PH_REFRESH, s0);
            GLR_LAUNCH(h, 1, tc::split_lo(h->Mrow, h->Mlo, (int64_t)h->mp * h->np, s0));
        }
        rc = refresh_op(hs, tc::launch_pown, s0, [&](glr_handle* h, tc::TcMat& M) {
            if (!is_active(h)) return false;
            M.rows = h->mp; M.mA = tcl_map(h, kMapMrow); M.mA2 = tcl_map(h, kMapMlo); M.mB = tcl_map(h, kMapZTtB);
            M.split = it == h->s.power_iters - 1 ? 1 : 0;
            M.out = h->Q; M.outT = h->QTt; M.ld_out = h->k; M.ntiles = cdiv(h->mp, 256);
            return true;
        });
        if (rc != GLR_OK) return rc;
        std::vector<int> mid(hs.size(), 0);
        for (size_t i = 0; i < hs.size(); ++i) mid[i] = active[i] && it < hs[i]->s.power_iters - 1 ? 1 : 0;
        if ((rc = cholqr_tc(hs, false, s0, mid)) != GLR_OK) return rc;
    }
    // CholeskyQR2 in fp32 (grouped FFMA products and factors), then Q^T for the Rayleigh-Ritz
    // product
    for (int pass = 0; pass < 2; ++pass) {
        if ((rc = fp32_products(hs, s0, [](glr_handle* h, GemmMat& G) {      // Gram Q^T Q
                 G.M = h->k; G.N = h->k; G.K = h->mp;
                 G.A = h->Q; G.sAi = 1; G.sAp = h->k; G.B = h->Q; G.sBp = h->k; G.sBj = 1;
                 G.C = h->gram; G.sCi = h->k; G.sCj = 1;
             })) != GLR_OK)
            return rc;
        for (size_t c0 = 0; c0 < hs.size(); c0 += 64) {
            CholGroup cg{};
            for (size_t i = c0; i < hs.size() && i < c0 + 64; ++i) {
                glr_handle* h = hs[i];
                CholMat& C = cg.mat[cg.nmat++];
                C.part = h->gram; C.nparts = 1; C.ld = h->k; C.n = h->k; C.out = h->Linv; C.flag = h->dflags + 0;
            }
            PhaseScope ps(hs[c0], GLR_PH_REFRESH, s0);
            GLR_LAUNCH(hs[c0], 1, chol_group(cg, s0));
        }
        if ((rc = fp32_products(hs, s0, [](glr_handle* h, GemmMat& G) {      // Qn = Q L^{-T}
                 G.M = h->mp; G.N = h->k; G.K = h->k;
                 G.A = h->Q; G.sAi = h->k; G.sAp = 1; G.B = h->Linv; G.sBp = 1; G.sBj = h->k;
                 G.C = h->Qn; G.sCi = h->k; G.sCj = 1;
             })) != GLR_OK)
            return rc;
        for (glr_handle* h : hs) std::swap(h->Q, h->Qn);
    }
    for (glr_handle* h : hs) {
        PhaseScope ps(h, GLR_PH_REFRESH, s0);
        GLR_LAUNCH(h, 1, tc::transpose_round(h->QTt, h->mp, h->Q, h->mp, h->k, h->k, s0));
    }
    // Rayleigh-Ritz: Z = Mbar^T Q, H = Z^T Z (Gram partials), the eigenproblems
    rc = refresh_op(hs, tc::launch_powt, s0, [&](glr_handle* h, tc::TcMat& M) {
        M.rows = h->np; M.mA = tcl_map(h, kMapMbarT); M.mB = tcl_map(h, kMapQTtB);
        M.out = h->Z; M.outT = h->ZTt; M.ld_out = h->k; M.ntiles = cdiv(h->np, 256);
        return true;
    });
    if (rc != GLR_OK) return rc;
    rc = refresh_op(hs, tc::launch_gram, s0, [](glr_handle* h, tc::TcMat& M) {
        M.rows = h->np; M.mA = tcl_map(h, kMapZTtA); M.mB = tcl_map(h, kMapZTtB);
        M.out = h->gpart; M.ntiles = cdiv(h->np, tc::kGramChunk);
        return true;
    });
    if (rc != GLR_OK) return rc;
    // the k x k problems: the blocked Jacobi for k a multiple of 128 from 256, else one CTA each
    std::vector<glr_handle*> small;
    std::vector<BjItem> big;
    for (glr_handle* h : hs) {
        if (tcl_rr_blocked(h)) big.push_back(BjItem{h, h->k, 0, 0, false});
        else small.push_back(h);
        h->bj_V = nullptr;
    }
    for (size_t c0 = 0; c0 < small.size(); c0 += kEigGroupMax) {
        EigGroup g{};
        g.max_sweeps = 40;
        for (size_t i = c0; i < small.size() && i < c0 + (size_t)kEigGroupMax; ++i) {
            glr_handle* h = small[i];
            EigMat& M = g.mat[g.nmat++];
            const int n = h->k;
            M.n = n; M.tol = 4.f * 5.96e-8f * sqrtf(static_cast<float>(n)) + 1e-7f;
            M.H = h->gpart; M.nparts = cdiv(h->np, tc::kGramChunk); M.ld = h->kpad;
            M.V = h->Vk; M.evals = h->evals; M.sweeps = h->dflags + 1;
        }
        PhaseScope ps(small[c0], GLR_PH_REFRESH, s0);
        GLR_LAUNCH(small[c0], 1, eig_tmem_group(g, s0));
    }
    if (!big.empty()) {
        glr_handle* b0 = big[0].h;
        PhaseScope ps(b0, GLR_PH_REFRESH, s0);
        rc = bjac_prepare(big, b0, s0, [](glr_handle* h, BjacPrep& P) {
            P.part = h->gpart; P.nparts = cdiv(h->np, tc::kGramChunk); P.ld = h->kpad;
        });
        if (rc == GLR_OK) rc = bjac_run(big, b0, s0);
        if (rc != GLR_OK) return rc;
        for (const BjItem& S : big) {
            GLR_LAUNCH(S.h, 1, bjac_diag(S.h->Hbuf, S.n, S.h->evals, s0));
            S.h->bj_V = S.V();
        }
    }
    // the finish, grouped: sorted Ritz pairs, Q <- Q W, column signs, the Householder WY form,
    // Yt = Y T^T, then Y^T for the W = Y^T Mbar products
    for (size_t c0 = 0; c0 < hs.size(); c0 += 64) {
        FinishGroup fg{};
        for (size_t i = c0; i < hs.size() && i < c0 + 64; ++i) {
            glr_handle* h = hs[i];
            FinishMat& F = fg.mat[fg.nmat++];
            F.mp = h->mp; F.k = h->k; F.evals = h->evals; F.V = h->bj_V ? h->bj_V : h->Vk; F.W = h->gram;
            F.evals_sorted = h->evals_sorted;
            F.Wtop = h->scratch; F.Y = h->Y; F.T = h->T; F.s = h->dsign;
        }
        PhaseScope ps(hs[c0], GLR_PH_REFRESH, s0);
        GLR_LAUNCH(hs[c0], 1, finish_group(fg, 0, s0));
    }
    if ((rc = fp32_products(hs, s0, [](glr_handle* h, GemmMat& G) {          // Qn = Q W
             G.M = h->mp; G.N = h->k; G.K = h->k;
             G.A = h->Q; G.sAi = h->k; G.sAp = 1; G.B = h->gram; G.sBp = h->k; G.sBj = 1;
             G.C = h->Qn; G.sCi = h->k; G.sCj = 1;
         })) != GLR_OK)
        return rc;
    for (glr_handle* h : hs) std::swap(h->Q, h->Qn);
    for (int stage = 1; stage <= 2; ++stage) {
        for (size_t c0 = 0; c0 < hs.size(); c0 += 64) {
            FinishGroup fg{};
            for (size_t i = c0; i < hs.size() && i < c0 + 64; ++i) {
                glr_handle* h = hs[i];
                FinishMat& F = fg.mat[fg.nmat++];
                F.mp = h->mp; F.k = h->k; F.Q = h->Q; F.Wtop = h->scratch; F.Y = h->Y; F.T = h->T; F.s = h->dsign;
            }
            PhaseScope ps(hs[c0], GLR_PH_REFRESH, s0);
            GLR_LAUNCH(hs[c0], 1, finish_group(fg, stage, s0));
        }
    }
    // rows a >= k of Y: Y[a, :] Utilde = -Q[a, :] with Utilde the upper triangle the top-block
    // LU left in scratch: Utilde^{-1} (as the inverse of its transpose), then one product
    for (size_t c0 = 0; c0 < hs.size(); c0 += 64) {
        CholGroup cg{};
        for (size_t i = c0; i < hs.size() && i < c0 + 64; ++i) {
            glr_handle* h = hs[i];
            CholMat& C = cg.mat[cg.nmat++];
            C.part = h->scratch; C.nparts = 1; C.ld = h->k; C.n = h->k; C.out = h->Linv; C.tri_only = 1;
        }
        PhaseScope ps(hs[c0], GLR_PH_REFRESH, s0);
        GLR_LAUNCH(hs[c0], 1, chol_group(cg, s0));
    }
    if ((rc = fp32_products(hs, s0, [](glr_handle* h, GemmMat& G) {          // Y[k:] = -Q[k:] Utilde^{-1}
             G.M = h->mp - h->k; G.N = h->k; G.K = h->k; G.alpha = -1.f;
             G.A = h->Q + (size_t)h->k * h->k; G.sAi = h->k; G.sAp = 1;
             G.B = h->Linv; G.sBp = 1; G.sBj = h->k;
             G.C = h->Y + (size_t)h->k * h->k; G.sCi = h->k; G.sCj = 1;
         })) != GLR_OK)
        return rc;
    if ((rc = fp32_products(hs, s0, [](glr_handle* h, GemmMat& G) {          // Yt = Y T^T
             G.M = h->mp; G.N = h->k; G.K = h->k;
             G.A = h->Y; G.sAi = h->k; G.sAp = 1; G.B = h->T; G.sBp = 1; G.sBj = h->k;
             G.C = h->Yt; G.sCi = h->k; G.sCj = 1;
         })) != GLR_OK)
        return rc;
    for (glr_handle* h : hs) {
        PhaseScope ps(h, GLR_PH_REFRESH, s0);
        GLR_LAUNCH(h, 1, tc::transpose_round(h->YTk, h->mp, h->Y, h->mp, h->k, h->k, s0));
    }
    // every handle's side stream continues after the group's work
    GLR_CK(h0, cudaEventRecord(h0->rpow, s0));
    for (glr_handle* h : hs)
        if (h != h0) GLR_CK(h, cudaStreamWaitEvent(h->rstream, h0->rpow, 0));
    return GLR_OK;
}

}  // namespace host
}  // namespace glr
