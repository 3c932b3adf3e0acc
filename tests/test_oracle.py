"""Pins for the CPU oracle: each check ties the oracle to something other than itself
(published known-answer vectors, worked examples printed in the paper, closed forms,
invariants, brute force on tiny inputs, Monte-Carlo statements of the paper's
propositions)."""
import itertools
import json
import math
import os

import numpy as np
import pytest

from oracle import greedylore as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def _rand_orth(rng, m):
    q, r = np.linalg.qr(rng.standard_normal((m, m)))
    return q * np.sign(np.diag(r))


# ---------------------------------------------------------------------------------------------
# Philox4x32-10 and the Gaussian vectors of Eq. random-v
# ---------------------------------------------------------------------------------------------
def test_philox_known_answers():
    for case in _golden("philox4x32_10_kat.json")["cases"]:
        c = [int(x, 16) for x in case["ctr"]]
        k = [int(x, 16) for x in case["key"]]
        out = O.philox4x32_10(*c, *k)
        assert [int(x) for x in out] == [int(x, 16) for x in case["out"]]


def test_unit_open_is_exact_in_fp32_and_open():
    """The word-to-uniform map stays inside (0, 1) and every value it takes is an fp32 number,
    so an fp32 implementation draws the same uniforms (the extremes and a spread of words)."""
    words = np.array([0, 1, 511, 512, 2 ** 31 - 1, 2 ** 31, 0xFFFFFE00, 0xFFFFFFFE, 0xFFFFFFFF] +
                     list(np.random.default_rng(3).integers(0, 2 ** 32, 10000, dtype=np.uint64)), dtype=np.uint64)
    u = O._unit_open(words)
    assert u.min() == 2.0 ** -24 and u.max() == 1.0 - 2.0 ** -24
    assert np.all(u.astype(np.float32).astype(np.float64) == u)
    assert np.all(np.isfinite(np.sqrt(-2.0 * np.log(u)))) and np.all(-2.0 * np.log(u) > 0)


def test_gaussian_v_moments_and_freshness():
    V = O.gaussian_v(seed=12345, t=7, rows=400, cols=1001)
    n = V.size
    assert V.shape == (400, 1001)
    assert abs(V.mean()) < 5 / math.sqrt(n)
    assert abs(V.var() - 1.0) < 5 * math.sqrt(2.0 / n)
    kurt = np.mean(V ** 4) / np.mean(V ** 2) ** 2
    assert abs(kurt - 3.0) < 0.05
    # rows are independent draws: sample correlation between rows ~ N(0, 1/cols)
    C = np.corrcoef(V[:50])
    off = C[~np.eye(50, dtype=bool)]
    assert np.max(np.abs(off)) < 6 / math.sqrt(1001)
    # reproducible, fresh per step, distinct per seed
    assert np.array_equal(V, O.gaussian_v(12345, 7, 400, 1001))
    assert not np.allclose(V, O.gaussian_v(12345, 8, 400, 1001))
    assert not np.allclose(V, O.gaussian_v(12346, 7, 400, 1001))
    # a narrower draw is a prefix of the wider one (element (j, b) depends only on (j, b))
    assert np.array_equal(V[:10, :37], O.gaussian_v(12345, 7, 10, 37))


# ---------------------------------------------------------------------------------------------
# SVD basis, Eckart-Young, Householder completion
# ---------------------------------------------------------------------------------------------
def _jacobi_eig_bruteforce(H, sweeps=60):
    """Cyclic two-sided Jacobi in plain Python loops (tiny matrices only)."""
    H = [list(map(float, row)) for row in H]
    n = len(H)
    V = [[1.0 if i == j else 0.0 for j in range(n)] for i in range(n)]
    for _ in range(sweeps):
        off = sum(H[i][j] ** 2 for i in range(n) for j in range(n) if i != j)
        if off < 1e-30:
            break
        for p in range(n - 1):
            for q in range(p + 1, n):
                if abs(H[p][q]) < 1e-300:
                    continue
                theta = (H[q][q] - H[p][p]) / (2 * H[p][q])
                t = (1.0 if theta >= 0 else -1.0) / (abs(theta) + math.sqrt(theta * theta + 1))
                c = 1 / math.sqrt(t * t + 1)
                s = t * c
                for k in range(n):
                    hkp, hkq = H[k][p], H[k][q]
                    H[k][p], H[k][q] = c * hkp - s * hkq, s * hkp + c * hkq
                for k in range(n):
                    hpk, hqk = H[p][k], H[q][k]
                    H[p][k], H[q][k] = c * hpk - s * hqk, s * hpk + c * hqk
                for k in range(n):
                    vkp, vkq = V[k][p], V[k][q]
                    V[k][p], V[k][q] = c * vkp - s * vkq, s * vkp + c * vkq
    return np.array([H[i][i] for i in range(n)]), np.array(V)


@pytest.mark.parametrize("shape", [(3, 5), (5, 9), (6, 6), (8, 13)])
def test_left_singular_basis_against_bruteforce_jacobi(shape):
    rng = np.random.default_rng(shape[0] * 31 + shape[1])
    A = rng.standard_normal(shape)
    U, s = O.left_singular_basis(A)
    m = shape[0]
    assert np.allclose(U.T @ U, np.eye(m), atol=1e-12)
    assert np.all(np.diff(s) <= 0)
    ev, W = _jacobi_eig_bruteforce(A @ A.T)
    order = np.argsort(-ev)
    ev, W = ev[order], W[:, order]
    assert np.allclose(np.sqrt(np.maximum(ev, 0)), s[:m], rtol=1e-10, atol=1e-12)
    W = O.fix_signs(W)
    assert np.allclose(W, U, atol=1e-8)
    # sign convention: the largest-magnitude entry of every column is positive
    idx = np.argmax(np.abs(U), axis=0)
    assert np.all(U[idx, np.arange(m)] > 0)


def test_eckart_young_and_subset_optimality():
    rng = np.random.default_rng(5)
    A = rng.standard_normal((6, 10))
    U, s = O.left_singular_basis(A)
    for r in range(1, 6):
        P = U[:, :r]
        err = np.linalg.norm(A - P @ P.T @ A) ** 2
        assert err == pytest.approx(np.sum(s[r:] ** 2), rel=1e-10)
        # no other r-subset of U's columns does better
        for J in itertools.combinations(range(6), r):
            PJ = U[:, list(J)]
            assert np.linalg.norm(A - PJ @ PJ.T @ A) ** 2 >= err - 1e-10


@pytest.mark.parametrize("m,k", [(5, 1), (7, 3), (16, 8), (40, 5)])
def test_householder_complement(m, k):
    rng = np.random.default_rng(m * 100 + k)
    Q = np.linalg.qr(rng.standard_normal((m, k)))[0]
    U = O.householder_complement(Q)
    assert np.allclose(U.T @ U, np.eye(m), atol=1e-12)
    assert np.allclose(U[:, :k], Q, atol=1e-12)
    assert np.allclose(Q.T @ U[:, k:], 0, atol=1e-12)


def test_argtop_r_ties_and_order():
    s = np.array([1.0, 3.0, 3.0, 0.5, 3.0, 2.0])
    assert list(O.argtop_r(s, 2)) == [1, 2]
    assert list(O.argtop_r(s, 4)) == [1, 2, 4, 5]
    assert list(O.argtop_r(np.zeros(5), 3)) == [0, 1, 2]


# ---------------------------------------------------------------------------------------------
# Worked examples printed in the paper
# ---------------------------------------------------------------------------------------------
def test_prop2_counterexample():
    g = _golden("prop2_counterexample.json")
    G0, Gt = np.array(g["G0"]), np.array(g["Gt"])
    U, _ = O.left_singular_basis(G0)
    P = U[:, : g["r"]]
    assert np.allclose(P, g["P"])
    C = P @ P.T @ Gt
    assert np.allclose(C, g["C_Gt"])
    assert np.linalg.norm(C - Gt) ** 2 == pytest.approx(g["err_sq"])
    assert np.linalg.norm(Gt) ** 2 == pytest.approx(g["norm_sq"])


def test_appendix_c_quadratic():
    g = _golden("appC_quadratic.json")
    L = g["L"]
    for tau in g["taus"]:
        orc = O.GreedyLoreOracle(2, 2, 1, 1, tau=10 ** 9, refresh_mode="alg4", optimizer="msgd",
                                 lr=1.0 / (2 * L), beta1=0.0)
        X = np.diag(g["x0"])
        for _ in range(tau):
            grad = np.diag([L * X[0, 0], L * X[1, 1] / 2])
            X, info = orc.step(grad[None], X, force_J=[0])
            assert np.allclose(info.P, [[1.0], [0.0]])
        assert X[0, 0] == 2.0 ** -tau
        assert X[1, 1] == g["y_tau"]
        grad = np.diag([L * X[0, 0], L * X[1, 1] / 2])
        P = np.array([[1.0], [0.0]])
        alpha = np.linalg.norm(P @ P.T @ grad) ** 2 / np.linalg.norm(grad) ** 2
        assert alpha == pytest.approx(2.0 ** (-2 * tau) / (2.0 ** (-2 * tau) + 0.25), rel=1e-12)
        if tau > g["fp32_alpha_zero_for_tau_above"]:
            assert np.float32(2.0 ** (-2 * tau)) == 0.0


# ---------------------------------------------------------------------------------------------
# Propositions 1, 3, 4 and Lemma 2
# ---------------------------------------------------------------------------------------------
def test_prop1_fixed_projection_nullifies_error_feedback():
    rng = np.random.default_rng(11)
    m, n, r, N = 6, 9, 2, 3
    orc = O.GreedyLoreOracle(m, n, r, N, tau=100, refresh_mode="alg4", lr=0.0, beta1=0.0)
    X = np.zeros((m, n))
    J = [1, 4]
    for t in range(6):
        G = rng.standard_normal((N, m, n))
        X, info = orc.step(G, X, force_J=J if t else None)
        if t == 0:
            J = list(info.J)
            continue
        P = info.P
        for i in range(N):
            assert np.allclose(info.sent[i], P @ P.T @ G[i], atol=1e-12)


def test_prop3_contraction_and_pythagoras():
    rng = np.random.default_rng(3)
    for trial in range(20):
        m, n = rng.integers(3, 12), rng.integers(3, 15)
        r = int(rng.integers(1, m + 1))
        U = _rand_orth(rng, m)
        G = rng.standard_normal((m, n)) * rng.exponential(size=(m, 1))
        e = O.exact_energies(G, U)
        J = O.argtop_r(e, r)
        P = U[:, J]
        err = np.linalg.norm(G - P @ P.T @ G) ** 2
        nrm = np.linalg.norm(G) ** 2
        assert err == pytest.approx(nrm - np.sum(e[J]), rel=1e-10, abs=1e-12)   # Eq. sub_problem_derivation
        assert err <= (1 - r / m) * nrm + 1e-12                                  # Eq. contractive


def test_exact_rule_equals_bruteforce_subset_search():
    rng = np.random.default_rng(8)
    for trial in range(10):
        m, n, r = 7, 5, int(rng.integers(1, 7))
        U = _rand_orth(rng, m)
        G = rng.standard_normal((m, n))
        best, bestJ = None, None
        for J in itertools.combinations(range(m), r):
            P = U[:, list(J)]
            err = np.linalg.norm(G - P @ P.T @ G) ** 2
            if best is None or err < best - 1e-12:
                best, bestJ = err, J
        assert list(O.argtop_r(O.exact_energies(G, U), r)) == list(bestJ)


def test_lambda_linearity_over_nodes():
    rng = np.random.default_rng(4)
    m, n, N = 5, 8, 4
    U = _rand_orth(rng, m)
    Ms = rng.standard_normal((N, m, n))
    V = O.gaussian_v(99, 3, m, n)
    lam = O.approx_top_r_lambda(list(Ms), U, V)
    direct = np.array([U[:, j] @ Ms.mean(0) @ V[j] for j in range(m)])
    assert np.allclose(lam, direct, atol=1e-12)
    # a hand-written double loop for one node and one j
    j = 2
    acc = sum(U[a, j] * Ms[0, a, b] * V[j, b] for a in range(m) for b in range(n))
    assert O.approx_top_r_lambda([Ms[0]], U, V)[j] == pytest.approx(acc, rel=1e-12)


def test_prop4_unbiased_estimator_monte_carlo():
    rng = np.random.default_rng(21)
    m, n, N = 4, 6, 3
    U = _rand_orth(rng, m)
    Ms = rng.standard_normal((N, m, n)) + np.arange(N)[:, None, None]   # heterogeneous nodes
    target = O.exact_energies(Ms.mean(0), U)                           # ||u_j^T Gbar||^2
    T = 20000
    samples = np.empty((T, m))
    for t in range(T):
        V = O.gaussian_v(777, t, m, n)
        samples[t] = O.approx_top_r_lambda(list(Ms), U, V) ** 2
    mean, se = samples.mean(0), samples.std(0) / math.sqrt(T)
    assert np.all(np.abs(mean - target) < 5 * se)
    # averaging squares instead of squaring the average would be biased here
    per_node = np.mean([O.exact_energies(Mi, U) for Mi in Ms], axis=0)
    assert np.any(np.abs(per_node - target) > 10 * se)


def test_lemma2_contraction_in_expectation_monte_carlo():
    rng = np.random.default_rng(22)
    m, n, N, r = 8, 10, 2, 2
    U = _rand_orth(rng, m)
    Ms = rng.standard_normal((N, m, n)) * np.linspace(3, 0.2, m)[None, :, None]
    Gbar = Ms.mean(0)
    T = 4000
    errs = np.empty(T)
    for t in range(T):
        V = O.gaussian_v(4242, t, m, n)
        J = O.argtop_r(O.approx_top_r_lambda(list(Ms), U, V) ** 2, r)
        P = U[:, J]
        errs[t] = np.linalg.norm(Gbar - P @ P.T @ Gbar) ** 2
    bound = (1 - r / m) * np.linalg.norm(Gbar) ** 2
    assert errs.mean() <= bound + 5 * errs.std() / math.sqrt(T)


# ---------------------------------------------------------------------------------------------
# Error-feedback telescoping, reconstruction, refresh, orientation
# ---------------------------------------------------------------------------------------------
@pytest.mark.parametrize("mode", ["alg3", "alg4"])
@pytest.mark.parametrize("k", [0, 3])
def test_error_feedback_telescoping(mode, k):
    rng = np.random.default_rng(31)
    m, n, r, N, tau, T = 6, 10, 2, 3, 4, 11
    orc = O.GreedyLoreOracle(m, n, r, N, tau, refresh_mode=mode, seed=5, basis_rank=k, lr=0.0)
    X = np.zeros((m, n))
    total_G = np.zeros((N, m, n))
    total_sent = np.zeros((N, m, n))
    for t in range(T):
        G = rng.standard_normal((N, m, n))
        X, info = orc.step(G, X)
        total_G += G
        total_sent += info.sent
        assert info.refresh == (t % tau == 0)
    assert np.allclose(total_sent + orc.E, total_G, atol=1e-11)


def test_refresh_uses_uncompressed_mean_and_resets_error():
    rng = np.random.default_rng(6)
    m, n, r, N = 5, 7, 2, 3
    orc = O.GreedyLoreOracle(m, n, r, N, tau=3, lr=1.0, beta1=0.0)
    X = np.zeros((m, n))
    for t in range(7):
        G = rng.standard_normal((N, m, n))
        E_before = orc.E.copy()
        X_before = X.copy()
        X, info = orc.step(G, X)
        if info.refresh:
            assert np.allclose(info.Ghat, (G + E_before).mean(0))
            assert np.allclose(X, X_before - info.Ghat)
            assert np.all(orc.E == 0)
            U = orc.U
            assert np.allclose(U.T @ U, np.eye(m), atol=1e-12)
        else:
            assert info.J is not None and len(info.J) == r
            assert np.allclose(info.P.T @ info.P, np.eye(r), atol=1e-12)


def test_rank_r_input_is_reconstructed_exactly():
    rng = np.random.default_rng(9)
    m, n, r, N = 7, 11, 3, 2
    A = rng.standard_normal((m, r)) @ rng.standard_normal((r, n))
    orc = O.GreedyLoreOracle(m, n, r, N, tau=1000, refresh_mode="alg4", lr=0.0, selection="exact")
    X = np.zeros((m, n))
    for t in range(3):
        X, info = orc.step(np.stack([A, A]), X)
        assert np.allclose(info.Ghat, A, atol=1e-10)
        assert np.allclose(orc.E, 0, atol=1e-10)


def test_orientation_rule_matches_transposed_problem():
    rng = np.random.default_rng(12)
    m, n, r, N = 9, 5, 2, 2
    kw = dict(tau=3, seed=17, lr=0.1, beta1=0.5)
    tall = O.GreedyLoreOracle(m, n, r, N, **kw)
    wide = O.GreedyLoreOracle(n, m, r, N, **kw)
    assert tall.transposed and not wide.transposed
    X1, X2 = np.zeros((m, n)), np.zeros((n, m))
    for t in range(7):
        G = rng.standard_normal((N, m, n))
        X1, i1 = tall.step(G, X1)
        X2, i2 = wide.step(np.swapaxes(G, 1, 2), X2)
        assert np.allclose(X1, X2.T, atol=1e-12)


def test_truncated_basis_keeps_top_k_and_is_orthogonal():
    rng = np.random.default_rng(13)
    m, n, r, k, N = 10, 14, 2, 4, 2
    orc = O.GreedyLoreOracle(m, n, r, N, tau=5, basis_rank=k, lr=0.0)
    G = rng.standard_normal((N, m, n))
    orc.step(G, np.zeros((m, n)))
    U_full, _ = O.left_singular_basis(G.mean(0))
    assert np.allclose(orc.U[:, :k], U_full[:, :k], atol=1e-12)
    assert np.allclose(orc.U.T @ orc.U, np.eye(m), atol=1e-12)


# ---------------------------------------------------------------------------------------------
# Optimizers: closed forms for a constant compressed gradient
# ---------------------------------------------------------------------------------------------
def test_msgd_closed_form():
    g = np.array([[0.5, -2.0], [3.0, 0.0]])
    X, Mo, lr, beta = np.ones((2, 2)), np.zeros((2, 2)), 0.1, 0.9
    T = 25
    for _ in range(T):
        X, Mo = O.msgd_update(X, Mo, g, lr, beta)
    # M_t = (1 - beta^{t+1}) g  =>  X_T = X_0 - lr * g * sum_{t<T} (1 - beta^{t+1})
    S = sum(1 - beta ** (t + 1) for t in range(T))
    assert np.allclose(Mo, (1 - beta ** T) * g)
    assert np.allclose(X, 1 - lr * S * g)


def test_adam_closed_form():
    g = np.array([[0.5, -2.0], [3.0, 1e-3]])
    X, Mo, Vo = np.zeros((2, 2)), np.zeros((2, 2)), np.zeros((2, 2))
    lr, b1, b2, eps = 0.01, 0.9, 0.999, 1e-8
    T = 30
    expect = np.zeros((2, 2))
    for t in range(T):
        X, Mo, Vo = O.adam_update(X, Mo, Vo, g, lr, b1, b2, eps)
        m_t = (1 - b1 ** (t + 1)) * g
        v_t = (1 - b2 ** (t + 1)) * g * g
        expect -= lr * m_t / (np.sqrt(v_t) + eps)    # eps outside the square root, no bias correction
    assert np.allclose(X, expect, rtol=1e-12, atol=1e-15)


def test_step_selection_is_unbiased_and_takes_the_largest_squares():
    """Prop. 4 through the full oracle step (not the free function): with the state frozen
    after a refresh, the mean of lambda-bar^2 over fresh v draws equals ||u_j^T Gbar||^2 for
    the refreshed (non-symmetric) U, and J always holds the r largest lambda-bar^2."""
    import copy
    rng = np.random.default_rng(41)
    m, n, r, N = 5, 7, 2, 3
    base = O.GreedyLoreOracle(m, n, r, N, tau=10 ** 6, seed=3, lr=0.0)
    G = rng.standard_normal((N, m, n)) + rng.standard_normal((1, m, n))
    base.step(G, np.zeros((m, n)))                   # refresh: U = SVD basis, E = 0
    assert not np.allclose(base.U, base.U.T)
    T = 12000
    sq = np.empty((T, m))
    for trial in range(T):
        o = copy.deepcopy(base)
        o.t = 1 + trial                              # a fresh v draw, same state
        _, info = o.step(G, np.zeros((m, n)))
        lam2 = info.lam_bar ** 2
        notJ = np.setdiff1d(np.arange(m), info.J)
        assert lam2[info.J].min() >= lam2[notJ].max()
        sq[trial] = lam2
    target = O.exact_energies(G.mean(0), base.U)
    assert np.all(np.abs(sq.mean(0) - target) < 5 * sq.std(0) / math.sqrt(T))


def test_algorithm1_lazy_svd_sends_the_top_r_projection():
    """Algorithm 1 (selection fixed, no error feedback): every compressed step of a period sends
    U_r U_r^T Gbar_t with U_r the top-r left singular vectors (numpy's SVD) of the period's
    refresh mean, and keeps E = 0."""
    rng = np.random.default_rng(21)
    m, n, r, N, tau = 12, 20, 3, 4, 4
    orc = O.GreedyLoreOracle(m, n, r, N, tau, selection="fixed", error_feedback=False, seed=5)
    X = np.zeros((m, n))
    Ur = None
    for t in range(2 * tau):
        G = rng.standard_normal((N, m, n))
        X, info = orc.step(G, X)
        if t % tau == 0:
            U, _, _ = np.linalg.svd(G.mean(axis=0))
            Ur = U[:, :r]
            assert not info.compressed
            continue
        assert np.array_equal(info.J, np.arange(r))
        np.testing.assert_allclose(np.abs(info.P), np.abs(Ur), atol=1e-10)   # columns up to sign
        np.testing.assert_allclose(info.Ghat, Ur @ (Ur.T @ G.mean(axis=0)), atol=1e-10)
        assert np.all(info.E == 0.0)


def test_prop1_frozen_subspace_makes_error_feedback_inert():
    """Prop. 1 through the Lazy-SVD selection: with P = U[:, :r] frozen for the period, E_i stays
    orthogonal to range(P), so runs with and without error feedback send the same Ghat."""
    rng = np.random.default_rng(22)
    m, n, r, N, tau = 10, 16, 2, 3, 5
    a = O.GreedyLoreOracle(m, n, r, N, tau, selection="fixed", error_feedback=True, seed=1)
    b = O.GreedyLoreOracle(m, n, r, N, tau, selection="fixed", error_feedback=False, seed=1)
    Xa = np.zeros((m, n))
    Xb = np.zeros((m, n))
    for t in range(tau):
        G = rng.standard_normal((N, m, n))
        Xa, ia = a.step(G, Xa)
        Xb, ib = b.step(G, Xb)
        np.testing.assert_allclose(ia.Ghat, ib.Ghat, atol=1e-12)
        if ia.compressed:
            assert np.abs(ia.P.T @ ia.E[0]).max() < 1e-12       # E_i is orthogonal to range(P)
            assert np.abs(ia.E).max() > 0.1                     # ... and not zero


def test_amsgrad_closed_form_and_monotone_normaliser():
    """The AMSGrad-type step of Appendix A: from a zero state one step gives
    X = -lr (1 - b1) G / sqrt((1 - b2) max G^2 + eps); with zero gradients afterwards V decays but
    the scalar normaliser Vt does not, and M keeps decaying geometrically."""
    rng = np.random.default_rng(23)
    G = rng.standard_normal((5, 7))
    lr, b1, b2, eps = 0.01, 0.9, 0.999, 1e-8
    X, M, V, Vt = O.amsgrad_update(np.zeros((5, 7)), np.zeros((5, 7)), np.zeros((5, 7)), 0.0, G, lr, b1, b2, eps)
    vt1 = (1 - b2) * float(np.max(G * G))
    assert Vt == pytest.approx(vt1, rel=1e-15)
    np.testing.assert_allclose(X, -lr * (1 - b1) * G / np.sqrt(vt1 + eps), rtol=1e-13)
    prev = Vt
    for k in range(1, 6):
        X2, M, V, Vt = O.amsgrad_update(X, M, V, Vt, np.zeros((5, 7)), lr, b1, b2, eps)
        assert float(np.max(V)) < prev and Vt == prev               # V decays, Vt holds
        np.testing.assert_allclose(M, (1 - b1) * b1 ** k * G, rtol=1e-13)
        np.testing.assert_allclose(X2 - X, -lr * M / np.sqrt(vt1 + eps), rtol=1e-12)
        X = X2


def test_adamw_first_step_and_bias_correction():
    """Bias-corrected AdamW: the first step has Mh = G and Vh = G^2, so from X0 it moves by
    -lr (G / (|G| + eps) + wd X0); with a constant gradient the corrected moments stay G, G^2."""
    rng = np.random.default_rng(24)
    G = rng.standard_normal((4, 6))
    X0 = rng.standard_normal((4, 6))
    lr, b1, b2, eps, wd = 0.01, 0.9, 0.999, 1e-8, 0.1
    X, M, V = O.adamw_update(X0, np.zeros_like(G), np.zeros_like(G), 1, G, lr, b1, b2, eps, wd)
    np.testing.assert_allclose(X, X0 - lr * (G / (np.abs(G) + eps) + wd * X0), rtol=1e-12)
    for s in range(2, 6):
        X2, M, V = O.adamw_update(X, M, V, s, G, lr, b1, b2, eps, wd)
        np.testing.assert_allclose(M / (1 - b1 ** s), G, rtol=1e-12)
        np.testing.assert_allclose(V / (1 - b2 ** s), G * G, rtol=1e-12)
        np.testing.assert_allclose(X2, X - lr * (G / (np.abs(G) + eps) + wd * X), rtol=1e-12)
        X = X2


@pytest.mark.parametrize("transposed", [False, True])
def test_algorithm5_is_adam_on_the_selected_coordinates(transposed):
    """Algorithm 5 when the refresh means have orthogonal rows: Mbar = diag(s) W (W with orthonormal
    rows) has U = I up to the order of s, so P holds coordinate vectors e_j, Rbar is those rows of
    the node mean, and the subspace Adam is Eq. adam on those rows alone, started afresh at every
    refresh; every other row of X stays put.  The second period's P shares row 1 with the first,
    so a state carried over the refresh would show."""
    mp, npr, r, N, tau, lr, b1, b2, eps = 6, 10, 2, 2, 3, 0.01, 0.9, 0.999, 1e-8
    rng = np.random.default_rng(31)
    W = np.linalg.qr(rng.standard_normal((npr, npr)))[0][:mp]
    scale = {0: np.array([5.0, 4.0, 3.0, 2.0, 1.5, 1.0]), 3: np.array([1.0, 5.0, 2.0, 4.0, 1.5, 3.0])}
    rows = {0: [0, 1], 3: [1, 3]}
    m, n = (npr, mp) if transposed else (mp, npr)
    orc = O.GreedyLoreOracle(m, n, r, N, tau, refresh_mode="alg4", optimizer="galore_adam", lr=lr, beta1=b1,
                             beta2=b2, eps=eps, selection="fixed", error_feedback=False)
    X0 = rng.standard_normal((mp, npr))
    X = X0.T.copy() if transposed else X0.copy()
    Xe = X0.copy()                                   # expected, oriented
    for t in range(5):
        if t in scale:
            Gbar = scale[t][:, None] * W
            D = rng.standard_normal((mp, npr))
            G = np.stack([Gbar + D, Gbar - D])
            sel, Ms, Vs = rows[t], np.zeros((r, npr)), np.zeros((r, npr))
        else:
            G = rng.standard_normal((N, mp, npr))
        Xe[sel], Ms, Vs = O.adam_update(Xe[sel], Ms, Vs, G.mean(axis=0)[sel], lr, b1, b2, eps)
        X, info = orc.step(np.swapaxes(G, 1, 2) if transposed else G, X)
        assert info.compressed and info.refresh == (t % tau == 0)
        assert sorted(np.argmax(np.abs(info.P), axis=0).tolist()) == rows[3 if t >= 3 else 0]
        np.testing.assert_allclose(X.T if transposed else X, Xe, rtol=0, atol=1e-12)
        assert np.all(info.E == 0)


def test_algorithm5_closed_form_constant_gradient():
    """A constant gradient in every step and node: P and R = P^T G stay fixed within the period,
    so M_t = (1 - b1^(t+1)) R and V_t = (1 - b2^(t+1)) R^2 and after T steps
    X_T = X_0 - lr P sum_t (1 - b1^(t+1)) R / (sqrt(1 - b2^(t+1)) |R| + eps); the weighting of
    Eq. adam (beta on the old state) is what this checks."""
    m, n, r, N, T, lr, b1, b2, eps = 7, 5, 2, 3, 6, 0.02, 0.8, 0.95, 1e-3
    rng = np.random.default_rng(32)
    G = rng.standard_normal((m, n))
    orc = O.GreedyLoreOracle(m, n, r, N, 100, refresh_mode="alg4", optimizer="galore_adam", lr=lr, beta1=b1,
                             beta2=b2, eps=eps, selection="fixed", error_feedback=False)
    X0 = rng.standard_normal((m, n))
    X = X0.copy()
    for _ in range(T):
        X, info = orc.step(np.stack([G] * N), X)
    Uo, _, _ = np.linalg.svd(G.T)                    # m > n: the basis lives on the n side
    P = info.P
    assert abs(abs(np.linalg.det(P.T @ Uo[:, :r])) - 1.0) < 1e-10   # span of the top-r singular vectors
    R = P.T @ G.T
    step = sum((1 - b1 ** (t + 1)) * R / (np.sqrt(1 - b2 ** (t + 1)) * np.abs(R) + eps) for t in range(T))
    np.testing.assert_allclose(X, X0 - lr * (P @ step).T, rtol=1e-12, atol=1e-14)


def test_algorithm5_rejects_other_schedules():
    for kw in ({"refresh_mode": "alg3"}, {"selection": "approx"}, {"error_feedback": True}, {"compress_start": 2}):
        args = dict(refresh_mode="alg4", selection="fixed", error_feedback=False, compress_start=0)
        args.update(kw)
        with pytest.raises(ValueError):
            O.GreedyLoreOracle(6, 8, 2, 2, 3, optimizer="galore_adam", **args)


@pytest.mark.parametrize("m,n,N,mode,opt", [(1, 5, 3, "alg3", "msgd"), (4, 9, 2, "alg4", "msgd"), (9, 4, 3, "alg3", "adam"),
                                             (5, 5, 1, "alg4", "adam"), (6, 11, 4, "alg3", "msgd")])
def test_full_rank_selection_is_uncompressed_data_parallel(m, n, N, mode, opt):
    """r = m': P is square and orthogonal, so P P^T = I, every E_i stays 0 and Ghat is the plain node
    mean: GreedyLore reduces to data-parallel MSGD / Adam on the mean gradient (m' = 1, square,
    transposed and N = 1 cases included)."""
    rng = np.random.default_rng(41 + m + n)
    r = min(m, n)
    kw = dict(lr=0.03, beta1=0.8, beta2=0.95, eps=1e-6, optimizer=opt)
    orc = O.GreedyLoreOracle(m, n, r, N, 3, refresh_mode=mode, seed=2, **kw)
    X = rng.standard_normal((m, n))
    Xe = X.copy()
    Mo, Vo = np.zeros((m, n)), np.zeros((m, n))
    for t in range(7):
        G = rng.standard_normal((N, m, n))
        X, info = orc.step(G, X)
        Gbar = G.mean(axis=0)
        if opt == "msgd":
            Xe, Mo = O.msgd_update(Xe, Mo, Gbar, kw["lr"], kw["beta1"])
        else:
            Xe, Mo, Vo = O.adam_update(Xe, Mo, Vo, Gbar, kw["lr"], kw["beta1"], kw["beta2"], kw["eps"])
        assert np.abs(info.E).max() < 1e-12
        np.testing.assert_allclose(X, Xe, rtol=1e-10, atol=1e-12)


def test_compress_start_warmup_is_uncompressed_then_refreshes():
    """Appendix F warm-up: the first K steps use the plain node mean with no error feedback
    (data-parallel MSGD), step K is the first refresh and the refreshes then follow every tau
    steps from there."""
    rng = np.random.default_rng(47)
    m, n, r, N, tau, K, lr, beta = 5, 8, 2, 3, 4, 3, 0.05, 0.7
    orc = O.GreedyLoreOracle(m, n, r, N, tau, seed=3, lr=lr, beta1=beta, compress_start=K)
    X = rng.standard_normal((m, n))
    Xe, Mo = X.copy(), np.zeros((m, n))
    refreshes = []
    for t in range(K + 2 * tau + 1):
        G = rng.standard_normal((N, m, n))
        X, info = orc.step(G, X)
        if info.refresh:
            refreshes.append(t)
        if t < K:
            assert not info.compressed and not info.refresh
            assert np.all(info.E == 0)
            Xe, Mo = O.msgd_update(Xe, Mo, G.mean(axis=0), lr, beta)
            np.testing.assert_allclose(X, Xe, rtol=1e-12, atol=1e-14)
    assert refreshes == [K, K + tau, K + 2 * tau]


def test_lemma2_holds_for_the_truncated_basis():
    """The truncated-basis reading keeps Lemma 2: its U (top-k singular vectors of an earlier
    refresh matrix, completed by Householder reflectors) is orthogonal, which is all the lemma
    uses, so Approx-Top-r on it contracts E||Gbar - P P^T Gbar||^2 <= (1 - r/m) ||Gbar||^2 even
    though U was computed from a different (stale) matrix."""
    rng = np.random.default_rng(23)
    m, n, N, r, k = 8, 10, 2, 2, 3
    stale = rng.standard_normal((m, n)) * np.linspace(2, 0.5, m)[:, None]
    Uk, _ = O.left_singular_basis(stale)
    U = O.householder_complement(Uk[:, :k])
    np.testing.assert_allclose(U.T @ U, np.eye(m), atol=1e-12)
    Ms = rng.standard_normal((N, m, n)) * np.linspace(3, 0.2, m)[None, :, None]
    Gbar = Ms.mean(0)
    T = 4000
    errs = np.empty(T)
    for t in range(T):
        V = O.gaussian_v(4343, t, m, n)
        J = O.argtop_r(O.approx_top_r_lambda(list(Ms), U, V) ** 2, r)
        P = U[:, J]
        errs[t] = np.linalg.norm(Gbar - P @ P.T @ Gbar) ** 2
    bound = (1 - r / m) * np.linalg.norm(Gbar) ** 2
    assert errs.mean() <= bound + 5 * errs.std() / math.sqrt(T)
