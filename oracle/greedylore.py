"""GreedyLore CPU oracle (fp64) -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may import this module.  The CUDA
library never calls it, and it imports nothing from the CUDA package: the two
sides share no code.  It is a plain, slow, obviously correct restatement of
the method of "Greedy Low-Rank Gradient Compression for Distributed Learning
with Convergence Guarantees" (arXiv 2507.08784):

* Algorithm 3 (GreedyLore) for one layer matrix and N simulated nodes, with the
  orientation rule of Algorithm 4 (work on G^T when m > n, Appendix D);
* Algorithm 2 (Approx-Top-r): lambda_j^(i) = u_j^T G^(i) v_j, averaged over the
  nodes, squared, arg-top-r (Eq. lambda-bar, Eq. semi-lazy-svd-3);
* the exact-energy selection of Eq. semi-lazy-svd-2 (used by the Prop. 3 pins);
* the Semi-Lazy SVD refresh of Eq. SVD-P1 (full SVD every tau steps);
* error feedback Eq. ef1/ef2 as written in Algorithm 3 (E reset at a refresh)
  or Algorithm 4 (no reset, always compressed);
* the optimizers of Eq. msgd and Eq. adam (no bias correction, eps outside the
  square root), the AMSGrad-type Adam of the convergence analysis (Appendix A), and
  bias-corrected AdamW;
* the distributed Adam-type GaLore of Algorithm 5 (Appendix E): Adam state on the
  r x n' projected mean, reset at every refresh, with the Lazy-SVD projector and no
  error feedback;
* the truncated-basis reading: the top-k singular vectors of the refresh
  matrix completed to a full orthogonal U by Householder QR (the proofs of
  Prop. 3 and Lemma 2 only use that U is orthogonal).

Every routine works in float64.  Random vectors v_j come from Philox4x32-10
(Salmon et al., SC'11) + Box-Muller, implemented here from their published
definitions; the CUDA side implements the same integer generator on its own.

Parity status: every function in this file is pinned by ``tests/test_oracle.py``
(known-answer vectors, worked examples printed in the paper, closed forms,
invariants and brute force on tiny inputs).
"""
from __future__ import annotations

import dataclasses
import math
from typing import List, Optional, Sequence

import numpy as np

# ----------------------------------------------------------------------------
# Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel random numbers: as easy
# as 1, 2, 3", SC'11): 10 rounds of two 32x32->64 multiplies, key bumped by the
# Weyl constants between rounds.
# ----------------------------------------------------------------------------
PHILOX_M0 = 0xD2511F53
PHILOX_M1 = 0xCD9E8D57
PHILOX_W0 = 0x9E3779B9
PHILOX_W1 = 0xBB67AE85
_MASK32 = np.uint64(0xFFFFFFFF)

# Stream tags carried in counter word 3 (which draw a counter belongs to).
TAG_LAMBDA_V = 0x4C414D56   # the v_j of Algorithm 2


def philox4x32_10(c0, c1, c2, c3, k0: int, k1: int):
    """Philox4x32-10 on arrays of counters; returns four uint64 arrays of 32-bit words."""
    c0 = np.asarray(c0, dtype=np.uint64) & _MASK32
    c1 = np.asarray(c1, dtype=np.uint64) & _MASK32
    c2 = np.asarray(c2, dtype=np.uint64) & _MASK32
    c3 = np.asarray(c3, dtype=np.uint64) & _MASK32
    k0 = np.uint64(k0 & 0xFFFFFFFF)
    k1 = np.uint64(k1 & 0xFFFFFFFF)
    for rnd in range(10):
        if rnd:
            k0 = np.uint64((int(k0) + PHILOX_W0) & 0xFFFFFFFF)
            k1 = np.uint64((int(k1) + PHILOX_W1) & 0xFFFFFFFF)
        p0 = np.uint64(PHILOX_M0) * c0
        p1 = np.uint64(PHILOX_M1) * c2
        hi0, lo0 = p0 >> np.uint64(32), p0 & _MASK32
        hi1, lo1 = p1 >> np.uint64(32), p1 & _MASK32
        c0, c1, c2, c3 = (hi1 ^ c1 ^ k0), lo1, (hi0 ^ c3 ^ k1), lo0
    return c0, c1, c2, c3


def _unit_open(x):
    """Map a 32-bit word to (0, 1): its top 23 bits plus one half, times 2^-23.  Every value
    (k + 1/2) 2^-23, k < 2^23, has at most 24 significant bits, so it is exact in fp32 as well
    and lies in [2^-24, 1 - 2^-24]: fp32 and fp64 implementations draw identical uniforms, and
    neither ever reaches 0 or 1."""
    return ((np.asarray(x, dtype=np.uint64) >> np.uint64(9)).astype(np.float64) + 0.5) * 2.0 ** -23


def gaussian_v(seed: int, t: int, rows: int, cols: int, tag: int = TAG_LAMBDA_V) -> np.ndarray:
    """The random vectors v_j ~ N(0, I) of Eq. random-v, stacked as rows of a rows x cols matrix.

    Element (j, b) uses counter (b // 4, j, t, tag) and key (seed lo, seed hi); the four
    output words give two Box-Muller pairs (w0, w1) -> (z0, z1), (w2, w3) -> (z2, z3)
    and v_j[b] = z_{b mod 4}.  All nodes share the seed (Sec. 4.3), and v is drawn
    afresh at every step t.
    """
    nq = (cols + 3) // 4
    jj, qq = np.meshgrid(np.arange(rows, dtype=np.uint64), np.arange(nq, dtype=np.uint64), indexing="ij")
    w0, w1, w2, w3 = philox4x32_10(qq, jj, np.full_like(jj, t), np.full_like(jj, tag),
                                   seed & 0xFFFFFFFF, (seed >> 32) & 0xFFFFFFFF)
    out = np.empty((rows, nq, 4), dtype=np.float64)
    for (a, b), slot in (((w0, w1), 0), ((w2, w3), 2)):
        rad = np.sqrt(-2.0 * np.log(_unit_open(a)))
        ang = 2.0 * math.pi * _unit_open(b)
        out[:, :, slot] = rad * np.cos(ang)
        out[:, :, slot + 1] = rad * np.sin(ang)
    return out.reshape(rows, nq * 4)[:, :cols]


# ----------------------------------------------------------------------------
# Linear-algebra building blocks
# ----------------------------------------------------------------------------
def fix_signs(Q: np.ndarray) -> np.ndarray:
    """Sign convention for singular vectors: the largest-magnitude entry of each column is
    positive (first such index on ties).  The paper leaves the sign free."""
    idx = np.argmax(np.abs(Q), axis=0)
    sgn = np.sign(Q[idx, np.arange(Q.shape[1])])
    sgn[sgn == 0] = 1.0
    return Q * sgn[None, :]


def left_singular_basis(A: np.ndarray) -> tuple[np.ndarray, np.ndarray]:
    """U, sigma of SVD(A) (Eq. SVD-P1): full m x m U, singular values descending, signs fixed."""
    U, s, _ = np.linalg.svd(A, full_matrices=True)
    return fix_signs(U), s


def householder_complement(Q: np.ndarray) -> np.ndarray:
    """Complete orthonormal Q (m x k) to an orthogonal m x m U with U[:, :k] == Q.

    Textbook Householder QR of Q (Golub & Van Loan, Alg. 5.2.1): for column j,
    x = A[j:, j], beta = -sign(x_0) ||x||, v = x - beta e_1 scaled so v_0 = 1,
    H_j = I - tau v v^T with tau = (beta - x_0) / beta.  The product
    H_1 ... H_k is orthogonal; its first k columns are Q diag(beta) (|beta| = 1
    because Q is orthonormal), so multiplying those columns by beta gives Q back
    and the remaining m - k columns are the orthonormal complement.
    """
    m, k = Q.shape
    A = Q.astype(np.float64).copy()
    vs, taus, betas = [], [], []
    for j in range(k):
        x = A[j:, j].copy()
        alpha = x[0]
        sigma = np.linalg.norm(x)
        beta = -sigma if alpha >= 0 else sigma
        v = x.copy()
        v[0] = alpha - beta
        v = v / v[0]
        tau = (beta - alpha) / beta
        A[j:, j:] -= tau * np.outer(v, v @ A[j:, j:])
        vs.append(v)
        taus.append(tau)
        betas.append(beta)
    U = np.eye(m)
    for j in reversed(range(k)):        # U = H_1 (H_2 (... H_k I))
        v = vs[j]
        U[j:, :] -= taus[j] * np.outer(v, v @ U[j:, :])
    U[:, :k] *= np.array(betas)[None, :]
    return U


def argtop_r(scores: np.ndarray, r: int) -> np.ndarray:
    """Indices of the r largest scores (ties -> lower index), returned in ascending index order."""
    order = sorted(range(len(scores)), key=lambda j: (-scores[j], j))
    return np.array(sorted(order[:r]), dtype=np.int64)


# ----------------------------------------------------------------------------
# Optimizers (Sec. 2): MSGD Eq. msgd, Adam Eq. adam
# ----------------------------------------------------------------------------
def msgd_update(X, Mo, G, lr, beta):
    Mo = beta * Mo + (1.0 - beta) * G
    return X - lr * Mo, Mo


def amsgrad_update(X, Mo, Vo, Vt, G, lr, beta1, beta2, eps):
    """The AMSGrad-type Adam of the convergence analysis (Appendix A): the EMAs of Eq. adam and one
    scalar normaliser Vt = max(Vt, ||V||_max), X <- X - lr M / sqrt(Vt + eps)."""
    Mo = beta1 * Mo + (1.0 - beta1) * G
    Vo = beta2 * Vo + (1.0 - beta2) * G * G
    Vt = max(Vt, float(np.max(Vo)))
    return X - lr * Mo / np.sqrt(Vt + eps), Mo, Vo, Vt


def adamw_update(X, Mo, Vo, s, G, lr, beta1, beta2, eps, weight_decay):
    """Bias-corrected AdamW with decoupled weight decay (Loshchilov & Hutter) at optimizer step
    s = 1, 2, ...: Mh = M / (1 - b1^s), Vh = V / (1 - b2^s), X <- X - lr (Mh / (sqrt(Vh) + eps) + wd X)."""
    Mo = beta1 * Mo + (1.0 - beta1) * G
    Vo = beta2 * Vo + (1.0 - beta2) * G * G
    Mh = Mo / (1.0 - beta1 ** s)
    Vh = Vo / (1.0 - beta2 ** s)
    return X - lr * (Mh / (np.sqrt(Vh) + eps) + weight_decay * X), Mo, Vo


def adam_update(X, Mo, Vo, G, lr, beta1, beta2, eps):
    Mo = beta1 * Mo + (1.0 - beta1) * G
    Vo = beta2 * Vo + (1.0 - beta2) * G * G
    return X - lr * Mo / (np.sqrt(Vo) + eps), Mo, Vo


# ----------------------------------------------------------------------------
# Algorithm 2 and the exact-energy rule
# ----------------------------------------------------------------------------
def approx_top_r_lambda(M_nodes: Sequence[np.ndarray], U: np.ndarray, V: np.ndarray) -> np.ndarray:
    """lambda-bar of Algorithm 2: per node Lambda^(i)_j = u_j^T M_i v_j (row j of U^T M_i dotted
    with v_j), then the node mean."""
    lam = []
    for Mi in M_nodes:
        lam.append(np.sum((U.T @ Mi) * V, axis=1))
    return np.mean(lam, axis=0)


def exact_energies(Mbar: np.ndarray, U: np.ndarray) -> np.ndarray:
    """||u_j^T G||^2 for every column of U (Eq. semi-lazy-svd-2)."""
    return np.sum((U.T @ Mbar) ** 2, axis=1)


# ----------------------------------------------------------------------------
# Algorithm 3 / 4 for one layer matrix
# ----------------------------------------------------------------------------
@dataclasses.dataclass
class StepInfo:
    t: int
    refresh: bool
    compressed: bool
    J: Optional[np.ndarray]
    P: Optional[np.ndarray]
    lam_bar: Optional[np.ndarray]
    Rbar: Optional[np.ndarray]
    Mbar: np.ndarray
    Ghat: np.ndarray          # in the working (oriented) layout
    E: np.ndarray             # error buffers after the step, (N, m', n')
    sent: np.ndarray          # per node, what the node contributed this step (P R_i or M_i), oriented


class GreedyLoreOracle:
    """State and step of GreedyLore for one m x n layer and N nodes (Algorithms 3 and 4).

    refresh_mode "alg3": at t mod tau == 0 the node mean is used uncompressed and E is
    reset to 0 (Algorithm 3); "alg4": every step is compressed, the refresh takes
    P = U[:, :r], and E is never reset (Algorithm 4).  selection "fixed" keeps
    P = U[:, :r] for the whole period (the Lazy-SVD of Algorithm 1); error_feedback False
    keeps E = 0 (with selection "fixed": Algorithm 1).  basis_rank k = 0 keeps the full
    singular basis (paper-exact); 0 < k < m' keeps the top-k singular vectors and
    completes them with the Householder complement.  selection "approx" is
    Algorithm 2; "exact" is Eq. semi-lazy-svd-2.  compress_start K runs the first K
    steps uncompressed (plain mean, no error feedback; Appendix F warm-up).
    optimizer "galore_adam" is Algorithm 5: it needs refresh_mode "alg4" (the refresh step is
    compressed with the new P), selection "fixed", error_feedback False and compress_start 0.
    """

    def __init__(self, m, n, r, N, tau, *, refresh_mode="alg3", optimizer="msgd", lr=0.01,
                 beta1=0.9, beta2=0.999, eps=1e-8, seed=0, basis_rank=0, selection="approx",
                 compress_start=0, error_feedback=True, weight_decay=0.0):
        self.m, self.n, self.r, self.N, self.tau = m, n, r, N, tau
        self.transposed = m > n                      # Algorithm 4, m > n branch
        self.mp, self.np_ = min(m, n), max(m, n)
        if not (1 <= r <= self.mp):
            raise ValueError("need 1 <= r <= min(m, n)")
        self.refresh_mode, self.optimizer = refresh_mode, optimizer
        self.lr, self.beta1, self.beta2, self.eps = lr, beta1, beta2, eps
        self.seed, self.selection, self.compress_start = seed, selection, compress_start
        self.error_feedback, self.weight_decay = error_feedback, weight_decay
        self.k = self.mp if basis_rank in (0, None) else basis_rank
        if not (r <= self.k <= self.mp):
            raise ValueError("need r <= basis_rank <= min(m, n)")
        self.E = np.zeros((N, self.mp, self.np_))
        self.U = np.eye(self.mp)                     # Algorithm 3 input: U = I
        self.sigma = None
        self.Mo = np.zeros((m, n))
        self.Vo = np.zeros((m, n))
        self.Vt = 0.0                                # AMSGrad-type scalar normaliser
        if optimizer == "galore_adam":
            if refresh_mode != "alg4" or selection != "fixed" or error_feedback or compress_start != 0:
                raise ValueError("Algorithm 5 needs refresh_mode 'alg4', selection 'fixed', "
                                 "error_feedback False and compress_start 0")
        self.Ms = np.zeros((r, self.np_))            # Algorithm 5: subspace Adam state, r x n'
        self.Vs = np.zeros((r, self.np_))
        self.t = 0

    # -- helpers ---------------------------------------------------------------
    def orient(self, A):
        return np.swapaxes(A, -1, -2) if self.transposed else A

    def refresh_basis(self, Mbar):
        """Eq. SVD-P1 (full SVD); with k < m' keep the top-k columns + Householder complement."""
        U, s = left_singular_basis(Mbar)
        if self.k < self.mp:
            U = householder_complement(U[:, : self.k])
        return U, s

    def apply_optimizer(self, X, Ghat_oriented):
        G = self.orient(Ghat_oriented)               # back to m x n (transpose only when m > n)
        if self.optimizer == "msgd":
            X, self.Mo = msgd_update(X, self.Mo, G, self.lr, self.beta1)
        elif self.optimizer == "adamw":
            X, self.Mo, self.Vo = adamw_update(X, self.Mo, self.Vo, self.t + 1, G, self.lr, self.beta1, self.beta2,
                                               self.eps, self.weight_decay)
        elif self.optimizer == "amsgrad":
            X, self.Mo, self.Vo, self.Vt = amsgrad_update(X, self.Mo, self.Vo, self.Vt, G, self.lr, self.beta1,
                                                          self.beta2, self.eps)
        else:
            X, self.Mo, self.Vo = adam_update(X, self.Mo, self.Vo, G, self.lr, self.beta1, self.beta2, self.eps)
        return X

    def galore_adam(self, X, P, Rbar, refresh):
        """Algorithm 5's Adam-Update on the projected mean Rbar (r x n'): the state is zeroed at a
        refresh, M and V are the EMAs of Eq. adam (beta weighting the old state), and X moves by
        lr P (M / (sqrt(V) + eps)), transposed back when m > n; lr is applied once."""
        if refresh:
            self.Ms = np.zeros_like(Rbar)
            self.Vs = np.zeros_like(Rbar)
        self.Ms = self.beta1 * self.Ms + (1.0 - self.beta1) * Rbar
        self.Vs = self.beta2 * self.Vs + (1.0 - self.beta2) * Rbar * Rbar
        Rhat = self.Ms / (np.sqrt(self.Vs) + self.eps)
        return X - self.lr * self.orient(P @ Rhat)

    # -- one iteration -----------------------------------------------------------
    def step(self, G_nodes: np.ndarray, X: np.ndarray, force_J: Optional[Sequence[int]] = None):
        """One iteration t.  G_nodes: (N, m, n) local gradients; X: (m, n) weights.

        Returns (X_{t+1}, StepInfo).  force_J replaces the selection (used by the Prop. 1 pin).
        """
        t = self.t
        G = self.orient(np.asarray(G_nodes, dtype=np.float64))
        X = np.asarray(X, dtype=np.float64)
        if t < self.compress_start:                  # uncompressed warm-up: plain mean, no EF
            Mbar = G.mean(axis=0)
            X = self.apply_optimizer(X, Mbar)
            self.t += 1
            return X, StepInfo(t, False, False, None, None, None, None, Mbar, Mbar, self.E.copy(), G.copy())
        tt = t - self.compress_start
        M = G + self.E                               # Algorithm 3: G^(i) <- grad + E^(i)_{t-1}
        Mbar = M.mean(axis=0)
        refresh = tt % self.tau == 0
        lam_bar = None
        if refresh:
            self.U, self.sigma = self.refresh_basis(Mbar)
            if self.refresh_mode == "alg3":
                self.E = np.zeros_like(self.E)       # E reset, uncompressed mean is used
                X = self.apply_optimizer(X, Mbar)
                self.t += 1
                return X, StepInfo(t, True, False, None, None, None, None, Mbar, Mbar, self.E.copy(), M.copy())
            J = np.arange(self.r) if force_J is None else np.array(sorted(force_J))
        elif force_J is not None:
            J = np.array(sorted(force_J))
        elif self.selection == "exact":
            J = argtop_r(exact_energies(Mbar, self.U), self.r)
        elif self.selection == "fixed":
            J = np.arange(self.r)                    # Lazy-SVD (Algorithm 1): P = U[:, :r] all period
        else:
            V = gaussian_v(self.seed, t, self.mp, self.np_)
            lam_bar = approx_top_r_lambda(list(M), self.U, V)
            J = argtop_r(lam_bar ** 2, self.r)
        P = self.U[:, J]
        R = P.T @ M                                  # R_i = P^T G^(i)   (for every node i)
        self.E = M - P @ R                           # E_i = G^(i) - P R_i
        if not self.error_feedback:                  # Algorithm 1 / the no-EF comparison: E_i = 0
            self.E = np.zeros_like(self.E)
        Rbar = R.mean(axis=0)                        # All-Reduce
        Ghat = P @ Rbar
        if self.optimizer == "galore_adam":
            X = self.galore_adam(X, P, Rbar, refresh)
        else:
            X = self.apply_optimizer(X, Ghat)
        self.t += 1
        sent = P @ R
        return X, StepInfo(t, refresh, True, J, P, lam_bar, Rbar, Mbar, Ghat, self.E.copy(), sent)


def run(oracle: GreedyLoreOracle, grads: Sequence[np.ndarray], X0: np.ndarray):
    """Run len(grads) steps; returns the final X and the list of StepInfo."""
    X, infos = np.asarray(X0, dtype=np.float64), []
    for G in grads:
        X, info = oracle.step(G, X)
        infos.append(info)
    return X, infos
