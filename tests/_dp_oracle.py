"""A shard engine for the data-parallel driver built from the CPU oracle's pieces (test code).

One rank's shard of the N nodes of Algorithm 3, in fp64, with the exchange points of Sec. 4.3:
begin(G) exposes the shard's lambda-bar (Algorithm 2, on the shard's nodes) or its node mean,
select() takes the averaged value and exposes the shard's projected mean Rbar, finish(X) applies
the optimizer to the averaged Rbar and writes the shard's error feedback.  The exposed buffers are
torch CPU tensors sharing memory with the numpy state, so an in-place all-reduce lands in it.
"""
from __future__ import annotations

import numpy as np
import torch

from oracle import greedylore as O


class OracleShard:
    def __init__(self, m, n, r, N_local, tau, *, seed, basis_rank, optimizer="msgd", lr=0.01, beta1=0.9,
                 beta2=0.999, eps=1e-8, refresh_mode="alg3"):
        self.m, self.n, self.r, self.N, self.tau = m, n, r, N_local, tau
        self.transposed = m > n
        self.mp, self.np_ = min(m, n), max(m, n)
        self.k = self.mp if basis_rank in (0, None) else basis_rank
        self.seed, self.optimizer, self.refresh_mode = seed, optimizer, refresh_mode
        self.lr, self.beta1, self.beta2, self.eps = lr, beta1, beta2, eps
        self.E = np.zeros((N_local, self.mp, self.np_))
        self.U = np.eye(self.mp)
        self.Mo = np.zeros((m, n))
        self.Vo = np.zeros((m, n))
        self.t = 0

    def _orient(self, A):
        return np.swapaxes(A, -1, -2) if self.transposed else A

    def begin(self, G):
        self.M = self._orient(np.asarray(G, dtype=np.float64)) + self.E       # M_i = G_i + E_i
        self.refresh = self.t % self.tau == 0
        if self.refresh:
            self.mean = np.ascontiguousarray(self.M.mean(axis=0))
            return [torch.from_numpy(self.mean).view(-1)]
        V = O.gaussian_v(self.seed, self.t, self.mp, self.np_)
        self.lam = np.ascontiguousarray(O.approx_top_r_lambda(list(self.M), self.U, V))
        return [torch.from_numpy(self.lam)]

    def select(self):
        self.compressed = not (self.refresh and self.refresh_mode == "alg3")
        if self.refresh:                                                      # averaged node mean
            U, _ = O.left_singular_basis(self.mean)
            self.U = O.householder_complement(U[:, : self.k]) if self.k < self.mp else U
            if not self.compressed:
                return []
            J = np.arange(self.r)
        else:                                                                 # averaged lambda-bar
            J = O.argtop_r(self.lam ** 2, self.r)
        self.J = J
        self.P = self.U[:, J]
        self.R = np.stack([self.P.T @ Mi for Mi in self.M])                # R_i = P^T M_i
        self.rbar = np.ascontiguousarray(self.R.mean(axis=0))
        return [torch.from_numpy(self.rbar).view(-1)]

    def finish(self, X):
        if self.compressed:
            Ghat = self.P @ self.rbar                                         # averaged Rbar
            self.E = self.M - np.stack([self.P @ Ri for Ri in self.R])        # E_i = M_i - P R_i
        else:
            Ghat = self.mean
            self.E = np.zeros_like(self.E)
        G = self._orient(Ghat)
        Xn = np.asarray(X, dtype=np.float64)
        if self.optimizer == "msgd":
            Xn, self.Mo = O.msgd_update(Xn, self.Mo, G, self.lr, self.beta1)
        else:
            Xn, self.Mo, self.Vo = O.adam_update(Xn, self.Mo, self.Vo, G, self.lr, self.beta1, self.beta2, self.eps)
        X[...] = Xn
        self.t += 1
