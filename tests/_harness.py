"""Lockstep driver: the CUDA library (through the C ABI) and the CPU oracle on the same seeded
inputs, compared step by step.  No value flows from the CUDA side into the oracle; after a
refresh the oracle's basis may be injected into the CUDA side (glr_set_basis) so that both
continue from one U (the non-unique singular directions of a noisy matrix would otherwise
make the runs select different columns)."""
from __future__ import annotations

import dataclasses
from typing import Callable, List, Optional

import numpy as np

from oracle import greedylore as O


def rel(a, b):
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-30))


@dataclasses.dataclass
class StepReport:
    t: int
    refresh: bool
    J_dev: Optional[np.ndarray]
    J_orc: Optional[np.ndarray]
    near_tie: bool
    errs: dict


def same_selection(J_dev, J_orc, lam_orc, tie_rel):
    """True when the sets agree; 'tie' when they differ only by near-tied scores."""
    a, b = set(J_dev.tolist()), set(J_orc.tolist())
    if a == b:
        return True
    scores = lam_orc ** 2
    thr = np.sort(scores)[::-1][len(J_orc) - 1]
    diff = (a - b) | (b - a)
    if all(abs(scores[j] - thr) <= tie_rel * scores.max() for j in diff):
        return "tie"
    return False


def lockstep(m, n, r, N, steps, grads: Callable[[int], np.ndarray], *, dtype="f32", inject_basis=True,
             tie_rel=1e-5, check_errors=True, **schedule) -> List[StepReport]:
    import torch
    import paper_2507_08784_gb300 as glr

    dev = glr.GreedyLore(m, n, r, N, grad_dtype=dtype, **schedule)
    orc = O.GreedyLoreOracle(m, n, r, N, **schedule)
    tdtype = torch.float32 if dtype == "f32" else torch.bfloat16
    X = torch.zeros(m, n, device="cuda")
    Xo = np.zeros((m, n))
    out = []
    try:
        for t in range(steps):
            G = grads(t)
            Gd = [torch.from_numpy(G[i]).to(tdtype).cuda().contiguous() for i in range(N)]
            dev.step(Gd, X)
            torch.cuda.synchronize()
            Xo, info = orc.step(G, Xo)
            J, P, Rbar, lam, Mbar = dev.selection()
            errs = {"X": rel(X.cpu().numpy(), Xo), "Mbar": rel(Mbar.cpu().numpy(), info.Mbar)}
            tie = False
            Jo = info.J
            if info.compressed:
                ok = same_selection(J, Jo, info.lam_bar, tie_rel) if info.lam_bar is not None else \
                    set(J.tolist()) == set(Jo.tolist())
                assert ok, f"step {t}: selection {sorted(J.tolist())} vs oracle {sorted(Jo.tolist())}"
                tie = ok == "tie"
                if info.lam_bar is not None:
                    errs["lambda"] = rel(lam.cpu().numpy(), info.lam_bar)
                if not tie and info.refresh:
                    # a refresh picks U[:, :r] of the device's own basis: P and Rbar are unique only
                    # up to rotations inside tied singular values, their product Ghat always is
                    errs["Ghat"] = rel((P @ Rbar).cpu().numpy(), info.Ghat)
                elif not tie:
                    errs["Rbar"] = rel(Rbar.cpu().numpy(), info.Rbar)
                    errs["P"] = rel(P.cpu().numpy(), info.P)
            else:
                assert np.all(J == -1)
            if check_errors and not tie:
                # ||E_dev - E|| <= tol (||E|| + 0.1 ||M_i||): relative to E, with an absolute floor at
                # the fp32 rounding of M_i - P P^T M_i (E vanishes up to rounding when r = m')
                worst = 0.0
                for i in range(N):
                    Ed = dev.error(i).cpu().numpy().astype(np.float64)
                    Mnorm = np.linalg.norm(info.sent[i] + info.E[i])
                    worst = max(worst, np.linalg.norm(Ed - info.E[i]) /
                                max(np.linalg.norm(info.E[i]) + 0.1 * Mnorm, 1e-30))
                errs["E"] = worst
            out.append(StepReport(t, info.refresh, J, Jo, tie, errs))
            if tie:
                break            # the runs legitimately diverge after a near-tied selection
            if info.refresh and inject_basis:
                U = orc.U if orc.k == orc.mp else orc.U[:, : orc.k]
                dev.set_basis(torch.from_numpy(np.ascontiguousarray(U)).float().cuda())
        return out
    finally:
        dev.close()
