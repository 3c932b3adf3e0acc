"""Data-parallel GreedyLore across processes (world size 2, gloo, no GPU).

Each rank owns half of the N = 4 nodes; a step exchanges the shard's Approx-Top-r scores, then
its projected mean, or the node mean at a refresh (Algorithm 3's All-Reduce lines, Sec. 4.3),
through in-place all-reduces of the driver in `paper_2507_08784_gb300.dp`.  The shard engine is
built from the CPU oracle's pieces (tests/_dp_oracle.py), so the test checks the orchestration:
both ranks end with the same X, equal to the single-process oracle's with all four nodes, and the
floats a rank exchanges per step are Table 2's: m' + r n' on a compressed step, m' n' on an
Algorithm 3 refresh (m' n' + r n' under Algorithm 4, whose refresh step also compresses).
"""
import json
import os
import socket
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
N, N_LOCAL, STEPS = 4, 2, 7


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _grads(m, n, t, seed):
    """Node gradients of step t: a fixed rank-6 part plus fresh noise per node."""
    rng = np.random.default_rng(seed)
    S = rng.standard_normal((m, 6)) @ rng.standard_normal((6, n)) / np.sqrt(n)
    r2 = np.random.default_rng(1000 * seed + t)
    return np.stack([S + 0.1 * r2.standard_normal((m, n)) / np.sqrt(n) for _ in range(N)])


def _rank(rank, world, port, outdir, case):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    sys.path.insert(0, os.path.join(ROOT, "tests"))
    import torch.distributed as dist
    from _dp_oracle import OracleShard
    from paper_2507_08784_gb300.dp import DataParallelGreedyLore, allreduce_mean

    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        m, n, r, k, tau, opt, mode = case
        eng = OracleShard(m, n, r, N_LOCAL, tau, seed=11, basis_rank=k, optimizer=opt, lr=0.05,
                          refresh_mode=mode)
        dp = DataParallelGreedyLore(eng, allreduce_mean())
        X = np.zeros((m, n))
        floats = []
        for t in range(STEPS):
            G = _grads(m, n, t, seed=m + n)[rank * N_LOCAL:(rank + 1) * N_LOCAL]
            dp.step(G, X)
            floats.append(dp.last_step_floats)
        np.save(os.path.join(outdir, f"X{rank}.npy"), X)
        with open(os.path.join(outdir, f"floats{rank}.json"), "w") as f:
            json.dump(floats, f)
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("case", [
    (48, 80, 4, 12, 3, "msgd", "alg3"),      # truncated basis, m < n
    (80, 48, 5, 0, 3, "adam", "alg3"),       # paper-exact basis, m > n (worked on G^T)
    (40, 64, 4, 10, 3, "msgd", "alg4"),      # Algorithm 4: the refresh step compresses too
])
def test_two_ranks_match_single_process(tmp_path, case):
    mp = pytest.importorskip("torch.multiprocessing")
    sys.path.insert(0, ROOT)
    from oracle import greedylore as O
    world = 2
    mp.spawn(_rank, args=(world, _free_port(), str(tmp_path), case), nprocs=world, join=True)
    m, n, r, k, tau, opt, mode = case
    orc = O.GreedyLoreOracle(m, n, r, N, tau, refresh_mode=mode, optimizer=opt, lr=0.05, seed=11, basis_rank=k)
    Xo = np.zeros((m, n))
    for t in range(STEPS):
        Xo, _ = orc.step(_grads(m, n, t, seed=m + n), Xo)
    X0, X1 = np.load(tmp_path / "X0.npy"), np.load(tmp_path / "X1.npy")
    assert np.array_equal(X0, X1), "the ranks disagree"
    assert np.linalg.norm(X0 - Xo) <= 1e-10 * np.linalg.norm(Xo)
    mp_, np_ = min(m, n), max(m, n)
    want = []
    for t in range(STEPS):
        if t % tau == 0:
            want.append(mp_ * np_ + (r * np_ if mode == "alg4" else 0))
        else:
            want.append(mp_ + r * np_)
    for rk in range(world):
        assert json.load(open(tmp_path / f"floats{rk}.json")) == want
