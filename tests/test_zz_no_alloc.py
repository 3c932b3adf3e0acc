"""The allocation-free selection entry point (glr_select_noalloc) against glr_step's own
selection.  Collected last on purpose: the entry point keeps state in a library-wide device
array, and it must give the same answer whether it runs in a fresh process or after
everything else."""
import numpy as np
import pytest

import workloads as W

pytestmark = pytest.mark.gpu


def _grads(m, n, N, seed):
    cfg = W.Config("t", ((m, n),), N=N, r=1, basis_rank=0, tau=1, steps=1, grad_dtype="f32", optimizer="msgd",
                   lr=0.01, beta1=0.9, beta2=0.0, eps=0.0, spectrum=lambda k: 1.0 / k, rho=12, noise=0.05,
                   master_seed=seed)
    prob = W.make_problem(cfg)
    return lambda t: W.gradients_numpy(prob, 0, t)


def test_select_noalloc_matches_step_selection():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    import paper_2507_08784_gb300 as glr

    m, n, N, r, seed = 200, 333, 3, 6, 4242
    g = _grads(m, n, N, 31)
    dev = glr.GreedyLore(m, n, r, N, tau=100, seed=seed, basis_rank=0, lr=0.01)
    X = torch.zeros(m, n, device="cuda")
    for t in range(3):                      # a refresh, then two compressed steps
        G = g(t)
        dev.step([torch.from_numpy(G[i]).float().cuda() for i in range(N)], X)
    torch.cuda.synchronize()
    J_ref, _, _, lam_ref, Mbar = dev.selection()
    U = dev.basis()
    lam_ref = lam_ref.cpu().numpy()
    for call in range(2):                   # two calls in a row share the library's scratch array
        lam = torch.full((m,), float("nan"), device="cuda")
        J = torch.full((r,), -1, dtype=torch.int32, device="cuda")
        glr.glr_select_noalloc(U, Mbar, seed, 2, r, lam, J)
        torch.cuda.synchronize()
        lam_np = lam.cpu().numpy()
        assert np.linalg.norm(lam_np - lam_ref) <= 1e-4 * np.linalg.norm(lam_ref), call
        assert sorted(J.cpu().tolist()) == sorted(J_ref.tolist()), call
    dev.close()

    # sizes beyond the fixed scratch are refused before any device work
    big = torch.empty(1, device="cuda")
    with pytest.raises(glr.GlrError) as err:
        glr._check(glr.load().glr_select_noalloc(16384, 70000, 4, big.data_ptr(), big.data_ptr(), 1, 0,
                                                 big.data_ptr(), big.data_ptr(), None))
    assert "exceed the fixed scratch" in str(err.value)
