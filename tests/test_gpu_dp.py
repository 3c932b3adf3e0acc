"""Data-parallel steps of the GPU library (glr_dp_begin / glr_dp_select / glr_dp_finish), marked gpu.

Two shard handles of N = 2 nodes each stand for two ranks of a data-parallel group; between the
phases their exposed buffers (the Approx-Top-r scores, the projected mean, the node mean at a
refresh) are averaged in place, as an all-reduce over two ranks would.  Checked against one handle
holding all N = 4 nodes and stepped with glr_step: the shards end every step with bit-identical X,
their selections match the single handle's (near-ties of the TF32 scores within 1e-2 of the
largest accepted), X agrees within the bf16 bound of the tcgen05 path (2e-2), and the floats the
shards expose per step are Table 2's m' + r n' (compressed) and m' n' (refresh).
"""
import numpy as np
import pytest

from tests._harness import rel, same_selection

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()


def _grads(m, n, N, seed, rho=48, noise=0.01):
    rng = np.random.default_rng(seed)
    Ub = np.linalg.qr(rng.standard_normal((m, rho)))[0]
    Vb = np.linalg.qr(rng.standard_normal((n, rho)))[0]
    S = (Ub * np.arange(1, rho + 1) ** -1.2) @ Vb.T

    def at(t):
        r2 = np.random.default_rng(10_000 * seed + t)
        return np.stack([S + noise * r2.standard_normal((m, n)) / np.sqrt(n) for _ in range(N)])
    return at


@pytest.mark.parametrize("m,n,mode,k", [(256, 704, "alg3", 64), (704, 256, "alg3", 64), (256, 640, "alg4", 64),
                                        (1152, 1280, "alg3", 0)])      # the full basis (blocked Jacobi)
def test_dp_shards_match_single_handle(m, n, mode, k):
    import torch
    import paper_2507_08784_gb300 as glr
    from paper_2507_08784_gb300.dp import DataParallelGreedyLore, ShardEngine

    r, N, steps = 32, 4, 7
    sched = dict(tau=3, refresh_mode=mode, optimizer="adam", lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8, seed=5,
                 basis_rank=k, grad_dtype="bf16")
    grads = _grads(m, n, N, seed=m + n)
    full = glr.GreedyLore(m, n, r, N, **sched)
    shards = [glr.GreedyLore(m, n, r, N // 2, **sched) for _ in range(2)]
    assert all(h.stats()["path"] == 2 for h in shards + [full])
    engines = [ShardEngine(h) for h in shards]
    drivers = [DataParallelGreedyLore(e) for e in engines]      # the exchange is done below, in place
    Xf = torch.zeros(m, n, device="cuda")
    Xs = [torch.zeros(m, n, device="cuda") for _ in shards]
    mp_, np_, rpad = min(m, n), max(m, n), (r + 31) // 32 * 32
    try:
        for t in range(steps):
            G = [torch.from_numpy(g.astype(np.float32)).to(torch.bfloat16).cuda().contiguous() for g in grads(t)]
            full.step(G, Xf)
            floats = 0
            bufs = [e.begin(G[2 * i:2 * i + 2]) for i, e in enumerate(engines)]
            for a, b in zip(*bufs):                               # the all-reduce of two ranks
                avg = (a + b) / 2
                a.copy_(avg)
                b.copy_(avg)
                floats += a.numel()
            bufs = [e.select() for e in engines]
            for a, b in zip(*bufs):
                avg = (a + b) / 2
                a.copy_(avg)
                b.copy_(avg)
                floats += a.numel()
            for e, X in zip(engines, Xs):
                e.finish(X)
            torch.cuda.synchronize()
            refresh = t % 3 == 0
            want = mp_ * np_ + (rpad * np_ if mode == "alg4" else 0) if refresh else mp_ + rpad * np_
            assert floats == want, f"step {t}: {floats} floats exchanged, Table 2 gives {want}"
            assert torch.equal(Xs[0], Xs[1]), f"step {t}: the shards disagree"
            Jf, _, _, lamf, _ = full.selection()
            Js, _, _, _, _ = shards[0].selection()
            if not refresh:
                ok = same_selection(Js, Jf, lamf.double().cpu().numpy(), 1e-2)
                assert ok, f"step {t}: selection {sorted(Js.tolist())[:6]}... vs {sorted(Jf.tolist())[:6]}..."
                if ok == "tie":
                    break
            assert rel(Xs[0].cpu().numpy(), Xf.cpu().numpy()) <= 2e-2, f"step {t}: X"
        assert drivers[0].floats_exchanged == 0                   # the drivers were not used to step
    finally:
        for h in shards + [full]:
            h.close()


def test_dp_calls_out_of_order_are_rejected():
    import torch
    import paper_2507_08784_gb300 as glr
    h = glr.GreedyLore(256, 512, 32, 2, tau=3, optimizer="adam", lr=1e-3, seed=1, basis_rank=64, grad_dtype="bf16")
    X = torch.zeros(256, 512, device="cuda")
    try:
        with pytest.raises(glr.GlrError):
            glr.glr_dp_select(h.handle)
        with pytest.raises(glr.GlrError):
            glr.glr_dp_finish(h.handle, X)
        G = [torch.zeros(256, 512, dtype=torch.bfloat16, device="cuda") for _ in range(2)]
        glr.glr_dp_begin(h.handle, G)
        with pytest.raises(glr.GlrError):
            glr.glr_dp_begin(h.handle, G)
        glr.glr_dp_select(h.handle)
        glr.glr_dp_finish(h.handle, X)
    finally:
        h.close()
    f = glr.GreedyLore(64, 96, 4, 2, tau=3, seed=1, basis_rank=16)            # fp32: not the tcgen05 path
    try:
        with pytest.raises(glr.GlrError):
            glr.glr_dp_begin(f.handle, [torch.zeros(64, 96, device="cuda")] * 2)
    finally:
        f.close()
