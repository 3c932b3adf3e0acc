"""GPU-vs-oracle parity through the C ABI (marked gpu).

Tolerances: relative Frobenius error <= 1e-5 for fp32 arithmetic on fp32 or bf16-exact
inputs (the oracle works in fp64 on the same values) — X under every optimizer, E_i, Mbar,
P, Rbar and lambda-bar alike; selections compared as sets (a difference is accepted only
between lambda-bar^2 scores within 1e-5 of the largest, after which the runs are not compared
further).
"""
import math

import numpy as np
import pytest

import workloads as W
from oracle import greedylore as O
from tests._harness import lockstep, rel

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()


def _synthetic(m, n, N, rho, spectrum, noise, seed, dtype="f32"):
    cfg = W.Config("t", ((m, n),), N=N, r=1, basis_rank=0, tau=1, steps=1, grad_dtype=dtype, optimizer="msgd",
                   lr=0.01, beta1=0.9, beta2=0.0, eps=0.0, spectrum=spectrum, rho=rho, noise=noise,
                   master_seed=seed)
    prob = W.make_problem(cfg)
    return lambda t: W.gradients_numpy(prob, 0, t)


def _assert_reports(reps, tol=1e-5, lam_tol=1e-5):
    assert reps, "no steps compared"
    for rep in reps:
        for key, val in rep.errs.items():
            lim = lam_tol if key == "lambda" else tol
            assert val <= lim, f"step {rep.t} ({'refresh' if rep.refresh else 'compressed'}): {key} err {val:.3e}"


def test_cfg1_paper_exact_lockstep():
    """The small benchmark configuration: 256 x 128 fp32, N=4, r=4, tau=5, 20 steps, MSGD."""
    cfg = W.config("cfg1_tiny")
    prob = W.make_problem(cfg)
    m, n = cfg.shapes[0]
    reps = lockstep(m, n, cfg.r, cfg.N, cfg.steps, lambda t: W.gradients_numpy(prob, 0, t),
                    tau=cfg.tau, optimizer="msgd", lr=cfg.lr, beta1=cfg.beta1, seed=77, basis_rank=0)
    _assert_reports(reps)
    assert sum(r.refresh for r in reps) == math.ceil(cfg.steps / cfg.tau) or any(r.near_tie for r in reps)


def test_ragged_truncated_basis_lockstep():
    """Ragged sizes (several tiles + a tail), truncated basis k=12 with the Householder complement."""
    g = _synthetic(200, 333, 3, 24, lambda k: 1.0 / k, 0.05, 11)
    reps = lockstep(200, 333, 5, 3, 10, g, tau=4, optimizer="msgd", lr=0.05, beta1=0.8, seed=5, basis_rank=12)
    _assert_reports(reps)


def test_transposed_adam_bf16_lockstep():
    """m > n (Algorithm 4 orientation), bf16 gradients, Adam, full basis m' = 150."""
    g = _synthetic(333, 150, 2, 30, lambda k: k ** -1.0, 0.02, 12, dtype="bf16")
    reps = lockstep(333, 150, 6, 2, 8, g, dtype="bf16", tau=3, optimizer="adam", lr=1e-3, beta1=0.9,
                    beta2=0.999, eps=1e-8, seed=9, basis_rank=0)
    _assert_reports(reps, tol=1e-5)


def test_transposed_truncated_lockstep():
    g = _synthetic(410, 130, 4, 20, lambda k: 0.9 ** k, 0.03, 13)
    reps = lockstep(410, 130, 4, 4, 9, g, tau=4, optimizer="msgd", lr=0.02, beta1=0.9, seed=21, basis_rank=10)
    _assert_reports(reps)


def test_alg4_refresh_compressed_lockstep():
    """Algorithm 4 refresh (P = U[:, :r], no E reset).  The spectrum has clear gaps so the GPU's
    own refresh basis agrees with the oracle's top-r columns at the refresh step itself."""
    g = _synthetic(64, 100, 2, 8, lambda k: 2.0 ** (-k), 0.0, 14)
    reps = lockstep(64, 100, 3, 2, 7, g, tau=4, refresh_mode="alg4", optimizer="msgd", lr=0.1, beta1=0.5,
                    seed=3, basis_rank=0)
    _assert_reports(reps, tol=1e-5)


def test_compress_start_warmup_lockstep():
    g = _synthetic(96, 160, 2, 12, lambda k: 1.0 / k, 0.05, 15)
    reps = lockstep(96, 160, 4, 2, 8, g, tau=3, optimizer="msgd", lr=0.05, beta1=0.9, seed=4, basis_rank=0,
                    compress_start=3)
    _assert_reports(reps)
    assert [r.refresh for r in reps[:4]] == [False, False, False, True]


@pytest.mark.parametrize("m,n,k", [(96, 400, 16), (96, 400, 0), (300, 130, 24), (640, 1280, 16)])
def test_amsgrad_lockstep(m, n, k):
    """The AMSGrad-type optimizer of the analysis (scalar normaliser) on the tensor-core,
    paper-exact, transposed and FFMA-strip paths."""
    g = _synthetic(m, n, 3, 24, lambda j: 1.0 / j, 0.05, 90 + m + k)
    reps = lockstep(m, n, 5, 3, 6, g, tau=3, optimizer="amsgrad", lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8,
                    seed=12, basis_rank=k)
    _assert_reports(reps, tol=1e-5)


@pytest.mark.parametrize("m,n,k", [(96, 400, 16), (300, 130, 0), (640, 1280, 16)])
def test_adamw_lockstep(m, n, k):
    """Bias-corrected AdamW with weight decay on the tensor-core, transposed paper-exact and
    FFMA-strip paths."""
    g = _synthetic(m, n, 3, 24, lambda j: 1.0 / j, 0.05, 95 + m + k)
    reps = lockstep(m, n, 5, 3, 6, g, tau=3, optimizer="adamw", lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8,
                    weight_decay=0.01, seed=13, basis_rank=k)
    _assert_reports(reps, tol=1e-5)


@pytest.mark.parametrize("m,n,k", [(64, 100, 0), (96, 400, 16), (300, 130, 24), (640, 1280, 16), (256, 2304, 16)])
def test_galore_adam_lockstep(m, n, k):
    """Algorithm 5 (Adam state on the projected mean, zeroed at each refresh; Lazy-SVD P; no error
    feedback) on the paper-exact, tensor-core, transposed and FFMA-strip paths.  The spectra have
    clear gaps so the device's own refresh basis matches the oracle's at the refresh step, where
    Algorithm 5 already compresses with it."""
    g = _synthetic(m, n, 2, 8, lambda j: 2.0 ** (-j), 0.01, 100 + m + k)
    reps = lockstep(m, n, 3, 2, 7, g, tau=3, refresh_mode="alg4", optimizer="galore_adam", lr=1e-3, beta1=0.9,
                    beta2=0.999, eps=1e-8, seed=14, basis_rank=k, selection="fixed", error_feedback=False)
    _assert_reports(reps, tol=1e-5)
    assert [r.refresh for r in reps] == [True, False, False, True, False, False, True]


@pytest.mark.parametrize("m,n,k,selection", [(96, 400, 16, "fixed"), (96, 400, 0, "fixed"), (640, 1280, 16, "approx"),
                                              (300, 130, 24, "fixed"), (200, 824, 24, "approx")])
def test_without_error_feedback_lockstep(m, n, k, selection):
    """Algorithm 1 (Lazy-SVD selection, no error feedback) and Approx-Top-r without error
    feedback (the comparison of Sec. 4), on the tensor-core, FFMA-strip, transposed and
    paper-exact paths."""
    g = _synthetic(m, n, 3, 24, lambda j: 1.0 / j, 0.05, 80 + m + k)
    reps = lockstep(m, n, 5, 3, 6, g, tau=3, optimizer="msgd", lr=0.05, beta1=0.9, seed=11, basis_rank=k,
                    error_feedback=False, selection=selection)
    _assert_reports(reps)


@pytest.mark.parametrize("m,n,r,N,k", [(1, 5, 1, 1, 0), (7, 7, 7, 1, 0), (9, 40, 1, 3, 0), (40, 9, 2, 2, 3),
                                       (65, 65, 65, 2, 0)])
def test_edge_shapes(m, n, r, N, k):
    """Degenerate cases: m' = 1, r = m' (every column selected), r = 1, square, N = 1."""
    g = _synthetic(m, n, N, min(m, n), lambda j: 1.0 / j, 0.1, 16 + m)
    reps = lockstep(m, n, r, N, 6, g, tau=3, optimizer="msgd", lr=0.1, beta1=0.9, seed=2, basis_rank=k)
    _assert_reports(reps)


def test_refresh_full_basis_matches_svd():
    """The device eigen-solver's U against the oracle's SVD basis on a spectrum with gaps."""
    import torch
    import paper_2507_08784_gb300 as glr
    m, n, N = 96, 200, 2
    g = _synthetic(m, n, N, 96, lambda k: 0.93 ** k, 0.0, 17)
    G = g(0)
    dev = glr.GreedyLore(m, n, 2, N, tau=100, seed=1, basis_rank=0, lr=0.0)
    X = torch.zeros(m, n, device="cuda")
    dev.step([torch.from_numpy(G[i]).float().cuda() for i in range(N)], X)
    U = dev.basis().cpu().double().numpy()
    Uo, s = O.left_singular_basis(G.mean(0))
    assert np.abs(U.T @ U - np.eye(m)).max() < 1e-5
    # the leading columns are separated by >= 7% relative gaps: compare them elementwise
    cols = np.arange(24)
    assert np.abs(U[:, cols] - Uo[:, cols]).max() < 2e-4
    # every column is an eigenvector of Mbar Mbar^T: U^T H U is diagonal and sorted
    H = G.mean(0) @ G.mean(0).T
    D = U.T @ H @ U
    assert np.abs(D - np.diag(np.diag(D))).max() < 1e-5 * np.abs(D).max()
    assert np.all(np.diff(np.diag(D)) <= 1e-6 * D[0, 0])
    dev.close()


def test_refresh_truncated_principal_angles():
    """Block power iteration (q=4) + Rayleigh-Ritz on an input with sigma_k / sigma_{k+1} = 10:
    principal angles to the oracle's top-k subspace <= 1e-4 rad, Ritz vectors elementwise."""
    import torch
    import paper_2507_08784_gb300 as glr
    m, n, N, k = 300, 700, 2, 16
    spec = lambda j: 1.0 - 0.03 * (j - 1) if j <= k else 0.05 * 0.97 ** (j - k)  # noqa: E731
    g = _synthetic(m, n, N, 200, spec, 0.0, 18)
    G = g(0)
    dev = glr.GreedyLore(m, n, 4, N, tau=100, seed=1, basis_rank=k, power_iters=4, lr=0.0)
    X = torch.zeros(m, n, device="cuda")
    dev.step([torch.from_numpy(G[i]).float().cuda() for i in range(N)], X)
    U = dev.basis().cpu().double().numpy()
    Uo, s = O.left_singular_basis(G.mean(0))
    assert np.abs(U.T @ U - np.eye(m)).max() < 1e-5
    # sine of the largest principal angle = ||(I - Uo_k Uo_k^T) U_k||_2
    resid = U[:, :k] - Uo[:, :k] @ (Uo[:, :k].T @ U[:, :k])
    assert math.asin(min(1.0, np.linalg.norm(resid, 2))) <= 1e-4
    assert np.abs(U[:, :k] - Uo[:, :k]).max() < 1e-3
    dev.close()


@pytest.mark.parametrize("basis_rank", [0, 16])
def test_cfg2_full_size_lockstep(basis_rank):
    """The ResNet conv-gradient stack at its full sizes (8 matrices, N=8, r=8), three steps each
    (refresh + two compressed), with the launch configuration the benchmark uses."""
    cfg = W.config("cfg2_resnet")
    prob = W.make_problem(cfg)
    for li, (m, n) in enumerate(cfg.shapes):
        reps = lockstep(m, n, cfg.r, cfg.N, 3, lambda t, li=li: W.gradients_numpy(prob, li, t),
                        tau=cfg.tau, optimizer="msgd", lr=cfg.lr, beta1=cfg.beta1, seed=100 + li,
                        basis_rank=basis_rank, check_errors=(li % 2 == 0))
        _assert_reports(reps)


def test_invalid_step_arguments():
    import torch
    import paper_2507_08784_gb300 as glr
    dev = glr.GreedyLore(8, 12, 2, 2, tau=2)
    X = torch.zeros(8, 12, device="cuda")
    G = [torch.zeros(8, 12, device="cuda") for _ in range(2)]
    with pytest.raises(glr.GlrError):
        glr.glr_step(dev.handle, [G[0], 0], X)
    with pytest.raises(glr.GlrError):
        dev.force_selection([0, 0])
    dev.step(G, X)
    torch.cuda.synchronize()
    st = dev.stats()
    assert st["t"] == 1 and st["refreshes"] == 1 and st["comm_floats_total"] == 8 * 12
    dev.close()


def test_step_host_matches_device_step():
    import torch
    import paper_2507_08784_gb300 as glr
    m, n, N = 70, 90, 3
    g = _synthetic(m, n, N, 10, lambda k: 1.0 / k, 0.05, 19)
    a = glr.GreedyLore(m, n, 3, N, tau=3, seed=8)
    b = glr.GreedyLore(m, n, 3, N, tau=3, seed=8)
    Xa = torch.zeros(m, n, device="cuda")
    Xb = torch.zeros(m, n, device="cuda")
    Xh = torch.zeros(m, n).pin_memory()
    for t in range(5):
        G = g(t)
        Gd = [torch.from_numpy(G[i]).float().cuda() for i in range(N)]
        Gh = [torch.from_numpy(G[i]).float().pin_memory() for i in range(N)]
        a.step(Gd, Xa)
        b.step_host(Gh, Xb, Xh)
        torch.cuda.synchronize()
        assert torch.equal(Xa, Xb)
        assert torch.equal(Xa.cpu(), Xh)
    a.close()
    b.close()


@pytest.mark.parametrize("m,n,basis_rank,opt", [(200, 520, 16, "msgd"), (96, 300, 0, "adam"), (700, 300, 24, "msgd")])
def test_checkpoint_resume_is_bit_identical(m, n, basis_rank, opt):
    """glr_save after a few steps, glr_load into a fresh handle: both continue identically, across
    a refresh, on the tensor-core, paper-exact and transposed fused paths; a handle of another
    shape refuses the checkpoint."""
    import torch
    import paper_2507_08784_gb300 as glr
    r, N = 6, 3
    kw = dict(tau=3, optimizer=opt, lr=0.01, beta1=0.9, beta2=0.999, eps=1e-8, seed=31, basis_rank=basis_rank)
    a = glr.GreedyLore(m, n, r, N, **kw)
    b = glr.GreedyLore(m, n, r, N, **kw)
    rng = np.random.default_rng(9)
    grads = [[torch.from_numpy(rng.standard_normal((m, n)).astype(np.float32)).cuda() for _ in range(N)] for _ in range(8)]
    Xa = torch.zeros(m, n, device="cuda")
    for t in range(4):
        a.step(grads[t], Xa)
    state = a.state_dict()
    Xb = Xa.clone()
    b.load_state_dict(state)
    for t in range(4, 8):
        a.step(grads[t], Xa)
        b.step(grads[t], Xb)
        torch.cuda.synchronize()
        assert torch.equal(Xa, Xb), t
        Ja, *_ = a.selection()
        Jb, *_ = b.selection()
        assert np.array_equal(Ja, Jb), t
        assert torch.equal(a.error(0), b.error(0)), t
    assert a.stats()["t"] == b.stats()["t"] == 8
    c = glr.GreedyLore(m, n, r + 1, N, **kw)
    with pytest.raises(glr.GlrError):
        c.load_state_dict(state)
    with pytest.raises(glr.GlrError):
        b.load_state_dict(state[:100])
    for h in (a, b, c):
        h.close()


@pytest.mark.parametrize("basis_rank", [0, 16])
def test_step_group_host_matches_step_group(basis_rank):
    """The asynchronous grouped host step (double-buffered staging on a copy stream) gives the
    same X, bit for bit, as glr_step_group on device gradients; the host gradient buffers are
    rewritten between calls only after the stream has passed the step that read them."""
    import torch
    import paper_2507_08784_gb300 as glr
    shapes, r, N = [(256, 128), (64, 576), (128, 1152), (130, 96)], 4, 4
    kw = dict(tau=3, optimizer="adam", lr=1e-3, basis_rank=basis_rank)
    dev = [glr.GreedyLore(m, n, r, N, seed=70 + j, **kw) for j, (m, n) in enumerate(shapes)]
    hst = [glr.GreedyLore(m, n, r, N, seed=70 + j, **kw) for j, (m, n) in enumerate(shapes)]
    Xd = [torch.zeros(m, n, device="cuda") for m, n in shapes]
    Xg = [torch.zeros(m, n, device="cuda") for m, n in shapes]
    Xh = [torch.zeros(m, n).pin_memory() for m, n in shapes]
    rng = np.random.default_rng(5)
    # two sets of pinned host gradients, alternated, so a buffer is rewritten only two steps later
    hbuf = [[[torch.zeros(m, n).pin_memory() for _ in range(N)] for m, n in shapes] for _ in range(2)]
    for t in range(7):
        Gs = [[rng.standard_normal((m, n)).astype(np.float32) for _ in range(N)] for m, n in shapes]
        if t >= 2:
            torch.cuda.synchronize()                      # buffer t % 2 was read two steps ago
        for j in range(len(shapes)):
            for i in range(N):
                hbuf[t % 2][j][i].copy_(torch.from_numpy(Gs[j][i]))
        glr.glr_step_group(dev, [[torch.from_numpy(g).cuda() for g in Gs[j]] for j in range(len(shapes))], Xd)
        glr.glr_step_group_host(hst, hbuf[t % 2], Xg, Xh)
    torch.cuda.synchronize()
    for a, b, c in zip(Xd, Xg, Xh):
        assert torch.equal(a, b)
        assert torch.equal(a.cpu(), c)
    for h in dev + hst:
        h.close()


@pytest.mark.parametrize("basis_rank", [0, 16])
def test_step_group_equals_single_steps(basis_rank):
    """glr_step_group batches the streaming kernels of every matrix into shared launches; the
    results must be bit-identical to stepping each handle alone."""
    import torch
    import paper_2507_08784_gb300 as glr
    cfg = W.config("cfg2_resnet")
    prob = W.make_problem(cfg)
    shapes = list(cfg.shapes) + [(130, 96)]          # plus a transposed matrix
    kw = dict(tau=3, optimizer="msgd", lr=cfg.lr, beta1=cfg.beta1, basis_rank=basis_rank)
    solo = [glr.GreedyLore(m, n, cfg.r, cfg.N, seed=50 + j, **kw) for j, (m, n) in enumerate(shapes)]
    grp = [glr.GreedyLore(m, n, cfg.r, cfg.N, seed=50 + j, **kw) for j, (m, n) in enumerate(shapes)]
    Xs = [torch.zeros(m, n, device="cuda") for m, n in shapes]
    Xg = [torch.zeros(m, n, device="cuda") for m, n in shapes]
    gen = torch.Generator(device="cuda").manual_seed(7)
    for t in range(5):
        G = [[torch.randn(m, n, device="cuda", generator=gen) for _ in range(cfg.N)] for m, n in shapes]
        for h, g, x in zip(solo, G, Xs):
            h.step(g, x)
        glr.glr_step_group(grp, G, Xg)
        torch.cuda.synchronize()
        for j in range(len(shapes)):
            assert torch.equal(Xs[j], Xg[j]), (t, j)
            Ja, *_ = solo[j].selection()
            Jb, *_ = grp[j].selection()
            assert np.array_equal(Ja, Jb)
            assert torch.equal(solo[j].error(0), grp[j].error(0))
    for h in solo + grp:
        h.close()


@pytest.mark.parametrize("m,n,dtype,k", [(640, 1280, "f32", 16), (1280, 640, "bf16", 0), (1024, 256, "bf16", 16),
                                         (256, 1024, "f32", 0), (96, 2048, "f32", 8)])
def test_fused_kernel_shapes_lockstep(m, n, dtype, k):
    """Aligned shapes that take the fused kernels: m' > 512 runs the FFMA strip kernel, m' <= 512
    the tensor-core (3xTF32 mma.sync) strip kernel; transposed and bf16 gradients included."""
    g = _synthetic(m, n, 3, 24, lambda j: 1.0 / j, 0.05, 40 + m, dtype=dtype)
    reps = lockstep(m, n, 6, 3, 5, g, dtype=dtype, tau=3, optimizer="msgd", lr=0.05, beta1=0.9, seed=6,
                    basis_rank=k)
    _assert_reports(reps)


@pytest.mark.parametrize("m,n,dtype,k,r", [(384, 1536, "bf16", 16, 8), (200, 824, "f32", 24, 6),
                                           (256, 768, "f32", 16, 16), (768, 256, "f32", 16, 12),
                                           (64, 4096, "f32", 32, 8)])
def test_tensor_core_compose_paths_lockstep(m, n, dtype, k, r):
    """The tensor-core compose kernel's variants: tile copies with bf16 gradients, m' not a
    multiple of 16 and a partial last strip with k = 24, two q-tiles (r = 16), the cp.async path
    for transposed gradients with r = 12, and k = 32 at m' = 64 (epilogue partials outside the
    ring)."""
    g = _synthetic(m, n, 3, 24, lambda j: 1.0 / j, 0.05, 70 + m + r, dtype=dtype)
    reps = lockstep(m, n, r, 3, 5, g, dtype=dtype, tau=3, optimizer="msgd", lr=0.05, beta1=0.9, seed=8,
                    basis_rank=k)
    _assert_reports(reps)
