"""GPU parity of the tcgen05 tensor-core path (bf16 gradients, truncated basis, MSGD / Adam,
16 <= r <= 128) against the CPU oracle, through the C ABI (marked gpu).

Its products run as TF32 tensor-core MMAs (each fp32 operand read to 10 mantissa bits), so the
comparison uses the bf16 tolerance of the method's accuracy contract: relative Frobenius error
<= 2e-2 for X, Mbar, lambda-bar, P, Rbar and E_i.  Near-ties of the arg-top-r are accepted when
the swapped scores lie within 1e-2 of the largest score (a TF32 score carries a relative error of
about 1e-3).

Lockstep without drift: at every compressed step the device first takes the step with its own
Approx-Top-r selection from a saved state (glr_save), lambda-bar and J are compared with the
oracle's, then the state is restored (glr_load) and the step is taken again with the oracle's J
forced (glr_force_selection), so both sides continue from one selection even after a near-tie.
After each refresh the oracle's basis is copied into the device (glr_set_basis).  No device value
enters the oracle.
"""
import numpy as np
import pytest

from oracle import greedylore as O
from tests._harness import rel, same_selection

pytestmark = pytest.mark.gpu

TOL = 2e-2          # bf16 inputs, TF32 products
TIE = 1e-2


@pytest.fixture(scope="module", autouse=True)
def _lib():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()


def _bf16(x):
    x = np.asarray(x, dtype=np.float32)
    u = x.view(np.uint32)
    u = (u + np.uint32(0x7FFF) + ((u >> 16) & np.uint32(1))) & np.uint32(0xFFFF0000)
    return u.view(np.float32).astype(np.float64)


def _grads(m, n, N, seed, rho=48, noise=0.01):
    """Low rank plus noise (s_k = k^-1.2), rounded to bf16: G_i(t) = S + c Xi_i(t) / sqrt(n)."""
    rng = np.random.default_rng(seed)
    Ub = np.linalg.qr(rng.standard_normal((m, rho)))[0]
    Vb = np.linalg.qr(rng.standard_normal((n, rho)))[0]
    S = (Ub * np.arange(1, rho + 1) ** -1.2) @ Vb.T

    def at(t):
        r2 = np.random.default_rng(10_000 * seed + t)
        return np.stack([_bf16(S + noise * r2.standard_normal((m, n)) / np.sqrt(n)) for _ in range(N)])
    return at


def _sched(opt, tau, k, seed, mode="alg3"):
    return dict(tau=tau, refresh_mode=mode, optimizer=opt, lr=1e-3 if opt == "adam" else 0.01, beta1=0.9,
                beta2=0.999, eps=1e-8, seed=seed, basis_rank=k)


def _error_rel(Ed, E, M):
    return np.linalg.norm(Ed - E) / max(np.linalg.norm(E) + 0.1 * np.linalg.norm(M), 1e-30)


class _Pair:
    """One layer matrix on both sides."""

    def __init__(self, glr, m, n, r, N, sched, grads):
        import torch
        self.dev = glr.GreedyLore(m, n, r, N, grad_dtype="bf16", **sched)
        assert self.dev.stats()["path"] == 2, "expected the tcgen05 path (GLR_PATH_TCGEN05)"
        self.orc = O.GreedyLoreOracle(m, n, r, N, **sched)
        self.m, self.n, self.N, self.grads = m, n, N, grads
        self.X = torch.zeros(m, n, device="cuda")
        self.Xo = np.zeros((m, n))

    def device_grads(self, G):
        import torch
        return [torch.from_numpy(G[i]).to(torch.bfloat16).cuda().contiguous() for i in range(self.N)]


def _check_free_selection(p, Gd, info, t):
    """Device step with its own selection from a saved state; lambda-bar and J against the oracle;
    the state (and X) restored afterwards."""
    state = p.dev.state_dict()
    X0 = p.X.clone()
    p.dev.step(Gd, p.X)
    J, _, _, lam, _ = p.dev.selection()
    assert rel(lam.cpu().numpy(), info.lam_bar) <= TOL, f"step {t}: lambda-bar"
    ok = same_selection(J, info.J, info.lam_bar, TIE)
    assert ok, f"step {t}: selection {sorted(J.tolist())[:8]}... differs beyond near-ties"
    p.dev.load_state_dict(state)
    p.X.copy_(X0)


def _compare_step(p, info, t):
    import torch
    torch.cuda.synchronize()
    J, P, Rbar, lam, Mbar = p.dev.selection()
    assert rel(p.X.cpu().numpy(), p.Xo) <= TOL, f"step {t}: X"
    assert rel(Mbar.cpu().numpy(), info.Mbar) <= TOL, f"step {t}: Mbar"
    if info.compressed and info.refresh:
        # Algorithm 4's refresh step compresses with U[:, :r] of the device's own refresh: P and Rbar
        # are unique only up to rotations inside near-tied singular values, Ghat = P Rbar is not
        assert sorted(J.tolist()) == sorted(info.J.tolist()), f"step {t}: J = 0..r-1"
        assert rel((P @ Rbar).cpu().numpy(), info.Ghat) <= TOL, f"step {t}: Ghat"
        for i in range(p.N):
            Ed = p.dev.error(i).double().cpu().numpy()
            assert _error_rel(Ed, info.E[i], info.sent[i] + info.E[i]) <= TOL, f"step {t}: E_{i}"
    elif info.compressed:
        assert sorted(J.tolist()) == sorted(info.J.tolist()), f"step {t}: forced J"
        assert rel(P.cpu().numpy(), info.P) <= TOL, f"step {t}: P"
        assert rel(Rbar.cpu().numpy(), info.Rbar) <= TOL, f"step {t}: Rbar"
        for i in range(p.N):
            Ed = p.dev.error(i).double().cpu().numpy()
            assert _error_rel(Ed, info.E[i], info.sent[i] + info.E[i]) <= TOL, f"step {t}: E_{i}"
    else:
        assert np.all(J == -1)


def _run_pairs(glr, pairs, steps, grouped):
    import torch
    for t in range(steps):
        Gs = [p.grads(t) for p in pairs]
        Gds = [p.device_grads(G) for p, G in zip(pairs, Gs)]
        infos = []
        for p, G in zip(pairs, Gs):
            p.Xo, info = p.orc.step(G, p.Xo)
            infos.append(info)
        for p, Gd, info in zip(pairs, Gds, infos):
            if info.compressed and info.lam_bar is not None:
                _check_free_selection(p, Gd, info, t)
            if info.compressed and not info.refresh:
                p.dev.force_selection(info.J)
        if grouped:
            glr.glr_step_group([p.dev.handle for p in pairs], Gds, [p.X for p in pairs])
        else:
            for p, Gd in zip(pairs, Gds):
                p.dev.step(Gd, p.X)
        for p, info in zip(pairs, infos):
            _compare_step(p, info, t)
            if info.refresh:
                U = p.orc.U[:, : p.orc.k]
                p.dev.set_basis(torch.from_numpy(np.ascontiguousarray(U)).float().cuda())


@pytest.mark.parametrize("m,n,r,N,k,opt,mode", [
    (256, 704, 32, 4, 64, "adam", "alg3"),
    (704, 256, 32, 4, 64, "adam", "alg3"),       # m > n: worked on G^T (Algorithm 4 orientation)
    (392, 776, 48, 3, 96, "msgd", "alg3"),       # ragged row and column tiles
    (384, 1024, 128, 4, 256, "adam", "alg3"),    # r = 128, k = 256 (the d = 4096 decoder's ranks)
    (256, 512, 32, 8, 64, "msgd", "alg3"),       # N = 8: every accumulator column in use
    # Algorithm 4: the refresh step compresses with U[:, :r] of the device's own power-iteration
    # basis; MSGD keeps X linear in Ghat (Adam's first step is sign-like and turns the sub-tolerance
    # difference from the oracle's exact SVD basis into sign flips of near-zero entries)
    (256, 640, 32, 4, 64, "msgd", "alg4"),
])
def test_tcgen05_lockstep(m, n, r, N, k, opt, mode):
    import paper_2507_08784_gb300 as glr
    pair = _Pair(glr, m, n, r, N, _sched(opt, 4, k, 31 + r, mode), _grads(m, n, N, seed=m + n))
    try:
        _run_pairs(glr, [pair], 7, grouped=False)
    finally:
        pair.dev.close()


def _layer(d, ffn):
    return [(d, d)] * 4 + [(ffn, d)] * 2 + [(d, ffn)]


@pytest.mark.parametrize("name,d,ffn,N,r,k", [
    ("d4096_decoder_reduced", 512, 1376, 4, 64, 128),    # the d = 4096 stack's layer, N = 4, scaled down
    ("d2048_decoder_reduced", 256, 704, 8, 32, 64),      # the d = 2048 stack's layer, N = 8, scaled down
])
def test_tcgen05_grouped_layer_lockstep(name, d, ffn, N, r, k):
    """One decoder layer (Wq, Wk, Wv, Wo, Wgate, Wup, Wdown) through glr_step_group, as the
    benchmark runs the stacks, element by element against the oracle."""
    import paper_2507_08784_gb300 as glr
    pairs = [_Pair(glr, m, n, r, N, _sched("adam", 3, k, 700 + i), _grads(m, n, N, seed=50 + i))
             for i, (m, n) in enumerate(_layer(d, ffn))]
    try:
        _run_pairs(glr, pairs, 5, grouped=True)
    finally:
        for p in pairs:
            p.dev.close()


def test_tcgen05_group_equals_single_steps():
    """A grouped step is the same computation as per-handle steps: bit-identical results."""
    import torch
    import paper_2507_08784_gb300 as glr
    shapes = [(256, 704), (704, 256), (384, 768)]
    N, r, k = 4, 32, 64
    grads = [_grads(m, n, N, seed=9 + i) for i, (m, n) in enumerate(shapes)]
    mk = lambda: [glr.GreedyLore(m, n, r, N, grad_dtype="bf16", **_sched("adam", 3, k, 90 + i))
                  for i, (m, n) in enumerate(shapes)]
    A, B = mk(), mk()
    XA = [torch.zeros(m, n, device="cuda") for m, n in shapes]
    XB = [torch.zeros(m, n, device="cuda") for m, n in shapes]
    try:
        for t in range(5):
            Gd = [[torch.from_numpy(g).to(torch.bfloat16).cuda() for g in gr(t)] for gr in grads]
            glr.glr_step_group([h.handle for h in A], Gd, XA)
            for h, G, X in zip(B, Gd, XB):
                h.step(G, X)
        torch.cuda.synchronize()
        for i in range(len(shapes)):
            assert torch.equal(XA[i], XB[i]), f"matrix {i}: X differs"
            assert torch.equal(A[i].error(0), B[i].error(0)), f"matrix {i}: E_0 differs"
    finally:
        for h in A + B:
            h.close()


def test_tcgen05_checkpoint_resume_is_bit_identical():
    import torch
    import paper_2507_08784_gb300 as glr
    m, n, r, N, k = 384, 768, 32, 4, 64
    grads = _grads(m, n, N, seed=3)
    sch = _sched("adam", 3, k, 5)
    a = glr.GreedyLore(m, n, r, N, grad_dtype="bf16", **sch)
    b = glr.GreedyLore(m, n, r, N, grad_dtype="bf16", **sch)
    Xa = torch.zeros(m, n, device="cuda")
    dev = lambda t: [torch.from_numpy(g).to(torch.bfloat16).cuda() for g in grads(t)]
    try:
        for t in range(4):
            a.step(dev(t), Xa)
        b.load_state_dict(a.state_dict())
        Xb = Xa.clone()
        for t in range(4, 8):
            G = dev(t)
            a.step(G, Xa)
            b.step(G, Xb)
        torch.cuda.synchronize()
        assert torch.equal(Xa, Xb)
        assert torch.equal(a.error(1), b.error(1))
    finally:
        a.close()
        b.close()


@pytest.mark.parametrize("m,n,r,dtype,k", [(256, 704, 32, "bf16", 64), (512, 4608, 8, "f32", 16)])
def test_nonfinite_gradient_is_reported(m, n, r, dtype, k):
    """A NaN placed in one node's host-made gradient reaches the node mean: glr_get_stats returns
    GLR_ENONFINITE and counts it (tcgen05 path and the tensor-core compose of the fp32 stacks)."""
    import torch
    import paper_2507_08784_gb300 as glr
    N = 4
    h = glr.GreedyLore(m, n, r, N, grad_dtype=dtype, **_sched("msgd", 5, k, 1))
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    X = torch.zeros(m, n, device="cuda")
    try:
        G = [torch.randn(m, n).to(tdt).cuda() * 0.01 for _ in range(N)]
        h.step(G, X)
        assert h.stats()["nonfinite"] == 0
        Gh = torch.randn(m, n) * 0.01
        Gh[m // 3, n // 2] = float("nan")
        G[2] = Gh.to(tdt).cuda()
        h.step(G, X)
        with pytest.raises(glr.GlrError) as exc:
            h.stats()
        assert exc.value.code == -5
    finally:
        h.close()


# ---- the paper-exact (full) basis above m' = 1024 -------------------------------------------
# basis_rank = 0 keeps U = all m' left singular vectors of Mbar (Eq. SVD-P1 as the paper states
# it).  Above m' = 1024 the refresh is the blocked Jacobi (k_bjac.cu) and the scores are the dense
# U^T Mbar on the tensor cores; the rest of the step is the tcgen05 path above.

@pytest.mark.parametrize("m,n,r,N,opt,mode", [
    (2048, 2304, 32, 2, "adam", "alg3"),
    (2304, 2048, 64, 2, "msgd", "alg4"),      # m > n, and Algorithm 4 with the device's own basis
])
def test_tcgen05_full_basis_lockstep(m, n, r, N, opt, mode):
    import paper_2507_08784_gb300 as glr
    pair = _Pair(glr, m, n, r, N, _sched(opt, 3, 0, 61 + r, mode), _grads(m, n, N, seed=m + n + 1, rho=96))
    try:
        assert pair.dev.stats()["k"] == min(m, n)
        _run_pairs(glr, [pair], 5, grouped=False)
    finally:
        pair.dev.close()


def test_full_basis_blocked_refresh_matches_svd():
    """The blocked Jacobi's U at m' = 2048 against the oracle's SVD basis: orthonormal, the leading
    (gapped) columns elementwise, the leading 32-dimensional subspace (separated from the rest by
    a factor 0.3 in sigma) within 1e-4 rad in principal angle, U^T H U diagonal and sorted."""
    import torch
    import paper_2507_08784_gb300 as glr
    m, n, N = 2048, 2304, 2
    rng = np.random.default_rng(23)
    Ub = np.linalg.qr(rng.standard_normal((m, m)))[0]
    Vb = np.linalg.qr(rng.standard_normal((n, m)))[0]
    sig = 0.995 ** np.arange(m) * np.where(np.arange(m) < 32, 1.0, 0.3)
    S = (Ub * sig) @ Vb.T                               # every singular value distinct, 0.5 % gaps
    G = np.stack([_bf16(S + 0.02 * rng.standard_normal((m, n)) / np.sqrt(n)) for _ in range(N)])
    dev = glr.GreedyLore(m, n, 32, N, grad_dtype="bf16", tau=100, seed=1, basis_rank=0, lr=0.0)
    try:
        assert dev.stats()["path"] == 2
        X = torch.zeros(m, n, device="cuda")
        dev.step([torch.from_numpy(G[i]).to(torch.bfloat16).cuda() for i in range(N)], X)
        torch.cuda.synchronize()
        st = dev.stats()
        U = dev.basis().cpu().double().numpy()
    finally:
        dev.close()
    Mbar = G.mean(0)
    Uo, s = O.left_singular_basis(Mbar)
    H = Mbar @ Mbar.T
    orth = np.abs(U.T @ U - np.eye(m)).max()
    lead = np.abs(U[:, :24] - Uo[:, :24]).max()
    resid = U[:, :32] - Uo[:, :32] @ (Uo[:, :32].T @ U[:, :32])
    angle = float(np.arcsin(min(1.0, np.linalg.norm(resid, 2))))
    D = U.T @ H @ U
    off = np.abs(D - np.diag(np.diag(D))).max() / np.abs(D).max()
    msg = f"sweeps {st['last_refresh_sweeps']} orth {orth:.2e} lead {lead:.2e} angle {angle:.2e} off {off:.2e}"
    print(msg)
    # fp32 pair sweeps and split-TF32 block products (~2^-21 per product): a column passes ~30
    # rounds of 128-term products and 127-rotation pair sweeps per sweep, a few 1e-5 of accumulated
    # rounding over 15 sweeps (measured: orth 3.1e-5, leading columns 1.2e-4, off-diagonal 1e-5
    # relative)
    assert 1 <= st["last_refresh_sweeps"] <= 30, msg
    assert orth <= 2e-4, msg
    assert lead <= 5e-4, msg
    assert angle <= 1e-4, msg
    assert off <= 5e-5, msg
    assert np.all(np.diff(np.diag(D)) <= 1e-5 * D[0, 0]), msg


def test_full_basis_group_equals_single_steps():
    """Full-basis handles of two sizes (1152 x 1280, 2048 x 1536 stored transposed) through one
    grouped step are the same computation as per-handle steps, across two blocked-Jacobi refreshes
    (the grouped refresh solves each size on its own): bit-identical X, E_0 and basis."""
    import torch
    import paper_2507_08784_gb300 as glr
    shapes = [(1152, 1280), (2048, 1536)]
    N, r = 2, 32
    grads = [_grads(m, n, N, seed=71 + i, rho=64) for i, (m, n) in enumerate(shapes)]
    mk = lambda: [glr.GreedyLore(m, n, r, N, grad_dtype="bf16", **_sched("adam", 3, 0, 130 + i))
                  for i, (m, n) in enumerate(shapes)]
    A, B = mk(), mk()
    XA = [torch.zeros(m, n, device="cuda") for m, n in shapes]
    XB = [torch.zeros(m, n, device="cuda") for m, n in shapes]
    try:
        for t in range(5):
            Gd = [[torch.from_numpy(g).to(torch.bfloat16).cuda() for g in gr(t)] for gr in grads]
            glr.glr_step_group([h.handle for h in A], Gd, XA)
            for h, G, X in zip(B, Gd, XB):
                h.step(G, X)
        torch.cuda.synchronize()
        for i in range(len(shapes)):
            assert A[i].stats()["refreshes"] == 2
            assert torch.equal(XA[i], XB[i]), f"matrix {i}: X differs"
            assert torch.equal(A[i].error(0), B[i].error(0)), f"matrix {i}: E_0 differs"
            assert torch.equal(A[i].basis(), B[i].basis()), f"matrix {i}: U differs"
    finally:
        for h in A + B:
            h.close()


def test_full_basis_checkpoint_resume_is_bit_identical():
    """glr_save / glr_load of a full-basis handle on the tcgen05 path (U and its TF32 transpose are
    part of the state): both handles continue identically across a refresh."""
    import torch
    import paper_2507_08784_gb300 as glr
    m, n, r, N = 1280, 1536, 32, 2
    grads = _grads(m, n, N, seed=5, rho=64)
    kw = _sched("msgd", 3, 0, 44)
    a = glr.GreedyLore(m, n, r, N, grad_dtype="bf16", **kw)
    b = glr.GreedyLore(m, n, r, N, grad_dtype="bf16", **kw)
    try:
        Xa = torch.zeros(m, n, device="cuda")
        Gs = [[torch.from_numpy(g).to(torch.bfloat16).cuda() for g in grads(t)] for t in range(7)]
        for t in range(2):
            a.step(Gs[t], Xa)
        b.load_state_dict(a.state_dict())
        Xb = Xa.clone()
        for t in range(2, 7):
            a.step(Gs[t], Xa)
            b.step(Gs[t], Xb)
            torch.cuda.synchronize()
            assert torch.equal(Xa, Xb), t
            assert np.array_equal(a.selection()[0], b.selection()[0]), t
        assert torch.equal(a.basis(), b.basis())
    finally:
        a.close()
        b.close()


@pytest.mark.parametrize("m,n,kw", [
    (2048, 2304, dict(grad_dtype="f32")),          # fp32 gradients: no full-basis path above 1024
    (1100, 2304, dict(grad_dtype="bf16")),         # m' not a multiple of 128
    (8192, 8192, dict(grad_dtype="bf16")),         # m' above 4096
])
def test_full_basis_above_1024_needs_tcgen05_conditions(m, n, kw):
    import paper_2507_08784_gb300 as glr
    with pytest.raises(glr.GlrError) as e:
        glr.GreedyLore(m, n, 32, 2, basis_rank=0, tau=10, **kw)
    assert "full basis" in str(e.value)
