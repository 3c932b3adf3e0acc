"""Failure reporting through the C ABI (marked gpu).  Every failure here is made on the host: a
gradient set that is all zero, an allocation larger than the device, a bounded wait on an
mbarrier that nothing arrives on, a corrupted checkpoint header, malformed caller buffers.
Nothing faults, traps or hangs the GPU; each kernel returns and the device stays usable.
"""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu

GLR_ENOMEM, GLR_ENUMERIC, GLR_ETIMEOUT, GLR_EINVAL = -2, -4, -6, -1


@pytest.fixture(scope="module", autouse=True)
def _lib():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()


def _sched(k, seed=3):
    return dict(tau=4, optimizer="msgd", lr=0.01, beta1=0.9, seed=seed, basis_rank=k)


@pytest.mark.parametrize("m,n,r,k,dtype,path", [
    (256, 704, 32, 64, "bf16", 2),       # tcgen05 path: power iteration with the one-CTA CholeskyQR factor
    (512, 4608, 8, 16, "f32", 1),        # the fp32 stack's path: grouped power iteration (k <= 32)
])
def test_zero_gradients_make_the_refresh_report_enumeric(m, n, r, k, dtype, path):
    """All-zero gradients at a refresh leave a zero node mean: its Gram matrix cannot be factored,
    and glr_get_stats reports GLR_ENUMERIC instead of a silently non-orthonormal basis."""
    import torch
    import paper_2507_08784_gb300 as glr
    N = 4
    h = glr.GreedyLore(m, n, r, N, grad_dtype=dtype, **_sched(k))
    try:
        assert h.stats()["path"] == path
        tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
        G = [torch.zeros(m, n, dtype=tdt, device="cuda") for _ in range(N)]
        X = torch.zeros(m, n, device="cuda")
        h.step(G, X)                                    # t = 0: a refresh of the zero mean
        with pytest.raises(glr.GlrError) as exc:
            h.stats()
        assert exc.value.code == GLR_ENUMERIC
    finally:
        h.close()


def test_allocation_beyond_the_device_reports_enomem():
    """N = 64 error buffers of 2^31 elements (512 GiB) cannot be allocated: GLR_ENOMEM, and the
    partial allocations are released (a normal handle is created right after)."""
    import paper_2507_08784_gb300 as glr
    with pytest.raises(glr.GlrError) as exc:
        glr.GreedyLore(32768, 65536, 8, 64, grad_dtype="bf16", **_sched(16))
    assert exc.value.code == GLR_ENOMEM
    h = glr.GreedyLore(256, 512, 8, 2, grad_dtype="f32", **_sched(16))
    h.close()


def test_bounded_wait_gives_up_and_the_device_stays_usable():
    """A bounded device wait that runs out (an mbarrier nothing arrives on, 1000 polls) counts the
    event: glr_get_stats reports GLR_ETIMEOUT; the kernel returned, and the next steps of another
    handle compute normally."""
    import torch
    import paper_2507_08784_gb300 as glr
    a = glr.GreedyLore(256, 704, 32, 4, grad_dtype="bf16", **_sched(64))
    b = glr.GreedyLore(256, 704, 32, 4, grad_dtype="bf16", **_sched(64))
    try:
        assert a.stats()["t"] == 0
        glr.glr_test_expire_wait(a.handle, 1000)
        torch.cuda.synchronize()
        with pytest.raises(glr.GlrError) as exc:
            a.stats()
        assert exc.value.code == GLR_ETIMEOUT
        X = torch.zeros(256, 704, device="cuda")
        for t in range(3):
            G = [torch.randn(256, 704, device="cuda").to(torch.bfloat16) * 0.01 for _ in range(4)]
            b.step(G, X)
        torch.cuda.synchronize()
        st = b.stats()
        assert st["t"] == 3 and bool(torch.isfinite(X).all()) and float(X.abs().max()) > 0
        with pytest.raises(glr.GlrError):
            glr.glr_test_expire_wait(a.handle, 0)       # out of range: GLR_EINVAL
    finally:
        a.close()
        b.close()


def _header_offsets():
    # CkptHeader: magic, version, m, n (8 B each), r, N, k, grad_dtype, optimizer, refresh_mode
    # (4 B each), seed, nbuf, buf_bytes, t, refreshes, comm, period_start (8 B each), e_zero,
    # force_refresh, last_uncompressed, basis_from_user, has_forceJ, pad (4 B each), role[6]
    return {"seed": 56, "has_forceJ": 128, "role": 136, "end": 160}


def test_corrupt_checkpoints_are_rejected():
    import torch
    import paper_2507_08784_gb300 as glr
    off = _header_offsets()
    m, n, r, N = 256, 704, 32, 4
    h = glr.GreedyLore(m, n, r, N, grad_dtype="bf16", **_sched(64, seed=11))
    other = glr.GreedyLore(m, n, r, N, grad_dtype="bf16", **_sched(64, seed=12))
    try:
        X = torch.zeros(m, n, device="cuda")
        for t in range(2):
            h.step([torch.randn(m, n, device="cuda").to(torch.bfloat16) for _ in range(N)], X)
        good = h.state_dict()
        h.load_state_dict(good)                                   # the intact checkpoint loads

        bad = good.copy()
        bad[off["role"]:off["role"] + 4] = np.frombuffer(np.int32(999).tobytes(), np.uint8)
        with pytest.raises(glr.GlrError) as exc:
            h.load_state_dict(bad)                                # a role past the buffers
        assert exc.value.code == GLR_EINVAL

        bad = good.copy()
        bad[off["role"]:off["role"] + 4] = bad[off["role"] + 8:off["role"] + 12]   # P names the Q buffer
        with pytest.raises(glr.GlrError):
            h.load_state_dict(bad)

        with pytest.raises(glr.GlrError) as exc:
            other.load_state_dict(good)                           # another seed: another v_j stream
        assert exc.value.code == GLR_EINVAL

        h.force_selection(list(range(r)))
        pend = h.state_dict()                                     # carries the pending selection
        assert int(np.frombuffer(pend[off["has_forceJ"]:off["has_forceJ"] + 4].tobytes(), np.int32)[0]) == 1
        bad = pend.copy()
        bad[off["end"]:off["end"] + 4] = np.frombuffer(np.int32(m + 5).tobytes(), np.uint8)
        with pytest.raises(glr.GlrError) as exc:
            h.load_state_dict(bad)                                # J outside [0, m')
        assert exc.value.code == GLR_EINVAL
        h.load_state_dict(pend)
    finally:
        h.close()
        other.close()


def test_noalloc_binding_checks_the_caller_buffers():
    import torch
    import paper_2507_08784_gb300 as glr
    mp, np_, r = 128, 256, 8
    U = torch.eye(mp, device="cuda")
    Mb = torch.randn(mp, np_, device="cuda")
    lam = torch.empty(mp, device="cuda")
    J = torch.empty(r, dtype=torch.int32, device="cuda")
    glr.glr_select_noalloc(U, Mb, 1, 1, r, lam, J)
    torch.cuda.synchronize()
    with pytest.raises(ValueError):
        glr.glr_select_noalloc(U[:64], Mb, 1, 1, r, lam, J)                 # U not m' x m'
    with pytest.raises(ValueError):
        glr.glr_select_noalloc(U.double(), Mb, 1, 1, r, lam, J)             # not fp32
    with pytest.raises(ValueError):
        glr.glr_select_noalloc(U, Mb.t(), 1, 1, r, lam, J)                  # not contiguous
    with pytest.raises(ValueError):
        glr.glr_select_noalloc(U, Mb, 1, 1, r, lam[: mp - 1], J)            # lambda too small
    with pytest.raises(ValueError):
        glr.glr_select_noalloc(U, Mb, 1, 1, r, lam, J.long())               # J not int32
    with pytest.raises(ValueError):
        glr.glr_select_noalloc(U, Mb, 1, 1, r, lam, J[: r - 1])             # J too small
