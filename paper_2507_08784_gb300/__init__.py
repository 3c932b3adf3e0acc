"""GreedyLore on GB300: Python binding of libglr.so.

The functions below carry the names of the C entry points declared in
``include/glr.h`` and only marshal arguments (tensor addresses, the CUDA
stream, the schedule struct).  Every step of the method runs in the CUDA
library; PyTorch provides device memory and streams.  There is no CPU path:
if ``libglr.so`` is missing, ``load()`` raises.
"""
from __future__ import annotations

import ctypes
from typing import Optional, Sequence

import numpy as np
import torch

from . import _lib
from ._lib import (GLR_ADAM, GLR_ADAMW, GLR_ALG3, GLR_ALG4, GLR_AMSGRAD, GLR_BF16, GLR_F32,  # noqa: F401
                   GLR_GALORE_ADAM, GLR_MSGD, GLR_OK, PHASE_NAMES, GlrProfile, GlrSchedule, GlrStats, load)

__all__ = ["GlrError", "make_schedule", "glr_create", "glr_destroy", "glr_step", "glr_step_group",
           "glr_step_group_host", "glr_step_host", "glr_save", "glr_load", "glr_refresh", "glr_get_stats", "glr_last_error", "glr_get_error", "glr_get_selection",
           "glr_get_basis", "glr_set_basis", "glr_force_selection", "glr_test_expire_wait", "glr_profile_enable",
           "glr_profile_read", "glr_select_noalloc", "GreedyLore", "load"]


class GlrError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"GLR error {code}: {msg}")
        self.code = code


def _check(rc: int, handle=None, group=()):
    if rc != GLR_OK:
        lib = load()
        msg = lib.glr_last_error(handle)
        for h in group:                       # a grouped call reports on the failing handle
            if msg:
                break
            msg = lib.glr_last_error(h)
        raise GlrError(rc, msg.decode() if msg else "")


def _stream_ptr(stream) -> int:
    if stream is None:
        stream = torch.cuda.current_stream()
    return int(stream.cuda_stream) if hasattr(stream, "cuda_stream") else int(stream)


# "galore_adam" is Algorithm 5; it needs refresh_mode "alg4", selection "fixed" and
# error_feedback False (glr_create rejects other combinations)
_OPTIMIZERS = {"msgd": GLR_MSGD, "adam": GLR_ADAM, "amsgrad": GLR_AMSGRAD, "adamw": GLR_ADAMW,
               "galore_adam": GLR_GALORE_ADAM}


def make_schedule(tau: int, refresh_mode: str = "alg3", optimizer: str = "msgd", lr: float = 0.01,
                  beta1: float = 0.9, beta2: float = 0.999, eps: float = 1e-8, seed: int = 0,
                  basis_rank: int = 0, power_iters: int = 4, grad_dtype: str = "f32",
                  compress_start: int = 0, error_feedback: bool = True, selection: str = "approx",
                  weight_decay: float = 0.0) -> GlrSchedule:
    """The glr_schedule of include/glr.h from keyword arguments.

    tau            refresh period of the Semi-Lazy SVD (>= 1)
    refresh_mode   "alg3" (refresh step uses the uncompressed mean and resets E) or "alg4"
                   (the refresh step is compressed with P = U[:, :r], E kept)
    optimizer      "msgd" (Eq. msgd), "adam" (Eq. adam), "amsgrad" (the analysis' AMSGrad-type
                   rule), "adamw" (bias-corrected, decoupled weight_decay) or "galore_adam"
                   (Algorithm 5: needs refresh_mode "alg4", selection "fixed",
                   error_feedback False); lr, beta1, beta2, eps as in those equations
    seed           key of the shared random vectors v_j (give every matrix its own)
    basis_rank     0: the full singular basis (paper-exact, min(m, n) <= 1024); r..512: the top-k
                   singular vectors completed by Householder reflectors, refreshed with
                   power_iters block power iterations
    grad_dtype     "f32" or "bf16" (the gradients' storage type)
    compress_start the first compress_start steps run uncompressed (Appendix F warm-up)
    error_feedback False drops error feedback (with selection "fixed": Algorithm 1)
    selection      "approx" (Algorithm 2) or "fixed" (P = U[:, :r] for the whole period)
    """
    return GlrSchedule(tau=tau, refresh_mode={"alg3": GLR_ALG3, "alg4": GLR_ALG4}[refresh_mode],
                       optimizer=_OPTIMIZERS[optimizer], lr=lr, beta1=beta1,
                       beta2=beta2, eps=eps, seed=seed & (2 ** 64 - 1), basis_rank=basis_rank,
                       power_iters=power_iters, grad_dtype={"f32": GLR_F32, "bf16": GLR_BF16}[grad_dtype],
                       compress_start=compress_start, no_error_feedback=0 if error_feedback else 1,
                       selection={"approx": 0, "fixed": 1}[selection], weight_decay=weight_decay)


def glr_create(m: int, n: int, r: int, N: int, schedule: GlrSchedule) -> ctypes.c_void_p:
    lib = load()
    h = ctypes.c_void_p()
    _check(lib.glr_create(m, n, r, N, ctypes.byref(schedule), ctypes.byref(h)))
    return h


def glr_destroy(h) -> None:
    _check(load().glr_destroy(h), h)


def _ptr_array(tensors: Sequence) -> ctypes.Array:
    arr = (ctypes.c_void_p * len(tensors))()
    for i, t in enumerate(tensors):
        arr[i] = t.data_ptr() if isinstance(t, torch.Tensor) else int(t)
    return arr


def glr_step(h, G: Sequence[torch.Tensor], X: torch.Tensor, stream=None) -> None:
    _check(load().glr_step(h, _ptr_array(G), X.data_ptr(), _stream_ptr(stream)), h)


def _exchange(ex) -> list:
    return [(int(ex.ptr[i]), int(ex.floats[i])) for i in range(ex.count)]


def glr_dp_begin(h, G: Sequence[torch.Tensor], stream=None) -> list:
    """First phase of a data-parallel step (see glr.h): [(device pointer, floats)] to average."""
    ex = _lib.GlrDpExchange()
    _check(load().glr_dp_begin(h, _ptr_array(G), _stream_ptr(stream), ctypes.byref(ex)), h)
    return _exchange(ex)


def glr_dp_select(h, stream=None) -> list:
    """Second phase: the selection (or refresh) on the averaged buffers; returns Rbar^T to average."""
    ex = _lib.GlrDpExchange()
    _check(load().glr_dp_select(h, _stream_ptr(stream), ctypes.byref(ex)), h)
    return _exchange(ex)


def glr_dp_finish(h, X: torch.Tensor, stream=None) -> None:
    """Third phase: the update of X with the averaged Rbar and the local error feedback."""
    _check(load().glr_dp_finish(h, X.data_ptr(), _stream_ptr(stream)), h)


def glr_step_group(handles: Sequence, G: Sequence[Sequence[torch.Tensor]], X: Sequence[torch.Tensor],
                   stream=None) -> None:
    """One step of several handles with batched launches (see glr.h)."""
    n = len(handles)
    hs = (ctypes.c_void_p * n)(*[h.handle if isinstance(h, GreedyLore) else h for h in handles])
    gp = [_ptr_array(g) for g in G]
    garr = (ctypes.c_void_p * n)(*[ctypes.addressof(a) for a in gp])
    xarr = (ctypes.c_void_p * n)(*[x.data_ptr() for x in X])
    _check(load().glr_step_group(hs, n, garr, xarr, _stream_ptr(stream)), group=list(hs))


def glr_step_group_host(handles: Sequence, G_host: Sequence[Sequence[torch.Tensor]], X: Sequence[torch.Tensor],
                        X_host_out: Optional[Sequence[torch.Tensor]] = None, stream=None) -> None:
    """One grouped step from host gradients; only enqueues the work (see glr.h)."""
    n = len(handles)
    hs = (ctypes.c_void_p * n)(*[h.handle if isinstance(h, GreedyLore) else h for h in handles])
    gp = [_ptr_array(g) for g in G_host]
    garr = (ctypes.c_void_p * n)(*[ctypes.addressof(a) for a in gp])
    xarr = (ctypes.c_void_p * n)(*[x.data_ptr() for x in X])
    oarr = None if X_host_out is None else (ctypes.c_void_p * n)(*[o.data_ptr() for o in X_host_out])
    _check(load().glr_step_group_host(hs, n, garr, xarr, oarr, _stream_ptr(stream)), group=list(hs))


def glr_step_host(h, G_host: Sequence[torch.Tensor], X: torch.Tensor, X_host_out: Optional[torch.Tensor] = None,
                  stream=None) -> None:
    _check(load().glr_step_host(h, _ptr_array(G_host), X.data_ptr(),
                                None if X_host_out is None else X_host_out.data_ptr(), _stream_ptr(stream)), h)


def glr_save(h, stream=None) -> np.ndarray:
    """The handle's whole state as a host byte array (see glr.h)."""
    lib = load()
    size = ctypes.c_int64(0)
    _check(lib.glr_state_size(h, ctypes.byref(size)), h)
    buf = np.empty(size.value, dtype=np.uint8)
    _check(lib.glr_save(h, buf.ctypes.data, size.value, _stream_ptr(stream)), h)
    return buf


def glr_load(h, state, stream=None) -> None:
    """Restore a checkpoint written by glr_save into a handle of the same shape and schedule."""
    buf = np.ascontiguousarray(state, dtype=np.uint8)
    _check(load().glr_load(h, buf.ctypes.data, buf.size, _stream_ptr(stream)), h)


def glr_refresh(h) -> None:
    _check(load().glr_refresh(h), h)


def glr_get_stats(h) -> dict:
    st = GlrStats()
    _check(load().glr_get_stats(h, ctypes.byref(st)), h)
    return {name: getattr(st, name) for name, _ in GlrStats._fields_}


def glr_last_error(h=None) -> str:
    msg = load().glr_last_error(h)
    return msg.decode() if msg else ""


def glr_get_error(h, i: int, out: torch.Tensor, stream=None) -> None:
    _check(load().glr_get_error(h, i, out.data_ptr(), _stream_ptr(stream)), h)


def glr_get_selection(h, r: int, P: Optional[torch.Tensor] = None, Rbar: Optional[torch.Tensor] = None,
                      lam: Optional[torch.Tensor] = None, Mbar: Optional[torch.Tensor] = None,
                      stream=None) -> np.ndarray:
    J = np.zeros(r, dtype=np.int32)
    ptr = lambda t: None if t is None else t.data_ptr()  # noqa: E731
    _check(load().glr_get_selection(h, J.ctypes.data, ptr(P), ptr(Rbar), ptr(lam), ptr(Mbar),
                                    _stream_ptr(stream)), h)
    return J


def glr_get_basis(h, out: torch.Tensor, stream=None) -> None:
    _check(load().glr_get_basis(h, out.data_ptr(), _stream_ptr(stream)), h)


def glr_set_basis(h, Q: torch.Tensor, stream=None) -> None:
    _check(load().glr_set_basis(h, Q.data_ptr(), _stream_ptr(stream)), h)


def glr_force_selection(h, J) -> None:
    arr = np.ascontiguousarray(np.asarray(J, dtype=np.int32))
    _check(load().glr_force_selection(h, arr.ctypes.data), h)


def glr_test_expire_wait(h, polls: int, stream=None) -> None:
    """Let one bounded device wait run out on the handle's flags (test aid, see glr.h)."""
    _check(load().glr_test_expire_wait(h, int(polls), _stream_ptr(stream)), h)


def glr_profile_enable(h, enable: bool = True) -> None:
    _check(load().glr_profile_enable(h, 1 if enable else 0), h)


def glr_profile_read(h, reset: bool = False) -> dict:
    p = GlrProfile()
    _check(load().glr_profile_read(h, ctypes.byref(p), 1 if reset else 0), h)
    return {name: {"ms": p.ms[i], "launches": p.launches[i], "count": p.count[i]}
            for i, name in enumerate(PHASE_NAMES)}


def glr_select_noalloc(U: torch.Tensor, Mbar: torch.Tensor, seed: int, t: int, r: int,
                       lambda_out: torch.Tensor, J_out: torch.Tensor, stream=None) -> None:
    """Approx-Top-r selection into caller buffers; the library allocates nothing (see glr.h).
    The library cannot see the buffers' sizes, so they are checked here: U (m' x m') and Mbar
    (m' x n') contiguous fp32 on the GPU, lambda_out at least m' fp32, J_out at least r int32."""
    if Mbar.dim() != 2:
        raise ValueError("Mbar must be a 2-D m' x n' tensor")
    mp, np_ = Mbar.shape
    for name, x in (("U", U), ("Mbar", Mbar)):
        if not (x.is_cuda and x.dtype == torch.float32 and x.is_contiguous()):
            raise ValueError(f"{name} must be a contiguous float32 CUDA tensor")
    if tuple(U.shape) != (mp, mp):
        raise ValueError(f"U must be {mp} x {mp}")
    if not (lambda_out.is_cuda and lambda_out.dtype == torch.float32 and lambda_out.is_contiguous()
            and lambda_out.numel() >= mp):
        raise ValueError(f"lambda_out must be a contiguous float32 CUDA tensor of at least {mp} elements")
    if not (J_out.is_cuda and J_out.dtype == torch.int32 and J_out.is_contiguous() and J_out.numel() >= r):
        raise ValueError(f"J_out must be a contiguous int32 CUDA tensor of at least {r} elements")
    _check(load().glr_select_noalloc(mp, np_, r, U.data_ptr(), Mbar.data_ptr(), seed & (2 ** 64 - 1), t,
                                     lambda_out.data_ptr(), J_out.data_ptr(), _stream_ptr(stream)))


class GreedyLore:
    """One layer matrix's GreedyLore state for N simulated nodes (owns a glr handle).

    GreedyLore(m, n, r, N, **schedule) with the keywords of make_schedule; step(G, X) runs one
    iteration on the N device gradients G (m x n, the schedule's dtype) and updates the device
    weights X (m x n float32) in place.  close() frees the device state.
    """

    def __init__(self, m: int, n: int, r: int, N: int, **schedule):
        self.m, self.n, self.r, self.N = m, n, r, N
        self.mp, self.np_ = min(m, n), max(m, n)
        self.schedule = make_schedule(**schedule)
        self.handle = glr_create(m, n, r, N, self.schedule)

    def step(self, G, X, stream=None):
        glr_step(self.handle, G, X, stream)

    def step_host(self, G_host, X, X_host_out=None, stream=None):
        glr_step_host(self.handle, G_host, X, X_host_out, stream)

    def state_dict(self, stream=None) -> np.ndarray:
        return glr_save(self.handle, stream)

    def load_state_dict(self, state, stream=None):
        glr_load(self.handle, state, stream)

    def refresh(self):
        glr_refresh(self.handle)

    def stats(self):
        return glr_get_stats(self.handle)

    def error(self, i: int) -> torch.Tensor:
        out = torch.empty(self.mp, self.np_, device="cuda", dtype=torch.float32)
        glr_get_error(self.handle, i, out)
        return out

    def selection(self):
        P = torch.empty(self.mp, self.r, device="cuda")
        Rbar = torch.empty(self.r, self.np_, device="cuda")
        lam = torch.empty(self.mp, device="cuda")
        Mbar = torch.empty(self.mp, self.np_, device="cuda")
        J = glr_get_selection(self.handle, self.r, P, Rbar, lam, Mbar)
        return J, P, Rbar, lam, Mbar

    def basis(self) -> torch.Tensor:
        out = torch.empty(self.mp, self.mp, device="cuda")
        glr_get_basis(self.handle, out)
        return out

    def set_basis(self, Q: torch.Tensor):
        glr_set_basis(self.handle, Q.contiguous().float())

    def force_selection(self, J):
        glr_force_selection(self.handle, J)

    def profile(self, enable: bool = True):
        glr_profile_enable(self.handle, enable)

    def profile_read(self, reset: bool = False) -> dict:
        return glr_profile_read(self.handle, reset)

    def close(self):
        if self.handle is not None:
            glr_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
