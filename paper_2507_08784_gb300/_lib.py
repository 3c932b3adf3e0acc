"""ctypes declarations for libglr.so (the C ABI declared in include/glr.h).

Loading never falls back to anything: if the library is missing or cannot be
loaded, ``load()`` raises and no GreedyLore call is possible.
"""
from __future__ import annotations

import ctypes
import os
import re

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "lib", "libglr.so")
HEADER = os.path.join(os.path.dirname(PKG), "include", "glr.h")

GLR_OK, GLR_EINVAL, GLR_ENOMEM, GLR_ECUDA, GLR_ENUMERIC, GLR_ENONFINITE, GLR_ETIMEOUT = 0, -1, -2, -3, -4, -5, -6
GLR_ALG3, GLR_ALG4 = 0, 1
GLR_MSGD, GLR_ADAM, GLR_AMSGRAD, GLR_ADAMW, GLR_GALORE_ADAM = 0, 1, 2, 3, 4
GLR_F32, GLR_BF16 = 0, 1
GLR_MAX_NODES = 64

_c_void_pp = ctypes.POINTER(ctypes.c_void_p)
_c_float_p = ctypes.c_void_p     # device/host float buffers are passed as raw addresses


class GlrSchedule(ctypes.Structure):
    _fields_ = [
        ("tau", ctypes.c_int32),
        ("refresh_mode", ctypes.c_int32),
        ("optimizer", ctypes.c_int32),
        ("lr", ctypes.c_float),
        ("beta1", ctypes.c_float),
        ("beta2", ctypes.c_float),
        ("eps", ctypes.c_float),
        ("seed", ctypes.c_uint64),
        ("basis_rank", ctypes.c_int32),
        ("power_iters", ctypes.c_int32),
        ("grad_dtype", ctypes.c_int32),
        ("compress_start", ctypes.c_int32),
        ("no_error_feedback", ctypes.c_int32),
        ("selection", ctypes.c_int32),
        ("weight_decay", ctypes.c_float),
    ]


class GlrStats(ctypes.Structure):
    _fields_ = [
        ("t", ctypes.c_int64),
        ("refreshes", ctypes.c_int64),
        ("comm_floats_total", ctypes.c_int64),
        ("state_bytes", ctypes.c_int64),
        ("m_prime", ctypes.c_int32),
        ("n_prime", ctypes.c_int32),
        ("r", ctypes.c_int32),
        ("k", ctypes.c_int32),
        ("transposed", ctypes.c_int32),
        ("last_refresh_sweeps", ctypes.c_int32),
        ("launches", ctypes.c_int64),
        ("path", ctypes.c_int32),
        ("nonfinite", ctypes.c_int32),
        ("numeric_failures", ctypes.c_int32),
        ("reserved", ctypes.c_int32),
    ]


class GlrDpExchange(ctypes.Structure):
    """glr_dp_exchange: the device buffers a data-parallel phase exposes for averaging."""
    _fields_ = [
        ("count", ctypes.c_int32),
        ("pad_", ctypes.c_int32),
        ("ptr", ctypes.c_void_p * 2),
        ("floats", ctypes.c_int64 * 2),
    ]


GLR_PHASES = 7
PHASE_NAMES = ["prev_project", "compose", "lambda", "select", "project", "update", "refresh"]


class GlrProfile(ctypes.Structure):
    _fields_ = [
        ("ms", ctypes.c_double * GLR_PHASES),
        ("launches", ctypes.c_int64 * GLR_PHASES),
        ("count", ctypes.c_int64 * GLR_PHASES),
    ]


_SIGNATURES = {
    "glr_create": (ctypes.c_int, [ctypes.c_int64, ctypes.c_int64, ctypes.c_int32, ctypes.c_int32,
                                  ctypes.POINTER(GlrSchedule), ctypes.POINTER(ctypes.c_void_p)]),
    "glr_destroy": (ctypes.c_int, [ctypes.c_void_p]),
    "glr_step": (ctypes.c_int, [ctypes.c_void_p, _c_void_pp, ctypes.c_void_p, ctypes.c_void_p]),
    "glr_step_group": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_int32, ctypes.c_void_p, ctypes.c_void_p,
                                      ctypes.c_void_p]),
    "glr_step_host": (ctypes.c_int, [ctypes.c_void_p, _c_void_pp, ctypes.c_void_p, ctypes.c_void_p,
                                     ctypes.c_void_p]),
    "glr_step_group_host": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_int32, ctypes.c_void_p, ctypes.c_void_p,
                                           ctypes.c_void_p, ctypes.c_void_p]),
    "glr_state_size": (ctypes.c_int, [ctypes.c_void_p, ctypes.POINTER(ctypes.c_int64)]),
    "glr_save": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p]),
    "glr_load": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p]),
    "glr_refresh": (ctypes.c_int, [ctypes.c_void_p]),
    "glr_get_stats": (ctypes.c_int, [ctypes.c_void_p, ctypes.POINTER(GlrStats)]),
    "glr_last_error": (ctypes.c_char_p, [ctypes.c_void_p]),
    "glr_get_error": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_int32, ctypes.c_void_p, ctypes.c_void_p]),
    "glr_get_selection": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                                         ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p]),
    "glr_get_basis": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p]),
    "glr_set_basis": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p]),
    "glr_force_selection": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p]),
    "glr_test_expire_wait": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_int32, ctypes.c_void_p]),
    "glr_profile_enable": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_int32]),
    "glr_profile_read": (ctypes.c_int, [ctypes.c_void_p, ctypes.POINTER(GlrProfile), ctypes.c_int32]),
    "glr_dp_begin": (ctypes.c_int, [ctypes.c_void_p, _c_void_pp, ctypes.c_void_p, ctypes.POINTER(GlrDpExchange)]),
    "glr_dp_select": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p, ctypes.POINTER(GlrDpExchange)]),
    "glr_dp_finish": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p]),
    "glr_select_noalloc": (ctypes.c_int, [ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_void_p,
                                          ctypes.c_void_p, ctypes.c_uint64, ctypes.c_int64, ctypes.c_void_p,
                                          ctypes.c_void_p, ctypes.c_void_p]),
}

_lib = None


def header_symbols(path: str = HEADER):
    """Names of the functions declared in glr.h."""
    with open(path) as f:
        text = f.read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(glr_[a-z_0-9]+)\s*\(", text)))


def load(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load libglr.so (once) and declare the signatures.  Raises if it is missing."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise ImportError(f"libglr.so not found at {path}: build it with "
                          f"`python -c 'import __graft_entry__ as g; g.build()'` (no CPU fallback exists)")
    try:  # the CUDA runtime of the running PyTorch satisfies libglr's libcudart dependency
        import torch  # noqa: F401
    except Exception:
        pass
    lib = ctypes.CDLL(path)
    for name, (res, args) in _SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib
