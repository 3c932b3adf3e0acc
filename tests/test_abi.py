"""Host-side checks of the C ABI that need no GPU: the library builds for sm_103a, loads, and
exports every function declared in include/glr.h; glr_create rejects bad arguments before it
touches the device; the ctypes structs match the C layout."""
import ctypes
import os
import subprocess

import pytest

import __graft_entry__
from paper_2507_08784_gb300 import _lib


@pytest.fixture(scope="module")
def lib():
    __graft_entry__.build()
    return _lib.load()


def test_exports_every_declared_symbol(lib):
    names = _lib.header_symbols()
    assert len(names) >= 12
    missing = [nm for nm in names if not hasattr(lib, nm)]
    assert not missing, missing
    out = subprocess.run(["nm", "-D", "--defined-only", _lib.LIB_PATH], capture_output=True, text=True).stdout
    exported = {line.split()[-1] for line in out.splitlines() if line.strip()}
    assert set(names) <= exported


def test_bindings_cover_every_symbol():
    assert set(_lib.header_symbols()) == set(_lib._SIGNATURES)


def test_struct_layouts(tmp_path):
    """The ctypes mirrors match the C layout of glr.h, field by field (a C program compiled
    against the header prints its sizes and offsets)."""
    import shutil
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    fields = {"glr_schedule": _lib.GlrSchedule, "glr_stats": _lib.GlrStats, "glr_dp_exchange": _lib.GlrDpExchange}
    lines = ['#include <stdio.h>', '#include <stddef.h>', '#include "glr.h"', 'int main(void) {']
    for cname, cls in fields.items():
        lines.append(f'printf("{cname} %zu\\n", sizeof({cname}));')
        for f, _ in cls._fields_:
            lines.append(f'printf("{cname}.{f} %zu\\n", offsetof({cname}, {f}));')
    lines += ['return 0;', '}']
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines) + "\n")
    exe = tmp_path / "layout"
    inc = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include")
    subprocess.run([cc, "-std=c99", "-I", inc, str(src), "-o", str(exe)], check=True)
    got = dict(line.split() for line in subprocess.run([str(exe)], capture_output=True, text=True,
                                                        check=True).stdout.splitlines())
    for cname, cls in fields.items():
        assert int(got[cname]) == ctypes.sizeof(cls), cname
        for f, _ in cls._fields_:
            assert int(got[f"{cname}.{f}"]) == getattr(cls, f).offset, f"{cname}.{f}"


@pytest.mark.parametrize("m,n,r,N,kw,frag", [
    (0, 5, 1, 1, {}, "matrix sizes"),
    (5, 5, 0, 1, {}, "1 <= r"),
    (5, 5, 6, 1, {}, "1 <= r"),
    (5, 5, 2, 0, {}, "N"),
    (5, 5, 2, 65, {}, "N"),
    (5, 5, 2, 1, {"tau": 0}, "tau"),
    (8, 20, 4, 1, {"basis_rank": 3}, "basis_rank"),
    (2000, 3000, 4, 1, {"basis_rank": 0}, "full basis"),
    (8, 20, 4, 1, {"power_iters": 0, "basis_rank": 5}, "power_iters"),
    (8, 20, 4, 1, {"optimizer": "galore_adam", "selection": "fixed", "error_feedback": False}, "Algorithm 5"),
    (8, 20, 4, 1, {"optimizer": "galore_adam", "refresh_mode": "alg4", "error_feedback": False}, "Algorithm 5"),
    (8, 20, 4, 1, {"optimizer": "galore_adam", "refresh_mode": "alg4", "selection": "fixed"}, "Algorithm 5"),
    (8, 20, 4, 1, {"optimizer": "galore_adam", "refresh_mode": "alg4", "selection": "fixed", "error_feedback": False,
                   "compress_start": 1}, "Algorithm 5"),
])
def test_create_rejects_bad_arguments(lib, m, n, r, N, kw, frag):
    import paper_2507_08784_gb300 as glr
    sched = dict(tau=5)
    sched.update(kw)
    s = glr.make_schedule(**sched)
    h = ctypes.c_void_p()
    rc = lib.glr_create(m, n, r, N, ctypes.byref(s), ctypes.byref(h))
    assert rc == _lib.GLR_EINVAL
    assert not h.value
    assert frag in lib.glr_last_error(None).decode()


def test_null_arguments(lib):
    h = ctypes.c_void_p()
    assert lib.glr_create(4, 4, 1, 1, None, ctypes.byref(h)) == _lib.GLR_EINVAL
    assert lib.glr_step(None, None, None, None) == _lib.GLR_EINVAL
    assert lib.glr_destroy(None) == _lib.GLR_OK
    assert lib.glr_refresh(None) == _lib.GLR_EINVAL


def test_build_is_sm103a_only():
    from paper_2507_08784_gb300 import build
    assert build.ARCH == ["-gencode", "arch=compute_103a,code=sm_103a"]
