"""The blocked Jacobi's tournament schedule (the host/device index maps of glr_internal.cuh),
compiled for the host with nvcc and checked exhaustively for 4 to 64 blocks: a permutation of
the blocks in every round, every two blocks paired exactly once per sweep, and every block's data
moved to its place of the next round (tests/bjac_schedule_check.cu)."""
import os
import shutil
import subprocess
import tempfile

import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)


def test_bjac_round_robin_schedule():
    nvcc = shutil.which("nvcc") or ("/usr/local/cuda/bin/nvcc" if os.path.exists("/usr/local/cuda/bin/nvcc") else None)
    if nvcc is None:
        pytest.skip("nvcc not found")
    with tempfile.TemporaryDirectory() as d:
        exe = os.path.join(d, "check")
        subprocess.run([nvcc, "-std=c++17", "-O1", "-I", os.path.join(ROOT, "include"),
                        "-I", os.path.join(ROOT, "paper_2507_08784_gb300", "csrc"),
                        os.path.join(HERE, "bjac_schedule_check.cu"), "-o", exe], check=True)
        out = subprocess.run([exe], capture_output=True, text=True, timeout=60)
    assert out.returncode == 0 and out.stdout.strip() == "ok", out.stdout
