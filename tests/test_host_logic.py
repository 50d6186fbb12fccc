"""Host-side logic of the library checked on the CPU (no GPU): the Gram tile table that
the persistent Gram kernel and its reduction share, and the lower-triangle tile walk of the
persistent Cholesky update (tests/host/tile_table.cu, compiled with nvcc as a host-only
program)."""
import os
import shutil
import subprocess
import tempfile

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2609_14706_gb300", "csrc")


@pytest.mark.skipif(shutil.which("nvcc") is None, reason="nvcc not on PATH")
def test_gram_tile_table():
    src = os.path.join(ROOT, "tests", "host", "tile_table.cu")
    with tempfile.TemporaryDirectory() as tmp:
        exe = os.path.join(tmp, "tile_table")
        subprocess.run(["nvcc", "-std=c++17", "-O1", "-I", CSRC, src, "-o", exe], check=True,
                       capture_output=True, timeout=300)
        out = subprocess.run([exe], capture_output=True, text=True, timeout=120)
    assert out.returncode == 0, out.stdout + out.stderr
    assert out.stdout.strip() == "ok"
