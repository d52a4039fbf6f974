"""Host logic of the kernels' tile geometry (tiles.cuh, compiled as plain C++
with g++): the per-item range of tiles that skip the element-wise mask agrees
with the per-tile predicate, no skipped tile holds an invisible (row, key)
pair, the split-K units cover each dense M-tile once, and every lane maps to
its query head's KV head with each (batch, head, row) held once, over many
shapes, all three modes, the dense tail and the GQA head packings; and the
two-CTA kernel's clusters always pair two heads of one row tile."""
import os
import shutil
import subprocess
import tempfile

import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(os.path.dirname(HERE), "paper_2505_11254_gb300", "csrc")


@pytest.mark.skipif(shutil.which("g++") is None, reason="needs g++")
def test_unmasked_tile_ranges():
    with tempfile.TemporaryDirectory() as d:
        exe = os.path.join(d, "tile_geometry_check")
        subprocess.run(["g++", "-O2", "-std=c++17", "-I", CSRC, os.path.join(HERE, "tile_geometry_check.cpp"),
                        "-o", exe], check=True)
        r = subprocess.run([exe], capture_output=True, text=True, timeout=600)
        assert r.returncode == 0, r.stdout + r.stderr
