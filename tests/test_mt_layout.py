"""The batched skinny projections' shared-memory plan, checked on the host.

tests/mt_layout_check.cpp includes the layout header the kernel and its
launcher use (csrc/wf_skinny_mt_layout.h) and walks every (units, K split,
ring depth) plan the launcher may choose, at every pass size up to 144 token
rows, for the Whisper-large, Whisper-tiny and toy projection shapes: each
region the kernel addresses lies inside the launch's dynamic shared memory,
the regions do not overlap and the copies' alignments hold."""
import os
import shutil
import subprocess

import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(os.path.dirname(HERE), "paper_2609_32869_gb300", "csrc")


def test_every_plan_fits_its_shared_memory(tmp_path):
    cxx = shutil.which("g++") or shutil.which("c++")
    if not cxx:
        pytest.skip("no host C++ compiler")
    exe = str(tmp_path / "mt_layout_check")
    subprocess.run([cxx, "-std=c++17", "-O1", "-I", CSRC, os.path.join(HERE, "mt_layout_check.cpp"), "-o", exe],
                   check=True, capture_output=True, text=True)
    r = subprocess.run([exe], capture_output=True, text=True)
    assert r.returncode == 0, r.stdout
    assert r.stdout.startswith("0 violations"), r.stdout
