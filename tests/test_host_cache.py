"""Host logic of the launchers' per-device setup cache (pbb::cached_per_device), checked on
the CPU: a small C++ program exercises it from 16 threads, with failing setups and device
indices outside the cached range."""
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2606_02680_gb300", "csrc")
CUDA_INC = os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "include")


def test_cached_per_device(tmp_path):
    cxx = shutil.which("g++")
    if cxx is None or not os.path.exists(os.path.join(CUDA_INC, "cuda.h")):
        pytest.skip("needs g++ and the CUDA headers")
    exe = tmp_path / "host_cache_check"
    src = os.path.join(os.path.dirname(os.path.abspath(__file__)), "host_cache_check.cpp")
    subprocess.run([cxx, "-std=c++17", "-O2", "-pthread", "-I", CSRC, "-I", CUDA_INC, src, "-o", str(exe)],
                   check=True, capture_output=True, text=True)
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert r.returncode == 0, r.stdout + r.stderr
    assert r.stdout.strip() == "ok"
