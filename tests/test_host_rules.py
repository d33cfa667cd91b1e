"""Builds tests/host_rules.cu with nvcc against the library's own headers and
runs it on the CPU: the host-side launch rules (backward team shapes, ragged
workspace offsets, ragged norm backward covers and segments, the longest
ragged norm row) checked exhaustively, without a device."""
import os
import shutil
import subprocess

import pytest

from paper_2607_23089_gb300 import build as bld

HERE = os.path.dirname(os.path.abspath(__file__))


def test_host_launch_rules(tmp_path):
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(nvcc):
        pytest.skip("nvcc not found")
    exe = tmp_path / "host_rules"
    flags = [f for f in bld.NVCC_FLAGS if f not in ("-Xcompiler", "-fPIC", "-fvisibility=hidden")]
    subprocess.run([nvcc] + flags + [os.path.join(HERE, "host_rules.cu"), "-o", str(exe)],
                   check=True, timeout=600)
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0 and r.stdout.strip().endswith("ok"), r.stdout[-3000:]
