"""The decode work plan (host logic of decode.cu): every tile of every (sequence, KV
head) pool in exactly one CTA's range, partial slots inside the pair's stride, one
wave of CTAs.  tests/plan_check.cu includes decode.cu and runs make_decode_plan on the
CPU for the workloads' shapes, edge cases and seeded random shapes; no GPU is used.
"""
import os
import shutil
import subprocess

import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)


def test_decode_plan_covers_every_tile_once(tmp_path):
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(nvcc):
        pytest.skip("nvcc not found")
    exe = str(tmp_path / "plan_check")
    cmd = [nvcc, "-std=c++17", "-O1", "--expt-relaxed-constexpr",
           "-gencode", "arch=compute_103a,code=sm_103a",
           "-I", os.path.join(ROOT, "include"),
           "-I", os.path.join(ROOT, "paper_2608_28911_gb300", "csrc"),
           os.path.join(HERE, "plan_check.cu"), "-o", exe]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr[-3000:]
    r = subprocess.run([exe], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stdout[-3000:]
    assert "all plans ok" in r.stdout
