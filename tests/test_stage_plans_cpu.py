"""The weight-stream stage planner (plan_stages / stage_desc, shared by the
host and the kernels) checked on the host: tests/plan_check.cu, compiled with
nvcc against the kernel header, walks every bulk copy of every phase of every
workload (float32, 8-bit and 4-bit rows; several SM counts; the standalone
GEMV with its K split) and checks exact coverage, bounds, the 16-byte rules of
bulk copies, whole row pairs and the deferred-partial scratch."""
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_stage_plans_cover_each_matrix_once_with_aligned_copies():
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(nvcc):
        pytest.skip("nvcc not found")
    out_dir = os.path.join(ROOT, "tests", "_build")
    os.makedirs(out_dir, exist_ok=True)
    exe = os.path.join(out_dir, "plan_check")
    subprocess.run([nvcc, "-O2", "-std=c++17", "-gencode", "arch=compute_103a,code=sm_103a",
                    "-o", exe, os.path.join(ROOT, "tests", "plan_check.cu")],
                   check=True, capture_output=True)
    r = subprocess.run([exe], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0 and r.stdout.startswith("ok"), r.stdout[-2000:]
