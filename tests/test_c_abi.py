"""The C ABI from plain C: tests/c_abi_check.c includes only include/rl_loss.h and links the
shared library (and, for the GPU part, the CUDA runtime), with no Python or torch in between.
The host part runs anywhere; the GPU part checks a closed-form loss and gradient."""

import os
import shutil
import subprocess

import pytest

from paper_2608_16798_gb300 import build as B

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "tests", "c_abi_check.c")


def _compile(tmp_path):
    B.build()
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    cuda_lib = os.path.join(os.path.dirname(os.path.dirname(os.path.realpath(B.nvcc()))), "lib64")
    exe = str(tmp_path / "c_abi_check")
    pkg = os.path.dirname(B.LIB)
    cmd = [cc, "-std=c99", "-O1", "-Wall", "-I", os.path.join(ROOT, "include"), SRC, "-o", exe, "-L", pkg, "-lrl_loss",
           "-L", cuda_lib, "-lcudart", f"-Wl,-rpath,{pkg}", f"-Wl,-rpath,{cuda_lib}", "-lm"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stdout + r.stderr
    return exe


def test_c_caller_host_checks(tmp_path):
    exe = _compile(tmp_path)
    r = subprocess.run([exe, "host"], capture_output=True, text=True, timeout=60)
    assert r.returncode == 0, r.stdout + r.stderr


@pytest.mark.gpu
def test_c_caller_closed_form_on_gpu(tmp_path):
    exe = _compile(tmp_path)
    r = subprocess.run([exe, "gpu"], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "c_abi_check ok" in r.stdout
