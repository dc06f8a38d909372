"""The C ABI from plain C: tests/c_abi_check.c is compiled with gcc against
include/vqc.h and libvqc.so and run.  Without a GPU it checks compilation,
plan statistics, export and the documented error codes; the GPU build also
evaluates the circuit (E against its closed form, device and host buffers)."""
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = os.path.join(ROOT, "paper_2607_11985_gb300")
CUDA = "/usr/local/cuda"


@pytest.fixture(scope="module")
def lib():
    from paper_2607_11985_gb300 import build
    return build.build()


def build_and_run(gpu):
    cc = shutil.which("gcc")
    if cc is None:
        pytest.skip("no gcc")
    out_dir = os.path.join(PKG, "_build")
    os.makedirs(out_dir, exist_ok=True)
    exe = os.path.join(out_dir, "c_abi_check_gpu" if gpu else "c_abi_check")
    cmd = [cc, "-std=c99", "-O1", "-Wall", "-I" + os.path.join(ROOT, "include"),
           os.path.join(ROOT, "tests", "c_abi_check.c"), "-o", exe, "-L" + PKG, "-lvqc",
           "-Wl,-rpath," + PKG, "-lm"]
    if gpu:
        cmd[1:1] = ["-DVQC_CHECK_GPU", "-I" + os.path.join(CUDA, "include")]
        cmd += ["-L" + os.path.join(CUDA, "lib64"), "-lcudart", "-Wl,-rpath," + os.path.join(CUDA, "lib64")]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "warning" not in r.stderr, r.stderr
    r = subprocess.run([exe], capture_output=True, text=True, timeout=120)
    return r


def test_c_abi_host(lib):
    r = build_and_run(gpu=False)
    assert r.returncode == 0 and r.stdout.strip().endswith("ok"), r.stdout + r.stderr


@pytest.mark.gpu
def test_c_abi_gpu(lib):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    r = build_and_run(gpu=True)
    assert r.returncode == 0 and "gpu ok" in r.stdout and r.stdout.strip().endswith("ok"), \
        r.stdout + r.stderr
