"""The C ABI from C: include/dard.h passes a strict C99 compile by itself, the C client
(tests/c_client/dard_c_client.c) builds and links against libdard.so with a C compiler
(CPU), and on the GPU it passes its closed-form checks of both entry points."""
import glob
import os
import shutil
import subprocess

import pytest

from paper_2608_26574_gb300 import build as BUILD

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
INCLUDE = os.path.join(ROOT, "include")
SRC = os.path.join(ROOT, "tests", "c_client", "dard_c_client.c")


def _cc():
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    return cc


def _cuda():
    """(include dir, directory holding libcudart.so) of the CUDA toolkit nvcc belongs to."""
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    home = os.path.dirname(os.path.dirname(os.path.realpath(nvcc)))
    libs = [os.path.join(home, "lib64")] + glob.glob(os.path.join(home, "targets", "*", "lib"))
    for d in libs:
        if os.path.exists(os.path.join(d, "libcudart.so")):
            return os.path.join(home, "include"), d
    pytest.skip("libcudart.so not found")


def _build_client(tmp_path):
    lib = BUILD.build()
    libdir = os.path.dirname(lib)
    cuda_inc, cuda_lib = _cuda()
    exe = str(tmp_path / "dard_c_client")
    cmd = [_cc(), "-std=c11", "-O2", "-Wall", "-Wextra", "-Werror", "-pedantic", SRC,
           "-I", INCLUDE, "-I", cuda_inc, "-L", libdir, "-ldard", "-L", cuda_lib, "-lcudart",
           f"-Wl,-rpath,{libdir}", f"-Wl,-rpath,{cuda_lib}", "-lm", "-o", exe]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    return exe


def test_header_is_strict_c99():
    r = subprocess.run([_cc(), "-fsyntax-only", "-x", "c", "-std=c99", "-Wall", "-Wextra",
                        "-Werror", "-pedantic", os.path.join(INCLUDE, "dard.h")],
                       capture_output=True, text=True)
    assert r.returncode == 0, r.stderr


def test_c_client_builds_and_links(tmp_path):
    assert os.path.exists(_build_client(tmp_path))


@pytest.mark.gpu
def test_c_client_runs(tmp_path):
    exe = _build_client(tmp_path)
    r = subprocess.run([exe], capture_output=True, text=True, timeout=120)
    print(r.stdout, r.stderr)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "all checks passed" in r.stdout
