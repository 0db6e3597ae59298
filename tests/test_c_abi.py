"""The boundary used from plain C: programs under tests/c are compiled with
gcc as C99 against include/acrl.h and linked to the in-tree library."""

import os
import shutil
import subprocess

import pytest

from paper_2607_24062_gb300 import build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CDIR = os.path.join(ROOT, "tests", "c")
LIBDIR = os.path.dirname(build.LIB)


def _missing(what):
    """A C client that cannot be built: a failure where a GPU is present (the
    C clients are the evidence that the boundary works from plain C), a
    skip on a CPU-only machine."""
    import torch
    if torch.cuda.is_available():
        pytest.fail(f"{what}: the C99 clients must build and run on a GPU machine")
    pytest.skip(what)


def _compile(tmp_path, src, cflags=(), libs=()):
    if shutil.which("gcc") is None:
        _missing("gcc not available")
    if shutil.which("nvcc") is None and not build.up_to_date():
        _missing("no nvcc to build the library")
    build.build()
    exe = str(tmp_path / os.path.splitext(src)[0])
    cmd = ["gcc", "-std=c99", "-Wall", "-Wextra", "-Werror", "-pedantic", f"-I{ROOT}/include", *cflags,
           os.path.join(CDIR, src), "-o", exe, f"-L{LIBDIR}", "-lacrl", f"-Wl,-rpath,{LIBDIR}", *libs, "-lm"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    return exe


def test_c_client_host_calls(tmp_path):
    exe = _compile(tmp_path, "abi_host.c")
    r = subprocess.run([exe], capture_output=True, text=True, timeout=60)
    assert r.returncode == 0 and r.stdout.strip() == "ok", r.stderr


@pytest.mark.gpu
def test_c_client_device_call(tmp_path):
    cuda = os.environ.get("CUDA_HOME", "/usr/local/cuda")
    exe = _compile(tmp_path, "abi_device.c", cflags=("-isystem", f"{cuda}/include"),
                   libs=(f"-L{cuda}/lib64", "-lcudart", f"-Wl,-rpath,{cuda}/lib64"))
    r = subprocess.run([exe], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0 and r.stdout.strip() == "ok", r.stdout + r.stderr


@pytest.mark.gpu
def test_c_client_whole_chain(tmp_path):
    """The whole on-policy pass through the C ABI alone, checked in C."""
    cuda = os.environ.get("CUDA_HOME", "/usr/local/cuda")
    exe = _compile(tmp_path, "abi_chain.c", cflags=("-isystem", f"{cuda}/include"),
                   libs=(f"-L{cuda}/lib64", "-lcudart", f"-Wl,-rpath,{cuda}/lib64"))
    r = subprocess.run([exe], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0 and r.stdout.strip() == "ok", r.stdout + r.stderr


@pytest.mark.gpu
def test_c_client_host_pipeline(tmp_path):
    """The host-buffer pipeline from C, bitwise against the device calls."""
    cuda = os.environ.get("CUDA_HOME", "/usr/local/cuda")
    exe = _compile(tmp_path, "abi_host_pipeline.c", cflags=("-isystem", f"{cuda}/include"),
                   libs=(f"-L{cuda}/lib64", "-lcudart", f"-Wl,-rpath,{cuda}/lib64"))
    r = subprocess.run([exe], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0 and r.stdout.strip() == "ok", r.stdout + r.stderr
