"""The header is plain C, and a C99 program linked against libspo.so runs
the whole path without Python (closed-form checks inside the program)."""

import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CUDA = os.environ.get("CUDA_HOME", "/usr/local/cuda")
CC = shutil.which("gcc") or shutil.which("cc")


def _build(tmp_path):
    from paper_2607_20908_gb300 import build
    lib = build.build()
    exe = str(tmp_path / "abi_demo")
    libdir = os.path.dirname(lib)
    cmd = [CC, "-std=c99", "-Wall", "-Wextra", "-Werror", "-O1",
           os.path.join(ROOT, "tests", "c", "abi_demo.c"), "-I", os.path.join(ROOT, "include"),
           "-I", os.path.join(CUDA, "include"), "-L", libdir, "-lspo",
           "-L", os.path.join(CUDA, "lib64"), "-lcudart", "-lm", f"-Wl,-rpath,{libdir}",
           f"-Wl,-rpath,{os.path.join(CUDA, 'lib64')}", "-o", exe]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stdout + r.stderr
    return exe


@pytest.mark.skipif(CC is None, reason="no C compiler")
def test_header_is_strict_c99(tmp_path):
    src = tmp_path / "h.c"
    src.write_text('#include "spo.h"\nint main(void) { return (int)SPO_OK + (int)SPO_AGG_TOKEN; }\n')
    r = subprocess.run([CC, "-std=c99", "-pedantic", "-Wall", "-Wextra", "-Werror", "-fsyntax-only",
                        "-I", os.path.join(ROOT, "include"), str(src)], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr


@pytest.mark.skipif(CC is None or not os.path.exists(os.path.join(CUDA, "include", "cuda_runtime_api.h")),
                    reason="no C compiler or CUDA runtime headers")
def test_c_program_builds(tmp_path):
    _build(tmp_path)


@pytest.mark.gpu
def test_c_program_runs_the_path(tmp_path):
    exe = _build(tmp_path)
    r = subprocess.run([exe], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "bad=0" in r.stdout
