"""The boundary is a C ABI: a plain C99 program (tests/c/abi_client.c) that
includes every public header compiles warning-free under -pedantic, links
against libshard.so by the headers' names alone, and runs.  It calls only
entry points whose argument checks fail on the host, so no GPU is needed.
The same source also compiles as C++ (the headers' extern "C" guards)."""
import os
import shutil
import subprocess

import pytest

from paper_2608_19147_gb300 import build as libbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "tests", "c", "abi_client.c")
INC = os.path.join(ROOT, "include")


@pytest.fixture(scope="module")
def lib():
    try:
        libbuild.build()
    except RuntimeError as e:  # no nvcc here
        if not os.path.exists(libbuild.LIB):
            pytest.skip(str(e))
    return libbuild.LIB


def _cc(name):
    exe = shutil.which(name)
    if not exe:
        pytest.skip("%s not found" % name)
    return exe


def test_c99_client_compiles_links_and_runs(lib, tmp_path):
    exe = tmp_path / "abi_client"
    libdir = os.path.dirname(lib)
    cmd = [_cc("gcc"), "-std=c99", "-Wall", "-Wextra", "-Werror", "-pedantic", "-I", INC, SRC, "-o", str(exe),
           "-L", libdir, "-lshard", "-Wl,-rpath," + libdir]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    run = subprocess.run([str(exe)], capture_output=True, text=True, timeout=120)
    assert run.returncode == 0 and "abi client ok" in run.stdout, (run.returncode, run.stdout, run.stderr)


def test_headers_compile_as_cxx(tmp_path):
    obj = tmp_path / "abi_client.o"
    cmd = [_cc("g++"), "-x", "c++", "-std=c++17", "-Wall", "-Wextra", "-Werror", "-I", INC, "-c", SRC, "-o", str(obj)]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
