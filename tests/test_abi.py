"""The C-ABI library loads on a machine without a GPU and exports every
symbol the headers in include/ declare (no compute call is made)."""
import ctypes
import os
import re

import pytest

import paper_2608_19147_gb300 as pkg
from paper_2608_19147_gb300 import build as libbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    names = set()
    for h in ("shard.h", "shard_debug.h", "head.h"):
        src = open(os.path.join(ROOT, "include", h)).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        for m in re.finditer(r"^\s*(?:const\s+)?\w+\**\s+\**(\w+)\s*\(", src, flags=re.M):
            names.add(m.group(1))
    return names


@pytest.fixture(scope="module")
def lib():
    try:
        libbuild.build()
    except RuntimeError as e:  # no nvcc here
        if not os.path.exists(libbuild.LIB):
            pytest.skip(str(e))
    return ctypes.CDLL(libbuild.LIB)


def test_headers_declare_the_binding_exports():
    assert _declared() == set(pkg.EXPORTS)


def test_library_exports_every_declared_symbol(lib):
    for name in sorted(_declared()):
        assert hasattr(lib, name), name


def test_no_device_call_needed_for_errors(lib):
    pkg.load_library()
    assert pkg.shard_last_error() == ""
    # argument validation happens on the host before any CUDA call
    lib.shard_destroy.argtypes = [ctypes.c_void_p]
    assert lib.shard_destroy(None) == pkg.SHARD_EINVAL
    assert "null" in pkg.shard_last_error()
    lib.head_destroy.argtypes = [ctypes.c_void_p]
    assert lib.head_destroy(None) == pkg.SHARD_EINVAL
    assert "null" in pkg.shard_last_error()
