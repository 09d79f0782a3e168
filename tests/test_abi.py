"""The C-ABI library builds for sm_103a, loads, and exports every symbol the header
declares (no compute calls: runs without a GPU)."""
import ctypes
import os

import pytest

import paper_2402_15758_gb300 as pkg
from paper_2402_15758_gb300 import build as pkg_build


@pytest.fixture(scope="module")
def lib_path():
    return pkg_build.build()


def test_library_exports_every_declared_symbol(lib_path):
    lib = ctypes.CDLL(lib_path)
    declared = pkg.declared_symbols()
    assert "chimera_init" in declared and "chimera_step" in declared
    missing = [s for s in declared if not hasattr(lib, s)]
    assert not missing, missing


def test_binding_signatures_cover_header():
    assert set(pkg.declared_symbols()) == set(pkg._SIGS)


def test_init_rejects_bad_config_without_touching_the_gpu(lib_path):
    lib = pkg.load()
    c = pkg.Config()  # all zero: invalid shapes -> EINVAL before any CUDA call
    h = ctypes.c_void_p()
    assert lib.chimera_init(ctypes.byref(c), None, None, ctypes.byref(h)) == -1
    assert lib.chimera_init(None, None, None, None) == -1
    assert not h.value
