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


def test_no_restrict_pointer_in_dependent_launch_kernels():
    """Every kernel is launched with programmatic dependent launch and reads its inputs
    only after griddepcontrol.wait.  A `__restrict__` parameter would let the compiler
    treat its loads as invariant and schedule them ahead of that wait (an fp32 prefill
    read a stale residual this way), so no kernel source may declare one."""
    csrc = os.path.join(os.path.dirname(pkg.__file__), "csrc")
    offenders = []
    for name in sorted(os.listdir(csrc)):
        if name.endswith((".cu", ".cuh", ".h")):
            with open(os.path.join(csrc, name)) as f:
                for i, line in enumerate(f, 1):
                    code = line.split("//")[0]
                    if "__restrict__" in code:
                        offenders.append(f"{name}:{i}")
    assert not offenders, offenders


def test_prewait_attention_follows_a_tensor_core_linear():
    """The tensor-core tree attention with fused RoPE (its `qkv` argument set) reads
    n_ctx, the page table and committed KV rows before its dependency wait.  That is
    only safe when the launch directly before it is a tensor-core linear or chain (both
    let their dependents launch only after their own wait).  Every such call site in
    the runtime must therefore have one of them as its previous launch."""
    import re
    src = open(os.path.join(os.path.dirname(pkg.__file__), "csrc", "runtime.cu")).read()
    lines = src.split("\n")
    launch = re.compile(r"\b(RUN|CK)\(")
    sites = 0
    for i, line in enumerate(lines):
        if "RUN(run_attention(" not in line and "CK(run_attention(" not in line:
            continue
        stmt = line
        j = i
        while not stmt.rstrip().endswith(");"):
            j += 1
            stmt += lines[j]
        if "ctx->qkv" not in stmt:
            continue
        sites += 1
        k = i - 1
        while k >= 0 and not launch.search(lines[k]):
            k -= 1
        assert k >= 0 and ("run_lin(" in lines[k] or "run_chain(" in lines[k]), \
            f"runtime.cu:{i + 1}: previous launch is {lines[k].strip()!r}"
    assert sites >= 2  # the verify layers and the draft block
