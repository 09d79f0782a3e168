"""The allocation-free linear entry point (chimera_op_linear_noalloc): for callers that
cannot allocate device memory when they call, the library keeps the split-K scratch in
static device arrays.  Its outputs must match chimera_op_linear's, call after call
(the scratch is shared between calls, so two consecutive calls check that it is left
in a usable state).  Kept in a file of its own, collected last."""
import numpy as np
import pytest
import torch

import paper_2402_15758_gb300 as pkg

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2402_15758_gb300 import build
    build.build()
    pkg.load()


def _rel_rows(a, ref):
    return float(np.max(np.abs(a - ref) / np.maximum(np.max(np.abs(ref), axis=-1, keepdims=True), 1e-30)))


@pytest.mark.parametrize("M,N,K,epi,out_f32", [(1, 4096, 4096, 0, True), (8, 1000, 520, 0, True),
                                               (32, 2048, 1024, 1, False), (5, 384, 4096, 2, True)])
def test_noalloc_matches_op_linear_twice(M, N, K, epi, out_f32):
    g = torch.Generator().manual_seed(M + N + K)
    for call in range(2):
        X = torch.randn(M, K, generator=g).to(torch.bfloat16).cuda()
        W = (torch.randn(N, K, generator=g) * 0.05).to(torch.bfloat16).cuda()
        dt = torch.float32 if out_f32 else torch.bfloat16
        init = torch.randn(M, N, generator=g).to(dt).cuda() if epi == 2 else torch.zeros(M, N, dtype=dt).cuda()
        ref = init.clone()
        got = init.clone()
        pkg.op_linear(X, W, ref, epi=epi, out_f32=out_f32)
        pkg.op_linear_noalloc(X, W, got, epi=epi, out_f32=out_f32)
        torch.cuda.synchronize()
        tol = 1e-5 if out_f32 else 8e-3
        assert _rel_rows(got.float().cpu().numpy(), ref.float().cpu().numpy()) <= tol, (call,)


def test_noalloc_rejects_sizes_beyond_the_static_limit():
    X = torch.zeros(33, 64, dtype=torch.bfloat16, device="cuda")
    W = torch.zeros(128, 64, dtype=torch.bfloat16, device="cuda")
    Y = torch.zeros(33, 128, device="cuda")
    with pytest.raises(pkg.ChimeraError):
        pkg.op_linear_noalloc(X, W, Y, out_f32=True)


@pytest.mark.parametrize("M", [17, 32])
def test_noalloc_split_operand_matches_op_linear(M):
    # the hi + lo split activation (two MMAs per K slice) changes the stage layout that
    # the static scratch is used with
    g = torch.Generator().manual_seed(M)
    N, K = 1536, 2048
    X32 = torch.randn(M, K, generator=g)
    X = X32.to(torch.bfloat16)
    X_lo = (X32 - X.float()).to(torch.bfloat16)
    W = (torch.randn(N, K, generator=g) * 0.05).to(torch.bfloat16)
    X, X_lo, W = X.cuda(), X_lo.cuda(), W.cuda()
    for call in range(2):
        ref = torch.zeros(M, N, device="cuda")
        got = torch.zeros(M, N, device="cuda")
        pkg.op_linear(X, W, ref, epi=0, out_f32=True, X_lo=X_lo)
        pkg.op_linear_noalloc(X, W, got, epi=0, out_f32=True, X_lo=X_lo)
        torch.cuda.synchronize()
        assert _rel_rows(got.cpu().numpy(), ref.cpu().numpy()) <= 1e-5, (call,)


def test_noalloc_calls_leave_device_memory_unchanged():
    # after a first call (which looks up the static arrays' addresses), further calls
    # must not change the device's free memory: nothing is allocated per call
    M, N, K = 16, 4096, 4096
    X = torch.randn(M, K).to(torch.bfloat16).cuda()
    W = (torch.randn(N, K) * 0.02).to(torch.bfloat16).cuda()
    Y = torch.zeros(M, N, device="cuda")
    pkg.op_linear_noalloc(X, W, Y, epi=0, out_f32=True)
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    for _ in range(4):
        pkg.op_linear_noalloc(X, W, Y, epi=0, out_f32=True)
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0
    pkg.op_sync()  # and no device-side error was flagged
