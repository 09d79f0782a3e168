"""Kernel-level parity through the C ABI: the tcgen05 / fp32 linear and the paged
tree attention against the fp64 oracle's definitions, at ragged sizes."""
import numpy as np
import pytest
import torch

import paper_2402_15758_gb300 as pkg
from oracle import chimera_oracle as co

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2402_15758_gb300 import build
    build.build()
    pkg.load()


def _rel_rows(a, ref):
    return float(np.max(np.abs(a - ref) / np.maximum(np.max(np.abs(ref), axis=-1, keepdims=True), 1e-30)))


LINEAR_SHAPES = [(1, 128, 64), (5, 300, 72), (16, 256, 512), (17, 1000, 520), (64, 1536, 1024),
                 (100, 384, 1024), (256, 512, 2048), (300, 256, 256), (64, 4096, 4096), (8, 32000, 512),
                 (1, 4096, 12288)]


@pytest.mark.parametrize("M,N,K", LINEAR_SHAPES)
def test_linear_bf16_fp32_out(M, N, K):
    g = torch.Generator().manual_seed(M * 7 + N + K)
    X = torch.randn(M, K, generator=g).to(torch.bfloat16)
    W = (torch.randn(N, K, generator=g) * 0.05).to(torch.bfloat16)
    Y = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
    pkg.op_linear(X.cuda(), W.cuda(), Y, epi=0, out_f32=True)
    torch.cuda.synchronize()
    ref = X.double().numpy() @ W.double().numpy().T
    assert _rel_rows(Y.cpu().numpy(), ref) <= 1e-4


@pytest.mark.parametrize("M,N,K", [(3, 640, 192), (64, 1408, 512), (33, 256, 1408)])
def test_linear_bf16_epilogues(M, N, K):
    g = torch.Generator().manual_seed(99 + M)
    X = torch.randn(M, K, generator=g).to(torch.bfloat16)
    W = (torch.randn(N, K, generator=g) * 0.05).to(torch.bfloat16)
    ref = X.double().numpy() @ W.double().numpy().T
    # bf16 store: one rounding of the fp32 accumulator
    Y = torch.zeros(M, N, dtype=torch.bfloat16, device="cuda")
    pkg.op_linear(X.cuda(), W.cuda(), Y, epi=0)
    assert _rel_rows(Y.float().cpu().numpy(), ref) <= 8e-3
    # SiLU
    pkg.op_linear(X.cuda(), W.cuda(), Y, epi=1)
    assert _rel_rows(Y.float().cpu().numpy(), co.silu(ref)) <= 8e-3
    # residual add into fp32
    R0 = torch.randn(M, N, generator=g)
    R = R0.clone().cuda()
    pkg.op_linear(X.cuda(), W.cuda(), R, epi=2)
    torch.cuda.synchronize()
    assert _rel_rows(R.cpu().numpy(), R0.double().numpy() + ref) <= 1e-5


@pytest.mark.parametrize("M,N,K", [(1, 256, 512), (64, 1536, 1024), (100, 384, 4096)])
def test_linear_bf16_split_operand(M, N, K):
    # X = hi + lo (two bf16 halves): W (hi + lo) reproduces the fp32 activation
    g = torch.Generator().manual_seed(3 * M + K)
    X32 = torch.randn(M, K, generator=g)
    hi = X32.to(torch.bfloat16)
    lo = (X32 - hi.float()).to(torch.bfloat16)
    W = (torch.randn(N, K, generator=g) * 0.05).to(torch.bfloat16)
    Y = torch.zeros(M, N, dtype=torch.float32, device="cuda")
    pkg.op_linear(hi.cuda(), W.cuda(), Y, epi=0, out_f32=True, X_lo=lo.cuda())
    torch.cuda.synchronize()
    ref = X32.double().numpy() @ W.double().numpy().T
    assert _rel_rows(Y.cpu().numpy(), ref) <= 2e-5
    # without the lo half the error is the bf16 rounding of X
    pkg.op_linear(hi.cuda(), W.cuda(), Y, epi=0, out_f32=True)
    torch.cuda.synchronize()
    assert _rel_rows(Y.cpu().numpy(), ref) > 1e-4


def test_linear_deterministic():
    g = torch.Generator().manual_seed(5)
    X = torch.randn(64, 4096, generator=g).to(torch.bfloat16).cuda()
    W = (torch.randn(4096, 4096, generator=g) * 0.02).to(torch.bfloat16).cuda()
    a = torch.zeros(64, 4096, device="cuda")
    b = torch.zeros(64, 4096, device="cuda")
    pkg.op_linear(X, W, a, out_f32=True)
    pkg.op_linear(X, W, b, out_f32=True)
    torch.cuda.synchronize()
    assert torch.equal(a, b)


@pytest.mark.parametrize("M,N,K", [(1, 64, 8), (16, 1024, 768), (64, 688, 256)])
def test_linear_fp32(M, N, K):
    g = torch.Generator().manual_seed(N)
    X = torch.randn(M, K, generator=g)
    W = torch.randn(N, K, generator=g) * 0.05
    Y = torch.zeros(M, N, device="cuda")
    pkg.op_linear(X.cuda(), W.cuda(), Y, epi=0)
    torch.cuda.synchronize()
    assert _rel_rows(Y.cpu().numpy(), X.double().numpy() @ W.double().numpy().T) <= 1e-5


def _random_tree_anc(n, rng):
    parent = [-1] + [int(rng.integers(0, j)) for j in range(1, n)]
    anc = []
    for i in range(n):
        m, j = 0, i
        while j >= 0:
            m |= 1 << j
            j = parent[j]
        anc.append(m)
    return anc


ATT_CASES = [
    # B, H, hd, n_ctx per seq, n_local, nq, q_local0, splits
    (1, 4, 64, [77], 16, 16, 0, 1),
    (1, 4, 64, [77], 16, 16, 0, 5),
    (2, 3, 128, [0, 300], 64, 64, 0, 7),
    (3, 2, 128, [16, 1, 129], 5, 1, 4, 3),     # draft-style: one query, local rows 0..4
    (1, 2, 128, [1000], 64, 64, 0, 8),
    (2, 3, 128, [700, 3], 64, 64, 0, 4),     # a split whose key range is empty for b=1
]


@pytest.mark.parametrize("dtype", ["fp32", "bf16", "bf16_split"])
@pytest.mark.parametrize("case", range(len(ATT_CASES)))
def test_attention_tree_masked_paged(dtype, case):
    B, H, hd, nctx, n_local, nq, q0, splits = ATT_CASES[case]
    rng = np.random.default_rng(case)
    max_pages = (max(nctx) + n_local + 15) // 16 + 1
    n_blocks = B * max_pages + 3
    perm = rng.permutation(n_blocks)[: B * max_pages].reshape(B, max_pages).astype(np.int32)
    assert perm.max() < n_blocks
    kv32 = torch.randn(n_blocks, H, 2, 16, hd, generator=torch.Generator().manual_seed(case))
    if dtype == "fp32":
        pool, Kref = kv32, kv32.double()
        odt = torch.float32
    elif dtype == "bf16":
        pool = kv32.to(torch.bfloat16)
        Kref = pool.double()
        odt = torch.bfloat16
    else:  # K_hi, K_lo, V_hi, V_lo planes; the reference uses the fp32 values
        hi = kv32.to(torch.bfloat16)
        lo = (kv32 - hi.float()).to(torch.bfloat16)
        pool = torch.stack([hi[:, :, 0], lo[:, :, 0], hi[:, :, 1], lo[:, :, 1]], dim=2).contiguous()
        Kref = kv32.double()
        odt = torch.bfloat16
    q = torch.randn(B * nq, H * hd, generator=torch.Generator().manual_seed(100 + case))
    anc = _random_tree_anc(n_local, rng) if q0 == 0 else [(1 << (i + 1)) - 1 for i in range(n_local)]
    out = torch.zeros(B * nq, H * hd, dtype=odt, device="cuda")
    out_lo = torch.zeros_like(out) if odt == torch.bfloat16 else None
    anc_t = torch.tensor(np.array(anc, dtype=np.uint64).view(np.int64), device="cuda")
    pkg.op_attention(q.cuda(), pool.cuda(), torch.tensor(perm, device="cuda"),
                     torch.tensor(nctx, dtype=torch.int32, device="cuda"), anc_t, out, nq=nq, q_local0=q0,
                     n_local=n_local, q_rows=nq, n_heads=H, head_dim=hd, splits=splits, out_lo=out_lo)
    torch.cuda.synchronize()
    got = out.float().cpu().numpy().reshape(B, nq, H, hd)
    if out_lo is not None:
        got = got + out_lo.float().cpu().numpy().reshape(B, nq, H, hd)
    P = Kref.numpy()
    Q = q.double().numpy().reshape(B, nq, H, hd)

    def kv(b, slot):
        blk = perm[b, slot // 16]
        return P[blk, :, 0, slot % 16], P[blk, :, 1, slot % 16]

    # fp32 path: fp32 arithmetic; tensor-core path (head_dim 128, bf16 model): bf16
    # split products of the fp32 query / probabilities (and of the split K/V planes),
    # which drop the lo*lo terms (~2^-16 relative)
    tol = 1e-5 if (dtype == "fp32" or hd != 128) else 5e-5
    for b in range(B):
        for i in range(nq):
            m = anc[q0 + i]
            slots = list(range(nctx[b])) + [nctx[b] + j for j in range(n_local) if (m >> j) & 1]
            Ks = np.array([kv(b, s)[0] for s in slots])
            Vs = np.array([kv(b, s)[1] for s in slots])
            ref = co.attend(Q[b, i], Ks, Vs)
            err = np.max(np.abs(got[b, i] - ref)) / np.max(np.abs(ref))
            assert err <= tol, (b, i, err)


@pytest.mark.parametrize("jump", [40.0, 150.0])
@pytest.mark.parametrize("splits", [1, 2])
def test_attention_rescale_after_one_sided_tile(jump, splits):
    """Online softmax with a far move of the running maximum. Every query row sees the 20
    context keys, local row 0 and itself, so row 50's first tile has visible keys in its
    first key half only; its own key (second tile) scores `jump` nats above zero, which
    moves the maximum by far more than the lazy-rescale threshold (the correction is
    about 2^-53 at 40 nats and underflows to 0 at 150). All 128 output columns of the
    row must then be rescaled, whichever key half saw keys before."""
    import math
    H, hd, nctx, n_local, nq = 2, 128, 20, 64, 64
    max_pages = (nctx + n_local + 15) // 16 + 1
    perm = np.arange(max_pages, dtype=np.int32).reshape(1, max_pages)
    kv32 = torch.randn(max_pages, H, 2, 16, hd, generator=torch.Generator().manual_seed(7))
    q = torch.randn(nq, H * hd, generator=torch.Generator().manual_seed(8))
    anc = [1 | (1 << i) for i in range(n_local)]
    r, slot = 50, nctx + 50
    for h in range(H):
        qv = q[r, h * hd:(h + 1) * hd]
        kv32[slot // 16, h, 0, slot % 16] = qv * (jump * math.sqrt(hd) / float(qv @ qv))
    hi = kv32.to(torch.bfloat16)
    lo = (kv32 - hi.float()).to(torch.bfloat16)
    pool = torch.stack([hi[:, :, 0], lo[:, :, 0], hi[:, :, 1], lo[:, :, 1]], dim=2).contiguous()
    out = torch.zeros(nq, H * hd, dtype=torch.bfloat16, device="cuda")
    out_lo = torch.zeros_like(out)
    anc_t = torch.tensor(np.array(anc, dtype=np.uint64).view(np.int64), device="cuda")
    pkg.op_attention(q.cuda(), pool.cuda(), torch.tensor(perm, device="cuda"),
                     torch.tensor([nctx], dtype=torch.int32, device="cuda"), anc_t, out, nq=nq, q_local0=0,
                     n_local=n_local, q_rows=nq, n_heads=H, head_dim=hd, splits=splits, out_lo=out_lo)
    torch.cuda.synchronize()
    got = (out.float() + out_lo.float()).cpu().numpy().reshape(nq, H, hd)
    P = kv32.double().numpy()
    Q = q.double().numpy().reshape(nq, H, hd)
    for i in range(nq):
        slots = list(range(nctx)) + [nctx + j for j in range(n_local) if (anc[i] >> j) & 1]
        Ks = np.array([P[s // 16, :, 0, s % 16] for s in slots])
        Vs = np.array([P[s // 16, :, 1, s % 16] for s in slots])
        ref = co.attend(Q[i], Ks, Vs)
        err = np.max(np.abs(got[i] - ref)) / np.max(np.abs(ref))
        assert err <= 5e-5, (i, err)
