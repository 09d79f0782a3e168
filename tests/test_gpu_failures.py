"""Failure paths of the C ABI, none of which faults the GPU.

Host-side refusals: a step before prefill (ESTATE), out-of-range token ids in a prompt,
an override or a root (EINVAL), a prompt or a step beyond max_seq_len (ECAPACITY), each
leaving the context usable.  Device-side: the tensor-core linear's bounded waits given
a limit of a few ns give up, the kernel leaves cleanly (copies and MMAs drained, tensor
memory freed) and chimera_op_sync reports ETIMEDOUT; the next call computes correctly.
"""
import numpy as np
import pytest
import torch

import paper_2402_15758_gb300 as pkg
import synth

pytestmark = pytest.mark.gpu

EINVAL, ECAPACITY, ETIMEDOUT, ESTATE = -1, -3, -5, -6


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2402_15758_gb300 import build
    build.build()
    pkg.load()


@pytest.fixture(scope="module")
def tiny():
    cfg = synth.get_config("tiny")
    w = {k: v.cuda() for k, v in synth.make_weights(cfg).items()}
    return cfg, w, synth.make_prompts(cfg)[0]


def _status(fn, *a):
    with pytest.raises(pkg.ChimeraError) as e:
        fn(*a)
    return e.value.status


def test_step_before_prefill_is_estate(tiny):
    cfg, w, prompt = tiny
    ctx = pkg.Chimera(cfg, w, max_batch=1, max_seq_len=256)
    ctx.batch = 1
    assert _status(ctx.step) == ESTATE
    assert _status(ctx.override_tree, [[0] * cfg["tree_nodes"]]) == ESTATE
    ctx.prefill([prompt])  # still usable
    assert len(ctx.step()[0]) >= 1
    ctx.close()


def test_bad_token_ids_are_einval(tiny):
    cfg, w, prompt = tiny
    V = cfg["vocab"]
    ctx = pkg.Chimera(cfg, w, max_batch=1, max_seq_len=256)
    assert _status(ctx.prefill, [prompt[:10] + [V] + prompt[11:]]) == EINVAL
    assert _status(ctx.prefill, [[-1] + prompt[1:]]) == EINVAL
    ctx.prefill([prompt])
    bad = [0] + [1] * (cfg["tree_nodes"] - 2) + [V + 5]
    assert _status(ctx.override_tree, [bad]) == EINVAL
    assert _status(ctx.set_root, [V]) == EINVAL
    n0 = int(ctx.read("n")[0])
    e = ctx.step()[0]
    assert int(ctx.read("n")[0]) == n0 + len(e)
    ctx.close()


def test_capacity_limits_are_ecapacity(tiny):
    cfg, w, prompt = tiny
    cap = 128
    ctx = pkg.Chimera(cfg, w, max_batch=1, max_seq_len=cap)
    assert _status(ctx.prefill, [prompt + prompt]) == ECAPACITY  # 128 tokens + tree slots > cap
    ctx.prefill([prompt + prompt[:36]])  # 100 tokens
    steps, st = 0, 0
    while True:
        try:
            ctx.step()
            steps += 1
        except pkg.ChimeraError as e:
            st = e.status
            break
        assert steps < cap
    assert st == ECAPACITY and steps >= 1
    n = int(ctx.read("n")[0])
    # refused before it could overrun: n plus one step's tree and path still fits
    assert n + cfg["tree_nodes"] + 1 <= cap
    ctx.close()


def test_bounded_wait_timeout_is_reported_and_recovered():
    g = torch.Generator().manual_seed(5)
    M, N, K = 64, 4096, 4096
    X = torch.randn(M, K, generator=g).to(torch.bfloat16).cuda()
    W = (torch.randn(N, K, generator=g) * 0.02).to(torch.bfloat16).cuda()
    ref = (X.double().cpu() @ W.double().cpu().T).numpy()
    pkg.op_sync()  # nothing pending
    Y = torch.zeros(M, N, device="cuda")
    try:
        pkg.set_wait_limit(2)  # ns: every wait that is not satisfied at once gives up
        pkg.op_linear(X, W, Y, epi=0, out_f32=True)  # split-K tiles finished by arrival counters
    finally:
        pkg.set_wait_limit(0)
    with pytest.raises(pkg.ChimeraError) as e:
        pkg.op_sync()
    assert e.value.status == ETIMEDOUT
    pkg.op_sync()  # the word was cleared
    for _ in range(2):  # the workspace counters were reset: the next calls are correct
        Y.zero_()
        pkg.op_linear(X, W, Y, epi=0, out_f32=True)
        pkg.op_sync()
        got = Y.cpu().double().numpy()
        assert np.max(np.abs(got - ref)) / np.max(np.abs(ref)) <= 1e-2
