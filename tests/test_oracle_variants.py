"""Pins of the oracle's variants of the method: typical acceptance (Section
"Verification", temperature 1) by hand-computed examples, and the draft ablations (the
one-pass draft, and heads without the residual input) by closed forms and brute force.
"""
import math

import numpy as np
import pytest
import torch

import synth
from oracle import chimera_oracle as co
from oracle import tree as ot


# ----------------------------------------------------------------------------
# typical acceptance
# ----------------------------------------------------------------------------
def _log(p):
    return np.log(np.asarray(p, dtype=np.float64))


def test_typical_threshold_hand_values():
    # p = (1/2, 1/4, 1/8, 1/8): H = 1.75 ln 2, exp(-H) = 2^-1.75 = 0.29730...
    p, thr = co.typical_threshold(_log([0.5, 0.25, 0.125, 0.125]), eps=0.09, delta=0.3)
    np.testing.assert_allclose(p, [0.5, 0.25, 0.125, 0.125], rtol=1e-14)
    assert abs(thr - 0.3 * 2 ** -1.75) < 1e-15  # 0.08919 < eps
    # uniform over 8: H = ln 8, delta * exp(-H) = 0.3 / 8 = 0.0375
    _, thr = co.typical_threshold(np.zeros(8), eps=0.09, delta=0.3)
    assert abs(thr - 0.0375) < 1e-15
    # peaked (0.97, 0.01, 0.01, 0.01): delta * exp(-H) = 0.2537 > eps, the threshold is eps
    _, thr = co.typical_threshold(_log([0.97, 0.01, 0.01, 0.01]), eps=0.09, delta=0.3)
    H = -(0.97 * math.log(0.97) + 3 * 0.01 * math.log(0.01))
    assert 0.3 * math.exp(-H) > 0.09 and thr == 0.09


def _tree4():
    # nodes: root, "0", "1", "00"   (top-k [2, 1])
    return ot.build_tree([2, 1], 4)


def test_typical_acceptance_hand_example():
    t = _tree4()
    assert t["parent"] == [-1, 0, 0, 1]
    root = _log([0.5, 0.25, 0.125, 0.125])   # threshold 0.0892: tokens 2 and 3 (p = 1/8) pass
    n1 = _log([0.97, 0.01, 0.01, 0.01])      # threshold 0.09: only token 0 passes
    n2 = _log([0.1, 0.2, 0.3, 0.4])
    n3 = _log([0.05, 0.05, 0.6, 0.3])
    logits = np.stack([root, n1, n2, n3])
    # node 3 ("00") carries token 1: p = 0.01 at node 1 fails -> depth 1; nodes 1 and 2
    # both pass, the smaller index wins; bonus = argmax at node 1 = 0
    path, bonus = co.accept_typical(t, [0, 2, 3, 1], logits, 0.09, 0.3)
    assert path == [0, 1] and bonus == 0
    # node 3 carries token 0 (p = 0.97): the path goes one deeper, bonus = argmax at node 3
    path, bonus = co.accept_typical(t, [0, 2, 3, 0], logits, 0.09, 0.3)
    assert path == [0, 1, 3] and bonus == 2
    # a root row (0.9, 0.04, 0.03, 0.03) has threshold 0.09: only token 0 passes there.
    # Node 1 with token 1 fails, so its child node 3 fails too although token 0 has
    # p = 0.97 at node 1; node 2 with token 0 passes; bonus = argmax at node 2 = 3
    logits_b = np.stack([_log([0.9, 0.04, 0.03, 0.03]), n1, n2, n3])
    path, bonus = co.accept_typical(t, [0, 1, 0, 0], logits_b, 0.09, 0.3)
    assert path == [0, 2] and bonus == 3
    # no child of the root passes: the root alone, bonus = argmax at the root
    path, bonus = co.accept_typical(t, [0, 1, 2, 0], logits_b, 0.09, 0.3)
    assert path == [0] and bonus == 0


def test_typical_acceptance_extremes():
    # eps <= 0: the threshold is non-positive, every node passes, the deepest path wins
    t = ot.build_tree([3, 2, 1], 9)
    rng = np.random.default_rng(1)
    logits = rng.standard_normal((t["n"], 16))
    toks = [0] + [int(v) for v in rng.integers(0, 16, t["n"] - 1)]
    path, _ = co.accept_typical(t, toks, logits, 0.0, 0.3)
    deepest = [i for i in range(t["n"]) if t["depth"][i] == max(t["depth"])]
    assert path[-1] == min(deepest)
    # eps > 1 and delta > max(1/p): nothing passes, the root alone with its argmax
    path, bonus = co.accept_typical(t, toks, logits, 2.0, 1e9)
    assert path == [0] and bonus == co.argmax_desc(logits[0])


# ----------------------------------------------------------------------------
# draft ablations
# ----------------------------------------------------------------------------
def _cfg(mode, d=64, V=64):
    cfg = synth.get_config("tiny")
    cfg.update(n_layers=1, d_model=d, n_heads=2, head_dim=d // 2, ffn_dim=96, vocab=V, draft_mode=mode)
    return cfg


def _setup(mode):
    cfg = _cfg(mode)
    w = synth.make_weights(cfg, seed=4)
    for k in w:
        if not k.endswith("norm"):
            w[k] = w[k] * 10.0
    d = cfg["d_model"]
    for k in range(cfg["n_draft_heads"]):
        if mode & 2:   # Theta_k = I: the scores are h_full itself
            w[f"heads.{k}"] = torch.eye(d)
        else:          # Theta_k = [0 | I]: the scores are the h_full half of the input
            m = torch.zeros(d, 2 * d)
            m[:, d:] = torch.eye(d)
            w[f"heads.{k}"] = m
    W = co.OracleWeights(w, cache=False)
    st = co.prefill(W, cfg, [7, 3, 9, 44, 12], 64)
    return cfg, W, st


@pytest.mark.parametrize("mode", [0, 2])
def test_sequential_heads_score_their_own_row(mode):
    cfg, W, st = _setup(mode)
    dr = co.draft(W, cfg, st, 2)
    brute = co.draft_bruteforce(W, cfg, st, dr["chain"][: cfg["n_draft_heads"]])
    for k in range(cfg["n_draft_heads"]):
        np.testing.assert_allclose(dr["logits"][k], brute[k], rtol=1e-10, atol=1e-11)
    assert np.max(np.abs(brute[1] - brute[0])) > 1e-3  # the rows differ: each head has its own


@pytest.mark.parametrize("mode", [1, 3])
def test_one_pass_heads_all_score_the_first_row(mode):
    cfg, W, st = _setup(mode)
    dr = co.draft(W, cfg, st, 2)
    brute = co.draft_bruteforce(W, cfg, st, [st.tokens[st.n]])  # one trigram row: x[n-2..n]
    assert len(dr["htri"]) == 1
    for k in range(cfg["n_draft_heads"]):
        np.testing.assert_allclose(dr["logits"][k], brute[0], rtol=1e-10, atol=1e-11)
        np.testing.assert_array_equal(dr["hfull"][k], dr["hfull"][0])


def test_no_residual_head_shape():
    cfg = _cfg(2, d=64, V=97)
    shapes = dict(synth.weight_shapes(cfg))
    assert shapes["heads.0"] == (97, 64)
    assert dict(synth.weight_shapes(_cfg(0, d=64, V=97)))["heads.0"] == (97, 128)
