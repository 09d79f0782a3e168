"""Closed-form pins of the draft model's parts that brute force cannot separate.

The trigram encoder (eq. "trigram_calculations"), the residual heads (eq. "residual
decoding head": Theta_k applied to [h_LLM_n ; h_full_{n+1+k}]) and the chain of draft
sub-steps (head k's top-1 becomes the last token of the next trigram) are checked here
with hand-built weights whose answers are known without running the oracle's own
formulas: identity blocks select one input, a doubled identity separates "SiLU then
W2" from "W2 then SiLU", and one-hot head rows force each head's top-1.

Mistakes each test is built to catch: SiLU applied after W2, a swapped trigram or
head concatenation, x_{i-1} / x_i mixed up, Hs[n] (not yet committed) read instead of
Hs[n-1] (the paper's h_LLM_n), and a sub-step that does not shift its trigram by the
previous head's top-1.
"""
import numpy as np
import pytest
import scipy.special
import torch

import synth
from oracle import chimera_oracle as co


def _silu(x):
    return x * scipy.special.expit(x)


def _cfg(d=64, V=64):
    cfg = synth.get_config("tiny")
    cfg.update(n_layers=1, d_model=d, n_heads=2, head_dim=d // 2, ffn_dim=96, vocab=V)
    return cfg


def _weights(cfg, seed=3):
    w = synth.make_weights(cfg, seed=seed)
    for k in w:  # a larger init so hidden states are far from zero
        if not k.endswith("norm"):
            w[k] = w[k] * 10.0
    return w


def _state(cfg, w, prompt):
    W = co.OracleWeights(dict(w), cache=False)
    return co.prefill(W, cfg, prompt, 64)


def _eye_block(d, which, scale=1.0):
    """W1 [d][3d] = scale * I on block `which` (0: x_{i-2}, 1: x_{i-1}, 2: x_i)."""
    m = torch.zeros(d, 3 * d)
    m[:, which * d:(which + 1) * d] = torch.eye(d) * scale
    return m


@pytest.mark.parametrize("which", [0, 1, 2])
def test_trigram_encoder_selects_one_embedding(which):
    # W1 = I on one block, W2 = 2 I:  h_tri = 2 SiLU(E[token of that block]).
    # SiLU after W2 would give SiLU(2 E[.]); a swapped concatenation picks another token.
    cfg = _cfg()
    w = _weights(cfg)
    d = cfg["d_model"]
    prompt = [11, 23, 35, 47, 59]
    st = _state(cfg, w, prompt)
    w["tri_w1"] = _eye_block(d, which)
    w["tri_w2"] = torch.eye(d) * 2.0
    W = co.OracleWeights(w, cache=False)
    dr = co.draft(W, cfg, st, 1)
    n = st.n
    toks = st.tokens[: n + 1] + dr["chain"][1:]  # x[0..n] then the drafted top-1 tokens
    E = w["embed"].double().numpy()
    for k in range(cfg["n_draft_heads"]):
        t = toks[n - 2 + k + which]  # block 0 holds x[n-2+k], block 2 holds x[n+k]
        np.testing.assert_allclose(dr["htri"][k], 2.0 * _silu(E[t]), rtol=1e-13, atol=1e-15)


def test_trigram_zero_block_before_the_sequence_start():
    # a one-token prompt: sub-step 0's trigram [x_{-2}; x_{-1}; x_0]... has no x_{n-2}
    # (reading R3: a zero block, so SiLU(0) = 0 comes out of that block)
    cfg = _cfg()
    w = _weights(cfg)
    st = _state(cfg, w, [9])
    w["tri_w1"] = _eye_block(cfg["d_model"], 0)
    w["tri_w2"] = torch.eye(cfg["d_model"])
    dr = co.draft(co.OracleWeights(w, cache=False), cfg, st, 1)
    np.testing.assert_array_equal(dr["htri"][0], np.zeros(cfg["d_model"]))


@pytest.mark.parametrize("half", [0, 1])
def test_residual_head_input_halves(half):
    # V = d; Theta_k = [I | 0] scores exactly h_LLM_n = Hs[n-1] (the last committed
    # row, post final norm); Theta_k = [0 | I] scores exactly h_full_{n+1+k}.
    cfg = _cfg(d=64, V=64)
    w = _weights(cfg)
    d = cfg["d_model"]
    st = _state(cfg, w, [3, 14, 15, 9, 26, 53])
    for k in range(cfg["n_draft_heads"]):
        m = torch.zeros(d, 2 * d)
        m[:, half * d:(half + 1) * d] = torch.eye(d)
        w[f"heads.{k}"] = m
    dr = co.draft(co.OracleWeights(w, cache=False), cfg, st, 2)
    hs_last = co.causal_forward(co.OracleWeights(w, cache=False), cfg, st.tokens[: st.n])[0][-1]
    for k in range(cfg["n_draft_heads"]):
        want = st.Hs[st.n - 1] if half == 0 else dr["hfull"][k]
        np.testing.assert_array_equal(dr["logits"][k], want)
        if half == 0:  # and that row is the from-scratch forward's last hidden state
            np.testing.assert_allclose(dr["logits"][k], hs_last, rtol=1e-11, atol=1e-12)
    if half == 0:
        assert np.max(np.abs(hs_last)) > 0.1  # the pinned row is not the zero row Hs[n]


def test_draft_chain_shifts_trigram_by_previous_top1():
    # one-hot head rows force head k's top-1 to a chosen token c_k; with W1 = I on the
    # x_i block the trigram of sub-step k+1 must end at c_k, and with W1 = I on the
    # x_{i-2} block sub-step k+2 must start at c_k.
    cfg = _cfg(d=64, V=97)
    w = _weights(cfg)
    d, V = cfg["d_model"], cfg["vocab"]
    st = _state(cfg, w, [5, 6, 7, 8])
    forced = [41, 2, 77, 60]
    hs_last = co.causal_forward(co.OracleWeights(w, cache=False), cfg, st.tokens[: st.n])[0][-1]
    for k, c in enumerate(forced):
        m = torch.zeros(V, 2 * d)
        m[c, :d] = torch.from_numpy(np.sign(hs_last)).float() * 100.0  # z[c] = 100 |h_LLM_n|_1 > 0
        w[f"heads.{k}"] = m
    E = w["embed"].double().numpy()
    root = st.tokens[st.n]
    for which, shift in ((2, 0), (0, 2)):
        w["tri_w1"] = _eye_block(d, which)
        w["tri_w2"] = torch.eye(d)
        dr = co.draft(co.OracleWeights(w, cache=False), cfg, st, 3)
        assert dr["chain"] == [root] + forced
        x = st.tokens[: st.n] + [root] + forced  # x[0..n] then the forced top-1 tokens
        for k in range(cfg["n_draft_heads"]):
            np.testing.assert_allclose(dr["htri"][k], _silu(E[x[st.n + k - shift]]), rtol=1e-13, atol=1e-15)
