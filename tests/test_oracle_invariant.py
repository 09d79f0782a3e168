"""Losslessness pin: greedy speculative decoding emits exactly the greedy
autoregressive stream (the paper's title claim; eq. 1 with argmax)."""
import numpy as np
import pytest

from oracle import chimera_oracle as co
from oracle import tree as ot


@pytest.fixture(scope="module")
def tiny_ar(tiny_setup):
    cfg, _, W, prompt = tiny_setup
    return co.ar_generate(W, cfg, prompt, cfg["gen_tokens"] + 5)


def test_spec_equals_ar_tiny(tiny_setup, tiny_ar):
    cfg, _, W, prompt = tiny_setup
    t = ot.build_tree(cfg["topk"], cfg["tree_nodes"])
    out, recs = co.generate(W, cfg, prompt, cfg["gen_tokens"], t)
    assert out == tiny_ar[: cfg["gen_tokens"]]
    assert all(len(r["emitted"]) == len(r["path"]) for r in recs)


@pytest.mark.parametrize("forced", [0, 1, 2, 3, 4])
def test_spec_equals_ar_with_forced_acceptance(tiny_setup, tiny_ar, forced):
    # draft injection: the rank-0 branch carries the true continuation for `forced`
    # tokens, every other node is wrong -> acceptance length == forced every step
    cfg, _, W, prompt = tiny_setup
    t = ot.build_tree(cfg["topk"], cfg["tree_nodes"])
    V = cfg["vocab"]

    def override(st):
        base = st.n - len(prompt)  # index of the root in the AR stream
        toks = [0] * t["n"]
        for i in range(1, t["n"]):
            dep = t["depth"][i]
            want = tiny_ar[base + dep]
            on_branch = all(r == 0 for r in t["nodes"][i])
            toks[i] = want if (on_branch and dep <= forced) else (want + 1 + t["rank"][i]) % V
        return toks

    n_new = 20
    out, recs = co.generate(W, cfg, prompt, n_new, t, override_fn=override)
    assert out == tiny_ar[:n_new]
    assert all(len(r["path"]) - 1 == forced for r in recs[:-1])
