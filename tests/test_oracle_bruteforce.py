"""Brute-force pins of the oracle: the KV-cached tree/draft paths against from-scratch
causal forwards over explicit sequences."""
import numpy as np
import pytest

import synth
from oracle import chimera_oracle as co
from oracle import tree as ot


def _small_cfg():
    cfg = synth.get_config("tiny")
    cfg.update(n_layers=2, d_model=64, n_heads=2, head_dim=32, ffn_dim=96, vocab=97)
    return cfg


@pytest.fixture(scope="module")
def small():
    cfg = _small_cfg()
    w = synth.make_weights(cfg, seed=11)
    # larger init so the random model is far from uniform attention
    for k in w:
        if not k.endswith("norm"):
            w[k] = w[k] * 10.0
    W = co.OracleWeights(w)
    prompt = [int(t) for t in np.random.default_rng(5).integers(0, cfg["vocab"], 13)]
    return cfg, W, prompt


def test_prefill_matches_causal_forward(small):
    cfg, W, prompt = small
    st = co.prefill(W, cfg, prompt, 64)
    hs, logits = co.causal_forward(W, cfg, prompt)
    np.testing.assert_allclose(st.Hs[: len(prompt)], hs, rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(st.prefill_logits, logits[-1], rtol=1e-11, atol=1e-12)
    assert st.tokens[-1] == co.argmax_desc(logits[-1])


@pytest.mark.parametrize("topk,N", [([4, 2, 1, 1], 16), ([3, 3], 9), ([2, 1], 2)])
def test_verify_logits_equal_path_forward(small, topk, N):
    # each node's logits = a from-scratch causal forward over prefix + root->node path
    cfg, W, prompt = small
    st = co.prefill(W, cfg, prompt, 64)
    t = ot.build_tree(topk, N)
    rng = np.random.default_rng(N)
    toks = [st.tokens[-1]] + [int(v) for v in rng.integers(0, cfg["vocab"], N - 1)]
    ver = co.verify(W, cfg, st, t, toks)
    for i in range(N):
        path, j = [], i
        while j >= 0:
            path.append(toks[j])
            j = t["parent"][j]
        seq = prompt + path[::-1]
        hs, logits = co.causal_forward(W, cfg, seq)
        np.testing.assert_allclose(ver["logits"][i], logits[-1], rtol=1e-10, atol=1e-11)
        np.testing.assert_allclose(ver["hidden"][i], hs[-1], rtol=1e-10, atol=1e-11)


def test_draft_incremental_equals_full_context_block(small):
    cfg, W, prompt = small
    st = co.prefill(W, cfg, prompt, 64)
    dr = co.draft(W, cfg, st, 4)
    brute = co.draft_bruteforce(W, cfg, st, dr["chain"][: cfg["n_draft_heads"]])
    np.testing.assert_allclose(dr["hfull"], brute, rtol=1e-10, atol=1e-11)
    # head k = Theta_k [h_LLM_n ; h_full_{n+1+k}], top-k of it
    for k in range(cfg["n_draft_heads"]):
        z = W(f"heads.{k}") @ np.concatenate([st.Hs[st.n - 1], brute[k]])
        np.testing.assert_allclose(dr["logits"][k], z, rtol=1e-10, atol=1e-11)
        assert dr["chain"][k + 1] == co.argmax_desc(z)


def test_trigram_collapse_for_short_prefix(small):
    # n = 1: the first sub-step's trigram lacks x_{n-2}: zero block (reading R3)
    cfg, W, _ = small
    st = co.prefill(W, cfg, [5], 16)
    dr = co.draft(W, cfg, st, 2)
    t0 = np.concatenate([np.zeros(cfg["d_model"]), W.rows("embed", [5])[0],
                         W.rows("embed", [st.tokens[1]])[0]])
    np.testing.assert_allclose(dr["htri"][0], W("tri_w2") @ co.silu(W("tri_w1") @ t0), rtol=1e-12)


def test_step_commit_equals_prefill_of_committed(small):
    # after a step (forced to accept 2 drafted tokens), the committed state equals a
    # from-scratch prefill of the committed tokens
    cfg, W, prompt = small
    t = ot.build_tree([4, 2, 1, 1], 16)
    ar = co.ar_generate(W, cfg, prompt, 5)
    st = co.prefill(W, cfg, prompt, 64)
    ov = _force_branch(t, ar, 2, cfg["vocab"])
    rec = co.step(W, cfg, st, t, ov)
    assert rec["path"] == [0, 1, 5] and rec["emitted"] == ar[:3]
    ref = co.prefill(W, cfg, prompt + ar[:3], 64)
    n = st.n
    assert n == len(prompt) + 3 and st.tokens == ref.tokens
    np.testing.assert_allclose(st.K[:, :n], ref.K[:, :n], rtol=1e-10, atol=1e-11)
    np.testing.assert_allclose(st.V[:, :n], ref.V[:, :n], rtol=1e-10, atol=1e-11)
    np.testing.assert_allclose(st.Hs[:n], ref.Hs[:n], rtol=1e-10, atol=1e-11)
    np.testing.assert_allclose(st.dK[:n], ref.dK[:n], rtol=1e-10, atol=1e-11)
    np.testing.assert_allclose(st.dV[:n], ref.dV[:n], rtol=1e-10, atol=1e-11)


def _force_branch(t, ar, L, V):
    """Node tokens so that the rank-0 branch carries the true AR continuation for L
    drafted tokens and every other node (and depth L+1 of the branch) is wrong."""
    toks = [0] * t["n"]
    for i in range(1, t["n"]):
        dep = t["depth"][i]
        want = ar[dep]  # AR token at depth dep (ar[0] is the root)
        on_branch = all(r == 0 for r in t["nodes"][i])
        toks[i] = want if (on_branch and dep <= L) else (want + 1 + t["rank"][i]) % V
    return toks


def test_block_rows_attention_equals_per_row_key_lists(small):
    # block_rows scores each query against [context ; local] at once; the same rows,
    # attended one at a time over an explicit list of their visible keys (attend),
    # must give the same block output
    cfg, W, _ = small
    H, hd, d = cfg["n_heads"], cfg["head_dim"], cfg["d_model"]
    rng = np.random.default_rng(21)
    R, m = 6, 9
    x = rng.standard_normal((R, d))
    pos = np.array([9, 10, 10, 11, 11, 12])
    ctx_k, ctx_v = rng.standard_normal((m, H, hd)), rng.standard_normal((m, H, hd))
    parent = [-1, 0, 0, 1, 2, 3]
    mask = np.zeros((R, R), dtype=bool)
    for i in range(R):
        j = i
        while j >= 0:
            mask[i, j] = True
            j = parent[j]
    out, k, v = co.block_rows(W, "layers.0", cfg, x, pos, ctx_k, ctx_v, mask)
    p = "layers.0"
    h = co.rmsnorm(x, W(f"{p}.attn_norm"), cfg["rms_eps"])
    q = co.rope((h @ W(f"{p}.wqkv").T)[:, :d].reshape(R, H, hd), pos, cfg["rope_theta"])
    att = np.stack([co.attend(q[i], np.concatenate([ctx_k, k[mask[i]]]), np.concatenate([ctx_v, v[mask[i]]]))
                    for i in range(R)])
    x1 = x + att.reshape(R, d) @ W(f"{p}.wo").T
    h2 = co.rmsnorm(x1, W(f"{p}.ffn_norm"), cfg["rms_eps"])
    ref = x1 + (co.silu(h2 @ W(f"{p}.w_gate").T) * (h2 @ W(f"{p}.w_up").T)) @ W(f"{p}.w_down").T
    np.testing.assert_allclose(out, ref, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("chunk", [1, 4, 5])
def test_chunked_prefill_equals_one_pass(small, chunk):
    cfg, W, prompt = small
    a = co.prefill(W, cfg, prompt, 64)
    b = co.prefill(W, cfg, prompt, 64, chunk=chunk)
    n = len(prompt)
    assert a.tokens == b.tokens
    np.testing.assert_allclose(b.K[:, :n], a.K[:, :n], rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(b.V[:, :n], a.V[:, :n], rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(b.Hs[:n], a.Hs[:n], rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(b.prefill_logits, a.prefill_logits, rtol=1e-11, atol=1e-12)
