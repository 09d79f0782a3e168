"""GPU parity of the method's variants against the fp64 oracle (through the C ABI):

* the trigram cache (Section "Trigram encoder", lookup table): results identical with
  the cache on and off, and a cached h_tri row identical bit for bit to the computed one;
* typical acceptance (Section "Verification", T = 1): accepted paths equal the oracle's
  except where one of the thresholds is a near-tie (flagged and counted);
* the draft ablations: the one-pass draft and heads without the residual input.
"""
import numpy as np
import pytest

import paper_2402_15758_gb300 as pkg
import synth
from oracle import chimera_oracle as co
from oracle import tree as ot
from parity import NEAR_TIE, check_choice, check_topk, rel_rows, tol_of

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2402_15758_gb300 import build
    build.build()
    pkg.load()


def _setup(name, **over):
    cfg = synth.get_config(name)
    cfg.update(over)
    w_cpu = synth.make_weights(cfg)
    w_dev = {k: v.cuda() for k, v in w_cpu.items()}
    return cfg, w_cpu, w_dev


# ----------------------------------------------------------------------------
# trigram cache
# ----------------------------------------------------------------------------
def _free_run(ctx, prompt, steps):
    ctx.prefill([prompt])
    rec = []
    for _ in range(steps):
        e = ctx.step()[0]
        rec.append(dict(emitted=e, draft=ctx.read("draft_logits").copy(), verify=ctx.read("verify_logits").copy(),
                        hits=ctx.read("trigram_hits").copy() if ctx.cfg.get("trigram_cache") else None,
                        htri=ctx.read("htri").copy() if ctx.cfg.get("trigram_cache") else None))
    return rec


def test_tiny_trigram_cache_is_exact():
    # fp32 path (deterministic): the same prompt twice through a cached context; the
    # second pass meets the trigrams of the first, so its sub-steps hit, and every
    # result equals the first pass, a context without the cache and the oracle
    cfg, w_cpu, w_dev = _setup("tiny", trigram_cache=64)
    prompt = synth.make_prompts(cfg)[0]
    ctx = pkg.Chimera(cfg, w_dev, max_batch=1, max_seq_len=256)
    first = _free_run(ctx, prompt, 8)
    second = _free_run(ctx, prompt, 8)
    hits = int(sum(r["hits"].sum() for r in second))
    assert hits >= 8  # at least sub-step 0 of every step of the second pass
    plain = pkg.Chimera(dict(cfg, trigram_cache=0), w_dev, max_batch=1, max_seq_len=256)
    ref = _free_run(plain, prompt, 8)
    for a, b, c in zip(first, second, ref):
        assert a["emitted"] == b["emitted"] == c["emitted"]
        np.testing.assert_array_equal(a["draft"], b["draft"])
        np.testing.assert_array_equal(a["draft"], c["draft"])
        np.testing.assert_array_equal(a["verify"], c["verify"])
        np.testing.assert_array_equal(a["htri"], b["htri"])
    W = co.OracleWeights(w_cpu)
    out = sum((r["emitted"] for r in second), [])
    assert out == co.ar_generate(W, cfg, prompt, len(out))
    ctx.close()
    plain.close()
    print(f"tiny trigram cache: {hits} hits in the second pass")


def test_mini_trigram_cache_rows_match():
    # bf16: a cached h_tri row equals the row computed for the same trigram bit for
    # bit, and both match the oracle's trigram encoder
    cfg, w_cpu, w_dev = _setup("mini", trigram_cache=256)
    prompt = synth.make_prompts(cfg)[0]
    W = co.OracleWeights(w_cpu)
    ctx = pkg.Chimera(cfg, w_dev, max_batch=1, max_seq_len=256)
    tol = tol_of(cfg)
    seen = {}
    hits = 0
    for rnd in range(2):
        ctx.prefill([prompt])
        for _ in range(3):
            toks_before = ctx.read("tokens")[0].tolist()
            n = int(ctx.read("n")[0])
            ctx.step()
            topk = ctx.read("topk")[0]
            hit = ctx.read("trigram_hits")[:, 0]
            htri = ctx.read("htri")[:, 0]
            x = toks_before[: n + 1] + [int(topk[j, 0]) for j in range(cfg["n_draft_heads"])]
            for k in range(cfg["n_draft_heads"]):
                tri = tuple(x[n - 2 + k: n + 1 + k])
                ref = co.trigram_encoder(W, co.trigram_input(W, cfg, list(tri)))
                assert rel_rows(htri[k], ref) <= tol
                if tri in seen:
                    np.testing.assert_array_equal(htri[k], seen[tri])
                seen.setdefault(tri, htri[k].copy())
                hits += int(hit[k])
    assert hits >= 3
    ctx.close()


# ----------------------------------------------------------------------------
# typical acceptance
# ----------------------------------------------------------------------------
def _typical_flags(tree, toks, logits, eps, delta):
    """Relative margins |p - thr| / thr of every node's typical decision (oracle)."""
    m = []
    for c in range(1, tree["n"]):
        p, thr = co.typical_threshold(logits[tree["parent"][c]], eps, delta)
        m.append(abs(p[toks[c]] - thr) / max(thr, 1e-300))
    return min(m) if m else np.inf


@pytest.mark.parametrize("name", ["tiny", "mini"])
def test_typical_acceptance_matches_oracle(name):
    cfg, w_cpu, w_dev = _setup(name, accept_mode=1, typical_eps=0.09, typical_delta=0.3)
    W = co.OracleWeights(w_cpu)
    prompt = synth.make_prompts(cfg)[0]
    tree = ot.build_tree(cfg["topk"], cfg["tree_nodes"])
    tol = tol_of(cfg)
    ctx = pkg.Chimera(cfg, w_dev, max_batch=1, max_seq_len=320)
    st = co.prefill(W, cfg, prompt, 320)
    ctx.prefill([prompt])
    ctx.set_root([st.tokens[st.n]])
    flags, lens = 0, []
    for _ in range(4):
        dr = co.draft(W, cfg, st, max(cfg["topk"]))
        toks = co.tree_tokens(tree, st.tokens[st.n], dr["topk"])
        ctx.override_tree([toks])
        n0 = st.n
        e = ctx.step()[0]
        ver = co.verify(W, cfg, st, tree, toks)
        assert rel_rows(ctx.read("verify_logits")[0], ver["logits"]) <= tol
        path, bonus = co.accept_typical(tree, toks, ver["logits"], 0.09, 0.3)
        L = int(ctx.read("accept_len")[0])
        gpath = ctx.read("path")[0][: L + 1].tolist()
        if gpath != path:
            assert _typical_flags(tree, toks, ver["logits"], 0.09, 0.3) < NEAR_TIE, (gpath, path)
            flags += 1
        else:
            assert e == [toks[i] for i in path]
            flags += check_choice(int(ctx.read("tokens")[0, n0 + L + 1]), ver["logits"][path[-1]], bonus)
            for layer in range(cfg["n_layers"]):
                k, v = ctx.read_kv(layer, 0, n0, L + 1)
                assert rel_rows(k, ver["k"][layer][path]) <= tol and rel_rows(v, ver["v"][layer][path]) <= tol
        lens.append(len(path) - 1)
        co.commit(W, cfg, st, toks, ver, path, bonus)
        if gpath != path:
            ctx.prefill([st.tokens[: st.n]])
        ctx.set_root([st.tokens[st.n]])
        assert int(ctx.read("n")[0]) == st.n
    ctx.close()
    print(f"{name} typical: accepted {lens}, flags {flags}")
    assert max(lens) >= 1


# ----------------------------------------------------------------------------
# draft ablations
# ----------------------------------------------------------------------------
@pytest.mark.parametrize("mode", [1, 2, 3])
def test_tiny_draft_variants(mode):
    # still lossless (greedy acceptance), and every head's scores match the oracle's draft
    cfg, w_cpu, w_dev = _setup("tiny", draft_mode=mode)
    W = co.OracleWeights(w_cpu)
    prompt = synth.make_prompts(cfg)[0]
    tree = ot.build_tree(cfg["topk"], cfg["tree_nodes"])
    ctx = pkg.Chimera(cfg, w_dev, max_batch=1, max_seq_len=256)
    ctx.prefill([prompt])
    st = co.prefill(W, cfg, prompt, 256)
    out, flags = [], 0
    while len(out) < 16:
        e = ctx.step()[0]
        rec = co.step(W, cfg, st, tree)
        dl = ctx.read("draft_logits")[:, 0]
        topk = ctx.read("topk")[0]
        for k in range(cfg["n_draft_heads"]):
            assert rel_rows(dl[k], rec["draft"]["logits"][k]) <= tol_of(cfg)
            flags += check_topk(topk[k], rec["draft"]["logits"][k], max(cfg["topk"]))
        assert e == rec["emitted"]
        out += e
    assert out[:16] == co.ar_generate(W, cfg, prompt, 16)
    ctx.close()


@pytest.mark.parametrize("fused", [0, 1])
def test_mini_draft_one_pass_no_residual(fused):
    cfg, w_cpu, w_dev = _setup("mini", draft_mode=3, fused_chain=fused)
    W = co.OracleWeights(w_cpu)
    prompt = synth.make_prompts(cfg)[0]
    ctx = pkg.Chimera(cfg, w_dev, max_batch=1, max_seq_len=256)
    st = co.prefill(W, cfg, prompt, 256)
    ctx.prefill([prompt])
    ctx.set_root([st.tokens[st.n]])
    ctx.step()
    dr = co.draft(W, cfg, st, max(cfg["topk"]))
    dl = ctx.read("draft_logits")[:, 0]
    hf = ctx.read("hfull")[:, 0]
    for k in range(cfg["n_draft_heads"]):
        assert rel_rows(dl[k], dr["logits"][k]) <= tol_of(cfg)
        np.testing.assert_array_equal(hf[k], hf[0])
    ctx.close()
