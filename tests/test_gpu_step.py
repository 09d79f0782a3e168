"""Step-level parity of the CUDA path (through the C ABI) against the fp64 oracle.

tiny (fp32): the whole generation is compared free-running: every draft score,
top-k list, tree token, verify logit/hidden row, argmax, accepted path and emitted
token, and the stream must equal plain greedy decoding.
mini / mini_b4 / 7b (bf16): the oracle drives the trajectory: each step the GPU
verifies the oracle's tree (tree override) and, when a near-tie made the GPU accept
a different path, it is re-synchronised to the oracle's committed tokens (prefill
with the oracle's tokens).  The GPU's own draft is checked against the oracle's draft
on the same state.  Acceptance lengths 0..depth are forced by setting the rank-0
branch to the base model's own greedy continuation.
"""
import os

import numpy as np
import pytest
import torch

import synth
import paper_2402_15758_gb300 as pkg
from oracle import chimera_oracle as co
from oracle import tree as ot
from parity import check_choice, check_topk, rel_rows, tol_of

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2402_15758_gb300 import build
    build.build()
    pkg.load()


def _setup(name, device_gen="cpu"):
    cfg = synth.get_config(name)
    w = synth.make_weights(cfg, device=device_gen)
    if device_gen == "cpu":
        w_cpu = w
        w_dev = {k: v.cuda() for k, v in w.items()}
    else:
        w_dev = w
        w_cpu = {k: v.cpu() for k, v in w.items()}
    return cfg, w_cpu, w_dev


@pytest.fixture(scope="module")
def tiny():
    cfg, w_cpu, w_dev = _setup("tiny")
    return cfg, w_dev, co.OracleWeights(w_cpu), synth.make_prompts(cfg)[0]


def _tree_equal(ctx, t):
    assert ctx.tree["depth"] == t["depth"]
    assert ctx.tree["parent"] == t["parent"]
    assert ctx.tree["rank"][1:] == t["rank"][1:]
    assert ctx.tree["anc"] == t["anc"]


def test_tiny_generation_matches_oracle(tiny):
    cfg, w_dev, W, prompt = tiny
    T, K, kmax, tol = cfg["gen_tokens"], cfg["n_draft_heads"], max(cfg["topk"]), tol_of(cfg)
    tree = ot.build_tree(cfg["topk"], cfg["tree_nodes"])
    ctx = pkg.Chimera(cfg, w_dev, max_batch=1, max_seq_len=256)
    _tree_equal(ctx, tree)
    ctx.prefill([prompt])
    st = co.prefill(W, cfg, prompt, 256)
    assert rel_rows(ctx.read("prefill_logits")[0], st.prefill_logits) <= tol
    out_g, out_o, flags = [], [], 0
    while len(out_o) < T:
        e = ctx.step()[0]
        rec = co.step(W, cfg, st, tree)
        dl = ctx.read("draft_logits")[:, 0]
        topk = ctx.read("topk")[0]
        for k in range(K):
            assert rel_rows(dl[k], rec["draft"]["logits"][k]) <= tol
            flags += check_topk(topk[k], rec["draft"]["logits"][k], kmax)
        assert rel_rows(ctx.read("hfull")[:, 0], rec["draft"]["hfull"]) <= tol
        assert ctx.read("node_tokens")[0].tolist() == rec["node_tokens"]
        assert rel_rows(ctx.read("verify_logits")[0], rec["verify"]["logits"]) <= tol
        assert rel_rows(ctx.read("verify_hidden")[0], rec["verify"]["hidden"]) <= tol
        am = ctx.read("argmax")[0]
        for i in range(tree["n"]):
            flags += check_choice(int(am[i]), rec["verify"]["logits"][i], co.argmax_desc(rec["verify"]["logits"][i]))
        L = int(ctx.read("accept_len")[0])
        assert ctx.read("path")[0][: L + 1].tolist() == rec["path"]
        assert e == rec["emitted"]
        out_g += e
        out_o += rec["emitted"]
    assert out_g[:T] == out_o[:T]
    assert out_o[:T] == co.ar_generate(W, cfg, prompt, T)
    print(f"tiny: {T} tokens bit-exact, near-tie flags {flags}")


def _forced_tokens(tree, base, forced, V):
    """Tree tokens whose rank-0 branch carries `base` (AR continuation, base[0] = root)
    for `forced` drafted tokens; every other node is wrong."""
    toks = [0] * tree["n"]
    for i in range(1, tree["n"]):
        dep = tree["depth"][i]
        on = all(r == 0 for r in tree["nodes"][i])
        toks[i] = base[dep] if (on and dep <= forced) else (base[dep] + 1 + tree["rank"][i]) % V
    return toks


@pytest.mark.parametrize("forced", [0, 1, 2, 3, 4])
def test_tiny_forced_acceptance_and_compaction(tiny, forced):
    cfg, w_dev, W, prompt = tiny
    tol = tol_of(cfg)
    tree = ot.build_tree(cfg["topk"], cfg["tree_nodes"])
    ar = co.ar_generate(W, cfg, prompt, 16)
    ctx = pkg.Chimera(cfg, w_dev, max_batch=1, max_seq_len=256)
    ctx.prefill([prompt])
    st = co.prefill(W, cfg, prompt, 256)
    out = []
    for _ in range(3):
        base = ar[len(out):]
        toks = _forced_tokens(tree, base, forced, cfg["vocab"])
        ctx.override_tree([toks])
        n0 = st.n
        e = ctx.step()[0]
        rec = co.step(W, cfg, st, tree, toks)
        assert e == rec["emitted"] == ar[len(out): len(out) + forced + 1]
        assert int(ctx.read("accept_len")[0]) == forced
        # compacted base KV (first and last layer) and appended draft KV
        for layer in (0, cfg["n_layers"] - 1, -1):
            k, v = ctx.read_kv(layer, 0, n0, forced + 1)
            rk = st.dK[n0:n0 + forced + 1] if layer < 0 else st.K[layer, n0:n0 + forced + 1]
            rv = st.dV[n0:n0 + forced + 1] if layer < 0 else st.V[layer, n0:n0 + forced + 1]
            assert rel_rows(k, rk) <= tol and rel_rows(v, rv) <= tol
        out += e
    assert ctx.read("n")[0] == len(prompt) + len(out)


def _branch_tokens(tree, base, branch, V):
    """Tree tokens whose nodes on `branch` (a rank tuple, e.g. (1, 0, 0)) carry `base`
    (AR continuation, base[0] = root); every other node is wrong."""
    toks = [0] * tree["n"]
    for i in range(1, tree["n"]):
        r, dep = tree["nodes"][i], tree["depth"][i]
        on = tuple(r) == tuple(branch[:dep])
        toks[i] = base[dep] if on else (base[dep] + 1 + tree["rank"][i] + 7 * dep) % V
    return toks


@pytest.mark.parametrize("branch", [(1, 0), (1, 0, 0), (2, 0, 0)])
def test_tiny_overlapping_compaction(tiny, branch):
    # accepted path off the rank-0 branch: e.g. "1" -> "10" -> "100" is nodes [0, 2, 7, 12],
    # so slot n+2 is both the destination of node 7 and the source of node 2; every
    # layer's compacted KV and the appended draft KV must equal the oracle's
    cfg, w_dev, W, prompt = tiny
    tol = tol_of(cfg)
    tree = ot.build_tree(cfg["topk"], cfg["tree_nodes"])
    ar = co.ar_generate(W, cfg, prompt, 12)
    ctx = pkg.Chimera(cfg, w_dev, max_batch=1, max_seq_len=256)
    ctx.prefill([prompt])
    st = co.prefill(W, cfg, prompt, 256)
    out = []
    for _ in range(2):
        toks = _branch_tokens(tree, ar[len(out):], branch, cfg["vocab"])
        ctx.override_tree([toks])
        n0 = st.n
        e = ctx.step()[0]
        rec = co.step(W, cfg, st, tree, toks)
        L = len(branch)
        want_path = [0] + [tree["nodes"].index(tuple(branch[:j])) for j in range(1, L + 1)]
        assert rec["path"] == want_path
        assert ctx.read("path")[0][: L + 1].tolist() == want_path
        # some entry's source slot is another entry's destination slot
        assert any(want_path[j] == j2 for j in range(1, L + 1) for j2 in range(1, L + 1) if j2 != j)
        assert e == rec["emitted"] == ar[len(out): len(out) + L + 1]
        for layer in list(range(cfg["n_layers"])) + [-1]:
            k, v = ctx.read_kv(layer, 0, n0, L + 1)
            rk = st.dK[n0:n0 + L + 1] if layer < 0 else st.K[layer, n0:n0 + L + 1]
            rv = st.dV[n0:n0 + L + 1] if layer < 0 else st.V[layer, n0:n0 + L + 1]
            assert rel_rows(k, rk) <= tol and rel_rows(v, rv) <= tol, layer
        out += e
    assert ctx.read("n")[0] == len(prompt) + len(out)


# ----------------------------------------------------------------------------
# bf16 configs, oracle-driven
# ----------------------------------------------------------------------------
def _force_chain(W, cfg, st, tree, toks, L, branch=(0, 0, 0, 0)):
    """Set the nodes of `branch` (a rank tuple; default the rank-0 branch) to the base
    model's greedy continuation for L tokens; a sibling that happens to carry the same
    token is moved off it, so the accepted path is exactly that branch."""
    toks = list(toks)
    V = cfg["vocab"]
    chain = [0]
    for d in range(1, len(branch) + 1):
        r = tuple(branch[:d])
        if r not in tree["nodes"]:
            break
        chain.append(tree["nodes"].index(r))
    for j in range(1, min(L, len(chain) - 1) + 1):
        ver = co.verify(W, cfg, st, tree, toks)
        t = co.argmax_desc(ver["logits"][chain[j - 1]])
        toks[chain[j]] = t
        for c in tree["children"][chain[j - 1]]:
            if c != chain[j] and toks[c] == t:
                toks[c] = (t + 1) % V
    return toks


def _run_bf16(name, n_steps, forced_seq, device_gen="cpu", max_seq=None, precision=1, branch=(0, 0, 0, 0), **over):
    cfg, w_cpu, w_dev = _setup(name, device_gen)
    cfg.update(over)
    W = co.OracleWeights(w_cpu, cache=(name != "7b"))
    prompts = synth.make_prompts(cfg)
    B, K, kmax, V, tol = len(prompts), cfg["n_draft_heads"], max(cfg["topk"]), cfg["vocab"], tol_of(cfg)
    cap = max(len(p) for p in prompts) + n_steps * 5 + cfg["tree_nodes"] + 16
    cap = max_seq or ((cap + 15) // 16) * 16
    tree = ot.build_tree(cfg["topk"], cfg["tree_nodes"])
    ctx = pkg.Chimera(cfg, w_dev, max_batch=B, max_seq_len=cap, precision=precision)
    _tree_equal(ctx, tree)
    states = [co.prefill(W, cfg, p, cap + 8) for p in prompts]
    ctx.prefill(prompts)
    flags, skipped, resync, accepted = 0, 0, 0, []
    pl = ctx.read("prefill_logits")
    gtok = ctx.read("tokens")
    for b in range(B):
        assert rel_rows(pl[b], states[b].prefill_logits) <= tol
        n = states[b].n
        flags += check_choice(int(gtok[b, n]), states[b].prefill_logits, states[b].tokens[n])
    ctx.set_root([s.tokens[s.n] for s in states])
    for step in range(n_steps):
        drafts, toks_all = [], []
        for b in range(B):
            dr = co.draft(W, cfg, states[b], kmax)
            toks = co.tree_tokens(tree, states[b].tokens[states[b].n], dr["topk"])
            toks = _force_chain(W, cfg, states[b], tree, toks, forced_seq[(step + b) % len(forced_seq)], branch)
            drafts.append(dr)
            toks_all.append(toks)
        n_before = [s.n for s in states]
        ctx.override_tree(toks_all)
        emitted = ctx.step()
        dl = ctx.read("draft_logits")
        gtopk = ctx.read("topk")
        vl = ctx.read("verify_logits")
        vh = ctx.read("verify_hidden")
        am = ctx.read("argmax")
        gpath = ctx.read("path")
        glen = ctx.read("accept_len")
        diverged = False
        for b in range(B):
            dr = drafts[b]
            # draft: head k is comparable while the GPU's top-1 chain equals the oracle's
            for k in range(K):
                if [int(gtopk[b, j, 0]) for j in range(k)] != dr["chain"][1:k + 1]:
                    skipped += K - k
                    break
                assert rel_rows(dl[k, b], dr["logits"][k]) <= tol, (step, b, k)
                flags += check_topk(gtopk[b, k], dr["logits"][k], kmax)
            ver = co.verify(W, cfg, states[b], tree, toks_all[b])
            assert rel_rows(vl[b], ver["logits"]) <= tol, (step, b)
            assert rel_rows(vh[b], ver["hidden"]) <= tol, (step, b)
            f = 0
            for i in range(tree["n"]):
                f += check_choice(int(am[b, i]), ver["logits"][i], co.argmax_desc(ver["logits"][i]))
            flags += f
            path, bonus = co.accept(tree, toks_all[b], ver["logits"])
            L = int(glen[b])
            if gpath[b, : L + 1].tolist() != path:
                assert f > 0, "accepted path differs without a near-tie"
                diverged = True
            else:
                assert emitted[b] == [toks_all[b][i] for i in path]
                # compacted KV of the accepted rows in every layer, and draft KV
                for layer in range(cfg["n_layers"]):
                    k_g, v_g = ctx.read_kv(layer, b, n_before[b], L + 1)
                    assert rel_rows(k_g, ver["k"][layer][path]) <= tol
                    assert rel_rows(v_g, ver["v"][layer][path]) <= tol
            accepted.append(len(path) - 1)
            co.commit(W, cfg, states[b], toks_all[b], ver, path, bonus)
            if not diverged:
                dk_g, dv_g = ctx.read_kv(-1, b, n_before[b], len(path))
                assert rel_rows(dk_g, states[b].dK[n_before[b]:n_before[b] + len(path)]) <= tol
                assert rel_rows(dv_g, states[b].dV[n_before[b]:n_before[b] + len(path)]) <= tol
        if diverged:
            resync += 1
            ctx.prefill([s.tokens[: s.n] for s in states])
        ctx.set_root([s.tokens[s.n] for s in states])
        assert ctx.read("n").tolist() == [s.n for s in states]
    ctx.close()
    print(f"{name} (precision {precision}): {n_steps} steps x {B} seqs, accepted {accepted}, flags {flags}, "
          f"draft heads skipped {skipped}, resyncs {resync}")
    return accepted


def test_mini_bf16_steps():
    acc = _run_bf16("mini", 6, [0, 4, 2, 1, 3])
    assert max(acc) >= 3


def test_mini_bf16_plain_precision():
    # activations rounded once to bf16 and bf16 KV caches (precision 0)
    _run_bf16("mini", 3, [4, 2, 0], precision=0)


def test_mini_overlapping_compaction():
    # accepted paths along "1" -> "10" -> "100" -> "1000" (nodes 2, 11, 39, 62 of the
    # 64-node tree): destination slots n+1.. are sources of later path entries
    acc = _run_bf16("mini", 3, [4, 2, 3], branch=(1, 0, 0, 0))
    assert max(acc) >= 3


@pytest.mark.parametrize("name", ["mini", "mini_b4"])
def test_bf16_steps_fused_chain(name):
    # the persistent chain launches (fused_chain = 1) against the oracle, with forced
    # acceptance along an off-rank-0 branch (overlapping compaction)
    acc = _run_bf16(name, 3, [4, 1, 3], branch=(1, 0, 0, 0), fused_chain=1)
    assert max(acc) >= 1


def test_mini_b4_ragged_batch():
    acc = _run_bf16("mini_b4", 3, [1, 0, 4, 2])
    assert max(acc) >= 2


def _host_mem_gb():
    try:
        return os.sysconf("SC_PAGE_SIZE") * os.sysconf("SC_PHYS_PAGES") / 2**30
    except (ValueError, OSError):
        return 0


@pytest.mark.skipif(_host_mem_gb() < 96, reason="the fp64 oracle of the 7B model needs >= 96 GB of host memory")
def test_7b_full_size_step():
    # the benchmark's workload: 7B shape, bs1, 512-token prompt, 64-node tree
    _run_bf16("7b", 1, [2], device_gen="cuda", max_seq=1024)


@pytest.mark.skipif(_host_mem_gb() < 96, reason="the fp64 oracle of the 7B model needs >= 96 GB of host memory")
def test_7b_full_size_step_fused_chain():
    _run_bf16("7b", 1, [3], device_gen="cuda", max_seq=1024, fused_chain=1)


# ----------------------------------------------------------------------------
# plain autoregressive steps (eq. 1): the baseline path on the same kernels
# ----------------------------------------------------------------------------
def test_tiny_ar_generation_matches_oracle(tiny):
    cfg, w_dev, W, prompt = tiny
    T = cfg["gen_tokens"]
    ctx = pkg.Chimera(cfg, w_dev, max_batch=1, max_seq_len=256)
    ctx.prefill([prompt])
    out = ctx.ar_generate(T)[0]
    assert out == co.ar_generate(W, cfg, prompt, T)
    ctx.close()


def test_tiny_ar_and_spec_steps_mix(tiny):
    # both kinds of step leave the same state: any interleaving emits the AR stream
    cfg, w_dev, W, prompt = tiny
    ref = co.ar_generate(W, cfg, prompt, 40)
    ctx = pkg.Chimera(cfg, w_dev, max_batch=1, max_seq_len=256)
    ctx.prefill([prompt])
    out = []
    for kind in ["ar", "spec", "spec", "ar", "ar", "spec", "ar", "spec"]:
        out += ctx.ar_generate(2)[0] if kind == "ar" else ctx.step()[0]
    assert out == ref[: len(out)]
    n = int(ctx.read("n")[0])
    assert n == len(prompt) + len(out)
    # the committed KV rows equal a from-scratch prefill of the committed tokens
    st = co.prefill(W, cfg, prompt + out, 256)
    for layer in list(range(cfg["n_layers"])) + [-1]:
        k, v = ctx.read_kv(layer, 0, 0, n)
        rk = st.dK[:n] if layer < 0 else st.K[layer, :n]
        rv = st.dV[:n] if layer < 0 else st.V[layer, :n]
        assert rel_rows(k, rk) <= tol_of(cfg) and rel_rows(v, rv) <= tol_of(cfg), layer
    ctx.close()


@pytest.mark.parametrize("name,fused", [("mini", 0), ("mini_b4", 0), ("mini", 1)])
def test_bf16_ar_steps_match_oracle(name, fused):
    cfg, w_cpu, w_dev = _setup(name)
    cfg["fused_chain"] = fused
    W = co.OracleWeights(w_cpu)
    prompts = synth.make_prompts(cfg)
    B, tol = len(prompts), tol_of(cfg)
    ctx = pkg.Chimera(cfg, w_dev, max_batch=B, max_seq_len=256)
    ctx.prefill(prompts)
    seqs = [list(p) for p in prompts]
    flags = 0
    for b in range(B):  # the roots: the oracle's greedy next token (a near-tie may differ)
        _, lg = co.causal_forward(W, cfg, seqs[b])
        flags += check_choice(int(ctx.read("tokens")[b, len(seqs[b])]), lg[-1], co.argmax_desc(lg[-1]))
        seqs[b].append(co.argmax_desc(lg[-1]))
    ctx.set_root([s[-1] for s in seqs])
    for step in range(5):
        out = ctx.ar_generate(1)
        logits = ctx.read("prefill_logits")  # the LM-head rows of the step's B query rows
        toks = ctx.read("tokens")
        for b in range(B):
            assert out[b] == [seqs[b][-1]]
            _, lg = co.causal_forward(W, cfg, seqs[b])
            assert rel_rows(logits[b], lg[-1]) <= tol, (step, b)
            ref = co.argmax_desc(lg[-1])
            flags += check_choice(int(toks[b, len(seqs[b])]), lg[-1], ref)
            seqs[b].append(ref)
        ctx.set_root([s[-1] for s in seqs])
    assert ctx.read("n").tolist() == [len(s) - 1 for s in seqs]
    ctx.close()
    print(f"{name} AR: 5 steps x {B} seqs, near-tie flags {flags}")
