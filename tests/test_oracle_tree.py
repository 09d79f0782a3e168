"""Pins of the static tree, the tree mask and greedy acceptance (hand examples)."""
import heapq
import os

import numpy as np
import pytest

from oracle import chimera_oracle as co
from oracle import tree as ot

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "static_trees.txt")


def _golden():
    out = []
    for line in open(GOLDEN):
        if line.startswith("#") or not line.strip():
            continue
        topk, n, nodes = line.strip().split(";")
        out.append(([int(t) for t in topk.split(",")], int(n), nodes.split()))
    return out


def test_marginals_from_table4():
    assert ot.marginals() == [[66, 12, 5, 4, 3], [49, 6, 5, 8, 7], [38, 6, 5, 6, 7], [33, 5, 5, 3, 8]]


@pytest.mark.parametrize("case", range(3))
def test_static_tree_matches_hand_lists(case):
    topk, n, nodes = _golden()[case]
    t = ot.build_tree(topk, n)
    assert t["n"] == n
    assert [ot.tuple_str(r) for r in t["nodes"][1:]] == nodes


def _best_first(topk, n):
    """Independent construction: best-first expansion from the root with a heap,
    using products of Table 4 marginals as fractions of 100 (prefix-closed)."""
    marg = ot.marginals()
    heap = [(-marg[0][r] * 100 ** 3, 1, (r,)) for r in range(topk[0])]
    heapq.heapify(heap)
    chosen = []
    while len(chosen) < n - 1:
        s, d, r = heapq.heappop(heap)
        chosen.append(r)
        if d < len(topk):
            for c in range(topk[d]):
                heapq.heappush(heap, (s // 100 * marg[d][c], d + 1, r + (c,)))
    return sorted(chosen, key=lambda r: (len(r), r))


@pytest.mark.parametrize("topk,n", [([4, 2, 1, 1], 16), ([5, 5, 5, 5], 32), ([5, 5, 5, 5], 64),
                                    ([3, 3, 3], 20), ([5, 5, 5, 5], 2), ([2, 2, 2, 2], 31)])
def test_static_tree_best_first_agrees(topk, n):
    t = ot.build_tree(topk, n)
    assert t["nodes"][1:] == _best_first(topk, n)
    # prefix closed, parents precede children, anc = ancestors-or-self
    for i in range(1, t["n"]):
        assert t["parent"][i] < i
        assert t["nodes"][t["parent"][i]] == t["nodes"][i][:-1]
        assert t["depth"][i] == t["depth"][t["parent"][i]] + 1


def test_tree_mask_hand_example():
    # nodes {root, "0", "1", "00"} with top-k [2, 1]
    t = ot.build_tree([2, 1], 4)
    assert [ot.tuple_str(r) for r in t["nodes"]] == ["", "0", "1", "00"]
    assert t["anc"] == [0b0001, 0b0011, 0b0101, 0b1011]
    assert t["depth"] == [0, 1, 1, 2]      # positions n, n+1, n+1, n+2


def test_acceptance_hand_example():
    # root = 7; head0 top-2 = [3, 9]; head1 top-1 = [5]
    t = ot.build_tree([2, 1], 4)
    topk = np.array([[3, 9], [5, 0]])
    toks = co.tree_tokens(t, 7, topk)
    assert toks == [7, 3, 9, 5]
    V = 12
    logits = np.zeros((4, V))
    logits[0, 9] = 1.0   # argmax(root) = 9  -> child "1" (token 9)
    logits[2, 4] = 1.0   # argmax("1") = 4   -> no child of "1": stop
    logits[1, 5] = 1.0
    logits[3, 2] = 1.0
    path, bonus = co.accept(t, toks, logits)
    assert path == [0, 2] and bonus == 4


def test_compaction_hand_example():
    # accepted path [0, 2] moves KV slot n+2 -> n+1 and emits [7, 9]
    cfg = dict(n_layers=2, n_heads=1, head_dim=2, d_model=2, rms_eps=1e-6, rope_theta=1e4)
    g = np.random.default_rng(0)
    W = co.OracleWeights({"draft.attn_norm": np.ones(2), "draft.wqkv": g.normal(size=(6, 2))})
    st = co.SeqState(cfg, 16)
    st.n, st.tokens = 5, [1, 2, 3, 4, 5, 7]
    ver = dict(k=g.normal(size=(2, 4, 1, 2)), v=g.normal(size=(2, 4, 1, 2)),
               hidden=g.normal(size=(4, 2)))
    emitted = co.commit(W, cfg, st, [7, 3, 9, 5], ver, [0, 2], 4)
    assert emitted == [7, 9]
    assert st.n == 7 and st.tokens == [1, 2, 3, 4, 5, 7, 9, 4]
    np.testing.assert_array_equal(st.K[:, 5], ver["k"][:, 0])
    np.testing.assert_array_equal(st.K[:, 6], ver["k"][:, 2])
    np.testing.assert_array_equal(st.V[:, 6], ver["v"][:, 2])
    np.testing.assert_array_equal(st.Hs[6], ver["hidden"][2])


def test_compaction_overlapping_slots():
    # path [0, 2, 5] on the 64-node tree: slot n+2 is both a source (of j=1) and a
    # destination (of j=2); every destination must get its own source row
    t = ot.build_tree([5, 5, 5, 5], 64)
    assert t["parent"][2] == 0 and t["parent"][t["children"][2][0]] == 2
    cfg = dict(n_layers=1, n_heads=1, head_dim=2, d_model=2, rms_eps=1e-6, rope_theta=1e4)
    g = np.random.default_rng(1)
    W = co.OracleWeights({"draft.attn_norm": np.ones(2), "draft.wqkv": g.normal(size=(6, 2))})
    st = co.SeqState(cfg, 128)
    st.n, st.tokens = 3, [1, 2, 3, 4]
    ver = dict(k=g.normal(size=(1, 64, 1, 2)), v=g.normal(size=(1, 64, 1, 2)),
               hidden=g.normal(size=(64, 2)))
    path = [0, 2, t["children"][2][0]]
    co.commit(W, cfg, st, list(range(64)), ver, path, 0)
    for j, node in enumerate(path):
        np.testing.assert_array_equal(st.K[0, 3 + j], ver["k"][0, node])
