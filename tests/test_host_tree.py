"""The library's static tree (host code, no GPU) against the oracle's, node by node.

Reading of Section "Inference" with the Table 4 marginals: the N-1 rank tuples of
largest marginal product, ordered by depth then rank tuple.  The oracle enumerates
every tuple with itertools; the library enumerates them recursively and sorts; both
must give the same depth, parent, rank and ancestor mask at every node, bit for bit,
over every head-limit tuple and node count the configuration allows.
"""
import itertools
import random

import pytest

import paper_2402_15758_gb300 as pkg
from oracle import tree as otree
from paper_2402_15758_gb300 import build as pkg_build


@pytest.fixture(scope="module", autouse=True)
def _lib():
    pkg_build.build()
    pkg.load()


def _rank_space(topk):
    n, prod = 0, 1
    for t in topk:
        prod *= min(t, 5)
        n += prod
    return n


def _same(topk, n_nodes):
    got = pkg.static_tree(topk, n_nodes)
    ref = otree.build_tree([min(t, 5) for t in topk], n_nodes)
    for key in ("depth", "parent", "rank", "anc"):
        assert got[key] == ref[key], (topk, n_nodes, key)


def test_every_limit_tuple_up_to_three_heads():
    for k in (1, 2, 3):
        for topk in itertools.product(range(1, 6), repeat=k):
            for n in range(2, min(64, _rank_space(topk) + 1) + 1):
                _same(list(topk), n)


def test_four_heads_sampled_limits_every_node_count():
    rng = random.Random(2402)
    tuples = list(itertools.product(range(1, 6), repeat=4))
    picks = rng.sample(tuples, 40) + [(5, 5, 5, 5), (4, 2, 1, 1), (1, 1, 1, 1), (5, 1, 5, 1)]
    for topk in picks:
        for n in range(2, min(64, _rank_space(topk) + 1) + 1):
            _same(list(topk), n)


def test_limits_past_table4_add_nothing():
    # top-k limits 6..8 are valid for the draft's selection; the tree stops at rank 4
    for topk in ([8, 8, 8, 8], [6, 5, 7, 5], [8, 1], [6]):
        for n in (2, min(64, _rank_space(topk) + 1)):
            _same(topk, n)


def test_the_bench_tree_shape():
    # 7B bs1: N = 64 from topk 5,5,5,5 — one root, the rest down to depth 4
    t = pkg.static_tree([5, 5, 5, 5], 64)
    assert t["parent"][0] == -1 and t["depth"][0] == 0
    assert all(t["parent"][i] < i for i in range(1, 64))
    assert all(t["depth"][i] == t["depth"][t["parent"][i]] + 1 for i in range(1, 64))
    assert max(t["depth"]) == 4


@pytest.mark.parametrize("topk,n", [
    ([5, 5, 5, 5], 65),      # the ancestor masks are 64-bit
    ([5, 5, 5, 5], 1),       # at least the root and one candidate
    ([5, 5, 5, 5, 5], 16),   # Table 4 covers four heads
    ([0, 5], 8),             # a head must offer one rank
    ([9, 5], 8),             # beyond the draft's top-k capacity
    ([1, 1], 4),             # only two tuples: (0) and (0, 0)
    ([2], 4),                # only two tuples at depth 1
])
def test_out_of_range_is_einval(topk, n):
    with pytest.raises(pkg.ChimeraError) as e:
        pkg.static_tree(topk, n)
    assert e.value.status == -1
