"""Static candidate tree of the oracle (test infrastructure: only tests/, the smoke
check and the benchmark's CPU baseline may import this package).

The paper builds its tree from the per-head top-k tokens (Section "Inference":
candidate sequences from the top-k of every Chimera head; Section "Verification":
Medusa-style tree attention), but does not say which rank combinations form the
tree.  Reading used here: rank the combinations by the product of per-head
marginal top-k accuracies taken from Table 4 (Chimera rows, Vicuna-7B) and keep
the N-1 best.

  marginal m_k(r) = TopAcc_k(r+1) - TopAcc_k(r)      (hundredths, Table 4)
  score(r_0..r_{d-1}) = prod_i m_i(r_i) * 100**(4-d)  (exact integers)

Order of selection: score descending, then shallower first, then the
lexicographically smaller rank tuple.  Node order in the verify batch: root, then
(depth, rank tuple) ascending.  Every marginal is < 100 so a node always scores
strictly below its parent and the selection is prefix-closed.
"""
from __future__ import annotations

import itertools

# Table 4, Chimera rows: cumulative top-1..top-5 accuracy of heads 0..3.
TABLE4_CHIMERA = [
    [0.66, 0.78, 0.83, 0.87, 0.90],
    [0.49, 0.55, 0.60, 0.68, 0.75],
    [0.38, 0.44, 0.49, 0.55, 0.62],
    [0.33, 0.38, 0.43, 0.46, 0.54],
]


def marginals() -> list[list[int]]:
    """Per-rank marginal accuracy in hundredths (successive differences of Table 4)."""
    out = []
    for row in TABLE4_CHIMERA:
        cum = [round(a * 100) for a in row]
        out.append([cum[0]] + [cum[i] - cum[i - 1] for i in range(1, len(cum))])
    return out


def build_tree(topk: list[int], n_nodes: int) -> dict:
    """Return the static tree: rank tuples, depth, parent, rank, ancestor masks.

    topk[k] limits the ranks drawn from head k; n_nodes counts the root.
    """
    marg = marginals()
    depth_max = len(topk)
    assert depth_max <= len(marg)
    cands = []
    for d in range(1, depth_max + 1):
        for ranks in itertools.product(*[range(topk[i]) for i in range(d)]):
            s = 1
            for i, r in enumerate(ranks):
                s *= marg[i][r]
            s *= 100 ** (len(marg) - d)
            cands.append((-s, d, ranks))
    cands.sort()
    if n_nodes - 1 > len(cands):
        raise ValueError("tree larger than the rank space")
    chosen = [c[2] for c in cands[: n_nodes - 1]]
    chosen.sort(key=lambda r: (len(r), r))
    nodes = [()] + chosen
    index = {r: i for i, r in enumerate(nodes)}
    parent = [-1] + [index[r[:-1]] for r in chosen]
    depth = [len(r) for r in nodes]
    rank = [0] + [r[-1] for r in chosen]
    anc = []
    for i in range(len(nodes)):
        m, j = 0, i
        while j >= 0:
            m |= 1 << j
            j = parent[j]
        anc.append(m)
    children = [[c for c in range(len(nodes)) if parent[c] == i] for i in range(len(nodes))]
    return dict(nodes=nodes, parent=parent, depth=depth, rank=rank, anc=anc,
                children=children, n=len(nodes))


def tuple_str(r: tuple) -> str:
    return "".join(str(x) for x in r)
