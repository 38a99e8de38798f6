"""Sparse draft trees for TREE mode (arXiv 2609.37007, Sec. 2.2 and Sec. 3.1): host-side
construction from measured acceptance statistics.

The paper calibrates its sparse tree offline: per drafted depth d and candidate rank r it
measures how often the rank-r candidate of depth d is the code finally emitted at that
position, then grows the tree greedily, each step adding the node with the largest
expected contribution to the accepted length (the product of the statistics along the
node's path), until the node budget N; depth is capped at K.

  measure_acceptance  acc[d][r] from traced TREE-mode frames of a probe tree
  grow_tree           the greedy growth (ties: the earlier-added parent, then the lower rank),
                      returned in the breadth-first order mcd_set_tree expects
"""
from __future__ import annotations

from typing import List, Sequence, Tuple

import numpy as np


def grow_tree(acc: Sequence[Sequence[float]], n_nodes: int) -> Tuple[List[int], List[int]]:
    """(parent, rank) of the greedy tree of at most n_nodes nodes; acc[d-1][r] is the
    probability that the rank-r candidate of depth d is the emitted code."""
    K = len(acc)
    nodes: List[Tuple[int, int, int, float]] = []        # (parent, rank, depth, value)
    n_children = {-1: 0}
    while len(nodes) < n_nodes:
        best = None
        for pa in range(-1, len(nodes)):
            d = 1 if pa < 0 else nodes[pa][2] + 1
            r = n_children.get(pa, 0)
            if d > K or r >= len(acc[d - 1]):
                continue
            v = (1.0 if pa < 0 else nodes[pa][3]) * float(acc[d - 1][r])
            if best is None or v > best[0]:
                best = (v, pa, r, d)
        if best is None:
            break
        v, pa, r, d = best
        nodes.append((pa, r, d, v))
        n_children[pa] = r + 1
        n_children[len(nodes) - 1] = 0

    def path(i):
        out = []
        while i >= 0:
            out.append(nodes[i][1])
            i = nodes[i][0]
        return out[::-1]

    order = sorted(range(len(nodes)), key=lambda i: (nodes[i][2], path(i)))
    new = {old: k for k, old in enumerate(order)}
    parent = [new[nodes[i][0]] if nodes[i][0] >= 0 else -1 for i in order]
    rank = [nodes[i][1] for i in order]
    return parent, rank


def probe_tree(depth: int, ranks: int) -> Tuple[List[int], List[int]]:
    """A tree whose every depth proposes `ranks` candidates (rank-0 spine with `ranks`
    children per spine node), at most 31 nodes: every (depth, rank) statistic is observed."""
    parent, rank = [], []
    spine = -1
    for d in range(depth):
        first = len(parent)
        for r in range(ranks):
            parent.append(spine)
            rank.append(r)
        spine = first
    assert len(parent) <= 31
    return parent, rank


def measure_acceptance(records, codes: Sequence[Sequence[int]], depth: int, ranks: int, n_pos: int):
    """acc[d-1][r] from traced frames: records[f] = list of (a', next_cand) per call of frame f
    (the candidates proposed for positions a'+1..), codes[f] = the frame's codes c1..c_P."""
    hits = np.zeros((depth, ranks))
    seen = np.zeros(depth)
    for recs, cds in zip(records, codes):
        for a_next, cand in recs:
            for d in range(1, min(depth, n_pos - a_next) + 1):
                c = cds[a_next + d - 1]
                seen[d - 1] += 1
                for r in range(min(ranks, len(cand[d - 1]))):
                    if cand[d - 1][r] == c:
                        hits[d - 1, r] += 1
    return (hits / np.maximum(seen, 1)[:, None]).tolist()
