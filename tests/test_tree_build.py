"""The library's greedy tree growth (paper_2609_37007_gb300.tree) against the oracle's
(oracle.tree.grow_tree, pinned against brute force), and the acceptance statistics on a
hand-made trace."""
import numpy as np

from paper_2609_37007_gb300 import tree as lt
from oracle.tree import Tree, expected_accepted, grow_tree


def test_grow_tree_matches_the_oracle():
    rng = np.random.default_rng(9)
    for _ in range(20):
        K = int(rng.integers(1, 5))
        acc = [list(np.sort(rng.uniform(0, 1, int(rng.integers(1, 8))))[::-1]) for _ in range(K)]
        for n in (1, 3, 8, 16, 31):
            parent, rank = lt.grow_tree(acc, n)
            ref = grow_tree(acc, n)
            assert (parent, rank) == (ref.parent, ref.rank), (acc, n)
            Tree(parent=parent, rank=rank)               # well formed (breadth-first, ranks distinct)


def test_probe_tree_observes_every_statistic():
    parent, rank = lt.probe_tree(3, 8)
    t = Tree(parent=parent, rank=rank)
    assert t.n == 24 and t.max_depth == 3 and t.ranks_needed() == [8, 8, 8]


def test_measure_acceptance_counts_hits():
    # frame codes c1..c4; after emitting c1 (a' = 1) the candidates for c2, c3 were proposed
    codes = [[5, 7, 9, 11]]
    records = [[(1, [[7, 1], [2, 9]]), (3, [[11, 4], [0, 0]])]]
    acc = lt.measure_acceptance(records, codes, depth=2, ranks=2, n_pos=4)
    # depth 1: 2 observations (c2 = 7 at rank 0, c4 = 11 at rank 0); depth 2: 1 (c3 = 9, rank 1)
    assert acc == [[1.0, 0.0], [0.0, 1.0]]
    assert abs(expected_accepted(Tree(*lt.grow_tree(acc, 2)), acc) - 1.0) < 1e-12
