"""Pins of oracle.tree (sparse tree drafting and verification, Sec. 2.2 and Fig. 2).

  * the attention mask of the figure's tree against the mask printed in Fig. 2
    (tests/golden/fig2_tree_mask.txt), and the figure's node labels against the
    per-depth candidate ranking;
  * a chain tree (one rank-0 node per depth) against the greedy-draft chain procedure of
    oracle.frame: identical codes, frame for frame;
  * losslessness: the exact law of tree decoding equals the autoregressive law on the tiny
    model (rationals), and sampled tree frames match that law (chi-square);
  * the greedy sparse-tree growth on a worked example and against brute force over all
    trees of a few nodes."""
import itertools
from collections import Counter
from fractions import Fraction

import numpy as np
import pytest

from conftest import read_golden
from paper_2609_37007_gb300.synth import DRAFT_GREEDY, TINY, make_frame, make_weights, weights_as_f32
from oracle.enumeration import PrefixModel, ar_distribution, tree_distribution
from oracle.frame import decode_frame
from oracle.model import Model
from oracle.tree import Tree, attention_mask, decode_frame_tree, expected_accepted, grow_tree, ranked

FIG2 = Tree(parent=[-1, -1, 0, 0, 1, 2, 4, 4], rank=[0, 1, 0, 1, 0, 0, 0, 1])


def test_fig2_mask_and_labels():
    want = []
    for line in read_golden("fig2_tree_mask.txt"):
        _, cols = line.split(":")
        want.append([int(c) for c in cols.split()])
    assert attention_mask(FIG2) == want
    # labels 1=t1 2=t2 3=t3 4=t4 5=t3 6=t5 7=t5 8=t6: every node of depth d and rank r shows
    # the rank-r candidate of depth d (t1, t2 | t3, t4 | t5, t6)
    labels = ["t1", "t2", "t3", "t4", "t3", "t5", "t5", "t6"]
    names = {(1, 0): "t1", (1, 1): "t2", (2, 0): "t3", (2, 1): "t4", (3, 0): "t5", (3, 1): "t6"}
    assert [names[(FIG2.depth[i], FIG2.rank[i])] for i in range(FIG2.n)] == labels


def test_ranked_order_and_ties():
    z = np.array([0.5, 2.0, 2.0, -1.0, 2.0, 1.5], dtype=np.float32)
    assert ranked(z, 4) == [1, 2, 4, 5]
    assert ranked(z, 1) == [1]


@pytest.mark.parametrize("K", [2, 3])
def test_chain_tree_equals_greedy_chain(K):
    cfg = TINY.replace(draft_len=K, n_pos=6)
    m = Model(cfg, weights_as_f32(cfg, make_weights(cfg)))
    for f in range(6):
        fr = make_frame(cfg, f)
        codes, calls = decode_frame_tree(m, fr, Tree.chain(K), stream=2, frame_idx=f)
        ref = decode_frame(m, fr, stream=2, frame_idx=f, draft_mode=DRAFT_GREEDY)
        assert codes == ref.codes, f
        assert len(calls) == ref.calls


SMALL = Tree(parent=[-1, -1, 0, 1], rank=[0, 1, 0, 0])


# the sizes of the paper's tree sweep (Fig. 4: N = 32 deployed, N = 64 the largest), grown
# greedily for rank-decreasing statistics: 8 candidates at depth 1, the rest at depth 2
_ACC = [[0.6 / (r + 1) ** 0.5 for r in range(8)] for _ in range(2)]


@pytest.mark.parametrize("tree", [SMALL, Tree(parent=[-1, -1, -1, 0], rank=[0, 1, 2, 0]), Tree.chain(2),
                                  grow_tree(_ACC, 32), grow_tree(_ACC, 64)],
                         ids=["small", "wide3", "chain2", "grown32", "grown64"])
def test_tree_law_equals_autoregressive_law(tree):
    cfg = TINY
    m = Model(cfg, weights_as_f32(cfg, make_weights(cfg)))
    fr = make_frame(cfg, 3)
    pm = PrefixModel(m, fr)
    ar = ar_distribution(pm, cfg.n_pos)
    law, calls = tree_distribution(pm, cfg.n_pos, tree)
    assert sum(law.values()) == 1
    assert set(law) <= set(ar)
    for seq, pr in ar.items():
        assert law.get(seq, Fraction(0)) == pr
    assert 1 < calls <= cfg.n_pos


def test_sampled_tree_frames_match_the_exact_law():
    cfg = TINY
    m = Model(cfg, weights_as_f32(cfg, make_weights(cfg)))
    fr = make_frame(cfg, 3)
    pm = PrefixModel(m, fr)
    ar = ar_distribution(pm, cfg.n_pos)
    n = 1200
    first = Counter()
    for i in range(n):
        codes, _ = decode_frame_tree(m, fr, SMALL, stream=5, frame_idx=10_000 + i)
        first[codes[0]] += 1
    marg = Counter()
    for seq, pr in ar.items():
        marg[seq[0]] += float(pr)
    chi2 = sum((first[x] - n * px) ** 2 / (n * px) for x, px in marg.items() if n * px > 0)
    dof = len(marg) - 1
    assert chi2 < dof + 6 * np.sqrt(2 * dof), chi2


def test_grow_tree_worked_example():
    acc = [[0.6, 0.2, 0.1], [0.5, 0.2], [0.4]]
    t = grow_tree(acc, 4)
    assert t.parent == [-1, -1, 0, 0] and t.rank == [0, 1, 0, 1]
    assert abs(expected_accepted(t, acc) - (0.6 + 0.2 + 0.3 + 0.12)) < 1e-12
    t6 = grow_tree(acc, 6)
    assert t6.n == 6 and t6.max_depth == 3


def _all_trees(n, K, m):
    """Every tree of n nodes whose children take consecutive ranks from 0 (depth <= K, rank < m)."""
    out = []

    def rec(parent, rank, depth):
        if len(parent) == n:
            out.append(Tree(parent=list(parent), rank=list(rank)))
            return
        for pa in [-1] + list(range(len(parent))):
            d = 1 if pa < 0 else depth[pa] + 1
            r = sum(1 for q in parent if q == pa)
            if d > K or r >= m:
                continue
            # canonical order: add nodes in nondecreasing (parent, rank) to avoid repeats
            if parent and (pa, r) < (parent[-1], rank[-1]):
                continue
            rec(parent + [pa], rank + [r], depth + [d])

    rec([], [], [])
    return out


def test_grow_tree_is_optimal_for_rank_decreasing_statistics():
    rng = np.random.default_rng(4)
    for _ in range(5):
        acc = [sorted(rng.uniform(0.05, 0.9, 3), reverse=True) for _ in range(3)]
        for n in (2, 3, 4, 5):
            best = max(expected_accepted(t, acc) for t in _all_trees(n, 3, 3))
            got = expected_accepted(grow_tree(acc, n), acc)
            assert abs(got - best) < 1e-12, (n, got, best)
