"""Sparse tree drafting and verification (Sec. 2.2, "Tree attention increases acceptance
rate" and "RVQ position aware offsets with sparse tree attention"; Fig. 2).
TEST INFRASTRUCTURE ONLY.

What the paper fixes: the drafter proposes the top m candidates at each of the K drafted
codebook positions and arranges them as a tree of depth K; the N tree nodes are packed,
with the committed prefix, into one query of N + 1 rows verified in one MultiCodeDecoder
call, each row attending only to its ancestors and itself (Fig. 2); verification applies
the standard acceptance rule with residual resampling along the tree; a sparse tree keeps
a subset of the paths and is grown greedily from per-depth, per-rank acceptance
statistics, each step adding the node with the largest expected contribution to the
accepted length, until the node budget N is reached (depth at most K).

Readings of what the paper leaves open (R-T1..R-T6):
  R-T1 a tree is a list of nodes in breadth-first order; node i has a parent (-1: a child
       of the call's first row) and a rank; depth = parent's depth + 1 <= K; siblings have
       distinct ranks.
  R-T2 the candidate of a node of depth d and rank r is the id of rank r in the draft
       logits z_d (fp32 logit descending, id ascending), z_d = LMH_{a'+d}(h_{a'} + b_d)
       of the row whose LM head emitted the call's last code (as in the chain drafter).
  R-T3 rows of a call: row 0 feeds the last emitted code c_a at position a + 1; node rows
       follow in tree order at position a + 1 + depth, fed while their code position
       a + depth < P (a node at code position P is tested but feeds no row).  A row attends
       to the committed positions 0..a, to row 0, to its ancestors and to itself (Fig. 2).
  R-T4 verification walks from row 0.  At a node with verify distribution p (its row's LM
       head) the children are tested in rank order; test i keeps candidate x with
       probability p'(x), p' being p without the candidates already rejected at this node
       (the acceptance rule for a one-hot draft distribution, whose residual is p' without
       x): U * (S - sum of rejected W) < 2^53 * W_x, U from counter (round, code position,
       purpose 1 for the first test, 0x10000 + i for test i >= 1).  A kept child becomes
       the current node; if every child is rejected, or the node has none, a code is drawn
       from p' with purpose 0 (residual / bonus) when a position is left, and the call ends.
  R-T5 the accepted path's keys and values become the committed cache at positions a+1..
       (row 0 and the kept nodes); the next call's row 0 is the last emitted code.
  R-T6 greedy construction from statistics acc[d][r] (probability that the rank-r
       candidate of depth d is the emitted code): a node's value is the product of acc
       along its path; from the empty tree, repeatedly add, among the next-rank children
       of the root and of every node of depth < K, the one of largest value (ties to the
       earlier-added parent, then the lower rank) until N nodes.
With every node of rank 0 and one child per depth the tree is the greedy-draft chain:
the first test of a node uses the chain's accept counter, so both procedures take the
same decisions (pinned in the tests).
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import Dict, List, Optional, Sequence, Tuple

import numpy as np

from paper_2609_37007_gb300.synth import FrameInput

from . import philox
from .frame import Sampling, to_f32
from .model import Model, rmsnorm, rope, silu
from .sampler import Dist, draw

PURPOSE_SIBLING = 0x10000          # + i: test i >= 1 at a tree node (R-T4)


@dataclass
class Tree:
    parent: List[int]
    rank: List[int]
    depth: List[int] = field(default_factory=list)

    def __post_init__(self):
        self.depth = []
        for i, (pa, r) in enumerate(zip(self.parent, self.rank)):
            assert pa < i, "nodes must be listed parents first"
            self.depth.append(1 if pa < 0 else self.depth[pa] + 1)
        for i in range(len(self.parent)):
            sib = [self.rank[j] for j in range(len(self.parent)) if self.parent[j] == self.parent[i]]
            assert len(sib) == len(set(sib)), "siblings need distinct ranks"

    @property
    def n(self) -> int:
        return len(self.parent)

    @property
    def max_depth(self) -> int:
        return max(self.depth) if self.depth else 0

    def children(self, node: int) -> List[int]:
        """Children of node (-1: of row 0) in rank order."""
        ch = [i for i in range(self.n) if self.parent[i] == node]
        return sorted(ch, key=lambda i: self.rank[i])

    def ancestors(self, node: int) -> List[int]:
        out = []
        while node >= 0:
            out.append(node)
            node = self.parent[node]
        return out[::-1]

    def ranks_needed(self) -> List[int]:
        """m_d: candidates needed at depth d (index d - 1)."""
        m = [0] * self.max_depth
        for d, r in zip(self.depth, self.rank):
            m[d - 1] = max(m[d - 1], r + 1)
        return m

    @staticmethod
    def chain(K: int) -> "Tree":
        return Tree(parent=[i - 1 for i in range(K)], rank=[0] * K)


def attention_mask(tree: Tree) -> List[List[int]]:
    """Fig. 2: row 0 is the committed prefix's last row, row 1 + i is node i; row i attends
    to the rows listed (its ancestors and itself)."""
    rows = [[0]]
    for i in range(tree.n):
        rows.append([0] + [1 + j for j in tree.ancestors(i)])
    return rows


def ranked(z: Sequence[float], m: int) -> List[int]:
    """R-T2: the m ids of largest fp32 logit, ties to the lower id."""
    z32 = np.asarray(z, dtype=np.float32)
    order = np.lexsort((np.arange(len(z32)), -z32.astype(np.float64)))
    return [int(i) for i in order[:m]]


# ---- model rows with an explicit key set (R-T3) --------------------------------------------
def tree_row(model: Model, kv: np.ndarray, n_prefix: int, anc: List[List[Tuple[np.ndarray, np.ndarray]]],
             x_in: np.ndarray, pos: int):
    """One row at RoPE position pos attending to cache positions 0..n_prefix-1, then to the
    keys / values of its ancestor rows (anc[t][l] = (k, v) of ancestor t at layer l), then
    to its own.  Returns (post-norm h, per-layer (k, v) of this row)."""
    c, w = model.cfg, model.w
    D, Hq, Hkv = c.head_dim, c.n_q_heads, c.n_kv_heads
    group = Hq // Hkv
    x = np.asarray(x_in, dtype=np.float64).copy()
    own = []
    for l in range(c.n_layers):
        p = f"layers.{l}."
        xn = rmsnorm(x, w[p + "attn_norm"], c.rms_eps)
        q = (w[p + "wq"] @ xn).reshape(Hq, D)
        k = (w[p + "wk"] @ xn).reshape(Hkv, D)
        v = (w[p + "wv"] @ xn).reshape(Hkv, D)
        if c.qk_norm:
            q = np.stack([rmsnorm(q[h], w[p + "q_norm"], c.rms_eps) for h in range(Hq)])
            k = np.stack([rmsnorm(k[h], w[p + "k_norm"], c.rms_eps) for h in range(Hkv)])
        q = rope(q, pos, c.rope_base)
        k = model.kv_store(rope(k, pos, c.rope_base))
        v = model.kv_store(v)
        own.append((k, v))
        o = np.empty((Hq, D))
        for h in range(Hq):
            g = h // group
            keys = [kv[l, 0, g, j] for j in range(n_prefix)] + [a[l][0][g] for a in anc] + [k[g]]
            vals = [kv[l, 1, g, j] for j in range(n_prefix)] + [a[l][1][g] for a in anc] + [v[g]]
            s = np.array([kk @ q[h] for kk in keys]) / math.sqrt(D)
            e = np.exp(s - s.max())
            e /= e.sum()
            o[h] = e @ np.stack(vals)
        x = x + w[p + "wo"] @ o.reshape(-1)
        xn = rmsnorm(x, w[p + "ffn_norm"], c.rms_eps)
        x = x + w[p + "wd"] @ (silu(w[p + "wg"] @ xn) * (w[p + "wu"] @ xn))
    return rmsnorm(x, w["final_norm"], c.rms_eps), own


# ---- verification walk (R-T4) ----------------------------------------------------------------
def remove(p: Dist, rejected: Sequence[int]) -> Dist:
    """p without the rejected ids (their weights set to zero; the order is kept)."""
    ids, W = list(p.ids), [0 if x in rejected else wv for x, wv in zip(p.ids, p.W)]
    return Dist(ids=ids, W=W, S=sum(W))


def test_child(p: Dist, rejected: Sequence[int], x: int, U: int) -> bool:
    """Keep x with probability p'(x): U * S' < 2^53 * W'_x (W'_x = 0 if x is not in p')."""
    pr = remove(p, rejected)
    wx = pr.weight(x)
    return wx > 0 and U * pr.S < (1 << 53) * wx


def sibling_purpose(i: int) -> int:
    return philox.PURPOSE_ACCEPT if i == 0 else PURPOSE_SIBLING + i


@dataclass
class TreeCall:
    rnd: int
    a: int
    rows: List[Tuple[int, int, int]]          # (node or -1, position, input id)
    cand: List[List[int]]                     # candidates used by this call's nodes
    path: List[int]                           # kept nodes
    emitted: List[int]
    draft_row: int                            # row whose drafts feed the next call
    next_cand: List[List[int]]
    verify_logits: Dict[int, np.ndarray] = field(default_factory=dict)   # row -> fp32 logits
    draft_logits: List[np.ndarray] = field(default_factory=list)


def walk(S: Sampling, rnd: int, a: int, P: int, tree: Tree, cand: List[List[int]],
         p_of_row, row_of_node: Dict[int, int]) -> Tuple[List[int], List[int], int]:
    """R-T4 from row 0.  Returns (emitted codes, kept nodes, row of the last visited node)."""
    emitted: List[int] = []
    path: List[int] = []
    node, row = -1, 0
    while True:
        s = a + 1 + len(path)                 # code position of the node's children
        p = p_of_row(row)
        rejected: List[int] = []
        kept = None
        for i, ch in enumerate([c for c in tree.children(node) if a + tree.depth[c] <= P]):
            x = cand[tree.depth[ch] - 1][tree.rank[ch]]
            if x in rejected:
                continue
            if test_child(p, rejected, x, S.u(rnd, s, sibling_purpose(i))):
                kept = (ch, x)
                break
            rejected.append(x)
        if kept is not None:
            ch, x = kept
            emitted.append(x)
            path.append(ch)
            if s == P:                         # the last code: nothing follows
                return emitted, path, row
            node, row = ch, row_of_node[ch]
            continue
        if s <= P:
            emitted.append(draw(remove(p, rejected), S.u(rnd, s, philox.PURPOSE_TARGET)))
        return emitted, path, row


def decode_frame_tree(model: Model, frame: FrameInput, tree: Tree, stream: int = 0, frame_idx: int = 0,
                      keep_logits: bool = False):
    """One frame of tree-drafted speculative decoding.  Returns (codes c1..c_P, calls)."""
    cfg = model.cfg
    P, K = cfg.n_pos, tree.max_depth
    assert K <= cfg.draft_len or K == 0
    S = Sampling(cfg, stream, frame_idx)
    m_need = tree.ranks_needed()
    kv = model.new_kv()
    codes: Dict[int, int] = {}
    calls: List[TreeCall] = []
    # first call: rows (cond, c0) at positions 0, 1 -- c1 from LM head 1 (plain AR)
    model.row(kv, np.asarray(frame.cond, dtype=np.float64), 0)
    h1 = model.row(kv, model.c0_row(frame.c0, frame.c0_emb), 1)
    lg1 = to_f32(model.verify_logits(1, h1))
    codes[1] = draw(S.dist(lg1), S.u(0, 1, philox.PURPOSE_TARGET))
    a = 1
    z = [to_f32(model.draft_logits(1, d, h1)) for d in range(1, min(K, P - a) + 1)]
    cand = [ranked(z[d], m_need[d]) for d in range(len(z))]
    rec = TreeCall(rnd=0, a=0, rows=[(-1, 0, -1), (-1, 1, -1)], cand=[], path=[], emitted=[codes[1]], draft_row=1,
                   next_cand=cand)
    if keep_logits:
        rec.verify_logits = {1: lg1}
        rec.draft_logits = z
    calls.append(rec)
    rnd = 1
    while a < P:
        # rows: 0 = c_a at position a + 1, then the nodes whose code position a + depth < P
        rows = [(-1, a + 1, codes[a])]
        row_of_node: Dict[int, int] = {}
        for i in range(tree.n):
            d = tree.depth[i]
            if a + d < P and d <= len(cand):
                row_of_node[i] = len(rows)
                rows.append((i, a + 1 + d, cand[d - 1][tree.rank[i]]))
        h: Dict[int, np.ndarray] = {}
        own: Dict[int, list] = {}
        h[0], own[0] = tree_row(model, kv, a + 1, [], model.code_row(a, codes[a]), a + 1)
        for r in range(1, len(rows)):
            node, pos, x = rows[r]
            anc = [own[0]] + [own[row_of_node[j]] for j in tree.ancestors(node)[:-1]]
            h[r], own[r] = tree_row(model, kv, a + 1, anc, model.code_row(pos - 1, x), pos)
        vl = {r: to_f32(model.verify_logits(rows[r][1], h[r])) for r in range(len(rows))}
        emitted, path, drow = walk(S, rnd, a, P, tree, cand, lambda r: S.dist(vl[r]), row_of_node)
        # R-T5: commit row 0 and the kept nodes at positions a + 1 ..
        for t, r in enumerate([0] + [row_of_node[n] for n in path if n in row_of_node]):
            for l in range(cfg.n_layers):
                kv[l, 0, :, a + 1 + t] = own[r][l][0]
                kv[l, 1, :, a + 1 + t] = own[r][l][1]
        for t, x in enumerate(emitted):
            codes[a + 1 + t] = x
        a_new = a + len(emitted)
        n_next = min(K, P - a_new)
        pos_d = rows[drow][1]
        z = [to_f32(model.draft_logits(pos_d, d, h[drow])) for d in range(1, n_next + 1)]
        nc = [ranked(z[d], m_need[d]) for d in range(n_next)]
        rec = TreeCall(rnd=rnd, a=a, rows=rows, cand=cand, path=path, emitted=emitted, draft_row=drow,
                       next_cand=nc)
        if keep_logits:
            rec.verify_logits = vl
            rec.draft_logits = z
        calls.append(rec)
        cand, a, rnd = nc, a_new, rnd + 1
    return [codes[i] for i in range(1, P + 1)], calls


# ---- greedy sparse-tree construction (R-T6) ----------------------------------------------------
def grow_tree(acc: Sequence[Sequence[float]], n_nodes: int) -> Tree:
    """acc[d-1][r]: probability that the rank-r candidate of depth d is the emitted code."""
    K = len(acc)
    parent: List[int] = []
    rank: List[int] = []
    value: List[float] = []
    depth: List[int] = []
    n_children = {-1: 0}
    while len(parent) < n_nodes:
        best = None
        for pa in [-1] + list(range(len(parent))):
            d = 1 if pa < 0 else depth[pa] + 1
            r = n_children.get(pa, 0)
            if d > K or r >= len(acc[d - 1]):
                continue
            v = (1.0 if pa < 0 else value[pa]) * acc[d - 1][r]
            if best is None or v > best[0]:
                best = (v, pa, r, d)
        if best is None:
            break
        v, pa, r, d = best
        parent.append(pa)
        rank.append(r)
        value.append(v)
        depth.append(d)
        n_children[pa] = r + 1
        n_children[len(parent) - 1] = 0
    # breadth-first order, siblings by rank
    order = sorted(range(len(parent)), key=lambda i: (depth[i], _path_key(parent, rank, i)))
    pos = {old: new for new, old in enumerate(order)}
    return Tree(parent=[pos[parent[i]] if parent[i] >= 0 else -1 for i in order], rank=[rank[i] for i in order])


def _path_key(parent, rank, i):
    key = []
    while i >= 0:
        key.append(rank[i])
        i = parent[i]
    return key[::-1]


def expected_accepted(tree: Tree, acc: Sequence[Sequence[float]]) -> float:
    """Sum over nodes of the product of acc along the path: the tree's expected number of
    kept drafts under independent per-depth acceptance (the quantity the growth maximises)."""
    val = []
    for i in range(tree.n):
        v = acc[tree.depth[i] - 1][tree.rank[i]]
        if tree.parent[i] >= 0:
            v *= val[tree.parent[i]]
        val.append(v)
    return float(sum(val))
