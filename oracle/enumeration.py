"""Exact output distributions of the autoregressive and speculative frame procedures.
TEST INFRASTRUCTURE ONLY.

The paper's correctness claim (Abstract; Sec. 3.2) is that the speculative decoder is
distributionally lossless under the deployed top-k sampling: the law of the emitted
codes c1..c_P equals the autoregressive law prod_s p_s(c_s | c_<s).  The sampler's
distributions are integer weights (oracle.sampler R-S2), so on a small model both laws
can be written out exactly as rationals (fractions.Fraction):

  * AR: product of the top-k/temperature probabilities along every sequence.
  * speculative: the procedure of oracle.frame, with every random choice replaced by
    its probability -- drafts d_j ~ q_j (independent, all from h_a + b_j), a draft kept
    with probability min(1, p(d)/q(d)), otherwise a residual code with probability
    r(x)/R, and a bonus code ~ p when every draft is kept.

Hidden states and distributions are memoised by code prefix: the row at sequence
position s depends only on c0 and c1..c_{s-1}.
"""
from __future__ import annotations

import itertools
from collections import defaultdict
from fractions import Fraction
from typing import Dict, Tuple

import numpy as np

from paper_2609_37007_gb300.synth import DRAFT_GREEDY, FrameInput

from .model import Model
from .sampler import Dist, greedy_dist, residual_weights, topk_dist


def to_f32(x) -> np.ndarray:
    return np.asarray(x, dtype=np.float64).astype(np.float32)


class PrefixModel:
    """h_s, p_s and the drafts of one frame input, memoised by code prefix."""

    def __init__(self, model: Model, frame: FrameInput, draft_mode: int = 0):
        self.m, self.frame, self.mode = model, frame, draft_mode
        self.k, self.T = model.cfg.top_k, model.cfg.temperature
        self._h: Dict[Tuple[int, ...], Tuple[np.ndarray, np.ndarray]] = {}
        self._p: Dict[Tuple[int, ...], Dist] = {}
        self._q: Dict[Tuple[Tuple[int, ...], int], Dist] = {}

    def state(self, prefix: Tuple[int, ...]):
        """(KV cache, h_s) after the rows up to position s = len(prefix) + 1."""
        if prefix not in self._h:
            if not prefix:
                kv = self.m.new_kv()
                self.m.row(kv, np.asarray(self.frame.cond, dtype=np.float64), 0)
                h = self.m.row(kv, self.m.c0_row(self.frame.c0, self.frame.c0_emb), 1)
            else:
                kv0, _ = self.state(prefix[:-1])
                kv = kv0.copy()
                s = len(prefix) + 1
                h = self.m.row(kv, self.m.code_row(s - 1, prefix[-1]), s)
            self._h[prefix] = (kv, h)
        return self._h[prefix]

    def target(self, prefix: Tuple[int, ...]) -> Dist:
        """p for c_{len(prefix)+1} given c1..c_len."""
        if prefix not in self._p:
            s = len(prefix) + 1
            self._p[prefix] = topk_dist(to_f32(self.m.verify_logits(s, self.state(prefix)[1])),
                                        self.k, self.T)
        return self._p[prefix]

    def draft(self, prefix: Tuple[int, ...], j: int) -> Dist:
        """q for c_{a+j} drafted from h_a, a = len(prefix) (prefix = c1..c_a)."""
        key = (prefix, j)
        if key not in self._q:
            a = len(prefix)
            h = self.state(prefix[:-1])[1]
            z = to_f32(self.m.draft_logits(a, j, h))
            self._q[key] = greedy_dist(z) if self.mode == DRAFT_GREEDY else \
                topk_dist(z, self.k, self.T)
        return self._q[key]


def ar_distribution(pm: PrefixModel, n_pos: int) -> Dict[Tuple[int, ...], Fraction]:
    out: Dict[Tuple[int, ...], Fraction] = {}

    def rec(prefix, pr):
        if len(prefix) == n_pos:
            out[prefix] = pr
            return
        p = pm.target(prefix)
        for x in p.ids:
            rec(prefix + (x,), pr * p.frac(x))

    rec((), Fraction(1))
    return out


def spec_distribution(pm: PrefixModel, n_pos: int, draft_len: int):
    """(law of c1..c_P, expected model calls per frame) of the speculative procedure."""
    memo: Dict[Tuple[int, ...], Tuple[Dict[Tuple[int, ...], Fraction], Fraction]] = {}

    def add(res, calls, head, sub, w):
        sub_law, sub_calls = sub
        for tail, pv in sub_law.items():
            res[head + tail] += w * pv
        return calls + w * sub_calls

    def from_state(prefix):
        """Law of the remaining codes and expected remaining calls, drafts pending."""
        if prefix in memo:
            return memo[prefix]
        a = len(prefix)
        res: Dict[Tuple[int, ...], Fraction] = defaultdict(Fraction)
        calls = Fraction(1)
        if a == n_pos:
            memo[prefix] = ({(): Fraction(1)}, Fraction(0))
            return memo[prefix]
        n_d = min(draft_len, n_pos - a)
        qs = [pm.draft(prefix, j) for j in range(1, n_d + 1)]
        for dt in itertools.product(*[q.ids for q in qs]):
            pr = Fraction(1)
            for q, d in zip(qs, dt):
                pr *= q.frac(d)
            cur = prefix
            for i in range(n_d):
                p, q, d = pm.target(cur), qs[i], dt[i]
                alpha = min(Fraction(1), p.frac(d) / q.frac(d))
                if alpha < 1:
                    xs, r, R = residual_weights(p, q)
                    for x, rx in zip(xs, r):
                        if rx > 0:
                            calls = add(res, calls, cur[a:] + (x,), from_state(cur + (x,)),
                                        pr * (1 - alpha) * Fraction(rx, R))
                pr *= alpha
                if pr == 0:
                    break
                cur = cur + (d,)
            else:
                if len(cur) < n_pos:
                    p = pm.target(cur)
                    for x in p.ids:
                        calls = add(res, calls, cur[a:] + (x,), from_state(cur + (x,)),
                                    pr * p.frac(x))
                else:
                    res[cur[a:]] += pr
        memo[prefix] = (dict(res), calls)
        return memo[prefix]

    # first call: rows (cond, c0), emits c1 from LM head 1 -- plain AR
    p1 = pm.target(())
    law: Dict[Tuple[int, ...], Fraction] = defaultdict(Fraction)
    calls = Fraction(1)
    for x in p1.ids:
        calls = add(law, calls, (x,), from_state((x,)), p1.frac(x))
    return dict(law), calls


def alpha(p: Dist, q: Dist) -> Fraction:
    """Acceptance probability of one draft: sum_x min(p(x), q(x))."""
    return sum((min(p.frac(x), q.frac(x)) for x in set(p.ids) | set(q.ids)), Fraction(0))


def tree_distribution(pm: PrefixModel, n_pos: int, tree, m_need=None):
    """(law of c1..c_P, expected calls) of tree-drafted decoding (oracle.tree, R-T1..R-T5),
    written with probabilities: at a node with target p and candidates x_1, x_2, .. (the
    node's children in rank order), test i keeps x_i with probability p(x_i) / (1 - sum of
    p over the candidates rejected before it); when none is kept a code is drawn from p
    restricted to the rejected candidates' complement, renormalised."""
    from .tree import ranked                               # the candidate ranking (R-T2)
    K = tree.max_depth
    m_need = tree.ranks_needed() if m_need is None else m_need
    memo: Dict[Tuple[int, ...], Tuple[Dict[Tuple[int, ...], Fraction], Fraction]] = {}

    def cands(prefix):
        a = len(prefix)
        h = pm.state(prefix[:-1])[1]
        out = []
        for d in range(1, min(K, n_pos - a) + 1):
            z = to_f32(pm.m.draft_logits(a, d, h))
            out.append(ranked(z, m_need[d - 1]))
        return out

    def from_state(prefix):
        if prefix in memo:
            return memo[prefix]
        a = len(prefix)
        if a == n_pos:
            memo[prefix] = ({(): Fraction(1)}, Fraction(0))
            return memo[prefix]
        cand = cands(prefix)
        res: Dict[Tuple[int, ...], Fraction] = defaultdict(Fraction)
        calls = [Fraction(1)]

        def visit(node, cur, pr):
            """Walk at `node` (-1: the call's first row) with codes `cur` emitted so far."""
            p = pm.target(cur)
            s = len(cur) + 1
            left = Fraction(1)
            rejected = []
            for ch in tree.children(node):
                if a + tree.depth[ch] > n_pos:
                    continue
                x = cand[tree.depth[ch] - 1][tree.rank[ch]]
                keep = p.frac(x) / left if left > 0 else Fraction(0)
                if keep > 0:
                    if s == n_pos:
                        res[cur[a:] + (x,)] += pr * keep
                    else:
                        visit(ch, cur + (x,), pr * keep)
                pr *= 1 - keep
                left -= p.frac(x)
                rejected.append(x)
                if pr == 0:
                    return
            if s > n_pos:
                res[cur[a:]] += pr
                return
            for x in p.ids:
                if x in rejected or p.frac(x) == 0:
                    continue
                w = pr * p.frac(x) / left
                sub_law, sub_calls = from_state(cur + (x,))
                for tail, pv in sub_law.items():
                    res[cur[a:] + (x,) + tail] += w * pv
                calls[0] += w * sub_calls

        visit(-1, prefix, Fraction(1))
        # a walk that ended by keeping the last position's code finishes the frame
        memo[prefix] = (dict(res), calls[0])
        return memo[prefix]

    p1 = pm.target(())
    law: Dict[Tuple[int, ...], Fraction] = defaultdict(Fraction)
    calls = Fraction(1)
    for x in p1.ids:
        sub_law, sub_calls = from_state((x,))
        for tail, pv in sub_law.items():
            law[(x,) + tail] += p1.frac(x) * pv
        calls += p1.frac(x) * sub_calls
    return dict(law), calls
