"""Top-k / temperature sampling and the lossless acceptance rule.  TEST INFRASTRUCTURE ONLY.

The paper keeps the deployed top-k sampling of the model (Abstract; Sec. 3.1, "original
sampling configuration") and verifies drafts with the standard speculative acceptance
rule with residual resampling (Sec. 2.2 "Tree attention ..."; Sec. 3.2): a draft d drawn
from q is kept with probability min(1, p(d)/q(d)); otherwise a replacement is drawn from
max(0, p - q) renormalised.  The paper fixes no tie-breaks or summation orders, so this
module fixes them (readings R-S1..R-S7 of the design notes):

  R-S1 top-k set: sort by (fp32 logit descending, id ascending), keep the first k;
       k >= V keeps every id.
  R-S2 z = double(logit) / double(T); e_i = exp(z_i - z_max); S = sum of e in that order.
  R-S3 categorical draw with uniform u: first entry i (in the sorted order) with
       u*S < e_0 + ... + e_i (sequential fp64 sums).
  R-S4 accept test: u * q(d) < p(d), with p(x) = e_x / S and p(x) = 0 outside the top-k.
  R-S5 residual: r(x) = max(0, p(x) - q(x)) over p's support in ascending id order,
       R = sequential sum; draw the first x with u*R < r_1 + ... + r_x; R == 0 draws from p.
  R-S6 greedy drafts: q is one-hot at the first id of the sorted order.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import Dict, List, Sequence

import numpy as np


@dataclass
class Dist:
    """A top-k / temperature distribution: ids in sampling order, unnormalised weights."""
    ids: List[int]
    e: List[float]
    S: float
    index: Dict[int, int] = field(default_factory=dict)

    def __post_init__(self):
        if not self.index:
            self.index = {x: i for i, x in enumerate(self.ids)}

    def prob(self, x: int) -> float:
        i = self.index.get(int(x))
        return 0.0 if i is None else self.e[i] / self.S


def f32(x: float) -> float:
    return float(np.float32(x))


def topk_order(logits: Sequence[float], k: int) -> List[int]:
    """R-S1: ids sorted by (logit desc, id asc), truncated to k."""
    vals = [float(v) for v in np.asarray(logits, dtype=np.float32)]
    order = sorted(range(len(vals)), key=lambda i: (-vals[i], i))
    return order[: min(k, len(vals))]


def topk_dist(logits: Sequence[float], k: int, temperature: float) -> Dist:
    """R-S1, R-S2 on an fp32 logits row; the temperature is taken as its fp32 value."""
    l32 = np.asarray(logits, dtype=np.float32)
    ids = topk_order(l32, k)
    T = f32(temperature)
    z = [float(l32[i]) / T for i in ids]
    m = z[0]
    e = [math.exp(zi - m) for zi in z]
    S = 0.0
    for v in e:
        S += v
    return Dist(ids=ids, e=e, S=S)


def greedy_dist(logits: Sequence[float]) -> Dist:
    """R-S6: one-hot distribution on the top-1 id."""
    return Dist(ids=[topk_order(logits, 1)[0]], e=[1.0], S=1.0)


def draw(d: Dist, u: float) -> int:
    """R-S3: inverse-CDF draw over the sorted order."""
    t = u * d.S
    c = 0.0
    for x, v in zip(d.ids, d.e):
        c += v
        if t < c:
            return x
    return d.ids[-1]


def accept(p: Dist, q: Dist, d: int, u: float) -> bool:
    """R-S4: keep draft d iff u*q(d) < p(d) (probability min(1, p(d)/q(d)))."""
    return u * q.prob(d) < p.prob(d)


def residual_weights(p: Dist, q: Dist):
    """R-S5 weights: (ids ascending, r(x) = max(0, p(x) - q(x)), R)."""
    xs = sorted(p.ids)
    r = [max(0.0, p.prob(x) - q.prob(x)) for x in xs]
    R = 0.0
    for v in r:
        R += v
    return xs, r, R


def residual_draw(p: Dist, q: Dist, u: float) -> int:
    """R-S5: draw from normalise(max(0, p - q))."""
    xs, r, R = residual_weights(p, q)
    if R == 0.0:
        return draw(p, u)
    t = u * R
    c = 0.0
    last = xs[-1]
    for x, v in zip(xs, r):
        c += v
        if v > 0.0:
            last = x
        if t < c:
            return x
    return last
