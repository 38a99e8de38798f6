"""Top-k / temperature sampling and the lossless acceptance rule.  TEST INFRASTRUCTURE ONLY.

The paper keeps the deployed top-k sampling of the model (Abstract; Sec. 3.1, "original
sampling configuration") and verifies drafts with the standard speculative acceptance
rule with residual resampling (Sec. 2.2 "Tree attention ..."; Sec. 3.2): a draft d drawn
from q is kept with probability min(1, p(d)/q(d)); otherwise a replacement is drawn from
max(0, p - q) renormalised.  The paper fixes no arithmetic for this, so this module fixes
it (readings R-S1..R-S7, stated here).  Every distribution is a list of integer
weights, so that each decision is an exact rational comparison:

  R-S1 top-k set: sort by (fp32 logit descending, id ascending), keep the first k;
       k >= V keeps every id.  A distribution lists its set in ascending id order.
  R-S2 weights: z_i = fp32(logit_i) / fp32(T) and d_i = z_i - z_max in fp32,
       e_i = exp32(d_i) (below), W_i = floor(2^24 * e_i); S = sum of W.  The
       distribution is p(x) = W_x / S exactly (p(x) = 0 outside the top-k).
  R-S3 categorical draw with a 53-bit integer uniform U (u = U / 2^53): the first entry i
       in ascending id order with U * S < 2^53 * (W_0 + ... + W_i).
  R-S4 accept test: keep draft d iff U * Wq_d * S_p < 2^53 * Wp_d * S_q, i.e. u < p(d)/q(d).
  R-S5 residual: N_x = max(0, Wp_x * S_q - Wq_x * S_p) = S_p S_q max(0, p(x) - q(x)) over
       p's support in ascending id order, R = sum N; draw the first x with
       U * R < 2^53 * (N_1 + ... + N_x); R == 0 draws from p.
  R-S6 greedy drafts: q is one-hot at the largest logit, ties to the lowest id (W = [1]).
  R-S7 exp32: fp32 exponential by Cody and Waite's range reduction ("Software Manual for
       the Elementary Functions", 1980): n = rint(d * log2 e), r = (d - n*C1) - n*C2 with
       ln 2 = C1 + C2 split so that n*C1 is exact, then e^r by the degree-7 Taylor
       polynomial (Horner, one fp32 rounding per multiply and per add, no fused
       multiply-add), then * 2^n; d < -87 gives 0.  Both implementations perform the same
       IEEE single-precision operations, so their weights agree bit for bit.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from fractions import Fraction
from typing import Dict, List, Sequence

import numpy as np

F32 = np.float32
WEIGHT_BITS = 24
LOG2E = F32(1.4426950408889634)
LN2_C1 = F32(0.693359375)              # 9 significant bits: n * C1 is exact for |n| < 2^15
LN2_C2 = F32(-2.12194440e-4)           # ln 2 - C1 (rounded to fp32)
EXP_CUTOFF = F32(-87.0)
TAYLOR = [F32(1.0 / math.factorial(k)) for k in range(7, -1, -1)]   # Horner order: 1/7! .. 1/0!


def exp32(d) -> np.float32:
    """R-S7 on an fp32 argument d <= 0."""
    d = F32(d)
    if d < EXP_CUTOFF:
        return F32(0.0)
    n = np.rint(d * LOG2E)
    r = (d - n * LN2_C1) - n * LN2_C2
    p = TAYLOR[0]
    for c in TAYLOR[1:]:
        p = p * r + c
    return p * F32(2.0 ** int(n))


@dataclass
class Dist:
    """A top-k / temperature distribution: ids in draw order, integer weights W, S = sum W."""
    ids: List[int]
    W: List[int]
    S: int = 0
    index: Dict[int, int] = field(default_factory=dict)

    def __post_init__(self):
        if not self.S:
            self.S = sum(self.W)
        if not self.index:
            self.index = {x: i for i, x in enumerate(self.ids)}

    def weight(self, x: int) -> int:
        i = self.index.get(int(x))
        return 0 if i is None else self.W[i]

    def frac(self, x: int) -> Fraction:
        return Fraction(self.weight(x), self.S)

    def prob(self, x: int) -> float:
        return self.weight(x) / self.S


def topk_order(logits: Sequence[float], k: int) -> List[int]:
    """R-S1: ids sorted by (logit desc, id asc), truncated to k."""
    vals = [float(v) for v in np.asarray(logits, dtype=np.float32)]
    order = sorted(range(len(vals)), key=lambda i: (-vals[i], i))
    return order[: min(k, len(vals))]


def topk_dist(logits: Sequence[float], k: int, temperature: float) -> Dist:
    """R-S1, R-S2 on an fp32 logits row; the temperature is taken as its fp32 value."""
    l32 = np.asarray(logits, dtype=np.float32)
    top = topk_order(l32, k)
    T = F32(temperature)
    z_max = l32[top[0]] / T
    ids = sorted(top)
    W = [int(math.floor(float(exp32(l32[i] / T - z_max)) * 2.0 ** WEIGHT_BITS)) for i in ids]
    return Dist(ids=ids, W=W)


def greedy_dist(logits: Sequence[float]) -> Dist:
    """R-S6: one-hot distribution on the top-1 id."""
    return Dist(ids=[topk_order(logits, 1)[0]], W=[1])


def draw(d: Dist, U: int) -> int:
    """R-S3: inverse-CDF draw over the listed order with a 53-bit integer uniform."""
    lhs = U * d.S
    c = 0
    for x, w in zip(d.ids, d.W):
        c += w
        if lhs < (c << 53):
            return x
    return d.ids[-1]


def accept(p: Dist, q: Dist, d: int, U: int) -> bool:
    """R-S4: keep draft d iff u < p(d)/q(d) (probability min(1, p(d)/q(d)))."""
    return U * q.weight(d) * p.S < (p.weight(d) * q.S) << 53


def residual_weights(p: Dist, q: Dist):
    """R-S5 weights: (p's ids in its listed order, N_x, R), N_x / R = normalise(max(0, p - q))."""
    xs = list(p.ids)
    n = [max(0, p.weight(x) * q.S - q.weight(x) * p.S) for x in xs]
    return xs, n, sum(n)


def residual_draw(p: Dist, q: Dist, U: int) -> int:
    """R-S5: draw from normalise(max(0, p - q))."""
    xs, n, R = residual_weights(p, q)
    if R == 0:
        return draw(p, U)
    lhs = U * R
    c = 0
    last = xs[-1]
    for x, v in zip(xs, n):
        c += v
        if v > 0:
            last = x
        if lhs < (c << 53):
            return x
    return last
