"""Autoregressive and speculative frame procedures.  TEST INFRASTRUCTURE ONLY.

Per 80 ms frame the MultiCodeDecoder emits c1..c_P (P = 15) after the outer model's
c0 (Sec. 1, Fig. 1).  Autoregressive decoding spends one model call per code.  The
speculative procedure (Sec. 2.2, Fig. 3) runs one call per round:

  * the call feeds the last emitted code c_a (table a, sequence position a+1) and the
    pending drafts d_{a+1..a+n} (tables a+1..a+n); row i reads LM head a+1+i, whose
    distribution p verifies draft d_{a+1+i} or, after the last draft, gives the bonus code;
  * drafts are tested in order with the acceptance rule (oracle.sampler.accept); the
    first rejection is replaced by a residual sample and ends the round; if every draft
    is kept a bonus code is drawn from the next row's p (when a position is left);
  * the hidden state h_{a'} that emitted the last code c_{a'} drafts the next round:
    LMH_{a'+j}(h_{a'} + b_j), j = 1..min(K, P - a');
  * the first call feeds the conditioning vector (position 0) and c0 (position 1) and
    emits c1 from LM head 1, which is exact autoregressive decoding (Fig. 3 caption).

Readings of what the paper leaves open (R-F1..R-F4):
  R-F1 rows per verify call = min(n_drafts + 1, P - a): no row is fed for a bonus past c_P.
  R-F2 round r uses counters (round r, position s, purpose); see oracle.philox.
  R-F3 NOISY_TARGET drafts (controlled-acceptance workload): q for position s is the
       target's own logits for s given the drafted prefix, plus sigma * N(0,1) per entry,
       rounded to fp32.  The target logits come from extra one-row passes on a copy of
       the KV cache, so sigma = 0 gives q = p and every draft is kept.
  R-F4 "tokens per call" = codes emitted / model calls, the first call included.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Dict, List, Optional, Sequence, Tuple

import numpy as np

from paper_2609_37007_gb300.synth import (DRAFT_GREEDY, DRAFT_NOISY_TARGET, DRAFT_SAMPLE,
                                          FrameInput, MCDConfig)

from . import philox
from .model import Model
from .sampler import (Dist, accept, draw, greedy_dist, residual_draw, topk_dist)


def to_f32(x) -> np.ndarray:
    return np.asarray(x, dtype=np.float64).astype(np.float32)


@dataclass
class RoundRecord:
    rnd: int
    a: int                          # codes emitted before this call
    positions: List[int]            # sequence positions of the rows fed
    input_ids: List[int]            # code fed at each row (-1: conditioning / c0 vector)
    drafts: List[int]               # drafts tested in this call (positions a+1..)
    n_acc: int
    emitted: List[int]
    next_drafts: List[int]
    verify_logits: Dict[int, np.ndarray] = field(default_factory=dict)   # pos -> fp32 row
    draft_logits: List[np.ndarray] = field(default_factory=list)          # fp32 rows


@dataclass
class FrameResult:
    codes: List[int]                # c1..c_P
    rounds: List[RoundRecord]

    @property
    def calls(self) -> int:
        return len(self.rounds)


class Sampling:
    """Sampling parameters plus the counter-based uniforms of one frame of one stream."""

    def __init__(self, cfg: MCDConfig, stream: int, frame_idx: int, draft_mode=None,
                 noise_sigma=None):
        self.k, self.T, self.seed = cfg.top_k, cfg.temperature, cfg.sample_seed
        self.stream, self.frame = stream, frame_idx
        self.mode = cfg.draft_mode if draft_mode is None else draft_mode
        self.sigma = cfg.noise_sigma if noise_sigma is None else noise_sigma

    def u(self, rnd: int, pos: int, purpose: int) -> int:
        """The 53-bit integer uniform of a decision (oracle.sampler R-S3..R-S5)."""
        return philox.uniform_int(self.seed, self.stream, self.frame, rnd, pos, purpose)

    def dist(self, logits) -> Dist:
        return topk_dist(logits, self.k, self.T)

    def noisy(self, logits32: np.ndarray, rnd: int, pos: int) -> np.ndarray:
        """R-F3: fp32(logit + sigma * n) with n from the Box-Muller pairs of (rnd, pos)."""
        out = np.empty(len(logits32), dtype=np.float32)
        for pair in range((len(logits32) + 1) // 2):
            n = philox.normal_pair(self.seed, self.stream, self.frame, rnd, pos, pair)
            for t in range(2):
                v = 2 * pair + t
                if v < len(logits32):
                    out[v] = np.float32(float(logits32[v]) + self.sigma * n[t])
        return out


def verify_round(S: Sampling, rnd: int, a: int, n_pos: int, p_rows: Sequence[np.ndarray],
                 drafts: Sequence[Tuple[int, Dist]]) -> Tuple[int, List[int]]:
    """Acceptance over one call.  p_rows[i] = fp32 logits of position a+1+i.

    Returns (accepted draft count, emitted codes)."""
    emitted: List[int] = []
    for i, (d, q) in enumerate(drafts):
        s = a + 1 + i
        p = S.dist(p_rows[i])
        if accept(p, q, d, S.u(rnd, s, philox.PURPOSE_ACCEPT)):
            emitted.append(int(d))
        else:
            emitted.append(residual_draw(p, q, S.u(rnd, s, philox.PURPOSE_TARGET)))
            return i, emitted
    s = a + 1 + len(drafts)
    if s <= n_pos:
        emitted.append(draw(S.dist(p_rows[len(drafts)]), S.u(rnd, s, philox.PURPOSE_TARGET)))
    return len(drafts), emitted


def sample_drafts(S: Sampling, rnd: int, a_new: int, z_rows: Sequence[np.ndarray]
                  ) -> List[Tuple[int, Dist]]:
    """Draft positions a_new+1.. from fp32 draft logits rows (SAMPLE / GREEDY / NOISY)."""
    out = []
    for j, z in enumerate(z_rows, start=1):
        q = greedy_dist(z) if S.mode == DRAFT_GREEDY else S.dist(z)
        out.append((draw(q, S.u(rnd, a_new + j, philox.PURPOSE_DRAFT)), q))
    return out


def decode_frame(model: Model, frame: FrameInput, stream: int = 0, frame_idx: int = 0,
                 draft_len: Optional[int] = None, draft_mode: Optional[int] = None,
                 noise_sigma: Optional[float] = None, keep_logits: bool = False,
                 zero_offsets: bool = False) -> FrameResult:
    """One frame of speculative decoding (draft_len = 0 is plain autoregressive decoding)."""
    cfg = model.cfg
    K = cfg.draft_len if draft_len is None else draft_len
    P = cfg.n_pos
    S = Sampling(cfg, stream, frame_idx, draft_mode, noise_sigma)
    kv = model.new_kv()
    codes: Dict[int, int] = {}
    a, rnd = 0, 0
    drafts: List[Tuple[int, Dist]] = []
    rounds: List[RoundRecord] = []
    while a < P:
        if rnd == 0:
            rows = [(0, -1, np.asarray(frame.cond, dtype=np.float64)),
                    (1, -1, model.c0_row(frame.c0, frame.c0_emb))]
        else:
            n_rows = min(len(drafts) + 1, P - a)                      # R-F1
            fed = [codes[a]] + [d for d, _ in drafts][: n_rows - 1]
            rows = [(a + 1 + i, int(c), model.code_row(a + i, c)) for i, c in enumerate(fed)]
        h = {pos: model.row(kv, x, pos) for pos, _, x in rows}
        p_rows = [to_f32(model.verify_logits(pos, h[pos])) for pos, _, _ in rows if pos >= 1]
        n_acc, emitted = verify_round(S, rnd, a, P, p_rows, drafts)
        for t, x in enumerate(emitted):
            codes[a + 1 + t] = x
        a_new = a + len(emitted)
        n_next = min(K, P - a_new)
        if S.mode == DRAFT_NOISY_TARGET:
            z_rows = _noisy_target_rows(model, S, kv, codes, rnd, a_new, n_next, h)
        elif zero_offsets:          # reused LM heads without offsets (Table 2, row i)
            z_rows = [to_f32(model.verify_logits(a_new + j, h[a_new]))
                      for j in range(1, n_next + 1)]
        else:
            z_rows = [to_f32(model.draft_logits(a_new, j, h[a_new]))
                      for j in range(1, n_next + 1)]
        new_drafts = sample_drafts(S, rnd, a_new, z_rows)
        rec = RoundRecord(rnd=rnd, a=a, positions=[r[0] for r in rows],
                          input_ids=[r[1] for r in rows], drafts=[d for d, _ in drafts],
                          n_acc=n_acc, emitted=list(emitted),
                          next_drafts=[d for d, _ in new_drafts])
        if keep_logits:
            rec.verify_logits = {pos: l for (pos, _, _), l in
                                 zip([r for r in rows if r[0] >= 1], p_rows)}
            rec.draft_logits = list(z_rows)
        rounds.append(rec)
        drafts, a, rnd = new_drafts, a_new, rnd + 1
    return FrameResult(codes=[codes[i] for i in range(1, P + 1)], rounds=rounds)


def _noisy_target_rows(model: Model, S: Sampling, kv: np.ndarray, codes: Dict[int, int],
                       rnd: int, a_new: int, n_next: int, h: Dict[int, np.ndarray]):
    """R-F3: target logits of the drafted positions from one-row passes on a KV copy.

    Draft j's distribution depends on draft j-1, so the drafts are drawn here one by
    one with the same counters sample_drafts would use; the rows returned reproduce
    them when fed to sample_drafts."""
    kv2 = kv.copy()
    prev = codes[a_new]
    rows = []
    for j in range(1, n_next + 1):
        s = a_new + j
        hs = model.row(kv2, model.code_row(s - 1, prev), s)
        z = S.noisy(to_f32(model.verify_logits(s, hs)), rnd, s)
        rows.append(z)
        prev = draw(S.dist(z), S.u(rnd, s, philox.PURPOSE_DRAFT))
    return rows
