"""fp64 outer CodeDecoder and the full frame pipeline.  TEST INFRASTRUCTURE ONLY.

What the paper fixes (Sec. 1 and Fig. 1 with its caption): text-to-speech generation
runs one CodeDecoder call per 80 ms frame; that call emits the frame's seed code c0,
then the MultiCodeDecoder emits c1..c15 conditioned on it.  The next frame's CodeDecoder
input is the sum of the frame's text-token embedding and the embeddings of all 16 codes
of the frame before.  The CodeDecoder has 28 layers; its block is not described, so it
is the MultiCodeDecoder's block (readings R-M1..R-M6 of oracle.model).

Readings of what the paper leaves open (R-C1..R-C7):
  R-C1 positions are absolute over the utterance: the text prompt fills positions
       0..T-1 (one prefill), frame i >= 1 feeds one row at position T - 1 + i.
  R-C2 frame 0's c0 and MultiCodeDecoder input come from the last prompt row; after the
       prompt the text input of a frame is a zero (pad) vector unless a text id is given.
  R-C3 the input row of frame i >= 1 is t_i + E_c0(c0) + sum_{j=1..P} E_j(c_j) of frame
       i - 1, summed in that order; tables E_1..E_{P-1} are the MultiCodeDecoder's own
       code tables, E_P (never fed inside a frame) belongs to the outer model.
  R-C4 for bf16 models the KV cache holds K (after QK-norm and RoPE) and V rounded to
       bf16: fp64 -> fp32 (nearest) -> bf16 (nearest, ties to even); every read of a
       cached position, the row's own included, sees the rounded value.  fp32 models
       keep the values exactly.
  R-C5 c0 ~ top-k / temperature of the c0 logits fp32(W_c0 h) with the sampler of
       oracle.sampler, uniform from counter (stream, frame, round 0, position 0,
       purpose 0): position 0 is never used by a MultiCodeDecoder decision.
  R-C6 the MultiCodeDecoder receives cond = fp32(h) (post-final-norm hidden of the
       frame's CodeDecoder row) and the c0 embedding vector fp32(E_c0(c0)).
  R-C7 a batched prefill is the causal forward of all prompt rows at once; each row's
       result is the same function of its prefix as a row-by-row decode.
"""
from __future__ import annotations

import math
from dataclasses import dataclass
from typing import Dict, List, Optional, Sequence

import numpy as np

from paper_2609_37007_gb300.synth import WEIGHT_BF16, FrameInput, MCDConfig, OuterConfig

from . import philox
from .frame import FrameResult, decode_frame, to_f32
from .model import Model, rmsnorm, rope, silu
from .sampler import draw, topk_dist


def round_bf16(a) -> np.ndarray:
    """R-C4 rounding: fp64 -> fp32 (nearest) -> bf16 (nearest, ties to even), as fp64."""
    u = np.ascontiguousarray(np.asarray(a, dtype=np.float64).astype(np.float32)).view(np.uint32)
    keep = u >> np.uint32(16)
    rest = u & np.uint32(0xFFFF)
    up = (rest > np.uint32(0x8000)) | ((rest == np.uint32(0x8000)) & ((keep & np.uint32(1)) == np.uint32(1)))
    bits = (keep + up.astype(np.uint32)) << np.uint32(16)
    return bits.view(np.float32).astype(np.float64)


class CodeDecoder(Model):
    """The outer model: Model's block over an absolute-position KV cache (R-C1, R-C4)."""

    def __init__(self, cfg: OuterConfig, weights_f32: Dict[str, np.ndarray], inner: Model):
        big = {"text_embed"}
        super().__init__(cfg, {k: v for k, v in weights_f32.items() if k not in big})
        self.text = np.asarray(weights_f32["text_embed"], dtype=np.float32)   # rows widened on use
        self.inner = inner
        self.P = inner.cfg.n_pos

    def kv_store(self, v: np.ndarray) -> np.ndarray:
        return round_bf16(v) if self.cfg.weight_dtype == WEIGHT_BF16 else v

    def new_kv(self) -> np.ndarray:
        c = self.cfg
        return np.zeros((c.n_layers, 2, c.n_kv_heads, c.max_tokens, c.head_dim))

    # ---- inputs ------------------------------------------------------------------------
    def text_row(self, tid: int) -> np.ndarray:
        return self.text[int(tid)].astype(np.float64)

    def frame_input(self, codes: Sequence[int], text_id: int = -1) -> np.ndarray:
        """R-C3: codes = (c0, c1, ..., c_P) of the previous frame."""
        assert len(codes) == self.P + 1
        x = self.text_row(text_id) if text_id >= 0 else np.zeros(self.cfg.hidden)
        x = x + self.w["c0_embed"][int(codes[0])]
        for j in range(1, self.P):
            x = x + self.inner.code_row(j, int(codes[j]))
        return x + self.w[f"code_embed.{self.P}"][int(codes[self.P])]

    def c0_vector(self, c0: int) -> np.ndarray:
        return self.w["c0_embed"][int(c0)].copy()

    def c0_logits(self, h: np.ndarray) -> np.ndarray:
        return self.w["c0_head"] @ h

    # ---- batched prefill (R-C7) -----------------------------------------------------------
    def rows(self, kv: np.ndarray, X: np.ndarray, pos0: int) -> np.ndarray:
        """Rows X[n] at positions pos0 + n, causal among themselves and over the cache
        positions < pos0; writes their K/V; returns the post-norm hidden states."""
        c, w = self.cfg, self.w
        D, Hq, Hkv = c.head_dim, c.n_q_heads, c.n_kv_heads
        group = Hq // Hkv
        x = np.array(X, dtype=np.float64)
        n = x.shape[0]
        pos = np.arange(pos0, pos0 + n)
        for l in range(c.n_layers):
            p = f"layers.{l}."
            xn = np.stack([rmsnorm(r, w[p + "attn_norm"], c.rms_eps) for r in x])
            q = (xn @ w[p + "wq"].T).reshape(n, Hq, D)
            k = (xn @ w[p + "wk"].T).reshape(n, Hkv, D)
            v = (xn @ w[p + "wv"].T).reshape(n, Hkv, D)
            if c.qk_norm:
                q = np.stack([[rmsnorm(q[i, h], w[p + "q_norm"], c.rms_eps) for h in range(Hq)] for i in range(n)])
                k = np.stack([[rmsnorm(k[i, h], w[p + "k_norm"], c.rms_eps) for h in range(Hkv)] for i in range(n)])
            q = np.stack([rope(q[i], int(pos[i]), c.rope_base) for i in range(n)])
            k = np.stack([rope(k[i], int(pos[i]), c.rope_base) for i in range(n)])
            for i in range(n):
                kv[l, 0, :, pos[i]] = self.kv_store(k[i])
                kv[l, 1, :, pos[i]] = self.kv_store(v[i])
            o = np.empty((n, Hq, D))
            for h in range(Hq):
                g = h // group
                keys = kv[l, 0, g, : pos0 + n]                      # [keys, D]
                vals = kv[l, 1, g, : pos0 + n]
                s = q[:, h, :] @ keys.T / math.sqrt(D)              # [n, keys]
                s[np.arange(pos0 + n)[None, :] > pos[:, None]] = -np.inf
                a = np.exp(s - s.max(axis=1, keepdims=True))
                a /= a.sum(axis=1, keepdims=True)
                o[:, h, :] = a @ vals
            x = x + o.reshape(n, -1) @ w[p + "wo"].T
            xn = np.stack([rmsnorm(r, w[p + "ffn_norm"], c.rms_eps) for r in x])
            x = x + (silu(xn @ w[p + "wg"].T) * (xn @ w[p + "wu"].T)) @ w[p + "wd"].T
        return np.stack([rmsnorm(r, w["final_norm"], c.rms_eps) for r in x])


def sample_c0(cfg: OuterConfig, logits32: np.ndarray, stream: int, frame: int) -> int:
    """R-C5."""
    U = philox.uniform_int(cfg.sample_seed, stream, frame, 0, 0, philox.PURPOSE_TARGET)
    return draw(topk_dist(logits32, cfg.top_k, cfg.temperature), U)


@dataclass
class PipelineFrame:
    c0: int
    codes: List[int]               # c0, c1..c_P
    c0_logits: np.ndarray          # fp32 [c0_vocab]
    cond: np.ndarray               # fp32 [H] (R-C6)
    c0_emb: np.ndarray             # fp32 [H]
    inner: Optional[FrameResult]


class Pipeline:
    """One utterance: prompt prefill, then per frame CodeDecoder row -> c0 -> MultiCodeDecoder."""

    def __init__(self, outer: CodeDecoder, stream: int = 0):
        self.outer, self.stream = outer, stream
        self.kv = outer.new_kv()
        self.n_tok = 0
        self.frame = 0
        self.h: Optional[np.ndarray] = None

    def prefill(self, text_ids: Sequence[int]) -> np.ndarray:
        X = np.stack([self.outer.text_row(t) for t in text_ids])
        hs = self.outer.rows(self.kv, X, 0)
        self.n_tok = len(text_ids)
        self.h = hs[-1]
        return self.h

    def step(self, prev_codes: Sequence[int], text_id: int = -1) -> np.ndarray:
        """One CodeDecoder row for frame `self.frame` (>= 1) from the previous frame's codes."""
        x = self.outer.frame_input(prev_codes, text_id)
        self.h = self.outer.row(self.kv, x, self.n_tok)
        self.n_tok += 1
        return self.h

    def c0_of_current(self):
        lg = to_f32(self.outer.c0_logits(self.h))
        c0 = sample_c0(self.outer.cfg, lg, self.stream, self.frame)
        return c0, lg

    def run_frame(self, draft_len: Optional[int] = None, prev_codes=None, text_id: int = -1,
                  keep_logits: bool = False) -> PipelineFrame:
        """The current frame (prefill done; frames >= 1 first take their CodeDecoder row)."""
        if self.frame > 0:
            self.step(prev_codes, text_id)
        c0, lg = self.c0_of_current()
        cond, emb = to_f32(self.h), to_f32(self.outer.c0_vector(c0))
        res = decode_frame(self.outer.inner, FrameInput(cond=cond, c0=-1, c0_emb=emb), stream=self.stream,
                           frame_idx=self.frame, draft_len=draft_len, keep_logits=keep_logits)
        self.frame += 1
        return PipelineFrame(c0=c0, codes=[c0] + list(res.codes), c0_logits=lg, cond=cond, c0_emb=emb, inner=res)


def decode_utterance(outer: CodeDecoder, text_ids: Sequence[int], n_frames: int, stream: int = 0,
                     draft_len: Optional[int] = None) -> List[PipelineFrame]:
    pl = Pipeline(outer, stream)
    pl.prefill(text_ids)
    out: List[PipelineFrame] = []
    prev = None
    for _ in range(n_frames):
        fr = pl.run_frame(draft_len=draft_len, prev_codes=prev)
        prev = fr.codes
        out.append(fr)
    return out
