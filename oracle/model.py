"""fp64 MultiCodeDecoder, one sequence row at a time.  TEST INFRASTRUCTURE ONLY.

What the paper fixes (Sec. 1, Fig. 1; Sec. 2.1): the MultiCodeDecoder is a 5-layer
transformer run inside each 80 ms frame; code c_i is looked up in its own embedding
table i and the hidden state read by LM head i emits c_i; it restarts every frame from
the outer model's output.  The block internals are not in the paper; they follow the
Qwen3 decoder layer that Qwen3-TTS uses (readings R-M1..R-M6, stated here):

  R-M1 pre-norm block without biases:
         x += Wo * Attn(RoPE(QKnorm(Wq n(x), Wk n(x))), Wv n(x))
         x += Wd * (silu(Wg n'(x)) * (Wu n'(x)))
       n(x) = x / sqrt(mean(x^2) + eps) * gain (RMSNorm), silu(z) = z / (1 + e^-z).
  R-M2 optional per-head RMSNorm of q and k (gains shared by all heads), before RoPE.
  R-M3 RoPE rotate-half: angle_i = pos * base^(-2i/D), i < D/2;
       (a, b) -> (a cos - b sin, b cos + a sin) for the pair (v[i], v[i + D/2]).
  R-M4 sequence positions: 0 = conditioning vector, 1 = c0 embedding,
       s >= 2 = embedding of c_{s-1} in table s-1; reset every frame.
  R-M5 causal softmax attention, scale 1/sqrt(D), GQA: q head h reads kv head h // (Hq/Hkv).
  R-M6 the hidden state h_s read by LM head s is the final-RMSNorm output of row s.

Rows are processed one at a time against a KV cache indexed by position, so a row's
output depends only on the rows at lower positions: a verify call's rows equal the
autoregressive rows bit for bit inside this oracle.
"""
from __future__ import annotations

import math
from typing import Dict

import numpy as np

from paper_2609_37007_gb300.synth import MCDConfig


def rmsnorm(x: np.ndarray, gain: np.ndarray, eps: float) -> np.ndarray:
    return x / math.sqrt(float(np.mean(x * x)) + eps) * gain


def silu(z: np.ndarray) -> np.ndarray:
    return z / (1.0 + np.exp(-z))


def rope(v: np.ndarray, pos: int, base: float) -> np.ndarray:
    """R-M3 on a [heads, D] array."""
    D = v.shape[-1]
    half = D // 2
    i = np.arange(half, dtype=np.float64)
    ang = pos * np.power(base, -2.0 * i / D)
    c, s = np.cos(ang), np.sin(ang)
    a, b = v[..., :half], v[..., half:]
    return np.concatenate([a * c - b * s, b * c + a * s], axis=-1)


class Model:
    def __init__(self, cfg: MCDConfig, weights_f32: Dict[str, np.ndarray]):
        self.cfg = cfg
        self.w = {k: np.asarray(v, dtype=np.float64) for k, v in weights_f32.items()}

    # ---- inputs -------------------------------------------------------------------
    def c0_row(self, c0: int, c0_emb) -> np.ndarray:
        if self.cfg.c0_vocab > 0:
            return self.w["embed.0"][c0].copy()
        return np.asarray(c0_emb, dtype=np.float64).copy()

    def code_row(self, i: int, code: int) -> np.ndarray:
        """Embedding of code c_i (table i), the input of sequence position i+1."""
        return self.w[f"embed.{i}"][int(code)].copy()

    # ---- KV cache -----------------------------------------------------------------
    def new_kv(self) -> np.ndarray:
        c = self.cfg
        return np.zeros((c.n_layers, 2, c.n_kv_heads, c.n_pos + 2, c.head_dim))

    def kv_store(self, v: np.ndarray) -> np.ndarray:
        """Values as the KV cache keeps them (the MultiCodeDecoder's cache is exact)."""
        return v

    # ---- one row --------------------------------------------------------------------
    def row(self, kv: np.ndarray, x_in: np.ndarray, pos: int) -> np.ndarray:
        """Run the row at sequence position `pos`; writes its K/V, returns post-norm h."""
        c, w = self.cfg, self.w
        D, Hq, Hkv = c.head_dim, c.n_q_heads, c.n_kv_heads
        group = Hq // Hkv
        x = np.asarray(x_in, dtype=np.float64).copy()
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
            k = rope(k, pos, c.rope_base)
            kv[l, 0, :, pos] = self.kv_store(k)
            kv[l, 1, :, pos] = self.kv_store(v)
            o = np.empty((Hq, D))
            for h in range(Hq):
                g = h // group
                keys = kv[l, 0, g, : pos + 1]
                vals = kv[l, 1, g, : pos + 1]
                s = keys @ q[h] / math.sqrt(D)
                a = np.exp(s - s.max())
                a /= a.sum()
                o[h] = a @ vals
            x = x + w[p + "wo"] @ o.reshape(-1)
            xn = rmsnorm(x, w[p + "ffn_norm"], c.rms_eps)
            x = x + w[p + "wd"] @ (silu(w[p + "wg"] @ xn) * (w[p + "wu"] @ xn))
        return rmsnorm(x, w["final_norm"], c.rms_eps)

    # ---- heads ----------------------------------------------------------------------
    def verify_logits(self, P: int, h: np.ndarray) -> np.ndarray:
        """LMH_P(h_P): logits of c_P (fp64)."""
        return self.w[f"head.{P}"] @ h

    def draft_logits(self, P: int, j: int, h: np.ndarray) -> np.ndarray:
        """LMH_{P+j}(h_P + b_j): position-aware offset draft of c_{P+j} (Sec. 2.2, Fig. 3).

        With offsets forced to zero this is the reused-heads ablation (Table 2, row i)."""
        return self.w[f"head.{P + j}"] @ (h + self.w[f"offset.{j}"])
