"""Pins of oracle.model: RoPE/RMSNorm identities and a cross-check of the row-wise fp64
model against an independent batched formulation written with torch library routines
(F.rms_norm, scaled_dot_product_attention with a causal mask, F.silu)."""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from paper_2609_37007_gb300.synth import TINY, make_weights, weights_as_f32
from oracle.model import Model, rmsnorm, rope


def test_rope_identity_at_zero_and_norm_preserving():
    rng = np.random.default_rng(0)
    v = rng.standard_normal((3, 64))
    assert np.array_equal(rope(v, 0, 1e4), v)
    for pos in (1, 5, 16):
        assert np.allclose(np.linalg.norm(rope(v, pos, 1e4), axis=-1),
                           np.linalg.norm(v, axis=-1), rtol=1e-13)


def test_rope_scores_depend_on_relative_position_only():
    rng = np.random.default_rng(1)
    q, k = rng.standard_normal((1, 128)), rng.standard_normal((1, 128))
    s = [float(rope(q, m, 1e4)[0] @ rope(k, m - 3, 1e4)[0]) for m in (3, 7, 12)]
    assert np.allclose(s, s[0], rtol=1e-12)


def test_rope_pair_rotation_closed_form():
    v = np.zeros((1, 4))
    v[0, 0] = 1.0                                 # pair (v0, v2) with angle pos * base^0
    out = rope(v, 2, 10000.0)
    assert np.allclose(out[0], [math.cos(2), 0, math.sin(2), 0], atol=1e-15)


def test_rmsnorm_closed_form():
    x = np.array([3.0, 4.0])
    g = np.array([1.0, 2.0])
    r = math.sqrt((9 + 16) / 2 + 1e-6)
    assert np.allclose(rmsnorm(x, g, 1e-6), [3 / r, 8 / r], rtol=1e-15)


def _torch_reference(cfg, W, xs):
    """Batched causal forward of all rows at once, written with torch library calls."""
    t = {k: torch.tensor(v, dtype=torch.float64) for k, v in W.items()}
    x = torch.tensor(np.stack(xs), dtype=torch.float64)             # [S, H]
    S, D = x.shape[0], cfg.head_dim
    pos = torch.arange(S, dtype=torch.float64)
    inv = cfg.rope_base ** (-torch.arange(0, D, 2, dtype=torch.float64) / D)
    ang = pos[:, None] * inv[None, :]                                 # [S, D/2]
    cos, sin = torch.cos(ang), torch.sin(ang)

    def rot(v):                                                       # v [heads, S, D]
        a, b = v[..., : D // 2], v[..., D // 2:]
        return torch.cat([a * cos - b * sin, b * cos + a * sin], dim=-1)

    for l in range(cfg.n_layers):
        p = f"layers.{l}."
        xn = F.rms_norm(x, (cfg.hidden,), t[p + "attn_norm"], cfg.rms_eps)
        q = (xn @ t[p + "wq"].T).view(S, cfg.n_q_heads, D).transpose(0, 1)
        k = (xn @ t[p + "wk"].T).view(S, cfg.n_kv_heads, D).transpose(0, 1)
        v = (xn @ t[p + "wv"].T).view(S, cfg.n_kv_heads, D).transpose(0, 1)
        if cfg.qk_norm:
            q = F.rms_norm(q, (D,), t[p + "q_norm"], cfg.rms_eps)
            k = F.rms_norm(k, (D,), t[p + "k_norm"], cfg.rms_eps)
        q, k = rot(q), rot(k)
        rep = cfg.n_q_heads // cfg.n_kv_heads
        k, v = k.repeat_interleave(rep, 0), v.repeat_interleave(rep, 0)
        o = F.scaled_dot_product_attention(q[None], k[None], v[None], is_causal=True)[0]
        x = x + o.transpose(0, 1).reshape(S, -1) @ t[p + "wo"].T
        xn = F.rms_norm(x, (cfg.hidden,), t[p + "ffn_norm"], cfg.rms_eps)
        x = x + (F.silu(xn @ t[p + "wg"].T) * (xn @ t[p + "wu"].T)) @ t[p + "wd"].T
    return F.rms_norm(x, (cfg.hidden,), t["final_norm"], cfg.rms_eps).numpy()


@pytest.mark.parametrize("gqa", [False, True])
def test_rows_match_batched_torch_reference(gqa):
    cfg = TINY.replace(n_kv_heads=2) if gqa else TINY
    W = weights_as_f32(cfg, make_weights(cfg))
    m = Model(cfg, W)
    rng = np.random.default_rng(3)
    xs = [rng.standard_normal(cfg.hidden) for _ in range(cfg.n_pos + 2)]
    kv = m.new_kv()
    rows = np.stack([m.row(kv, x, s) for s, x in enumerate(xs)])
    ref = _torch_reference(cfg, W, xs)
    assert np.allclose(rows, ref, rtol=0, atol=1e-11)


def test_verify_rows_equal_autoregressive_rows_bitwise(tiny_model):
    m = tiny_model
    rng = np.random.default_rng(4)
    xs = [rng.standard_normal(m.cfg.hidden) for _ in range(6)]
    kv1, kv2 = m.new_kv(), m.new_kv()
    seq = [m.row(kv1, x, s) for s, x in enumerate(xs)]
    # stale rows at higher positions (rejected drafts) must not influence lower rows
    m.row(kv2, xs[0], 0)
    m.row(kv2, xs[1], 1)
    m.row(kv2, rng.standard_normal(m.cfg.hidden), 2)
    m.row(kv2, rng.standard_normal(m.cfg.hidden), 3)
    again = [m.row(kv2, xs[s], s) for s in range(2, 6)]
    for s in range(2, 6):
        assert np.array_equal(seq[s], again[s - 2])


def test_offsets_enter_only_the_draft_stream(tiny_model):
    m = tiny_model
    h = np.random.default_rng(5).standard_normal(m.cfg.hidden)
    assert np.array_equal(m.draft_logits(1, 1, h), m.w["head.2"] @ (h + m.w["offset.1"]))
    assert np.array_equal(m.verify_logits(2, h), m.w["head.2"] @ h)
