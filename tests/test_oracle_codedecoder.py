"""Pins of oracle.codedecoder (outer CodeDecoder and frame pipeline, Fig. 1).

  * the batched prompt prefill against an independent torch formulation (library
    rms_norm, causal scaled_dot_product_attention, silu; RoPE as a complex rotation),
    with the bf16 KV rounding done by torch's own bfloat16 conversion;
  * a row-by-row decode of the same rows against the batched prefill;
  * the incremental pipeline (prefill, then one row per frame) against one causal
    forward over the whole token sequence;
  * the frame input sum on planted one-hot tables (exact integers);
  * the c0 counter (position 0) against every counter a MultiCodeDecoder frame uses."""
import numpy as np
import pytest
import torch
import torch.nn.functional as F

from paper_2609_37007_gb300.synth import (OUTER_TINY, TINY, WEIGHT_BF16, make_frame, make_outer_weights,
                                          make_prompt, make_weights, outer_weights_as_f32, weights_as_f32)
from oracle import philox
from oracle.codedecoder import CodeDecoder, Pipeline, decode_utterance, round_bf16, sample_c0
from oracle.frame import decode_frame
from oracle.model import Model
from oracle.sampler import draw, topk_dist


def _models(cfg=OUTER_TINY, inner_cfg=TINY):
    inner = Model(inner_cfg, weights_as_f32(inner_cfg, make_weights(inner_cfg)))
    W = outer_weights_as_f32(cfg, make_outer_weights(cfg, inner_cfg))
    return CodeDecoder(cfg, W, inner), W


def _torch_forward(cfg, W, X, kv_bf16):
    """Causal forward of all rows at positions 0..S-1 with torch library routines."""
    t = {k: torch.tensor(v, dtype=torch.float64) for k, v in W.items() if k != "text_embed"}
    x = torch.tensor(np.asarray(X), dtype=torch.float64)
    S, D = x.shape[0], cfg.head_dim
    inv = cfg.rope_base ** (-torch.arange(0, D, 2, dtype=torch.float64) / D)
    rot = torch.polar(torch.ones(S, D // 2, dtype=torch.float64),
                      torch.arange(S, dtype=torch.float64)[:, None] * inv[None, :])   # e^{i pos w}

    def rope(v):                       # pair (v_i, v_{i+D/2}) as the complex number v_i + i v_{i+D/2}
        z = torch.complex(v[..., : D // 2], v[..., D // 2:]) * rot
        return torch.cat([z.real, z.imag], dim=-1)

    def cache(v):
        return v.to(torch.float32).to(torch.bfloat16).to(torch.float64) if kv_bf16 else v

    for l in range(cfg.n_layers):
        p = f"layers.{l}."
        xn = F.rms_norm(x, (cfg.hidden,), t[p + "attn_norm"], cfg.rms_eps)
        q = (xn @ t[p + "wq"].T).view(S, cfg.n_q_heads, D).transpose(0, 1)
        k = (xn @ t[p + "wk"].T).view(S, cfg.n_kv_heads, D).transpose(0, 1)
        v = (xn @ t[p + "wv"].T).view(S, cfg.n_kv_heads, D).transpose(0, 1)
        if cfg.qk_norm:
            q = F.rms_norm(q, (D,), t[p + "q_norm"], cfg.rms_eps)
            k = F.rms_norm(k, (D,), t[p + "k_norm"], cfg.rms_eps)
        q, k, v = rope(q), cache(rope(k)), cache(v)
        rep = cfg.n_q_heads // cfg.n_kv_heads
        k, v = k.repeat_interleave(rep, 0), v.repeat_interleave(rep, 0)
        o = F.scaled_dot_product_attention(q[None], k[None], v[None], is_causal=True)[0]
        x = x + o.transpose(0, 1).reshape(S, -1) @ t[p + "wo"].T
        xn = F.rms_norm(x, (cfg.hidden,), t[p + "ffn_norm"], cfg.rms_eps)
        x = x + (F.silu(xn @ t[p + "wg"].T) * (xn @ t[p + "wu"].T)) @ t[p + "wd"].T
    return F.rms_norm(x, (cfg.hidden,), t["final_norm"], cfg.rms_eps).numpy()


@pytest.mark.parametrize("bf16", [False, True])
def test_prefill_matches_torch_formulation(bf16):
    cfg = OUTER_TINY.replace(weight_dtype=WEIGHT_BF16) if bf16 else OUTER_TINY
    oc, W = _models(cfg)
    X = np.stack([oc.text_row(t) for t in make_prompt(cfg)])
    hs = oc.rows(oc.new_kv(), X, 0)
    ref = _torch_forward(cfg, W, X, bf16)
    assert np.allclose(hs, ref, rtol=0, atol=1e-11)


def test_prefill_rows_equal_row_by_row_decode():
    cfg = OUTER_TINY.replace(weight_dtype=WEIGHT_BF16)
    oc, _ = _models(cfg)
    X = np.stack([oc.text_row(t) for t in make_prompt(cfg)])
    kv1, kv2 = oc.new_kv(), oc.new_kv()
    hs = oc.rows(kv1, X, 0)
    one = np.stack([oc.row(kv2, X[i], i) for i in range(len(X))])
    assert np.allclose(hs, one, rtol=0, atol=1e-12)
    assert np.allclose(kv1, kv2, rtol=0, atol=1e-12)


def test_bf16_cache_rounding_against_torch_and_ties():
    rng = np.random.default_rng(0)
    a = rng.standard_normal(4096) * 3.0
    ties = (np.arange(64, dtype=np.uint32) << np.uint32(16)) | np.uint32(0x3F808000)   # exact midpoints
    b = ties.view(np.float32).astype(np.float64)
    for v in (a, b):
        ref = torch.tensor(v).to(torch.float32).to(torch.bfloat16).to(torch.float64).numpy()
        assert np.array_equal(round_bf16(v), ref)
    # ties go to the even neighbour
    assert round_bf16(np.array([np.float32(1.0 + 2.0 ** -8)]))[0] == 1.0
    assert round_bf16(np.array([np.float32(1.0 + 3 * 2.0 ** -8)]))[0] == 1.0 + 2.0 ** -6


def test_pipeline_rows_equal_one_forward_over_the_whole_sequence():
    oc, W = _models()
    prompt = make_prompt(OUTER_TINY)
    pl = Pipeline(oc)
    h0 = pl.prefill(prompt)
    frames = [pl.run_frame()]
    hs = [h0]
    for _ in range(3):
        frames.append(pl.run_frame(prev_codes=frames[-1].codes))
        hs.append(pl.h)
    assert pl.n_tok == len(prompt) + 3
    X = [oc.text_row(t) for t in prompt] + [oc.frame_input(f.codes) for f in frames[:-1]]
    ref = _torch_forward(OUTER_TINY, W, np.stack(X), False)
    for i, h in enumerate(hs):
        assert np.allclose(h, ref[len(prompt) - 1 + i], rtol=0, atol=1e-11), i
    for f in frames:
        assert len(f.codes) == TINY.n_pos + 1 and 0 <= f.c0 < OUTER_TINY.c0_vocab
        assert np.array_equal(f.cond, np.asarray(f.cond, dtype=np.float32))


def test_frame_input_sum_on_planted_tables():
    oc, _ = _models()
    H, P = OUTER_TINY.hidden, TINY.n_pos
    oc.w["c0_embed"] = np.zeros_like(oc.w["c0_embed"])
    oc.w["c0_embed"][5, 0] = 1.0
    for j in range(1, P):
        oc.inner.w[f"embed.{j}"] = np.zeros_like(oc.inner.w[f"embed.{j}"])
        oc.inner.w[f"embed.{j}"][7 + j, j] = 10.0 ** j
    oc.w[f"code_embed.{P}"] = np.zeros_like(oc.w[f"code_embed.{P}"])
    oc.w[f"code_embed.{P}"][3, 0] = 1000.0
    oc.text = np.zeros_like(oc.text)
    oc.text[9, H - 1] = -2.0
    codes = [5] + [7 + j for j in range(1, P)] + [3]
    x = oc.frame_input(codes, text_id=9)
    want = np.zeros(H)
    want[0] = 1001.0
    for j in range(1, P):
        want[j] = 10.0 ** j
    want[H - 1] = -2.0
    assert np.array_equal(x, want)
    assert np.array_equal(oc.frame_input(codes), np.where(np.arange(H) == H - 1, 0.0, want))
    # a wrong code moves the row it reads: nothing else contributes
    codes2 = list(codes)
    codes2[2] = 0
    assert oc.frame_input(codes2, 9)[2] == 0.0


def test_c0_counter_is_outside_every_inner_counter(monkeypatch):
    seen = set()
    real = philox.uniform_int

    def spy(seed, stream, frame, rnd, pos, purpose):
        seen.add((stream, frame, rnd, pos, purpose))
        return real(seed, stream, frame, rnd, pos, purpose)

    monkeypatch.setattr(philox, "uniform_int", spy)
    oc, _ = _models()
    for K in (0, 2):
        for f in range(3):
            decode_frame(oc.inner, make_frame(TINY, f), stream=0, frame_idx=f, draft_len=K)
    assert seen and all(pos >= 1 for (_, _, _, pos, _) in seen)
    lg = np.random.default_rng(2).standard_normal(OUTER_TINY.c0_vocab).astype(np.float32)
    U = real(OUTER_TINY.sample_seed, 0, 4, 0, 0, philox.PURPOSE_TARGET)
    assert sample_c0(OUTER_TINY, lg, 0, 4) == draw(topk_dist(lg, OUTER_TINY.top_k, OUTER_TINY.temperature), U)


def test_utterance_is_deterministic_and_frames_chain():
    oc, _ = _models()
    a = decode_utterance(oc, make_prompt(OUTER_TINY), 3)
    b = decode_utterance(oc, make_prompt(OUTER_TINY), 3)
    assert [f.codes for f in a] == [f.codes for f in b]
    # the autoregressive inner loop (K = 0) keeps the same frame-0 c0 (drawn before it runs)
    c = decode_utterance(oc, make_prompt(OUTER_TINY), 1, draft_len=0)
    assert c[0].c0 == a[0].c0 and np.array_equal(c[0].c0_logits, a[0].c0_logits)
