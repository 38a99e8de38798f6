"""Training the RVQ-position-aware draft offsets b_1..b_K on synthetic teacher-forced data
(Sec. 2.2, "RVQ position aware offsets"; Table 2).

The paper keeps the MultiCodeDecoder backbone and its per-position LM heads frozen and learns
one hidden-size vector b_j per lookahead j: the draft of position k + j reads
LMH_{k+j}(h_k + b_j), where h_k is the post-norm hidden state whose head emitted c_k.  The
offsets are fitted by the cross-entropy of those draft logits against the code c_{k+j} the
target actually emitted, teacher-forced (h_k comes from the frozen model run on the true
prefix).  The paper trains on speech data and a trained Qwen3-TTS model; here the same
procedure runs on a synthetic random-init model, so only the procedure (not the paper's
numbers) is reproduced.

Steps:
  1. codes: frames decoded by the library (mcd_decode_frame: whatever the draft length, the
     emitted codes follow the target's top-k law);
  2. hidden states: one batched causal forward of the frozen model over the rows
     [cond, c0, c_1 .. c_{P-2}] of every frame (PyTorch, fp32) -- a training tool, not the
     decode path, which runs only in the library's kernels;
  3. training: Adam on b_j only.  The draft logits are linear in b_j,
     LMH_P (h + b) = LMH_P h + LMH_P b, so LMH_P h of every (frame, k, j) sample is computed
     once and each step adds LMH_P b_j;  the loss is the mean cross-entropy of
     softmax(z / T) (T = the sampling temperature) against c_{k+j};
  4. evaluation: the learned offsets loaded into a library context, tokens per verify call
     measured on frames not used for training, against the initial (random) offsets.
"""
from __future__ import annotations

import argparse
import json
import math
from typing import Dict, List, Optional, Tuple

import numpy as np

from .synth import (CONFIGS, MCD, WEIGHT_BF16, WEIGHT_INT8, MCDConfig, make_frames, make_weights,
                    round_to_bf16_bits, weights_as_f32)


# ---- 2. teacher-forced hidden states of the frozen model ---------------------------------
def _rmsnorm(x, gain, eps):
    import torch
    return x * torch.rsqrt((x * x).mean(dim=-1, keepdim=True) + eps) * gain


def _rope(v, base: float):
    """Rotate-half RoPE of v [N, S, heads, D] at sequence positions 0..S-1."""
    import torch
    S, D = v.shape[1], v.shape[-1]
    half = D // 2
    i = torch.arange(half, dtype=v.dtype, device=v.device)
    pos = torch.arange(S, dtype=v.dtype, device=v.device)
    ang = pos[:, None] * torch.pow(torch.tensor(base, dtype=v.dtype, device=v.device), -2.0 * i / D)[None, :]
    c, s = torch.cos(ang)[None, :, None, :], torch.sin(ang)[None, :, None, :]
    a, b = v[..., :half], v[..., half:]
    return torch.cat([a * c - b * s, b * c + a * s], dim=-1)


def input_rows(cfg: MCDConfig, w: Dict[str, "object"], cond, c0, c0_emb, codes, n_rows: Optional[int] = None):
    """Rows [N, n_rows] fed at sequence positions 0..n_rows-1 of a teacher-forced frame
    (default n_rows = P, the rows whose hidden states draft): the conditioning vector, the c0
    embedding (table 0 or the given vector), then code c_s from table s at position s + 1."""
    import torch
    S = cfg.n_pos if n_rows is None else n_rows
    rows = [cond]
    rows.append(w["embed.0"][c0.long()] if cfg.c0_vocab > 0 else c0_emb)
    for s in range(1, S - 1):
        rows.append(w[f"embed.{s}"][codes[:, s - 1].long()])
    return torch.stack(rows[:S], dim=1)


def teacher_forced_hidden(cfg: MCDConfig, w: Dict[str, "object"], x):
    """Post-final-norm hidden states h [N, S, H] of the frozen model on input rows x [N, S, H]
    (causal; pre-norm blocks with QK-norm, rotate-half RoPE and grouped-query attention, the
    block the library runs).  h[:, s] is what LM head s reads."""
    import torch
    N, S, H = x.shape
    D, Hq, Hkv = cfg.head_dim, cfg.n_q_heads, cfg.n_kv_heads
    mask = torch.ones(S, S, dtype=torch.bool, device=x.device).tril()
    for l in range(cfg.n_layers):
        p = f"layers.{l}."
        xn = _rmsnorm(x, w[p + "attn_norm"], cfg.rms_eps)
        q = (xn @ w[p + "wq"].T).view(N, S, Hq, D)
        k = (xn @ w[p + "wk"].T).view(N, S, Hkv, D)
        v = (xn @ w[p + "wv"].T).view(N, S, Hkv, D)
        if cfg.qk_norm:
            q = _rmsnorm(q, w[p + "q_norm"], cfg.rms_eps)
            k = _rmsnorm(k, w[p + "k_norm"], cfg.rms_eps)
        q, k = _rope(q, cfg.rope_base), _rope(k, cfg.rope_base)
        g = Hq // Hkv
        k, v = k.repeat_interleave(g, dim=2), v.repeat_interleave(g, dim=2)
        s = torch.einsum("nqhd,nkhd->nhqk", q, k) / math.sqrt(D)
        s = s.masked_fill(~mask, float("-inf"))
        o = torch.einsum("nhqk,nkhd->nqhd", torch.softmax(s, dim=-1), v).reshape(N, S, Hq * D)
        x = x + o @ w[p + "wo"].T
        xn = _rmsnorm(x, w[p + "ffn_norm"], cfg.rms_eps)
        gate, up = xn @ w[p + "wg"].T, xn @ w[p + "wu"].T
        x = x + (gate * torch.sigmoid(gate) * up) @ w[p + "wd"].T
    return _rmsnorm(x, w["final_norm"], cfg.rms_eps)


def torch_weights(cfg: MCDConfig, weights: Dict[str, np.ndarray], device, dtype=None):
    """The weights as tensors of the values they represent (bf16 widened exactly)."""
    import torch
    dt = torch.float32 if dtype is None else dtype
    return {k: torch.from_numpy(np.asarray(v, dtype=np.float32)).to(device=device, dtype=dt)
            for k, v in weights_as_f32(cfg, weights).items()}


# ---- 3. training samples, loss and Adam -------------------------------------------------
class OffsetSamples:
    """Every (frame n, source position k, lookahead j) with k + j <= P: the frozen logits
    LMH_{k+j} h_k (base [m, V]), the head index k + j and the target code c_{k+j}."""

    def __init__(self, cfg: MCDConfig, w: Dict[str, "object"], h, codes, K: int):
        import torch
        P, N = cfg.n_pos, h.shape[0]
        self.cfg, self.K = cfg, K
        self.blocks: List[Tuple[int, int]] = []               # (head P = k + j, offset j), N rows each
        bases, targets = [], []
        for k in range(1, P):
            for j in range(1, min(K, P - k) + 1):
                self.blocks.append((k + j, j))
                bases.append(h[:, k] @ w[f"head.{k + j}"].T)     # [N, V]
                targets.append(codes[:, k + j - 1].long())
        self.n = N
        self.base = torch.cat(bases)
        self.target = torch.cat(targets)
        self.w_heads = {Ph: w[f"head.{Ph}"] for Ph, _ in self.blocks}

    def loss(self, b):
        """Mean cross-entropy of softmax((LMH_P h_k + LMH_P b_j) / T) against c_{k+j}; b [K, H]."""
        import torch
        T = float(self.cfg.temperature)
        shift = torch.cat([(self.w_heads[Ph] @ b[j - 1]).expand(self.n, -1) for Ph, j in self.blocks])
        return torch.nn.functional.cross_entropy((self.base + shift) / T, self.target)


def train_offsets(samples: OffsetSamples, b0, steps: int = 300, lr: float = 1e-3):
    """Adam on the offsets only (the backbone and the heads stay frozen).  Returns the
    trained offsets [K, H] and the loss before each step plus after the last."""
    import torch
    b = b0.clone().detach().requires_grad_(True)
    opt = torch.optim.Adam([b], lr=lr)
    hist = []
    for _ in range(steps):
        opt.zero_grad()
        loss = samples.loss(b)
        hist.append(float(loss.detach()))
        loss.backward()
        opt.step()
    with torch.no_grad():
        hist.append(float(samples.loss(b)))
    return b.detach(), hist


def offsets_of(cfg: MCDConfig, weights: Dict[str, np.ndarray]) -> np.ndarray:
    """The offsets b_1..b_K stored in a weight dictionary, as float32 [K, H]."""
    w = weights_as_f32(cfg, {f"offset.{j}": weights[f"offset.{j}"] for j in range(1, cfg.draft_len + 1)})
    return np.stack([w[f"offset.{j}"] for j in range(1, cfg.draft_len + 1)]).astype(np.float32)


def with_offsets(cfg: MCDConfig, weights: Dict[str, np.ndarray], b: np.ndarray) -> Dict[str, np.ndarray]:
    """A copy of the weight dictionary whose offsets are b [K, H] (rounded to bf16 for bf16
    models, the precision the library loads them in)."""
    out = dict(weights)
    for j in range(1, cfg.draft_len + 1):
        v = np.asarray(b[j - 1], dtype=np.float32)
        out[f"offset.{j}"] = round_to_bf16_bits(v) if cfg.weight_dtype in (WEIGHT_BF16, WEIGHT_INT8) else v
    return out


# ---- 1. and 4. frames decoded by the library --------------------------------------------
def decode_codes(cfg: MCDConfig, weights: Dict[str, np.ndarray], n: int, first: int, stream_id: int = 0):
    """n frames (inputs first .. first + n - 1) decoded by the library: frame inputs, codes
    [n, P] and the per-frame stats [n, 8] (calls, codes, drafted, accepted, status, ...)."""
    import torch
    from . import mcd
    dev = torch.device("cuda", torch.cuda.current_device())
    cond_h, c0_h, emb_h = make_frames(cfg, n, first=first)
    cond = torch.from_numpy(cond_h).to(dev)
    c0 = torch.from_numpy(c0_h).to(dev)
    emb = torch.from_numpy(emb_h).to(dev) if emb_h is not None else None
    codes = torch.zeros((n, cfg.n_pos), dtype=torch.int32, device=dev)
    stats = torch.zeros((n, 8), dtype=torch.int32, device=dev)
    dec = mcd.Decoder(cfg, weights)
    try:
        for i in range(n):
            mcd.mcd_decode_frame(dec.ctx, stream_id, first + i, cond[i], c0[i:i + 1] if cfg.c0_vocab else None,
                                 emb[i] if emb is not None else None, codes[i], stats[i])
        mcd.mcd_sync(dec.ctx)
    finally:
        dec.close()
    st = stats.cpu().numpy()
    if (st[:, 4] != 0).any():
        raise RuntimeError("a frame failed on the device")
    return (cond_h, c0_h, emb_h), codes.cpu().numpy(), st


def tokens_per_call(stats: np.ndarray) -> float:
    """Codes emitted per model call over whole frames (the first call, which emits c1, included)."""
    return float(stats[:, 1].sum() / stats[:, 0].sum())


def fit(cfg: MCDConfig, weights: Dict[str, np.ndarray], train_frames: int, steps: int, lr: float = 1e-3,
        first: int = 5_000_000, device=None):
    """Steps 1-3: decode train_frames frames with the current offsets, teacher-force the frozen
    model on their codes and train the offsets.  Returns (b [K, H] float32, loss history)."""
    import torch
    dev = device or torch.device("cuda", torch.cuda.current_device())
    (cond_h, c0_h, emb_h), codes, _ = decode_codes(cfg, weights, train_frames, first)
    w = torch_weights(cfg, weights, dev)
    with torch.no_grad():
        x = input_rows(cfg, w, torch.from_numpy(cond_h).to(dev), torch.from_numpy(c0_h).to(dev),
                       torch.from_numpy(emb_h).to(dev) if emb_h is not None else None,
                       torch.from_numpy(codes).to(dev))
        h = teacher_forced_hidden(cfg, w, x)
        samples = OffsetSamples(cfg, w, h, torch.from_numpy(codes).to(dev), cfg.draft_len)
    b0 = torch.from_numpy(offsets_of(cfg, weights)).to(dev)
    b, hist = train_offsets(samples, b0, steps=steps, lr=lr)
    return b.cpu().numpy(), hist


def main(argv=None):
    ap = argparse.ArgumentParser(description="train the draft offsets b_j on synthetic teacher-forced frames "
                                             "and measure tokens per call before and after")
    ap.add_argument("--config", default=MCD.name, choices=sorted(CONFIGS))
    ap.add_argument("--train-frames", type=int, default=1000)
    ap.add_argument("--eval-frames", type=int, default=1000)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--lr", type=float, default=1e-3)
    args = ap.parse_args(argv)
    cfg = CONFIGS[args.config]
    weights = make_weights(cfg)
    b, hist = fit(cfg, weights, args.train_frames, args.steps, args.lr)
    _, _, st0 = decode_codes(cfg, weights, args.eval_frames, 6_000_000, stream_id=1)
    _, _, st1 = decode_codes(cfg, with_offsets(cfg, weights, b), args.eval_frames, 6_000_000, stream_id=1)
    print(json.dumps({"offsets": "teacher-forced cross-entropy of LMH_{k+j}(h_k + b_j) against c_{k+j}, Adam",
                      "config": cfg.name, "train_frames": args.train_frames, "steps": args.steps, "lr": args.lr,
                      "loss_initial": hist[0], "loss_trained": hist[-1],
                      "eval_frames": args.eval_frames,
                      "tokens_per_call_initial_offsets": tokens_per_call(st0),
                      "tokens_per_call_trained_offsets": tokens_per_call(st1),
                      "accepted_per_draft_initial": float(st0[:, 3].sum() / max(1, st0[:, 2].sum())),
                      "accepted_per_draft_trained": float(st1[:, 3].sum() / max(1, st1[:, 2].sum())),
                      "offset_norms": [float(np.linalg.norm(v)) for v in b]}), flush=True)


if __name__ == "__main__":
    main()
