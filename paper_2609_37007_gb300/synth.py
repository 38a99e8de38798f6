"""Seeded synthetic workloads for the MultiCodeDecoder speculative-decoding path.

This module only *draws* inputs: model shapes, random-init weights and the per-frame
inputs (conditioning hidden state and c0).  It holds none of the method's arithmetic,
so both the CUDA path and the CPU oracle can consume the same tensors without sharing
any computation.

Shapes follow the paper's MultiCodeDecoder (Sec. 1 and Fig. 1: 5 layers, 15 residual
codebook positions, one embedding table and one LM head per position; Sec. 2.2: K=3
offset vectors b_j).  The paper publishes no weights, so every tensor is synthetic:
  * matrices, embedding tables, LM heads and offsets ~ N(0, 0.02^2) (fp32 draw,
    rounded to bf16 with round-to-nearest-even for bf16 configurations);
  * RMSNorm gains ~ 1 + N(0, 0.1^2), so a dropped gain is visible in parity tests;
  * per-frame conditioning vector ~ N(0, 1); c0 ~ U[0, c0_vocab) or, when the
    configuration has no c0 table, a c0 embedding vector ~ N(0, 1).
Every tensor has its own PCG64 stream seeded by (seed, tensor index), and every frame
its own stream seeded by (seed, 7, frame index), so one tensor or frame never depends
on the shapes of the others.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List, Tuple

import numpy as np

WEIGHT_F32 = 0
WEIGHT_BF16 = 1
WEIGHT_INT8 = 2      # W8A16: the library quantises the bf16 matrices it streams at load time

DRAFT_SAMPLE = 0
DRAFT_GREEDY = 1
DRAFT_NOISY_TARGET = 2
DRAFT_TREE = 3


@dataclasses.dataclass(frozen=True)
class MCDConfig:
    """Shape and sampling configuration of one MultiCodeDecoder workload."""
    name: str
    n_layers: int
    hidden: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    ffn: int
    n_pos: int            # residual codebook positions c1..c_{n_pos}
    vocab: int            # entries per residual codebook (and per LM head)
    c0_vocab: int         # rows of the c0 table; 0 = the frame supplies a c0 embedding
    rms_eps: float
    rope_base: float
    qk_norm: int
    weight_dtype: int     # WEIGHT_F32 or WEIGHT_BF16
    draft_len: int        # K; 0 = plain autoregressive decoding
    top_k: int
    temperature: float
    draft_mode: int = DRAFT_SAMPLE
    noise_sigma: float = 0.0
    weight_seed: int = 0
    sample_seed: int = 1
    frames: int = 1
    max_streams: int = 1  # streams one launch may decode together
    # Synthetic structure for the offset-training harness: the table feeding sequence
    # position s (table 0 -> position 1, table i -> position i + 1) gets s * d added to every
    # row, d ~ N(0, position_drift^2 / hidden) per dim from its own seeded stream, so hidden
    # states drift with the position the way a per-lookahead offset can undo.  0 = none.
    position_drift: float = 0.0

    def replace(self, **kw) -> "MCDConfig":
        return dataclasses.replace(self, **kw)


# Tiny fp32 model for brute-force checks: 2 layers, hidden 256, 4x64 MHA, FFN 768,
# 4 positions, vocab 64, K=2, top-k 8, T=1, 200 frames, weight seed 0, Philox seed 1.
TINY = MCDConfig(name="tiny_fp32", n_layers=2, hidden=256, n_q_heads=4, n_kv_heads=4,
                 head_dim=64, ffn=768, n_pos=4, vocab=64, c0_vocab=0, rms_eps=1e-6,
                 rope_base=10000.0, qk_norm=1, weight_dtype=WEIGHT_F32, draft_len=2,
                 top_k=8, temperature=1.0, weight_seed=0, sample_seed=1, frames=200)

# MultiCodeDecoder-shaped bf16 model: 5 layers, hidden 1024, 16q/8kv x 128, FFN 3072,
# 15 positions with 2048-entry codebooks, K=3, top-k 50, T=0.9, 1000 frames.
MCD = MCDConfig(name="mcd_bf16", n_layers=5, hidden=1024, n_q_heads=16, n_kv_heads=8,
                head_dim=128, ffn=3072, n_pos=15, vocab=2048, c0_vocab=2048, rms_eps=1e-6,
                rope_base=10000.0, qk_norm=1, weight_dtype=WEIGHT_BF16, draft_len=3,
                top_k=50, temperature=0.9, weight_seed=0, sample_seed=1, frames=1000)

# The same models with a position drift in their embedding tables (offset-training harness).
TINY_DRIFT = TINY.replace(name="tiny_fp32_drift", position_drift=2.0)
MCD_DRIFT = MCD.replace(name="mcd_bf16_drift", position_drift=2.0)

CONFIGS = {c.name: c for c in (TINY, MCD, TINY_DRIFT, MCD_DRIFT)}


def tensor_specs(cfg: MCDConfig) -> List[Tuple[str, Tuple[int, ...], str]]:
    """Canonical (name, shape, kind) list; kind is 'mat' (N(0,0.02)) or 'gain' (1+N(0,0.1)).

    Matrices are stored [out, in] (row-major, one output per row)."""
    H, D = cfg.hidden, cfg.head_dim
    qd, kd = cfg.n_q_heads * D, cfg.n_kv_heads * D
    specs: List[Tuple[str, Tuple[int, ...], str]] = []
    for l in range(cfg.n_layers):
        p = f"layers.{l}."
        specs += [(p + "attn_norm", (H,), "gain"),
                  (p + "wq", (qd, H), "mat"), (p + "wk", (kd, H), "mat"), (p + "wv", (kd, H), "mat")]
        if cfg.qk_norm:
            specs += [(p + "q_norm", (D,), "gain"), (p + "k_norm", (D,), "gain")]
        specs += [(p + "wo", (H, qd), "mat"), (p + "ffn_norm", (H,), "gain"),
                  (p + "wg", (cfg.ffn, H), "mat"), (p + "wu", (cfg.ffn, H), "mat"),
                  (p + "wd", (H, cfg.ffn), "mat")]
    specs.append(("final_norm", (H,), "gain"))
    if cfg.c0_vocab > 0:
        specs.append(("embed.0", (cfg.c0_vocab, H), "mat"))
    # Table i embeds code c_i (i = 1..n_pos-1); c_{n_pos} is never fed back inside a frame.
    for i in range(1, cfg.n_pos):
        specs.append((f"embed.{i}", (cfg.vocab, H), "mat"))
    for P in range(1, cfg.n_pos + 1):
        specs.append((f"head.{P}", (cfg.vocab, H), "mat"))
    for j in range(1, max(cfg.draft_len, 1) + 1):
        specs.append((f"offset.{j}", (H,), "mat"))
    return specs


def round_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """fp32 -> bf16 bit patterns (uint16), round to nearest even (inputs are finite)."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32)
    bias = ((u >> np.uint32(16)) & np.uint32(1)) + np.uint32(0x7FFF)
    return ((u + bias) >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (b.astype(np.uint32) << np.uint32(16)).view(np.float32)


def _drift(cfg: MCDConfig) -> np.ndarray:
    rng = np.random.Generator(np.random.PCG64(np.random.SeedSequence([cfg.weight_seed, 13])))
    return rng.standard_normal(cfg.hidden) * (cfg.position_drift / np.sqrt(cfg.hidden))


def make_weights(cfg: MCDConfig) -> Dict[str, np.ndarray]:
    """All weights of `cfg`: float32 arrays for F32 configs, uint16 bf16 bits for BF16."""
    out: Dict[str, np.ndarray] = {}
    for idx, (name, shape, kind) in enumerate(tensor_specs(cfg)):
        rng = np.random.Generator(np.random.PCG64(np.random.SeedSequence([cfg.weight_seed, idx])))
        draw = rng.standard_normal(shape, dtype=np.float32)
        if kind == "gain":
            vals = (1.0 + 0.1 * draw.astype(np.float64)).astype(np.float32)
        else:
            vals = (0.02 * draw.astype(np.float64)).astype(np.float32)
        if cfg.position_drift and name.startswith("embed."):
            pos = int(name.split(".")[1]) + 1                       # the sequence position it feeds
            vals = (vals.astype(np.float64) + pos * _drift(cfg)[None, :]).astype(np.float32)
        out[name] = round_to_bf16_bits(vals) if cfg.weight_dtype in (WEIGHT_BF16, WEIGHT_INT8) else vals
    return out


def weights_as_f32(cfg: MCDConfig, w: Dict[str, np.ndarray]) -> Dict[str, np.ndarray]:
    """The exact values the weights represent, as float32 (bf16 widening is exact)."""
    if cfg.weight_dtype in (WEIGHT_BF16, WEIGHT_INT8):
        return {k: bf16_bits_to_f32(v) for k, v in w.items()}
    return dict(w)


@dataclasses.dataclass
class FrameInput:
    cond: np.ndarray            # float32 [H]: the outer model's hidden state for this frame
    c0: int                     # c0 id (c0_vocab > 0), else -1
    c0_emb: np.ndarray | None   # float32 [H] when the configuration has no c0 table


def make_frame(cfg: MCDConfig, frame_idx: int, seed: int | None = None) -> FrameInput:
    s = cfg.weight_seed if seed is None else seed
    rng = np.random.Generator(np.random.PCG64(np.random.SeedSequence([s, 7, frame_idx])))
    cond = rng.standard_normal(cfg.hidden, dtype=np.float32)
    if cfg.c0_vocab > 0:
        return FrameInput(cond=cond, c0=int(rng.integers(0, cfg.c0_vocab)), c0_emb=None)
    return FrameInput(cond=cond, c0=-1, c0_emb=rng.standard_normal(cfg.hidden, dtype=np.float32))


def make_frames(cfg: MCDConfig, n: int, first: int = 0, seed: int | None = None):
    """Stacked frame inputs: cond [n,H] f32, c0 ids [n] i32, c0 embeddings [n,H] f32 or None."""
    fr = [make_frame(cfg, first + i, seed) for i in range(n)]
    cond = np.stack([f.cond for f in fr]).astype(np.float32)
    c0 = np.array([f.c0 for f in fr], dtype=np.int32)
    emb = None if cfg.c0_vocab > 0 else np.stack([f.c0_emb for f in fr]).astype(np.float32)
    return cond, c0, emb


def random_logits(rng: np.random.Generator, rows: int, vocab: int, scale: float = 1.0,
                  tie_frac: float = 0.0) -> np.ndarray:
    """fp32 logits for sampler tests; `tie_frac` of entries are snapped to a coarse grid
    so that exact ties (broken by the lower id) occur often."""
    x = (scale * rng.standard_normal((rows, vocab))).astype(np.float32)
    if tie_frac > 0:
        m = rng.random((rows, vocab)) < tie_frac
        x[m] = np.round(x[m] * 4.0).astype(np.float32) / np.float32(4.0)
    return x


# ---------------------------------------------------------------------------------------
# Outer CodeDecoder (full frame pipeline, Fig. 1): one decoder call per 80 ms frame emits
# the seed code c0; its hidden state and c0 start the MultiCodeDecoder's frame.
# ---------------------------------------------------------------------------------------
@dataclasses.dataclass(frozen=True)
class OuterConfig:
    """Shape and sampling configuration of the outer CodeDecoder of a frame pipeline."""
    name: str
    n_layers: int
    hidden: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    ffn: int
    c0_vocab: int         # rows of the c0 table and of the c0 head
    text_vocab: int       # rows of the text-token table
    rms_eps: float
    rope_base: float
    qk_norm: int
    weight_dtype: int     # WEIGHT_F32 or WEIGHT_BF16; the KV cache is kept in this dtype
    top_k: int
    temperature: float
    prompt_len: int       # text tokens prefilled before frame 0
    frames: int           # frames of one utterance
    weight_seed: int = 0
    sample_seed: int = 1

    @property
    def max_tokens(self) -> int:
        """KV positions one utterance fills: the prompt plus one row per frame after the first."""
        return self.prompt_len + self.frames - 1

    def replace(self, **kw) -> "OuterConfig":
        return dataclasses.replace(self, **kw)


# Tiny fp32 pipeline for brute-force checks (inner model: TINY, which takes the c0
# embedding vector from the outer model).
OUTER_TINY = OuterConfig(name="outer_tiny_fp32", n_layers=2, hidden=256, n_q_heads=4, n_kv_heads=2,
                         head_dim=64, ffn=768, c0_vocab=96, text_vocab=512, rms_eps=1e-6,
                         rope_base=10000.0, qk_norm=1, weight_dtype=WEIGHT_F32, top_k=8,
                         temperature=1.0, prompt_len=12, frames=8)

# CodeDecoder-shaped bf16 model: 28 layers, hidden 1024, 16q/8kv x 128, FFN 3072, c0 vocab
# 3072, text vocab 151936, 256-token text prompt, 375 frames (30 s), top-k 50, T = 0.9.
OUTER = OuterConfig(name="codedecoder_bf16", n_layers=28, hidden=1024, n_q_heads=16, n_kv_heads=8,
                    head_dim=128, ffn=3072, c0_vocab=3072, text_vocab=151936, rms_eps=1e-6,
                    rope_base=10000.0, qk_norm=1, weight_dtype=WEIGHT_BF16, top_k=50,
                    temperature=0.9, prompt_len=256, frames=375)

# The MultiCodeDecoder of the pipeline: config-2 shapes, c0 embedding supplied by the outer model.
PIPE_INNER = MCD.replace(name="mcd_bf16_pipeline", c0_vocab=0)
PIPELINES = {"tiny": (OUTER_TINY, TINY), "full": (OUTER, PIPE_INNER)}


def outer_tensor_specs(cfg: OuterConfig, inner: MCDConfig) -> List[Tuple[str, Tuple[int, ...], str]]:
    """Tensors of the outer model: its layers (same names as the inner model's), final norm,
    c0 head and c0 table, the text table, and the table of the inner model's last code
    c_{n_pos}, which only the outer model's input sum reads."""
    H, D = cfg.hidden, cfg.head_dim
    qd, kd = cfg.n_q_heads * D, cfg.n_kv_heads * D
    specs: List[Tuple[str, Tuple[int, ...], str]] = []
    for l in range(cfg.n_layers):
        p = f"layers.{l}."
        specs += [(p + "attn_norm", (H,), "gain"),
                  (p + "wq", (qd, H), "mat"), (p + "wk", (kd, H), "mat"), (p + "wv", (kd, H), "mat")]
        if cfg.qk_norm:
            specs += [(p + "q_norm", (D,), "gain"), (p + "k_norm", (D,), "gain")]
        specs += [(p + "wo", (H, qd), "mat"), (p + "ffn_norm", (H,), "gain"),
                  (p + "wg", (cfg.ffn, H), "mat"), (p + "wu", (cfg.ffn, H), "mat"),
                  (p + "wd", (H, cfg.ffn), "mat")]
    specs += [("final_norm", (H,), "gain"), ("c0_head", (cfg.c0_vocab, H), "mat"),
              ("c0_embed", (cfg.c0_vocab, H), "mat"), ("text_embed", (cfg.text_vocab, H), "mat"),
              (f"code_embed.{inner.n_pos}", (inner.vocab, H), "mat")]
    return specs


def make_outer_weights(cfg: OuterConfig, inner: MCDConfig) -> Dict[str, np.ndarray]:
    """Outer-model weights, drawn like make_weights but from streams (seed, 5, index) so
    that they never repeat the inner model's."""
    out: Dict[str, np.ndarray] = {}
    for idx, (name, shape, kind) in enumerate(outer_tensor_specs(cfg, inner)):
        rng = np.random.Generator(np.random.PCG64(np.random.SeedSequence([cfg.weight_seed, 5, idx])))
        draw = rng.standard_normal(shape, dtype=np.float32)
        if kind == "gain":
            vals = (1.0 + 0.1 * draw.astype(np.float64)).astype(np.float32)
        else:
            vals = (0.02 * draw.astype(np.float64)).astype(np.float32)
        out[name] = round_to_bf16_bits(vals) if cfg.weight_dtype == WEIGHT_BF16 else vals
    return out


def outer_weights_as_f32(cfg: OuterConfig, w: Dict[str, np.ndarray]) -> Dict[str, np.ndarray]:
    if cfg.weight_dtype == WEIGHT_BF16:
        return {k: bf16_bits_to_f32(v) for k, v in w.items()}
    return dict(w)


def make_prompt(cfg: OuterConfig, utterance: int = 0, seed: int | None = None) -> np.ndarray:
    """Text-token ids of one utterance's prompt, uniform over [0, text_vocab)."""
    s = cfg.weight_seed if seed is None else seed
    rng = np.random.Generator(np.random.PCG64(np.random.SeedSequence([s, 11, utterance])))
    return rng.integers(0, cfg.text_vocab, size=cfg.prompt_len).astype(np.int32)
