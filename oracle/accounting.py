"""The paper's real-time call arithmetic.  TEST INFRASTRUCTURE ONLY.

Sec. 1 / Fig. 1 caption: 12.5 frames/s (80 ms frames) x 16 codes = 200 tokens/s, one
outer CodeDecoder call plus 15 inner MultiCodeDecoder calls per frame.  With speculation
the inner loop needs 15 / (tokens per call) calls per frame (Sec. 1: 12.5 + 187.5/2.47
~= 88 sequential calls/s).  Sec. 3.4 prices the inner loop per second of audio as
inner calls/s x latency per call, and the speculative cost as that divided by the speedup.
"""
from __future__ import annotations

import math

FRAME_SECONDS = 0.080
CODES_PER_FRAME = 16          # c0 .. c15
RESIDUAL_CODES = 15           # c1 .. c15


def frames_per_second() -> float:
    return 1.0 / FRAME_SECONDS


def tokens_per_second() -> float:
    return frames_per_second() * CODES_PER_FRAME


def inner_calls_per_second_ar() -> float:
    return frames_per_second() * RESIDUAL_CODES


def sequential_calls_per_second(tokens_per_call: float) -> float:
    """Outer calls plus inner calls per second of audio at a given inner acceptance."""
    return frames_per_second() + inner_calls_per_second_ar() / tokens_per_call


def inner_ms_per_audio_second(ms_per_call: float) -> float:
    return inner_calls_per_second_ar() * ms_per_call


def offset_parameters(draft_len: int, hidden: int) -> int:
    """Sec. 2.2: K offset vectors b_1..b_K of the hidden size."""
    return draft_len * hidden


def medusa_head_parameters(n_heads: int, hidden: int, vocab: int) -> int:
    """Table 2 row ii: K fresh heads per position, each hidden x vocab."""
    return n_heads * hidden * vocab


def chain_calls_per_frame_all_accepted(draft_len: int, n_pos: int = RESIDUAL_CODES) -> int:
    """Calls when every draft is kept: the first call emits c1, then K+1 codes per call."""
    return 1 + math.ceil((n_pos - 1) / (draft_len + 1))


def chain_max_tokens_per_call(draft_len: int, n_pos: int = RESIDUAL_CODES) -> float:
    return n_pos / chain_calls_per_frame_all_accepted(draft_len, n_pos)
