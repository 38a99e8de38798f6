"""W8A16 weights (Sec. 3.3: the deployed model streams 8-bit weights with 16-bit
activations).  TEST INFRASTRUCTURE ONLY.

The paper does not give its quantiser; the reading taken here (R-Q1):
  R-Q1 every matrix the decoder streams (Wq, Wk, Wv, Wo, Wg, Wu, Wd of every layer and
       every LM head) is quantised per output row, symmetrically: with w the row's values
       as fp32 (the bf16 model's values, exact in fp32), m = max |w|,
       s = fp32(m / 127) (one IEEE single division, round to nearest even),
       q = clamp(rint(fp32(w / s)), -127, 127) (fp32 division, ties to even), and the
       row's weights are q * s; a row of zeros has s = 0 and q = 0.
       Embedding tables, offsets and norm gains keep their 16- / 32-bit values.
"""
from __future__ import annotations

from typing import Dict, Tuple

import numpy as np

QUANTISED = ("wq", "wk", "wv", "wo", "wg", "wu", "wd")


def quantise_rows(w: np.ndarray) -> Tuple[np.ndarray, np.ndarray]:
    """R-Q1 on a [rows, cols] fp32 matrix: (q int8 [rows, cols], s fp32 [rows])."""
    w32 = np.asarray(w, dtype=np.float32)
    m = np.max(np.abs(w32), axis=1)
    s = (m / np.float32(127.0)).astype(np.float32)
    q = np.zeros(w32.shape, dtype=np.int8)
    nz = s > 0
    ratio = (w32[nz] / s[nz, None]).astype(np.float32)
    q[nz] = np.clip(np.rint(ratio), -127, 127).astype(np.int8)
    return q, s


def dequantise(q: np.ndarray, s: np.ndarray) -> np.ndarray:
    return q.astype(np.float64) * s.astype(np.float64)[:, None]


def is_quantised(name: str) -> bool:
    return name.startswith("head.") or name.split(".")[-1] in QUANTISED


def w8a16_weights(w_f32: Dict[str, np.ndarray]) -> Dict[str, np.ndarray]:
    """The values a W8A16 decoder computes with: quantised matrices replaced by q * s."""
    out = {}
    for k, v in w_f32.items():
        out[k] = dequantise(*quantise_rows(v)) if is_quantised(k) else np.asarray(v, dtype=np.float64)
    return out
