"""Philox4x32-10 (Salmon, Moraes, Dror, Shaw: "Parallel random numbers: as easy as
1, 2, 3", SC'11) and the draws the sampler takes from it.  TEST INFRASTRUCTURE ONLY.

The paper only says the sampler is the deployed top-k sampling with the standard
speculative acceptance rule; which uniform drives which decision is fixed here as a
counter contract so that two independent implementations can be compared draw by draw:

  key     = (seed & 0xffffffff, seed >> 32)
  counter = (stream, frame, (round << 8) | position, purpose)

  purpose 0: sample from the target distribution (first code, bonus, AR, residual)
  purpose 1: accept test of the draft at `position`
  purpose 2: draft sample for `position`
  purpose 3 + v//2: Gaussian pair for vocabulary entries (v, v+1) of a noisy draft row

A uniform in [0, 1) uses words 0 and 1 of the block: ((w0 >> 5) * 2^26 + (w1 >> 6)) * 2^-53,
the 53-bit construction of Matsumoto and Nishimura's genrand_res53; the sampler's decisions
use its integer numerator U directly.
"""
from __future__ import annotations

import math

MASK = 0xFFFFFFFF
_M0, _M1 = 0xD2511F53, 0xCD9E8D57          # Philox multipliers (SC'11, Table 2)
_W0, _W1 = 0x9E3779B9, 0xBB67AE85          # Weyl key increments (golden ratio, sqrt(3)-1)

PURPOSE_TARGET = 0
PURPOSE_ACCEPT = 1
PURPOSE_DRAFT = 2
PURPOSE_NOISE = 3


def philox4x32_10(ctr, key):
    """Ten Philox rounds on a 4x32-bit counter with a 2x32-bit key; key bumped between rounds."""
    c0, c1, c2, c3 = (int(v) & MASK for v in ctr)
    k0, k1 = (int(v) & MASK for v in key)
    for r in range(10):
        if r:
            k0 = (k0 + _W0) & MASK
            k1 = (k1 + _W1) & MASK
        p0 = _M0 * c0          # 64-bit products: hi word is mulhi, lo word is mullo
        p1 = _M1 * c2
        c0, c1, c2, c3 = ((p1 >> 32) ^ c1 ^ k0, p1 & MASK, (p0 >> 32) ^ c3 ^ k1, p0 & MASK)
    return (c0, c1, c2, c3)


def key_of(seed: int):
    return (seed & MASK, (seed >> 32) & MASK)


def counter(stream: int, frame: int, rnd: int, position: int, purpose: int):
    return (stream & MASK, frame & MASK, ((rnd << 8) | position) & MASK, purpose & MASK)


def res53(w0: int, w1: int) -> float:
    """53-bit uniform in [0, 1) from two 32-bit words (exact in binary64)."""
    return ((w0 >> 5) * 67108864.0 + (w1 >> 6)) * (1.0 / 9007199254740992.0)


def int53(w0: int, w1: int) -> int:
    """The 53-bit integer U behind res53: res53(w0, w1) == U / 2^53 exactly."""
    return ((w0 >> 5) << 26) | (w1 >> 6)


def uniform(seed: int, stream: int, frame: int, rnd: int, position: int, purpose: int) -> float:
    w = philox4x32_10(counter(stream, frame, rnd, position, purpose), key_of(seed))
    return res53(w[0], w[1])


def uniform_int(seed: int, stream: int, frame: int, rnd: int, position: int, purpose: int) -> int:
    """The decision uniform as its 53-bit integer (u = U / 2^53)."""
    w = philox4x32_10(counter(stream, frame, rnd, position, purpose), key_of(seed))
    return int53(w[0], w[1])


def normal_pair(seed: int, stream: int, frame: int, rnd: int, position: int, pair: int):
    """Two N(0,1) draws by the Box-Muller transform (Box and Muller, 1958).

    u1 from words (0,1), u2 from words (2,3); radius sqrt(-2 ln(1-u1)) keeps the log finite."""
    w = philox4x32_10(counter(stream, frame, rnd, position, PURPOSE_NOISE + pair), key_of(seed))
    u1 = res53(w[0], w[1])
    u2 = res53(w[2], w[3])
    r = math.sqrt(-2.0 * math.log(1.0 - u1))
    t = 2.0 * math.pi * u2
    return r * math.cos(t), r * math.sin(t)
