"""Philox4x32-10 counter-based generator -- oracle side (test infrastructure).

Written from the published definition (Salmon, Moraes, Dror, Shaw,
"Parallel random numbers: as easy as 1, 2, 3", SC'11, Section 5): four
32-bit counter words and two key words; each of the ten rounds multiplies
words 0 and 2 by the constants M0 and M1, mixes the high halves with the
other two words and the key, and the key is bumped by the Weyl constants
between rounds.

The PARD speculative-sampling path draws its uniforms from this generator
(the CUDA side has its own implementation of the same definition).
Stream layout used by both sides:
    key     = (seed mod 2^32, seed div 2^32)
    counter = (v div 4, (stream << 16) | i, b, step mod 2^32)
    word    = v mod 4
with stream 0: draft Gumbel noise (i = draft row, v = vocab id),
     stream 1: acceptance uniform (i = draft row, v = 0),
     stream 2: bonus / residual Gumbel noise (i = 0, v = vocab id).
"""
from __future__ import annotations

import numpy as np

M0, M1 = 0xD2511F53, 0xCD9E8D57
W0, W1 = 0x9E3779B9, 0xBB67AE85
MASK32 = 0xFFFFFFFF

STREAM_DRAFT, STREAM_ACCEPT, STREAM_BONUS = 0, 1, 2


def philox4x32_10(ctr, key):
    """ctr: 4 arrays (or ints) of uint32 values; key: 2 ints.  Returns the
    four output words as uint64 arrays holding 32-bit values."""
    c0, c1, c2, c3 = (np.asarray(c, dtype=np.uint64) & MASK32 for c in ctr)
    k0, k1 = int(key[0]) & MASK32, int(key[1]) & MASK32
    for r in range(10):
        if r > 0:
            k0 = (k0 + W0) & MASK32
            k1 = (k1 + W1) & MASK32
        p0 = c0 * np.uint64(M0)
        p1 = c2 * np.uint64(M1)
        hi0, lo0 = p0 >> np.uint64(32), p0 & np.uint64(MASK32)
        hi1, lo1 = p1 >> np.uint64(32), p1 & np.uint64(MASK32)
        c0, c1, c2, c3 = (hi1 ^ c1 ^ np.uint64(k0), lo1, hi0 ^ c3 ^ np.uint64(k1), lo0)
    return c0, c1, c2, c3


def raw_words(seed: int, stream: int, step: int, b: int, i: int, v) -> np.ndarray:
    """32-bit draws for vocab ids v (array) of row i, sequence b, step."""
    v = np.asarray(v, dtype=np.uint64)
    key = (seed & MASK32, (seed >> 32) & MASK32)
    ctr = (v >> np.uint64(2), np.uint64(((stream & 0xFFFF) << 16) | (i & 0xFFFF)),
           np.uint64(b & MASK32), np.uint64(step & MASK32))
    out = philox4x32_10(ctr, key)
    w = (v & np.uint64(3)).astype(np.int64)
    stacked = np.stack([np.broadcast_to(o, v.shape) for o in out], axis=0)
    return np.take_along_axis(stacked, w[None, ...], axis=0)[0].astype(np.uint32)


def uniform01(x: np.ndarray) -> np.ndarray:
    """[0, 1) from the top 24 bits: (x >> 8) * 2^-24, exact in fp32."""
    return ((x >> 8).astype(np.float32) * np.float32(2.0 ** -24)).astype(np.float32)


def uniform_open01(x: np.ndarray) -> np.ndarray:
    """(0, 1) from the top 23 bits: ((x >> 9) + 0.5) * 2^-23, exact in fp32
    (with 24 bits the largest value would round to 1.0)."""
    return (((x >> 9).astype(np.float32) + np.float32(0.5)) * np.float32(2.0 ** -23)).astype(np.float32)


def gumbel(x: np.ndarray) -> np.ndarray:
    """Standard Gumbel noise -log(-log u) in fp32."""
    u = uniform_open01(x)
    return (-np.log(-np.log(u))).astype(np.float32)
