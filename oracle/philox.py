"""Philox4x32-10 (Salmon, Moraes, Dror, Shaw: "Parallel random numbers: as easy as
1, 2, 3", SC'11), written from the paper's definition, plus the uniform and
Gumbel conversions used by relaxed verification.

The AtSpeed paper only states r ~ U(0,1) (Alg. 2); the stream layout is a
reading of this build:
  key     = (seed & 0xffffffff, seed >> 32)
  counter = (draw >> 2, level | stream << 8, sd_step, user), output word draw & 3
  stream  0 draft sampling, 1 accept test, 2 subset keys, 3 resampling.
"""
from __future__ import annotations

import numpy as np

M0 = 0xD2511F53
M1 = 0xCD9E8D57
W0 = 0x9E3779B9   # golden ratio
W1 = 0xBB67AE85   # sqrt(3) - 1
MASK = 0xFFFFFFFF

STREAM_DRAFT, STREAM_ACCEPT, STREAM_SUBSET, STREAM_RESAMPLE = 0, 1, 2, 3


def philox4x32_10(c0, c1, c2, c3, k0, k1):
    """Vectorised Philox4x32 with 10 rounds; all arguments uint32-valued arrays/ints."""
    c0, c1, c2, c3 = (np.asarray(x, dtype=np.uint64) & MASK for x in (c0, c1, c2, c3))
    k0 = np.asarray(k0, dtype=np.uint64) & MASK
    k1 = np.asarray(k1, dtype=np.uint64) & MASK
    for r in range(10):
        if r:
            k0 = (k0 + W0) & MASK
            k1 = (k1 + W1) & MASK
        p0 = np.uint64(M0) * c0          # < 2**64: exact in uint64
        p1 = np.uint64(M1) * c2
        hi0, lo0 = p0 >> np.uint64(32), p0 & MASK
        hi1, lo1 = p1 >> np.uint64(32), p1 & MASK
        c0, c1, c2, c3 = hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0
    return tuple(x.astype(np.uint32) for x in (c0, c1, c2, c3))


def draw_u32(seed: int, stream: int, level: int, sd_step: int, user: int, draw) -> np.ndarray:
    """The uint32 word for draw index ``draw`` (array) of the given stream."""
    draw = np.asarray(draw, dtype=np.uint64)
    words = philox4x32_10(draw >> np.uint64(2), (level | (stream << 8)) & MASK, sd_step & MASK, user & MASK,
                          seed & MASK, (seed >> 32) & MASK)
    sel = (draw & np.uint64(3)).astype(np.int64)
    stacked = np.stack(words, axis=-1)
    return np.take_along_axis(stacked, sel[..., None], axis=-1)[..., 0]


def u_accept(w: np.ndarray) -> np.ndarray:
    """u = ((w >> 8) + 1) * 2**-24 in (0, 1], exact in fp32: u <= ratio accepts every
    draft with p >= q and none with p = 0."""
    w = np.asarray(w, dtype=np.uint32)
    return ((w >> np.uint32(8)).astype(np.float32) + np.float32(1.0)) * np.float32(2.0 ** -24)


def u_open(w: np.ndarray) -> np.ndarray:
    """u = (2 * (w >> 9) + 1) * 2**-24 in (0, 1), exact in fp32 (argument of the Gumbel map)."""
    w = np.asarray(w, dtype=np.uint32)
    return ((w >> np.uint32(9)).astype(np.float32) * np.float32(2.0) + np.float32(1.0)) * np.float32(2.0 ** -24)


def gumbel(w: np.ndarray) -> np.ndarray:
    """Standard Gumbel variate -log(-log(u)) in fp32."""
    u = u_open(w)
    return (-np.log(-np.log(u, dtype=np.float32), dtype=np.float32)).astype(np.float32)
