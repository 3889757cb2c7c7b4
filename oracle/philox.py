"""Philox4x32-10 and the random draws of the sampling path (oracle side).

TEST INFRASTRUCTURE ONLY (see the package docstring).

Philox4x32-10 follows its published definition (J. Salmon, M. Moraes,
R. Dror, D. Shaw, "Parallel random numbers: as easy as 1, 2, 3", SC'11):
a 4x32-bit counter and a 2x32-bit key; each of 10 rounds multiplies counter
words 0 and 2 by fixed constants into 64-bit products, and the new counter is
(hi(M1*x2) ^ x1 ^ k0, lo(M1*x2), hi(M0*x0) ^ x3 ^ k1, lo(M0*x0)); the key is
bumped by the Weyl constants between rounds.

Stream layout used by the sampling path (App. A.4 asks for per-position
independent draft samples and FP32 acceptance arithmetic; the paper does not
fix a generator, so this layout is this implementation's choice):
  key     = (seed mod 2^32, seed >> 32)
  counter = (index, row, step, tag << 24 | sequence id)
  index   = vocabulary id >> 2 for per-token Gumbel noise (word = id & 3), else 0
  tags    = DRAFT (candidate draws), ACCEPT (accept coins), RESIDUAL, BONUS
"""
from __future__ import annotations

import numpy as np

PHILOX_M0 = 0xD2511F53
PHILOX_M1 = 0xCD9E8D57
PHILOX_W0 = 0x9E3779B9
PHILOX_W1 = 0xBB67AE85

TAG_DRAFT = 1
TAG_ACCEPT = 2
TAG_RESIDUAL = 3
TAG_BONUS = 4

_MASK32 = np.uint64(0xFFFFFFFF)


def philox4x32_10(counter, key):
    """counter: uint32 array [..., 4]; key: uint32 array broadcastable to [..., 2].
    Returns uint32 [..., 4]."""
    c = np.asarray(counter, dtype=np.uint64)
    k = np.asarray(key, dtype=np.uint64)
    x0, x1, x2, x3 = c[..., 0], c[..., 1], c[..., 2], c[..., 3]
    k0 = np.broadcast_to(k[..., 0], x0.shape).copy()
    k1 = np.broadcast_to(k[..., 1], x0.shape).copy()
    m0 = np.uint64(PHILOX_M0)
    m1 = np.uint64(PHILOX_M1)
    for rnd in range(10):
        if rnd > 0:
            k0 = (k0 + np.uint64(PHILOX_W0)) & _MASK32
            k1 = (k1 + np.uint64(PHILOX_W1)) & _MASK32
        p0 = m0 * x0                       # < 2^64: exact in uint64
        p1 = m1 * x2
        hi0, lo0 = p0 >> np.uint64(32), p0 & _MASK32
        hi1, lo1 = p1 >> np.uint64(32), p1 & _MASK32
        x0, x1, x2, x3 = hi1 ^ x1 ^ k0, lo1, hi0 ^ x3 ^ k1, lo0
    return np.stack([x0, x1, x2, x3], axis=-1).astype(np.uint32)


def _key(seed: int):
    seed = int(seed) & 0xFFFFFFFFFFFFFFFF
    return np.array([seed & 0xFFFFFFFF, seed >> 32], dtype=np.uint32)


def _counter(index, row, step, tag, seq):
    index = np.asarray(index, dtype=np.uint64)
    shape = index.shape
    c = np.empty(shape + (4,), dtype=np.uint64)
    c[..., 0] = index
    c[..., 1] = np.uint64(row)
    c[..., 2] = np.uint64(step)
    c[..., 3] = np.uint64(((tag & 0xFF) << 24) | (seq & 0xFFFFFF))
    return c


def word_to_uniform(w) -> np.ndarray:
    """u in [0, 1): the top 24 bits of a 32-bit word, exact in float32."""
    return ((np.asarray(w, dtype=np.uint32) >> np.uint32(8)).astype(np.float32)
            * np.float32(1.0 / 16777216.0))


def word_to_open_uniform(w) -> np.ndarray:
    """u in (0, 1): the top 23 bits plus one half, times 2^-23; exact in float32
    (24 significant bits), so neither 0 nor 1 can occur."""
    return (((np.asarray(w, dtype=np.uint32) >> np.uint32(9)).astype(np.float32) + np.float32(0.5))
            * np.float32(1.0 / 8388608.0))


def gumbel_noise(seed: int, seq: int, step: int, row: int, tag: int, vocab: int) -> np.ndarray:
    """Standard Gumbel noise G_v = -log(-log u_v), one per vocabulary id, float32."""
    ids = np.arange(vocab, dtype=np.uint64)
    out = philox4x32_10(_counter(ids >> np.uint64(2), row, step, tag, seq), _key(seed))
    w = np.take_along_axis(out, (ids & np.uint64(3)).astype(np.int64)[:, None], axis=1)[:, 0]
    u = word_to_open_uniform(w)
    return (-np.log(-np.log(u))).astype(np.float32)


def accept_uniform(seed: int, seq: int, step: int, row: int) -> np.float32:
    """The accept coin for candidate `row` (1-based) of one speculative step."""
    out = philox4x32_10(_counter(np.zeros((), np.uint64), row, step, TAG_ACCEPT, seq), _key(seed))
    return word_to_uniform(out[..., 0])[()]
