"""Philox4x32-10 counter-based generator and the Gumbel(0, 1) draw built on it.

TEST INFRASTRUCTURE ONLY: this module belongs to the CPU oracle.  Only tests,
the smoke check and the benchmark's CPU-baseline leg may import it.

The paper draws g ~ Gumbel(0, 1) per level and per weight (Alg. 1) and resamples
it on every forward pass (§3.3, "Gradient accumulation"), but names no
generator.  This oracle reads the draw as Philox4x32-10, written here from its
published definition (Salmon, Moraes, Dror, Shaw: "Parallel Random Numbers: As
Easy as 1, 2, 3", SC'11, §4: the Philox S-box with multipliers 0xD2511F53 and
0xCD9E8D57 and the Weyl key schedule 0x9E3779B9, 0xBB67AE85).

Stream layout (a reading; the paper is silent):
  counter = (lo32(i), hi32(i), t, k div 4), key = (lo32(seed), hi32(seed)),
  where i = (e*R + r)*C + c is the flat weight index, t the step index and k the
  grid level; level k takes 32-bit word (k mod 4) of that block.
  u = ((x mod 2^23) + 1/2) * 2^-23     (low 23 bits; exactly representable in fp32, in (0,1))
  g = -ln(-ln(u))                       (inverse-CDF of Gumbel(0, 1)), in fp64.

Binary instances (the ternary mask x sign variant, Alg. 2) need only the
difference of their two Gumbel draws, which is Logistic(0, 1); it is drawn
directly by its inverse CDF from one word: lambda = ln(u) - ln(1 - u).  Two
weights share one block: weight i takes the block of counter
(lo32(i'), hi32(i'), t, 0) with i' = i - (i mod 2), and instance k (0 mask,
1 sign) takes word 2 (i mod 2) + k.
"""
from __future__ import annotations

import numpy as np

PHILOX_M0 = np.uint64(0xD2511F53)
PHILOX_M1 = np.uint64(0xCD9E8D57)
PHILOX_W0 = 0x9E3779B9
PHILOX_W1 = 0xBB67AE85
_MASK32 = np.uint64(0xFFFFFFFF)


def philox4x32_10(c0, c1, c2, c3, k0: int, k1: int):
    """Ten Philox rounds on arrays of 32-bit counter words; returns 4 uint32 arrays."""
    x0 = np.asarray(c0, dtype=np.uint64) & _MASK32
    x1 = np.asarray(c1, dtype=np.uint64) & _MASK32
    x2 = np.asarray(c2, dtype=np.uint64) & _MASK32
    x3 = np.asarray(c3, dtype=np.uint64) & _MASK32
    x0, x1, x2, x3 = np.broadcast_arrays(x0, x1, x2, x3)
    ka, kb = int(k0) & 0xFFFFFFFF, int(k1) & 0xFFFFFFFF
    for r in range(10):
        if r:
            ka = (ka + PHILOX_W0) & 0xFFFFFFFF
            kb = (kb + PHILOX_W1) & 0xFFFFFFFF
        p0 = PHILOX_M0 * x0           # < 2^64: exact in uint64
        p1 = PHILOX_M1 * x2
        hi0, lo0 = p0 >> np.uint64(32), p0 & _MASK32
        hi1, lo1 = p1 >> np.uint64(32), p1 & _MASK32
        x0, x1, x2, x3 = (hi1 ^ x1 ^ np.uint64(ka), lo1, hi0 ^ x3 ^ np.uint64(kb), lo0)
    return tuple(v.astype(np.uint32) for v in (x0, x1, x2, x3))


def uniform_from_word(x) -> np.ndarray:
    """u = ((x mod 2^23) + 1/2) * 2^-23, in float64 (exact)."""
    j = (np.asarray(x, dtype=np.uint64) & np.uint64(0x7FFFFF)).astype(np.float64)
    return (j + 0.5) * 2.0 ** -23


def level_words(seed: int, t: int, flat_index, K: int) -> np.ndarray:
    """The 32-bit word assigned to every (level k, weight i): shape [K, *flat_index.shape]."""
    i = np.asarray(flat_index, dtype=np.uint64)
    lo = i & _MASK32
    hi = i >> np.uint64(32)
    k0, k1 = int(seed) & 0xFFFFFFFF, (int(seed) >> 32) & 0xFFFFFFFF
    out = np.empty((K,) + i.shape, dtype=np.uint32)
    for blk in range((K + 3) // 4):
        words = philox4x32_10(lo, hi, np.uint64(t), np.uint64(blk), k0, k1)
        for w in range(4):
            k = 4 * blk + w
            if k < K:
                out[k] = words[w]
    return out


def gumbel(seed: int, t: int, flat_index, K: int) -> np.ndarray:
    """g[k, ...] ~ Gumbel(0, 1): one draw per level and weight (Alg. 1), fresh for
    every step t (§3.3).  fp64."""
    u = uniform_from_word(level_words(seed, t, flat_index, K))
    return -np.log(-np.log(u))


def pair_words(seed: int, t: int, flat_index) -> np.ndarray:
    """Words [2, ...] of the two binary instances of every weight: one Philox
    block per pair of weights (2j, 2j + 1), words (0, 1) for the even weight and
    (2, 3) for the odd one."""
    i = np.asarray(flat_index, dtype=np.uint64)
    odd = (i & np.uint64(1)).astype(bool)
    even = i - (i & np.uint64(1))
    k0, k1 = int(seed) & 0xFFFFFFFF, (int(seed) >> 32) & 0xFFFFFFFF
    w = philox4x32_10(even & _MASK32, even >> np.uint64(32), np.uint64(t), np.uint64(0), k0, k1)
    return np.stack([np.where(odd, w[2], w[0]), np.where(odd, w[3], w[1])])


def logistic(seed: int, t: int, flat_index) -> np.ndarray:
    """lam[k, ...] ~ Logistic(0, 1), the law of g1 - g0 for two independent
    Gumbel(0, 1) draws: one per binary instance (k = 0 mask, 1 sign) and
    weight, fresh for every step t.  Inverse CDF: lam = ln(u / (1 - u)).  fp64."""
    u = uniform_from_word(pair_words(seed, t, flat_index))
    return np.log(u) - np.log1p(-u)
