"""Pins for the oracle's noise draw (Alg. 1: g ~ Gumbel(0, 1) per level; §3.3:
resampled every forward pass) against facts that do not come from the oracle:
the generator's published known-answer vectors, the Gumbel distribution's
moments, and the Gumbel-max property (argmax of logit + Gumbel noise is a
sample of softmax(logit)), which is what makes Alg. 1 a relaxation of sampling."""
import math
import os

import numpy as np
import pytest

from oracle import philox

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "philox4x32_10_kat.txt")


def _kat_rows():
    rows = []
    with open(GOLDEN) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            v = [int(x, 16) for x in line.split()]
            rows.append((v[0:4], v[4:6], v[6:10]))
    return rows


def test_philox_known_answers():
    rows = _kat_rows()
    assert len(rows) == 3
    for ctr, key, expect in rows:
        out = philox.philox4x32_10(*[np.array([c], dtype=np.uint64) for c in ctr], key[0], key[1])
        assert [int(o[0]) for o in out] == expect


def test_philox_vectorised_matches_scalar():
    ctr0 = np.arange(1000, dtype=np.uint64) * 7919
    out = philox.philox4x32_10(ctr0, 3, 5, 1, 0x1234, 0x9876)
    for j in (0, 1, 17, 999):
        single = philox.philox4x32_10(np.array([ctr0[j]]), 3, 5, 1, 0x1234, 0x9876)
        assert [int(o[j]) for o in out] == [int(s[0]) for s in single]


def test_uniform_is_exact_open_interval_fp32():
    x = np.array([0, 1, 0x800000, 0x800001, 0xFFFFFFFF, 0x400000, 0x7FFFFF], dtype=np.uint32)
    u = philox.uniform_from_word(x)
    assert u[0] == 2.0 ** -24 and u[2] == 2.0 ** -24          # only the low 23 bits count
    assert u[1] == 3 * 2.0 ** -24 and u[3] == 3 * 2.0 ** -24
    assert u[4] == 1.0 - 2.0 ** -24 and u[6] == 1.0 - 2.0 ** -24
    assert u[5] == 0.5 + 2.0 ** -24
    assert np.all(u.astype(np.float32).astype(np.float64) == u)   # representable in fp32
    assert np.all((u > 0) & (u < 1))


def test_level_words_layout():
    """Levels 0..3 share one Philox block (words 0..3); levels 4..7 use block 1."""
    idx = np.array([0, 5, (1 << 33) + 7], dtype=np.int64)
    w = philox.level_words(seed=(7 << 32) | 3, t=11, flat_index=idx, K=8)
    for j, i in enumerate(idx):
        lo, hi = int(i) & 0xFFFFFFFF, int(i) >> 32
        b0 = philox.philox4x32_10(np.array([lo]), hi, 11, 0, 3, 7)
        b1 = philox.philox4x32_10(np.array([lo]), hi, 11, 1, 3, 7)
        assert [int(w[k, j]) for k in range(4)] == [int(b[0]) for b in b0]
        assert [int(w[k, j]) for k in range(4, 8)] == [int(b[0]) for b in b1]


def test_fresh_noise_per_step_and_seed():
    idx = np.arange(4096, dtype=np.int64)
    g0 = philox.gumbel(0, 0, idx, 4)
    g1 = philox.gumbel(0, 1, idx, 4)
    g2 = philox.gumbel(1, 0, idx, 4)
    assert np.mean(g0 == g1) < 1e-3 and np.mean(g0 == g2) < 1e-3
    assert np.array_equal(g0, philox.gumbel(0, 0, idx, 4))      # reproducible


def test_gumbel_moments():
    """Gumbel(0,1): mean = Euler-Mascheroni gamma, variance = pi^2/6."""
    n = 1_000_000
    g = philox.gumbel(12345, 3, np.arange(n // 4, dtype=np.int64), 4).reshape(-1)
    mean, var = g.mean(), g.var()
    gamma = 0.5772156649015329
    sd_mean = math.sqrt(math.pi ** 2 / 6 / n)
    sd_var = (math.pi ** 2 / 6) * math.sqrt((5.4 - 1.0) / n)   # Gumbel kurtosis 5.4
    assert abs(mean - gamma) < 5 * sd_mean
    assert abs(var - math.pi ** 2 / 6) < 5 * sd_var
    # tail bounds implied by the 23-bit uniform: g in [-ln(-ln 2^-24), -ln(-ln(1-2^-24))]
    assert g.min() >= -math.log(-math.log(2.0 ** -24)) - 1e-12
    assert g.max() <= -math.log(-math.log1p(-2.0 ** -24)) + 1e-9


def test_gumbel_max_is_softmax_sample():
    """argmax_k (kappa*l_k + g_k) ~ Categorical(softmax(kappa*l)): chi-square test."""
    K, n, kappa = 4, 400_000, 1.7
    l = np.array([0.3, -0.2, 1.1, 0.0])
    g = philox.gumbel(99, 0, np.arange(n, dtype=np.int64), K)
    pick = np.argmax(kappa * l[:, None] + g, axis=0)
    counts = np.bincount(pick, minlength=K).astype(np.float64)
    p = np.exp(kappa * l) / np.exp(kappa * l).sum()
    chi2 = np.sum((counts - n * p) ** 2 / (n * p))
    # 3 degrees of freedom: P(chi2 > 21.1) ~ 1e-4
    assert chi2 < 21.1, (chi2, counts / n, p)
