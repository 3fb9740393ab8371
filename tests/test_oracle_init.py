"""Pins for the oracle's warm start from a supplied code vector (§3.1
"Initialization", Eq. 3-4; App. A): the noise-free prior logits by hand for each
parameterisation, the prior's mode at the supplied code, its Gaussian shape
(softmax ratios exp(-alpha ((c_k - mu)^2 - (c_j - mu)^2) / 2)), the mean
subtraction, and the linear noisy form l = sigma (eps + alpha l_GPTQ)."""
import numpy as np

from oracle import gsq_oracle as O

GRID2 = np.array([-1.5, -0.5, 0.5, 1.5])
GRID3 = np.linspace(-3.5, 3.5, 8)
TERN = np.array([-1.0, 0.0, 1.0])


def _prob(grid, **kw):
    C = 16
    return O.Problem(E=1, R=2, C=C, grid=grid, group=8, H=np.eye(C)[None], **kw)


def test_prior_by_hand():
    # 2-bit grid, code 1 (mu = -0.5): -(c - mu)^2 / 2 = (-0.5, 0, -0.5, -2), mean -0.75
    l = O.prior_logits(_prob(GRID2), np.array([1]))
    assert l[:, 0].tolist() == [0.25, 0.75, 0.25, -1.25]
    # local shift: candidates -2..2, mu = 0: (-2, -0.5, 0, -0.5, -2), mean -1
    l = O.prior_logits(_prob(GRID3, shift=True), np.array([6]))
    assert l[:, 0].tolist() == [-1.0, 0.5, 1.0, 0.5, -1.0]
    # mask x sign, Eq. 3: codes (-1, 0, +1) -> (l_m, l_b) = (1, -1), (-1, 0), (1, 1)
    l = O.prior_logits(_prob(TERN, mask_sign=True), np.array([0, 1, 2]))
    assert l[0].tolist() == [1.0, -1.0, 1.0] and l[1].tolist() == [-1.0, 0.0, 1.0]


def test_prior_mode_is_the_supplied_solution():
    codes = np.arange(8)
    l = O.prior_logits(_prob(GRID3), codes)
    assert np.array_equal(np.argmax(l, axis=0), codes)
    assert np.allclose(l.mean(axis=0), 0.0)
    l = O.prior_logits(_prob(GRID3, shift=True), codes)
    assert np.all(np.argmax(l, axis=0) == 2)                      # delta = 0: stay put
    l = O.prior_logits(_prob(TERN, mask_sign=True), np.array([0, 1, 2]))
    c, _ = O.project(l.astype(np.float32), mask_sign=True)
    assert c.tolist() == [0, 1, 2]


def test_prior_softmax_is_a_discretised_gaussian():
    alpha = 6.0
    for code in range(4):
        l = O.prior_logits(_prob(GRID2), np.array([code]))[:, 0]
        p = O.relax(alpha * l[:, None], np.zeros((4, 1)), 1.0, 1.0)[:, 0]
        d2 = (GRID2 - GRID2[code]) ** 2
        for j in range(4):
            np.testing.assert_allclose(p / p[j], np.exp(-alpha * (d2 - d2[j]) / 2), rtol=1e-12)


def test_noisy_init_is_linear_in_eps_and_prior():
    prob = _prob(GRID2)
    rng = np.random.default_rng(4)
    W = (0.02 * rng.standard_normal((2, 16))).astype(np.float32)
    codes = rng.integers(0, 4, (2, 16))
    eps = rng.standard_normal((4, 2, 16))
    prior = O.prior_logits(prob, codes)
    st = O.init_from_codes(prob, W, np.arange(2), codes, eps, alpha=6.0, sigma=0.01)
    np.testing.assert_allclose(st.logits, 0.01 * (eps + 6.0 * prior), rtol=1e-6, atol=1e-9)
    st0 = O.init_from_codes(prob, W, np.arange(2), codes, None, alpha=6.0, sigma=0.01)
    np.testing.assert_allclose(st0.logits, 0.06 * prior, rtol=1e-6, atol=1e-9)
    stn = O.init_from_codes(prob, W, np.arange(2), codes, eps, alpha=0.0, sigma=0.5)
    np.testing.assert_allclose(stn.logits, 0.5 * eps, rtol=1e-6, atol=1e-9)
    assert not st.m_logits.any() and not st.m_scales.any()
    # supplied scales replace the absmax ones
    sc = np.full((2, 2), 0.125, np.float32)
    st1 = O.init_from_codes(prob, W, np.arange(2), codes, None, 1.0, 1.0, scales=sc)
    assert np.array_equal(st1.scales, sc)


def test_shift_init_takes_j0_from_the_codes():
    prob = _prob(GRID3, shift=True)
    W = np.zeros((2, 16), np.float32)
    codes = np.tile(np.arange(8), 4).reshape(2, 16)
    st = O.init_from_codes(prob, W, np.arange(2), codes, None, alpha=6.0, sigma=0.01)
    assert np.array_equal(st.j0, codes.astype(np.uint8))
    fw = O.forward(O.Problem(E=1, R=2, C=16, grid=GRID3, group=8, H=np.eye(16)[None], shift=True,
                             noise=False), st, 0, 1e-3, 1.0)
    s = np.repeat(st.scales.astype(np.float64), 8, axis=1)
    np.testing.assert_allclose(fw.What, s * GRID3[codes], rtol=0, atol=1e-12)
