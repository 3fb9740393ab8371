"""Pins for the oracle's ternary mask x sign parameterisation (§3.1, Alg. 2):
two binary GS instances per weight (mask over {0, 1}, sign over {-1, 1}) with
tied logits (-l, l), whose softmax is a sigmoid of the noisy logit 2l (§3
notation paragraph); w~ = a m~ b~ on the grid {-a, 0, a}; hard rule
m = [l_m >= 0], b = 2 [l_b >= 0] - 1 (Alg. 2, final lines); Eq. 3 logit init.

Checked against the closed-form sigmoid, the logistic law of a Gumbel
difference (hand values and a Kolmogorov-Smirnov test), the tau -> 0 limit, the
Gumbel-max sampling frequencies, central finite differences, and hand examples
of the hard rule and the init table."""
import numpy as np
import pytest

from oracle import gsq_oracle as O
from oracle import philox

A = 0.75
GRID = np.array([-A, 0.0, A])


def _problem(R=4, C=32, group=16, noise=True, seed=3):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((1, 24, C))
    H = np.einsum("etc,etd->ecd", X, X)
    prob = O.Problem(E=1, R=R, C=C, grid=GRID, group=group, seed=seed, H=H, noise=noise,
                     mask_sign=True)
    W = (0.02 * rng.standard_normal((R, C))).astype(np.float32)
    st = O.init_state(prob, W, np.arange(R))
    st.logits = rng.standard_normal(st.logits.shape).astype(np.float32)
    return prob, st


def test_grid_must_be_symmetric_ternary():
    with pytest.raises(AssertionError):
        O.Problem(E=1, R=1, C=8, grid=np.array([-1.0, 0.0, 2.0]), group=8, mask_sign=True)
    with pytest.raises(AssertionError):
        O.Problem(E=1, R=1, C=8, grid=np.array([-1.5, -0.5, 0.5, 1.5]), group=8, mask_sign=True)


def test_binary_gs_is_sigmoid_of_twice_the_logit():
    prob, st = _problem()
    tau, kappa = 0.6, 1.3
    fw = O.forward(prob, st, 2, tau, kappa)
    lm, lb = st.logits.astype(np.float64)
    sig = lambda x: 1.0 / (1.0 + np.exp(-x))
    mt = sig((2 * kappa * lm + fw.g[0]) / tau)
    bt = 2 * sig((2 * kappa * lb + fw.g[1]) / tau) - 1
    np.testing.assert_allclose(fw.soft[0], mt, rtol=1e-13, atol=1e-15)
    np.testing.assert_allclose(fw.soft[1], bt, rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(fw.wtil, A * mt * bt, rtol=1e-12, atol=1e-15)
    s = np.repeat(st.scales.astype(np.float64), prob.group, axis=1)
    np.testing.assert_allclose(fw.What, s * A * mt * bt, rtol=1e-12, atol=1e-16)


def test_logistic_noise_hand_values_and_symmetry():
    # word with low 23 bits j gives u = (j + 1/2) 2^-23 and lambda = ln(u / (1 - u))
    for j, want in ((0, np.log(0.5 / (2 ** 23 - 0.5))),
                    (2 ** 22 - 1, np.log((2 ** 22 - 0.5) / (2 ** 22 + 0.5))),   # ~ -2^-22
                    (2 ** 22, np.log((2 ** 22 + 0.5) / (2 ** 22 - 0.5)))):
        u = philox.uniform_from_word(np.uint32(j | 0xAB800000))        # high bits ignored
        assert np.log(u) - np.log1p(-u) == pytest.approx(want, rel=1e-12)
    assert abs(np.log((2 ** 22 - 0.5) / (2 ** 22 + 0.5)) + 2.0 ** -22) < 1e-18
    # complementing the 23 bits maps u -> 1 - u, hence lambda -> -lambda
    words = np.arange(0, 2 ** 23, 4099, dtype=np.uint32)
    u, v = philox.uniform_from_word(words), philox.uniform_from_word(~words)
    np.testing.assert_allclose(np.log(u) - np.log1p(-u), -(np.log(v) - np.log1p(-v)),
                               rtol=1e-12, atol=1e-12)


def test_pair_words_layout():
    """Weights 2j and 2j + 1 split the four words of one block (counter of the
    even weight, block 0): the even weight takes words (0, 1), the odd (2, 3)."""
    idx = np.array([0, 1, 6, 7, 2 ** 33 + 4, 2 ** 33 + 5], dtype=np.uint64)
    got = philox.pair_words(99, 12, idx)
    for j, i in enumerate(idx):
        e = int(i) - int(i) % 2
        w = philox.philox4x32_10(e & 0xFFFFFFFF, e >> 32, 12, 0, 99, 0)
        o = 2 * (int(i) % 2)
        assert (got[0, j], got[1, j]) == (w[o], w[o + 1])
    # the even weight's words equal the first two words of its own block
    assert np.array_equal(philox.pair_words(5, 1, np.arange(0, 64, 2)),
                          philox.level_words(5, 1, np.arange(0, 64, 2), 2))


def test_logistic_law_matches_gumbel_difference():
    """The drawn lambda and the difference of two independent Gumbel draws both
    follow F(x) = 1 / (1 + e^-x) (Kolmogorov-Smirnov at n = 200000)."""
    idx = np.arange(200_000)
    lam = philox.logistic(7, 3, idx)
    g = philox.gumbel(7, 5, idx, 2)
    cdf = lambda x: 1.0 / (1.0 + np.exp(-x))
    for sample in (lam[0], lam[1], g[1] - g[0]):
        x = np.sort(sample)
        n = x.size
        F = cdf(x)
        d = max(np.max(np.arange(1, n + 1) / n - F), np.max(F - np.arange(n) / n))
        assert d < 1.63 / np.sqrt(n)          # 1% critical value
    assert abs(np.corrcoef(lam[0], lam[1])[0, 1]) < 0.01   # mask and sign draws independent


def test_zero_temperature_limit_is_the_hard_rule():
    prob, st = _problem(noise=False)
    st.logits[np.abs(st.logits) < 0.05] = 0.3
    fw = O.forward(prob, st, 0, 1e-3, 1.0)
    codes, _ = O.project(st.logits, mask_sign=True)
    np.testing.assert_allclose(fw.wtil, GRID[codes], rtol=0, atol=1e-12)


def test_uniform_logits():
    prob, st = _problem(noise=False)
    st.logits[:] = 0.0
    fw = O.forward(prob, st, 0, 0.9, 1.0)
    assert np.all(fw.soft[0] == 0.5) and np.all(fw.soft[1] == 0.0) and np.all(fw.wtil == 0.0)
    st.logits[1] = 40.0                         # sign certain: w~ = a * 1/2
    fw = O.forward(prob, st, 0, 0.9, 1.0)
    np.testing.assert_allclose(fw.wtil, A / 2, rtol=1e-14)


def test_sampling_frequencies_follow_the_logits():
    """Gumbel-max: at tau -> 0 the relaxed sample is the hard sample of the
    binary distributions, P(m = 1) = sigmoid(2 kappa l_m), P(b = 1 | m = 1) =
    sigmoid(2 kappa l_b); the three ternary values occur with the product
    probabilities."""
    prob = O.Problem(E=1, R=1, C=8, grid=GRID, group=8, seed=11, H=np.eye(8)[None], mask_sign=True)
    st = O.init_state(prob, np.zeros((1, 8), np.float32), np.arange(1))
    lm = np.array([-1.0, -0.3, 0.0, 0.2, 0.5, 1.0, 0.0, 0.4], np.float32)
    lb = np.array([0.0, 0.5, -0.5, 1.0, -1.0, 0.3, 0.0, -0.2], np.float32)
    st.logits = np.stack([lm, lb])[:, None, :]
    T, kappa = 4000, 0.8
    counts = np.zeros((3, 8))
    for t in range(T):
        fw = O.forward(prob, st, t, 1e-4, kappa)
        v = np.rint(fw.wtil[0] / A).astype(int)
        for c in (-1, 0, 1):
            counts[c + 1] += v == c
    sig = lambda x: 1.0 / (1.0 + np.exp(-x))
    pm, pb = sig(2 * kappa * lm.astype(float)), sig(2 * kappa * lb.astype(float))
    expect = np.stack([pm * (1 - pb), 1 - pm, pm * pb])
    assert np.all(np.abs(counts / T - expect) <= 4.5 * np.sqrt(expect * (1 - expect) / T) + 1e-9)


def test_gradients_match_central_differences():
    prob, st = _problem()
    st.logits = st.logits.astype(np.float64)
    st.scales = st.scales.astype(np.float64)
    t, tau, kappa = 1, 0.7, 1.2
    res = O.step(prob, st, t, tau, kappa, update=False)

    def loss_at(logits=None, scales=None):
        s2 = st.copy()
        if logits is not None:
            s2.logits = logits
        if scales is not None:
            s2.scales = scales
        fw = O.forward(prob, s2, t, tau, kappa)
        return O.loss_and_grad(prob, s2.row_ids, fw.D)[0]

    rng = np.random.default_rng(9)
    for _ in range(12):
        k, r, c = rng.integers(2), rng.integers(prob.R), rng.integers(prob.C)
        h = 1e-6 * max(1.0, abs(st.logits[k, r, c]))
        lp, lm = st.logits.copy(), st.logits.copy()
        lp[k, r, c] += h
        lm[k, r, c] -= h
        fd = (loss_at(logits=lp) - loss_at(logits=lm)) / (2 * h)
        assert abs(fd - res.d_logits[k, r, c]) <= 1e-6 * (abs(fd) + np.abs(res.d_logits).max())
    for _ in range(4):
        r, g = rng.integers(prob.R), rng.integers(prob.C // prob.group)
        h = 1e-7 * abs(st.scales[r, g])
        sp, sm = st.scales.copy(), st.scales.copy()
        sp[r, g] += h
        sm[r, g] -= h
        fd = (loss_at(scales=sp) - loss_at(scales=sm)) / (2 * h)
        assert abs(fd - res.d_scales[r, g]) <= 1e-6 * (abs(fd) + np.abs(res.d_scales).max())


def test_hard_rule_and_margins_by_hand():
    lm = np.float32([-0.5, 0.0, 0.25, 3.0, 1.0])
    lb = np.float32([9.0, 0.0, -1.0, 0.5, -0.0])
    codes, margin = O.project(np.stack([lm, lb]), mask_sign=True)
    # m = [l_m >= 0]: 0, 1, 1, 1, 1;  b = [l_b >= 0]: -, +, -, +, + (-0.0 >= 0)
    assert codes.tolist() == [1, 2, 0, 2, 2]
    assert margin.tolist() == [1.0, 0.0, 0.5, 1.0, 0.0]


def test_init_follows_eq3():
    prob = O.Problem(E=1, R=1, C=8, grid=GRID, group=8, H=np.eye(8)[None], mask_sign=True)
    W = np.float32([[-0.9, -0.2, 0.0, 0.1, 0.5, 0.9, -0.6, 0.3]])
    st = O.init_state(prob, W, np.arange(1), init_bias=1.5)
    # scale = absmax / a = 0.9 / 0.75 = 1.2; codes round W / 1.2 to {-0.75, 0, 0.75}
    assert st.scales[0, 0] == np.float32(np.float32(0.9) / np.float32(0.75))
    codes = [0, 1, 1, 1, 2, 2, 0, 1]
    want_m = [1.5 if c != 1 else -1.5 for c in codes]
    want_b = [1.5 if c == 2 else (-1.5 if c == 0 else 0.0) for c in codes]
    assert st.logits[0, 0].tolist() == want_m and st.logits[1, 0].tolist() == want_b
    # at init with no noise and tau -> 0 the soft weight is the RTN weight
    prob.noise = False
    fw = O.forward(prob, st, 0, 1e-3, 1.0)
    np.testing.assert_allclose(fw.What[0], st.scales[0, 0] * GRID[codes], rtol=0, atol=1e-12)
