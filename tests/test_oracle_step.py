"""Pins for the oracle's relaxation, loss, gradients and optimiser against what the
paper and the mathematics fix:
  * softmax rows sum to 1; the two-element case equals a sigmoid of 2*l (§3 notation
    paragraph: one logit l and -l for a binary set);
  * tau -> 0 turns the soft weight into the argmax-rounded weight (Alg. 1 caption
    text: annealing tau makes the weighted sum converge to one element);
  * uniform logits, no noise: W^ = s * mean(grid);
  * the loss equals brute force sum_t ||(W - W^) x_t||^2 (Eq. 1, linear layer);
  * gradients match central finite differences; shift invariance of the softmax;
    homogeneity in the scale; the Lemma of App. B bounds the logit gradient;
  * Lion: sign update of size lr after decoupled decay; a hand-worked two-step case.
"""
import numpy as np
import pytest

from oracle import gsq_oracle as O

GRID4 = np.array([-1.5, -0.5, 0.5, 1.5])
GRID_SKEW = np.array([-2.0, -1.0, 0.0, 1.0])


def _problem(E=1, R=4, C=32, grid=GRID4, group=16, T=24, seed=5, noise=True, rng=None):
    rng = rng or np.random.default_rng(0)
    X = rng.standard_normal((E, T, C))
    H = np.einsum("etc,etd->ecd", X, X)
    return O.Problem(E=E, R=R, C=C, grid=np.asarray(grid, float), group=group, seed=seed,
                     H=H, noise=noise), X


def _random_state(prob, rng, logit_scale=1.0):
    nr = prob.E * prob.R
    W = 0.02 * rng.standard_normal((nr, prob.C))
    st = O.init_state(prob, W.astype(np.float32), np.arange(nr))
    st.logits = (logit_scale * rng.standard_normal(st.logits.shape)).astype(np.float32)
    st.scales = (st.scales * (1 + 0.3 * rng.standard_normal(st.scales.shape))).astype(np.float32)
    return st


def test_softmax_sums_to_one():
    rng = np.random.default_rng(1)
    l = rng.standard_normal((8, 100)) * 5
    g = rng.gumbel(size=(8, 100))
    for tau in (2.0, 0.5, 0.05):
        p = O.relax(l, g, tau, 3.0)
        assert np.all(p >= 0)
        np.testing.assert_allclose(p.sum(0), 1.0, rtol=0, atol=1e-14)


def test_binary_case_is_sigmoid_of_twice_logit():
    l = np.linspace(-3, 3, 61)
    for tau, kappa in ((1.0, 1.0), (0.3, 2.0)):
        p = O.relax(np.stack([-l, l]), 0.0, tau, kappa)
        sig = 1.0 / (1.0 + np.exp(-2.0 * kappa * l / tau))
        np.testing.assert_allclose(p[1], sig, rtol=1e-13, atol=1e-15)


def test_low_temperature_gives_argmax_rounded_weight():
    rng = np.random.default_rng(2)
    prob, _ = _problem()
    st = _random_state(prob, rng)
    fw = O.forward(prob, st, t=3, tau=1e-4, kappa=1.0)
    a = prob.grid.size
    z = st.logits.astype(np.float64) + fw.g
    srt = np.sort(z, axis=0)
    clear = (srt[-1] - srt[-2]) > 1e-2            # away from ties
    k = np.argmax(z, axis=0)
    hard = fw.s * prob.grid[k]
    np.testing.assert_allclose(fw.What[clear], hard[clear], rtol=0, atol=1e-12)
    # with noise off, it is the projected weight of Alg. 2
    prob.noise = False
    fw0 = O.forward(prob, st, t=3, tau=1e-4, kappa=1.0)
    codes, margin = O.project(st.logits)
    ok = margin > 1e-2
    np.testing.assert_allclose(fw0.What[ok], (fw0.s * prob.grid[codes])[ok], atol=1e-12)


def test_uniform_logits_give_scaled_grid_mean():
    rng = np.random.default_rng(3)
    for grid in (GRID4, GRID_SKEW):
        prob, _ = _problem(grid=grid, noise=False)
        st = _random_state(prob, rng)
        st.logits[:] = 0.37
        fw = O.forward(prob, st, t=0, tau=0.7, kappa=2.0)
        np.testing.assert_allclose(fw.What, fw.s * grid.mean(), rtol=1e-14, atol=0)
    assert GRID_SKEW.mean() == -0.5


@pytest.mark.parametrize("use_x", [False, True])
def test_loss_equals_bruteforce_token_sum(use_x):
    rng = np.random.default_rng(4)
    prob, X = _problem(E=2, R=3, C=32, T=9, rng=rng)
    if use_x:
        prob.X, prob.H = X, None
    st = _random_state(prob, rng)
    res = O.step(prob, st, t=0, tau=0.8, kappa=1.0, update=False)
    brute = 0.0
    for e in range(prob.E):
        rows = slice(e * prob.R, (e + 1) * prob.R)
        brute += O.loss_bruteforce(st.W[rows], res.fw.What[rows], X[e])
    assert res.loss > 0
    np.testing.assert_allclose(res.loss, brute, rtol=1e-12)


def test_identity_calibration_gives_frobenius_norm():
    rng = np.random.default_rng(5)
    prob, _ = _problem()
    prob.H = np.eye(prob.C)[None]
    st = _random_state(prob, rng)
    res = O.step(prob, st, 0, 1.0, 1.0, update=False)
    np.testing.assert_allclose(res.loss, np.sum(res.fw.D ** 2), rtol=1e-13)
    np.testing.assert_allclose(res.G, 2 * res.fw.D, rtol=1e-13)


def _loss_at(prob, st, t, tau, kappa, logits=None, scales=None):
    s2 = st.copy()
    if logits is not None:
        s2.logits = logits
    if scales is not None:
        s2.scales = scales
    fw = O.forward(prob, s2, t, tau, kappa)
    return O.loss_and_grad(prob, s2.row_ids, fw.D)[0]


@pytest.mark.parametrize("grid", [GRID4, np.array([-1.0, 0.0, 1.0]),
                                  np.linspace(-3.5, 3.5, 8)])
def test_gradients_match_central_differences(grid):
    rng = np.random.default_rng(6)
    prob, _ = _problem(R=3, C=32, grid=grid, group=16, T=12, rng=rng)
    st = _random_state(prob, rng)
    st.logits = st.logits.astype(np.float64)
    st.scales = st.scales.astype(np.float64)
    t, tau, kappa = 2, 0.6, 1.3
    res = O.step(prob, st, t, tau, kappa, update=False)
    for _ in range(12):
        k, r, c = rng.integers(prob.K), rng.integers(3), rng.integers(32)
        h = 1e-6 * max(1.0, abs(st.logits[k, r, c]))
        lp, lm = st.logits.copy(), st.logits.copy()
        lp[k, r, c] += h
        lm[k, r, c] -= h
        fd = (_loss_at(prob, st, t, tau, kappa, logits=lp) -
              _loss_at(prob, st, t, tau, kappa, logits=lm)) / (2 * h)
        assert abs(fd - res.d_logits[k, r, c]) <= 1e-6 * (abs(fd) + np.abs(res.d_logits).max())
    for _ in range(6):
        r, gi = rng.integers(3), rng.integers(2)
        h = 1e-6 * max(1.0, abs(st.scales[r, gi]))
        sp, sm = st.scales.copy(), st.scales.copy()
        sp[r, gi] += h
        sm[r, gi] -= h
        fd = (_loss_at(prob, st, t, tau, kappa, scales=sp) -
              _loss_at(prob, st, t, tau, kappa, scales=sm)) / (2 * h)
        assert abs(fd - res.d_scales[r, gi]) <= 1e-6 * (abs(fd) + np.abs(res.d_scales).max())


def test_gradient_invariants_and_lemma_bound():
    rng = np.random.default_rng(7)
    prob, _ = _problem(R=4, C=64, grid=np.linspace(-3.5, 3.5, 8), group=32, rng=rng)
    st = _random_state(prob, rng, logit_scale=3.0)
    tau, kappa = 0.4, 2.0
    res = O.step(prob, st, 1, tau, kappa, update=False)
    scale = np.abs(res.d_logits).max()
    # softmax shift invariance: sum_k dL/dl_k = 0
    assert np.abs(res.d_logits.sum(0)).max() <= 1e-12 * scale
    # homogeneity: sum_g s_g dL/ds_g = sum G * W^
    lhs = np.sum(st.scales * res.d_scales)
    np.testing.assert_allclose(lhs, np.sum(res.G * res.fw.What), rtol=1e-12)
    # Lemma (App. B): ||dL/da||_inf <= (||dL/dy||_1 / tau) (1 - y_max), a = kappa*l + g
    dLdp = (res.G * res.fw.s)[None] * prob.grid[:, None, None]
    bound = (np.abs(dLdp).sum(0) / tau) * (1.0 - res.fw.p.max(0))
    da = np.abs(res.d_logits).max(0) / kappa
    assert np.all(da <= bound * (1 + 1e-12) + 1e-300)
    # second form of the bound: (K-1) (G/tau) exp(-Delta/tau)
    a = kappa * st.logits.astype(np.float64) + res.fw.g
    srt = np.sort(a, 0)
    bound2 = (prob.K - 1) * (np.abs(dLdp).sum(0) / tau) * np.exp(-(srt[-1] - srt[-2]) / tau)
    assert np.all(da <= bound2 * (1 + 1e-12) + 1e-300)


def test_lion_update_is_sign_of_size_lr_after_decay():
    rng = np.random.default_rng(8)
    theta = rng.standard_normal(10000).astype(np.float32)
    m = (0.01 * rng.standard_normal(10000)).astype(np.float32)
    g = rng.standard_normal(10000) * 1e-3
    lr, wd = 1e-4, 1.0
    tn, mn = O.lion(theta, m, g, lr, 0.9, 0.95, wd)
    step = tn.astype(np.float64) - theta.astype(np.float64) * (1 - lr * wd)
    ulp = np.spacing(np.abs(theta)).astype(np.float64)
    assert np.all(np.min(np.abs(step[:, None] - np.array([-lr, 0.0, lr])[None]), axis=1) <= ulp)
    # zero gradient and zero momentum: pure decay
    tz, mz = O.lion(theta, np.zeros_like(m), np.zeros(10000), lr, 0.9, 0.95, wd)
    np.testing.assert_array_equal(tz, (theta.astype(np.float64) * (1 - lr * wd)).astype(np.float32))
    assert np.all(mz == 0)


def test_lion_hand_worked_two_steps():
    """theta0 = 1, m0 = 0, lr = 0.1, wd = 0.5, b1 = 0.9, b2 = 0.95.
    step 1, g = 2:   c = 0.2 > 0       -> theta1 = 1 - 0.1*(1 + 0.5*1)     = 0.85
                     m1 = 0.05*2       = 0.1
    step 2, g = -1:  c = 0.09 - 0.1 < 0 -> theta2 = 0.85 - 0.1*(-1 + 0.425) = 0.9075
                     m2 = 0.095 - 0.05 = 0.045"""
    t1, m1 = O.lion(np.float32([1.0]), np.float32([0.0]), np.array([2.0]), 0.1, 0.9, 0.95, 0.5)
    assert t1[0] == np.float32(0.85) and m1[0] == np.float32(0.1)
    t2, m2 = O.lion(t1, m1, np.array([-1.0]), 0.1, 0.9, 0.95, 0.5)
    assert abs(t2[0] - 0.9075) < 1e-7 and abs(m2[0] - 0.045) < 1e-8


def test_step_updates_state_and_freezes_scales_when_lr_zero():
    rng = np.random.default_rng(9)
    prob, _ = _problem(rng=rng)
    st = _random_state(prob, rng)
    s0 = st.scales.copy()
    l0 = st.logits.copy()
    O.step(prob, st, 0, 1.0, 1.0)
    assert not np.array_equal(st.logits, l0) and not np.array_equal(st.scales, s0)
    prob.lr_scales = 0.0
    st2 = _random_state(prob, np.random.default_rng(9))
    s2 = st2.scales.copy()
    res = O.step(prob, st2, 0, 1.0, 1.0)
    assert res.d_scales is None and np.array_equal(st2.scales, s2)


@pytest.mark.parametrize("grid,group", [(GRID4, 16), (np.array([-1.0, 0.0, 1.0]), 32),
                                        (np.linspace(-3.5, 3.5, 8), 16)])
def test_initial_cold_weight_is_rtn_dequantised(grid, group):
    """At init (bias on the RTN level), noise off and tau -> 0, W^ is the
    round-to-nearest weight s_{floor(c/G)} q_{k0}: within half a grid step of W
    inside the grid's range, and exactly the clamped end level outside it."""
    rng = np.random.default_rng(10)
    prob = O.Problem(E=1, R=5, C=64, grid=np.asarray(grid, float), group=group, noise=False)
    W = (0.02 * rng.standard_normal((5, 64))).astype(np.float32)
    st = O.init_state(prob, W, np.arange(5))
    fw = O.forward(prob, st, t=0, tau=1e-3, kappa=1.0)
    s_true = np.repeat(O.init_group_scales(W, group, grid), group, axis=1).astype(np.float64)
    half_step = 0.5 * np.max(np.diff(grid))
    assert np.all(np.abs(fw.What - W) <= s_true * half_step * (1 + 1e-6) + 1e-12)
    np.testing.assert_allclose(fw.What / s_true, grid[O.rtn_codes(W, s_true.astype(np.float32), grid)],
                               rtol=0, atol=1e-9)
