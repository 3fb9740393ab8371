"""Pins for the oracle's step on per-step token batches with gradient
accumulation over resampled noise (§3.3 "Objective", "Gradient accumulation"):
one micro-batch reduces to the already pinned single step on those tokens; the
accumulated gradient is the gradient of the mean micro-batch loss (central
finite differences, each micro-batch with its own noise); the Lion update uses
that mean; and resampling the noise cuts the gradient's sampling variance by
the number of micro-batches (which reusing one draw would not)."""
import numpy as np

from oracle import gsq_oracle as O

GRID = np.array([-1.5, -0.5, 0.5, 1.5])


def _setup(R=3, C=32, T=12, M=3, seed=0, **kw):
    rng = np.random.default_rng(seed)
    batches = [rng.standard_normal((1, T, C)) for _ in range(M)]
    prob = O.Problem(E=1, R=R, C=C, grid=kw.pop("grid", GRID), group=16, seed=5,
                     H=np.eye(C)[None], **kw)
    W = (0.02 * rng.standard_normal((R, C))).astype(np.float32)
    st = O.init_state(prob, W, np.arange(R))
    st.logits = (0.5 * rng.standard_normal(st.logits.shape)).astype(np.float32)
    return prob, st, batches


def test_single_microbatch_is_the_token_step():
    prob, st, batches = _setup(M=1)
    t = 4
    res = O.step_microbatches(prob, st.copy(), t, batches, 0.7, 1.0, update=False)
    px = O.Problem(E=1, R=prob.R, C=prob.C, grid=GRID, group=16, seed=5, X=batches[0])
    ref = O.step(px, st.copy(), t, 0.7, 1.0, update=False)
    assert res.losses == [ref.loss]
    np.testing.assert_allclose(res.d_logits, ref.d_logits, rtol=1e-13, atol=1e-18)
    np.testing.assert_allclose(res.d_scales, ref.d_scales, rtol=1e-13, atol=1e-18)
    # and the token loss is the brute-force sum over the tokens (Eq. 1)
    fw = O.forward(px, st, t, 0.7, 1.0)
    assert abs(O.loss_bruteforce(st.W, fw.What, batches[0][0]) - ref.loss) <= 1e-12 * ref.loss


def test_accumulated_gradient_is_gradient_of_mean_loss():
    for kw in ({}, {"shift": True, "grid": np.linspace(-3.5, 3.5, 8)},
               {"mask_sign": True, "grid": np.array([-1.0, 0.0, 1.0])}):
        prob, st, batches = _setup(**kw)
        st.logits = st.logits.astype(np.float64)
        st.scales = st.scales.astype(np.float64)
        t, tau, kappa, M = 2, 0.8, 1.1, len(batches)
        res = O.step_microbatches(prob, st.copy(), t, batches, tau, kappa, update=False)

        def mean_loss(logits=None, scales=None):
            s2 = st.copy()
            if logits is not None:
                s2.logits = logits
            if scales is not None:
                s2.scales = scales
            tot = 0.0
            for j, X in enumerate(batches):
                pj = O.Problem(E=1, R=prob.R, C=prob.C, grid=prob.grid, group=16, seed=5, X=X,
                               shift=prob.shift, mask_sign=prob.mask_sign)
                fw = O.forward(pj, s2, t * M + j, tau, kappa)
                tot += O.loss_and_grad(pj, s2.row_ids, fw.D)[0]
            return tot / M

        rng = np.random.default_rng(3)
        for _ in range(8):
            k, r, c = rng.integers(st.logits.shape[0]), rng.integers(prob.R), rng.integers(prob.C)
            h = 1e-6
            lp, lm = st.logits.copy(), st.logits.copy()
            lp[k, r, c] += h
            lm[k, r, c] -= h
            fd = (mean_loss(logits=lp) - mean_loss(logits=lm)) / (2 * h)
            assert abs(fd - res.d_logits[k, r, c]) <= 1e-6 * (abs(fd) + np.abs(res.d_logits).max())
        r, g = 1, 1
        h = 1e-7 * abs(st.scales[r, g])
        sp, sm = st.scales.copy(), st.scales.copy()
        sp[r, g] += h
        sm[r, g] -= h
        fd = (mean_loss(scales=sp) - mean_loss(scales=sm)) / (2 * h)
        assert abs(fd - res.d_scales[r, g]) <= 1e-6 * (abs(fd) + np.abs(res.d_scales).max())


def test_update_uses_the_mean_gradient():
    prob, st, batches = _setup()
    res = O.step_microbatches(prob, st.copy(), 1, batches, 0.9, 1.0, update=False)
    st2 = st.copy()
    O.step_microbatches(prob, st2, 1, batches, 0.9, 1.0, update=True)
    want_l, want_m = O.lion(st.logits, st.m_logits, res.d_logits, prob.lr_logits, prob.beta1,
                            prob.beta2, prob.wd_logits)
    assert np.array_equal(st2.logits, want_l) and np.array_equal(st2.m_logits, want_m)


def test_resampled_noise_cuts_gradient_variance():
    """Over 300 steps, the variance of one logit's accumulated gradient with M = 8
    micro-batches (same tokens in each, so only the noise differs) is about 1/8
    of the single-draw variance."""
    prob, st, batches = _setup(R=1, C=16, T=8, M=1)
    X = batches[0]
    one, eight = [], []
    for t in range(300):
        one.append(O.step_microbatches(prob, st.copy(), t, [X], 1.0, 1.0, update=False).d_logits[1, 0, 3])
        eight.append(O.step_microbatches(prob, st.copy(), t, [X] * 8, 1.0, 1.0,
                                         update=False).d_logits[1, 0, 3])
    ratio = np.var(eight) / np.var(one)
    assert 0.6 / 8 < ratio < 1.6 / 8, ratio


def test_token_loss_through_the_gram_matrix():
    """The micro-batch's loss and gradient through its Gram matrix, H = X^T X, equal the
    token-literal ones (Eq. 1 with a linear f: sum_t ||D x_t||^2 = tr(D X^T X D^T) and
    2 (D X^T) X = 2 D (X^T X)): the identity the GPU's Gram route rests on, on a
    micro-batch with more tokens than inputs and with fewer."""
    for T, C in ((40, 16), (6, 32)):
        prob, st, batches = _setup(C=C, T=T, M=1, seed=T)
        X = batches[0]
        px = O.Problem(E=1, R=prob.R, C=C, grid=GRID, group=16, seed=5, X=X)
        ph = O.Problem(E=1, R=prob.R, C=C, grid=GRID, group=16, seed=5,
                       H=np.einsum("etc,etd->ecd", X, X))
        fw = O.forward(px, st, 2, 0.6, 1.0)
        ids = np.arange(prob.R)
        Lx, Gx = O.loss_and_grad(px, ids, fw.D)
        Lh, Gh = O.loss_and_grad(ph, ids, fw.D)
        assert abs(Lx - Lh) <= 1e-12 * Lx
        np.testing.assert_allclose(Gh, Gx, rtol=1e-11, atol=1e-14 * np.abs(Gx).max())
        assert abs(O.loss_bruteforce(st.W, fw.What, X[0]) - Lh) <= 1e-12 * Lh
