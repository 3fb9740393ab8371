"""Pins for the oracle's diagnostics: displacement and margin histograms and the
mean noise-free max-probability, by hand on small logits for every
parameterisation, and the closed forms at uniform and one-hot logits."""
import numpy as np

from oracle import gsq_oracle as O

GRID4 = np.array([-1.5, -0.5, 0.5, 1.5])


def _st(prob, logits, j0=None):
    nr, C = logits.shape[1:]
    st = O.init_state(prob, np.zeros((nr, C), np.float32), np.arange(nr))
    st.logits = np.asarray(logits, np.float32)
    st.j0 = j0
    return st


def test_full_grid_by_hand():
    prob = O.Problem(E=1, R=1, C=4, grid=GRID4, group=4, H=np.eye(4)[None])
    l = np.zeros((4, 1, 4), np.float32)
    l[3, 0, 0] = 2.0          # code 3, margin 2
    l[1, 0, 1] = 1e-5 * 5     # code 1, margin 5e-5
    l[0, 0, 2] = 0.3          # code 0, margin 0.3
    # weight 3: all equal -> code 0, margin 0
    st = _st(prob, l)
    disp, pmax, marg = O.diagnostics(prob, st, np.array([[1, 1, 2, 0]]), tau=1.0, kappa=1.0)
    assert disp.tolist() == [2, 0, 2, 0, 0, 0, 0, 0]     # |3-1| = 2, 0, |0-2| = 2, 0
    # bins: [0, 1e-6) | [1e-6, 1e-5) | [1e-5, 1e-4) | ... | [0.1, 1) | [1, 10) | >= 10
    assert marg.tolist() == [1, 0, 1, 0, 0, 0, 1, 1, 0]  # 0 | 5e-5 | 0.3 | 2
    want = [np.exp(2) / (np.exp(2) + 3), np.exp(5e-5) / (np.exp(5e-5) + 3),
            np.exp(0.3) / (np.exp(0.3) + 3), 0.25]
    np.testing.assert_allclose(pmax, np.mean(want), rtol=1e-6)


def test_uniform_and_one_hot_saturation():
    prob = O.Problem(E=1, R=2, C=8, grid=GRID4, group=8, H=np.eye(8)[None])
    st = _st(prob, np.zeros((4, 2, 8)))
    assert O.diagnostics(prob, st, np.zeros((2, 8), int), 0.5, 1.0)[1] == 0.25
    l = np.zeros((4, 2, 8), np.float32)
    l[2] = 60.0
    st = _st(prob, l)
    disp, pmax, marg = O.diagnostics(prob, st, np.full((2, 8), 2), 0.1, 1.0)
    assert pmax == 1.0 and disp[0] == 16 and marg[-1] == 16


def test_shift_and_mask_sign():
    g8 = np.linspace(-3.5, 3.5, 8)
    prob = O.Problem(E=1, R=1, C=2, grid=g8, group=2, H=np.eye(2)[None], shift=True)
    l = np.zeros((5, 1, 2), np.float32)
    l[4, 0, 0] = 1.0          # delta +2 from j0 = 6 -> clipped to 7: displacement 1
    l[0, 0, 1] = 1.0          # delta -2 from j0 = 3 -> 1: displacement 2
    st = _st(prob, l, j0=np.array([[6, 3]], np.uint8))
    disp, _, _ = O.diagnostics(prob, st, np.array([[6, 3]]), 1.0, 1.0)
    assert disp.tolist() == [0, 1, 1, 0, 0, 0, 0, 0]
    pm = O.Problem(E=1, R=1, C=2, grid=np.array([-1.0, 0, 1]), group=2, H=np.eye(2)[None],
                   mask_sign=True)
    st = _st(pm, np.float32([[[0.0, -3.0]], [[0.0, 1.0]]]))
    disp, pmax, _ = O.diagnostics(pm, st, np.array([[1, 1]]), 1.0, 1.0)
    # weight 0: l_m = 0 -> on, l_b = 0 -> +: code 2, |2-1| = 1; p = (1/4, 1/2, 1/4) -> 1/2
    # weight 1: off: code 1; pm = s(-6), so max is 1 - pm
    assert disp.tolist() == [1, 1, 0, 0, 0, 0, 0, 0]
    s = lambda x: 1 / (1 + np.exp(-x))
    np.testing.assert_allclose(pmax, (0.5 + 1 - s(-6.0)) / 2, rtol=1e-12)
