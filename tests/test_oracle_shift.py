"""Pins for the oracle's local-shift parameterisation (§3.2 "Higher bit-widths",
Fig. 1): 5 logits per weight for delta in {-2..2}; the level of shift delta is
G[clip(j0 + delta)].  Checked against hand-written windows, against the full
K-level parameterisation (already pinned) with the logits outside the window at
-inf, a closed form at the clipped edge, finite differences, the projection map,
and the cold start."""
import numpy as np
import pytest

from oracle import gsq_oracle as O

GRID8 = np.linspace(-3.5, 3.5, 8)


def test_shift_windows_by_hand():
    j0 = np.array([0, 1, 3, 6, 7])
    idx = O.shift_index(j0, 8)
    assert idx[:, 0].tolist() == [0, 0, 0, 1, 2]       # clipped at the bottom
    assert idx[:, 1].tolist() == [0, 0, 1, 2, 3]
    assert idx[:, 2].tolist() == [1, 2, 3, 4, 5]       # interior
    assert idx[:, 3].tolist() == [4, 5, 6, 7, 7]
    assert idx[:, 4].tolist() == [5, 6, 7, 7, 7]       # clipped at the top


def _shift_problem(R=3, C=32, group=16, noise=False, seed=1):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((1, 20, C))
    H = np.einsum("etc,etd->ecd", X, X)
    prob = O.Problem(E=1, R=R, C=C, grid=GRID8, group=group, seed=3, H=H, noise=noise, shift=True)
    W = (0.02 * rng.standard_normal((R, C))).astype(np.float32)
    st = O.init_state(prob, W, np.arange(R))
    st.logits = rng.standard_normal(st.logits.shape).astype(np.float32)
    return prob, st


def test_interior_window_equals_full_parameterisation():
    prob, st = _shift_problem()
    st.j0 = np.random.default_rng(2).integers(2, 6, st.j0.shape).astype(np.uint8)   # interior
    full = O.Problem(E=1, R=prob.R, C=prob.C, grid=GRID8, group=prob.group, H=prob.H, noise=False)
    fst = st.copy()
    fl = np.full((8,) + st.j0.shape, -1e30, dtype=np.float64)
    for d in range(5):
        np.put_along_axis(fl, (st.j0.astype(np.int64) + d - 2)[None], st.logits[d][None].astype(np.float64), 0)
    fst.logits = fl
    fst.j0 = None
    rs = O.step(prob, st, 0, 0.7, 1.3, update=False)
    rf = O.step(full, fst, 0, 0.7, 1.3, update=False)
    np.testing.assert_allclose(rs.fw.What, rf.fw.What, rtol=1e-12, atol=0)
    np.testing.assert_allclose(rs.loss, rf.loss, rtol=1e-12)
    for d in range(5):
        g_full = np.take_along_axis(rf.d_logits, (st.j0.astype(np.int64) + d - 2)[None], 0)[0]
        np.testing.assert_allclose(rs.d_logits[d], g_full, rtol=1e-10, atol=1e-14)
    np.testing.assert_allclose(rs.d_scales, rf.d_scales, rtol=1e-12)


def test_clipped_edge_uniform_logits_closed_form():
    prob, st = _shift_problem()
    st.j0[:] = 0
    st.logits[:] = 0.25
    fw = O.forward(prob, st, 0, 0.9, 1.0)
    expect = (3 * GRID8[0] + GRID8[1] + GRID8[2]) / 5.0          # levels (0,0,0,1,2) equally likely
    np.testing.assert_allclose(fw.wtil, expect, rtol=1e-14)
    st.j0[:] = 7
    fw = O.forward(prob, st, 0, 0.9, 1.0)
    np.testing.assert_allclose(fw.wtil, (GRID8[5] + GRID8[6] + 3 * GRID8[7]) / 5.0, rtol=1e-14)


def test_shift_gradients_match_central_differences():
    prob, st = _shift_problem(noise=True)
    st.j0 = np.random.default_rng(4).integers(0, 8, st.j0.shape).astype(np.uint8)
    st.logits = st.logits.astype(np.float64)
    st.scales = st.scales.astype(np.float64)
    t, tau, kappa = 1, 0.6, 1.1
    res = O.step(prob, st, t, tau, kappa, update=False)
    rng = np.random.default_rng(5)

    def loss_at(logits):
        s2 = st.copy()
        s2.logits = logits
        fw = O.forward(prob, s2, t, tau, kappa)
        return O.loss_and_grad(prob, s2.row_ids, fw.D)[0]

    for _ in range(10):
        d, r, c = rng.integers(5), rng.integers(prob.R), rng.integers(prob.C)
        h = 1e-6 * max(1.0, abs(st.logits[d, r, c]))
        lp, lm = st.logits.copy(), st.logits.copy()
        lp[d, r, c] += h
        lm[d, r, c] -= h
        fd = (loss_at(lp) - loss_at(lm)) / (2 * h)
        assert abs(fd - res.d_logits[d, r, c]) <= 1e-6 * (abs(fd) + np.abs(res.d_logits).max())
    assert np.abs(res.d_logits.sum(0)).max() <= 1e-12 * np.abs(res.d_logits).max()


def test_shift_projection_maps_through_j0():
    l = np.float32([[0, 0, 0], [1, 0, 0], [0, 3, 0], [0, 0, 0], [0, 0, 5]])   # argmax 1, 2, 4
    codes, margin = O.project(l, j0=np.array([0, 3, 6]), levels=8)
    assert codes.tolist() == [0, 3, 7]        # clip(0-1)=0, 3+0=3, clip(6+2)=7
    assert margin.tolist() == [1.0, 3.0, 5.0]


def test_shift_cold_start_is_rtn_weight():
    prob, st = _shift_problem()
    W = st.W.astype(np.float32)
    st = O.init_state(prob, W, np.arange(prob.R))
    assert np.all(st.logits[2] == 2.0) and not st.logits[[0, 1, 3, 4]].any()
    fw = O.forward(prob, st, 0, 1e-3, 1.0)
    s = np.repeat(st.scales.astype(np.float64), prob.group, axis=1)
    np.testing.assert_allclose(fw.What, s * GRID8[st.j0], rtol=0, atol=1e-12)
