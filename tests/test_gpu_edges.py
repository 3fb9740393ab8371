"""Edge and degenerate cases of the step on the GPU against the oracle: the
smallest legal shapes (one row, C = 8 with group 4), ragged tails (weights not a
multiple of a warp's 128 or a pack chunk's 32), the binary grid (K = 2, whose
softmax is a sigmoid of twice the logit, §3 notation paragraph), all-zero weight
groups (scale 1), weights exactly on the grid, kappa = 0 (the logits drop out:
p is a pure Gumbel sample), temperatures from 1e-3 to 1e3, noise off, and the
rejection of bad arguments before any launch."""
import numpy as np
import pytest
import torch

from gpu_common import TOL_F32, assert_close, gsq
from oracle import gsq_oracle as O

pytestmark = pytest.mark.gpu


def _layer(W, grid, group, gemm="f32", noise=True, H=None, seed=3):
    g = gsq()
    E, R, C = W.shape
    if H is None:
        rng = np.random.default_rng(5)
        X = rng.standard_normal((E, 16, C)).astype(np.float32)
        H = np.einsum("etc,etd->ecd", X, X).astype(np.float32)
    Hd = torch.from_numpy(np.ascontiguousarray(H)).cuda()
    Wd = torch.from_numpy(np.ascontiguousarray(W)).cuda()
    layer = g.Layer(Wd, Hd, grid, group, gemm=gemm, noise=noise, seed=seed)
    prob = O.Problem(E=E, R=R, C=C, grid=np.asarray(grid, float), group=group, seed=seed,
                     H=H.astype(np.float64), noise=noise)
    return layer, prob


U32 = 2.0 ** -24


def _check_step(layer, prob, W, t, tau, kappa, tol=TOL_F32):
    g = gsq()
    E, R, C = W.shape
    n = E * R * C
    loss = torch.zeros(1, device="cuda")
    gl = torch.empty(prob.K * n, device="cuda")
    gs = torch.zeros(n // prob.group, device="cuda")
    layer.step(t, tau, kappa, loss=loss, grad_logits=gl, grad_scales=gs)
    what = torch.empty(n, device="cuda")
    layer.forward(t, tau, kappa, what=what)
    torch.cuda.synchronize()
    st = O.init_state(prob, W.reshape(E * R, C), np.arange(E * R))
    ref = O.step(prob, st, t, tau, kappa, update=False)
    # fp32 conditioning: z = (kappa l + g)/tau is evaluated with relative error
    # ~u, i.e. an absolute error u |z| that moves p by the same relative amount,
    # and w~ = sum p_k q_k cancels when p is flat over a symmetric grid (its
    # rounding is u sum |p_k q_k|).  At ordinary temperatures these stay far below
    # 1e-4; at the extremes the tolerance widens to what fp32 can resolve.
    zmax = float(np.max(np.abs(kappa * st.logits.astype(np.float64) + ref.fw.g))) / tau
    tol_p = max(tol, 8 * U32 * zmax)
    smax = float(np.max(np.abs(ref.fw.s))) * float(np.max(np.abs(prob.grid)))
    got_w = what.cpu().numpy().astype(np.float64)
    err = np.abs(got_w - ref.fw.What.reshape(-1))
    b = np.abs(ref.fw.What.reshape(-1))
    assert np.all(err <= tol_p * (b + np.sqrt(np.mean(b * b))) + 8 * U32 * smax), "W^"
    assert_close(loss.cpu().numpy(), [ref.loss], tol_p, "loss")
    assert_close(gl.cpu().numpy(), ref.d_logits, tol_p, "dL/dlogits")
    # dL/ds_g = sum_g G w~ inherits w~'s rounding u sum|p_k q_k| per weight
    ds = ref.d_scales.reshape(-1)
    cond = (8 * U32 * float(np.max(np.abs(prob.grid))) *
            np.abs(ref.G).reshape(-1, prob.group).sum(1))
    err = np.abs(gs.cpu().numpy().astype(np.float64) - ds)
    assert np.all(err <= tol_p * (np.abs(ds) + np.sqrt(np.mean(ds * ds))) + cond), "dL/dscales"
    return ref


def _w(shape, seed=0, scale=0.02):
    return (scale * np.random.default_rng(seed).standard_normal(shape)).astype(np.float32)


@pytest.mark.parametrize("shape,group", [((1, 1, 8), 4), ((1, 3, 24), 8), ((2, 5, 40), 8),
                                         ((1, 7, 136), 8)])
def test_smallest_and_ragged_shapes(shape, group):
    W = _w(shape)
    layer, prob = _layer(W, (-1.5, -0.5, 0.5, 1.5), group)
    _check_step(layer, prob, W, 2, 0.7, 1.0)
    # projection and packing of a ragged tail (n not a multiple of 32)
    n = int(np.prod(shape))
    codes = torch.empty(n, dtype=torch.uint8, device="cuda")
    layer.project(codes)
    buf = torch.empty(layer.packed_size(), dtype=torch.uint8, device="cuda")
    layer.pack(buf)
    st = O.init_state(prob, W.reshape(-1, shape[2]), np.arange(shape[0] * shape[1]))
    oc, _ = O.project(st.logits)
    assert np.array_equal(codes.cpu().numpy(), oc.reshape(-1))
    assert buf.cpu().numpy().tobytes() == O.pack_group(oc.reshape(-1), st.scales.reshape(-1), 4)


def test_binary_grid_is_sigmoid():
    W = _w((1, 4, 64), seed=1)
    layer, prob = _layer(W, (-1.0, 1.0), 16, noise=False)
    ref = _check_step(layer, prob, W, 0, 0.5, 1.0)
    l = O.init_state(prob, W[0], np.arange(4)).logits.astype(np.float64)
    sig = 1.0 / (1.0 + np.exp(-(l[1] - l[0]) / 0.5))
    np.testing.assert_allclose(ref.fw.p[1], sig, rtol=1e-12)


def test_all_zero_groups_and_exact_grid_points():
    W = _w((1, 4, 64), seed=2)
    W[0, 1, :] = 0.0                              # all-zero groups: scale 1, RTN code = nearest to 0
    W[0, 2, :16] = 0.01 * np.array([-1.5, -0.5, 0.5, 1.5] * 4, np.float32)
    layer, prob = _layer(W, (-1.5, -0.5, 0.5, 1.5), 16)
    st = O.init_state(prob, W[0], np.arange(4))
    got = layer.get_tensor(gsq().GSQ_T_SCALES, torch.float32).cpu().numpy().reshape(4, 4)
    assert np.array_equal(got, st.scales) and np.all(st.scales[1] == 1.0)
    _check_step(layer, prob, W, 1, 1.0, 1.0)


@pytest.mark.parametrize("tau,kappa", [(1e-3, 1.0), (1e3, 1.0), (0.5, 0.0), (0.05, 3.0)])
def test_temperature_and_kappa_extremes(tau, kappa):
    W = _w((1, 6, 128), seed=4)
    layer, prob = _layer(W, tuple(np.linspace(-3.5, 3.5, 8)), 32)
    _check_step(layer, prob, W, 5, tau, kappa)


def test_bad_step_arguments_are_rejected():
    g = gsq()
    W = _w((1, 2, 32), seed=6)
    layer, _ = _layer(W, (-1.0, 0.0, 1.0), 16)
    for tau, kappa, t in ((0.0, 1.0, 0), (-1.0, 1.0, 0), (float("nan"), 1.0, 0),
                          (1.0, float("inf"), 0), (1.0, 1.0, 1 << 32)):
        with pytest.raises(g.GsqError) as ei:
            layer.step(t, tau, kappa)
        assert ei.value.status == g.GSQ_ERR_INVALID_ARG
    with pytest.raises(g.GsqError):
        layer.set_tensor(g.GSQ_T_LOGITS, torch.zeros(5, device="cuda"))   # wrong size
    layer.sync_status()


def test_nonfinite_inputs_are_rejected():
    g = gsq()
    W = _w((1, 2, 32), seed=7)
    W[0, 1, 3] = np.nan
    with pytest.raises(g.GsqError) as ei:
        _layer(W, (-1.0, 0.0, 1.0), 16)
    assert ei.value.status == g.GSQ_ERR_NONFINITE
