"""GPU parity of the local-shift parameterisation (§3.2 "Higher bit-widths",
Fig. 1) against the oracle: 5 logits per weight for the shifts delta = -2..2
around the initial grid index j0, level G[clip(j0 + delta)].  Covered: the
initial state (j0 = RTN index, +bias on delta = 0) bit-exact; the soft weight,
loss and gradients on random logits and random j0 that reach both clipped ends
of the grid; the Lion update; the look-ahead forward; projection through j0 and
packing bit-exact; a multi-step trajectory.  Shapes are small versions of the
3-bit down_proj and MoE K-Quant workloads and of the 2-bit / ternary grids
(where the 5-wide window is clipped on both sides), with ragged GEMM tiles."""
import dataclasses

import numpy as np
import pytest
import torch

from gpu_common import (TOL_BF16, TOL_F32, Case, assert_close, assert_gemm_bound,
                        assert_grad_close, check_lion, check_momentum, grad_bounds, gsq)
from oracle import gsq_oracle as O
from paper_2604_18556_gb300 import configs as C

pytestmark = pytest.mark.gpu

W = C.WORKLOADS


def _shift(w):
    return dataclasses.replace(w, param="shift5")


SMALL = {
    "down_proj": C.shrunk(W["llama8b_down_proj_shift5"], rows=160, cols=640, tokens=4096),
    "moe_kquant": _shift(C.shrunk(W["moe64_kquant3"], experts=3, rows=64, cols=512, tokens=1024)),
    "q_proj": _shift(C.shrunk(W["llama8b_q_proj"], rows=96, cols=384, tokens=2048)),
    "ternary": _shift(W["ternary_256x512"]),
}
TAU = {"down_proj": 0.5, "moe_kquant": 1.0, "q_proj": 0.55, "ternary": 1.0}


def _n(w):
    return w.experts * w.rows * w.cols


def _randomise(case, seed):
    """Random logits N(0, 1) and random initial indices over the whole grid
    (both clipped ends included), written through the C ABI."""
    g = gsq()
    w = case.w
    rng = np.random.default_rng(seed)
    nr = w.experts * w.rows
    L = rng.standard_normal((5, nr, w.cols)).astype(np.float32)
    j0 = rng.integers(0, w.K, (nr, w.cols)).astype(np.uint8)
    case.layer.set_tensor(g.GSQ_T_LOGITS, torch.from_numpy(L).cuda())
    case.layer.set_tensor(g.GSQ_T_J0, torch.from_numpy(j0).cuda())
    return case.state()


def _q(case, st):
    return O.level_values(case.prob, st)


@pytest.mark.parametrize("name", list(SMALL))
def test_shift_init_bit_exact(name):
    case = Case(SMALL[name], gemm="f32")
    st, ref = case.state(), case.oracle_init()
    assert st.logits.shape[0] == 5
    assert np.array_equal(st.j0, ref.j0)
    assert np.array_equal(st.logits, ref.logits)
    assert np.array_equal(st.scales, ref.scales)
    assert not st.m_logits.any() and not st.m_scales.any()
    if SMALL[name].scale_mode == "kquant2":
        assert np.array_equal(st.kq_d, ref.kq_d) and np.array_equal(st.kq_sc, ref.kq_sc)


@pytest.mark.parametrize("noise", [True, False])
@pytest.mark.parametrize("name", list(SMALL))
def test_shift_forward_soft_weight(name, noise):
    w = SMALL[name]
    case = Case(w, gemm="f32", noise=noise)
    st = _randomise(case, 11)
    what = torch.empty(_n(w), device="cuda")
    case.layer.forward(7, 0.7, 1.3, what=what)
    ref = O.forward(case.prob, st, 7, 0.7, 1.3)
    assert_close(what.cpu().numpy(), ref.What, TOL_F32, "W^")
    assert_close(case.D(), ref.D, TOL_F32, "D")


@pytest.mark.parametrize("gemm", ["f32", "bf16"])
@pytest.mark.parametrize("name", list(SMALL))
def test_shift_step_loss_and_gradients(name, gemm):
    w = SMALL[name]
    case = Case(w, gemm=gemm)
    st = _randomise(case, 12)
    tol = TOL_F32 if gemm == "f32" else TOL_BF16
    n = _n(w)
    loss = torch.zeros(1, device="cuda")
    gl = torch.empty(5 * n, device="cuda")
    gs = torch.zeros(n // w.group, device="cuda")
    case.layer.step(3, TAU[name], 1.0, loss=loss, grad_logits=gl, grad_scales=gs)
    torch.cuda.synchronize()
    ref = O.step(case.prob, st.copy(), 3, TAU[name], 1.0, update=False)
    assert_close(loss.cpu().numpy(), [ref.loss], tol, "loss")
    assert_close(case.G(), ref.G, tol, "G")
    if gemm == "f32":
        assert_close(gl.cpu().numpy(), ref.d_logits, tol, "dL/dlogits")
        if ref.d_scales is not None:
            assert_close(gs.cpu().numpy(), ref.d_scales, tol, "dL/dscales")
    else:
        assert_grad_close(gl.cpu().numpy(), gs.cpu().numpy() if ref.d_scales is not None else None,
                          ref, case.prob, TAU[name], 1.0, tol, name, q=_q(case, st))
        D, H, G = case.D(), case.H_operand(), case.G()
        rows = np.arange(w.experts * w.rows)
        for e in range(w.experts):
            sel = rows // w.rows == e
            assert_gemm_bound(G[sel], D[sel], H[e], f"tcgen05 GEMM vs its operands, expert {e}")
    # the 5 logit gradients of a weight sum to zero (softmax shift invariance)
    gl5 = gl.cpu().numpy().astype(np.float64).reshape(5, -1)
    assert np.all(np.abs(gl5.sum(0)) <= 1e-5 * np.abs(gl5).max())


@pytest.mark.parametrize("gemm", ["f32", "bf16"])
@pytest.mark.parametrize("name", ["down_proj", "moe_kquant", "q_proj"])
def test_shift_step_update(name, gemm):
    w = SMALL[name]
    case = Case(w, gemm=gemm)
    _randomise(case, 13)
    tol = TOL_F32 if gemm == "f32" else TOL_BF16
    for t in range(2):
        loss = torch.zeros(1, device="cuda")
        before = case.state()
        case.layer.step(t, TAU[name], 1.0, loss=loss)
        torch.cuda.synchronize()
        st_sync = before.copy()
        res = O.step(case.prob, st_sync, t, TAU[name], 1.0, update=True)
        gpu = case.state()
        assert np.array_equal(gpu.j0, before.j0)          # j0 is fixed for the whole run
        assert_close(loss.cpu().numpy(), [res.loss], tol, f"loss t={t}")
        c_l = w.beta1 * before.m_logits.astype(np.float64) + (1 - w.beta1) * res.d_logits
        check_lion(gpu.logits, st_sync.logits, before.logits, c_l, w.lr_logits, 2 * tol, "logits")
        if gemm == "f32":
            gb_l = tol * (np.abs(res.d_logits) + np.sqrt(np.mean(res.d_logits ** 2)))
            gb_s = None if res.d_scales is None else \
                tol * (np.abs(res.d_scales) + np.sqrt(np.mean(res.d_scales ** 2)))
        else:
            f, gscale, bs = grad_bounds(res, case.prob, tol, q=_q(case, before))
            gb_l = (1.0 / TAU[name]) * f * gscale[None] + tol * np.abs(res.d_logits)
            gb_s = None if res.d_scales is None else bs + tol * np.abs(res.d_scales)
        check_momentum(gpu.m_logits, st_sync.m_logits, gb_l, w.beta2, "logit momentum")
        if res.d_scales is not None:
            c_s = w.beta1 * before.m_scales.astype(np.float64) + (1 - w.beta1) * res.d_scales
            check_lion(gpu.scales, st_sync.scales, before.scales, c_s, w.lr_scales, 2 * tol,
                       "scales")
            check_momentum(gpu.m_scales, st_sync.m_scales, gb_s, w.beta2, "scale momentum")
        else:
            assert np.array_equal(gpu.scales, before.scales)


@pytest.mark.parametrize("name", ["down_proj", "moe_kquant"])
def test_shift_lookahead_is_bit_identical(name):
    w = SMALL[name]
    a, b = Case(w, gemm="bf16"), Case(w, gemm="bf16")
    for t in range(4):
        la, lb = torch.zeros(1, device="cuda"), torch.zeros(1, device="cuda")
        a.layer.step(t, w.tau(t), 1.0, next_tau=w.tau(t + 1), next_kappa=1.0, loss=la)
        b.layer.step(t, w.tau(t), 1.0, loss=lb)
        torch.cuda.synchronize()
        assert la.item() == lb.item()
        sa, sb = a.state(), b.state()
        for f in ("logits", "m_logits", "scales", "m_scales", "j0"):
            assert np.array_equal(getattr(sa, f), getattr(sb, f)), (t, f)


@pytest.mark.parametrize("name", list(SMALL))
def test_shift_project_and_pack_bit_exact(name):
    g = gsq()
    w = SMALL[name]
    case = Case(w, gemm="bf16")
    for t in range(2):
        case.layer.step(t, 0.3, 1.0, next_tau=0.3)
    st = _randomise(case, 14)
    L = st.logits.copy()
    L[:, :, ::7] = L[:, :, ::7].max(0, keepdims=True)      # exact ties in every 7th column
    case.layer.set_tensor(g.GSQ_T_LOGITS, torch.from_numpy(L.copy()).cuda())
    n = _n(w)
    codes = torch.empty(n, dtype=torch.uint8, device="cuda")
    margin = torch.empty(n, device="cuda")
    case.layer.project(codes, margin)
    st = case.state()
    oc, om = O.project(st.logits, j0=st.j0, levels=w.K)
    assert np.array_equal(codes.cpu().numpy(), oc.reshape(-1))
    assert np.array_equal(margin.cpu().numpy(), om.reshape(-1))
    buf = torch.full((case.layer.packed_size(),), 0xAB, dtype=torch.uint8, device="cuda")
    assert case.layer.pack(buf) == buf.numel()
    got = buf.cpu().numpy().tobytes()
    if w.scale_mode == "kquant2":
        ref = O.pack_kquant2(oc.reshape(-1), st.kq_d.reshape(-1), st.kq_sc.reshape(-1))
    else:
        ref = O.pack_group(oc.reshape(-1), st.scales.reshape(-1), w.K)
    assert got == ref


def test_shift_trajectory():
    """30 steps of the 3-bit shift problem in the fp32 path, oracle and GPU each
    on their own trajectory: per-step losses within 1e-4, final logits within
    the Lion flip allowance, final codes bit-exact where the margin is >= 1e-5."""
    w = dataclasses.replace(SMALL["down_proj"], w_dtype="f32", steps=30, tau0=1.0, tau1=0.3)
    case = Case(w, gemm="f32")
    st = case.oracle_init()
    for t in range(w.steps):
        loss = torch.zeros(1, device="cuda")
        case.layer.step(t, w.tau(t), 1.0, next_tau=w.tau(t + 1), next_kappa=1.0, loss=loss)
        res = O.step(case.prob, st, t, w.tau(t), 1.0)
        assert_close(loss.cpu().numpy(), [res.loss], TOL_F32, f"loss t={t}")
    gpu = case.state()
    diff = np.abs(gpu.logits.astype(np.float64) - st.logits)
    assert int((diff > 0.5 * w.lr_logits).sum()) <= 1e-4 * diff.size
    assert diff[diff <= 0.5 * w.lr_logits].max() <= 1e-5
    oc, om = O.project(st.logits, j0=st.j0, levels=w.K)
    gc, _ = O.project(gpu.logits, j0=gpu.j0, levels=w.K)
    keep = om >= 1e-5
    assert np.array_equal(gc[keep], oc[keep])
