"""GPU parity of the ternary mask x sign parameterisation (§3.1, Alg. 2) against
the oracle: a mask logit and a sign logit per weight, each relaxed by a binary
GS with tied logits (-l, l), W^ = s a m~ b~ on the grid {-a, 0, a}.  Covered:
the Eq. 3 initial logits bit-exact; the soft weight, loss and both logit
gradients on random logits; the Lion update; the look-ahead forward; the hard
rule l >= 0 (zeros and negative zeros included) and packing bit-exact; a
multi-step trajectory.  Shapes: the ternary layer (fp32, calibration tokens
kept), a small q_proj-shaped layer, and K-Quant-style scales."""
import dataclasses

import numpy as np
import pytest
import torch

from gpu_common import (TOL_BF16, TOL_F32, Case, assert_close, assert_gemm_bound, check_lion,
                        check_momentum, gsq, mask_sign_grad_bounds)
from oracle import gsq_oracle as O
from paper_2604_18556_gb300 import configs as C

pytestmark = pytest.mark.gpu

W = C.WORKLOADS
SMALL = {
    "ternary": dataclasses.replace(W["ternary_256x512"], param="mask_sign"),
    "q_proj": C.shrunk(W["llama8b_q_proj_mask_sign"], rows=96, cols=384, tokens=2048),
    "moe_kquant": dataclasses.replace(
        C.shrunk(W["moe64_kquant3"], experts=3, rows=64, cols=512, tokens=1024),
        grid=C.GRID_TERNARY, param="mask_sign"),
}
TAU = {"ternary": 1.0, "q_proj": 0.55, "moe_kquant": 0.8}


def _n(w):
    return w.experts * w.rows * w.cols


def _randomise(case, seed):
    g = gsq()
    w = case.w
    rng = np.random.default_rng(seed)
    L = rng.standard_normal((2, w.experts * w.rows, w.cols)).astype(np.float32)
    case.layer.set_tensor(g.GSQ_T_LOGITS, torch.from_numpy(L).cuda())
    return case.state()


@pytest.mark.parametrize("name", list(SMALL))
def test_mask_sign_init_bit_exact(name):
    case = Case(SMALL[name], gemm="f32")
    st, ref = case.state(), case.oracle_init()
    assert st.logits.shape[0] == 2
    assert np.array_equal(st.logits, ref.logits)
    assert np.array_equal(st.scales, ref.scales)
    assert not st.m_logits.any() and not st.m_scales.any()
    if SMALL[name].scale_mode == "kquant2":
        assert np.array_equal(st.kq_d, ref.kq_d) and np.array_equal(st.kq_sc, ref.kq_sc)


@pytest.mark.parametrize("noise", [True, False])
@pytest.mark.parametrize("name", list(SMALL))
def test_mask_sign_forward_soft_weight(name, noise):
    w = SMALL[name]
    case = Case(w, gemm="f32", noise=noise)
    st = _randomise(case, 21)
    what = torch.empty(_n(w), device="cuda")
    case.layer.forward(7, 0.7, 1.3, what=what)
    ref = O.forward(case.prob, st, 7, 0.7, 1.3)
    assert_close(what.cpu().numpy(), ref.What, TOL_F32, "W^")
    assert_close(case.D(), ref.D, TOL_F32, "D")


@pytest.mark.parametrize("gemm", ["f32", "bf16"])
@pytest.mark.parametrize("name", list(SMALL))
def test_mask_sign_step_loss_and_gradients(name, gemm):
    w = SMALL[name]
    case = Case(w, gemm=gemm)
    st = _randomise(case, 22)
    tol = TOL_F32 if gemm == "f32" else TOL_BF16
    n = _n(w)
    loss = torch.zeros(1, device="cuda")
    gl = torch.empty(2 * n, device="cuda")
    gs = torch.zeros(n // w.group, device="cuda")
    case.layer.step(3, TAU[name], 1.0, loss=loss, grad_logits=gl, grad_scales=gs)
    torch.cuda.synchronize()
    ref = O.step(case.prob, st.copy(), 3, TAU[name], 1.0, update=False)
    assert_close(loss.cpu().numpy(), [ref.loss], tol, "loss")
    assert_close(case.G(), ref.G, tol, "G")
    got_l = gl.cpu().numpy().astype(np.float64).reshape(ref.d_logits.shape)
    if gemm == "f32":
        assert_close(got_l, ref.d_logits, tol, "dL/dlogits")
        if ref.d_scales is not None:
            assert_close(gs.cpu().numpy(), ref.d_scales, tol, "dL/dscales")
    else:
        bl, bs = mask_sign_grad_bounds(ref, case.prob, TAU[name], 1.0, tol)
        assert np.all(np.abs(got_l - ref.d_logits) <= bl * 1.0001 + 1e-30), "dL/dlogits"
        if ref.d_scales is not None:
            err = np.abs(gs.cpu().numpy().astype(np.float64).reshape(ref.d_scales.shape) - ref.d_scales)
            assert np.all(err <= bs * 1.0001 + 1e-30), "dL/dscales"
        D, H, G = case.D(), case.H_operand(), case.G()
        rows = np.arange(w.experts * w.rows)
        for e in range(w.experts):
            sel = rows // w.rows == e
            assert_gemm_bound(G[sel], D[sel], H[e], f"tcgen05 GEMM vs its operands, expert {e}")


@pytest.mark.parametrize("gemm", ["f32", "bf16"])
@pytest.mark.parametrize("name", list(SMALL))
def test_mask_sign_step_update(name, gemm):
    w = SMALL[name]
    case = Case(w, gemm=gemm)
    _randomise(case, 23)
    tol = TOL_F32 if gemm == "f32" else TOL_BF16
    for t in range(2):
        loss = torch.zeros(1, device="cuda")
        before = case.state()
        case.layer.step(t, TAU[name], 1.0, loss=loss)
        torch.cuda.synchronize()
        st_sync = before.copy()
        res = O.step(case.prob, st_sync, t, TAU[name], 1.0, update=True)
        gpu = case.state()
        assert_close(loss.cpu().numpy(), [res.loss], tol, f"loss t={t}")
        c_l = w.beta1 * before.m_logits.astype(np.float64) + (1 - w.beta1) * res.d_logits
        check_lion(gpu.logits, st_sync.logits, before.logits, c_l, w.lr_logits, 2 * tol, "logits")
        if gemm == "f32":
            gb_l = tol * (np.abs(res.d_logits) + np.sqrt(np.mean(res.d_logits ** 2)))
            gb_s = None if res.d_scales is None else \
                tol * (np.abs(res.d_scales) + np.sqrt(np.mean(res.d_scales ** 2)))
        else:
            gb_l, gb_s = mask_sign_grad_bounds(res, case.prob, TAU[name], 1.0, tol)
        check_momentum(gpu.m_logits, st_sync.m_logits, gb_l, w.beta2, "logit momentum")
        if res.d_scales is not None:
            c_s = w.beta1 * before.m_scales.astype(np.float64) + (1 - w.beta1) * res.d_scales
            check_lion(gpu.scales, st_sync.scales, before.scales, c_s, w.lr_scales, 2 * tol, "scales")
            check_momentum(gpu.m_scales, st_sync.m_scales, gb_s, w.beta2, "scale momentum")
        else:
            assert np.array_equal(gpu.scales, before.scales)


@pytest.mark.parametrize("name", ["q_proj", "moe_kquant"])
def test_mask_sign_lookahead_is_bit_identical(name):
    w = SMALL[name]
    a, b = Case(w, gemm="bf16"), Case(w, gemm="bf16")
    for t in range(4):
        la, lb = torch.zeros(1, device="cuda"), torch.zeros(1, device="cuda")
        a.layer.step(t, w.tau(t), 1.0, next_tau=w.tau(t + 1), next_kappa=1.0, loss=la)
        b.layer.step(t, w.tau(t), 1.0, loss=lb)
        torch.cuda.synchronize()
        assert la.item() == lb.item()
        sa, sb = a.state(), b.state()
        for f in ("logits", "m_logits", "scales", "m_scales"):
            assert np.array_equal(getattr(sa, f), getattr(sb, f)), (t, f)


@pytest.mark.parametrize("name", list(SMALL))
def test_mask_sign_project_and_pack_bit_exact(name):
    g = gsq()
    w = SMALL[name]
    case = Case(w, gemm="bf16")
    for t in range(2):
        case.layer.step(t, 0.3, 1.0, next_tau=0.3)
    L = _randomise(case, 24).logits.copy()
    L[:, :, ::7] = 0.0                      # the rule's boundary: l = 0 is "on" / "+"
    L[:, :, 3::11] = -0.0
    case.layer.set_tensor(g.GSQ_T_LOGITS, torch.from_numpy(L.copy()).cuda())
    n = _n(w)
    codes = torch.empty(n, dtype=torch.uint8, device="cuda")
    margin = torch.empty(n, device="cuda")
    case.layer.project(codes, margin)
    st = case.state()
    oc, om = O.project(st.logits, mask_sign=True)
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


def test_mask_sign_trajectory():
    """The ternary layer (fp32, tokens kept) for 40 steps, GPU and oracle each
    on their own trajectory: per-step losses within 1e-4, final logits within
    the Lion flip allowance, final codes bit-exact where the margin is >= 1e-5."""
    w = dataclasses.replace(SMALL["ternary"], steps=40, tau0=1.0, tau1=0.2)
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
    oc, om = O.project(st.logits, mask_sign=True)
    gc, _ = O.project(gpu.logits, mask_sign=True)
    keep = om >= 1e-5
    assert np.array_equal(gc[keep], oc[keep])
    assert_close(gpu.scales, st.scales, TOL_F32, "scales after 40 steps")
