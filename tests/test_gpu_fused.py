"""The fused tensor-core step (GSQ_FLAG_FUSED: the loss contraction with the backward,
Lion and the look-ahead forward as its epilogue): its contraction against exact products of its
own bf16 operands (G kept on request), the loss, Lion updates against the oracle for
every parameterisation and for scale groups narrower than, equal to and wider than a
warp (4, 32, 64, 128 columns), ragged tiles in rows and columns, several experts, and
agreement with the separate GEMM + backward kernels."""
from dataclasses import replace

import numpy as np
import pytest
import torch

from gpu_common import (TOL_BF16, Case, assert_close, assert_gemm_bound, bf16_operand_bounds,
                        check_lion, check_momentum, grad_bounds, gsq, mask_sign_grad_factors)
from oracle import gsq_oracle as O
from paper_2604_18556_gb300 import configs as C

pytestmark = pytest.mark.gpu

W = C.WORKLOADS
BASE = C.shrunk(W["llama8b_q_proj"], rows=200, cols=384, tokens=2048)
CASES = {
    # rows 200 = one full and one ragged 128-row tile; columns 384 = 3 column tiles
    "full_g128": BASE,
    "full_g64": replace(BASE, group=64),
    "full_g32": replace(BASE, group=32),
    "full_g4": replace(BASE, group=4),
    # columns 320: a ragged 128-column tile (64 of 128 lanes idle), 3 experts
    "experts_ragged": C.shrunk(W["llama70b_gate_proj"], experts=3, rows=70, cols=320, tokens=2048),
    "kquant_frozen": C.shrunk(W["moe64_kquant3"], experts=2, rows=96, cols=512, tokens=1024),
    "shift5": C.shrunk(W["llama8b_down_proj_shift5"], rows=150, cols=256, tokens=2048),
    "mask_sign": C.shrunk(W["llama8b_q_proj_mask_sign"], rows=136, cols=384, tokens=2048),
    "mask_sign_g32": replace(C.shrunk(W["llama8b_q_proj_mask_sign"], rows=66, cols=256, tokens=2048),
                             group=32),
}
TAU = 0.6


def _randomise(case, seed):
    """Spread the logits so that every level carries probability mass."""
    g = gsq()
    w = case.w
    rng = np.random.default_rng(seed)
    Lg = (1.5 * rng.standard_normal((w.L, w.experts * w.rows, w.cols))).astype(np.float32)
    case.layer.set_tensor(g.GSQ_T_LOGITS, torch.from_numpy(Lg).cuda())
    return case.state()


@pytest.mark.parametrize("name", list(CASES))
def test_fused_contraction_and_loss(name):
    """G kept by the fused kernel equals the exact product of its own bf16 operands
    within fp32 accumulation, and the loss is 1/2 sum D G and the oracle's."""
    w = CASES[name]
    case = Case(w, gemm="bf16", keep_g=True, fused=True)
    st = _randomise(case, 5)
    loss = torch.zeros(1, device="cuda")
    case.layer.step(4, TAU, 1.0, loss=loss)        # no look-ahead: D stays step 4's
    torch.cuda.synchronize()
    D, H, G = case.D(), case.H_operand(), case.G()
    rows = np.arange(w.experts * w.rows)
    for e in range(w.experts):
        sel = rows // w.rows == e
        assert_gemm_bound(G[sel], D[sel], H[e], f"fused contraction, expert {e}")
    half = 0.5 * np.sum(D.astype(np.float64) * G)
    assert abs(loss.item() - half) <= 1e-5 * abs(half), (loss.item(), half)
    ref = O.step(case.prob, st.copy(), 4, TAU, 1.0, update=False)
    assert_close(loss.cpu().numpy(), [ref.loss], TOL_BF16, "loss")
    # G within the worst-case error of one bf16 rounding of each operand
    zmax = float(np.max(np.abs(st.logits.astype(np.float64) + ref.fw.g))) / TAU
    zmax *= 2 if w.param == "mask_sign" else 1
    dD, _, gb = bf16_operand_bounds(ref, case.prob, zmax)
    assert np.all(np.abs(D - ref.fw.D) <= dD), "D operand"
    assert np.all(np.abs(G - ref.G) <= gb), "G"


@pytest.mark.parametrize("name", list(CASES))
def test_fused_updates_match_oracle(name):
    """Two fused steps with look-ahead, each against the oracle's step from the GPU's
    state before it (logits, momenta, scales and scale momenta)."""
    w = CASES[name]
    case = Case(w, gemm="bf16", fused=True)
    _randomise(case, 9)
    for t in range(2):
        before = case.state()
        loss = torch.zeros(1, device="cuda")
        case.layer.step(t, TAU, 1.0, next_tau=TAU, next_kappa=1.0, loss=loss)
        torch.cuda.synchronize()
        orc = before.copy()
        res = O.step(case.prob, orc, t, TAU, 1.0, update=True)
        gpu = case.state()
        assert_close(loss.cpu().numpy(), [res.loss], TOL_BF16, f"loss t={t}")
        c_l = w.beta1 * before.m_logits.astype(np.float64) + (1 - w.beta1) * res.d_logits
        check_lion(gpu.logits, orc.logits, before.logits, c_l, w.lr_logits, 2 * TOL_BF16, "logits")
        if w.param == "mask_sign":
            Gs = TOL_BF16 * (np.abs(res.G) + np.sqrt(np.mean(res.G ** 2)))
            gb_l = mask_sign_grad_factors(res, case.prob, TAU, 1.0) * Gs[None] + \
                TOL_BF16 * np.abs(res.d_logits)
            gb_s = None
        else:
            q = O.level_values(case.prob, before) if w.param == "shift5" else None
            f, gscale, bs = grad_bounds(res, case.prob, TOL_BF16, q)
            gb_l = (1.0 / TAU) * f * gscale[None] + TOL_BF16 * np.abs(res.d_logits)
            gb_s = None if res.d_scales is None else bs + TOL_BF16 * np.abs(res.d_scales)
        check_momentum(gpu.m_logits, orc.m_logits, gb_l, w.beta2, "logit momentum")
        if res.d_scales is not None:
            c_s = w.beta1 * before.m_scales.astype(np.float64) + (1 - w.beta1) * res.d_scales
            check_lion(gpu.scales, orc.scales, before.scales, c_s, w.lr_scales, 2 * TOL_BF16, "scales")
            if gb_s is not None:
                check_momentum(gpu.m_scales, orc.m_scales, gb_s, w.beta2, "scale momentum")
        else:
            assert np.array_equal(gpu.scales, before.scales)


@pytest.mark.parametrize("name", ["full_g128", "full_g4", "experts_ragged", "shift5", "mask_sign"])
def test_fused_agrees_with_separate_kernels(name):
    """Three steps with look-ahead, fused against the separate GEMM + backward kernels
    from the same state: logits and momenta agree to rounding (Lion sign flips only
    where the momentum mix is below the tolerance), the look-ahead D to one bf16
    rounding, the losses to fp32 summation order."""
    w = CASES[name]
    fused = Case(w, gemm="bf16", fused=True)
    sep = Case(w, gemm="bf16")
    g = gsq()
    for c in (fused, sep):
        _randomise(c, 13)
    for t in range(3):
        before = sep.state()
        la, lb = torch.zeros(1, device="cuda"), torch.zeros(1, device="cuda")
        fused.layer.step(t, TAU, 1.0, next_tau=TAU, next_kappa=1.0, loss=la)
        sep.layer.step(t, TAU, 1.0, next_tau=TAU, next_kappa=1.0, loss=lb)
        torch.cuda.synchronize()
        assert abs(la.item() - lb.item()) <= 1e-5 * abs(lb.item()), (t, la.item(), lb.item())
        a, b = fused.state(), sep.state()
        # a Lion step moves a logit by lr (sign) plus the decay: apart from rounding
        # the two paths differ only where sign(c) flipped, by at most 2 lr
        diff = np.abs(a.logits.astype(np.float64) - b.logits)
        mag = np.maximum(np.maximum(np.abs(b.logits), np.abs(before.logits)), w.lr_logits)
        flip = diff > 4 * np.spacing(mag.astype(np.float32))
        assert np.all(diff[flip] <= 2.002 * w.lr_logits), t
        assert flip.sum() <= 1e-3 * a.logits.size, (t, int(flip.sum()))
        scale = np.sqrt(np.mean(b.m_logits.astype(np.float64) ** 2))
        assert np.max(np.abs(a.m_logits - b.m_logits)) <= 1e-3 * scale, t
        Da = fused.layer.get_tensor(g.GSQ_T_D, torch.bfloat16).float().cpu().numpy()
        Db = sep.layer.get_tensor(g.GSQ_T_D, torch.bfloat16).float().cpu().numpy()
        assert np.max(np.abs(Da - Db)) <= 2 * 2.0 ** -8 * np.max(np.abs(Db)), t


def test_g_is_not_readable_after_a_fused_step_without_keep():
    g = gsq()
    w = CASES["full_g128"]
    case = Case(w, gemm="bf16", fused=True)
    case.layer.step(0, TAU, 1.0)
    torch.cuda.synchronize()
    with pytest.raises(g.GsqError) as ei:
        case.layer.get_tensor(g.GSQ_T_G, torch.float32)
    assert ei.value.status == g.GSQ_ERR_STATE
    case.layer.close()
