"""GPU parity of the step on per-step calibration tokens with gradient
accumulation over resampled noise (gsq_step_tokens; §3.3 "Objective",
"Gradient accumulation") against the oracle's step_microbatches: every
micro-batch's loss, and after the last micro-batch the Lion update with the
mean gradient, for two consecutive steps (so the look-ahead crosses a step
boundary and the momenta are nonzero), in both GEMM precisions and all three
parameterisations.  Shapes span several GEMM tiles with ragged tails (rows not
a multiple of 128, tokens not a multiple of 256).  Also: the call order is
enforced, and such a layer refuses the plain gsq_step."""
import dataclasses

import numpy as np
import pytest
import torch

from gpu_common import TOL_BF16, TOL_F32, Case, assert_close, assert_gemm_bound, check_lion, gsq
from oracle import gsq_oracle as O
from paper_2604_18556_gb300 import configs as C
from paper_2604_18556_gb300 import inputs

pytestmark = pytest.mark.gpu

BASE = C.shrunk(C.WORKLOADS["llama8b_q_proj_tokens"], rows=136, cols=384, tokens=328)
CASES = {
    "full": dataclasses.replace(BASE, micro=3),
    "shift5": dataclasses.replace(BASE, grid=C.GRID_3BIT_SYM, param="shift5", micro=2),
    "mask_sign": dataclasses.replace(BASE, grid=C.GRID_TERNARY, param="mask_sign", micro=3),
    "single": dataclasses.replace(BASE, micro=1),
}


def _batches(w, step):
    return [inputs.make_token_batch(w, step, j, device="cuda") for j in range(w.micro)]


@pytest.mark.parametrize("gemm,route", [("f32", "direct"), ("bf16", "direct"), ("bf16", "gram")])
@pytest.mark.parametrize("name", list(CASES))
def test_token_steps_match_oracle(name, gemm, route, monkeypatch):
    """route: the tensor-core contraction as Y = D X^T, G = 2 Y X ("direct") or through the
    micro-batch's Gram matrix H = X^T X, G = 2 D H ("gram"); the fp32 path is direct."""
    monkeypatch.setenv("GSQ_TOKEN_ROUTE", route)
    _check_token_steps(CASES[name], gemm)


@pytest.mark.parametrize("route", ["direct", "gram"])
@pytest.mark.parametrize("mode,kernel", [("0", "k_tc_gemm"), ("1", "k_tc_gemm_pair"),
                                         ("2", "k_tc_gemm_quad")])
def test_token_steps_on_every_contraction_kernel(mode, kernel, route, monkeypatch):
    """Both token contractions of either route (Y = D X^T with bf16 output and G = 2 Y X
    with fp32 output; or H = X^T X with bf16 output and G = 2 D H) on single CTAs, CTA
    pairs and clusters of two pairs sharing operand tiles by TMA multicast, against the
    oracle."""
    monkeypatch.setenv("GSQ_GEMM_PAIR", mode)
    monkeypatch.setenv("GSQ_TOKEN_ROUTE", route)
    w = dataclasses.replace(CASES["full"], rows=600)   # three 256-row tiles: a ragged cluster
    case = _check_token_steps(w, "bf16")
    assert case.layer.kernel_name(gsq().GSQ_K_GEMM) == kernel


@pytest.mark.parametrize("sym", ["1", "0"], ids=["upper_triangle", "every_tile"])
@pytest.mark.parametrize("mode", ["0", "1", "2"])
@pytest.mark.parametrize("cols", [384, 1152])
def test_gram_route_contractions(cols, mode, sym, monkeypatch):
    """The Gram route on the kernels' own bf16 operands, two experts: the micro-batch's
    H = X^T X (fp32 accumulation of the bf16 tokens, then one rounding to bf16) within
    the accumulation bound plus that rounding, and exactly symmetric, whether formed
    from the tiles of its upper triangle and mirrored (default) or from every tile;
    G = 2 D H within the accumulation bound of the bf16 D and H; the loss as 1/2 sum
    D G.  1,152 inputs: ragged tiles on both sides of the diagonal."""
    monkeypatch.setenv("GSQ_TOKEN_ROUTE", "gram")
    monkeypatch.setenv("GSQ_TOKEN_SYM", sym)
    monkeypatch.setenv("GSQ_GEMM_PAIR", mode)
    w = dataclasses.replace(BASE, experts=2, rows=600, cols=cols, micro=1)
    case = Case(w, gemm="bf16")
    g = gsq()
    X = inputs.make_token_batch(w, 0, 0, device="cuda")
    loss = torch.zeros(1, device="cuda")
    case.layer.step_tokens(0, 0, 1, w.tau(0), X, loss=loss)   # no look-ahead: D stays
    torch.cuda.synchronize()
    case.layer.sync_status()
    Cc, T = w.cols, X.shape[1]
    Hj = case.tensor(g.GSQ_T_H, torch.bfloat16).float().view(w.experts, Cc, Cc).cpu().numpy()
    Xb = X.bfloat16().double().cpu().numpy()
    D, G = case.D(), case.G()
    rows = np.arange(w.experts * w.rows)
    for e in range(w.experts):
        assert np.array_equal(Hj[e], Hj[e].T), ("H = X^T X not symmetric", e)
        exact = Xb[e].T @ Xb[e]
        absum = np.abs(Xb[e]).T @ np.abs(Xb[e])
        bound = 1.01 * T * 2.0 ** -24 * absum + 2.0 ** -8 * np.abs(exact) + 1e-30
        worst = float((np.abs(Hj[e] - exact) / bound).max())
        assert worst <= 1.0, ("H = X^T X", e, worst)
        sel = rows // w.rows == e
        assert_gemm_bound(G[sel], D[sel], Hj[e], f"G = 2 D H, expert {e}")
    assert abs(loss.item() - 0.5 * np.sum(D.astype(np.float64) * G)) <= 1e-5 * abs(loss.item())


def _check_token_steps(w, gemm):
    case = Case(w, gemm=gemm)
    tol = TOL_F32 if gemm == "f32" else TOL_BF16
    rng = np.random.default_rng(5)
    L = (0.7 * rng.standard_normal(case.logits().shape)).astype(np.float32)
    case.layer.set_tensor(gsq().GSQ_T_LOGITS, torch.from_numpy(L).cuda())
    for step in range(2):
        Xs = _batches(w, step)
        before = case.state()
        losses = torch.zeros(w.micro, device="cuda")
        tau, tau_next = w.tau(step), w.tau(step + 1)
        for j, X in enumerate(Xs):
            case.layer.step_tokens(step, j, w.micro, tau, X, next_tau=tau_next,
                                   loss=losses[j:j + 1])
            if j + 1 < w.micro:   # the state only changes after the last micro-batch
                assert np.array_equal(case.state().logits, before.logits)
        torch.cuda.synchronize()
        st = before.copy()
        res = O.step_microbatches(case.prob, st, step, [X.double().cpu().numpy() for X in Xs],
                                  tau, 1.0, update=True)
        assert_close(losses.cpu().numpy(), res.losses, tol, f"micro-batch losses, step {step}")
        gpu = case.state()
        c_l = w.beta1 * before.m_logits.astype(np.float64) + (1 - w.beta1) * res.d_logits
        check_lion(gpu.logits, st.logits, before.logits, c_l, w.lr_logits, 2 * tol, "logits")
        if gemm == "f32":
            assert_close(gpu.m_logits, st.m_logits, tol, "logit momentum (mean gradient)")
            if res.d_scales is not None:
                assert_close(gpu.m_scales, st.m_scales, tol, "scale momentum")
        else:
            # the mean gradient through bf16 GEMMs: tensor-level relative error
            for a, b, what in ((gpu.m_logits, st.m_logits, "logit momentum"),
                               (gpu.m_scales, st.m_scales, "scale momentum")):
                d = np.linalg.norm(a.astype(np.float64) - b) / np.linalg.norm(b)
                assert d <= tol, (what, d)
    case.layer.sync_status()
    return case


def test_token_steps_enforce_order_and_mode():
    g = gsq()
    w = CASES["full"]
    case = Case(w, gemm="f32")
    X = inputs.make_token_batch(w, 0, 0, device="cuda")
    case.layer.step_tokens(0, 0, 3, 0.9, X)
    with pytest.raises(g.GsqError) as ei:           # micro-batch 1 skipped
        case.layer.step_tokens(0, 2, 3, 0.9, X)
    assert ei.value.status == g.GSQ_ERR_STATE
    for micro, n_micro, Xbad in ((3, 3, X), (0, 0, X), (0, 1, X[:, :12]), (0, 1, X[:, :0])):
        with pytest.raises(g.GsqError) as ei:
            case.layer.step_tokens(0, micro, n_micro, 0.9, Xbad)
        assert ei.value.status == g.GSQ_ERR_INVALID_ARG
    with pytest.raises(g.GsqError) as ei:           # more tokens than the workspace holds
        case.layer.step_tokens(0, 0, 1, 0.9, torch.zeros(1, w.tokens + 8, w.cols, device="cuda"))
    assert ei.value.status == g.GSQ_ERR_INVALID_ARG
    with pytest.raises(g.GsqError) as ei:           # the H-based step needs an H
        case.layer.step(0, 0.9)
    assert ei.value.status == g.GSQ_ERR_INVALID_ARG
    case.layer.sync_status()
