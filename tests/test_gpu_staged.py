"""The staged backward (input streams brought into shared memory by bulk asynchronous
copies, one tile of 1,024 weights ahead) against the same kernel body reading its
streams with direct global loads (GSQ_FLAG_UNSTAGED): both run identical arithmetic
on every weight, so every updated tensor and the look-ahead D must agree bit for
bit; the loss, a reduction whose order follows each kernel's grid, to 1e-6.  Shapes cover blocks that reuse both stages several
times, a ragged last tile read with direct loads, a layer smaller than one tile,
fp32 and bf16 weights, scale groups of 4 to 128, frozen K-Quant scales, 2 to 8
logits per weight (momenta staged up to 5, loaded directly above), local shift and
mask x sign.  Each case runs under every staging plan that applies (forced through
GSQ_STAGED_PLAN, which also lifts the rule that small layers are not staged) and
under the layer's own choice."""
from dataclasses import replace

import numpy as np
import pytest
import torch

from gpu_common import Case, gsq
from paper_2604_18556_gb300 import configs as C

pytestmark = pytest.mark.gpu

W = C.WORKLOADS
Q = W["llama8b_q_proj"]
CASES = {
    # 1,278,720 weights: 1,248 full tiles (about 4 per block) and a ragged 768-weight tile
    "k4_ragged_multi_tile": C.shrunk(Q, rows=999, cols=1280, tokens=2048),
    # 768 weights: no full tile, the whole layer through the direct-load tail
    "k4_below_one_tile": C.shrunk(Q, rows=3, cols=256, tokens=1024),
    "k4_g4": replace(C.shrunk(Q, rows=130, cols=1024, tokens=2048), group=4),
    "k2_g32": replace(C.shrunk(Q, rows=257, cols=512, tokens=2048), group=32, grid=(-0.5, 0.5)),
    "k3_fp32_w": C.shrunk(W["ternary_256x512"], rows=300, cols=512),
    "k8_momenta_direct": C.shrunk(W["llama8b_down_proj"], rows=300, cols=1792, tokens=2048),
    "kquant_frozen": C.shrunk(W["moe64_kquant3"], experts=2, rows=96, cols=2048, tokens=1024),
    "shift5": C.shrunk(W["llama8b_down_proj_shift5"], rows=200, cols=1536, tokens=2048),
    "mask_sign": C.shrunk(W["llama8b_q_proj_mask_sign"], rows=257, cols=1024, tokens=2048),
}
TAU = 0.7


def _randomise(case, seed):
    g = gsq()
    w = case.w
    rng = np.random.default_rng(seed)
    Lg = (1.5 * rng.standard_normal((w.L, w.experts * w.rows, w.cols))).astype(np.float32)
    case.layer.set_tensor(g.GSQ_T_LOGITS, torch.from_numpy(Lg).cuda())


PLANS = ("auto", "1", "3", "5")


@pytest.mark.parametrize("plan", PLANS)
@pytest.mark.parametrize("name", list(CASES))
def test_staged_backward_is_bit_identical(name, plan, monkeypatch):
    g = gsq()
    w = CASES[name]
    if plan == "3" and w.L > 4:
        pytest.skip("plan 3 serves up to 4 logits per weight")
    if plan != "auto":
        monkeypatch.setenv("GSQ_STAGED_PLAN", plan)
    gemm = "f32" if w.w_dtype == "f32" else "bf16"
    staged = Case(w, gemm=gemm)
    direct = Case(w, gemm=gemm, unstaged=True)
    for c in (staged, direct):
        _randomise(c, 21)
    start = staged.logits()
    d_dtype = torch.bfloat16 if gemm == "bf16" else torch.float32
    for t in range(3):
        la, lb = torch.zeros(1, device="cuda"), torch.zeros(1, device="cuda")
        staged.layer.step(t, TAU, 1.0, next_tau=TAU, next_kappa=1.0, loss=la)
        direct.layer.step(t, TAU, 1.0, next_tau=TAU, next_kappa=1.0, loss=lb)
        torch.cuda.synchronize()
        staged.layer.sync_status()
        direct.layer.sync_status()
        assert abs(la.item() - lb.item()) <= 1e-6 * abs(lb.item()), (t, la.item(), lb.item())
        for which in (g.GSQ_T_LOGITS, g.GSQ_T_MOM_LOGITS, g.GSQ_T_SCALES, g.GSQ_T_MOM_SCALES):
            a = staged.tensor(which, torch.float32)
            b = direct.tensor(which, torch.float32)
            assert torch.equal(a.view(torch.int32), b.view(torch.int32)), (t, which)
        Da = staged.tensor(g.GSQ_T_D, d_dtype)
        Db = direct.tensor(g.GSQ_T_D, d_dtype)
        assert torch.equal(Da.view(torch.int16 if gemm == "bf16" else torch.int32),
                           Db.view(torch.int16 if gemm == "bf16" else torch.int32)), t
    # the steps did update the state
    assert not np.array_equal(staged.logits(), start)


def test_kernel_names_follow_the_layer():
    """gsq_kernel_name reports what gsq_step launches: staged up to 4 logits per weight
    on layers with more tiles than resident blocks, direct loads with 5 (local shift),
    on request and on small layers; the CTA-pair contraction by default."""
    g = gsq()
    big = C.shrunk(Q, rows=999, cols=1280, tokens=2048)
    cases = [(big, {}, "k_backward_staged"),
             (big, {"unstaged": True}, "k_backward"),
             (CASES["shift5"], {}, "k_backward"),
             (CASES["k4_below_one_tile"], {}, "k_backward")]
    for w, kw, want in cases:
        case = Case(w, gemm="bf16", **kw)
        assert case.layer.kernel_name(g.GSQ_K_BACKWARD) == want, (w.name, kw)
        assert case.layer.kernel_name(g.GSQ_K_GEMM) == "k_tc_gemm_pair"
        assert case.layer.kernel_name(g.GSQ_K_PROJECT) is None
    f32 = Case(CASES["k3_fp32_w"], gemm="f32")
    assert f32.layer.kernel_name(g.GSQ_K_GEMM) == "k_simt_gemm"
