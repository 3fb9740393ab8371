"""GPU parity of the warm start from supplied codes (gsq_init_logits; §3.1
"Initialization", Eq. 3-4; App. A) against the oracle: for the full grid (2- and
3-bit, group and K-Quant scales), local shift and mask x sign, random codes
(a few beyond the grid, which act as the top level), with and without the
caller's eps, at the paper's Llama strengths (alpha 3 and 6, sigma_init 0.01)
and at a large one.  Logits within fp32 rounding of three operations, j0
bit-exact, momenta zero, scales untouched; the next step then matches the
oracle's step from the same state."""
import dataclasses

import numpy as np
import pytest
import torch

from gpu_common import TOL_F32, Case, assert_close, gsq
from oracle import gsq_oracle as O
from paper_2604_18556_gb300 import configs as C

pytestmark = pytest.mark.gpu

W = C.WORKLOADS
CASES = {
    "q_proj": C.shrunk(W["llama8b_q_proj"], rows=96, cols=384, tokens=2048),
    "down_proj": C.shrunk(W["llama8b_down_proj"], rows=40, cols=640, tokens=2048),
    "moe_kquant": C.shrunk(W["moe64_kquant3"], experts=2, rows=32, cols=512, tokens=1024),
    "shift5": C.shrunk(W["llama8b_down_proj_shift5"], rows=40, cols=640, tokens=2048),
    "mask_sign": C.shrunk(W["llama8b_q_proj_mask_sign"], rows=96, cols=384, tokens=2048),
}


@pytest.mark.parametrize("alpha,sigma,with_eps", [(6.0, 0.01, True), (3.0, 0.01, False),
                                                  (2.0, 1.5, True)])
@pytest.mark.parametrize("name", list(CASES))
def test_init_from_codes_matches_oracle(name, alpha, sigma, with_eps):
    g = gsq()
    w = CASES[name]
    case = Case(w, gemm="f32")
    nr = w.experts * w.rows
    rng = np.random.default_rng(31)
    codes = rng.integers(0, w.K, (nr, w.cols)).astype(np.uint8)
    codes[0, :5] = [w.K, w.K + 3, 255, w.K - 1, 0]          # beyond the grid: act as K - 1
    eps = rng.standard_normal((w.L, nr, w.cols)).astype(np.float32) if with_eps else None
    scales_before = case.tensor(g.GSQ_T_SCALES, torch.float32).clone()
    case.layer.init_logits(torch.from_numpy(codes).cuda(),
                           None if eps is None else torch.from_numpy(eps).cuda(), alpha, sigma)
    st = case.state()
    ref = O.init_from_codes(case.prob, case.W_host, np.arange(nr), np.minimum(codes, w.K - 1),
                            eps, alpha, sigma)
    mag = sigma * (np.abs(0.0 if eps is None else eps) + abs(alpha) * 8.0 * max(1.0, np.max(np.abs(w.grid))) ** 2)
    assert np.all(np.abs(st.logits - ref.logits) <= 16 * 2.0 ** -24 * mag + 1e-30)
    assert not st.m_logits.any()
    assert torch.equal(case.tensor(g.GSQ_T_SCALES, torch.float32), scales_before)
    if w.param == "shift5":
        assert np.array_equal(st.j0, np.minimum(codes, w.K - 1))
    # the next step starts from the new logits (no stale look-ahead), as the oracle's
    loss = torch.zeros(1, device="cuda")
    case.layer.step(0, 0.8, 1.0, next_tau=0.8)              # produces a look-ahead for t = 1
    case.layer.init_logits(torch.from_numpy(codes).cuda(),
                           None if eps is None else torch.from_numpy(eps).cuda(), alpha, sigma)
    st = case.state()
    case.layer.step(1, 0.8, 1.0, loss=loss)
    torch.cuda.synchronize()
    res = O.step(case.prob, st, 1, 0.8, 1.0, update=False)
    assert_close(loss.cpu().numpy(), [res.loss], TOL_F32, "loss after warm start")


def test_init_logits_rejects_bad_arguments():
    g = gsq()
    case = Case(CASES["q_proj"], gemm="f32")
    codes = torch.zeros(CASES["q_proj"].n, dtype=torch.uint8, device="cuda")
    for args in ((None, None, 1.0, 1.0), (codes, None, float("nan"), 1.0),
                 (codes, None, 1.0, float("inf"))):
        with pytest.raises(g.GsqError) as ei:
            c, e, a, s = args
            g.gsq_init_logits(case.layer.handle, None if c is None else c.data_ptr(), e, a, s, 0)
        assert ei.value.status == g.GSQ_ERR_INVALID_ARG
