"""GPU parity of gsq_diagnose against the oracle's diagnostics: displacement and
margin histograms bit-exact (integer results of fp32 decisions), mean noise-free
max-probability to fp32 rounding, for every parameterisation and both scale
modes, after a few steps and after a warm start from supplied codes."""
import dataclasses

import numpy as np
import pytest
import torch

from gpu_common import Case, gsq
from oracle import gsq_oracle as O
from paper_2604_18556_gb300 import configs as C

pytestmark = pytest.mark.gpu

W = C.WORKLOADS
CASES = {
    "full": C.shrunk(W["llama8b_q_proj"], rows=96, cols=384, tokens=1024),
    "kquant": C.shrunk(W["moe64_kquant3"], experts=2, rows=32, cols=512, tokens=1024),
    "shift5": C.shrunk(W["llama8b_down_proj_shift5"], rows=40, cols=640, tokens=1024),
    "mask_sign": C.shrunk(W["llama8b_q_proj_mask_sign"], rows=96, cols=384, tokens=1024),
}


def _check(case, code0, tau, kappa):
    got = case.layer.diagnose(tau, kappa)
    st = case.state()
    # the entry point takes tau and kappa as fp32
    disp, pmax, marg = O.diagnostics(case.prob, st, code0, float(np.float32(tau)),
                                     float(np.float32(kappa)))
    assert got["displacement"] == disp.tolist()
    assert got["margin"] == marg.tolist()
    # the kernel evaluates each max-probability in fp32 (a few ulp), then averages
    # in double: the mean agrees to about the fp32 unit roundoff
    assert abs(got["mean_max_prob"] - pmax) <= 1e-6 * pmax
    return got


@pytest.mark.parametrize("name", list(CASES))
def test_diagnostics_after_steps(name):
    w = CASES[name]
    case = Case(w, gemm="bf16", keep_calib_host=False)
    st0 = case.oracle_init()
    code0, _ = O.project(st0.logits, j0=st0.j0, levels=w.K, mask_sign=w.param == "mask_sign")
    rng = np.random.default_rng(8)
    L = case.logits() + 1.5 * rng.standard_normal(case.logits().shape).astype(np.float32)
    case.layer.set_tensor(gsq().GSQ_T_LOGITS, torch.from_numpy(L).cuda())
    for t in range(3):
        case.layer.step(t, 0.7, 1.0, next_tau=0.7)
    got = _check(case, code0, 0.7, 1.0)
    assert sum(got["displacement"]) == w.n and sum(got["margin"]) == w.n
    _check(case, code0, 0.05, 2.0)                 # near saturation


@pytest.mark.parametrize("name", ["full", "shift5", "mask_sign"])
def test_diagnostics_after_warm_start(name):
    w = CASES[name]
    case = Case(w, gemm="bf16", keep_calib_host=False)
    rng = np.random.default_rng(9)
    codes = rng.integers(0, w.K, w.n).astype(np.uint8)
    case.layer.init_logits(torch.from_numpy(codes).cuda(), None, alpha=3.0, sigma=0.5)
    got = _check(case, codes.reshape(-1, w.cols), 1.0, 1.0)
    assert got["displacement"][0] == w.n           # the prior's mode is the supplied code
