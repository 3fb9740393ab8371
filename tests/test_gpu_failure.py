"""Bounded device-side waits: every mbarrier wait of the persistent kernels gives up
after 2 s of %globaltimer, records an error code and lets its kernel finish, and
gsq_sync_status turns the code into GSQ_ERR_TIMEOUT.  The test hook GSQ_TEST_STALL
makes a layer's kernel skip one copy, so a wait runs out on something nothing will
complete (no fault, no trap, no unbounded spin); the context stays usable and the
next layer steps cleanly."""
import pytest
import torch

from gpu_common import Case, gsq
from paper_2604_18556_gb300 import configs as C

pytestmark = pytest.mark.gpu

# 1,278,720 weights: more tiles than the staged backward's blocks, so every block
# reaches its second stage; 999 x 1280 also spans several GEMM tiles
W = C.shrunk(C.WORKLOADS["llama8b_q_proj"], rows=999, cols=1280, tokens=2048)


@pytest.mark.parametrize("stall,pair,code,kernel", [
    ("backward", "1", 0x7C03, "k_backward_staged"),
    ("gemm", "1", 0x7C04, "k_tc_gemm_pair"),
    ("gemm", "2", 0x7C05, "k_tc_gemm_quad"),
    ("gemm", "0", 0x7C01, "k_tc_gemm"),
])
def test_bounded_wait_reports_timeout(stall, pair, code, kernel, monkeypatch):
    g = gsq()
    monkeypatch.setenv("GSQ_GEMM_PAIR", pair)
    monkeypatch.setenv("GSQ_TEST_STALL", stall)
    case = Case(W, gemm="bf16", keep_calib_host=False)
    which = g.GSQ_K_BACKWARD if stall == "backward" else g.GSQ_K_GEMM
    assert case.layer.kernel_name(which) == kernel
    case.layer.step(0, 0.7, 1.0, next_tau=0.7)
    with pytest.raises(g.GsqError) as ei:
        case.layer.sync_status()
    assert ei.value.status == g.GSQ_ERR_TIMEOUT
    assert f"0x{code:x}" in g.gsq_last_error().lower()
    case.layer.sync_status()                          # the error word was cleared
    case.layer.close()
    # the context stays usable: a layer without the hook steps and reports no error
    monkeypatch.delenv("GSQ_TEST_STALL")
    fresh = Case(W, gemm="bf16", keep_calib_host=False)
    loss = torch.zeros(1, device="cuda")
    fresh.layer.step(0, 0.7, 1.0, next_tau=0.7, loss=loss)
    fresh.layer.step(1, 0.7, 1.0, next_tau=0.7, loss=loss)
    torch.cuda.synchronize()
    fresh.layer.sync_status()
    assert torch.isfinite(loss).all()
