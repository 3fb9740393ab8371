"""Workspace canaries: 256 bytes after every buffer of a layer's workspace are
written at init and compared by gsq_sync_status, which reports the buffer whose
end was overrun (GSQ_ERR_STATE).  A clean run passes; a canary overwritten from
outside is caught and named."""
import pytest
import torch

from gpu_common import Case, gsq
from paper_2604_18556_gb300 import configs as C

pytestmark = pytest.mark.gpu


def test_canaries_clean_after_steps_and_named_when_overrun():
    g = gsq()
    w = C.shrunk(C.WORKLOADS["llama8b_q_proj"], rows=96, cols=384, tokens=1024)
    case = Case(w, gemm="bf16", keep_calib_host=False)
    for t in range(3):
        case.layer.step(t, 0.8, 1.0, next_tau=0.8)
    codes = torch.empty(w.n, dtype=torch.uint8, device="cuda")
    case.layer.project(codes)
    buf = torch.empty(case.layer.packed_size(), dtype=torch.uint8, device="cuda")
    case.layer.pack(buf)
    case.layer.sync_status()                                   # every canary intact
    ws = case.layer.workspace
    saved = ws[-256:].cpu().numpy().copy()
    ws[-256:] = 0                                              # the last buffer overrun
    with pytest.raises(g.GsqError) as ei:
        case.layer.sync_status()
    assert ei.value.status == g.GSQ_ERR_STATE and "'diag'" in g.gsq_last_error()
    ws[-256:] = torch.from_numpy(saved)                        # restored: clean again
    case.layer.sync_status()
    ws[256:512] = 7                                            # the first buffer (flags) overrun
    with pytest.raises(g.GsqError) as ei:
        case.layer.sync_status()
    assert ei.value.status == g.GSQ_ERR_STATE and "'flags'" in g.gsq_last_error()
