"""Parity at the workloads' full sizes, in the launch configuration the benchmark
times (bf16 tensor-core GEMM, fused backward with look-ahead).  The oracle
follows a sample of rows exactly (rows are independent given H); quantities
that couple all rows are checked through properties that hold at any size
(L = 1/2 sum D*G for the GPU's own D and G)."""
import numpy as np
import pytest
import torch

from gpu_common import TOL_BF16, Case, assert_close, assert_gemm_bound, assert_grad_close, gsq
from oracle import gsq_oracle as O
from paper_2604_18556_gb300 import configs as C

pytestmark = pytest.mark.gpu

FULL = ["llama8b_q_proj", "llama8b_down_proj", "llama70b_gate_proj", "moe64_kquant3"]


def _rows_view(t, K, nr, C_):
    return t.view(K, nr, C_) if K else t.view(nr, C_)


def _sample_rows(w, k=6):
    nr = w.experts * w.rows
    rng = np.random.default_rng(17)
    rows = {0, nr - 1, w.rows - 1, (nr // 2) | 1}
    rows |= set(rng.integers(0, nr, k).tolist())
    return np.array(sorted(rows), dtype=np.int64)


def _gather_state(case, rows):
    g = gsq()
    w = case.w
    nr, K, Cc = w.experts * w.rows, w.K, w.cols
    idx = torch.from_numpy(rows).cuda()
    f = lambda which: case.layer.get_tensor(which, torch.float32)
    L = f(g.GSQ_T_LOGITS).view(K, nr, Cc)[:, idx].cpu().numpy()
    M = f(g.GSQ_T_MOM_LOGITS).view(K, nr, Cc)[:, idx].cpu().numpy()
    S = f(g.GSQ_T_SCALES).view(nr, Cc // w.group)[idx].cpu().numpy()
    MS = f(g.GSQ_T_MOM_SCALES).view(nr, Cc // w.group)[idx].cpu().numpy()
    return O.RowState(row_ids=rows, W=case.W.view(nr, Cc)[idx].float().cpu().double().numpy(),
                      logits=L, scales=S, m_logits=M, m_scales=MS)


@pytest.mark.parametrize("name", FULL)
def test_full_size_step_sampled_rows(name):
    g = gsq()
    w = C.WORKLOADS[name]
    case = Case(w, gemm="bf16", keep_calib_host=False)
    rows = _sample_rows(w)
    experts = sorted(set((rows // w.rows).tolist()))
    H = np.zeros((w.experts, 1, 1))
    Hs = {e: case.calib[e].double().cpu().numpy() for e in experts}
    del case.calib
    torch.cuda.empty_cache()

    class _H:  # expert -> H lookup for the oracle, only the sampled experts on the host
        def __getitem__(self, e):
            return Hs[int(e)]
    case.prob.H = _H()
    nr, K, Cc = w.experts * w.rows, w.K, w.cols
    tau0, tau1 = w.tau(0), w.tau(1)

    # (a) gradient export at t = 0 (no update): G, D, loss property, sampled rows
    st0 = _gather_state(case, rows)
    loss = torch.zeros(1, device="cuda")
    gl = torch.empty(K * w.n, device="cuda")
    gs = torch.zeros(w.n // w.group, device="cuda")
    case.layer.step(0, tau0, w.kappa, loss=loss, grad_logits=gl, grad_scales=gs)
    torch.cuda.synchronize()
    Gd = case.layer.get_tensor(g.GSQ_T_G, torch.float32).view(nr, Cc)
    Dd = case.layer.get_tensor(g.GSQ_T_D, torch.bfloat16).view(nr, Cc)
    half_DG = 0.5 * torch.sum(Dd.double() * Gd.double()).item()
    assert abs(loss.item() - half_DG) <= 1e-5 * abs(half_DG), (loss.item(), half_DG)
    idx = torch.from_numpy(rows).cuda()
    Gs, Ds = Gd[idx].double().cpu().numpy(), Dd[idx].double().cpu().numpy()
    glr = gl.view(K, nr, Cc)[:, idx].cpu().numpy()
    gsr = gs.view(nr, Cc // w.group)[idx].cpu().numpy()
    del Gd, Dd, gl, gs
    torch.cuda.empty_cache()
    ref = O.step(case.prob, st0.copy(), 0, tau0, w.kappa, update=False)
    assert_close(Ds, ref.fw.D, TOL_BF16, "D rows")
    assert_close(Gs, ref.G, TOL_BF16, "G rows vs oracle")
    # the GEMM against exact products of its own bf16 operands on these rows
    Hb = case.layer.get_tensor(g.GSQ_T_H, torch.bfloat16).view(w.experts, Cc, Cc)
    for e in experts:
        sel = rows // w.rows == e
        assert_gemm_bound(Gs[sel], Ds[sel], Hb[e].double().cpu().numpy(),
                          f"tcgen05 GEMM rows, expert {e}")
    del Hb
    torch.cuda.empty_cache()
    assert_grad_close(glr, gsr if ref.d_scales is not None else None, ref, case.prob, tau0,
                      w.kappa, TOL_BF16, "rows")

    # (b) the benchmark's step: update with look-ahead, state-synced on the rows
    case.layer.step(0, tau0, w.kappa, next_tau=tau1, next_kappa=w.kappa, loss=loss)
    torch.cuda.synchronize()
    st1 = _gather_state(case, rows)
    orc = st0.copy()
    res = O.step(case.prob, orc, 0, tau0, w.kappa, update=True)
    d = np.abs(st1.logits.astype(np.float64) - orc.logits)
    flip = d > 0.5 * w.lr_logits
    assert flip.mean() < 1e-3 and d[~flip].max() < 1e-5 and d.max() <= 2.001 * w.lr_logits
    c = np.abs((1 - w.beta1) * res.d_logits)
    assert np.all(c[flip] <= 2 * TOL_BF16 * np.sqrt(np.mean(c * c)))
    if res.d_scales is None:
        assert np.array_equal(st1.scales, st0.scales)
    # look-ahead D of step 1 from the updated state (oracle uses the GPU's updated rows)
    D1 = case.layer.get_tensor(g.GSQ_T_D, torch.bfloat16).view(nr, Cc)[idx].double().cpu().numpy()
    fw1 = O.forward(case.prob, st1, 1, tau1, w.kappa)
    assert_close(D1, fw1.D, 2 ** -8, "look-ahead D rows (bf16 storage)")
    case.layer.sync_status()
    case.layer.close()
