"""GPU parity: the CUDA path through the C ABI against the CPU oracle, element by
element, on the same seeded inputs.  Shapes are small versions of the five
workloads, chosen to span several GEMM tiles with ragged tails (rows not a
multiple of 128, columns not a multiple of 256) and every group size / level
count / scale mode."""
import numpy as np
import pytest
import torch

from gpu_common import (TOL_BF16, TOL_F32, Case, assert_close, assert_gemm_bound,
                        assert_grad_close, check_lion, check_momentum, grad_bounds, gsq)
from oracle import gsq_oracle as O
from paper_2604_18556_gb300 import configs as C

pytestmark = pytest.mark.gpu

W = C.WORKLOADS
SMALL = {
    "ternary": W["ternary_256x512"],
    "q_proj": C.shrunk(W["llama8b_q_proj"], rows=96, cols=384, tokens=2048),
    "down_proj": C.shrunk(W["llama8b_down_proj"], rows=160, cols=640, tokens=4096),
    "gate_proj": C.shrunk(W["llama70b_gate_proj"], rows=130, cols=320, tokens=2048),
    "moe_kquant": C.shrunk(W["moe64_kquant3"], experts=3, rows=64, cols=512, tokens=1024),
}
TAU = {"ternary": 1.0, "q_proj": 0.55, "down_proj": 0.5, "gate_proj": 1.0, "moe_kquant": 1.0}


def _n(w):
    return w.experts * w.rows * w.cols


@pytest.mark.parametrize("name", list(SMALL))
def test_init_bit_exact(name):
    case = Case(SMALL[name], gemm="f32")
    st, ref = case.state(), case.oracle_init()
    assert np.array_equal(st.logits, ref.logits)
    assert np.array_equal(st.scales, ref.scales)
    assert not st.m_logits.any() and not st.m_scales.any()
    if SMALL[name].scale_mode == "kquant2":
        assert np.array_equal(st.kq_d, ref.kq_d) and np.array_equal(st.kq_sc, ref.kq_sc)


@pytest.mark.parametrize("noise", [True, False])
@pytest.mark.parametrize("name", list(SMALL))
def test_forward_soft_weight(name, noise):
    w = SMALL[name]
    case = Case(w, gemm="f32", noise=noise)
    what = torch.empty(_n(w), device="cuda")
    case.layer.forward(7, 0.7, 1.3, what=what)
    ref = O.forward(case.prob, case.oracle_init(), 7, 0.7, 1.3)
    assert_close(what.cpu().numpy(), ref.What, TOL_F32, "W^")
    assert_close(case.D(), ref.D, TOL_F32, "D")


@pytest.mark.parametrize("gemm", ["f32", "bf16"])
@pytest.mark.parametrize("name", list(SMALL))
def test_step_loss_and_gradients(name, gemm):
    w = SMALL[name]
    case = Case(w, gemm=gemm)
    tol = TOL_F32 if gemm == "f32" else TOL_BF16
    g = gsq()
    n, K = _n(w), w.K
    loss = torch.zeros(1, device="cuda")
    gl = torch.empty(K * n, device="cuda")
    gs = torch.zeros(n // w.group, device="cuda")
    case.layer.step(3, TAU[name], 1.0, loss=loss, grad_logits=gl, grad_scales=gs)
    torch.cuda.synchronize()
    ref = O.step(case.prob, case.oracle_init(), 3, TAU[name], 1.0, update=False)
    assert_close(loss.cpu().numpy(), [ref.loss], tol, "loss")
    assert_close(case.G(), ref.G, tol, "G")
    if gemm == "f32":
        assert_close(gl.cpu().numpy(), ref.d_logits, tol, "dL/dlogits")
        if ref.d_scales is not None:
            assert_close(gs.cpu().numpy(), ref.d_scales, tol, "dL/dscales")
    else:
        # gradients are linear in G: G's bf16 tolerance carried through (see grad_bounds)
        assert_grad_close(gl.cpu().numpy(), gs.cpu().numpy() if ref.d_scales is not None else None,
                          ref, case.prob, TAU[name], 1.0, tol, name)
    if gemm == "bf16":
        # the tensor-core GEMM against exact products of its own bf16 operands
        D, H, G = case.D(), case.H_operand(), case.G()
        rows = np.arange(w.experts * w.rows)
        for e in range(w.experts):
            sel = rows // w.rows == e
            assert_gemm_bound(G[sel], D[sel], H[e], f"tcgen05 GEMM vs its operands, expert {e}")
        assert_close(loss.cpu().numpy(), [0.5 * np.sum(D * case.G())], 1e-5, "loss = 1/2 sum D*G")


@pytest.mark.parametrize("gemm", ["f32", "bf16"])
@pytest.mark.parametrize("name", list(SMALL))
def test_step_update(name, gemm):
    w = SMALL[name]
    case = Case(w, gemm=gemm)
    tol = TOL_F32 if gemm == "f32" else TOL_BF16
    # two steps, so the second update sees a nonzero momentum
    st = case.oracle_init()
    losses = []
    for t in range(2):
        loss = torch.zeros(1, device="cuda")
        st_gpu_before = case.state()
        case.layer.step(t, TAU[name], 1.0, loss=loss)
        torch.cuda.synchronize()
        # state-synced: the oracle takes the GPU's pre-step state
        st_sync = st_gpu_before.copy()
        res = O.step(case.prob, st_sync, t, TAU[name], 1.0, update=True)
        gpu = case.state()
        assert_close(loss.cpu().numpy(), [res.loss], tol, f"loss t={t}")
        m0 = st_gpu_before.m_logits.astype(np.float64)
        c_l = w.beta1 * m0 + (1 - w.beta1) * res.d_logits
        check_lion(gpu.logits, st_sync.logits, st_gpu_before.logits, c_l, w.lr_logits, 2 * tol,
                    "logits")
        if gemm == "f32":
            gb_l = tol * (np.abs(res.d_logits) + np.sqrt(np.mean(res.d_logits ** 2)))
            gb_s = None if res.d_scales is None else \
                tol * (np.abs(res.d_scales) + np.sqrt(np.mean(res.d_scales ** 2)))
        else:
            f, gscale, bs = grad_bounds(res, case.prob, tol)
            gb_l = (1.0 / TAU[name]) * f * gscale[None] + tol * np.abs(res.d_logits)
            gb_s = None if res.d_scales is None else bs + tol * np.abs(res.d_scales)
        check_momentum(gpu.m_logits, st_sync.m_logits, gb_l, w.beta2, "logit momentum")
        if res.d_scales is not None:
            c_s = w.beta1 * st_gpu_before.m_scales.astype(np.float64) + (1 - w.beta1) * res.d_scales
            check_lion(gpu.scales, st_sync.scales, st_gpu_before.scales, c_s, w.lr_scales,
                        2 * tol, "scales")
            check_momentum(gpu.m_scales, st_sync.m_scales, gb_s, w.beta2, "scale momentum")
        else:
            assert np.array_equal(gpu.scales, st_gpu_before.scales)
        losses.append(float(loss.item()))
    assert all(np.isfinite(losses))


@pytest.mark.parametrize("name", ["q_proj", "down_proj", "moe_kquant"])
def test_lookahead_is_bit_identical(name):
    w = SMALL[name]
    a, b = Case(w, gemm="bf16"), Case(w, gemm="bf16")
    for t in range(4):
        la, lb = torch.zeros(1, device="cuda"), torch.zeros(1, device="cuda")
        tau, tau_next = w.tau(t), w.tau(t + 1)
        a.layer.step(t, tau, 1.0, next_tau=tau_next, next_kappa=1.0, loss=la)
        b.layer.step(t, tau, 1.0, loss=lb)
        torch.cuda.synchronize()
        assert la.item() == lb.item()
        sa, sb = a.state(), b.state()
        for f in ("logits", "m_logits", "scales", "m_scales"):
            assert np.array_equal(getattr(sa, f), getattr(sb, f)), (t, f)


def test_resume_is_bit_identical():
    g = gsq()
    w = SMALL["q_proj"]
    full = Case(w, gemm="bf16")
    part = Case(w, gemm="bf16")
    losses_full = []
    for t in range(6):
        loss = torch.zeros(1, device="cuda")
        full.layer.step(t, w.tau(t), 1.0, next_tau=w.tau(t + 1), loss=loss)
        losses_full.append(loss.item())
    for t in range(3):
        part.layer.step(t, w.tau(t), 1.0, next_tau=w.tau(t + 1))
    saved = {k: part.layer.get_tensor(k).clone()
             for k in (g.GSQ_T_LOGITS, g.GSQ_T_SCALES, g.GSQ_T_MOM_LOGITS, g.GSQ_T_MOM_SCALES)}
    part.layer.close()
    resumed = Case(w, gemm="bf16")
    for k, v in saved.items():
        resumed.layer.set_tensor(k, v)
    for t in range(3, 6):
        loss = torch.zeros(1, device="cuda")
        resumed.layer.step(t, w.tau(t), 1.0, next_tau=w.tau(t + 1), loss=loss)
        assert loss.item() == losses_full[t]
    sf, sr = full.state(), resumed.state()
    for f in ("logits", "m_logits", "scales", "m_scales"):
        assert np.array_equal(getattr(sf, f), getattr(sr, f)), f


@pytest.mark.parametrize("name", list(SMALL))
def test_project_and_pack_bit_exact(name):
    g = gsq()
    w = SMALL[name]
    case = Case(w, gemm="bf16")
    for t in range(3):
        case.layer.step(t, 0.3, 1.0, next_tau=0.3)
    # make the logits less trivial than init: random perturbation through set_tensor
    rng = np.random.default_rng(3)
    L = case.logits() + rng.standard_normal(case.logits().shape).astype(np.float32)
    L[:, :, ::7] = L[:, :, ::7].max(0, keepdims=True)  # exact ties in every 7th column
    case.layer.set_tensor(g.GSQ_T_LOGITS, torch.from_numpy(L.copy()).cuda())
    n = _n(w)
    codes = torch.empty(n, dtype=torch.uint8, device="cuda")
    margin = torch.empty(n, device="cuda")
    case.layer.project(codes, margin)
    st = case.state()
    oc, om = O.project(st.logits)
    assert np.array_equal(codes.cpu().numpy(), oc.reshape(-1))
    assert np.array_equal(margin.cpu().numpy(), om.reshape(-1))
    buf = torch.full((case.layer.packed_size(),), 0xAB, dtype=torch.uint8, device="cuda")
    wrote = case.layer.pack(buf)
    assert wrote == buf.numel()
    got = buf.cpu().numpy().tobytes()
    if w.scale_mode == "kquant2":
        ref = O.pack_kquant2(oc.reshape(-1), st.kq_d.reshape(-1), st.kq_sc.reshape(-1))
    else:
        ref = O.pack_group(oc.reshape(-1), st.scales.reshape(-1), w.K)
    assert got == ref


def test_trajectory_ternary_full_run():
    """The ternary workload (256 x 512, calibration tokens kept, fp32 path) for all
    50 steps: per-step losses within 1e-4; final codes bit-exact where the
    margin is at least 1e-5; final state within the Lion flip allowance."""
    w = SMALL["ternary"]
    case = Case(w, gemm="f32")
    st = case.oracle_init()
    flips = 0
    for t in range(w.steps):
        loss = torch.zeros(1, device="cuda")
        case.layer.step(t, w.tau(t), w.kappa, next_tau=w.tau(t + 1), next_kappa=w.kappa, loss=loss)
        res = O.step(case.prob, st, t, w.tau(t), w.kappa)
        assert_close(loss.cpu().numpy(), [res.loss], TOL_F32, f"loss t={t}")
    gpu = case.state()
    diff = np.abs(gpu.logits.astype(np.float64) - st.logits)
    # a Lion sign flip moves a logit by 2 lr; fp32 rounding drift over 50 steps
    # stays orders of magnitude below lr / 2
    flips = int((diff > 0.5 * w.lr_logits).sum())
    assert flips <= 1e-4 * diff.size, flips
    drift = diff[diff <= 0.5 * w.lr_logits]
    assert drift.max() <= 1e-5, drift.max()
    assert diff.max() <= 2 * w.lr_logits * w.steps
    oc, om = O.project(st.logits)
    gc, _ = O.project(gpu.logits)
    keep = om >= 1e-5
    assert np.array_equal(gc[keep], oc[keep])
    assert_close(gpu.scales, st.scales, TOL_F32, "scales after 50 steps")


@pytest.mark.parametrize("tile_n", ["128", "224", "256"])
@pytest.mark.parametrize("name", ["q_proj", "gate_proj", "moe_kquant"])
def test_tc_gemm_tile_widths(name, tile_n, monkeypatch):
    """The single-CTA contraction: every tensor-core tile width (chosen per layer by wave balance) on ragged
    shapes, against exact products of the kernel's own bf16 operands."""
    monkeypatch.setenv("GSQ_GEMM_TILE_N", tile_n)
    monkeypatch.setenv("GSQ_GEMM_PAIR", "0")  # single CTAs (pairs: test_tc_gemm_cta_pairs)
    w = SMALL[name]
    case = Case(w, gemm="bf16")
    loss = torch.zeros(1, device="cuda")
    case.layer.step(0, TAU[name], 1.0, loss=loss)
    torch.cuda.synchronize()
    D, H, G = case.D(), case.H_operand(), case.G()
    rows = np.arange(w.experts * w.rows)
    for e in range(w.experts):
        sel = rows // w.rows == e
        assert_gemm_bound(G[sel], D[sel], H[e], f"tile N = {tile_n}, expert {e}")
    assert abs(loss.item() - 0.5 * np.sum(D.astype(np.float64) * G)) <= 1e-5 * abs(loss.item())


PAIR_CASES = dict(SMALL, **{
    # 2,000 rows: eight 256-row pair tiles, the last ragged; 2,688 columns: 12 tiles 224
    # wide, 11 (the last ragged) 256 wide, 21 of 128; 42 k-blocks; more tiles (88 to
    # 168) than CTA pairs on the GPU, so every pair runs several
    "q_proj_multi_wave": C.shrunk(W["llama8b_q_proj"], rows=2000, cols=2688, tokens=4096),
})


@pytest.mark.parametrize("tile_n", ["128", "224", "256"])
@pytest.mark.parametrize("name", ["q_proj", "gate_proj", "moe_kquant", "q_proj_multi_wave"])
def test_tc_gemm_cta_pairs(name, tile_n, monkeypatch):
    """The CTA-pair contraction (tcgen05.mma.cta_group::2, 256-row tiles over two SMs)
    at every tile width on ragged shapes and several experts, against exact products of
    the kernel's own bf16 operands, and the loss as 1/2 sum D G."""
    monkeypatch.setenv("GSQ_GEMM_TILE_N", tile_n)
    monkeypatch.setenv("GSQ_GEMM_PAIR", "1")
    w = PAIR_CASES[name]
    case = Case(w, gemm="bf16")
    loss = torch.zeros(1, device="cuda")
    case.layer.step(0, TAU.get(name, 0.55), 1.0, loss=loss)
    torch.cuda.synchronize()
    case.layer.sync_status()
    D, H, G = case.D(), case.H_operand(), case.G()
    rows = np.arange(w.experts * w.rows)
    for e in range(w.experts):
        sel = rows // w.rows == e
        assert_gemm_bound(G[sel], D[sel], H[e], f"pairs, tile N = {tile_n}, expert {e}")
    assert abs(loss.item() - 0.5 * np.sum(D.astype(np.float64) * G)) <= 1e-5 * abs(loss.item())


CLUSTER_CASES = dict(PAIR_CASES, **{
    # 700 rows: three 256-row tiles, so the last cluster tile has one pair with rows
    "q_proj_odd_tiles": C.shrunk(W["llama8b_q_proj"], rows=700, cols=1024, tokens=2048),
})


@pytest.mark.parametrize("tile_n", ["128", "224", "256"])
@pytest.mark.parametrize("name", ["q_proj", "gate_proj", "moe_kquant", "q_proj_multi_wave",
                                  "q_proj_odd_tiles"])
def test_tc_gemm_pair_clusters(name, tile_n, monkeypatch):
    """Clusters of two CTA pairs sharing each tile of H by TMA multicast: every tile width,
    ragged shapes (an odd number of 256-row tiles leaves the second pair of the last
    cluster tile without rows), several experts, against exact products of the kernel's
    own bf16 operands, and the loss as 1/2 sum D G."""
    monkeypatch.setenv("GSQ_GEMM_TILE_N", tile_n)
    monkeypatch.setenv("GSQ_GEMM_PAIR", "2")
    w = CLUSTER_CASES[name]
    case = Case(w, gemm="bf16")
    assert case.layer.kernel_name(gsq().GSQ_K_GEMM) == "k_tc_gemm_quad"
    loss = torch.zeros(1, device="cuda")
    case.layer.step(0, TAU.get(name, 0.55), 1.0, loss=loss)
    torch.cuda.synchronize()
    case.layer.sync_status()
    D, H, G = case.D(), case.H_operand(), case.G()
    rows = np.arange(w.experts * w.rows)
    for e in range(w.experts):
        sel = rows // w.rows == e
        assert_gemm_bound(G[sel], D[sel], H[e], f"pair clusters, tile N = {tile_n}, expert {e}")
    assert abs(loss.item() - 0.5 * np.sum(D.astype(np.float64) * G)) <= 1e-5 * abs(loss.item())
