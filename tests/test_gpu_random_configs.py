"""Seeded random layer problems against the oracle: shapes (E, R, C including odd
rows and tiny layers), grids (2 to 8 levels at random spacing, a symmetric
ternary grid for mask x sign), group sizes 4 to 128 or K-Quant scales, every
parameterisation, fp32 or bf16 weights, calibration as H or as tokens, fp32 or
tensor-core GEMM, temperatures 0.05 to 3, kappa 0 to 3, noise on or off.  Per
case: the initial state bit-exact, the step's loss and gradients (gradient
export) on random logits (on the bf16 path also its GEMM operands and product),
one Lion update, and projection and packing bit-exact."""
import dataclasses
import math

import numpy as np
import pytest
import torch

from gpu_common import (TOL_BF16, TOL_F32, Case, assert_close, assert_gemm_bound, assert_grad_close,
                        bf16_criterion, bf16_operand_bounds, check_lion, gsq,
                        mask_sign_grad_bounds)
from oracle import gsq_oracle as O
from paper_2604_18556_gb300 import configs as C

pytestmark = pytest.mark.gpu

U32 = 2.0 ** -24


def _config(i):
    rng = np.random.default_rng(1000 + i)
    param = rng.choice(["full", "full", "full", "shift5", "mask_sign"])
    if param == "mask_sign":
        a = float(rng.uniform(0.5, 2.0))
        grid = (-a, 0.0, a)
    else:
        K = int(rng.integers(2, 9)) if param == "full" else int(rng.integers(3, 9))
        gaps = rng.uniform(0.2, 1.5, K - 1)
        g = np.concatenate([[0.0], np.cumsum(gaps)])
        grid = tuple(float(v) for v in (g - rng.uniform(0.2, 0.8) * g[-1]))
    kquant = rng.random() < 0.2
    if kquant:
        group, cols = 16, 256 * int(rng.integers(1, 3))
    else:
        group = int(rng.choice([4, 8, 16, 32, 64, 128]))
        step = group * 8 // math.gcd(group, 8)
        cols = step * int(rng.integers(1, max(2, 1024 // step + 1)))
    w = C.Workload(
        name=f"random_{i}", experts=int(rng.choice([1, 1, 2, 3])), rows=int(rng.integers(1, 300)),
        cols=cols, grid=grid, group=group, w_dtype=str(rng.choice(["f32", "bf16"])),
        calib=str(rng.choice(["H", "X"])), tokens=int(rng.integers(16, 300)),
        token_dist=str(rng.choice(["normal", "student_t3"])), outliers=int(rng.integers(0, 3)),
        outlier_scale=10.0, steps=10, tau0=1.0, tau1=1.0,
        scale_mode="kquant2" if kquant else "group", init_bias=float(rng.uniform(0.5, 3.0)),
        lr_scales=0.0 if kquant else 5e-5, data_seed=7000 + i, param=param)
    gemm = str(rng.choice(["f32", "bf16"]))
    tau = float(np.exp(rng.uniform(np.log(0.05), np.log(3.0))))
    kappa = float(rng.uniform(0.0, 3.0))
    noise = bool(rng.random() < 0.85)
    seed = int(rng.integers(0, 2 ** 40))
    return w, gemm, float(np.float32(tau)), float(np.float32(kappa)), noise, seed, rng


@pytest.mark.parametrize("i", range(32))
def test_random_config(i):
    g = gsq()
    w, gemm, tau, kappa, noise, seed, rng = _config(i)
    case = Case(w, gemm=gemm, noise=noise, seed=seed)
    nr, L, n = w.experts * w.rows, w.L, w.n
    # (1) initial state
    st, ref = case.state(), case.oracle_init()
    for f in ("logits", "scales", "m_logits", "m_scales"):
        assert np.array_equal(getattr(st, f), getattr(ref, f)), f
    if w.param == "shift5":
        assert np.array_equal(st.j0, ref.j0)
    if w.scale_mode == "kquant2":
        assert np.array_equal(st.kq_d, ref.kq_d) and np.array_equal(st.kq_sc, ref.kq_sc)
    # (2) loss and gradients on random logits
    Lg = (1.5 * rng.standard_normal((L, nr, w.cols))).astype(np.float32)
    case.layer.set_tensor(g.GSQ_T_LOGITS, torch.from_numpy(Lg).cuda())
    st = case.state()
    t = int(rng.integers(0, 1000))
    loss = torch.zeros(1, device="cuda")
    gl = torch.empty(L * n, device="cuda")
    gs = torch.zeros(n // w.group, device="cuda")
    case.layer.step(t, tau, kappa, loss=loss, grad_logits=gl, grad_scales=gs)
    torch.cuda.synchronize()
    res = O.step(case.prob, st.copy(), t, tau, kappa, update=False)
    got_l = gl.cpu().numpy().astype(np.float64).reshape(res.d_logits.shape)
    got_s = gs.cpu().numpy().astype(np.float64)
    # fp32 conditioning of z = (kappa l + g)/tau and of w~ (see test_gpu_edges)
    zmax = float(np.max(np.abs(kappa * st.logits.astype(np.float64) + res.fw.g))) / tau
    zmax *= 2 if w.param == "mask_sign" else 1
    if gemm == "f32":
        tol = max(TOL_F32, 8 * U32 * zmax)
        assert_close(loss.cpu().numpy(), [res.loss], tol, "loss")
        assert_close(got_l, res.d_logits, tol, "dL/dlogits")
        if res.d_scales is not None:
            qmax = float(np.max(np.abs(w.grid)))
            cond = 8 * U32 * qmax * np.abs(res.G).reshape(-1, w.group).sum(1)
            ds = res.d_scales.reshape(-1)
            err = np.abs(got_s - ds)
            assert np.all(err <= tol * (np.abs(ds) + np.sqrt(np.mean(ds * ds))) + cond), "dL/ds"
    else:
        assert_close(loss.cpu().numpy(), [res.loss], TOL_BF16, "loss")
        # the tensor-core operands within one bf16 rounding of the oracle's, their product
        # within fp32 accumulation of the exact one; the gradients then within the larger
        # of G's relative tolerance and the operands' worst-case error carried through
        dD, dH, gb = bf16_operand_bounds(res, case.prob, zmax)
        Dg, Hg, Gg = case.D(), case.H_operand(), case.G()
        assert np.all(np.abs(Dg - res.fw.D) <= dD), "D operand"
        Hr = case.prob.H if case.prob.H is not None else np.einsum("etc,etd->ecd", case.prob.X,
                                                                   case.prob.X)
        assert np.all(np.abs(Hg - Hr) <= dH), "H operand"
        for e in range(w.experts):
            rows = slice(e * w.rows, (e + 1) * w.rows)
            assert_gemm_bound(Gg[rows], Dg[rows], Hg[e], f"G expert {e}")
        assert np.all(np.abs(Gg - res.G) <= gb), "G"
        bf16_criterion(Gg, res.G, gb, f"case {i} ({w.name}, {w.experts}x{w.rows}x{w.cols}, "
                                      f"calib {w.calib})")
        if w.param == "mask_sign":
            bl, bs = mask_sign_grad_bounds(res, case.prob, tau, kappa, TOL_BF16, gb)
            assert np.all(np.abs(got_l - res.d_logits) <= bl * 1.0001 + 1e-30), "dL/dlogits"
            if res.d_scales is not None:
                assert np.all(np.abs(got_s - res.d_scales.reshape(-1)) <= bs.reshape(-1) * 1.0001
                              + 1e-30), "dL/ds"
        else:
            q = O.level_values(case.prob, st) if w.param == "shift5" else None
            assert_grad_close(got_l, got_s if res.d_scales is not None else None, res, case.prob,
                              tau, kappa, TOL_BF16, w.name, q=q, g_bound=gb)
    # (3) one Lion update from the same state
    case.layer.step(t, tau, kappa)
    torch.cuda.synchronize()
    after = case.state()
    orc = st.copy()
    res = O.step(case.prob, orc, t, tau, kappa, update=True)
    c_l = w.beta1 * st.m_logits.astype(np.float64) + (1 - w.beta1) * res.d_logits
    check_lion(after.logits, orc.logits, st.logits, c_l, w.lr_logits,
               2 * (TOL_F32 if gemm == "f32" else TOL_BF16), "logits")
    # (4) projection and packing
    codes = torch.empty(n, dtype=torch.uint8, device="cuda")
    margin = torch.empty(n, device="cuda")
    case.layer.project(codes, margin)
    oc, om = O.project(after.logits, j0=after.j0, levels=w.K, mask_sign=w.param == "mask_sign")
    assert np.array_equal(codes.cpu().numpy(), oc.reshape(-1))
    assert np.array_equal(margin.cpu().numpy(), om.reshape(-1))
    buf = torch.empty(case.layer.packed_size(), dtype=torch.uint8, device="cuda")
    case.layer.pack(buf)
    if w.scale_mode == "kquant2":
        want = O.pack_kquant2(oc.reshape(-1), after.kq_d.reshape(-1), after.kq_sc.reshape(-1))
    else:
        want = O.pack_group(oc.reshape(-1), after.scales.reshape(-1), w.K)
    assert buf.cpu().numpy().tobytes() == want
    case.layer.sync_status()
    case.layer.close()
