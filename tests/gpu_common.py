"""Helpers shared by the GPU parity tests: build a layer through the C ABI and the
matching oracle problem from the same seeded inputs, read GPU state back into
oracle form, and the tolerance checks the acceptance criteria name.

Tolerances (from the acceptance criteria of the step):
  * hard assignments and packed bits: bit-exact (entries whose top-two logit
    margin is below 1e-5 excluded where the logits themselves came from two
    trajectories);
  * fp32 path (GEMM on fp32 operands): loss, gradients and W^ within 1e-4 relative;
  * bf16 tensor-core GEMM path: GEMM-backed quantities within 2e-2 relative.
"Relative" is applied elementwise as |a - b| <= tol * (|b| + rms(b)) -- the rms
term keeps entries that are tiny by cancellation from failing on absolute
noise -- and, for the whole tensor, ||a - b|| <= tol * ||b||.
"""
from __future__ import annotations

import numpy as np
import torch

from oracle import gsq_oracle as O
from paper_2604_18556_gb300 import configs as C
from paper_2604_18556_gb300 import inputs

TOL_F32 = 1e-4
TOL_BF16 = 2e-2


def gsq():
    from paper_2604_18556_gb300 import build
    build.build()
    from paper_2604_18556_gb300 import gsq as g
    return g


def assert_close(a, b, tol, what=""):
    a = np.asarray(a, dtype=np.float64).reshape(-1)
    b = np.asarray(b, dtype=np.float64).reshape(-1)
    assert a.shape == b.shape, (what, a.shape, b.shape)
    if b.size == 0:
        return
    rms = float(np.sqrt(np.mean(b * b)))
    err = np.abs(a - b)
    bad = err > tol * (np.abs(b) + rms)
    if bad.any():
        i = int(np.argmax(err / (np.abs(b) + rms + 1e-300)))
        raise AssertionError(f"{what}: {int(bad.sum())}/{b.size} elements beyond {tol}; worst at {i}: "
                             f"got {a[i]!r} want {b[i]!r} (rms {rms:.3e})")
    nrm = float(np.linalg.norm(b))
    assert float(np.linalg.norm(a - b)) <= tol * nrm + 1e-300, (what, float(np.linalg.norm(a - b)) / nrm)


def assert_gemm_bound(G, D, H, what="", alpha=2.0):
    """fp32-accumulated G = alpha D H against exact products of the same operands:
    every entry within the summation error bound |g^ - g| <= gamma_n sum_k |d_k h_k|
    with gamma_n ~ n u, u = 2^-24 (Higham, Accuracy and Stability of Numerical
    Algorithms, Thm 3.5; holds for any summation order).  Returns the largest
    error as a fraction of its bound."""
    D = np.asarray(D, np.float64)
    H = np.asarray(H, np.float64)
    exact = alpha * D @ H
    absum = abs(alpha) * np.abs(D) @ np.abs(H)
    n = D.shape[-1]
    bound = 1.01 * n * 2.0 ** -24 * absum + 1e-30
    err = np.abs(np.asarray(G, np.float64) - exact)
    worst = float((err / bound).max())
    assert worst <= 1.0, (what, worst)
    return worst


U_BF16 = 2.0 ** -8


def bf16_operand_bounds(ref, prob, zmax):
    """Elementwise worst-case bounds for the tensor-core path's operands and product,
    G = 2 D H with D and H each rounded once to bf16 (unit roundoff u = 2^-8):
      W^ in fp32 from p = softmax(z), |z| <= zmax: the rounding of z (relative 2^-24 each
        for kappa l + g and /tau) moves p_k by <= 6 * 2^-24 zmax p_k, the exp, the sum
        and the level mix by <= (K + 4) 2^-24, so |dW^| <= 2^-24 |s| qmax (6 zmax + K + 4);
      D = fl(W^ - W) then bf16:  |dD| <= u |D| + (1 + u)(|dW^| + 2^-24 |D|);
      H given in fp32 (H mode) or formed in fp32 from T tokens (X mode; |X^T X| <= |X|^T |X|),
        then bf16:  |dH| <= (u + (T + 2) 2^-24) |H|;
      fp32 accumulation over C terms, doubled for the tensor core's order: 2 C 2^-24 |D| |H|;
    so |dG| <= 2 [|dD| |H| + |D| |dH| + 2 C 2^-24 |D| |H|] to first order (Higham, Accuracy
    and Stability of Numerical Algorithms, Thm 3.5 with perturbed operands).  Returns
    (dD, dH per expert, dG).  Where G cancels (rank-deficient or outlier-dominated H) dG
    exceeds a relative tolerance on G."""
    u = U_BF16
    e24 = 2.0 ** -24
    D = np.abs(ref.fw.D)
    nr, Cc = D.shape
    R = nr // prob.E
    qmax = float(np.max(np.abs(prob.grid)))
    K = len(prob.grid)
    s = np.abs(ref.fw.s)
    dW = e24 * s * qmax * (6.0 * zmax + K + 4)
    dD = u * D + (1 + u) * (dW + e24 * D)
    dG = np.empty_like(D)
    dH = []
    for e in range(prob.E):
        if prob.H is not None:
            Ha, T = np.abs(prob.H[e]), 0
        else:
            Xa = np.abs(prob.X[e])
            Ha, T = Xa.T @ Xa, Xa.shape[0]
        dH.append((u + (T + 2) * e24) * Ha)
        rows = slice(e * R, (e + 1) * R)
        dG[rows] = dD[rows] @ Ha + D[rows] @ dH[-1] + 2 * Cc * e24 * (D[rows] @ Ha)
    return dD, np.stack(dH), 2.0 * (1 + 4 * u) * dG


def bf16_criterion(G, ref_G, g_bound, what, tol=TOL_BF16):
    """The 2e-2 relative criterion on the bf16 path's G, made visible.  Prints the
    worst elementwise error in units of tol (|b| + rms b), the fraction of entries
    beyond it and the tensor-norm relative error; asserts that every entry beyond
    the criterion is one where the operands' own worst-case error (g_bound: D and
    H each one bf16 rounding from the oracle's, bf16_operand_bounds) already
    exceeds it -- cancellation in G, not an error of the kernel.  Returns the
    worst ratio."""
    a = np.asarray(G, np.float64).reshape(-1)
    b = np.asarray(ref_G, np.float64).reshape(-1)
    gb = np.asarray(g_bound, np.float64).reshape(-1)
    scale = tol * (np.abs(b) + np.sqrt(np.mean(b * b)))
    ratio = np.abs(a - b) / scale
    beyond = ratio > 1.0
    norm_rel = float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))
    worst = float(ratio.max()) if ratio.size else 0.0
    print(f"bf16 criterion {what}: worst |dG| = {worst:.3f} x 2e-2 (|G| + rms G), "
          f"{int(beyond.sum())}/{beyond.size} entries beyond, ||dG||/||G|| = {norm_rel:.2e}")
    explained = gb[beyond] > scale[beyond]
    assert explained.all(), (what, int((~explained).sum()), worst)
    return worst


def grad_bounds(ref, prob, tol, q=None, g_bound=None):
    """Elementwise bounds for the logit and scale gradients when the only
    reduced-precision input is G (the bf16 tensor-core GEMM): both gradients
    are linear in G,
        dL/dl_k = f_k G,  f_k = (kappa/tau) s p_k (q_k - w~),   dL/ds_g = sum_g w~ G,
    so G's tolerance tol (|G| + rms G), or the larger elementwise bound g_bound
    (bf16_operand_bounds), carries through |f_k| and |w~|."""
    G = ref.G
    gscale = tol * (np.abs(G) + np.sqrt(np.mean(G * G)))
    if g_bound is not None:
        gscale = np.maximum(gscale, g_bound)
    fw = ref.fw
    if q is None:
        q = np.asarray(prob.grid, np.float64)[:, None, None]
    f = np.abs(fw.s[None] * fw.p * O.centred_values(fw.p, q))   # |f_k| / (kappa/tau)
    bl = None
    nr, C = G.shape
    bs = (np.abs(fw.wtil) * gscale).reshape(nr, C // prob.group, prob.group).sum(2)
    return f, gscale, bs


def assert_grad_close(got_l, got_s, ref, prob, tau, kappa, tol, what="", q=None, g_bound=None):
    f, gscale, bs = grad_bounds(ref, prob, tol, q, g_bound)
    bl = (kappa / tau) * f * gscale[None] + tol * np.abs(ref.d_logits)
    err = np.abs(np.asarray(got_l, np.float64).reshape(ref.d_logits.shape) - ref.d_logits)
    bad = err > bl * 1.0001 + 1e-30
    assert not bad.any(), (what + " dL/dlogits", int(bad.sum()), float((err / (bl + 1e-30)).max()))
    if got_s is not None and ref.d_scales is not None:
        bsc = bs + tol * np.abs(ref.d_scales)
        err = np.abs(np.asarray(got_s, np.float64).reshape(ref.d_scales.shape) - ref.d_scales)
        bad = err > bsc * 1.0001 + 1e-30
        assert not bad.any(), (what + " dL/dscales", int(bad.sum()))


def mask_sign_grad_factors(ref, prob, tau, kappa):
    """|dL/dl| / |G| for both planes: (kappa/tau) s a |b~ dm~| and (kappa/tau) s a |m~ db~|."""
    fw = ref.fw
    a = float(prob.grid[2])
    gm = O.binary_gs_grad(fw.p[0], fw.soft[0], O.BINARY_VALUES[0], tau, kappa)
    gb = O.binary_gs_grad(fw.p[1], fw.soft[1], O.BINARY_VALUES[1], tau, kappa)
    return np.abs(np.stack([fw.s * a * fw.soft[1] * gm, fw.s * a * fw.soft[0] * gb]))


def mask_sign_grad_bounds(ref, prob, tau, kappa, tol, g_bound=None):
    """Gradients are linear in G; with G the only reduced-precision input (bf16
    GEMM) its tolerance (or the larger g_bound) carries through the factors above."""
    G = ref.G
    gscale = tol * (np.abs(G) + np.sqrt(np.mean(G * G)))
    if g_bound is not None:
        gscale = np.maximum(gscale, g_bound)
    bl = mask_sign_grad_factors(ref, prob, tau, kappa) * gscale[None] + tol * np.abs(ref.d_logits)
    nr, Cc = G.shape
    bs = (np.abs(ref.fw.wtil) * gscale).reshape(nr, Cc // prob.group, prob.group).sum(2)
    return bl, bs + (0 if ref.d_scales is None else tol * np.abs(ref.d_scales))


def check_lion(gpu, orc, theta_in, c_orc, lr, flip_frac, what):
    """Lion results agree to rounding except where the sign of the momentum mix
    c is decided by a difference below the path's tolerance; such flips move a
    parameter by at most 2 lr."""
    gpu = np.asarray(gpu, np.float64).reshape(-1)
    orc = np.asarray(orc, np.float64).reshape(-1)
    theta_in = np.asarray(theta_in, np.float64).reshape(-1)
    c = np.abs(np.asarray(c_orc, np.float64).reshape(-1))
    diff = np.abs(gpu - orc)
    # rounding is relative to the operands (theta, lr), not to a result that may
    # cancel to ~0 (theta = lr, sign(c) = +1)
    mag = np.maximum(np.maximum(np.abs(orc), np.abs(theta_in)), lr)
    same = diff <= 4 * np.spacing(mag.astype(np.float32)).astype(np.float64)
    flip = ~same
    assert np.all(diff[flip] <= 2.0 * lr * 1.001 + 1e-7), what
    thresh = flip_frac * np.sqrt(np.mean(c * c))
    assert np.all(c[flip] <= thresh), (what, int(flip.sum()), float(c[flip].max()), thresh)
    return int(flip.sum())


def check_momentum(gpu, orc, grad_bound, b2, what):
    """m' = b2 m + (1 - b2) g with the same m on both sides: the difference is
    (1 - b2) times the gradient difference, so the gradient's bound carries
    over, plus fp32 rounding of m'."""
    gpu = np.asarray(gpu, np.float64).reshape(-1)
    orc = np.asarray(orc, np.float64).reshape(-1)
    bound = (1 - b2) * np.asarray(grad_bound, np.float64).reshape(-1) + \
        2 * np.spacing(np.abs(orc).astype(np.float32)).astype(np.float64)
    bad = np.abs(gpu - orc) > bound
    assert not bad.any(), (what, int(bad.sum()))


def rel_err(a, b) -> float:
    a = np.asarray(a, dtype=np.float64).reshape(-1)
    b = np.asarray(b, dtype=np.float64).reshape(-1)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


class Case:
    """A layer problem on the GPU (through the C ABI) and the same problem for the oracle."""

    def __init__(self, w: C.Workload, gemm: str = "f32", noise: bool = True, seed=None,
                 keep_calib_host: bool = True, device="cuda", unstaged: bool = False,
                 index_offset: int = 0):
        g = gsq()
        self.w = w
        self.gemm = gemm
        self.W = inputs.make_weight(w, device=device)
        if w.calib == "X":
            self.calib = inputs.make_tokens(w, device=device)
        elif w.calib == "batches":
            self.calib = None                      # tokens arrive with every micro-batch
        else:
            self.calib = inputs.make_gram(w, device=device)
        hyper = dict(init_bias=w.init_bias, seed=w.seed if seed is None else seed,
                     lr_logits=w.lr_logits, lr_scales=w.lr_scales, beta1=w.beta1, beta2=w.beta2,
                     wd_logits=w.wd_logits, wd_scales=w.wd_scales, noise=noise,
                     unstaged=unstaged, index_offset=index_offset)
        self.layer = g.Layer(self.W, self.calib, w.grid, w.group, calib_kind=w.calib,
                             scale_mode=w.scale_mode, gemm=gemm, param=w.param,
                             tokens_per_batch=w.tokens if w.calib == "batches" else 0, **hyper)
        self.prob = O.Problem(E=w.experts, R=w.rows, C=w.cols, grid=np.asarray(w.grid, float),
                              group=w.group, seed=hyper["seed"], scale_mode=w.scale_mode,
                              lr_logits=w.lr_logits, lr_scales=w.lr_scales, beta1=w.beta1,
                              beta2=w.beta2, wd_logits=w.wd_logits, wd_scales=w.wd_scales,
                              noise=noise, shift=w.param == "shift5",
                              mask_sign=w.param == "mask_sign")
        if keep_calib_host and self.calib is not None:
            host = self.calib.double().cpu().numpy()
            if w.calib == "X":
                self.prob.X = host
            else:
                self.prob.H = host
        self.W_host = self.W.float().cpu().numpy().reshape(w.experts * w.rows, w.cols)

    # ---- GPU state -> numpy ------------------------------------------------------
    def tensor(self, which, dtype):
        return self.layer.get_tensor(which, dtype)

    def logits(self):
        g = gsq()
        E, R, Cc, L = self.w.experts, self.w.rows, self.w.cols, self.w.L
        return self.tensor(g.GSQ_T_LOGITS, torch.float32).view(L, E * R, Cc).cpu().numpy()

    def state(self, rows=None) -> O.RowState:
        g = gsq()
        w = self.w
        nr = w.experts * w.rows
        K = w.L
        f = lambda which: self.tensor(which, torch.float32).cpu().numpy()
        st = O.RowState(row_ids=np.arange(nr, dtype=np.int64), W=self.W_host.astype(np.float64),
                        logits=f(g.GSQ_T_LOGITS).reshape(K, nr, w.cols),
                        scales=f(g.GSQ_T_SCALES).reshape(nr, w.cols // w.group),
                        m_logits=f(g.GSQ_T_MOM_LOGITS).reshape(K, nr, w.cols),
                        m_scales=f(g.GSQ_T_MOM_SCALES).reshape(nr, w.cols // w.group))
        if w.scale_mode == "kquant2":
            d16 = self.tensor(g.GSQ_T_KQ_D, torch.int16).cpu().numpy().view(np.uint16)
            st.kq_d = O.f16_bits_to_f32(d16).reshape(nr, w.cols // 256)
            st.kq_sc = self.tensor(g.GSQ_T_KQ_SC, torch.int8).cpu().numpy().astype(np.int32).reshape(
                nr, w.cols // 16)
        if w.param == "shift5":
            st.j0 = self.tensor(g.GSQ_T_J0, torch.uint8).cpu().numpy().reshape(nr, w.cols)
        return st if rows is None else st.subset(rows)

    def G(self):
        g = gsq()
        return self.tensor(g.GSQ_T_G, torch.float32).view(-1, self.w.cols).cpu().numpy()

    def D(self):
        g = gsq()
        dt = torch.bfloat16 if self.gemm == "bf16" else torch.float32
        return self.tensor(g.GSQ_T_D, dt).float().view(-1, self.w.cols).cpu().numpy()

    def H_operand(self):
        g = gsq()
        dt = torch.bfloat16 if self.gemm == "bf16" else torch.float32
        C_ = self.w.cols
        return self.tensor(g.GSQ_T_H, dt).float().view(self.w.experts, C_, C_).cpu().numpy()

    def oracle_init(self, rows=None) -> O.RowState:
        nr = self.w.experts * self.w.rows
        ids = np.arange(nr) if rows is None else np.asarray(rows)
        return O.init_state(self.prob, self.W_host[ids], ids, init_bias=self.w.init_bias)


def gather_rows(case, rows) -> O.RowState:
    """The GPU state of the given global rows (row id = e*R + r) as an oracle
    RowState, gathered on the device so only those rows cross to the host."""
    g = gsq()
    w = case.w
    nr, L, Cc = w.experts * w.rows, w.L, w.cols
    rows = np.asarray(rows, dtype=np.int64)
    idx = torch.from_numpy(rows).cuda()
    f = lambda which: case.layer.get_tensor(which, torch.float32)
    st = O.RowState(
        row_ids=rows, W=case.W.view(nr, Cc)[idx].float().cpu().double().numpy(),
        logits=f(g.GSQ_T_LOGITS).view(L, nr, Cc)[:, idx].cpu().numpy(),
        scales=f(g.GSQ_T_SCALES).view(nr, Cc // w.group)[idx].cpu().numpy(),
        m_logits=f(g.GSQ_T_MOM_LOGITS).view(L, nr, Cc)[:, idx].cpu().numpy(),
        m_scales=f(g.GSQ_T_MOM_SCALES).view(nr, Cc // w.group)[idx].cpu().numpy())
    if w.param == "shift5":
        st.j0 = case.layer.get_tensor(g.GSQ_T_J0, torch.uint8).view(nr, Cc)[idx].cpu().numpy()
    if w.scale_mode == "kquant2":
        d16 = case.layer.get_tensor(g.GSQ_T_KQ_D, torch.int16).view(nr, Cc // 256)[idx]
        st.kq_d = O.f16_bits_to_f32(d16.cpu().numpy().view(np.uint16))
        sc = case.layer.get_tensor(g.GSQ_T_KQ_SC, torch.int8).view(nr, Cc // 16)[idx]
        st.kq_sc = sc.cpu().numpy().astype(np.int32)
    return st


class HostH:
    """Expert -> float64 H lookup for the oracle holding only the experts of the
    sampled rows (a full-size layer's H for every expert need not be on the host)."""

    def __init__(self, calib, experts):
        self.H = {int(e): calib[int(e)].double().cpu().numpy() for e in experts}

    def __getitem__(self, e):
        return self.H[int(e)]
