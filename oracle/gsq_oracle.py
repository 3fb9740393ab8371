"""Plain CPU oracle for one GSQ optimisation step of a linear layer.

TEST INFRASTRUCTURE ONLY.  This is the slow, obviously-correct restatement of
the method that the CUDA path is checked against.  It shares no code with the
CUDA path; only tests, the smoke check and the benchmark's CPU-baseline leg may
import it.  Arithmetic is float64 (numpy) except where a floating-point value
decides an integer (initial round-to-nearest codes, the initial scales that
feed them, the K-Quant sub-scale codes): those decisions are taken in fp32,
the precision the kernels use, so both sides decide identically.  Optimiser
state is stored in fp32 between steps (the precision of the stored state on
both sides); within a step everything is float64.

What one step computes (paper references):
  noise      g_k ~ Gumbel(0,1) per weight and level, fresh each step
             (Alg. 1; §3.3 "Gradient accumulation")      -> philox.gumbel
  relax      p = softmax((kappa*l + g)/tau)  (Alg. 1)
  soft weight  w~ = sum_k p_k q_k  (Alg. 1 "return"); W^ = s_group * w~
             with one scale per group of consecutive inputs (§3.2 constraint
             set C_b-bit; §4.1 "Quantization configuration": symmetric,
             group-wise, groups row-wise over consecutive entries)
  loss       L = ||f(x; W^) - f(x; W)||_F^2 (Eq. 1) for a linear f:
             sum_t ||(W^ - W) x_t||^2 = tr(D H D^T), D = W^ - W, H = X^T X
  gradient   dL/dW^ = D (H + H^T); dL/ds_g = sum_{c in g} dL/dW^_c * w~_c;
             dL/dl_k = (kappa/tau) * dL/dW^ * s * p_k (q_k - w~)  (softmax
             Jacobian as written in the proof of the Lemma, App. B)
  optimiser  Lion (§3.3 "Optimizer"; App. B; Table 5 hyper-parameters):
             c = b1 m + (1-b1) g;  theta <- theta - lr (sign(c) + wd theta);
             m <- b2 m + (1-b2) g
  projection hard argmax of the noise-free logits (Alg. 2, final lines,
             generalised from the binary threshold to K levels)
  packing    symmetric group-wise b-bit codes + fp16 scale per group (§4.1),
             or a two-level K-Quant-like super-block (§4.4, App. E).
  local shift  (§3.2 "Higher bit-widths", Fig. 1): instead of one logit per grid
             level, 5 logits per weight for shifts delta in {-2..2} around the
             initial index j0; the level of shift delta is G[clip(j0 + delta)], so
             the same relaxation runs over a per-weight window of 5 levels.
  micro-batches (§3.3 "Objective", "Gradient accumulation"): a step on per-step
             token batches X_j; every forward pass draws fresh noise; the update
             uses the mean of the micro-batches' gradients.
  mask x sign  (§3.1, Alg. 2): ternary weights s * m * b with a mask logit l_m
             and a sign logit l_b per weight, each relaxed by a binary GS over
             {0, 1} resp. {-1, 1} with the tied logits (-l, l) (§3 notation
             paragraph: a sigmoid of the noisy logit 2l); hard rule
             m = [l_m >= 0], b = 2 [l_b >= 0] - 1.  The grid must be {-a, 0, a};
             w~ = a * m~ * b~.

Readings where the paper is silent are listed at the top of the design notes
(kappa multiplies the logit; summed, un-normalised loss; Philox stream; absmax
initial scale; RTN code with +bias logit init; weight decay on logits only;
sign(0) = 0; lowest index wins argmax ties; packing bit order; fp16 RNE).
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace
from typing import Optional

import numpy as np

from . import philox

SUB_BLOCK = 16      # K-Quant-like sub-block (one 6-bit sub-scale code)
SHIFTS = 5          # local-shift logits: delta in {-2, -1, 0, 1, 2} (§3.2)
SUPER_BLOCK = 256   # K-Quant-like super-block (one fp16 d)


# ----------------------------------------------------------------------------
# problem and state
# ----------------------------------------------------------------------------
@dataclass
class Problem:
    """Static inputs of one layer problem (the paper's problem statement, Eq. 1)."""
    E: int
    R: int
    C: int
    grid: np.ndarray                    # K ascending levels (float64)
    group: int                          # scale group size along the input dim
    seed: int = 0
    scale_mode: str = "group"           # "group" | "kquant2"
    H: Optional[np.ndarray] = None      # [E, C, C] float64
    X: Optional[np.ndarray] = None      # [E, T, C] float64 (loss taken literally over tokens)
    lr_logits: float = 1e-4
    lr_scales: float = 5e-5
    beta1: float = 0.9
    beta2: float = 0.95
    wd_logits: float = 1.0
    wd_scales: float = 0.0
    noise: bool = True
    shift: bool = False                 # local-shift parameterisation (§3.2)
    mask_sign: bool = False             # ternary mask x sign parameterisation (§3.1, Alg. 2)

    def __post_init__(self):
        if self.mask_sign:
            g = np.asarray(self.grid, dtype=np.float64)
            assert g.shape == (3,) and g[1] == 0.0 and g[0] == -g[2] and g[2] > 0, \
                "mask x sign needs the grid {-a, 0, a}"
            assert not self.shift

    @property
    def K(self) -> int:
        """Number of logits per weight: the grid size, 5 shifts, or 2 (mask, sign)."""
        if self.mask_sign:
            return 2
        return SHIFTS if self.shift else int(len(self.grid))

    @property
    def levels(self) -> int:
        return int(len(self.grid))


@dataclass
class RowState:
    """Optimiser state for a set of global rows (row id = e*R + r).

    Rows are independent in everything but the scalar loss, so the oracle can
    follow any subset of rows exactly."""
    row_ids: np.ndarray                 # int64 [nr]
    W: np.ndarray                       # float64 [nr, C] (values of the stored dtype)
    logits: np.ndarray                  # float32 [K, nr, C]
    scales: np.ndarray                  # float32 [nr, C // group]
    m_logits: np.ndarray                # float32 [K, nr, C]
    m_scales: np.ndarray                # float32 [nr, C // group]
    kq_d: Optional[np.ndarray] = None   # float32 [nr, C // 256] (fp16 values) for kquant2
    kq_sc: Optional[np.ndarray] = None  # int32 [nr, C // 16] for kquant2
    j0: Optional[np.ndarray] = None     # uint8 [nr, C]: initial grid index (local shift)

    def copy(self) -> "RowState":
        return RowState(self.row_ids.copy(), self.W.copy(), self.logits.copy(),
                        self.scales.copy(), self.m_logits.copy(), self.m_scales.copy(),
                        None if self.kq_d is None else self.kq_d.copy(),
                        None if self.kq_sc is None else self.kq_sc.copy(),
                        None if self.j0 is None else self.j0.copy())

    def subset(self, idx) -> "RowState":
        idx = np.asarray(idx)
        return RowState(self.row_ids[idx].copy(), self.W[idx].copy(),
                        self.logits[:, idx].copy(), self.scales[idx].copy(),
                        self.m_logits[:, idx].copy(), self.m_scales[idx].copy(),
                        None if self.kq_d is None else self.kq_d[idx].copy(),
                        None if self.kq_sc is None else self.kq_sc[idx].copy(),
                        None if self.j0 is None else self.j0[idx].copy())


def flat_index(prob: Problem, row_ids: np.ndarray) -> np.ndarray:
    """i = (e*R + r)*C + c for every weight of the given rows: [nr, C]."""
    return row_ids.astype(np.int64)[:, None] * prob.C + np.arange(prob.C, dtype=np.int64)[None, :]


def expand_scales(scales: np.ndarray, group: int) -> np.ndarray:
    """Per-weight scale s_{r, floor(c/G)} as float64 [nr, C]."""
    return np.repeat(scales.astype(np.float64), group, axis=1)


# ----------------------------------------------------------------------------
# forward: noise, relaxation, soft weight (Alg. 1, §3.2)
# ----------------------------------------------------------------------------
def relax(logits: np.ndarray, g, tau: float, kappa: float) -> np.ndarray:
    """p_k = exp((kappa l_k + g_k)/tau) / sum_j exp((kappa l_j + g_j)/tau)  (Alg. 1).

    Level axis first.  The common shift by max_j is the usual overflow guard and
    leaves the ratio unchanged."""
    z = (kappa * logits.astype(np.float64) + g) / tau
    z = z - z.max(axis=0, keepdims=True)
    e = np.exp(z)
    return e / e.sum(axis=0, keepdims=True)


def soft_value(p: np.ndarray, grid: np.ndarray) -> np.ndarray:
    """w~ = sum_k p_k q_k (Alg. 1, soft sample over the grid)."""
    return np.tensordot(np.asarray(grid, dtype=np.float64), p, axes=(0, 0))


def noise(prob: Problem, st: RowState, t: int) -> np.ndarray:
    """Gumbel draws [K, nr, C]; for mask x sign, one logistic draw per binary
    instance [2, nr, C] (mask, sign), the difference of its two Gumbel draws."""
    if not prob.noise:
        return np.zeros((prob.K, len(st.row_ids), prob.C))
    if prob.mask_sign:
        return philox.logistic(prob.seed, t, flat_index(prob, st.row_ids))
    return philox.gumbel(prob.seed, t, flat_index(prob, st.row_ids), prob.K)


def shift_index(j0: np.ndarray, levels: int) -> np.ndarray:
    """Grid index of every shift: clip(j0 + delta, 0, levels - 1), delta = -2..2
    (§3.2: j_i = clip(j_i^0 + delta_i, 1, 2^b) with 1-based indices).  [5, ...]."""
    delta = np.arange(-2, 3).reshape((SHIFTS,) + (1,) * np.ndim(j0))
    return np.clip(np.asarray(j0, dtype=np.int64)[None] + delta, 0, levels - 1)


def level_values(prob: Problem, st: RowState) -> np.ndarray:
    """q_k for every logit k of every weight, broadcastable against [K, nr, C]:
    the grid itself, or each weight's window G[clip(j0 + delta)] (local shift)."""
    grid = np.asarray(prob.grid, dtype=np.float64)
    if prob.shift:
        return grid[shift_index(st.j0, prob.levels)]
    return grid[:, None, None]


@dataclass
class Forward:
    g: np.ndarray
    p: np.ndarray
    wtil: np.ndarray
    s: np.ndarray
    What: np.ndarray
    D: np.ndarray
    soft: Optional[np.ndarray] = None   # mask x sign: [2, nr, C] = (m~, b~)


BINARY_VALUES = (np.array([0.0, 1.0]), np.array([-1.0, 1.0]))   # mask {0,1}, sign {-1,1}


def binary_gs(l, lam, values, tau: float, kappa: float):
    """One binary GS instance of Alg. 2: Alg. 1 over the two values with the
    tied logits (-l, l) (§3 notation paragraph) and the noise pair (0, lam),
    lam being the difference of the pair's two Gumbel draws (only the
    difference enters the softmax).  Returns (p [2, ...], soft value)."""
    l = np.asarray(l, dtype=np.float64)
    p = relax(np.stack([-l, l]), np.stack([np.zeros_like(lam), lam]), tau, kappa)
    return p, soft_value(p, values)


def forward(prob: Problem, st: RowState, t: int, tau: float, kappa: float) -> Forward:
    g = noise(prob, st, t)
    if prob.mask_sign:
        a = float(prob.grid[2])
        pm, mt = binary_gs(st.logits[0], g[0], BINARY_VALUES[0], tau, kappa)
        pb, bt = binary_gs(st.logits[1], g[1], BINARY_VALUES[1], tau, kappa)
        wtil = a * mt * bt                                # w~ = a m~ b~ (Alg. 2)
        s = expand_scales(st.scales, prob.group)
        What = s * wtil
        return Forward(g=g, p=np.stack([pm, pb]), wtil=wtil, s=s, What=What, D=What - st.W,
                       soft=np.stack([mt, bt]))
    p = relax(st.logits, g, tau, kappa)
    wtil = np.sum(p * level_values(prob, st), axis=0)     # w~ = sum_k p_k q_k
    s = expand_scales(st.scales, prob.group)
    What = s * wtil
    return Forward(g=g, p=p, wtil=wtil, s=s, What=What, D=What - st.W)


# ----------------------------------------------------------------------------
# loss and its gradient w.r.t. the soft weight (Eq. 1 with a linear layer)
# ----------------------------------------------------------------------------
def loss_and_grad(prob: Problem, row_ids: np.ndarray, D: np.ndarray):
    """L = sum_rows D_r H_e D_r^T and dL/dW^ = D (H_e + H_e^T), per expert e.

    With calibration tokens (prob.X) the loss is taken literally as
    sum_t ||D x_t||^2 and the gradient as 2 (D X^T) X."""
    G = np.empty_like(D)
    L = 0.0
    experts = row_ids // prob.R
    for e in np.unique(experts):
        sel = experts == e
        De = D[sel]
        if prob.X is not None:
            Xe = prob.X[e]
            Y = De @ Xe.T                        # rows of (W^ - W) x_t, one column per token
            L += float(np.sum(Y * Y))
            G[sel] = 2.0 * (Y @ Xe)
        else:
            He = prob.H[e]
            DH = De @ He
            L += float(np.sum(DH * De))
            G[sel] = DH + De @ He.T              # D (H + H^T)
    return L, G


def loss_bruteforce(W: np.ndarray, What: np.ndarray, X: np.ndarray) -> float:
    """sum over tokens of ||(W - W^) x_t||^2 with explicit Python loops (tiny inputs only)."""
    R, C = W.shape
    total = 0.0
    for x in X:
        for r in range(R):
            acc = 0.0
            for c in range(C):
                acc += (W[r, c] - What[r, c]) * x[c]
            total += acc * acc
    return total


# ----------------------------------------------------------------------------
# backward (App. B softmax Jacobian) and Lion (§3.3, App. B)
# ----------------------------------------------------------------------------
def centred_values(p, values):
    """d_k - w~ for every k, with w~ = sum_j p_j d_j, written as
    sum_j p_j (d_k - d_j) (equal because sum_j p_j = 1).  The direct difference
    cancels catastrophically when p is nearly one-hot (d_m - w~ is then tiny);
    this form keeps full relative accuracy in float64.  p: [K, ...]; values
    broadcastable against p."""
    p = np.asarray(p, dtype=np.float64)
    d = np.broadcast_to(np.asarray(values, dtype=np.float64), p.shape)
    out = np.zeros(p.shape)
    for k in range(p.shape[0]):
        out[k] = np.sum(p * (d[k][None] - d), axis=0)
    return out


def binary_gs_grad(p, soft, values, tau: float, kappa: float):
    """d(soft value)/dl of a binary instance: the softmax Jacobian (App. B)
    d w~/d l_k = (kappa/tau) p_k (d_k - w~), chained through the tied logits
    l_1 = l, l_0 = -l."""
    vals = np.asarray(values, dtype=np.float64).reshape((2,) + (1,) * (np.ndim(p) - 1))
    c = centred_values(p, vals)
    return (kappa / tau) * (p[1] * c[1] - p[0] * c[0])


def backward(prob: Problem, fw: Forward, G: np.ndarray, tau: float, kappa: float, q=None):
    """dL/dl [K, nr, C] and dL/ds [nr, C/G]; q: level values of every logit."""
    nr, C = G.shape
    if prob.mask_sign:
        a = float(prob.grid[2])
        mt, bt = fw.soft
        gm = binary_gs_grad(fw.p[0], mt, BINARY_VALUES[0], tau, kappa)
        gb = binary_gs_grad(fw.p[1], bt, BINARY_VALUES[1], tau, kappa)
        Gs = G * fw.s
        d_logits = np.stack([Gs * a * bt * gm, Gs * a * mt * gb])   # W^ = s a m~ b~
        d_scales = (G * fw.wtil).reshape(nr, C // prob.group, prob.group).sum(axis=2)
        return d_logits, d_scales
    if q is None:
        q = np.asarray(prob.grid, dtype=np.float64)[:, None, None]
    # softmax Jacobian (App. B): dL/dl_k = (kappa/tau) G s p_k (q_k - w~)
    d_logits = (kappa / tau) * (G * fw.s)[None] * fw.p * centred_values(fw.p, q)
    d_scales = (G * fw.wtil).reshape(nr, C // prob.group, prob.group).sum(axis=2)
    return d_logits, d_scales


def lion(theta32: np.ndarray, m32: np.ndarray, grad: np.ndarray, lr: float, b1: float,
         b2: float, wd: float):
    """One Lion update with decoupled weight decay (Chen et al. 2023, the
    optimiser the paper adopts in §3.3); sign(0) = 0.  Returns fp32 state."""
    theta = theta32.astype(np.float64)
    m = m32.astype(np.float64)
    c = b1 * m + (1.0 - b1) * grad
    theta_new = theta - lr * (np.sign(c) + wd * theta)
    m_new = b2 * m + (1.0 - b2) * grad
    return theta_new.astype(np.float32), m_new.astype(np.float32)


def scales_frozen(prob: Problem) -> bool:
    return prob.lr_scales == 0.0 and prob.wd_scales == 0.0


@dataclass
class StepResult:
    loss: float
    fw: Forward
    G: np.ndarray
    d_logits: np.ndarray
    d_scales: Optional[np.ndarray]


def step(prob: Problem, st: RowState, t: int, tau: float, kappa: float,
         update: bool = True) -> StepResult:
    """One optimisation step t on the given rows (Alg. 2's loop body generalised
    to K levels: sample, soft weight, loss, gradient, update).  Updates `st` in
    place unless update=False; the reported loss is this step's forward loss."""
    fw = forward(prob, st, t, tau, kappa)
    L, G = loss_and_grad(prob, st.row_ids, fw.D)
    q = None if prob.mask_sign else level_values(prob, st)
    d_logits, d_scales = backward(prob, fw, G, tau, kappa, q=q)
    if scales_frozen(prob):
        d_scales = None
    if update:
        st.logits, st.m_logits = lion(st.logits, st.m_logits, d_logits, prob.lr_logits,
                                      prob.beta1, prob.beta2, prob.wd_logits)
        if d_scales is not None:
            st.scales, st.m_scales = lion(st.scales, st.m_scales, d_scales, prob.lr_scales,
                                          prob.beta1, prob.beta2, prob.wd_scales)
    return StepResult(loss=L, fw=fw, G=G, d_logits=d_logits, d_scales=d_scales)


@dataclass
class MicroStepResult:
    losses: list                        # L_j of every micro-batch (before the update)
    d_logits: np.ndarray                # mean over the micro-batches
    d_scales: Optional[np.ndarray]


def step_microbatches(prob: Problem, st: RowState, t: int, batches, tau: float, kappa: float,
                      update: bool = True) -> MicroStepResult:
    """One optimisation step on per-step calibration tokens with gradient
    accumulation over resampled noise (§3.3 "Objective" and "Gradient
    accumulation").  batches: M token arrays X_j [E, T_j, C].  Micro-batch j
    draws fresh noise (counter t*M + j: every forward pass is a new draw),
    forms W^_j, its loss L_j = sum over its tokens of ||(W^_j - W) x||^2 (Eq. 1)
    and the gradients; the update applies the mean gradient over the
    micro-batches.  The state is unchanged until that update."""
    M = len(batches)
    q = None if prob.mask_sign else level_values(prob, st)
    acc_l = acc_s = None
    losses = []
    for j, X in enumerate(batches):
        pj = replace(prob, X=np.asarray(X, dtype=np.float64), H=None)
        fw = forward(pj, st, t * M + j, tau, kappa)
        L, G = loss_and_grad(pj, st.row_ids, fw.D)
        dl, ds = backward(pj, fw, G, tau, kappa, q=q)
        acc_l = dl if acc_l is None else acc_l + dl
        acc_s = ds if acc_s is None else acc_s + ds
        losses.append(L)
    d_logits = acc_l / M
    d_scales = None if scales_frozen(prob) else acc_s / M
    if update:
        st.logits, st.m_logits = lion(st.logits, st.m_logits, d_logits, prob.lr_logits,
                                      prob.beta1, prob.beta2, prob.wd_logits)
        if d_scales is not None:
            st.scales, st.m_scales = lion(st.scales, st.m_scales, d_scales, prob.lr_scales,
                                          prob.beta1, prob.beta2, prob.wd_scales)
    return MicroStepResult(losses=losses, d_logits=d_logits, d_scales=d_scales)


# ----------------------------------------------------------------------------
# initialisation (readings: absmax scale, round-to-nearest code, +bias logit)
# ----------------------------------------------------------------------------
def f32_to_f16_bits(x) -> np.ndarray:
    """IEEE 754 binary32 -> binary16, round to nearest, ties to even; returns uint16 bits.

    Written from the format definition: 1 sign, 5 exponent (bias 15), 10
    fraction bits; subnormal quantum 2^-24; magnitudes >= 65520 overflow to inf."""
    x = np.asarray(x, dtype=np.float32)
    a = np.abs(x.astype(np.float64))
    sign = np.where(np.signbit(x), 0x8000, 0).astype(np.uint32)
    out = np.zeros(x.shape, dtype=np.uint32)
    nan = np.isnan(x)
    big = (~nan) & (a >= 65520.0)
    fin = (~nan) & (~big)
    _, ex = np.frexp(np.where(fin & (a > 0), a, 1.0))
    e = ex - 1                                        # a = m * 2^e with m in [1, 2)
    e = np.maximum(e, -14)                            # below 2^-14 the quantum stays 2^-24
    quantum = np.ldexp(1.0, e - 10)
    v = np.rint(a / quantum) * quantum                # exact: a has <= 24 significant bits
    v = np.where(fin, v, 0.0)
    _, ev = np.frexp(np.where(v > 0, v, 1.0))
    ev = ev - 1
    normal = v >= 2.0 ** -14
    exp_field = np.where(normal, ev + 15, 0)
    frac = np.where(normal, v / np.ldexp(1.0, ev - 10) - 1024.0, v / 2.0 ** -24)
    bits = (exp_field.astype(np.uint32) << 10) | frac.astype(np.uint32)
    out = np.where(fin, bits, out)
    out = np.where(big, 0x7C00, out)
    out = np.where(nan, 0x7E00, out)
    return (out | sign).astype(np.uint16)


def f16_bits_to_f32(h) -> np.ndarray:
    """binary16 bits -> float value (exact)."""
    h = np.asarray(h, dtype=np.uint32)
    s = np.where(h & 0x8000, -1.0, 1.0)
    e = (h >> 10) & 0x1F
    f = (h & 0x3FF).astype(np.float64)
    v = np.where(e == 0, f * 2.0 ** -24, np.ldexp(1.0 + f / 1024.0, e.astype(np.int64) - 15))
    v = np.where(e == 31, np.where(f == 0, np.inf, np.nan), v)
    return (s * v).astype(np.float32)


def rtn_codes(W32: np.ndarray, s32: np.ndarray, grid: np.ndarray) -> np.ndarray:
    """Round-to-nearest grid index k0 = argmin_k |W/s - q_k| in fp32 (lowest k on
    ties); a zero scale maps to the level of smallest magnitude."""
    q32 = np.asarray(grid, dtype=np.float32)
    with np.errstate(divide="ignore", invalid="ignore"):
        x = W32 / s32
    dist = np.abs(x[None] - q32.reshape((-1,) + (1,) * W32.ndim))
    codes = np.argmin(dist, axis=0)
    zero_code = int(np.argmin(np.abs(q32)))
    return np.where(s32 == 0, zero_code, codes).astype(np.uint8)


def init_group_scales(W32: np.ndarray, group: int, grid: np.ndarray) -> np.ndarray:
    """s_g = max_{c in g} |W_c| / max_k |q_k| in fp32; 1 for an all-zero group."""
    nr, C = W32.shape
    absmax = np.abs(W32).reshape(nr, C // group, group).max(axis=2)
    qmax = np.float32(np.max(np.abs(np.asarray(grid, dtype=np.float32))))
    s = (absmax / qmax).astype(np.float32)
    return np.where(absmax == 0, np.float32(1.0), s).astype(np.float32)


def init_kquant2_scales(W32: np.ndarray, grid: np.ndarray):
    """Two-level scales: sub-scale s_j = absmax_16 / qmax; d = fp16(max_j s_j / 31)
    per 256-weight super-block; sc_j = clamp(rne(s_j / d), -32, 31) (0 when d = 0);
    effective scale d * sc_j (exact in fp32).  All fp32."""
    nr, C = W32.shape
    qmax = np.float32(np.max(np.abs(np.asarray(grid, dtype=np.float32))))
    sj = (np.abs(W32).reshape(nr, C // SUB_BLOCK, SUB_BLOCK).max(axis=2) / qmax).astype(np.float32)
    smax = sj.reshape(nr, C // SUPER_BLOCK, SUPER_BLOCK // SUB_BLOCK).max(axis=2)
    d = f16_bits_to_f32(f32_to_f16_bits((smax / np.float32(31.0)).astype(np.float32)))
    d_sub = np.repeat(d, SUPER_BLOCK // SUB_BLOCK, axis=1)
    with np.errstate(divide="ignore", invalid="ignore"):
        ratio = (sj / d_sub).astype(np.float32)
    sc = np.where(d_sub > 0, np.clip(np.rint(ratio), -32, 31), 0).astype(np.int32)
    s_eff = (d_sub * sc.astype(np.float32)).astype(np.float32)
    return s_eff, d, sc


def init_state(prob: Problem, W, row_ids, init_bias: float = 2.0) -> RowState:
    """Initial state: scales, RTN codes, logits = init_bias on the RTN level
    (0 elsewhere), zero Lion momenta.  W holds the rows' stored values."""
    W32 = np.asarray(W, dtype=np.float32)
    nr, C = W32.shape
    kq_d = kq_sc = None
    if prob.scale_mode == "kquant2":
        s, kq_d, kq_sc = init_kquant2_scales(W32, prob.grid)
        assert prob.group == SUB_BLOCK
    else:
        s = init_group_scales(W32, prob.group, prob.grid)
    codes = rtn_codes(W32, np.repeat(s, prob.group, axis=1), prob.grid)
    logits = np.zeros((prob.K, nr, C), dtype=np.float32)
    j0 = None
    if prob.mask_sign:
        # Eq. 3 with the RTN code in place of the GPTQ one, scaled by init_bias:
        # l_m = +1 if the code is nonzero else -1; l_b = sign of the code (0 for 0)
        b = np.float32(init_bias)
        logits[0] = np.where(codes != 1, b, -b)
        logits[1] = np.where(codes == 2, b, np.where(codes == 0, -b, np.float32(0.0)))
    elif prob.shift:
        logits[2] = np.float32(init_bias)             # delta = 0: stay on the RTN level
        j0 = codes.astype(np.uint8)
    else:
        for k in range(prob.K):
            logits[k][codes == k] = np.float32(init_bias)
    return RowState(row_ids=np.asarray(row_ids, dtype=np.int64), W=W32.astype(np.float64),
                    logits=logits, scales=s.astype(np.float32),
                    m_logits=np.zeros_like(logits), m_scales=np.zeros_like(s, dtype=np.float32),
                    kq_d=kq_d, kq_sc=kq_sc, j0=j0)


def prior_logits(prob: Problem, codes) -> np.ndarray:
    """The noise-free warm-start logits l_GPTQ around a supplied code vector
    ([K, nr, C] float64), for the code of every weight (a grid index):
      mask x sign (Eq. 3): l_m = +1 if the code is nonzero else -1;
                           l_b = +1, -1 or 0 by the code's sign;
      full grid (App. A, b = 2): l_k = -(c_k - mu)^2 / 2 with the candidates
                           c_k the grid values and mu the coded value;
      local shift (App. A, b > 2): the candidates are the shifts -2..2 and
                           mu = 0;
    in the last two cases minus each weight's mean logit (App. A)."""
    codes = np.asarray(codes, dtype=np.int64)
    if prob.mask_sign:
        lm = np.where(codes != 1, 1.0, -1.0)
        lb = np.where(codes == 2, 1.0, np.where(codes == 0, -1.0, 0.0))
        return np.stack([lm, lb])
    if prob.shift:
        c = np.arange(-2, 3, dtype=np.float64).reshape((SHIFTS,) + (1,) * codes.ndim)
        mu = np.zeros(codes.shape)
    else:
        grid = np.asarray(prob.grid, dtype=np.float64)
        c = grid.reshape((len(grid),) + (1,) * codes.ndim)
        mu = grid[codes]
    l = -0.5 * (c - mu[None]) ** 2
    return l - l.mean(axis=0, keepdims=True)


def init_from_codes(prob: Problem, W, row_ids, codes, eps, alpha: float, sigma: float,
                    scales=None) -> RowState:
    """Warm start from a supplied solution (§3.1 "Initialization", Eq. 3-4;
    App. A): logits l = sigma (eps + alpha l_GPTQ) with eps ~ N(0, I) given by
    the caller ([K, nr, C]; None for eps = 0), zero momenta, the given scales
    (default: the absmax scales of init_state), and for local shift j0 = the
    supplied codes."""
    st = init_state(prob, W, row_ids)
    codes = np.asarray(codes, dtype=np.int64)
    lg = prior_logits(prob, codes)
    e = np.zeros_like(lg) if eps is None else np.asarray(eps, dtype=np.float64)
    st.logits = (sigma * (e + alpha * lg)).astype(np.float32)
    st.m_logits = np.zeros_like(st.logits)
    if scales is not None:
        st.scales = np.asarray(scales, dtype=np.float32).copy()
    if prob.shift:
        st.j0 = codes.astype(np.uint8)
    return st


# ----------------------------------------------------------------------------
# hard projection (Alg. 2, final lines, generalised to K levels)
# ----------------------------------------------------------------------------
def project_mask_sign(logits32: np.ndarray):
    """Alg. 2, final lines: m = [l_m >= 0], b = 2 [l_b >= 0] - 1; grid code of
    s * m * b on {-a, 0, a}: 0, 1 or 2.  Margin: the top-two logit gap 2|l| of
    every instance that decides the code (the mask; the sign when m = 1)."""
    lm, lb = logits32[0], logits32[1]
    m = lm >= 0
    b = lb >= 0
    codes = np.where(m, np.where(b, 2, 0), 1).astype(np.uint8)
    gm = 2 * np.abs(lm.astype(np.float32))
    gb = 2 * np.abs(lb.astype(np.float32))
    margin = np.where(m, np.minimum(gm, gb), gm).astype(np.float32)
    return codes, margin


def project(logits32: np.ndarray, j0=None, levels: int = 0, mask_sign: bool = False):
    """k* = argmax_k l_k (lowest k on ties) and margin = l_(1) - l_(2) in fp32.
    With local shift the grid code is clip(j0 + k* - 2) (§3.2)."""
    if mask_sign:
        return project_mask_sign(logits32)
    k = np.argmax(logits32, axis=0)
    srt = np.sort(logits32, axis=0)
    margin = (srt[-1] - srt[-2]).astype(np.float32)
    if j0 is not None:
        k = np.clip(np.asarray(j0, dtype=np.int64) + k - 2, 0, levels - 1)
    return k.astype(np.uint8), margin


# ----------------------------------------------------------------------------
# diagnostics (not part of the step): displacement, saturation, margins
# ----------------------------------------------------------------------------
MARGIN_EDGES = np.float32([1e-6, 1e-5, 1e-4, 1e-3, 1e-2, 1e-1, 1.0, 10.0])   # 9 bins
SHIFT_BINS = 8


def diagnostics(prob: Problem, st: RowState, code0, tau: float, kappa: float):
    """Three diagnostics of the current logits (no noise):
      * displacement: histogram of |projected code - initial code| in grid steps
        (App. L's local-shift statistic, measured on the full parameterisation);
      * saturation: mean over weights of max_k p_k with p = softmax(kappa l / tau)
        (for mask x sign, of the three-value distribution the two binary instances
        define), the regime where the logit gradients vanish (App. B);
      * margins: histogram of the top-two logit gap of the projection (bins split
        at MARGIN_EDGES, compared in fp32).
    Returns (displacement counts [8], mean max-probability, margin counts [9])."""
    codes, margin = project(st.logits, j0=st.j0, levels=prob.levels, mask_sign=prob.mask_sign)
    disp = np.abs(codes.astype(np.int64) - np.asarray(code0, dtype=np.int64))
    disp_hist = np.bincount(np.minimum(disp, SHIFT_BINS - 1).reshape(-1), minlength=SHIFT_BINS)
    l = st.logits.astype(np.float64)
    if prob.mask_sign:
        pm = 1.0 / (1.0 + np.exp(-2.0 * kappa * l[0] / tau))
        pb = 1.0 / (1.0 + np.exp(-2.0 * kappa * l[1] / tau))
        pmax = np.maximum(np.maximum(pm * (1 - pb), 1 - pm), pm * pb)
    else:
        pmax = relax(st.logits, 0.0, tau, kappa).max(axis=0)
    m = np.asarray(margin, dtype=np.float32).reshape(-1)
    bins = np.zeros(m.shape, dtype=np.int64)
    for e in MARGIN_EDGES:
        bins += (m >= e)
    margin_hist = np.bincount(bins, minlength=len(MARGIN_EDGES) + 1)
    return disp_hist, float(pmax.mean()), margin_hist


# ----------------------------------------------------------------------------
# packing (§4.1 symmetric group-wise codes + fp16 scale; §4.4 / App. E K-Quant)
# ----------------------------------------------------------------------------
def code_bits(K: int) -> int:
    return 2 if K <= 4 else 3


def bits_per_param(K: int, group: int) -> float:
    """The paper's storage accounting: log2(#levels) bits per code plus a 16-bit
    scale per group (Table 1: 2.13, 3.13 and 1.71 bit/param at group 128)."""
    return float(np.log2(K)) + 16.0 / group


def _pack_stream(codes: np.ndarray, bits: int) -> np.ndarray:
    """Little-endian bit stream: element j of every 32-element chunk at bit bits*j
    of that chunk's bits-word (96-bit for 3-bit codes, 64-bit for 2-bit); words
    emitted as little-endian uint32.  Returns uint32 words."""
    c = codes.astype(np.uint64).reshape(-1)
    n = c.size
    pad = (-n) % 32
    if pad:
        c = np.concatenate([c, np.zeros(pad, dtype=np.uint64)])
    chunks = c.reshape(-1, 32)
    words = np.zeros((chunks.shape[0], bits), dtype=np.uint64)
    for j in range(32):
        p = bits * j
        w, o = p // 32, p % 32
        words[:, w] |= (chunks[:, j] << np.uint64(o)) & np.uint64(0xFFFFFFFF)
        if o + bits > 32:
            words[:, w + 1] |= chunks[:, j] >> np.uint64(32 - o)
    return words.reshape(-1).astype(np.uint32)


def _unpack_stream(words: np.ndarray, bits: int, n: int) -> np.ndarray:
    w = np.asarray(words, dtype=np.uint64).reshape(-1, bits)
    out = np.zeros((w.shape[0], 32), dtype=np.uint64)
    mask = np.uint64((1 << bits) - 1)
    for j in range(32):
        p = bits * j
        k, o = p // 32, p % 32
        v = w[:, k] >> np.uint64(o)
        if o + bits > 32:
            v = v | (w[:, k + 1] << np.uint64(32 - o))
        out[:, j] = v & mask
    return out.reshape(-1)[:n].astype(np.uint8)


def code_section_bytes(n: int, K: int) -> int:
    b = code_bits(K)
    raw = ((n + 31) // 32) * 4 * b
    return (raw + 15) // 16 * 16


def pack_group(codes: np.ndarray, scales32: np.ndarray, K: int) -> bytes:
    """codes [E*R*C] row-major, scales [E*R*C/G] row-major ->
    [code stream, padded to 16 B] || [fp16 scales, little-endian]."""
    n = codes.size
    words = _pack_stream(codes, code_bits(K))
    code_sec = words.astype("<u4").tobytes()
    code_sec += b"\0" * (code_section_bytes(n, K) - len(code_sec))
    return code_sec + f32_to_f16_bits(scales32.reshape(-1)).astype("<u2").tobytes()


def unpack_group(buf: bytes, n: int, K: int, n_groups: int):
    cs = code_section_bytes(n, K)
    bits = code_bits(K)
    nw = ((n + 31) // 32) * bits
    words = np.frombuffer(buf[: nw * 4], dtype="<u4")
    codes = _unpack_stream(words, bits, n)
    sc = np.frombuffer(buf[cs: cs + 2 * n_groups], dtype="<u2")
    return codes, sc


KQ_RECORD = 110   # 96 B codes || 12 B sub-scales || 2 B fp16 d


def pack_kquant2(codes: np.ndarray, d32: np.ndarray, sc: np.ndarray) -> bytes:
    """One 110-byte record per 256 consecutive weights (row-major):
    3-bit codes (same stream as pack_group) || 16 sub-scale codes sc+32 as a
    6-bit little-endian stream || fp16 d."""
    nb = codes.size // SUPER_BLOCK
    cw = _pack_stream(codes.reshape(nb, SUPER_BLOCK), 3).reshape(nb, 24)
    s6 = (sc.reshape(nb, 16).astype(np.int64) + 32).astype(np.uint64)
    sw = np.zeros((nb, 3), dtype=np.uint64)
    for j in range(16):
        p = 6 * j
        w, o = p // 32, p % 32
        sw[:, w] |= (s6[:, j] << np.uint64(o)) & np.uint64(0xFFFFFFFF)
        if o + 6 > 32:
            sw[:, w + 1] |= s6[:, j] >> np.uint64(32 - o)
    dh = f32_to_f16_bits(d32.reshape(nb)).astype("<u2")
    rec = np.zeros((nb, KQ_RECORD), dtype=np.uint8)
    rec[:, :96] = cw.astype("<u4").view(np.uint8).reshape(nb, 96)
    rec[:, 96:108] = sw.astype(np.uint32).astype("<u4").view(np.uint8).reshape(nb, 12)
    rec[:, 108:110] = dh.view(np.uint8).reshape(nb, 2)
    return rec.tobytes()


def unpack_kquant2(buf: bytes, n: int):
    nb = n // SUPER_BLOCK
    rec = np.frombuffer(buf, dtype=np.uint8)[: nb * KQ_RECORD].reshape(nb, KQ_RECORD)
    cw = rec[:, :96].copy().view("<u4").reshape(-1)
    codes = _unpack_stream(cw, 3, n)
    sw = rec[:, 96:108].copy().view("<u4").astype(np.uint64).reshape(nb, 3)
    sc = np.zeros((nb, 16), dtype=np.int32)
    for j in range(16):
        p = 6 * j
        w, o = p // 32, p % 32
        v = sw[:, w] >> np.uint64(o)
        if o + 6 > 32:
            v = v | (sw[:, w + 1] << np.uint64(32 - o))
        sc[:, j] = (v & np.uint64(63)).astype(np.int32) - 32
    d = f16_bits_to_f32(rec[:, 108:110].copy().view("<u2").reshape(nb))
    return codes, d, sc
