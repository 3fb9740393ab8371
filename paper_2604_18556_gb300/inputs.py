"""Seeded synthetic inputs for the GSQ step: weights W, calibration tokens X and
their Gram matrix H = X^T X.

These stand in for the paper's Llama-3.1 / Kimi-K2.5 weights and its
FineWeb-Edu / OpenThoughts calibration data (§4.1), which are not available
here.  Both the CUDA path and the CPU oracle consume these tensors; this module
holds none of the method's arithmetic (no noise, softmax, loss, gradients,
optimiser, projection or packing).

Recipe (per workload, see configs.py):
  * W[e, r, c] = 0.02 * z * rho_r,  z ~ N(0, 1),  log rho_r ~ U[log 0.5, log 2];
    rounded to bf16 (round-to-nearest-even) unless the workload keeps fp32.
  * tokens x ~ N(0, 1) (or Student-t with 3 degrees of freedom,
    z / sqrt(chi2_3 / 3)); a seeded random choice of `outliers` channels is
    multiplied by `outlier_scale`.
  * H_e = X_e^T X_e in fp32 (TF32 disabled), accumulated over chunks of 8192
    tokens so X is never held whole; symmetrised exactly as (H + H^T) / 2.
Every tensor draws from its own torch.Generator seeded with
data_seed + tensor id (+ 17 * expert), so results are reproducible per device
type.
"""
from __future__ import annotations

import math

import torch

from .configs import Workload

_W_ID, _ROWSCALE_ID, _X_ID, _OUTLIER_ID = 1, 2, 3, 4


def _gen(device, seed: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def make_weight(w: Workload, device="cpu", experts=None, rows=None) -> torch.Tensor:
    """W as [E, R, C] in the workload's storage dtype (fp32 or bf16).  experts /
    rows: [lo, hi) ranges of the layer's global expert and row indices to return
    (a shard's slice; default all), drawn exactly as in the whole layer."""
    out_dtype = torch.float32 if w.w_dtype == "f32" else torch.bfloat16
    e0, e1 = experts if experts is not None else (0, w.experts)
    r0, r1 = rows if rows is not None else (0, w.rows)
    W = torch.empty((e1 - e0, r1 - r0, w.cols), dtype=out_dtype, device=device)
    for e in range(e0, e1):
        g = _gen(device, w.data_seed + _W_ID + 17 * e)
        z = torch.randn((w.rows, w.cols), generator=g, device=device, dtype=torch.float32)
        gr = _gen(device, w.data_seed + _ROWSCALE_ID + 17 * e)
        u = torch.rand((w.rows, 1), generator=gr, device=device, dtype=torch.float32)
        rho = torch.exp(math.log(0.5) + u * (math.log(2.0) - math.log(0.5)))
        W[e - e0] = (0.02 * z * rho)[r0:r1].to(out_dtype)
    return W


def _outlier_channels(w: Workload, e: int, device) -> torch.Tensor:
    g = _gen("cpu", w.data_seed + _OUTLIER_ID + 17 * e)
    perm = torch.randperm(w.cols, generator=g)
    return perm[: w.outliers].to(device)


def _token_chunk(w: Workload, g: torch.Generator, ntok: int, device) -> torch.Tensor:
    z = torch.randn((ntok, w.cols), generator=g, device=device, dtype=torch.float32)
    if w.token_dist == "student_t3":
        c = torch.randn((3, ntok, w.cols), generator=g, device=device, dtype=torch.float32)
        chi2 = (c * c).sum(0)
        z = z / torch.sqrt(chi2 / 3.0)
    elif w.token_dist != "normal":
        raise ValueError(w.token_dist)
    return z


def make_tokens(w: Workload, device="cpu") -> torch.Tensor:
    """Calibration tokens X as [E, T, C] fp32 (small workloads only)."""
    X = torch.empty((w.experts, w.tokens, w.cols), dtype=torch.float32, device=device)
    for e in range(w.experts):
        g = _gen(device, w.data_seed + _X_ID + 17 * e)
        x = _token_chunk(w, g, w.tokens, device)
        if w.outliers:
            ch = _outlier_channels(w, e, device)
            x[:, ch] *= w.outlier_scale
        X[e] = x
    return X


def make_token_batch(w: Workload, step: int, micro: int, device="cpu") -> torch.Tensor:
    """Tokens of micro-batch `micro` of step `step` for a per-step-batch workload:
    [E, w.tokens, C] fp32, with the layer's outlier channels."""
    X = torch.empty((w.experts, w.tokens, w.cols), dtype=torch.float32, device=device)
    for e in range(w.experts):
        g = _gen(device, w.data_seed + _X_ID + 17 * e + 7919 * (step * max(w.micro, 1) + micro + 1))
        x = _token_chunk(w, g, w.tokens, device)
        if w.outliers:
            ch = _outlier_channels(w, e, device)
            x[:, ch] *= w.outlier_scale
        X[e] = x
    return X


def make_gram(w: Workload, device="cpu", chunk: int = 8192, experts=None) -> torch.Tensor:
    """H = X^T X as [E, C, C] fp32, built chunk by chunk with TF32 off; experts:
    [lo, hi) range of global expert indices to build (default all)."""
    prev = torch.backends.cuda.matmul.allow_tf32
    torch.backends.cuda.matmul.allow_tf32 = False
    e0, e1 = experts if experts is not None else (0, w.experts)
    try:
        H = torch.zeros((e1 - e0, w.cols, w.cols), dtype=torch.float32, device=device)
        for e in range(e0, e1):
            He = H[e - e0]
            g = _gen(device, w.data_seed + _X_ID + 17 * e)
            ch = _outlier_channels(w, e, device) if w.outliers else None
            done = 0
            while done < w.tokens:
                m = min(chunk, w.tokens - done)
                x = _token_chunk(w, g, m, device)
                if ch is not None:
                    x[:, ch] *= w.outlier_scale
                He.addmm_(x.t(), x)
                done += m
            H[e - e0] = 0.5 * (He + He.t())
        return H
    finally:
        torch.backends.cuda.matmul.allow_tf32 = prev
