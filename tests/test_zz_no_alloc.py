"""The allocation-free backward + Lion update against the handle-based step.

gsq_backward_update_noalloc serves callers that cannot allocate device memory
(a host that owns a fixed memory pool, a plugin whose host forbids allocation):
they keep the optimiser state in their own buffers and the call's only scratch
is a static array inside libgsq.  Here the state lives in caller-owned torch
buffers; each step, the handle-based gsq_step runs on a layer with the same
initial state, and the new entry point, given that step's dL/dW^ (read from the
layer), must leave the caller's buffers equal to the layer's state and report
the same loss.  Two calls in a row, in both GEMM precisions, and once at the
largest layer the static scratch serves (4096 x 4096, 2^24 weights).  This file sorts
last so that a run stopping at the first failure has run every other test."""
import ctypes

import numpy as np
import pytest
import torch

from gpu_common import TOL_F32, gsq
from paper_2604_18556_gb300 import configs as C
from paper_2604_18556_gb300 import inputs

pytestmark = pytest.mark.gpu


def _args(g, w, W, G, st, loss, t, tau, kappa, d_dtype):
    a = g.gsq_backward_args()
    a.num_experts, a.out_features, a.in_features = w.experts, w.rows, w.cols
    a.num_levels = w.K
    for k, q in enumerate(w.grid):
        a.grid[k] = q
    a.group_size = w.group
    a.w_dtype = g.GSQ_DTYPE_BF16 if W.dtype == torch.bfloat16 else g.GSQ_DTYPE_F32
    a.d_dtype = d_dtype
    a.flags = 0
    a.W, a.G = W.data_ptr(), G.data_ptr()
    a.logits = st[g.GSQ_T_LOGITS].data_ptr()
    a.m_logits = st[g.GSQ_T_MOM_LOGITS].data_ptr()
    a.scales = st[g.GSQ_T_SCALES].data_ptr()
    a.m_scales = st[g.GSQ_T_MOM_SCALES].data_ptr()
    a.loss_dev = loss.data_ptr()
    a.seed, a.step, a.tau, a.kappa = w.seed, t, tau, kappa
    a.lr_logits, a.lr_scales, a.beta1, a.beta2 = w.lr_logits, w.lr_scales, w.beta1, w.beta2
    a.wd_logits, a.wd_scales = w.wd_logits, w.wd_scales
    return a


@pytest.mark.parametrize("gemm,rows,cols", [
    ("f32", 192, 512), ("bf16", 192, 512),
    # exactly the documented limit of 2^24 weights: the last thread block writes the
    # last partial slot of the static scratch array
    ("bf16", 4096, 4096)])
def test_noalloc_update_matches_step(gemm, rows, cols):
    g = gsq()
    w = C.shrunk(C.WORKLOADS["llama8b_q_proj"], rows=rows, cols=cols,
                 tokens=2048 if rows * cols < (1 << 24) else None)
    W = inputs.make_weight(w, device="cuda").contiguous()
    H = inputs.make_gram(w, device="cuda")
    layer = g.Layer(W, H, w.grid, w.group, gemm=gemm, seed=w.seed, lr_logits=w.lr_logits,
                    lr_scales=w.lr_scales, beta1=w.beta1, beta2=w.beta2,
                    wd_logits=w.wd_logits, wd_scales=w.wd_scales)
    kinds = (g.GSQ_T_LOGITS, g.GSQ_T_MOM_LOGITS, g.GSQ_T_SCALES, g.GSQ_T_MOM_SCALES)
    st = {k: layer.get_tensor(k, torch.float32).clone() for k in kinds}   # caller-owned state
    d_dtype = g.GSQ_DTYPE_BF16 if gemm == "bf16" else g.GSQ_DTYPE_F32
    stream = torch.cuda.current_stream().cuda_stream
    for t, tau in ((0, 0.9), (1, 0.8)):
        loss_ref = torch.zeros(1, device="cuda")
        loss_na = torch.full((1,), float("nan"), device="cuda")
        layer.step(t, tau, 1.0, loss=loss_ref)
        G = layer.get_tensor(g.GSQ_T_G, torch.float32).clone()
        g.gsq_backward_update_noalloc(_args(g, w, W, G, st, loss_na, t, tau, 1.0, d_dtype), stream)
        torch.cuda.synchronize()
        for k in kinds:
            ref = layer.get_tensor(k, torch.float32)
            assert torch.equal(st[k], ref), (t, k, float((st[k] - ref).abs().max()))
        lr, ln = loss_ref.item(), loss_na.item()
        assert np.isfinite(ln) and abs(ln - lr) <= TOL_F32 * abs(lr), (t, ln, lr)
    layer.close()


def test_noalloc_rejects_layers_beyond_its_scratch():
    g = gsq()
    a = g.gsq_backward_args()
    a.num_experts, a.out_features, a.in_features = 1, 4097, 4096   # one row past 2^24 weights
    a.num_levels, a.group_size = 4, 128
    for k, q in enumerate((-1.5, -0.5, 0.5, 1.5)):
        a.grid[k] = q
    a.tau, a.kappa = 1.0, 1.0
    with pytest.raises(g.GsqError) as ei:
        g.gsq_backward_update_noalloc(a, 0)
    assert ei.value.status == g.GSQ_ERR_SHAPE
    assert "16777216" in g.gsq_last_error()
