"""Shards of one layer, stepped one after another on one GPU.

Rows are independent in Eq. 1 with a linear f (the loss is a sum over rows,
L = sum_r D_r H D_r^T; dL/dW^ of row r needs only row r and H; Lion acts
elementwise), and the noise is keyed on the whole layer's flat weight index, so
a layer split into row blocks (one-expert layers) or whole experts (the MoE
batch), each shard built from its slice of W, a copy of H and its index offset,
must step every weight exactly as the whole layer does: state bit for bit, the
look-ahead D bit for bit, codes and packed bytes bit for bit, and the shards'
losses summing to the layer's (only the reduction order differs)."""
import numpy as np
import pytest
import torch

from gpu_common import gsq
from paper_2604_18556_gb300 import configs as C
from paper_2604_18556_gb300 import inputs

pytestmark = pytest.mark.gpu

W_ = C.WORKLOADS
CASES = {
    # 520 rows: the whole layer runs the staged backward, its shards the direct one
    "rows_full": C.shrunk(W_["llama8b_q_proj"], rows=520, cols=1024, tokens=2048),
    "rows_mask_sign": C.shrunk(W_["llama8b_q_proj_mask_sign"], rows=264, cols=512, tokens=2048),
    "rows_shift5": C.shrunk(W_["llama8b_down_proj_shift5"], rows=136, cols=1024, tokens=2048),
    "experts_kquant": C.shrunk(W_["moe64_kquant3"], experts=5, rows=64, cols=512, tokens=1024),
}
STEPS = 3


def _layer(g, w, W, H, gemm, index_offset=0):
    return g.Layer(W, H, w.grid, w.group, scale_mode=w.scale_mode, gemm=gemm, param=w.param,
                   init_bias=w.init_bias, seed=w.seed, lr_logits=w.lr_logits,
                   lr_scales=w.lr_scales, beta1=w.beta1, beta2=w.beta2, wd_logits=w.wd_logits,
                   wd_scales=w.wd_scales, index_offset=index_offset)


def _run(layer, w):
    """STEPS updating steps with look-ahead (the benchmark's sequence); the losses."""
    losses = []
    for t in range(STEPS):
        loss = torch.zeros(1, device="cuda")
        layer.step(t, w.tau(t), w.kappa, next_tau=w.tau(t + 1), next_kappa=w.kappa, loss=loss)
        losses.append(loss)
    layer.sync_status()
    return [float(x.item()) for x in losses]


def _state(g, layer, w, E, R):
    """State tensors as [planes][E][R][C] / [E][R][...] views (CPU)."""
    C_, L = w.cols, w.L
    f32 = lambda k: layer.get_tensor(k, torch.float32).cpu()
    out = {"logits": f32(g.GSQ_T_LOGITS).view(L, E, R, C_),
           "m_logits": f32(g.GSQ_T_MOM_LOGITS).view(L, E, R, C_),
           "scales": f32(g.GSQ_T_SCALES).view(E, R, -1),
           "m_scales": f32(g.GSQ_T_MOM_SCALES).view(E, R, -1)}
    d = layer.get_tensor(g.GSQ_T_D).cpu()
    out["D"] = d.view(E, R, -1)
    n = E * R * C_
    codes = torch.empty(n, dtype=torch.uint8, device="cuda")
    layer.project(codes)
    out["codes"] = codes.cpu().view(E, R, C_)
    return out


@pytest.mark.parametrize("world", [2, 3])
@pytest.mark.parametrize("gemm", ["bf16", "f32"])
@pytest.mark.parametrize("name", list(CASES))
def test_shards_step_exactly_as_the_whole_layer(name, gemm, world):
    g = gsq()
    w = CASES[name]
    W = inputs.make_weight(w, device="cuda")
    H = inputs.make_gram(w, device="cuda")
    whole = _layer(g, w, W, H, gemm)
    loss_whole = _run(whole, w)
    ref = _state(g, whole, w, w.experts, w.rows)
    packed_whole = None
    if w.scale_mode == "kquant2":
        packed_whole = torch.empty(whole.packed_size(), dtype=torch.uint8, device="cuda")
        whole.pack(packed_whole)
        packed_whole = packed_whole.cpu()
    whole.close()

    loss_sum = np.zeros(STEPS)
    packed_parts = []
    for rank in range(world):
        sh = C.shard(w, rank, world)
        (e0, e1), (r0, r1) = sh.experts, sh.rows
        Ws = inputs.make_weight(w, device="cuda", experts=sh.experts, rows=sh.rows)
        assert torch.equal(Ws, W[e0:e1, r0:r1])          # the shard's slice of the whole W
        Hs = inputs.make_gram(w, device="cuda", experts=sh.experts)
        part = _layer(g, sh.workload, Ws, Hs, gemm, sh.index_offset)
        loss_sum += np.array(_run(part, sh.workload))
        got = _state(g, part, sh.workload, e1 - e0, r1 - r0)
        for key, t in got.items():
            want = ref[key][:, e0:e1, r0:r1] if key in ("logits", "m_logits") else \
                ref[key][e0:e1, r0:r1]
            assert torch.equal(t, want), (name, gemm, rank, key)
        if packed_whole is not None:
            buf = torch.empty(part.packed_size(), dtype=torch.uint8, device="cuda")
            part.pack(buf)
            packed_parts.append(buf.cpu())
        part.close()
    # the shards' losses add up to the layer's: the same double partial sums in
    # another grouping, each total rounded once to fp32
    lw = np.array(loss_whole)
    assert np.all(np.abs(loss_sum - lw) <= 4e-7 * np.abs(lw) * world), (loss_sum, lw)
    if packed_whole is not None:   # K-Quant records are per 256 weights: shards concatenate
        assert torch.equal(torch.cat(packed_parts), packed_whole)

