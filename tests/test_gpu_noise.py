"""The GPU's counter-based noise against the oracle's Philox words on many counters:
which draw is largest, and the sign of every logistic draw, weight by weight.

With kappa = 0 the logits drop out of the relaxation, and at tau = 1e-6 the soft
value is the grid level of the largest draw (Alg. 1 in its zero-temperature limit;
the binary mask x sign instances become the signs of their logistic draws, Alg. 2).
The Gumbel transform -ln(-ln u) is increasing in u, so the largest draw is the
level whose Philox word has the largest low 23 bits, and the sign of a logistic
draw ln(u / (1 - u)) is whether those bits reach 2^22.  The oracle side is
therefore integer work on the Philox4x32-10 words (oracle/philox.py); the GPU side
is the forward kernel's exported soft weight.  Weights whose top two draws are too
close for the fp32 softmax to saturate at this tau (or tie exactly) give a value
between levels; they are left out and must be rare."""
import numpy as np
import pytest
import torch

from gpu_common import gsq
from oracle import philox as P

pytestmark = pytest.mark.gpu

R, C = 2048, 4096            # 8,388,608 weights
SEED = 0x0123456789ABCDEF    # both key words nonzero
TAU = 1e-6


def _layer(grid, param):
    g = gsq()
    torch.manual_seed(3)
    W = (0.02 * torch.randn(1, R, C, device="cuda")).bfloat16()
    H = torch.zeros(1, C, C, device="cuda")
    layer = g.Layer(W, H, grid, 128, gemm="bf16", param=param, seed=SEED)
    layer.set_tensor(g.GSQ_T_SCALES, torch.ones(R * C // 128, device="cuda"))
    return layer


def _soft_values(layer, t):
    what = torch.empty(R * C, device="cuda")
    layer.forward(t, TAU, 0.0, what=what)
    torch.cuda.synchronize()
    return what.cpu().numpy().astype(np.float64)


@pytest.mark.parametrize("t", [0, 12345])
def test_largest_gumbel_draw_matches_the_oracle_words(t):
    """8 levels x 8.4 M weights = 67 M draws per step counter."""
    K = 8
    layer = _layer(tuple(float(k) for k in range(K)), "full")
    v = _soft_values(layer, t)
    layer.close()
    code = np.rint(v)
    ok = np.abs(v - code) < 1e-6
    idx = np.arange(R * C, dtype=np.uint64)
    j = (P.level_words(SEED, t, idx, K) & np.uint32(0x7FFFFF)).astype(np.int64)   # [K, n]
    top = j.max(axis=0)
    expect = j.argmax(axis=0)
    # an exact tie of the top two draws gives the mean of their levels, which is a
    # level itself when they are an even number of levels apart: left out
    tie = (j == top[None]).sum(axis=0) > 1
    keep = ok & ~tie
    assert np.array_equal(code[keep].astype(np.int64), expect[keep]), \
        int(np.sum(code[keep].astype(np.int64) != expect[keep]))
    assert (~keep).mean() < 1e-3, (~keep).mean()


@pytest.mark.parametrize("t", [0, 777])
def test_logistic_draw_signs_match_the_oracle_words(t):
    """Two binary instances x 8.4 M weights = 16.8 M logistic draws per step counter."""
    layer = _layer((-1.0, 0.0, 1.0), "mask_sign")
    v = _soft_values(layer, t)
    layer.close()
    code = np.rint(v)
    ok = np.abs(v - code) < 1e-6
    idx = np.arange(R * C, dtype=np.uint64)
    words = P.pair_words(SEED, t, idx)                       # [2 (mask, sign), n]
    pos = (words & np.uint32(0x7FFFFF)) >= (1 << 22)         # u > 1/2, i.e. the draw > 0
    expect = pos[0].astype(np.int64) * np.where(pos[1], 1, -1)
    assert np.array_equal(code[ok].astype(np.int64), expect[ok]), \
        int(np.sum(code[ok].astype(np.int64) != expect[ok]))
    assert (~ok).mean() < 1e-3, (~ok).mean()
