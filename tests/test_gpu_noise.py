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


def _layer(grid, param, rows=R, index_offset=0):
    g = gsq()
    torch.manual_seed(3)
    W = (0.02 * torch.randn(1, rows, C, device="cuda")).bfloat16()
    H = torch.zeros(1, C, C, device="cuda")
    layer = g.Layer(W, H, grid, 128, gemm="bf16", param=param, seed=SEED,
                    index_offset=index_offset)
    layer.set_tensor(g.GSQ_T_SCALES, torch.ones(rows * C // 128, device="cuda"))
    return layer


def _soft_values(layer, t, rows=R):
    what = torch.empty(rows * C, device="cuda")
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


ROWS_OFF = 256                     # 1,048,576 weights per shard
N_OFF = ROWS_OFF * C


@pytest.mark.parametrize("index_offset", [(1 << 32) + 5 * N_OFF, (1 << 32) - N_OFF // 2 - 4096,
                                          (3 << 32) - 12 * C])
def test_largest_gumbel_draw_of_a_shard_far_into_the_counter_space(index_offset):
    """A shard whose flat indices have a nonzero high word, and shards whose indices
    cross a multiple of 2^32 (the counter's high word changes inside the launch):
    every weight's draw must still be the oracle's for its whole-layer index."""
    K = 8
    t = 4242
    layer = _layer(tuple(float(k) for k in range(K)), "full", rows=ROWS_OFF,
                   index_offset=index_offset)
    v = _soft_values(layer, t, rows=ROWS_OFF)
    layer.close()
    code = np.rint(v)
    ok = np.abs(v - code) < 1e-6
    idx = np.uint64(index_offset) + np.arange(N_OFF, dtype=np.uint64)
    j = (P.level_words(SEED, t, idx, K) & np.uint32(0x7FFFFF)).astype(np.int64)
    top = j.max(axis=0)
    expect = j.argmax(axis=0)
    tie = (j == top[None]).sum(axis=0) > 1
    keep = ok & ~tie
    assert np.array_equal(code[keep].astype(np.int64), expect[keep]), \
        int(np.sum(code[keep].astype(np.int64) != expect[keep]))
    assert (~keep).mean() < 1e-3, (~keep).mean()
