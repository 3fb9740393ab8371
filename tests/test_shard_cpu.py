"""The multi-GPU partition of one layer on CPU: row blocks of a one-expert layer
or whole experts of a multi-expert layer (configs.shard), two gloo ranks each
following its shard with the oracle.  Rows are independent in Eq. 1 with a
linear f, so the shards' noise must be the whole layer's for the same weights
(keyed on the global flat index), their states the whole layer's rows, and
their losses, summed by one all-reduce, the whole layer's loss."""
import os
import socket
import sys

import numpy as np
import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
STEPS = 2


def _cases():
    sys.path.insert(0, ROOT)
    from paper_2604_18556_gb300 import configs as C
    W = C.WORKLOADS
    return {"rows": C.shrunk(W["llama8b_q_proj"], rows=22, cols=256, tokens=512),
            "experts": C.shrunk(W["moe64_kquant3"], experts=3, rows=6, cols=256, tokens=256)}


def _problem(w, H):
    from oracle import gsq_oracle as O
    return O.Problem(E=w.experts, R=w.rows, C=w.cols, grid=np.asarray(w.grid, float),
                     group=w.group, seed=w.seed, scale_mode=w.scale_mode, H=H,
                     lr_logits=w.lr_logits, lr_scales=w.lr_scales, beta1=w.beta1,
                     beta2=w.beta2, wd_logits=w.wd_logits, wd_scales=w.wd_scales)


def _follow(w, rows_ids, Wrows, H):
    """The oracle on the given global rows for STEPS steps: (noise of step 0,
    per-step losses, final logits, final scales)."""
    from oracle import gsq_oracle as O
    prob = _problem(w, H)
    st = O.init_state(prob, Wrows, rows_ids, init_bias=w.init_bias)
    g0 = O.noise(prob, st, 0)
    losses = []
    for t in range(STEPS):
        losses.append(O.step(prob, st, t, w.tau(t), w.kappa).loss)
    return g0, np.array(losses), st.logits, st.scales


def _global_rows(w, sh):
    (e0, e1), (r0, r1) = sh.experts, sh.rows
    return np.array([e * w.rows + r for e in range(e0, e1) for r in range(r0, r1)], np.int64)


def _worker(rank, world, port, name, out):
    sys.path.insert(0, ROOT)
    import torch
    import torch.distributed as dist
    from oracle import gsq_oracle as O
    from paper_2604_18556_gb300 import configs as C
    from paper_2604_18556_gb300 import inputs
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        w = _cases()[name]
        sh = C.shard(w, rank, world)
        ids = _global_rows(w, sh)
        H = inputs.make_gram(w).double().numpy()        # every rank holds H (replicated)
        Ws = inputs.make_weight(w, experts=sh.experts, rows=sh.rows).float().numpy()
        prob = _problem(w, H)
        # the shard's first flat index is its index offset
        assert O.flat_index(prob, ids)[0, 0] == sh.index_offset
        g0, losses, logits, scales = _follow(w, ids, Ws.reshape(-1, w.cols), H)
        t = torch.tensor(losses, dtype=torch.float64)
        dist.all_reduce(t)                               # the loss all-reduce of the partition
        out[rank] = (ids, g0, t.numpy(), logits, scales)
    finally:
        dist.destroy_process_group()


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


@pytest.mark.parametrize("name", ["rows", "experts"])
def test_two_gloo_rank_shards_reproduce_the_whole_layer(name):
    sys.path.insert(0, ROOT)
    from paper_2604_18556_gb300 import inputs
    world = 2
    with mp.Manager() as mgr:
        out = mgr.dict()
        mp.start_processes(_worker, args=(world, _free_port(), name, out), nprocs=world,
                           start_method="spawn")
        res = dict(out)
    w = _cases()[name]
    H = inputs.make_gram(w).double().numpy()
    Wall = inputs.make_weight(w).float().numpy().reshape(-1, w.cols)
    ids = np.arange(w.experts * w.rows)
    g0, losses, logits, scales = _follow(w, ids, Wall, H)
    got_ids = np.concatenate([res[r][0] for r in range(world)])
    assert np.array_equal(got_ids, ids)                  # the blocks cover every row once
    # noise keyed on the global index: identical draws
    assert np.array_equal(np.concatenate([res[r][1] for r in range(world)], axis=1), g0)
    for r in range(world):                               # the all-reduced loss is the layer's
        assert np.allclose(res[r][2], losses, rtol=1e-12, atol=0)
    # rows are independent: the same state up to float64 summation order
    assert np.max(np.abs(np.concatenate([res[r][3] for r in range(world)], axis=1) - logits)) <= 1e-6
    assert np.max(np.abs(np.concatenate([res[r][4] for r in range(world)]) - scales)) <= 1e-7


def test_shard_offsets_are_the_global_flat_index():
    """configs.shard: the blocks cover the layer once, in order, and each index
    offset is the flat index (e*R + r)*C of the shard's first weight."""
    sys.path.insert(0, ROOT)
    from paper_2604_18556_gb300 import configs as C
    W = C.WORKLOADS
    for w in (W["llama8b_q_proj"], W["moe64_kquant3"], W["llama70b_gate_proj"]):
        for world in (1, 2, 3, 8):
            seen = 0
            for rank in range(world):
                sh = C.shard(w, rank, world)
                (e0, e1), (r0, r1) = sh.experts, sh.rows
                assert sh.index_offset == (e0 * w.rows + r0) * w.cols
                assert sh.workload.n == (e1 - e0) * (r1 - r0) * w.cols
                assert sh.index_offset == seen
                seen += sh.workload.n
            assert seen == w.n
    with pytest.raises(ValueError):
        C.shard(C.shrunk(W["moe64_kquant3"], experts=2), 0, 4)   # fewer experts than ranks
