"""Steps replayed from a captured CUDA graph against the same steps launched eagerly.

The step's tensor-core GEMMs and backward kernels are launched as programmatic
dependents of the kernel before them (each waits with griddepcontrol before its
first global access), and a captured graph keeps those launches as programmatic
edges.  Whether the kernels are launched that way or plainly (GSQ_PDL=0), eagerly or
from a graph, with or without the library's profiling event records between them,
they run the same arithmetic on the same inputs: every updated tensor and the
look-ahead D must agree bit for bit, and the loss to 1e-6 (a reduction over the
grid).  Covered: the staged backward after the CTA-pair GEMM and after clusters of
pairs, the direct-load backward (local shift), the first step's forward inside the
graph, and the token step, whose contraction is two GEMMs back to back."""
import dataclasses

import numpy as np
import pytest
import torch

from gpu_common import Case, gsq
from paper_2604_18556_gb300 import configs as C
from paper_2604_18556_gb300 import inputs

pytestmark = pytest.mark.gpu

W = C.WORKLOADS
CASES = {
    # staged backward (more tiles than resident blocks), 256-row pair tiles with a ragged last one
    "staged_pairs": (C.shrunk(W["llama8b_q_proj"], rows=999, cols=1280, tokens=2048), "1"),
    "staged_clusters": (C.shrunk(W["llama8b_q_proj"], rows=999, cols=1280, tokens=2048), "2"),
    # 5 logits per weight: the direct-load backward
    "shift5_direct": (C.shrunk(W["llama8b_down_proj_shift5"], rows=300, cols=1536, tokens=2048),
                      "auto"),
}
STEPS = 4
TAU = 0.7


def _randomise(case):
    rng = np.random.default_rng(31)
    L = (1.5 * rng.standard_normal(case.logits().shape)).astype(np.float32)
    case.layer.set_tensor(gsq().GSQ_T_LOGITS, torch.from_numpy(L).cuda())


def _state(case, d_dtype):
    g = gsq()
    out = [case.tensor(w, torch.float32).view(torch.int32).clone()
           for w in (g.GSQ_T_LOGITS, g.GSQ_T_MOM_LOGITS, g.GSQ_T_SCALES, g.GSQ_T_MOM_SCALES)]
    out.append(case.tensor(g.GSQ_T_D, d_dtype).view(torch.int16).clone())
    return out


def _steps(case, loss):
    for t in range(STEPS):
        case.layer.step(t, TAU, 1.0, next_tau=TAU, next_kappa=1.0, loss=loss)


def _new_case(w, pair, pdl, monkeypatch):
    if pair != "auto":
        monkeypatch.setenv("GSQ_GEMM_PAIR", pair)
    if pdl:
        monkeypatch.delenv("GSQ_PDL", raising=False)
    else:
        monkeypatch.setenv("GSQ_PDL", "0")
    case = Case(w, gemm="bf16")       # GSQ_PDL and GSQ_GEMM_PAIR are read when the layer is made
    _randomise(case)
    return case


@pytest.mark.parametrize("events", [False, True], ids=["plain_graph", "graph_with_events"])
@pytest.mark.parametrize("name", list(CASES))
def test_graph_replay_matches_eager_steps(name, events, monkeypatch):
    w, pair = CASES[name]
    eager = _new_case(w, pair, pdl=False, monkeypatch=monkeypatch)
    graphed = _new_case(w, pair, pdl=True, monkeypatch=monkeypatch)
    assert eager.layer.kernel_name(gsq().GSQ_K_BACKWARD) == graphed.layer.kernel_name(
        gsq().GSQ_K_BACKWARD)

    loss_e = torch.zeros(1, device="cuda")
    _steps(eager, loss_e)
    torch.cuda.synchronize()
    eager.layer.sync_status()

    loss_g = torch.zeros(1, device="cuda")
    graphed.layer.profile_enable(events)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        _steps(graphed, loss_g)
    before = _state(graphed, torch.bfloat16)
    graph.replay()
    torch.cuda.synchronize()
    graphed.layer.sync_status()
    graphed.layer.profile_enable(False)

    after = _state(graphed, torch.bfloat16)
    assert not torch.equal(before[0], after[0]), "the replay did not update the logits"
    for a, b, what in zip(_state(eager, torch.bfloat16), after,
                          ("logits", "logit momenta", "scales", "scale momenta", "look-ahead D")):
        assert torch.equal(a, b), what
    assert abs(loss_g.item() - loss_e.item()) <= 1e-6 * abs(loss_e.item())


def test_token_step_graph_matches_eager(monkeypatch):
    """One token step (three micro-batches: two exporting passes, then the update) captured
    in a graph, against the same step launched eagerly without programmatic dependents."""
    w = dataclasses.replace(C.shrunk(W["llama8b_q_proj_tokens"], rows=600, cols=384, tokens=328),
                            micro=3)
    Xs = [inputs.make_token_batch(w, 0, j, device="cuda") for j in range(w.micro)]

    def run(case, losses):
        for j, X in enumerate(Xs):
            case.layer.step_tokens(0, j, w.micro, w.tau(0), X, next_tau=w.tau(1),
                                   loss=losses[j:j + 1])

    eager = _new_case(w, "auto", pdl=False, monkeypatch=monkeypatch)
    graphed = _new_case(w, "auto", pdl=True, monkeypatch=monkeypatch)
    le = torch.zeros(w.micro, device="cuda")
    run(eager, le)
    torch.cuda.synchronize()
    eager.layer.sync_status()

    lg = torch.zeros(w.micro, device="cuda")
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        run(graphed, lg)
    graph.replay()
    torch.cuda.synchronize()
    graphed.layer.sync_status()

    for a, b, what in zip(_state(eager, torch.bfloat16), _state(graphed, torch.bfloat16),
                          ("logits", "logit momenta", "scales", "scale momenta", "look-ahead D")):
        assert torch.equal(a, b), what
    assert torch.allclose(lg, le, rtol=1e-6, atol=0.0), (lg, le)
