"""Benchmark of the GSQ relaxed-scalar-quantizer step on one GB300 (per rank).

One step = one gsq_step: (look-ahead forward from the previous step) + the
tensor-core loss GEMM + the fused backward/Lion/next-forward kernel, on the
Llama-3.1-8B q_proj-shaped layer (4096 x 4096 bf16, 2-bit grid, group 128,
tau annealed 1.0 -> 0.1 over 500 steps).  Prints one JSON line.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl gsq|reference]
                  [--workload NAME]

--impl reference times the CPU oracle (the plain float64 restatement of the
method) on a row sample of the same layer; rows are independent, so the full
layer's step time is the sample's time scaled by R / rows.  Under torchrun,
every rank runs its own independent layer (weak scaling, no collective on the
data path); rank 0 prints the whole-job throughput.
"""
from __future__ import annotations

import argparse
import json
import os
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "GSQ steps/s per 8B-shaped layer"
UNIT = "steps/s"


def _args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="gsq", choices=["gsq", "reference"])
    ap.add_argument("--workload", default="llama8b_q_proj")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-graph", action="store_true",
                    help="time eager launches instead of one CUDA-graph replay of the timed steps")
    ap.add_argument("--cpu-sample-seconds", type=float, default=15.0)
    ap.add_argument("--unstaged", action="store_true",
                    help="time the backward with direct global loads (GSQ_FLAG_UNSTAGED)")
    return ap.parse_args()


def _dist():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


TRAFFIC_FILE = os.path.join(ROOT, "profiles", "dram_traffic.json")
CSRC = os.path.join(ROOT, "paper_2604_18556_gb300", "csrc")
# the source files each profiled kernel is compiled from
KERNEL_SOURCES = {
    "k_backward": ["gsq_backward.cu", "gsq_staged.cu", "gsq_backward.cuh", "gsq_relax.cuh",
                   "gsq_tc.cuh", "gsq_internal.h"],
}


def source_sha256(kernel: str = "k_backward") -> str:
    import hashlib
    h = hashlib.sha256()
    for name in KERNEL_SOURCES[kernel]:
        with open(os.path.join(CSRC, name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()


def committed_traffic(workload: str, kernel: str = "k_backward"):
    """DRAM bytes (read + write) per launch of `kernel` from the committed ncu
    capture, or None when there is none for this workload or the kernel's
    sources have changed since it was taken."""
    if not os.path.exists(TRAFFIC_FILE):
        return None
    with open(TRAFFIC_FILE) as f:
        d = json.load(f).get("kernels", {}).get(kernel)
    if not d or d.get("source_sha256") != source_sha256(kernel):
        return None
    return d.get("workloads", {}).get(workload, {}).get("dram_bytes_per_launch")


def rank_workload(w, rank: int, world: int):
    """Each rank quantizes its own independent layer of the same shape (weak
    scaling: rows and experts never exchange data, so ranks share nothing)."""
    if world <= 1:
        return w
    import dataclasses
    return dataclasses.replace(w, seed=w.seed + rank, data_seed=w.data_seed + 100 * rank)


def max_over_ranks(x: float, device) -> float:
    """Largest value over the process group (the slowest rank defines the time)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_steps_per_s(ms_per_step: float, world: int) -> float:
    """All ranks' steps per second: world layers advance one step every ms_per_step."""
    return world * 1000.0 / ms_per_step


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d.get("hbm_gbs", 6800.0), d.get("bf16_tflops", 1900.0), d.get(
            "bf16_tflops_sustained", 1700.0), "measured"
    return 6800.0, 1900.0, 1700.0, "fallback"


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms during the timed region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.dev = device_index
        self.lines = []
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200", "-i", str(self.dev)], stdout=subprocess.PIPE,
                stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except (OSError, ValueError):
            self.proc = None

    def _read(self):
        for ln in self.proc.stdout:
            self.lines.append(ln.strip())

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=2)
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
        sm.sort()
        return {"sm_mhz": sm[len(sm) // 2], "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm)}


def _workload(name):
    from paper_2604_18556_gb300 import configs as C
    return C.WORKLOADS[name]


def _config(w, extra=None):
    cfg = {"workload": f"{w.name}: E={w.experts} R={w.rows} C={w.cols} K={w.K} G={w.group} "
                       f"W={w.w_dtype} scales={w.scale_mode} logits/weight={w.L}",
           "tau": f"{w.tau0}->{w.tau1} over {w.steps} steps", "kappa": w.kappa,
           "gemm": "tcgen05 bf16 x bf16 -> fp32",
           "l2": "working set larger than L2 (logits + momenta = "
                 f"{8 * w.L * w.n / 2**20:.0f} MiB vs 126 MiB L2)"}
    if extra:
        cfg.update(extra)
    return cfg


# ----------------------------------------------------------------------------
# CPU oracle on a row sample (baseline / reference arm)
# ----------------------------------------------------------------------------
def _oracle_problem(w, H_host, rows):
    import numpy as np
    from oracle import gsq_oracle as O
    prob = O.Problem(E=w.experts, R=w.rows, C=w.cols, grid=np.asarray(w.grid, float), group=w.group,
                     seed=w.seed, scale_mode=w.scale_mode, H=H_host, lr_logits=w.lr_logits,
                     lr_scales=w.lr_scales, beta1=w.beta1, beta2=w.beta2, wd_logits=w.wd_logits,
                     wd_scales=w.wd_scales, shift=w.param == "shift5",
                     mask_sign=w.param == "mask_sign")
    return prob


def _cpu_inputs(w, rows):
    """The workload's W rows and H (expert 0) from the seeded generators (on the
    GPU when one is present: input preparation only, not the timed oracle)."""
    import torch
    from paper_2604_18556_gb300 import configs as C
    from paper_2604_18556_gb300 import inputs
    w1 = C.shrunk(w, experts=1)
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    if dev == "cpu":
        torch.set_num_threads(max(1, os.cpu_count() or 1))
    Wt = inputs.make_weight(w1, device=dev)[0, :rows].float().cpu().numpy()
    H = inputs.make_gram(w1, device=dev)[0].double().cpu().numpy()
    return Wt, H


def _oracle_rows_for(seconds_per_step, t_one_row):
    return max(1, int(seconds_per_step / max(t_one_row, 1e-6)))


def _single_thread_env():
    for v in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        os.environ[v] = "1"


def run_oracle_sample(w, step_budget_s: float, n_steps: int, n_warm: int, Wt=None, H=None):
    """Times the oracle's full step on a row sample.  Returns (seconds per step of
    the full layer, rows sampled, seconds measured)."""
    import numpy as np
    from oracle import gsq_oracle as O
    if Wt is None:
        Wt, H = _cpu_inputs(w, min(w.rows, 256))
    prob = _oracle_problem(w, H[None] if H.ndim == 2 else H, None)
    # size the sample from a probe of 16 rows (after one untimed call)
    probe = min(16, Wt.shape[0])
    st = O.init_state(prob, Wt[:probe], np.arange(probe), init_bias=w.init_bias)
    O.step(prob, st.copy(), 0, w.tau(0), w.kappa)
    t0 = time.perf_counter()
    O.step(prob, st, 0, w.tau(0), w.kappa)
    t_row = (time.perf_counter() - t0) / probe
    rows = min(Wt.shape[0], _oracle_rows_for(step_budget_s, t_row))
    st = O.init_state(prob, Wt[:rows], np.arange(rows), init_bias=w.init_bias)
    for t in range(n_warm):
        O.step(prob, st, t, w.tau(t), w.kappa)
    times = []
    for t in range(n_warm, n_warm + n_steps):
        t0 = time.perf_counter()
        O.step(prob, st, t, w.tau(t), w.kappa)
        times.append(time.perf_counter() - t0)
    per = float(np.median(times))
    return per * (w.experts * w.rows) / rows, rows, float(sum(times))


def run_oracle_tokens_sample(w, n_steps: int, rows: int = 256, tok=(512, 4096)):
    """Oracle step on per-step token batches, sampled in rows and tokens.  The
    micro-batch cost is linear in its tokens (the loss contractions) plus a part
    that is not (noise, softmax, backward, Lion): both are fitted from one
    micro-batch of tok[0] and of tok[1] tokens on `rows` rows, then scaled to the
    workload's tokens per micro-batch, micro-batches and rows.  Returns (seconds
    per full step, description of the sample, seconds measured)."""
    import dataclasses
    import numpy as np
    import torch
    from oracle import gsq_oracle as O
    from paper_2604_18556_gb300 import configs as C
    from paper_2604_18556_gb300 import inputs
    w1 = C.shrunk(w, experts=1)
    Wt = inputs.make_weight(w1)[0, :rows].float().numpy()
    prob = _oracle_problem(w1, None, None)
    per_tok = []
    measured = 0.0
    for T in tok:
        wt = dataclasses.replace(w1, tokens=T, micro=1)
        X = inputs.make_token_batch(wt, 0, 0).double().numpy()
        times = []
        for t in range(n_steps + 1):
            st = O.init_state(prob, Wt, np.arange(rows), init_bias=w.init_bias)
            t0 = time.perf_counter()
            O.step_microbatches(prob, st, t, [X], w.tau(t), w.kappa)
            times.append(time.perf_counter() - t0)
        measured += sum(times)
        per_tok.append(float(np.median(times[1:])))
    b = (per_tok[1] - per_tok[0]) / (tok[1] - tok[0])
    a = max(per_tok[0] - b * tok[0], 0.0)
    full = (a + b * w.tokens) * w.micro * (w.experts * w.rows) / rows
    desc = (f"{rows} rows x one micro-batch of {tok[0]} and of {tok[1]} tokens, {n_steps} timed "
            f"steps each ({measured:.1f} s measured); cost fitted as a + b*tokens and scaled to "
            f"{w.tokens} tokens x {w.micro} micro-batches x {w.experts * w.rows} rows")
    return full, desc, measured


def reference_arm(args, rank, world):
    if rank != 0:
        return 0
    _single_thread_env()
    w = _workload(args.workload)
    if w.calib == "batches":
        full_step_s, desc, _ = run_oracle_tokens_sample(w, max(args.steps, 1))
        value = 1.0 / full_step_s
        print(json.dumps({
            "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": full_step_s * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": _config(w, {"oracle": "numpy float64, one thread"}),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle",
                             "sample": desc},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        }), flush=True)
        return 0
    per_step_budget = 1.0
    full_step_s, rows, measured = run_oracle_sample(w, per_step_budget, args.steps, args.warmup)
    value = 1.0 / full_step_s
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": full_step_s * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": _config(w, {"oracle": "numpy float64, one thread"}),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle",
                         "sample": f"{rows} of {w.experts * w.rows} rows per step (rows are "
                                   f"independent; full-layer time = sample time x {w.rows}/{rows}); "
                                   f"{measured:.1f} s measured"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ----------------------------------------------------------------------------
# GPU arm
# ----------------------------------------------------------------------------
def gpu_arm(args, rank, world, local):
    import numpy as np
    import torch
    import torch.distributed as dist

    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    from paper_2604_18556_gb300 import build
    build.build()
    from paper_2604_18556_gb300 import gsq, inputs
    from paper_2604_18556_gb300 import configs as C

    w = rank_workload(_workload(args.workload), rank, world)
    W = inputs.make_weight(w, device="cuda")
    H = inputs.make_gram(w, device="cuda")
    H_host = H[0].double().cpu().numpy() if world == 1 and not args.no_cpu_baseline else None
    layer = gsq.Layer(W, H, w.grid, w.group, calib_kind="H", scale_mode=w.scale_mode, gemm="bf16",
                      init_bias=w.init_bias, seed=w.seed, lr_logits=w.lr_logits,
                      lr_scales=w.lr_scales, beta1=w.beta1, beta2=w.beta2,
                      wd_logits=w.wd_logits, wd_scales=w.wd_scales, param=w.param,
                      unstaged=args.unstaged)
    stream = torch.cuda.current_stream()
    loss = torch.zeros(1, device="cuda")
    T = w.steps

    def sched(t):
        return w.tau(t % T)

    t = 0
    for _ in range(args.warmup):
        layer.step(t, sched(t), w.kappa, next_tau=sched(t + 1), next_kappa=w.kappa, loss=loss)
        t += 1
    layer.sync_status()
    torch.cuda.synchronize()

    # The timed steps run as one CUDA graph (captured here, untimed): K distinct
    # steps t0..t0+K-1, so the replay does exactly the work of K eager steps
    # without the host launch gaps.  The library's profiling events are captured
    # as event-record nodes and time the kernels of the replay.
    graph = None
    if not args.no_graph:
        layer.profile_enable(True)
        layer.profile_read()
        graph = torch.cuda.CUDAGraph()
        t_cap = t
        with torch.cuda.graph(graph):
            for i in range(args.steps):
                layer.step(t_cap + i, sched(t_cap + i), w.kappa, next_tau=sched(t_cap + i + 1),
                           next_kappa=w.kappa, loss=loss)
        t += args.steps
        graph.replay()      # first replay (graph upload), untimed
        torch.cuda.synchronize()
    sampler = ClockSampler(local)
    sampler.start()
    time.sleep(0.3)
    if graph is None:
        layer.profile_enable(True)
        layer.profile_read()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    if graph is not None:
        graph.replay()
    else:
        for _ in range(args.steps):
            layer.step(t, sched(t), w.kappa, next_tau=sched(t + 1), next_kappa=w.kappa, loss=loss)
            t += 1
    e1.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clocks = sampler.stop()
    ms_total = e0.elapsed_time(e1)
    prof = layer.profile_read()
    layer.profile_enable(False)
    layer.sync_status()
    ms_total = max_over_ranks(ms_total, torch.device("cuda", local))
    ms_step = ms_total / args.steps
    value = whole_job_steps_per_s(ms_step, world)

    hbm, tf_burst, tf_sust, peak_src = _peaks()
    n = w.n
    bwd_n, bwd_ms = prof["backward"]
    gemm_n, gemm_ms = prof["gemm"]
    fwd_n, fwd_ms = prof["forward"]
    flops = w.gemm_flops_per_step()
    bwd_avg = bwd_ms / max(bwd_n, 1)
    gemm_avg = gemm_ms / max(gemm_n, 1)
    bytes_bwd = w.elementwise_bytes_per_weight() * n
    bwd_gbs = bytes_bwd / (bwd_avg * 1e-3) / 1e9
    gemm_tfs = flops / (gemm_avg * 1e-3) / 1e12
    kname = layer.kernel_name(gsq.GSQ_K_BACKWARD)
    roofline = {"kernel": f"{kname} (fused backward + Lion + next forward)", "bound": "hbm",
                "achieved": bwd_gbs, "peak": hbm, "unit": "GB/s", "frac": bwd_gbs / hbm,
                "traffic": committed_traffic(w.name),
                "peak_source": f"{peak_src} (MEASURED_PEAKS.json hbm_gbs)",
                "algorithmic_bytes_per_launch": bytes_bwd, "avg_launch_ms": bwd_avg,
                "frac_of_8TBps": bwd_gbs / 8000.0}
    roofline_gemm = {"kernel": f"{layer.kernel_name(gsq.GSQ_K_GEMM)} (tcgen05 loss contraction)",
                     "bound": "tensor",
                     "achieved": gemm_tfs, "peak": tf_sust, "unit": "TFLOP/s",
                     "frac": gemm_tfs / tf_sust, "frac_of_burst": gemm_tfs / tf_burst,
                     "flops_per_launch": flops, "avg_launch_ms": gemm_avg,
                     "peak_source": f"{peak_src} bf16_tflops_sustained"}
    launches = bwd_n + gemm_n + fwd_n

    # method diagnostics of the state after the timed steps (not timed)
    diag = layer.diagnose(sched(t), w.kappa)
    diag["after_step"] = t
    e2e = None
    if not args.no_e2e:
        e2e = e2e_run(args, w, W, H, gsq, torch, rank, world)
    cpu = None
    if world == 1 and not args.no_cpu_baseline:     # the oracle baseline: N = 1 only
        cpu = cpu_baseline(args, w, W, H_host)

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32 (tensor-core GEMM bf16 in, f32 acc)",
            "data": "synthetic (seeded; shapes and statistics of Llama-3.1-8B q_proj + calibration)",
            "config": _config(w, {"parallelism": f"{world} independent layer(s), one per GPU",
                                  "timing": ("one CUDA-graph replay of the timed steps (captured and "
                                             "replayed once before the timed region)")
                                  if graph is not None else "eager launches"}),
            "roofline": roofline, "roofline_gemm": roofline_gemm, "clocks": clocks,
            "diagnostics": diag,
            "gpu_launches": launches, "e2e": e2e, "cpu_baseline": cpu,
            "kernel_ms_per_step": {"gemm": gemm_ms / args.steps, "backward": bwd_ms / args.steps,
                                   "forward": fwd_ms / args.steps},
        }
        print(json.dumps(line), flush=True)
    del graph
    layer.close()
    if world > 1:
        dist.destroy_process_group()
    return 0


def gpu_arm_tokens(args, rank, world, local):
    """One step = w.micro micro-batches of w.tokens per-step tokens (gsq_step_tokens),
    Lion after the last; the token batches are resident in HBM and reused."""
    import torch
    import torch.distributed as dist

    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    from paper_2604_18556_gb300 import build
    build.build()
    from paper_2604_18556_gb300 import gsq, inputs

    w = rank_workload(_workload(args.workload), rank, world)
    W = inputs.make_weight(w, device="cuda")
    Xs = [inputs.make_token_batch(w, 0, j, device="cuda") for j in range(w.micro)]
    hyper = dict(init_bias=w.init_bias, seed=w.seed, lr_logits=w.lr_logits, lr_scales=w.lr_scales,
                 beta1=w.beta1, beta2=w.beta2, wd_logits=w.wd_logits, wd_scales=w.wd_scales,
                 param=w.param)
    layer = gsq.Layer(W, None, w.grid, w.group, calib_kind="batches", tokens_per_batch=w.tokens,
                      scale_mode=w.scale_mode, gemm="bf16", **hyper)
    stream = torch.cuda.current_stream()
    loss = torch.zeros(w.micro, device="cuda")
    T = w.steps

    def one_step(layer, t, Xs, loss):
        for j, X in enumerate(Xs):
            layer.step_tokens(t, j, w.micro, w.tau(t % T), X, kappa=w.kappa,
                              next_tau=w.tau((t + 1) % T), next_kappa=w.kappa, loss=loss[j:j + 1])

    t = 0
    for _ in range(args.warmup):
        one_step(layer, t, Xs, loss)
        t += 1
    layer.sync_status()
    torch.cuda.synchronize()
    sampler = ClockSampler(local)
    sampler.start()
    time.sleep(0.3)
    layer.profile_enable(True)
    layer.profile_read()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        one_step(layer, t, Xs, loss)
        t += 1
    e1.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clocks = sampler.stop()
    prof = layer.profile_read()
    layer.profile_enable(False)
    layer.sync_status()
    ms_step = max_over_ranks(e0.elapsed_time(e1), torch.device("cuda", local)) / args.steps
    value = whole_job_steps_per_s(ms_step, world)

    hbm, tf_burst, tf_sust, peak_src = _peaks()
    gemm_n, gemm_ms = prof["gemm"]
    bwd_n, bwd_ms = prof["backward"]
    tok_n, tok_ms = prof["tokens"]
    fwd_n, fwd_ms = prof["forward"]
    gemm_avg = gemm_ms / max(gemm_n, 1)
    flops_per_launch = w.gemm_flops_per_step() / w.micro      # Y = D X^T and G = 2 Y X
    gemm_tfs = flops_per_launch / (gemm_avg * 1e-3) / 1e12
    bytes_step = w.elementwise_bytes_per_step()
    bwd_gbs = bytes_step / (bwd_ms / args.steps * 1e-3) / 1e9
    roofline = {"kernel": f"{layer.kernel_name(gsq.GSQ_K_GEMM)} x 2 (Y = D X^T, then G = 2 Y X; "
                          "tcgen05, bf16 in, fp32 acc)",
                "bound": "tensor", "achieved": gemm_tfs, "peak": tf_sust, "unit": "TFLOP/s",
                "frac": gemm_tfs / tf_sust, "frac_of_burst": gemm_tfs / tf_burst, "traffic": None,
                "flops_per_launch": flops_per_launch, "avg_launch_ms": gemm_avg,
                "peak_source": f"{peak_src} bf16_tflops_sustained (MEASURED_PEAKS.json)"}
    roofline_bwd = {"kernel": "k_backward (accumulating / Lion + next forward), all micro-batches",
                    "bound": "hbm", "achieved": bwd_gbs, "peak": hbm, "unit": "GB/s",
                    "frac": bwd_gbs / hbm, "algorithmic_bytes_per_step": bytes_step,
                    "ms_per_step": bwd_ms / args.steps}
    launches = gemm_n * 2 + bwd_n + tok_n + fwd_n

    e2e = None
    if not args.no_e2e:
        e2e = e2e_run_tokens(args, w, W, Xs, hyper, gsq, torch, world, one_step)
    cpu = None
    if world == 1 and not args.no_cpu_baseline:     # the oracle baseline: N = 1 only
        cpu = cpu_baseline_tokens(args, w)
    if rank == 0:
        print(json.dumps({
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32 (tensor-core GEMMs bf16 in, f32 acc)",
            "data": "synthetic (seeded; Llama-3.1-8B q_proj shape, per-step token batches)",
            "config": _config(w, {"parallelism": f"{world} independent layer(s), one per GPU",
                                  "micro_batches": w.micro, "tokens_per_micro_batch": w.tokens,
                                  "l2": "token batches of "
                                        f"{w.tokens * w.cols * 4 / 2**20:.0f} MiB each, larger "
                                        "than L2"}),
            "roofline": roofline, "roofline_backward": roofline_bwd, "clocks": clocks,
            "gpu_launches": launches, "e2e": e2e, "cpu_baseline": cpu,
            "kernel_ms_per_step": {"gemm": gemm_ms / args.steps, "backward": bwd_ms / args.steps,
                                   "tokens": tok_ms / args.steps, "forward": fwd_ms / args.steps},
        }), flush=True)
    layer.close()
    if world > 1:
        dist.destroy_process_group()
    return 0


def e2e_run_tokens(args, w, W, Xs, hyper, gsq, torch, world, one_step):
    """The whole job through the public API from pinned host buffers: W and the
    micro-batch tokens uploaded, init, K steps (every micro-batch's loss read
    back), projection + packing, packed download."""
    W_host = W.cpu().pin_memory()
    X_host = [X.cpu().pin_memory() for X in Xs]
    K = args.steps
    loss_host = torch.zeros(K, w.micro, dtype=torch.float32).pin_memory()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    Wd = W_host.to("cuda", non_blocking=True)
    Xd = [X.to("cuda", non_blocking=True) for X in X_host]
    layer = gsq.Layer(Wd, None, w.grid, w.group, calib_kind="batches", tokens_per_batch=w.tokens,
                      scale_mode=w.scale_mode, gemm="bf16", **hyper)
    loss = torch.zeros(K, w.micro, device="cuda")
    for t in range(K):
        one_step(layer, t, Xd, loss[t])
        loss_host[t].copy_(loss[t], non_blocking=True)
    packed = torch.empty(layer.packed_size(), dtype=torch.uint8, device="cuda")
    layer.pack(packed)
    packed_host = torch.empty(packed.numel(), dtype=torch.uint8).pin_memory()
    packed_host.copy_(packed, non_blocking=True)
    torch.cuda.synchronize()
    dt = time.perf_counter() - t0
    layer.close()
    if not bool(torch.isfinite(loss_host).all()):
        raise RuntimeError("non-finite loss in the end-to-end run")
    h2d = W_host.numel() * W_host.element_size() + sum(X.numel() * 4 for X in X_host)
    return {"value": world * K / dt, "unit": UNIT, "h2d_bytes_per_step": h2d / K,
            "d2h_bytes_per_step": (4 * K * w.micro + packed_host.numel()) / K,
            "what": f"one {K}-step job: pinned W + {w.micro} token batches uploaded, init, "
                    f"{K} steps with every loss read back, projection + packing, download"}


def cpu_baseline_tokens(args, w):
    code = ("import sys, json; sys.path.insert(0, %r)\n"
            "import bench\n"
            "from paper_2604_18556_gb300 import configs as C\n"
            "full, desc, meas = bench.run_oracle_tokens_sample(C.WORKLOADS[%r], 3)\n"
            "print(json.dumps([full, desc]))\n") % (ROOT, w.name)
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1",
               CUDA_VISIBLE_DEVICES="")
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env,
                       cwd=ROOT, timeout=900)
    if r.returncode != 0:
        return {"value": None, "unit": UNIT, "cores": 1, "kind": "oracle",
                "sample": f"failed: {r.stderr[-300:]}"}
    full, desc = json.loads(r.stdout.strip().splitlines()[-1])
    return {"value": 1.0 / full, "unit": UNIT, "cores": 1, "kind": "oracle", "sample": desc}


def e2e_run(args, w, W, H, gsq, torch, rank, world):
    """The whole per-layer job through the public API with host buffers: pinned
    W and H copied to the GPU, init, K steps (each step's loss read back into
    pinned memory), projection + packing, packed result copied back."""
    W_host = W.cpu().pin_memory()
    H_host = H.cpu().pin_memory()
    stream = torch.cuda.current_stream()
    K = args.steps
    loss_host = torch.zeros(K, dtype=torch.float32).pin_memory()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    Wd = W_host.to("cuda", non_blocking=True)
    Hd = H_host.to("cuda", non_blocking=True)
    layer = gsq.Layer(Wd, Hd, w.grid, w.group, scale_mode=w.scale_mode, gemm="bf16",
                      init_bias=w.init_bias, seed=w.seed, lr_logits=w.lr_logits,
                      lr_scales=w.lr_scales, beta1=w.beta1, beta2=w.beta2,
                      wd_logits=w.wd_logits, wd_scales=w.wd_scales, param=w.param)
    loss = torch.zeros(K, device="cuda")
    for t in range(K):
        layer.step(t, w.tau(t % w.steps), w.kappa, next_tau=w.tau((t + 1) % w.steps),
                   next_kappa=w.kappa, loss=loss[t:t + 1])
        loss_host[t:t + 1].copy_(loss[t:t + 1], non_blocking=True)
    packed = torch.empty(layer.packed_size(), dtype=torch.uint8, device="cuda")
    layer.pack(packed)
    packed_host = torch.empty(packed.numel(), dtype=torch.uint8).pin_memory()
    packed_host.copy_(packed, non_blocking=True)
    torch.cuda.synchronize()
    dt = time.perf_counter() - t0
    layer.close()
    h2d = W_host.numel() * W_host.element_size() + H_host.numel() * H_host.element_size()
    d2h = 4 * K + packed_host.numel()
    if not bool(torch.isfinite(loss_host).all()):
        raise RuntimeError("non-finite loss in the end-to-end run")
    return {"value": world * K / dt, "unit": UNIT, "h2d_bytes_per_step": h2d / K,
            "d2h_bytes_per_step": d2h / K,
            "what": f"one {K}-step layer job: pinned W+H upload, init, {K} steps with the loss "
                    f"read back each step, projection + packing, packed download"}


def cpu_baseline(args, w, W, H_host):
    """Oracle step on a bounded row sample, in a single-threaded child process."""
    import numpy as np
    import tempfile
    rows = min(w.rows, 1024)
    with tempfile.TemporaryDirectory() as td:
        np.save(os.path.join(td, "W.npy"), W[0, :rows].float().cpu().numpy())
        np.save(os.path.join(td, "H.npy"), H_host)
        code = (
            "import sys, json, numpy as np; sys.path.insert(0, %r)\n"
            "import bench\n"
            "from paper_2604_18556_gb300 import configs as C\n"
            "w = C.WORKLOADS[%r]\n"
            "Wt = np.load(%r); H = np.load(%r)\n"
            "per, rows, meas = bench.run_oracle_sample(w, %f, 6, 1, Wt, H)\n"
            "print(json.dumps([per, rows, meas]))\n"
        ) % (ROOT, w.name, os.path.join(td, "W.npy"), os.path.join(td, "H.npy"),
             args.cpu_sample_seconds / 7)
        env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1")
        r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env,
                           cwd=ROOT, timeout=600)
        if r.returncode != 0:
            return {"value": None, "unit": UNIT, "cores": 1, "kind": "oracle",
                    "sample": f"failed: {r.stderr[-300:]}"}
        per, srows, meas = json.loads(r.stdout.strip().splitlines()[-1])
    return {"value": 1.0 / per, "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": f"{srows} of {w.rows} rows, 6 timed steps + 1 warm-up ({meas:.1f} s "
                      f"measured); full-layer step = sample x {w.rows}/{srows}"}


def main():
    args = _args()
    rank, world, local = _dist()
    if args.impl == "reference":
        return reference_arm(args, rank, world)
    if _workload(args.workload).calib == "batches":
        return gpu_arm_tokens(args, rank, world, local)
    return gpu_arm(args, rank, world, local)


if __name__ == "__main__":
    sys.exit(main())
