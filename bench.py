"""Benchmark of the GSQ relaxed-scalar-quantizer step on one GB300 (per rank).

One step = one gsq_step: (look-ahead forward from the previous step) + the
tensor-core loss GEMM + the fused backward/Lion/next-forward kernel, on the
Llama-3.1-8B q_proj-shaped layer (4096 x 4096 bf16, 2-bit grid, group 128,
tau annealed 1.0 -> 0.1 over 500 steps).  Prints one JSON line.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl gsq|reference]
                  [--workload NAME]

The K timed steps are captured once as a CUDA graph; the graph is replayed
until the timed window covers at least --min-window-ms, each replay (exactly K
steps) bracketed by a synchronize, and the median replay gives ms_per_step.  The
per-kernel times behind the rooflines come from a second graph of K steps with
the library's event records around every kernel, replayed in a window of its
own (those records slow a step by about 15 us, so they stay out of the headline).

--impl reference times the CPU oracle (the plain float64 restatement of the
method) on the host's cores: one single-threaded process per core, each
following its own block of rows (rows are independent, Eq. 1 with a linear f),
all blocks together covering the layer where the time allows it, else a row
sample scaled by R / rows.  Under torchrun, the layer is split across the ranks
(rows of a one-expert layer, whole experts of the MoE batch; no collective on
the data path), so the whole job advances one layer step per step (strong
scaling); rank 0 prints the whole layer's throughput.
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
    ap.add_argument("--cpu-step-seconds", type=float, default=1.5,
                    help="oracle baseline: target seconds per timed step of each host core")
    ap.add_argument("--min-window-ms", type=float, default=500.0,
                    help="replay the captured K-step graph until the timed window is this long")
    ap.add_argument("--unstaged", action="store_true",
                    help="time the backward with direct global loads (GSQ_FLAG_UNSTAGED)")
    ap.add_argument("--experts", type=int, default=0,
                    help="run a multi-expert workload with this many experts instead of all of "
                         "them (a smaller case of the same kernels, for profiling)")
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


def rank_shard(w, rank: int, world: int):
    """This rank's part of the layer: whole experts of a multi-expert layer, or a
    block of rows of a one-expert layer (rows and experts never exchange data, so
    the ranks share nothing but a copy of H)."""
    from paper_2604_18556_gb300 import configs as C
    return C.shard(w, rank, world)


def max_over_ranks(x: float, device) -> float:
    """Largest value over the process group (the slowest rank defines the time)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(x: float, device) -> float:
    """The whole layer's value of a per-shard sum (the loss: rows add up)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t)
    return float(t.item())


def layer_steps_per_s(ms_per_step: float) -> float:
    """Whole-layer steps per second: every rank advances its shard of the one
    layer once per step, so the job advances the layer once every ms_per_step."""
    return 1000.0 / ms_per_step


def replays_for_window(ms_per_replay: float, min_window_ms: float, cap: int = 1000) -> int:
    """Replays of the K-step graph that cover at least min_window_ms (>= 1)."""
    if ms_per_replay <= 0:
        return 1
    import math
    return max(1, min(cap, int(math.ceil(min_window_ms / ms_per_replay))))


def elementwise_bytes_8d(w) -> int:
    """Algorithmic HBM bytes of one step's elementwise work as the step is
    defined (separate forward, backward and Lion passes over the streams):
    forward reads the logits (4L) and W (b_W) and writes D (2); backward + Lion
    reads the logits, their momenta (4L each) and G (4) and writes the logits and
    momenta (4L each); local shift reads its base index j0 in both passes (2):
    n (20L + b_W + 6 [+ 2]) per step.  Scale terms are O(n / G) and left out."""
    return w.n * (20 * w.L + w.w_bytes() + 6 + (2 if w.param == "shift5" else 0))


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d.get("hbm_gbs", 6800.0), d.get("bf16_tflops", 1900.0), d.get(
            "bf16_tflops_sustained", 1700.0), "measured"
    return 6800.0, 1900.0, 1700.0, "fallback"


class ClockSampler:
    """nvidia-smi clocks, throttle reasons and utilisation sampled every 100 ms during the
    timed region; the SM clock reported is the median over samples with the GPU busy."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap,"
              "utilization.gpu")

    def __init__(self, device_index: int):
        self.dev = device_index
        self.lines = []
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100", "-i", str(self.dev)], stdout=subprocess.PIPE,
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
        sm, smax, reasons, busy = [], [], set(), []
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
            if len(parts) > 9:
                try:
                    if float(parts[9]) >= 50.0:
                        busy.append(float(parts[1]))
                except ValueError:
                    pass
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
        sm.sort()
        busy.sort()
        med = busy[len(busy) // 2] if busy else sm[len(sm) // 2]
        return {"sm_mhz": med, "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm), "samples_under_load": len(busy),
                "sm_mhz_all_samples": sm[len(sm) // 2]}


def _workload(name, experts=0):
    from paper_2604_18556_gb300 import configs as C
    w = C.WORKLOADS[name]
    if experts and w.experts > 1:
        w = C.shrunk(w, experts=min(experts, w.experts))
    return w


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
# CPU oracle on the host cores (baseline / reference arm)
# ----------------------------------------------------------------------------
_BLAS_THREAD_VARS = ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS")


def host_cores() -> int:
    """Cores this process may run on (its affinity mask, not the machine's count)."""
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def _oracle_problem(w, H_host):
    import numpy as np
    from oracle import gsq_oracle as O
    prob = O.Problem(E=w.experts, R=w.rows, C=w.cols, grid=np.asarray(w.grid, float), group=w.group,
                     seed=w.seed, scale_mode=w.scale_mode, H=H_host, lr_logits=w.lr_logits,
                     lr_scales=w.lr_scales, beta1=w.beta1, beta2=w.beta2, wd_logits=w.wd_logits,
                     wd_scales=w.wd_scales, shift=w.param == "shift5",
                     mask_sign=w.param == "mask_sign")
    return prob


def _input_device():
    import torch
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    if dev == "cpu":
        torch.set_num_threads(max(1, os.cpu_count() or 1))
    return dev


def _cpu_weight(w, rows):
    """Rows [0, rows) of expert 0's W from the seeded generator (on the GPU when
    one is present: input preparation only, not the timed oracle)."""
    from paper_2604_18556_gb300 import inputs
    return inputs.make_weight(w, device=_input_device(), experts=(0, 1),
                              rows=(0, rows))[0].float().cpu().numpy()


def _cpu_gram(w):
    """Expert 0's H (float64), prepared like the weights."""
    from paper_2604_18556_gb300 import inputs
    return inputs.make_gram(w, device=_input_device(), experts=(0, 1))[0].double().cpu().numpy()


def _oracle_block(root, w, w_path, h_path, lo, hi, n_warm, n_steps, barrier, queue, idx):
    """One spawned, single-threaded worker: the oracle's whole step on rows
    [lo, hi) of expert 0 -- n_warm untimed steps, then, once every worker is
    ready, n_steps timed ones.  Puts (idx, seconds of each timed step, error)."""
    for v in _BLAS_THREAD_VARS:
        os.environ[v] = "1"
    sys.path.insert(0, root)
    try:
        import numpy as np
        from oracle import gsq_oracle as O
        Wt = np.array(np.load(w_path, mmap_mode="r")[lo:hi])
        H = np.load(h_path, mmap_mode="r")          # pages shared by every worker
        prob = _oracle_problem(w, H[None])
        st = O.init_state(prob, Wt, np.arange(lo, hi), init_bias=w.init_bias)
        for t in range(n_warm):
            O.step(prob, st, t, w.tau(t), w.kappa)
        barrier.wait(timeout=900)
        times = []
        for t in range(n_warm, n_warm + n_steps):
            t0 = time.perf_counter()
            O.step(prob, st, t, w.tau(t), w.kappa)
            times.append(time.perf_counter() - t0)
        queue.put((idx, times, None))
    except Exception as e:  # report instead of leaving the parent waiting
        try:
            barrier.abort()
        except Exception:
            pass
        queue.put((idx, None, repr(e)))


def run_oracle_parallel(w, workers, rows_per_worker, n_warm, n_steps, Wt, H, timeout_s=1800):
    """`workers` spawned single-threaded oracle processes on consecutive blocks of
    rows_per_worker rows of Wt (the last block may be shorter), all timed over the
    same window.  Returns (seconds per timed step of the slowest worker, rows)."""
    import multiprocessing as mp
    import tempfile
    import numpy as np
    rows_total = Wt.shape[0]
    blocks = [(i * rows_per_worker, min(rows_total, (i + 1) * rows_per_worker))
              for i in range(workers)]
    blocks = [b for b in blocks if b[1] > b[0]]
    ctx = mp.get_context("spawn")             # never fork a process that holds a CUDA context
    saved = {v: os.environ.get(v) for v in _BLAS_THREAD_VARS}
    for v in _BLAS_THREAD_VARS:
        os.environ[v] = "1"
    try:
        with tempfile.TemporaryDirectory() as td:
            wp, hp = os.path.join(td, "W.npy"), os.path.join(td, "H.npy")
            np.save(wp, np.ascontiguousarray(Wt, dtype=np.float32))
            np.save(hp, np.ascontiguousarray(H, dtype=np.float64))
            barrier, queue = ctx.Barrier(len(blocks)), ctx.Queue()
            procs = [ctx.Process(target=_oracle_block,
                                 args=(ROOT, w, wp, hp, lo, hi, n_warm, n_steps, barrier,
                                       queue, i), daemon=True)
                     for i, (lo, hi) in enumerate(blocks)]
            for p in procs:
                p.start()
            times, errors = {}, []
            try:
                for _ in procs:
                    idx, tt, err = queue.get(timeout=timeout_s)
                    if err:
                        errors.append(err)
                    else:
                        times[idx] = tt
            finally:
                for p in procs:
                    p.join(timeout=30)
                    if p.is_alive():
                        p.terminate()
            if errors:
                raise RuntimeError("oracle worker failed: " + errors[0])
    finally:
        for v, x in saved.items():
            if x is None:
                os.environ.pop(v, None)
            else:
                os.environ[v] = x
    per_step = max(sum(t) for t in times.values()) / n_steps
    return per_step, sum(hi - lo for lo, hi in blocks)


def time_oracle(w, cores, step_s, n_warm, n_steps, single=True):
    """The oracle's whole-layer step time on `cores` host cores: one process per
    core on its own block of expert 0's rows; the blocks cover all R rows when
    that keeps a step near step_s seconds, else they are a sample and the time is
    scaled by (E R) / rows (rows are independent; every row costs the same).  The
    per-row cost comes from a 16-row probe.  With single=True the same block is
    also timed alone on one core.  Returns a dict for the JSON line."""
    import math
    R = w.rows
    H = _cpu_gram(w)
    probe = min(16, R)
    t_probe, _ = run_oracle_parallel(w, 1, probe, 1, 1, _cpu_weight(w, probe), H)
    t_row = t_probe / probe
    rpw = max(1, min(math.ceil(R / cores), int(step_s / max(t_row, 1e-9))))
    workers = min(cores, math.ceil(R / rpw))
    Wt = _cpu_weight(w, min(R, workers * rpw))
    per_step, covered = run_oracle_parallel(w, workers, rpw, n_warm, n_steps, Wt, H)
    scale = w.experts * w.rows / covered
    out = {"full_step_s": per_step * scale, "workers": workers, "rows": covered,
           "rows_per_worker": rpw, "per_step_s": per_step, "scale": scale,
           "n_warm": n_warm, "n_steps": n_steps}
    if single:
        n1 = max(1, min(n_steps, 2))
        t1, c1 = run_oracle_parallel(w, 1, rpw, 1, n1, Wt[:rpw], H)
        out["single_core_full_step_s"] = t1 * (w.experts * w.rows) / c1
        out["single_core_rows"] = c1
    return out


def oracle_sample_text(w, r, cores):
    whole = w.experts * w.rows
    what = ("the whole layer" if r["scale"] == 1.0 else
            f"a sample of {r['rows']} of {whole} rows, time scaled by {r['scale']:.3g}")
    return (f"{r['workers']} single-threaded oracle processes on {cores} host cores, "
            f"{r['rows_per_worker']} rows each ({what}); {r['n_warm']} untimed + "
            f"{r['n_steps']} timed steps each, slowest process's time per step")


def run_oracle_tokens_sample(w, n_steps: int, rows: int = 256, tok=(512, 4096), row0: int = 0):
    """Oracle step on per-step token batches, sampled in rows and tokens.  The
    micro-batch cost is linear in its tokens (the loss contractions) plus a part
    that is not (noise, softmax, backward, Lion): both are fitted from one
    micro-batch of tok[0] and of tok[1] tokens on rows [row0, row0 + rows), then
    scaled to the workload's tokens per micro-batch, micro-batches and rows.
    Returns (seconds per full step on one core, description of the sample,
    seconds measured)."""
    import dataclasses
    import numpy as np
    import torch
    from oracle import gsq_oracle as O
    from paper_2604_18556_gb300 import configs as C
    from paper_2604_18556_gb300 import inputs
    w1 = C.shrunk(w, experts=1)
    Wt = inputs.make_weight(w1)[0, row0:row0 + rows].float().numpy()
    prob = _oracle_problem(w1, None)
    per_tok = []
    measured = 0.0
    for T in tok:
        wt = dataclasses.replace(w1, tokens=T, micro=1)
        X = inputs.make_token_batch(wt, 0, 0).double().numpy()
        times = []
        for t in range(n_steps + 1):
            st = O.init_state(prob, Wt, np.arange(row0, row0 + rows), init_bias=w.init_bias)
            t0 = time.perf_counter()
            O.step_microbatches(prob, st, t, [X], w.tau(t), w.kappa)
            times.append(time.perf_counter() - t0)
        measured += sum(times)
        per_tok.append(float(np.median(times[1:])))
    b = (per_tok[1] - per_tok[0]) / (tok[1] - tok[0])
    if b <= 0.0:                 # timing noise swamped the slope: scale the larger batch
        b, a = per_tok[1] / tok[1], 0.0
    else:
        a = max(per_tok[0] - b * tok[0], 0.0)
    full = (a + b * w.tokens) * w.micro * (w.experts * w.rows) / rows
    desc = (f"{rows} rows x one micro-batch of {tok[0]} and of {tok[1]} tokens, {n_steps} timed "
            f"steps each ({measured:.1f} s measured); cost fitted as a + b*tokens and scaled to "
            f"{w.tokens} tokens x {w.micro} micro-batches x {w.experts * w.rows} rows")
    return full, desc, measured


def run_oracle_tokens_parallel(w, n_steps: int, cores: int, rows: int = 256):
    """run_oracle_tokens_sample in one single-threaded process per host core, all at
    once, each on its own block of rows; the whole layer's step takes the slowest
    process's one-core estimate divided by the number of processes.  Returns
    (seconds per full step, description, processes)."""
    procs = max(1, min(cores, w.rows // rows))
    code = ("import sys, json; sys.path.insert(0, %r)\n"
            "import bench\n"
            "w = bench._workload(%r)\n"
            "full, desc, meas = bench.run_oracle_tokens_sample(w, %d, rows=%d, row0=int(sys.argv[1]))\n"
            "print(json.dumps([full, desc]))\n") % (ROOT, w.name, n_steps, rows)
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1",
               CUDA_VISIBLE_DEVICES="")
    ps = [subprocess.Popen([sys.executable, "-c", code, str(i * rows)], stdout=subprocess.PIPE,
                           stderr=subprocess.PIPE, text=True, env=env, cwd=ROOT)
          for i in range(procs)]
    outs = []
    for p in ps:
        out, err = p.communicate(timeout=1800)
        if p.returncode != 0:
            raise RuntimeError(f"oracle worker failed: {err[-300:]}")
        outs.append(json.loads(out.strip().splitlines()[-1]))
    full = max(o[0] for o in outs) / procs
    desc = (f"{procs} single-threaded oracle processes at once, each on its own {rows} rows: "
            f"{outs[0][1]}; whole-layer time = slowest process's / {procs}")
    return full, desc, procs


def reference_arm(args, rank, world):
    """The oracle as it stands, on the host's cores, for the same workload and
    metric; rank 0 alone runs it under torchrun."""
    if rank != 0:
        return 0
    w = _workload(args.workload, args.experts)
    cores = host_cores()
    common = {"impl": "reference", "metric": METRIC, "unit": UNIT, "n_gpus": args.gpus,
              "steps": args.steps, "warmup": args.warmup, "higher_is_better": True,
              "scaling": "strong", "vs_baseline": None, "dtype": "f64", "data": "synthetic"}
    if w.calib == "batches":
        full_step_s, desc, procs = run_oracle_tokens_parallel(w, max(args.steps, 1), cores)
        value = 1.0 / full_step_s
        print(json.dumps(dict(common, **{
            "value": value, "ms_per_step": full_step_s * 1e3,
            "config": _config(w, {"oracle": "numpy float64, one process per host core"}),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": procs, "kind": "oracle",
                             "sample": desc},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        })), flush=True)
        return 0
    r = time_oracle(w, cores, step_s=3.0, n_warm=args.warmup, n_steps=max(args.steps, 1),
                    single=False)
    value = 1.0 / r["full_step_s"]
    print(json.dumps(dict(common, **{
        "value": value, "ms_per_step": r["full_step_s"] * 1e3,
        "config": _config(w, {"oracle": "numpy float64, one process per host core"}),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": r["workers"], "kind": "oracle",
                         "sample": oracle_sample_text(w, r, cores)},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    })), flush=True)
    return 0


# ----------------------------------------------------------------------------
# GPU arm
# ----------------------------------------------------------------------------
def _parallelism(w, sh, world):
    if world == 1:
        return "1 GPU, the whole layer"
    (e0, e1), (r0, r1) = sh.experts, sh.rows
    part = f"experts {e0}..{e1 - 1}" if w.experts > 1 else f"rows {r0}..{r1 - 1}"
    return (f"{world} GPUs, one layer split by {'experts' if w.experts > 1 else 'rows'} "
            f"(rank 0 holds {part}), H replicated, no collective in the timed region")


def _timed_replays(args, run_k_steps, stream, world, device, min_window_ms=None):
    """Times replays of exactly K steps, each bracketed by a barrier (N > 1) and a
    synchronize, until the window covers min_window_ms (default args.min_window_ms).
    Returns the list of per-replay milliseconds (the same count on every rank)."""
    if min_window_ms is None:
        min_window_ms = args.min_window_ms
    import torch
    import torch.distributed as dist

    def one():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        run_k_steps()
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1)

    reps = [one()]
    n = replays_for_window(max_over_ranks(reps[0], device), min_window_ms)
    for _ in range(n - 1):
        reps.append(one())
    if world > 1:
        dist.barrier()
    return reps


def gpu_arm(args, rank, world, local):
    import numpy as np
    import torch
    import torch.distributed as dist

    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=device)
    from paper_2604_18556_gb300 import build
    build.build()
    from paper_2604_18556_gb300 import gsq, inputs

    whole = _workload(args.workload, args.experts)
    sh = rank_shard(whole, rank, world)
    w = sh.workload
    W = inputs.make_weight(whole, device="cuda", experts=sh.experts, rows=sh.rows)
    H = inputs.make_gram(whole, device="cuda", experts=sh.experts)
    hyper = dict(init_bias=w.init_bias, seed=w.seed, lr_logits=w.lr_logits, lr_scales=w.lr_scales,
                 beta1=w.beta1, beta2=w.beta2, wd_logits=w.wd_logits, wd_scales=w.wd_scales,
                 param=w.param, index_offset=sh.index_offset)
    layer = gsq.Layer(W, H, w.grid, w.group, calib_kind="H", scale_mode=w.scale_mode, gemm="bf16",
                      unstaged=args.unstaged, **hyper)
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

    # The K timed steps are captured as CUDA graphs (untimed): K distinct steps
    # t0..t0+K-1, so a replay does exactly the work of K eager steps without host
    # launch gaps.  Two graphs: the headline times one with nothing but the step's
    # kernels; the per-kernel split comes from a second graph of K further steps
    # with the library's profiling events as event-record nodes around every
    # kernel, replayed in a window of its own (the record read at the end is the
    # last replay's).  Those records add gaps between the kernels, so that window
    # runs slower and its per-kernel averages over-state each kernel a little: the
    # roofline fractions drawn from them are conservative.  K is even, so the
    # look-ahead D a replay leaves behind sits in the buffer its first step reads.
    def capture(t0):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            for i in range(args.steps):
                layer.step(t0 + i, sched(t0 + i), w.kappa, next_tau=sched(t0 + i + 1),
                           next_kappa=w.kappa, loss=loss)
        g.replay()          # first replay (graph upload), untimed
        torch.cuda.synchronize()
        return g

    graph = graph_prof = None
    layer.profile_enable(False)
    if not args.no_graph:
        graph = capture(t)
        t += args.steps
        layer.profile_enable(True)
        graph_prof = capture(t)
        t += args.steps
        layer.profile_enable(False)

    state = {"t": t}

    def eager_k_steps():
        for _ in range(args.steps):
            tt = state["t"]
            layer.step(tt, sched(tt), w.kappa, next_tau=sched(tt + 1), next_kappa=w.kappa,
                       loss=loss)
            state["t"] = tt + 1

    def run_k_steps():
        if graph is not None:
            graph.replay()
        else:
            eager_k_steps()

    def run_k_steps_profiled():
        if graph_prof is not None:
            graph_prof.replay()
        else:
            eager_k_steps()

    sampler = ClockSampler(local)
    sampler.start()
    time.sleep(0.3)
    reps = _timed_replays(args, run_k_steps, stream, world, device)
    if graph_prof is None:   # eager steps record their events from here on (a captured
        layer.profile_enable(True)   # graph holds the events recorded at its capture)
        layer.profile_read()
    prof_reps = _timed_replays(args, run_k_steps_profiled, stream, world, device,
                               min_window_ms=min(200.0, args.min_window_ms))
    prof = layer.profile_read()
    layer.profile_enable(False)
    clocks = sampler.stop()
    layer.sync_status()
    ms_step = max_over_ranks(float(np.median(reps)), device) / args.steps
    value = layer_steps_per_s(ms_step)
    loss_total = sum_over_ranks(float(loss.item()), device)   # reporting only, untimed

    hbm, tf_burst, tf_sust, peak_src = _peaks()
    bwd_n, bwd_ms = prof["backward"]
    gemm_n, gemm_ms = prof["gemm"]
    fwd_n, fwd_ms = prof["forward"]
    bwd_avg = bwd_ms / max(bwd_n, 1)
    gemm_avg = gemm_ms / max(gemm_n, 1)
    per_weight_8d = 20 * w.L + w.w_bytes() + 6 + (2 if w.param == "shift5" else 0)
    bytes_8d = elementwise_bytes_8d(w)
    bytes_fused = w.elementwise_bytes_per_weight() * w.n
    traffic = committed_traffic(w.name) if world == 1 and not args.experts else None
    gbs = lambda nbytes: nbytes / (bwd_avg * 1e-3) / 1e9
    kname = layer.kernel_name(gsq.GSQ_K_BACKWARD)
    roofline = {
        "kernel": f"{kname} (backward + Lion + the next step's forward, one launch per step)",
        "bound": "hbm", "achieved": gbs(bytes_8d), "peak": hbm, "unit": "GB/s",
        "frac": gbs(bytes_8d) / hbm, "traffic": traffic,
        "peak_source": f"{peak_src}: MEASURED_PEAKS.json hbm_gbs (copy, burst)",
        "algorithmic_bytes_per_weight": per_weight_8d, "weights_per_launch": w.n,
        "algorithmic_bytes_per_launch": bytes_8d, "avg_launch_ms": bwd_avg,
        "frac_of_8TBps": gbs(bytes_8d) / 8000.0,
        "moved_bytes_per_launch_fused": bytes_fused,
        "frac_on_moved_bytes_fused": gbs(bytes_fused) / hbm,
        "frac_on_ncu_traffic": None if not traffic else gbs(traffic) / hbm}
    flops = w.gemm_flops_per_step()
    gemm_tfs = flops / (gemm_avg * 1e-3) / 1e12
    roofline_gemm = {"kernel": f"{layer.kernel_name(gsq.GSQ_K_GEMM)} (tcgen05 loss contraction)",
                     "bound": "tensor", "achieved": gemm_tfs, "peak": tf_burst, "unit": "TFLOP/s",
                     "frac": gemm_tfs / tf_burst, "frac_of_sustained": gemm_tfs / tf_sust,
                     "flops_per_launch": flops, "avg_launch_ms": gemm_avg,
                     "peak_source": f"{peak_src}: bf16_tflops (burst; the timed windows are "
                                    f"{sum(reps):.0f} + {sum(prof_reps):.0f} ms of replays)"}
    # kernels of the headline window: the profiled graph's last replay holds one replay's
    # launches; eager steps launch a GEMM and a backward kernel per step
    launches = ((bwd_n + gemm_n + fwd_n) * len(reps) if graph is not None
                else 2 * args.steps * len(reps))

    # method diagnostics of the state after the timed steps (not timed)
    diag = layer.diagnose(sched(state["t"]), w.kappa)
    diag["after_step"] = state["t"]
    e2e = None
    if not args.no_e2e:
        e2e = e2e_run(args, w, W, H, gsq, torch, device, hyper)
    cpu = None
    if world == 1 and not args.no_cpu_baseline:     # the oracle baseline: N = 1 only
        cpu = cpu_baseline(args, whole)

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
            "scaling": "strong", "vs_baseline": None,
            "dtype": "f32 (tensor-core GEMM bf16 in, f32 acc)",
            "data": "synthetic (seeded; shapes and statistics of Llama-3.1-8B q_proj + calibration)",
            "config": _config(whole, {
                "parallelism": _parallelism(whole, sh, world),
                "timing": (f"{len(reps)} replays of one CUDA graph of the {args.steps} timed steps "
                           f"(each replay bracketed by a synchronize; median replay), "
                           f"{sum(reps):.1f} ms timed in total; the per-kernel split from "
                           f"{len(prof_reps)} replays of a second graph of {args.steps} steps "
                           f"with event records around every kernel") if graph is not None else
                          f"{len(reps)} rounds of {args.steps} eager steps, median round; the "
                          f"per-kernel split from {len(prof_reps)} further rounds with event "
                          f"records around every kernel"}),
            "timed_window_ms": sum(reps), "replays": len(reps),
            "ms_per_step_with_kernel_events": float(np.median(prof_reps)) / args.steps,
            "roofline": roofline, "roofline_gemm": roofline_gemm, "clocks": clocks,
            "diagnostics": diag, "loss_last_step": loss_total,
            "gpu_launches": launches, "e2e": e2e, "cpu_baseline": cpu,
            "kernel_ms_per_step": {"gemm": gemm_ms / max(gemm_n, 1), "backward": bwd_avg,
                                   "forward": fwd_ms / max(args.steps, 1)},
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
    import numpy as np
    import torch
    import torch.distributed as dist

    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    from paper_2604_18556_gb300 import build
    build.build()
    from paper_2604_18556_gb300 import gsq, inputs

    whole = _workload(args.workload, args.experts)
    sh = rank_shard(whole, rank, world)
    w = sh.workload
    W = inputs.make_weight(whole, device="cuda", experts=sh.experts, rows=sh.rows)
    Xs = [inputs.make_token_batch(w, 0, j, device="cuda") for j in range(w.micro)]
    hyper = dict(init_bias=w.init_bias, seed=w.seed, lr_logits=w.lr_logits, lr_scales=w.lr_scales,
                 beta1=w.beta1, beta2=w.beta2, wd_logits=w.wd_logits, wd_scales=w.wd_scales,
                 param=w.param, index_offset=sh.index_offset)
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
    state = {"t": t}

    def run_k_steps():
        for _ in range(args.steps):
            one_step(layer, state["t"], Xs, loss)
            state["t"] += 1

    # the headline from rounds with nothing but the step's kernels; the per-kernel
    # split from further rounds with the library's event records around every kernel
    device = torch.device("cuda", local)
    reps = _timed_replays(args, run_k_steps, stream, world, device)
    layer.profile_enable(True)
    layer.profile_read()
    prof_reps = _timed_replays(args, run_k_steps, stream, world, device,
                               min_window_ms=min(200.0, args.min_window_ms))
    prof = layer.profile_read()
    layer.profile_enable(False)
    clocks = sampler.stop()
    layer.sync_status()
    n_timed = args.steps * len(prof_reps)     # steps of the profiled rounds
    ms_step = max_over_ranks(float(np.median(reps)), device) / args.steps
    value = layer_steps_per_s(ms_step)

    hbm, tf_burst, tf_sust, peak_src = _peaks()
    gemm_n, gemm_ms = prof["gemm"]
    bwd_n, bwd_ms = prof["backward"]
    tok_n, tok_ms = prof["tokens"]
    fwd_n, fwd_ms = prof["forward"]
    gemm_avg = gemm_ms / max(gemm_n, 1)
    gram = layer.tensor_size(gsq.GSQ_T_H) > 0     # the layer contracts through X^T X
    sym = os.environ.get("GSQ_TOKEN_SYM", "1") != "0"   # ... formed from its upper triangle
    flops_per_launch = w.gemm_flops_per_step(gram, sym) / w.micro   # a micro-batch's GEMMs
    gemm_tfs = flops_per_launch / (gemm_avg * 1e-3) / 1e12
    bytes_step = w.elementwise_bytes_per_step()
    bwd_gbs = bytes_step / (bwd_ms / n_timed * 1e-3) / 1e9
    route = ("H = X^T X" + (" (upper triangle, mirrored)" if sym else "") + ", then G = 2 D H"
             if gram else "Y = D X^T, then G = 2 Y X")
    roofline = {"kernel": f"{layer.kernel_name(gsq.GSQ_K_GEMM)} x 2 ({route}; "
                          "tcgen05, bf16 in, fp32 acc)",
                "bound": "tensor", "achieved": gemm_tfs, "peak": tf_burst, "unit": "TFLOP/s",
                "frac": gemm_tfs / tf_burst, "frac_of_sustained": gemm_tfs / tf_sust,
                "traffic": None, "flops_per_launch": flops_per_launch, "avg_launch_ms": gemm_avg,
                "peak_source": f"{peak_src}: bf16_tflops (burst; MEASURED_PEAKS.json)"}
    roofline_bwd = {"kernel": "k_backward (accumulating / Lion + next forward), all micro-batches",
                    "bound": "hbm", "achieved": bwd_gbs, "peak": hbm, "unit": "GB/s",
                    "frac": bwd_gbs / hbm, "algorithmic_bytes_per_step": bytes_step,
                    "ms_per_step": bwd_ms / n_timed}
    # kernels of the headline rounds (a GEMM profile entry covers a micro-batch's GEMMs)
    per_gemm = 3 if gram and sym else 2      # the GEMMs of a micro-batch (and the mirror)
    launches = (gemm_n * per_gemm + bwd_n + tok_n + fwd_n) * len(reps) // max(len(prof_reps), 1)

    e2e = None
    if not args.no_e2e:
        e2e = e2e_run_tokens(args, w, W, Xs, hyper, gsq, torch, device, one_step)
    cpu = None
    if world == 1 and not args.no_cpu_baseline:     # the oracle baseline: N = 1 only
        cpu = cpu_baseline_tokens(args, whole)
    if rank == 0:
        print(json.dumps({
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
            "scaling": "strong", "vs_baseline": None,
            "dtype": "f32 (tensor-core GEMMs bf16 in, f32 acc)",
            "data": "synthetic (seeded; Llama-3.1-8B q_proj shape, per-step token batches)",
            "timed_window_ms": sum(reps), "replays": len(reps),
            "ms_per_step_with_kernel_events": float(np.median(prof_reps)) / args.steps,
            "config": _config(whole, {"parallelism": _parallelism(whole, sh, world),
                                  "timing": f"{len(reps)} rounds of {args.steps} eager steps, "
                                            f"median round; the per-kernel split from "
                                            f"{len(prof_reps)} further rounds with event records "
                                            f"around every kernel",
                                  "micro_batches": w.micro, "tokens_per_micro_batch": w.tokens,
                                  "l2": "token batches of "
                                        f"{w.tokens * w.cols * 4 / 2**20:.0f} MiB each, larger "
                                        "than L2"}),
            "roofline": roofline, "roofline_backward": roofline_bwd, "clocks": clocks,
            "gpu_launches": launches, "e2e": e2e, "cpu_baseline": cpu,
            "kernel_ms_per_step": {"gemm": gemm_ms / n_timed, "backward": bwd_ms / n_timed,
                                   "tokens": tok_ms / n_timed, "forward": fwd_ms / n_timed},
        }), flush=True)
    layer.close()
    if world > 1:
        dist.destroy_process_group()
    return 0


def make_read_back(torch):
    """Per-step read-back of a step's loss into pinned host memory on a copy stream of
    its own: the copy waits for the step (an event on the compute stream) but does not
    hold the next step's kernels behind it."""
    copy_stream = torch.cuda.Stream()
    done = torch.cuda.Event()   # one event, recorded again every step: a wait takes the
                                # record current when it is enqueued

    def read_back(dst_host, src_dev):   # src_dev stays alive until the job's final sync
        done.record()
        copy_stream.wait_event(done)
        with torch.cuda.stream(copy_stream):
            dst_host.copy_(src_dev, non_blocking=True)
    return read_back


def e2e_run_tokens(args, w, W, Xs, hyper, gsq, torch, device, one_step):
    """The whole job through the public API from pinned host buffers: W and the
    micro-batch tokens uploaded, init, K steps (every micro-batch's loss read
    back), projection + packing, packed download."""
    W_host = W.cpu().pin_memory()
    X_host = [X.cpu().pin_memory() for X in Xs]
    K = args.steps
    loss_host = torch.zeros(K, w.micro, dtype=torch.float32).pin_memory()
    read_back = make_read_back(torch)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    Wd = W_host.to("cuda", non_blocking=True)
    Xd = [X.to("cuda", non_blocking=True) for X in X_host]
    layer = gsq.Layer(Wd, None, w.grid, w.group, calib_kind="batches", tokens_per_batch=w.tokens,
                      scale_mode=w.scale_mode, gemm="bf16", **hyper)
    loss = torch.zeros(K, w.micro, device="cuda")
    for t in range(K):
        one_step(layer, t, Xd, loss[t])
        read_back(loss_host[t], loss[t])
    packed = torch.empty(layer.packed_size(), dtype=torch.uint8, device="cuda")
    layer.pack(packed)
    packed_host = torch.empty(packed.numel(), dtype=torch.uint8).pin_memory()
    packed_host.copy_(packed, non_blocking=True)
    torch.cuda.synchronize()
    dt = max_over_ranks(time.perf_counter() - t0, device)
    layer.close()
    if not bool(torch.isfinite(loss_host).all()):
        raise RuntimeError("non-finite loss in the end-to-end run")
    h2d = W_host.numel() * W_host.element_size() + sum(X.numel() * 4 for X in X_host)
    return {"value": K / dt, "unit": UNIT, "h2d_bytes_per_step": h2d / K,
            "d2h_bytes_per_step": (4 * K * w.micro + packed_host.numel()) / K,
            "what": f"one {K}-step job: pinned W + {w.micro} token batches uploaded, init, "
                    f"{K} steps with every loss read back, projection + packing, download"}


def cpu_baseline_tokens(args, w):
    """The oracle on every host core (one single-threaded process per core, each on
    its own block of rows), per-step token batches."""
    cores = host_cores()
    try:
        full, desc, procs = run_oracle_tokens_parallel(w, 3, cores)
    except Exception as e:  # the baseline is reported, never required
        return {"value": None, "unit": UNIT, "cores": cores, "kind": "oracle",
                "sample": f"failed: {e!r}"[:300]}
    return {"value": 1.0 / full, "unit": UNIT, "cores": procs, "kind": "oracle", "sample": desc}


def e2e_run(args, w, W, H, gsq, torch, device, hyper):
    """The whole per-layer job through the public API with host buffers: pinned
    W and H copied to the GPU, init, K steps (each step's loss read back into
    pinned memory), projection + packing, packed result copied back.  Under
    torchrun every rank runs its shard's job; the slowest rank's time counts."""
    W_host = W.cpu().pin_memory()
    H_host = H.cpu().pin_memory()
    K = args.steps
    loss_host = torch.zeros(K, dtype=torch.float32).pin_memory()
    read_back = make_read_back(torch)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    Wd = W_host.to("cuda", non_blocking=True)
    Hd = H_host.to("cuda", non_blocking=True)
    layer = gsq.Layer(Wd, Hd, w.grid, w.group, scale_mode=w.scale_mode, gemm="bf16", **hyper)
    loss = torch.zeros(K, device="cuda")
    for t in range(K):
        layer.step(t, w.tau(t % w.steps), w.kappa, next_tau=w.tau((t + 1) % w.steps),
                   next_kappa=w.kappa, loss=loss[t:t + 1])
        read_back(loss_host[t:t + 1], loss[t:t + 1])
    packed = torch.empty(layer.packed_size(), dtype=torch.uint8, device="cuda")
    layer.pack(packed)
    packed_host = torch.empty(packed.numel(), dtype=torch.uint8).pin_memory()
    packed_host.copy_(packed, non_blocking=True)
    torch.cuda.synchronize()
    dt = max_over_ranks(time.perf_counter() - t0, device)
    layer.close()
    h2d = W_host.numel() * W_host.element_size() + H_host.numel() * H_host.element_size()
    d2h = 4 * K + packed_host.numel()
    if not bool(torch.isfinite(loss_host).all()):
        raise RuntimeError("non-finite loss in the end-to-end run")
    return {"value": K / dt, "unit": UNIT, "h2d_bytes_per_step": h2d / K,
            "d2h_bytes_per_step": d2h / K,
            "what": f"one {K}-step layer job: pinned W+H upload, init, {K} steps with the loss "
                    f"read back each step, projection + packing, packed download"}


def cpu_baseline(args, w):
    """The oracle on every host core (one single-threaded process per core, each on
    its own block of rows), with the same block on one core beside it."""
    cores = host_cores()
    try:
        r = time_oracle(w, cores, step_s=args.cpu_step_seconds, n_warm=1, n_steps=3, single=True)
    except Exception as e:  # the baseline is reported, never required
        return {"value": None, "unit": UNIT, "cores": cores, "kind": "oracle",
                "sample": f"failed: {e!r}"[:300]}
    return {"value": 1.0 / r["full_step_s"], "unit": UNIT, "cores": r["workers"], "kind": "oracle",
            "sample": oracle_sample_text(w, r, cores),
            "single_core": {"value": 1.0 / r["single_core_full_step_s"], "unit": UNIT, "cores": 1,
                            "sample": f"the first {r['single_core_rows']}-row block alone on one "
                                      f"core, time scaled to the whole layer"}}


def main():
    args = _args()
    rank, world, local = _dist()
    if args.impl == "reference":
        return reference_arm(args, rank, world)
    if _workload(args.workload, args.experts).calib == "batches":
        return gpu_arm_tokens(args, rank, world, local)
    return gpu_arm(args, rank, world, local)


if __name__ == "__main__":
    sys.exit(main())
