"""The five synthetic layer workloads the step is built and measured on.

Each workload fixes a layer shape, a grid, a group size, a calibration recipe
and a temperature schedule.  The shapes follow the layers the paper quantizes
(Llama-3.1-8B/70B linear layers and MoE experts, §4.1); the optimiser
hyper-parameters follow the paper's training tables (Table 5: Lion, logits lr
1e-4, group-scales lr 5e-5, betas (0.9, 0.95), weight decay 1.0; Table 7: the
K-Quant scales are frozen, scale lr 0).

Nothing here computes any part of the method.
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace
from typing import Tuple

GRID_TERNARY = (-1.0, 0.0, 1.0)
GRID_2BIT_SYM = (-1.5, -0.5, 0.5, 1.5)
GRID_2BIT_SKEWED = (-2.0, -1.0, 0.0, 1.0)          # §3.2 "The 2-bit case"
GRID_3BIT_SYM = (-3.5, -2.5, -1.5, -0.5, 0.5, 1.5, 2.5, 3.5)

SCALE_GROUP = "group"
SCALE_KQUANT2 = "kquant2"


@dataclass(frozen=True)
class Workload:
    name: str
    experts: int
    rows: int                  # R = out_features
    cols: int                  # C = in_features
    grid: Tuple[float, ...]
    group: int                 # scale group along the input dim (16 = K-Quant sub-block)
    w_dtype: str               # "f32" | "bf16"
    calib: str                 # "X" (tokens kept) | "H" (Gram matrix) | "batches" (per step)
    tokens: int                # calibration tokens per expert (per micro-batch for "batches")
    token_dist: str            # "normal" | "student_t3"
    outliers: int              # number of outlier channels
    outlier_scale: float
    steps: int
    tau0: float
    tau1: float
    kappa: float = 1.0
    scale_mode: str = SCALE_GROUP
    init_bias: float = 2.0
    seed: int = 0
    lr_logits: float = 1e-4
    lr_scales: float = 5e-5
    beta1: float = 0.9
    beta2: float = 0.95
    wd_logits: float = 1.0
    wd_scales: float = 0.0
    data_seed: int = 0
    pack: bool = False
    micro: int = 1             # "batches": micro-batches per step (gradient accumulation)
    param: str = "full"        # "full": one logit per level; "shift5": local shift (§3.2);
    #                            "mask_sign": ternary mask x sign (§3.1, Alg. 2)

    @property
    def K(self) -> int:
        return len(self.grid)

    @property
    def L(self) -> int:
        """Logits per weight: K, 5 shifts around the initial index, or (mask, sign)."""
        return {"shift5": 5, "mask_sign": 2}.get(self.param, self.K)

    @property
    def n(self) -> int:
        return self.experts * self.rows * self.cols

    def tau(self, t: int) -> float:
        """Linear temperature schedule tau0 -> tau1 over steps 0..T-1."""
        if self.steps <= 1:
            return self.tau0
        return self.tau0 + (self.tau1 - self.tau0) * t / (self.steps - 1)

    def w_bytes(self) -> int:
        return 4 if self.w_dtype == "f32" else 2

    def elementwise_bytes_per_weight(self) -> int:
        """Algorithmic HBM bytes per weight of one steady-state step's fused
        elementwise kernel (backward t + Lion + forward t+1):
        read logits, logit momentum (4L each, L logits per weight), G (4), W (b_W),
        the initial index j0 with local shift (1);
        write logits, logit momentum (4L each), D for the next step (2)."""
        return 16 * self.L + 4 + self.w_bytes() + 2 + (1 if self.param == "shift5" else 0)

    def gram_route(self, sym=True) -> bool:
        """Per-step tokens on the tensor cores contract through each micro-batch's Gram
        matrix (H = X^T X, then G = 2 D H) when that costs fewer flops than Y = D X^T,
        G = 2 Y X: C (T + 2R) < 4 R T with H formed from its upper triangle (sym), else
        C (T + R) < 2 R T."""
        if self.calib != "batches":
            return False
        C_, T, R = self.cols, self.tokens, self.rows
        return C_ * (T + 2 * R) < 4 * R * T if sym else C_ * (T + R) < 2 * R * T

    def gemm_flops_per_step(self, gram=None, sym=True) -> int:
        """Loss contraction flops of one step: G = 2 D H (2 R C^2 per expert), or per
        micro-batch Y = D X^T and G = 2 Y X (4 R C T per expert) or, on the Gram route
        (gram: the layer's choice; None: the cost rule), H = X^T X and G = 2 D H
        (2 C^2 T + 2 R C^2 per expert; C (C + 1) T for H's upper triangle when sym)."""
        E, R, Cc, T = self.experts, self.rows, self.cols, self.tokens
        if self.calib == "batches":
            if self.gram_route(sym) if gram is None else gram:
                h = Cc * (Cc + 1) * T if sym else 2 * Cc * Cc * T
                return E * (h + 2 * R * Cc * Cc) * self.micro
            return 4 * E * R * Cc * T * self.micro
        return 2 * E * R * Cc * Cc

    def elementwise_bytes_per_step(self) -> int:
        """Algorithmic HBM bytes of one step's fused elementwise kernels, all
        micro-batches: every pass reads the logits (4L), G (4), W (b_W) and j0
        (local shift) and writes the next D (2); the accumulator (4L) is written
        by the first pass, read and written by the middle ones and read by the
        last, which also reads and writes the momenta and writes the logits."""
        n = self.n
        if self.micro <= 1:
            return self.elementwise_bytes_per_weight() * n
        base = 4 * self.L + 4 + self.w_bytes() + 2 + (1 if self.param == "shift5" else 0)
        first = base + 4 * self.L
        middle = base + 8 * self.L
        last = base + 4 * self.L + 8 * self.L + 4 * self.L
        return (first + (self.micro - 2) * middle + last) * n


WORKLOADS = {
    w.name: w
    for w in [
        Workload(name="ternary_256x512", experts=1, rows=256, cols=512, grid=GRID_TERNARY,
                 group=128, w_dtype="f32", calib="X", tokens=256, token_dist="normal",
                 outliers=4, outlier_scale=20.0, steps=50, tau0=1.0, tau1=1.0, data_seed=1000),
        Workload(name="llama8b_q_proj", experts=1, rows=4096, cols=4096, grid=GRID_2BIT_SYM,
                 group=128, w_dtype="bf16", calib="H", tokens=128 * 2048, token_dist="normal",
                 outliers=41, outlier_scale=30.0, steps=500, tau0=1.0, tau1=0.1, data_seed=2000),
        Workload(name="llama8b_down_proj", experts=1, rows=4096, cols=14336, grid=GRID_3BIT_SYM,
                 group=128, w_dtype="bf16", calib="H", tokens=256 * 2048, token_dist="student_t3",
                 outliers=0, outlier_scale=1.0, steps=200, tau0=0.5, tau1=0.5, data_seed=3000),
        Workload(name="llama70b_gate_proj", experts=1, rows=28672, cols=8192, grid=GRID_2BIT_SYM,
                 group=64, w_dtype="bf16", calib="H", tokens=128 * 2048, token_dist="normal",
                 outliers=82, outlier_scale=30.0, steps=100, tau0=1.0, tau1=1.0, data_seed=4000,
                 pack=True),
        Workload(name="moe64_kquant3", experts=64, rows=2048, cols=7168, grid=GRID_3BIT_SYM,
                 group=16, w_dtype="bf16", calib="H", tokens=4096, token_dist="normal",
                 outliers=72, outlier_scale=30.0, steps=100, tau0=1.0, tau1=1.0,
                 scale_mode=SCALE_KQUANT2, lr_scales=0.0, data_seed=5000, pack=True),
        # The paper's own 3-bit method (§3.2 "Higher bit-widths"): the down_proj layer
        # with 5 local-shift logits per weight instead of 8.
        Workload(name="llama8b_down_proj_shift5", experts=1, rows=4096, cols=14336,
                 grid=GRID_3BIT_SYM, group=128, w_dtype="bf16", calib="H", tokens=256 * 2048,
                 token_dist="student_t3", outliers=0, outlier_scale=1.0, steps=200, tau0=0.5,
                 tau1=0.5, data_seed=3000, param="shift5"),
        # The paper's ternary method (§3.1, Alg. 2) on the q_proj layer: mask and sign
        # logits per weight, grid {-1, 0, 1}.
        Workload(name="llama8b_q_proj_mask_sign", experts=1, rows=4096, cols=4096,
                 grid=GRID_TERNARY, group=128, w_dtype="bf16", calib="H", tokens=128 * 2048,
                 token_dist="normal", outliers=41, outlier_scale=30.0, steps=500, tau0=1.0,
                 tau1=0.1, data_seed=2000, param="mask_sign"),
        # Per-step calibration tokens with gradient accumulation (§3.3): the q_proj
        # layer, one step = 8 micro-batches of 8 sequences x 4096 tokens (Table 5's
        # batch of 64 sequences), fresh noise per micro-batch.
        Workload(name="llama8b_q_proj_tokens", experts=1, rows=4096, cols=4096,
                 grid=GRID_2BIT_SYM, group=128, w_dtype="bf16", calib="batches",
                 tokens=8 * 4096, token_dist="normal", outliers=41, outlier_scale=30.0,
                 steps=500, tau0=1.0, tau1=0.1, data_seed=2000, micro=8),
    ]
}

ORDER = ["ternary_256x512", "llama8b_q_proj", "llama8b_down_proj", "llama70b_gate_proj",
         "moe64_kquant3"]


@dataclass(frozen=True)
class Shard:
    """One rank's part of a layer split across GPUs: whole experts of a
    multi-expert layer, or a contiguous block of rows of a one-expert layer
    (rows and experts are independent in Eq. 1 with a linear f, so the shards
    never exchange data).  `workload` is the shard's own layer problem; the
    input generators take `experts` and `rows` (ranges of the whole layer's
    global indices) to produce exactly its slice of W and H; `index_offset`
    is the flat index of its first weight in the whole layer, so it draws the
    whole layer's noise."""
    workload: Workload
    experts: Tuple[int, int]
    rows: Tuple[int, int]
    index_offset: int


def _block(n: int, rank: int, world: int) -> Tuple[int, int]:
    """[lo, hi) of block `rank` when n items split into `world` contiguous blocks
    whose sizes differ by at most one (the first n % world are one larger)."""
    base, extra = divmod(n, world)
    lo = rank * base + min(rank, extra)
    return lo, lo + base + (1 if rank < extra else 0)


def shard(w: Workload, rank: int, world: int) -> Shard:
    """Rank `rank` of `world`: experts split across ranks when the layer has
    several (each rank gets whole experts, every row), else rows."""
    if not 0 <= rank < world:
        raise ValueError(f"rank {rank} outside world {world}")
    if world == 1:
        return Shard(w, (0, w.experts), (0, w.rows), 0)
    if w.experts > 1:
        if w.experts < world:
            raise ValueError(f"{w.experts} experts cannot feed {world} ranks")
        e0, e1 = _block(w.experts, rank, world)
        return Shard(replace(w, experts=e1 - e0), (e0, e1), (0, w.rows), e0 * w.rows * w.cols)
    if w.rows < world:
        raise ValueError(f"{w.rows} rows cannot feed {world} ranks")
    r0, r1 = _block(w.rows, rank, world)
    return Shard(replace(w, rows=r1 - r0), (0, 1), (r0, r1), r0 * w.cols)


def shrunk(w: Workload, experts: int | None = None, rows: int | None = None,
           cols: int | None = None, tokens: int | None = None) -> Workload:
    """The same workload recipe at a smaller shape (for tests the oracle finishes in seconds)."""
    kw = {}
    if experts is not None:
        kw["experts"] = experts
    if rows is not None:
        kw["rows"] = rows
    if cols is not None:
        kw["cols"] = cols
        kw["outliers"] = min(w.outliers, max(1, cols // 100)) if w.outliers else 0
    if tokens is not None:
        kw["tokens"] = tokens
    return replace(w, **kw)
