"""The synthetic forecast workloads and their sampling schedules.

Shapes follow the DiT families the paper evaluates (Sec. 4.1): DiT-XL/2 class-to-image,
PixArt text-to-image, a large MMDiT text-to-image model and HunyuanVideo-class
text-to-video, each cached as a list of per-block feature tensors, plus the many-tensor
blockwise cache of Sec. 4.5.  Values are synthetic
(no model weights): per-element random polynomial trajectories in time plus noise
(:mod:`.synth`).  The schedule is the equal-spaced one of Sec. 3.3: a full step every
``interval`` steps, plus the first K steps to fill the window; every other step is a cache
forward that forecasts from the K most recent full steps (the sliding window of Eq. 6).
"""
from __future__ import annotations

from dataclasses import dataclass, field
from math import prod

DTYPE_F32, DTYPE_BF16 = 0, 1


@dataclass(frozen=True)
class Problem:
    """One skipped step: forecast at `t` from `nodes` (newest first)."""
    step: int
    t: float
    nodes: tuple[float, ...]
    node_steps: tuple[int, ...]
    dt: float  # t_next - t (Euler step to the following timestep)


@dataclass(frozen=True)
class Workload:
    name: str
    layer_shape: tuple[int, ...]
    n_layers: int
    dtype: int
    K: int
    steps: int
    interval: int
    time_kind: str            # "ddim": t = 980 - 20 i (1000-step model); "flow": t = 1 - i/steps
    degree: int               # polynomial degree of the synthetic trajectories
    noise_std: float
    outlier_frac: float = 0.0
    outlier_scale: float = 10.0
    euler_shape: tuple[int, ...] | None = None
    fixed_problem: tuple | None = None   # (t, nodes newest first) when the config names them
    K_sweep: tuple[int, ...] = field(default_factory=tuple)

    # ---- sizes
    @property
    def layer_numel(self) -> int:
        return prod(self.layer_shape)

    @property
    def numels(self) -> list[int]:
        n = [self.layer_numel] * self.n_layers
        if self.euler_shape:
            n.append(prod(self.euler_shape))
        return n

    @property
    def elem_bytes(self) -> int:
        return 2 if self.dtype == DTYPE_BF16 else 4

    @property
    def hidden(self) -> int:
        return self.layer_shape[-1]

    # ---- schedule
    def times(self) -> list[float]:
        if self.time_kind == "ddim":
            return [980.0 - 20.0 * i for i in range(self.steps)]
        return [1.0 - i / self.steps for i in range(self.steps)]

    def tau(self, t: float) -> float:
        """Normalised time for synthesising values (keeps trajectories O(1))."""
        return t / 1000.0 if self.time_kind == "ddim" else t

    def is_full(self, i: int, K: int | None = None) -> bool:
        K = self.K if K is None else K
        return i < K or i % self.interval == 0

    def problems(self, K: int | None = None) -> list[Problem]:
        """Every skipped step of the schedule with a full window of K nodes."""
        K = self.K if K is None else K
        ts = self.times()
        out, full = [], []
        for i, t in enumerate(ts):
            if self.is_full(i, K):
                full.append(i)
                continue
            if len(full) < K:
                continue
            node_steps = tuple(reversed(full[-K:]))
            t_next = ts[i + 1] if i + 1 < len(ts) else 0.0
            out.append(Problem(i, t, tuple(ts[j] for j in node_steps), node_steps, t_next - t))
        return out

    def representative(self, K: int | None = None) -> Problem:
        """The forecast measured and checked for this workload: the config's named nodes,
        else the first skipped step in the second half of the schedule."""
        K = self.K if K is None else K
        if self.fixed_problem is not None:
            t, nodes = self.fixed_problem
            return Problem(-1, t, tuple(nodes), (), 0.0)
        probs = self.problems(K)
        for p in probs:
            if p.step >= self.steps // 2:
                return p
        return probs[-1]

    # ---- bytes
    def cache_bytes(self, K: int | None = None) -> int:
        K = self.K if K is None else K
        per_slot = sum((n * self.elem_bytes + 255) // 256 * 256 for n in self.numels)
        return K * per_slot

    def forecast_bytes(self, K: int | None = None, out_elem_bytes: int | None = None,
                       x_elem_bytes: int = 4) -> int:
        """Algorithmic HBM bytes of one forecast: K reads + 1 write per element (+ the
        Euler state read and write for the fused step)."""
        K = self.K if K is None else K
        ob = self.elem_bytes if out_elem_bytes is None else out_elem_bytes
        n_feat = self.layer_numel * self.n_layers
        b = (K * self.elem_bytes + ob) * n_feat
        if self.euler_shape:
            nv = prod(self.euler_shape)
            b += K * self.elem_bytes * nv + 2 * x_elem_bytes * nv
        return b


WORKLOADS: dict[str, Workload] = {
    # DiT-XL/2 256 px: one cached tensor [B=2, 256 tokens, 1152] fp32, K = 3,
    # nodes t = 980, 960, 940 of DDIM-50, forecast at 920; quadratic trajectories.
    "c2i-256": Workload("c2i-256", (2, 256, 1152), 1, DTYPE_F32, 3, 50, 3, "ddim", 2, 1e-3,
                        fixed_problem=(920.0, (940.0, 960.0, 980.0))),
    # DiT-XL/2 512 px: 28 block outputs [8, 1024, 1152] bf16, K = 4, DDIM-50, full every
    # 3rd step; smooth cubic trajectories.
    "c2i-512": Workload("c2i-512", (8, 1024, 1152), 28, DTYPE_BF16, 4, 50, 3, "ddim", 3, 1e-2),
    # PixArt 1024 px: 28 block outputs [4, 4096, 1152] bf16, K = 3, 20-step flow schedule,
    # quadratic trajectories, 1 % of channels at 10x amplitude.
    "t2i-1024": Workload("t2i-1024", (4, 4096, 1152), 28, DTYPE_BF16, 3, 20, 3, "flow", 2,
                         5e-3, outlier_frac=0.01, outlier_scale=10.0),
    # Large MMDiT: 57 block outputs [1, 4608, 3072] bf16 + the velocity [1, 16, 128, 128]
    # forecast fused with the Euler update; K = 3, 28-step flow schedule.
    "mmdit-t2i": Workload("mmdit-t2i", (1, 4608, 3072), 57, DTYPE_BF16, 3, 28, 3, "flow", 2,
                          5e-3, euler_shape=(1, 16, 128, 128)),
    # Video DiT: 60 block outputs [1, 33*45*80 = 118800 tokens, 3072] bf16, K swept over
    # 2..4, 50-step flow schedule forecasting 2 of every 3 steps.
    "t2v": Workload("t2v", (1, 118800, 3072), 60, DTYPE_BF16, 3, 50, 3, "flow", 2, 1e-2,
                    K_sweep=(2, 3, 4)),
    # Blockwise (module-level) cache of Sec. 4.5 / Tables 5-6: many small tensors instead of
    # one per block -- 4096 tensors of 65,536 bf16 elements, K = 3 (1.6 GB of cache), the
    # per-tensor forecast of every one in one launch.
    "blockwise": Workload("blockwise", (65536,), 4096, DTYPE_BF16, 3, 20, 3, "flow", 2, 1e-2),
}

# Device-memory budget of the video workload (cache + forecast output) stated with it.
T2V_HBM_BUDGET = 180 * 10**9
