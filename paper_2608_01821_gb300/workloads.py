"""Seeded synthetic workloads for the DAVET step-conditioning path.

This module holds sizes, level schedules and seeded input generators only; it
contains none of the method's arithmetic.  The tests feed the same generated
tensors to the CUDA library and to the CPU oracle, and the benchmark uses it to
build its inputs.

Workloads (shapes of an 8B-class diffusion VLM backbone with 32 heads of
dimension 128 and 384px tiles of 27x27 visual tokens):

  tiny     1 request, 4x64 heads, one 12x12 tile, levels 12/6/3, prompt 16,
           response 32, 8 steps with levels [0,0,1,1,2,2,1,0], vocab 1024,
           top-4 per step, seed 0
  single   1 request, one 27x27 tile, levels 27/14/7/4, prompt 64,
           response 128, 64 steps, level floor(4t/64), vocab 126464, top-2,
           seed 1
  anyres   1 request, 5 tiles, prompt 128, response 256, 128 steps, level 0
           for t < 32 then level 2, top-2, seed 2
  highres  4 requests, 10 tiles each, prompt 256, response 512, 256 steps,
           level 2 for t < 224 then level 0, top-2, seed 3
  ragged   16 requests, tiles U{1..9}, prompt U{32..256}, response
           U{64..512}, 128 steps, level drawn per (step, request) from
           {0,1,2,3} with p = [0.25, 0.25, 0.30, 0.20], top-2, seed 4

Two more exercise the mixed view (coarse level 2 plus a centred stride-3
lattice of level-0 tokens, selected as view index n_levels):

  tiny_mixed    tiny with views [0,0,3,3,2,2,3,0] (3 = mixed, 25 rows)
  single_mixed  single with coarse / mixed / high thirds over 64 steps
                (49 / 130 / 729 visual rows)

Per-token channel count C = 3*H*D: each visual and text row carries the
packed [query | key | value] projections of its token, so a gathered row is
exactly one row of the attention input (pooling commutes with the linear
projection, so pooling the projected rows equals projecting pooled rows).

Value recipe: features, text rows ~ N(0, 1); logits ~ N(0, 2) (variance 2);
all rounded to bf16 (round to nearest even).  Each tensor has its own
torch.Generator seeded from (workload seed, tensor kind, index) through
splitmix64, so every tensor is reproducible on its own.  Integer workload
parameters of the ragged mix come from one splitmix64 stream (seed 4): the
per-request (tiles, prompt, response) triples first, request by request, then
the level schedule in step-major order.
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

MASK64 = (1 << 64) - 1
VOCAB_8B = 126464


def splitmix64(state: int) -> tuple[int, int]:
    """One step of splitmix64 (Steele, Lea, Flood 2014): (new_state, output)."""
    state = (state + 0x9E3779B97F4A7C15) & MASK64
    z = state
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & MASK64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & MASK64
    return state, z ^ (z >> 31)


class SplitMix64:
    def __init__(self, seed: int):
        self.state = seed & MASK64

    def next(self) -> int:
        self.state, out = splitmix64(self.state)
        return out

    def uniform_int(self, lo: int, hi: int) -> int:
        """Integer in [lo, hi] (modulo reduction; bias < 2^-50 here)."""
        return lo + self.next() % (hi - lo + 1)

    def uniform01(self) -> float:
        return (self.next() >> 11) * (1.0 / (1 << 53))


def derive_seed(*parts: int) -> int:
    s = 0x5DEECE66D
    for p in parts:
        s, _ = splitmix64(s ^ (p & MASK64))
        _, s = splitmix64(s)
    return s & ((1 << 63) - 1)


# tensor kinds for derive_seed
KIND_FEAT, KIND_TEXT, KIND_LOGITS, KIND_QKV, KIND_SCORE = 1, 2, 3, 4, 5


@dataclasses.dataclass
class Workload:
    name: str
    batch: int
    H: int
    D: int
    grid: int
    n_levels: int
    tiles: list[int]
    prompt: list[int]
    resp: list[int]
    T: int
    schedule: np.ndarray  # int32 [T, batch]
    V: int
    k: int
    seed: int
    # mixed view (coarse pyramid level, lattice stride), selected as view
    # index n_levels; None when the workload has no mixed view
    mixed: tuple[int, int] | None = None

    @property
    def C(self) -> int:
        return 3 * self.H * self.D

    @property
    def scale(self) -> float:
        return 1.0 / math.sqrt(self.D)

    def level_sides(self) -> list[int]:
        out, g = [], self.grid
        for _ in range(self.n_levels):
            out.append(g)
            g = (g + 1) // 2
        return out

    def pyramid_rows(self, b: int) -> int:
        return self.tiles[b] * sum(g * g for g in self.level_sides())

    @property
    def mixed_args(self) -> tuple[int, int]:
        """(mixed_level, mixed_stride) as the gather takes them; (0, 0) = none."""
        return self.mixed if self.mixed else (0, 0)

    def view_rows_per_tile(self, level: int) -> int:
        """Rows per tile of view `level`: a pyramid level, or the mixed view
        (index n_levels): the coarse level plus the centred lattice."""
        if level < self.n_levels:
            return self.level_sides()[level] ** 2
        assert level == self.n_levels and self.mixed, level
        coarse, s = self.mixed
        n = len(range(s // 2, self.grid, s))
        return self.level_sides()[coarse] ** 2 + n * n

    def sim_channels(self) -> tuple[int, int]:
        """(first channel, count) the merging realizer measures similarity on:
        the key slice [H*D, 2*H*D) of each packed [q | k | v] row."""
        return self.H * self.D, self.H * self.D

    def n_views(self) -> int:
        return self.n_levels + (1 if self.mixed else 0)

    def seq_len(self, b: int, level: int) -> int:
        return self.tiles[b] * self.view_rows_per_tile(level) + self.prompt[b] + self.resp[b]

    def step_lengths(self, t: int) -> list[int]:
        return [self.seq_len(b, int(self.schedule[t, b])) for b in range(self.batch)]

    def max_total_rows(self) -> int:
        return sum(max(self.seq_len(b, v) for v in range(self.n_views())) for b in range(self.batch))

    @property
    def total_resp(self) -> int:
        return sum(self.resp)

    def cu_resp(self) -> np.ndarray:
        return np.concatenate([[0], np.cumsum(self.resp)]).astype(np.int32)

    def text_offsets(self) -> np.ndarray:
        n = [p + r for p, r in zip(self.prompt, self.resp)]
        return np.concatenate([[0], np.cumsum(n)[:-1]]).astype(np.int64)

    def total_text(self) -> int:
        return sum(p + r for p, r in zip(self.prompt, self.resp))

    # ------------------------------------------------------ algorithmic work
    def attention_flops(self, t: int) -> float:
        """4 L^2 H D per request (two GEMMs of 2 L^2 D flops per head)."""
        return float(sum(4.0 * L * L * self.H * self.D for L in self.step_lengths(t)))

    def gather_bytes(self, t: int) -> float:
        """Read + write of every packed row (bf16)."""
        return 2.0 * sum(self.step_lengths(t)) * self.C * 2

    def pyramid_bytes(self) -> float:
        """Read level 0 + write levels >= 1 (bf16), all requests."""
        sides = self.level_sides()
        rows_in = sum(self.tiles) * sides[0] ** 2
        rows_out = sum(self.tiles) * sum(g * g for g in sides[1:])
        return float((rows_in + rows_out) * self.C * 2)

    def view_fill_bytes(self) -> float:
        """Bytes the view-block fill moves (read + write, bf16): every view
        block's copy of the request's text rows, and the mixed view's rows."""
        rows = 0
        for b in range(self.batch):
            rows += self.n_views() * (self.prompt[b] + self.resp[b])
            if self.mixed:
                rows += self.tiles[b] * self.view_rows_per_tile(self.n_levels)
        return float(rows * self.C * 2 * 2)

    def masked_rows(self, t: int) -> int:
        """|M_t| summed over requests when k positions are committed per step."""
        return sum(max(r - self.k * t, 0) for r in self.resp)

    def unmask_bytes(self, t: int) -> float:
        """Logit bytes of the masked rows (bf16)."""
        return float(self.masked_rows(t) * self.V * 2)


def _sched_const(T, batch, fn):
    s = np.empty((T, batch), dtype=np.int32)
    for t in range(T):
        s[t, :] = fn(t)
    return s


def make(name: str) -> Workload:
    if name == "tiny":
        return Workload("tiny", 1, 4, 64, 12, 3, [1], [16], [32], 8,
                        np.array([[0], [0], [1], [1], [2], [2], [1], [0]], dtype=np.int32),
                        1024, 4, 0)
    if name == "single":
        # level ramps 0 -> 3 linearly over 64 steps: 16 steps at each level
        return Workload("single", 1, 32, 128, 27, 4, [1], [64], [128], 64,
                        _sched_const(64, 1, lambda t: (4 * t) // 64), VOCAB_8B, 2, 1)
    if name == "anyres":
        return Workload("anyres", 1, 32, 128, 27, 4, [5], [128], [256], 128,
                        _sched_const(128, 1, lambda t: 0 if t < 32 else 2), VOCAB_8B, 2, 2)
    if name == "highres":
        return Workload("highres", 4, 32, 128, 27, 4, [10] * 4, [256] * 4, [512] * 4, 256,
                        _sched_const(256, 4, lambda t: 2 if t < 224 else 0), VOCAB_8B, 2, 3)
    if name == "ragged":
        rng = SplitMix64(4)
        tiles, prompt, resp = [], [], []
        for _ in range(16):
            tiles.append(rng.uniform_int(1, 9))
            prompt.append(rng.uniform_int(32, 256))
            resp.append(rng.uniform_int(64, 512))
        cum = [0.25, 0.50, 0.80, 1.00]
        sched = np.empty((128, 16), dtype=np.int32)
        for t in range(128):
            for b in range(16):
                u = rng.uniform01()
                sched[t, b] = next(i for i, c in enumerate(cum) if u < c)
        return Workload("ragged", 16, 32, 128, 27, 4, tiles, prompt, resp, 128, sched,
                        VOCAB_8B, 2, 4)
    if name == "tiny_mixed":
        # coarse (level 2, 9 rows), mixed (index 3: level 2 + the 4x4 lattice of
        # stride 3, 25 rows) and high (level 0, 144 rows)
        return Workload("tiny_mixed", 1, 4, 64, 12, 3, [1], [16], [32], 8,
                        np.array([[0], [0], [3], [3], [2], [2], [3], [0]], dtype=np.int32),
                        1024, 4, 0, mixed=(2, 3))
    if name == "single_mixed":
        # the three-view hierarchy on one 27x27 tile: coarse (level 2, 49 rows)
        # for t < 22, mixed (index 4: level 2 + the 9x9 lattice of stride 3,
        # 130 rows) for t < 43, then high (level 0, 729 rows)
        return Workload("single_mixed", 1, 32, 128, 27, 4, [1], [64], [128], 64,
                        _sched_const(64, 1, lambda t: 2 if t < 22 else (4 if t < 43 else 0)), VOCAB_8B, 2, 1,
                        mixed=(2, 3))
    raise ValueError(f"unknown workload {name!r}")


NAMES = ("tiny", "single", "anyres", "highres", "ragged")
MIXED_NAMES = ("tiny_mixed", "single_mixed")


# ------------------------------------------------------------ value sources
def normal_bf16(shape, seed: int, sigma: float = 1.0):
    """bf16 CPU tensor ~ N(0, sigma^2), reproducible from `seed`."""
    import torch
    g = torch.Generator(device="cpu")
    g.manual_seed(int(seed))
    x = torch.randn(tuple(shape), generator=g, dtype=torch.float32)
    if sigma != 1.0:
        x.mul_(sigma)
    return x.to(torch.bfloat16)


def features(w: Workload, b: int):
    """Visual tokens of request b: bf16 [tiles, G, G, C] ~ N(0,1)."""
    return normal_bf16((w.tiles[b], w.grid, w.grid, w.C), derive_seed(w.seed, KIND_FEAT, b))


def text_rows(w: Workload):
    """Prompt and response rows of all requests, request-major: bf16 [sum(P+R), C]."""
    import torch
    parts = [normal_bf16((w.prompt[b] + w.resp[b], w.C), derive_seed(w.seed, KIND_TEXT, b))
             for b in range(w.batch)]
    return torch.cat(parts, 0)


# Operation demand prior d(o) of the five operation categories (Table A:
# lexical readout, numerical reasoning, entity grounding, binary decision,
# general understanding).  The query parser that assigns a category is not
# part of this path; requests take the categories in turn.
DEMAND_PRIOR = (1.000, 0.941, 0.824, 0.647, 0.529)


def request_demands(w: Workload) -> list[float]:
    """d(o) of every request (categories assigned in turn, request b -> b mod 5)."""
    return [DEMAND_PRIOR[b % len(DEMAND_PRIOR)] for b in range(w.batch)]


def set_static_view(w: Workload, which: str) -> None:
    """Replace the level schedule by one view for every step and request:
    'high' (level 0), 'mid' or 'low' (the policy's other two views)."""
    lv = dict(zip(("low", "mid", "high"), policy_view_levels(w)))[which]
    w.schedule = np.full_like(w.schedule, lv)


def policy_view_levels(w: Workload) -> list[int]:
    """The views the allocation policy picks among, as the gather numbers
    them: [low, mid, high] = [pyramid level 2 (or the coarsest), the mixed
    view (or level 1), level 0]."""
    return [min(2, w.n_levels - 1), w.n_levels if w.mixed else 1, 0]


def token_scores(w: Workload, b: int):
    """Importance score of every visual token of request b for the pruning
    realizer (the paper leaves the score open): fp32 [tiles, G*G] ~ N(0,1)."""
    import torch
    g = torch.Generator(device="cpu")
    g.manual_seed(derive_seed(w.seed, KIND_SCORE, b))
    return torch.randn((w.tiles[b], w.grid * w.grid), generator=g, dtype=torch.float32)


def logits(w: Workload, t: int):
    """Step-t logits of all answer rows: bf16 [sum(R), V] ~ N(0, 2)."""
    return normal_bf16((w.total_resp, w.V), derive_seed(w.seed, KIND_LOGITS, t), math.sqrt(2.0))


def logits_device(w: Workload, t: int, device, out=None):
    """Device-generated step-t logits for timing runs (torch's device RNG,
    seeded per step; not bit-identical to `logits`)."""
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(derive_seed(w.seed, KIND_LOGITS, t))
    if out is None:
        out = torch.empty((w.total_resp, w.V), dtype=torch.bfloat16, device=device)
    tmp = torch.randn(out.shape, generator=g, dtype=torch.float32, device=device)
    out.copy_(tmp.mul_(math.sqrt(2.0)))
    return out


def qkv_rows(n_rows: int, H: int, D: int, seed: int):
    """Stand-alone attention input bf16 [n_rows, 3, H, D] ~ N(0,1)."""
    return normal_bf16((n_rows, 3, H, D), derive_seed(seed, KIND_QKV, n_rows))
