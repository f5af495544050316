"""Full backbone step with synthetic weights: host orchestration only.

Every denoising step (Sec. 3.1, Eq. 1-2) runs the whole backbone over the
step sequence [v_t || q || y^(t-1)]: the step's view rows and prompt rows
come from the evidence pyramid and the text store (davet_gather_view), the
answer rows are the embeddings of the current answer state (committed token
or the mask token; davet_embed_answers); then `n_layers` pre-normalization
layers (davet_linear with the rotary / residual / gated-MLP epilogues,
davet_step_attention), the final normalization of the answer rows
(davet_rmsnorm) and the LM head give the logits that davet_unmask_topk
commits from.  The rows carry hidden states of width C = H * D; the MLP
width is 3C.

The two normalizations of a layer are folded into the projections that
read them: the gains are multiplied into the QKV and gate/up weights once,
the residual projections (output, down) also emit each row's partial sums of
squares, and the next projection scales its product rows by 1 / rms (for the
first layer the sums come from davet_row_sumsq).  rmsnorm(x) W^T =
(x (W diag g)^T) / rms(x), so no normalized copy of x is written or read.

Each step's view comes either from the workload's schedule (known on the
host, so every launch is sized to the step's rows) or, after use_policy(),
from the allocation policy (Eq. 6-9) on the device, fed by the previous
step's unmasking statistics.  Then the row count exists only on the device
(cu_seqlens[batch] after the gather): the norms and projections are launched
for the largest view and read the count when they start, so a captured pass
runs whatever views the policy picks without a host round trip.

Weights are random (no checkpoint is available): each matrix ~ N(0, 1/fan_in),
normalization gains ~ 1 + N(0, 0.1^2), drawn on the device from torch
generators seeded per tensor.  This module performs no arithmetic of its own.
"""
from __future__ import annotations

import torch

from . import davet as _davet
from .workloads import Workload, derive_seed, policy_view_levels, request_demands

KIND_WEIGHT = 16
ROPE_THETA = 500000.0
RMS_EPS = 1e-5


class Backbone:
    def __init__(self, w: Workload, n_layers: int, device="cuda", lib=None, mask_id: int | None = None):
        self.w = w
        self.L = n_layers
        self.dev = torch.device(device)
        self.lib = lib if lib is not None else _davet.load()
        H, D = w.H, w.D
        self.C = C = H * D
        self.F = F = 3 * C
        self.HD = H * D
        self.V = w.V
        self.mask_id = w.V - 1 if mask_id is None else mask_id
        if C % 256 or F % 128 or w.V % 256:
            raise ValueError("hidden width and vocabulary must be multiples of 256, the MLP width of 128")
        dev = self.dev
        seed = w.seed

        def rnd(shape, k, std):
            g = torch.Generator(device=dev)
            g.manual_seed(derive_seed(seed, KIND_WEIGHT + k, 0))
            return (torch.randn(shape, generator=g, device=dev, dtype=torch.float32) * std).to(torch.bfloat16)

        def gain(k):
            return (1.0 + rnd((C,), k, 0.1).float()).to(torch.bfloat16)

        def fold(wt, g):  # W diag(g), rounded to bf16 once
            return (wt.float() * g.float()[None, :]).to(torch.bfloat16)

        self.layers = []
        for l in range(n_layers):
            base = 16 * (l + 1)
            wg = rnd((F, C), base + 4, C ** -0.5)
            wu = rnd((F, C), base + 5, C ** -0.5)
            g1, g2 = gain(base + 0), gain(base + 3)
            self.layers.append(dict(
                g1=g1,
                g2=g2,
                # the normalization gains folded in: wqkv = Wqkv diag(g1), wgu = Wgu diag(g2)
                wqkv=fold(rnd((3 * self.HD, C), base + 1, C ** -0.5), g1),
                wo=rnd((C, self.HD), base + 2, self.HD ** -0.5),
                # gate and up rows interleaved in blocks of 128 (the gated-MLP epilogue's layout)
                wgu=fold(torch.stack([wg.reshape(F // 128, 128, C), wu.reshape(F // 128, 128, C)], 1)
                         .reshape(2 * F, C), g2).contiguous(),
                wd=rnd((C, F), base + 6, F ** -0.5),
            ))
            del wg, wu
        self.gf = gain(1)
        self.wlm = rnd((w.V, C), 2, C ** -0.5)
        self.emb = rnd((w.V, C), 3, 1.0)

        # the evidence pyramids of the hidden rows (level-major, one buffer per request) and the prompt rows
        self.pyr = [torch.empty((max(w.tiles[b] * sum(g * g for g in w.level_sides()), 1), C), dtype=torch.bfloat16,
                                device=dev) for b in range(w.batch)]
        self.pyr_ptrs = torch.tensor([p.data_ptr() for p in self.pyr], dtype=torch.int64, device=dev)
        self.text = torch.zeros((max(w.total_text(), 1), C), dtype=torch.bfloat16, device=dev)
        self.tiles = torch.tensor(w.tiles, dtype=torch.int32, device=dev)
        self.prompt = torch.tensor(w.prompt, dtype=torch.int32, device=dev)
        self.resp = torch.tensor(w.resp, dtype=torch.int32, device=dev)
        self.text_off = torch.from_numpy(w.text_offsets()).to(dev)
        self.schedule = torch.from_numpy(w.schedule).to(dev).contiguous()
        self.max_rows = w.max_total_rows()
        R = w.total_resp
        self.R = R
        self.cu = torch.zeros(w.batch + 1, dtype=torch.int32, device=dev)
        self.cu_resp = torch.from_numpy(w.cu_resp()).to(dev)
        self.x = torch.empty((self.max_rows, C), dtype=torch.bfloat16, device=dev)
        # partial sums of squares of x's rows: from the input (one part) and
        # from the residual projections (one part per 256 columns)
        self.ss_in = torch.empty((self.max_rows, 1), dtype=torch.float32, device=dev)
        self.ss_parts = C // 256
        self.ss = [torch.empty((self.max_rows, self.ss_parts), dtype=torch.float32, device=dev) for _ in range(2)]
        self.qkv = torch.empty((self.max_rows, 3 * self.HD), dtype=torch.bfloat16, device=dev)
        self.att = torch.empty((self.max_rows, self.HD), dtype=torch.bfloat16, device=dev)
        self.a = torch.empty((self.max_rows, F), dtype=torch.bfloat16, device=dev)
        self.xa = torch.empty((max(R, 1), C), dtype=torch.bfloat16, device=dev)
        self.logits = torch.empty((max(R, 1), w.V), dtype=torch.bfloat16, device=dev)
        self.max_pos = max(max(w.seq_len(b, v) for v in range(w.n_views())) for b in range(w.batch))
        self.rope = torch.empty((D // 2, self.max_pos, 2), dtype=torch.float32, device=dev)
        self.lib.davet_rope_table(self.max_pos, D, ROPE_THETA, self.rope)
        self.masked = torch.ones(R, dtype=torch.uint8, device=dev)
        self.tokens = torch.full((R,), -1, dtype=torch.int32, device=dev)
        self.argmax = torch.full((R,), -1, dtype=torch.int32, device=dev)
        self.conf = torch.zeros(R, dtype=torch.float32, device=dev)
        self.committed = torch.full((w.T, w.batch, w.k), -1, dtype=torch.int32, device=dev)
        self.stats = torch.zeros((w.T, w.batch, 2), dtype=torch.float32, device=dev)
        ws = self.lib.davet_unmask_topk_workspace(R, w.V, w.batch)
        self.workspace = torch.zeros(max(ws, 256), dtype=torch.uint8, device=dev)
        # scratch of the projections' K split (steps with few rows)
        shapes = [(C, 3 * self.HD), (self.HD, C), (C, 2 * F), (F, C), (C, w.V)]
        rows = {self.rows(t) for t in range(w.T)} | {R, self.max_rows}
        gw = max(self.lib.davet_linear_workspace_bytes(m, k, n) for k, n in shapes for m in rows)
        self.gemm_ws = torch.empty(max(gw, 256), dtype=torch.uint8, device=dev)
        self.policy = None

    def use_policy(self, orientation: str = "early", B: float = 0.75, rho: float = 0.2, alpha: float = 1.0,
                   uniform_demand: bool = False):
        """Choose every step's view with the closed-loop allocation policy:
        the budget envelope (Eq. 6-7) at the start of each pass, the view of
        step t from step t-1's unmasking statistics (Eq. 8-9).  The demand
        prior d(o) comes from Table A by request, or is 1 for every request
        (uniform_demand, the paper's ablation of the prior)."""
        if orientation not in ("early", "late"):
            raise ValueError("orientation is 'early' or 'late'")
        w, dev = self.w, self.dev
        self.policy = dict(orientation=orientation, B=B, rho=rho, alpha=alpha, view_levels=policy_view_levels(w))
        self.lo = torch.empty((w.batch, w.T), dtype=torch.float64, device=dev)
        self.up = torch.empty_like(self.lo)
        self.demand = None if uniform_demand else torch.tensor(request_demands(w), dtype=torch.float64, device=dev)
        self.budget = torch.zeros((w.T, w.batch), dtype=torch.float64, device=dev)

    # -------------------------------------------------------------- inputs
    def load_inputs(self, feats, prompts, non_blocking=False):
        """feats: per-request bf16 [tiles, G, G, C] visual hidden states;
        prompts: per-request bf16 [P_b, C] prompt embeddings."""
        w = self.w
        for b, f in enumerate(feats):
            if w.tiles[b]:
                self.pyr[b][: f.numel() // self.C].copy_(f.reshape(-1, self.C), non_blocking=non_blocking)
        off = w.text_offsets()
        for b, p in enumerate(prompts):
            if w.prompt[b]:
                self.text[int(off[b]): int(off[b]) + w.prompt[b]].copy_(p, non_blocking=non_blocking)

    def reset_state(self):
        self.masked.fill_(1)
        self.tokens.fill_(-1)
        self.argmax.fill_(-1)

    def begin_pass(self, stream=None):
        """Fresh answer state; with the policy, the pass's budget envelope."""
        self.reset_state()
        if self.policy:
            pol = self.policy
            self.lib.davet_policy_envelope(self.w.T, 0 if pol["orientation"] == "early" else 1, pol["B"], pol["rho"],
                                           self.demand, self.w.batch, self.lo, self.up, stream)

    def build_pyramids(self, stream=None):
        w = self.w
        for b in range(w.batch):
            self.lib.davet_build_pyramid(self.pyr[b], self.pyr[b], w.tiles[b], w.grid, w.n_levels, self.C, None,
                                         stream)

    # ---------------------------------------------------------------- path
    def rows(self, t: int) -> int:
        """Rows of step t's packed sequence under the workload's schedule."""
        return int(sum(self.w.step_lengths(t)))

    def rows_of(self, levels) -> int:
        """Rows of a step whose requests take the views `levels`."""
        return int(sum(self.w.seq_len(b, int(v)) for b, v in enumerate(levels)))

    def forward(self, t: int, stream=None, timed=None):
        """Step t's input rows and every layer; leaves the answer logits.
        `timed(kind, fn)`, if given, runs each library call (for per-kernel
        timing); kind is "input", "norm", "gemm" or "attention"."""
        w, lib = self.w, self.lib
        run = timed if timed is not None else (lambda kind, fn: fn())
        if self.policy:
            N, nd = self.max_rows, self.cu[w.batch:]  # the count the gather writes
        else:
            N, nd = self.rows(t), None
        C, HD, F = self.C, self.HD, self.F
        ws = self.gemm_ws
        run("input", lambda: lib.davet_gather_view(self.pyr_ptrs, self.tiles, self.text, self.text_off, self.prompt,
                                                   self.resp, self.schedule[t], w.batch, w.grid, w.n_levels,
                                                   *w.mixed_args, C, self.x, self.cu, self.max_rows, stream))
        run("input", lambda: lib.davet_embed_answers(self.emb, w.V, C, self.tokens, self.mask_id, self.cu,
                                                     self.cu_resp, w.batch, self.R, self.x, stream))
        run("norm", lambda: lib.davet_row_sumsq(self.x, N, C, self.ss_in, rows_dev=nd, stream=stream))
        sa, sb, parts = self.ss[0], self.ss[1], self.ss_parts
        for i, p in enumerate(self.layers):
            ss, sp = (self.ss_in, 1) if i == 0 else (sb, parts)
            run("gemm", lambda: lib.davet_linear(self.x, N, C, p["wqkv"], 3 * HD, self.qkv, lib.EPI_ROPE, None,
                                                 self.cu, w.batch, 2 * HD, w.D, self.rope, self.max_pos, ws,
                                                 row_ss=ss, row_ss_parts=sp, row_ss_eps=RMS_EPS, rows_dev=nd,
                                                 stream=stream))
            run("attention", lambda: lib.davet_step_attention(self.qkv, self.cu, w.batch, self.max_rows, w.H, w.D,
                                                              w.scale, self.att, stream))
            run("gemm", lambda: lib.davet_linear(self.att, N, HD, p["wo"], C, self.x, lib.EPI_RESIDUAL, self.x,
                                                 workspace=ws, ss_out=sa, rows_dev=nd, stream=stream))
            run("gemm", lambda: lib.davet_linear(self.x, N, C, p["wgu"], 2 * F, self.a, lib.EPI_SWIGLU,
                                                 workspace=ws, row_ss=sa, row_ss_parts=parts, row_ss_eps=RMS_EPS,
                                                 rows_dev=nd, stream=stream))
            run("gemm", lambda: lib.davet_linear(self.a, N, F, p["wd"], C, self.x, lib.EPI_RESIDUAL, self.x,
                                                 workspace=ws, ss_out=sb, rows_dev=nd, stream=stream))
        run("norm", lambda: lib.davet_rmsnorm(self.x, self.R, C, self.gf, RMS_EPS, self.xa, self.cu, self.cu_resp,
                                              w.batch, stream))
        run("gemm", lambda: lib.davet_linear(self.xa, self.R, C, self.wlm, w.V, self.logits, workspace=ws,
                                             stream=stream))

    def step(self, t: int, stream=None, timed=None):
        w = self.w
        run = timed if timed is not None else (lambda kind, fn: fn())
        torch.cuda.nvtx.range_push(f"backbone step {t}")
        if self.policy:
            pol = self.policy
            run("policy", lambda: self.lib.davet_policy_step(t, w.T, self.lo, self.up,
                                                             self.stats[t - 1] if t else None, w.batch, pol["alpha"],
                                                             pol["view_levels"], self.schedule[t], self.budget[t],
                                                             stream))
        self.forward(t, stream, timed)
        run("unmask", lambda: self.lib.davet_unmask_topk(self.logits, w.V, self.cu_resp, w.batch, self.R, w.k,
                                                         self.masked, self.tokens, self.argmax, self.conf,
                                                         self.committed[t], self.stats[t], self.workspace,
                                                         stream=stream))
        torch.cuda.nvtx.range_pop()

    # ---------------------------------------------------- accounting (host)
    def gemm_flops(self, t: int, N: int | None = None) -> float:
        """Tensor-core FLOPs of step t's projections and LM head (N rows;
        default: the workload's schedule)."""
        N = self.rows(t) if N is None else N
        C, HD, F = self.C, self.HD, self.F
        per_layer = 2.0 * N * C * (3 * HD) + 2.0 * N * HD * C + 2.0 * N * C * (2 * F) + 2.0 * N * F * C
        return self.L * per_layer + 2.0 * self.R * C * self.w.V

    def gemm_launches(self, t: int) -> int:
        """Kernels of step t's projections: one per GEMM, two where K is split."""
        N = self.max_rows if self.policy else self.rows(t)
        C, HD, F = self.C, self.HD, self.F

        def k(m, kk, n):
            return 2 if self.lib.davet_linear_workspace_bytes(m, kk, n) > 0 else 1

        per_layer = k(N, C, 3 * HD) + k(N, HD, C) + k(N, C, 2 * F) + k(N, F, C)
        return self.L * per_layer + k(self.R, C, self.w.V)

    def launches(self, t: int) -> int:
        """Kernels of step t: gather, embedding, the input's sums of squares,
        per layer the attention, the projections, the final norm, two unmask
        kernels; with the policy, its step kernel."""
        return 3 + self.L + self.gemm_launches(t) + 1 + 2 + (1 if self.policy else 0)
