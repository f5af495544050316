"""Device-resident state of one DAVET batch and the per-step call sequence.

Host orchestration only: this module allocates the buffers a batch needs
(pyramids, packed step input, attention output, answer state, workspace) as
torch CUDA tensors and issues the four library calls in order.  It performs no
arithmetic of its own.

Per request the pyramid buffer is level-major; its level-0 rows are where the
visual encoding is written, so the pyramid build reads the encoding in place
and writes only the pooled levels.
"""
from __future__ import annotations

import torch

from . import davet as _davet
from .workloads import Workload


class Pipeline:
    def __init__(self, w: Workload, device="cuda", lib=None):
        self.w = w
        self.dev = torch.device(device)
        self.lib = lib if lib is not None else _davet.load()
        C, B = w.C, w.batch
        self.sides = w.level_sides()
        # pyramids: one allocation, request b at row pyr_row0[b]
        rows = [w.pyramid_rows(b) for b in range(B)]
        self.pyr_row0 = [0]
        for r in rows:
            self.pyr_row0.append(self.pyr_row0[-1] + r)
        self.pyr = torch.empty((self.pyr_row0[-1], C), dtype=torch.bfloat16, device=self.dev)
        self.pyr_views = [self.pyr[self.pyr_row0[b]:self.pyr_row0[b + 1]] for b in range(B)]
        self.pyr_ptrs = torch.tensor([v.data_ptr() for v in self.pyr_views], dtype=torch.int64, device=self.dev)
        self.text = torch.empty((max(w.total_text(), 1), C), dtype=torch.bfloat16, device=self.dev)
        self.tiles = torch.tensor(w.tiles, dtype=torch.int32, device=self.dev)
        self.prompt = torch.tensor(w.prompt, dtype=torch.int32, device=self.dev)
        self.resp = torch.tensor(w.resp, dtype=torch.int32, device=self.dev)
        self.text_off = torch.from_numpy(w.text_offsets()).to(self.dev)
        self.schedule = torch.from_numpy(w.schedule).to(self.dev).contiguous()
        self.max_rows = w.max_total_rows()
        self.packed = torch.empty((self.max_rows, C), dtype=torch.bfloat16, device=self.dev)
        self.cu = torch.zeros(B + 1, dtype=torch.int32, device=self.dev)
        self.attn_out = torch.empty((self.max_rows, w.H, w.D), dtype=torch.bfloat16, device=self.dev)
        R = w.total_resp
        self.cu_resp = torch.from_numpy(w.cu_resp()).to(self.dev)
        self.masked = torch.ones(R, dtype=torch.uint8, device=self.dev)
        self.tokens = torch.full((R,), -1, dtype=torch.int32, device=self.dev)
        self.argmax = torch.full((R,), -1, dtype=torch.int32, device=self.dev)
        self.conf = torch.zeros(R, dtype=torch.float32, device=self.dev)
        self.committed = torch.full((w.T, B, w.k), -1, dtype=torch.int32, device=self.dev)
        self.stats = torch.zeros((w.T, B, 2), dtype=torch.float32, device=self.dev)
        ws = self.lib.davet_unmask_topk_workspace(R, w.V, B)
        self.workspace = torch.zeros(max(ws, 256), dtype=torch.uint8, device=self.dev)

    # -------------------------------------------------------------- inputs
    def level0(self, b: int):
        """Rows of request b's encoding inside its pyramid buffer."""
        n = self.w.tiles[b] * self.w.grid * self.w.grid
        return self.pyr_views[b][:n]

    def load_inputs(self, feats, text, non_blocking=False):
        """feats: per-request bf16 [tiles, G, G, C]; text: bf16 [sum(P+R), C]."""
        for b, f in enumerate(feats):
            self.level0(b).copy_(f.reshape(-1, self.w.C), non_blocking=non_blocking)
        if self.w.total_text():
            self.text[: self.w.total_text()].copy_(text, non_blocking=non_blocking)

    def reset_state(self):
        self.masked.fill_(1)
        self.tokens.fill_(-1)
        self.argmax.fill_(-1)

    # ---------------------------------------------------------------- path
    def build_pyramids(self, stream=None):
        w = self.w
        for b in range(w.batch):
            v = self.pyr_views[b]
            self.lib.davet_build_pyramid(v, v, w.tiles[b], w.grid, w.n_levels, w.C, None, stream)

    def gather(self, t: int, stream=None):
        w = self.w
        self.lib.davet_gather_view(self.pyr_ptrs, self.tiles, self.text, self.text_off, self.prompt, self.resp,
                                   self.schedule[t], w.batch, w.grid, w.n_levels, *w.mixed_args, w.C,
                                   self.packed, self.cu, self.max_rows, stream)

    def attention(self, stream=None):
        w = self.w
        self.lib.davet_step_attention(self.packed, self.cu, w.batch, self.max_rows, w.H, w.D, w.scale,
                                      self.attn_out, stream)

    def unmask(self, t: int, logits, stream=None):
        w = self.w
        self.lib.davet_unmask_topk(logits, w.V, self.cu_resp, w.batch, w.total_resp, w.k, self.masked,
                                   self.tokens, self.argmax, self.conf, self.committed[t], self.stats[t],
                                   self.workspace, self.workspace.numel(), stream)

    def step(self, t: int, logits, stream=None):
        self.gather(t, stream)
        self.attention(stream)
        self.unmask(t, logits, stream)
