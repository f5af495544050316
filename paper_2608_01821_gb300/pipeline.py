"""Device-resident state of one DAVET batch and the per-step call sequence.

Host orchestration only: this module allocates the buffers a batch needs
(pyramids or view blocks, step input, attention output, answer state,
workspace) as torch CUDA tensors and issues the library calls in order.  It
performs no arithmetic of its own.

Two layouts:
  fused (default)  each request's buffer holds view blocks [view || text]
                   (davet_build_views), and a step is davet_view_attention,
                   which reads each request's sequence from the block of its
                   step view, then the unmasking;
  unfused          each request's buffer is its level-major pyramid, text
                   rows live apart, and a step is davet_gather_view (packing
                   the step input), davet_step_attention, then the unmasking.
In both, the encoding is written where level 0 lives (the first rows of the
request's buffer), so the build reads it in place.

The fused layout takes one of three evidence realizers (Sec. 4.3, 5.3):
"pool" (structured pooling, the default), "prune" (nested pruning by a
per-token score the caller loads) or "merge" (hierarchical similarity
merging on the key channels); all three give the same view lengths.
"""
from __future__ import annotations

import torch

from . import davet as _davet
from .workloads import Workload


class Pipeline:
    REALIZERS = ("pool", "prune", "merge")

    def __init__(self, w: Workload, device="cuda", lib=None, fused: bool = True, realizer: str = "pool"):
        if realizer not in self.REALIZERS or (realizer != "pool" and not fused):
            raise ValueError(f"realizer {realizer!r} needs the fused layout and one of {self.REALIZERS}")
        self.w = w
        self.realizer = realizer
        self.dev = torch.device(device)
        self.lib = lib if lib is not None else _davet.load()
        C, B = w.C, w.batch
        self.sides = w.level_sides()
        self.fused = fused
        mixed = w.mixed_args
        text_rows = [p + r for p, r in zip(w.prompt, w.resp)]
        # one allocation; request b's buffer starts at row buf_row0[b]
        if fused:
            self.blocks = [self.lib.davet_view_layout(w.grid, w.n_levels, *mixed, w.tiles[b], text_rows[b])
                           for b in range(B)]
            rows = [blk[-1] for blk in self.blocks]
        else:
            rows = [w.pyramid_rows(b) for b in range(B)]
        self.buf_row0 = [0]
        for r in rows:
            self.buf_row0.append(self.buf_row0[-1] + r)
        n_buf = self.buf_row0[-1]
        self.store = torch.empty((max(n_buf, 1), C), dtype=torch.bfloat16, device=self.dev)
        self.bufs = [self.store[self.buf_row0[b]:self.buf_row0[b + 1]] for b in range(B)]
        self.buf_row0_dev = torch.tensor(self.buf_row0[:-1], dtype=torch.int64, device=self.dev)
        # text rows (unfused: gathered from here; fused: copied into every block)
        self.text = torch.empty((max(w.total_text(), 1), C), dtype=torch.bfloat16, device=self.dev)
        self.pyr_views = self.bufs  # unfused: the level-major pyramids
        self.pyr_ptrs = torch.tensor([v.data_ptr() for v in self.bufs], dtype=torch.int64, device=self.dev)
        self.tiles = torch.tensor(w.tiles, dtype=torch.int32, device=self.dev)
        self.prompt = torch.tensor(w.prompt, dtype=torch.int32, device=self.dev)
        self.resp = torch.tensor(w.resp, dtype=torch.int32, device=self.dev)
        self.text_off = torch.from_numpy(w.text_offsets()).to(self.dev)
        self.text_off_host = w.text_offsets()
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
        # realizer inputs: per-token scores (prune), a workspace (merge)
        self.scores = [torch.zeros((t, w.grid * w.grid), dtype=torch.float32, device=self.dev) for t in w.tiles]
        self.merge_ws = None
        if realizer == "merge":
            mw = max(self.lib.davet_merge_workspace_bytes(t, w.grid, w.n_levels, w.sim_channels()[1])
                     for t in w.tiles)
            self.merge_ws = torch.empty(max(mw, 256), dtype=torch.uint8, device=self.dev)

    # -------------------------------------------------------------- inputs
    def level0(self, b: int):
        """Rows of request b's encoding inside its buffer (level 0 comes first
        in both layouts)."""
        n = self.w.tiles[b] * self.w.grid * self.w.grid
        return self.bufs[b][:n]

    def pyramid_cpu(self, b: int):
        """Request b's pooled levels as a level-major bf16 CPU tensor (for
        checks), from either layout."""
        w = self.w
        if not self.fused:
            return self.bufs[b].cpu()
        parts = []
        for lvl, g in enumerate(self.sides):
            r0 = self.blocks[b][lvl]
            parts.append(self.bufs[b][r0:r0 + w.tiles[b] * g * g])
        return torch.cat(parts).cpu()

    def load_inputs(self, feats, text, non_blocking=False, scores=None):
        """feats: per-request bf16 [tiles, G, G, C]; text: bf16 [sum(P+R), C];
        scores (pruning realizer): per-request fp32 [tiles, G*G]."""
        for b, f in enumerate(feats):
            self.level0(b).copy_(f.reshape(-1, self.w.C), non_blocking=non_blocking)
        if self.w.total_text():
            self.text[: self.w.total_text()].copy_(text, non_blocking=non_blocking)
        if scores is not None:
            for b, s in enumerate(scores):
                self.scores[b].copy_(s.reshape(self.scores[b].shape), non_blocking=non_blocking)

    def reset_state(self):
        self.masked.fill_(1)
        self.tokens.fill_(-1)
        self.argmax.fill_(-1)

    # ---------------------------------------------------------------- path
    def build_pyramids(self, stream=None):
        """The pyramids (unfused) or every view block (fused), once per batch."""
        w = self.w
        for b in range(w.batch):
            v = self.bufs[b]
            if self.fused:
                t0 = int(self.text_off_host[b])
                n = w.prompt[b] + w.resp[b]
                text = self.text[t0:t0 + n] if n else None
                geo = (w.tiles[b], w.grid, w.n_levels, *w.mixed_args, n, w.C)
                if self.realizer == "pool":
                    self.lib.davet_build_views(v, v, text, *geo, stream)
                elif self.realizer == "prune":
                    self.lib.davet_build_views_pruned(v, self.scores[b], v, text, *geo, stream)
                else:
                    self.lib.davet_build_views_merged(v, v, text, *geo, *w.sim_channels(), None, self.merge_ws,
                                                      stream=stream)
            else:
                self.lib.davet_build_pyramid(v, v, w.tiles[b], w.grid, w.n_levels, w.C, None, stream)

    def gather(self, t: int, stream=None):
        w = self.w
        self.lib.davet_gather_view(self.pyr_ptrs, self.tiles, self.text, self.text_off, self.prompt, self.resp,
                                   self.schedule[t], w.batch, w.grid, w.n_levels, *w.mixed_args, w.C,
                                   self.packed, self.cu, self.max_rows, stream)

    def view_attention(self, t: int, stream=None):
        w = self.w
        self.lib.davet_view_attention(self.store, self.store.shape[0], self.buf_row0_dev, self.tiles, self.prompt,
                                      self.resp, self.schedule[t], w.batch, w.grid, w.n_levels, *w.mixed_args, w.H,
                                      w.D, w.scale, self.attn_out, self.cu, self.max_rows, stream)

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
        """One denoising step; NVTX ranges name its parts for profilers
        (host-side marks: they cost nothing on a replayed CUDA graph)."""
        nvtx = torch.cuda.nvtx
        nvtx.range_push(f"davet step {t}")
        if self.fused:
            nvtx.range_push("view_attention")
            self.view_attention(t, stream)
            nvtx.range_pop()
        else:
            nvtx.range_push("gather + attention")
            self.gather(t, stream)
            self.attention(stream)
            nvtx.range_pop()
        nvtx.range_push("unmask")
        self.unmask(t, logits, stream)
        nvtx.range_pop()
        nvtx.range_pop()
