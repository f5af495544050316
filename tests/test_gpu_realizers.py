"""Parity of the pruning and merging realizers (Sec. 4.3 "compatible evidence
realizers", Sec. 5.3 / Table 2) with the oracle: every view block -- view
rows and text rows -- and the merge assignment must be bit-exact; the blocks
feed davet_view_attention unchanged."""
import numpy as np
import pytest
import torch

import oracle
from helpers import ATTN_MAX_ABS, ATTN_REL_L2, attn_errors, bits
from paper_2608_01821_gb300 import workloads
from paper_2608_01821_gb300.pipeline import Pipeline

pytestmark = pytest.mark.gpu


def expected_blocks(views, text_bits, layout, C):
    out = np.zeros((layout[-1], C), np.uint16)
    for v, rows in enumerate(views):
        out[layout[v]:layout[v] + len(rows)] = rows
        out[layout[v] + len(rows):layout[v + 1]] = text_bits
    return out


def make_request(davet, n_tiles, grid, levels, mixed, text_rows, C, seed, in_place):
    dev = torch.device("cuda")
    layout = davet.davet_view_layout(grid, levels, *mixed, n_tiles, text_rows)
    feat = workloads.normal_bf16((n_tiles, grid * grid, C), seed)
    text = workloads.normal_bf16((max(text_rows, 1), C), seed + 1)[:text_rows]
    buf = torch.full((layout[-1] + 64, C), float("nan"), dtype=torch.bfloat16, device=dev)
    if in_place:
        buf[: n_tiles * grid * grid].copy_(feat.reshape(-1, C))
        src = buf
    else:
        src = feat.reshape(-1, C).to(dev)
    return layout, feat, text, text.to(dev), buf, src


# ------------------------------------------------------------------ pruning
@pytest.mark.parametrize("n_tiles,grid,levels,mixed,C,text_rows,in_place", [
    (1, 12, 3, (2, 3), 768, 48, True),
    (3, 27, 4, (2, 3), 256, 37, False),
    (2, 27, 4, (0, 0), 264, 0, True),
    (1, 27, 4, (2, 3), 12288, 192, True),
])
def test_pruned_blocks_bit_exact(davet, n_tiles, grid, levels, mixed, C, text_rows, in_place):
    layout, feat, text, text_d, buf, src = make_request(davet, n_tiles, grid, levels, mixed, text_rows, C, 11,
                                                        in_place)
    rng = np.random.default_rng(grid + n_tiles)
    score = rng.standard_normal((n_tiles, grid * grid)).astype(np.float32)
    score[0, ::5] = score[0, 2]  # ties
    score[-1, [3, 30, 100]] = np.nan
    rpt = oracle.view_rows_per_tile(grid, levels, mixed if mixed[1] else None)
    davet.davet_build_views_pruned(src, torch.from_numpy(score).cuda(), buf, text_d if text_rows else None, n_tiles,
                                   grid, levels, *mixed, text_rows, C)
    torch.cuda.synchronize()
    assert davet.davet_device_status() == (0, 0)
    views = oracle.prune_views(feat, score, n_tiles, grid, rpt, C)
    want = expected_blocks(views, bits(text), layout, C)
    got = bits(buf)
    assert np.array_equal(got[: layout[-1]], want)
    assert torch.isnan(buf[layout[-1]:].float()).all()


def test_pruned_text_only_and_all_equal_scores(davet):
    """An image-free request gets its text in every block; equal scores keep
    the first tokens in raster order."""
    grid, levels, C = 12, 3, 64
    layout, feat, text, text_d, buf, src = make_request(davet, 0, grid, levels, (0, 0), 9, C, 3, False)
    davet.davet_build_views_pruned(None, None, buf, text_d, 0, grid, levels, 0, 0, 9, C)
    torch.cuda.synchronize()
    assert np.array_equal(bits(buf)[: layout[-1]], expected_blocks([np.zeros((0, C), np.uint16)] * 3, bits(text),
                                                                   layout, C))
    layout, feat, text, text_d, buf, src = make_request(davet, 2, grid, levels, (0, 0), 4, C, 4, True)
    score = torch.full((2, 144), 0.25, device="cuda")
    davet.davet_build_views_pruned(src, score, buf, text_d, 2, grid, levels, 0, 0, 4, C)
    torch.cuda.synchronize()
    fb = bits(feat)
    for v, m in enumerate([144, 36, 9]):
        rows = bits(buf)[layout[v]:layout[v] + 2 * m]
        assert np.array_equal(rows, np.concatenate([fb[0, :m], fb[1, :m]]))


# ------------------------------------------------------------------ merging
def merged_reference(feat, n_tiles, grid, levels, mixed, C, c0, Cs):
    lv, assign = oracle.merge_views(feat, n_tiles, grid, levels, C, c0, Cs)
    views = list(lv)
    if mixed[1]:
        pyr = torch.from_numpy(np.concatenate(lv).view(np.int16)).view(torch.bfloat16)
        views.append(oracle.mixed_view(pyr, n_tiles, grid, levels, *mixed, C))
    return views, assign


@pytest.mark.parametrize("n_tiles,grid,levels,mixed,C,sim,text_rows,in_place", [
    (1, 12, 3, (2, 3), 768, (256, 256), 48, True),
    (3, 27, 4, (2, 3), 256, (64, 128), 37, False),
    (2, 8, 4, (0, 0), 64, (0, 64), 5, True),
    (4, 5, 3, (1, 1), 96, (32, 32), 0, False),
])
def test_merged_blocks_and_assignment_bit_exact(davet, n_tiles, grid, levels, mixed, C, sim, text_rows, in_place):
    layout, feat, text, text_d, buf, src = make_request(davet, n_tiles, grid, levels, mixed, text_rows, C, 21,
                                                        in_place)
    ws = torch.empty(davet.davet_merge_workspace_bytes(n_tiles, grid, levels, sim[1]), dtype=torch.uint8,
                     device="cuda")
    assign = torch.full((levels, n_tiles, grid * grid), -7, dtype=torch.int32, device="cuda")
    davet.davet_build_views_merged(src, buf, text_d if text_rows else None, n_tiles, grid, levels, *mixed, text_rows,
                                   C, *sim, assign, ws)
    torch.cuda.synchronize()
    assert davet.davet_device_status() == (0, 0)
    views, ref_assign = merged_reference(feat, n_tiles, grid, levels, mixed, C, *sim)
    assert np.array_equal(assign.cpu().numpy(), ref_assign)
    want = expected_blocks(views, bits(text), layout, C)
    got = bits(buf)
    assert np.array_equal(got[: layout[-1]], want)
    assert torch.isnan(buf[layout[-1]:].float()).all()


def test_merged_full_width_single_tile(davet):
    """The 8B-class row (C = 12288, similarity on the 4096 key channels) on
    one 27x27 tile with the three-view mixed hierarchy."""
    grid, levels, mixed, C, sim = 27, 4, (2, 3), 12288, (4096, 4096)
    layout, feat, text, text_d, buf, src = make_request(davet, 1, grid, levels, mixed, 192, C, 31, True)
    ws = torch.empty(davet.davet_merge_workspace_bytes(1, grid, levels, sim[1]), dtype=torch.uint8, device="cuda")
    assign = torch.empty((levels, 1, grid * grid), dtype=torch.int32, device="cuda")
    davet.davet_build_views_merged(src, buf, text_d, 1, grid, levels, *mixed, 192, C, *sim, assign, ws)
    torch.cuda.synchronize()
    views, ref_assign = merged_reference(feat, 1, grid, levels, mixed, C, *sim)
    assert np.array_equal(assign.cpu().numpy(), ref_assign)
    assert np.array_equal(bits(buf)[: layout[-1]], expected_blocks(views, bits(text), layout, C))


def test_merge_is_deterministic_and_workspace_needs_no_init(davet):
    grid, levels, C, sim = 27, 4, 128, (0, 64)
    layout, feat, text, text_d, buf, src = make_request(davet, 2, grid, levels, (0, 0), 3, C, 41, False)
    nbytes = davet.davet_merge_workspace_bytes(2, grid, levels, sim[1])
    outs = []
    for fill in (0x00, 0xFF):
        ws = torch.full((nbytes,), fill, dtype=torch.uint8, device="cuda")
        buf.fill_(0)
        davet.davet_build_views_merged(src, buf, text_d, 2, grid, levels, 0, 0, 3, C, *sim, None, ws)
        torch.cuda.synchronize()
        outs.append(bits(buf).copy())
    assert np.array_equal(outs[0], outs[1])


# ------------------------------------------------------- through the attention
@pytest.mark.parametrize("realizer", ["prune", "merge"])
def test_pipeline_attention_over_realized_views(davet, realizer):
    """One step of the tiny mixed workload through davet_view_attention over
    the realizer's blocks equals the oracle's attention over the same step
    sequences [view || prompt || answer]."""
    w = workloads.make("tiny_mixed")
    pl = Pipeline(w, lib=davet, realizer=realizer)
    feats = [workloads.features(w, b) for b in range(w.batch)]
    scores = [workloads.token_scores(w, b) for b in range(w.batch)]
    pl.load_inputs(feats, workloads.text_rows(w), scores=scores)
    pl.build_pyramids()
    torch.cuda.synchronize()
    text = bits(workloads.text_rows(w))
    rpt = oracle.view_rows_per_tile(w.grid, w.n_levels, w.mixed)
    if realizer == "prune":
        views = oracle.prune_views(feats[0], scores[0].numpy(), w.tiles[0], w.grid, rpt, w.C)
    else:
        views, _ = merged_reference(feats[0], w.tiles[0], w.grid, w.n_levels, w.mixed, w.C, *w.sim_channels())
    assert np.array_equal(bits(pl.bufs[0]), expected_blocks(views, text, pl.blocks[0], w.C))
    for t in (0, 2, 4):  # high, mixed and coarse views
        pl.view_attention(t)
        torch.cuda.synchronize()
        v = int(w.schedule[t, 0])
        seq = np.concatenate([views[v], text])
        qkv = torch.from_numpy(seq.view(np.int16)).view(torch.bfloat16)
        cu = np.array([0, len(seq)], np.int32)
        assert list(pl.cu.cpu().numpy()) == list(cu)
        ref = oracle.attention(qkv, cu, w.H, w.D, w.scale)
        got = pl.attn_out[: len(seq)].float().cpu().numpy().astype(np.float64)
        max_abs, rel = attn_errors(got, ref)
        assert max_abs < ATTN_MAX_ABS and rel < ATTN_REL_L2
