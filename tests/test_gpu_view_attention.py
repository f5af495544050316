"""Parity of the view-block path (davet_build_views + davet_view_attention:
the view gather of Eq. 5 fused into the step attention of Sec. 3.1, Eq. 1)
with the unfused pair davet_gather_view + davet_step_attention, which the
other tests hold to the oracle.  The output rows and cu_seqlens must be
bit-identical (the kernels compute the same tiles; only where the rows come
from differs), for pooled levels, the mixed view, ragged and empty requests,
both head dimensions and a capacity overflow; the view blocks themselves
must hold exactly the pyramid's rows, the mixed view's rows and the text;
plus a direct oracle check on the tiny workloads."""
import math

import numpy as np
import pytest
import torch

import oracle
from helpers import ATTN_MAX_ABS, ATTN_REL_L2, attn_errors, bf16_to_f64, bits
from paper_2608_01821_gb300 import workloads
from paper_2608_01821_gb300.pipeline import Pipeline

pytestmark = pytest.mark.gpu


def build_both(davet, tiles, prompt, resp, grid, levels, H, D, seed, mixed):
    """The same requests as level-major pyramids + text (unfused) and as view
    blocks in one store (fused)."""
    C = 3 * H * D
    dev = torch.device("cuda")
    B = len(tiles)
    feats = [workloads.normal_bf16((t, grid, grid, C), seed * 100 + b) for b, t in enumerate(tiles)]
    n_text = int(sum(prompt) + sum(resp))
    text = workloads.normal_bf16((max(n_text, 1), C), seed * 7 + 1).to(dev)
    text_off = np.concatenate([[0], np.cumsum(np.add(prompt, resp))[:-1]]).astype(np.int64)
    pyrs = []
    for b, t in enumerate(tiles):
        off = davet.davet_pyramid_layout(grid, levels, t)[1]
        p = torch.empty((max(off[-1], 1), C), dtype=torch.bfloat16, device=dev)
        if t:
            p[: off[1]].copy_(feats[b].reshape(-1, C))
            davet.davet_build_pyramid(p, p, t, grid, levels, C)
        pyrs.append(p)
    blocks = [davet.davet_view_layout(grid, levels, *mixed, t, p + r) for t, p, r in zip(tiles, prompt, resp)]
    row0 = np.concatenate([[0], np.cumsum([blk[-1] for blk in blocks])]).astype(np.int64)
    store = torch.full((max(int(row0[-1]), 1), C), float("nan"), dtype=torch.bfloat16, device=dev)
    for b, t in enumerate(tiles):
        buf = store[int(row0[b]):int(row0[b + 1])]
        if t:
            buf[: t * grid * grid].copy_(feats[b].reshape(-1, C))
        n = prompt[b] + resp[b]
        tb = text[int(text_off[b]):int(text_off[b]) + n] if n else None
        davet.davet_build_views(buf, buf, tb, t, grid, levels, *mixed, n, C)
    return dict(C=C, pyrs=pyrs, text=text, text_off=text_off, store=store, row0=row0, blocks=blocks)


def run_both(davet, d, tiles, prompt, resp, view, grid, levels, H, D, cap, mixed):
    dev = torch.device("cuda")
    B = len(tiles)
    C = d["C"]
    t32 = lambda a: torch.tensor(a, dtype=torch.int32, device=dev)  # noqa: E731
    scale = 1 / math.sqrt(D)
    ptrs = torch.tensor([p.data_ptr() for p in d["pyrs"]], dtype=torch.int64, device=dev)
    packed = torch.empty((cap, C), dtype=torch.bfloat16, device=dev)
    cu_a = torch.full((B + 1,), -5, dtype=torch.int32, device=dev)
    davet.davet_gather_view(ptrs, t32(tiles), d["text"], torch.from_numpy(d["text_off"]).to(dev), t32(prompt),
                            t32(resp), t32(view), B, grid, levels, *mixed, C, packed, cu_a, cap)
    out_a = torch.full((cap, H, D), float("nan"), dtype=torch.bfloat16, device=dev)
    davet.davet_step_attention(packed, cu_a, B, cap, H, D, scale, out_a)
    cu_b = torch.full((B + 1,), -5, dtype=torch.int32, device=dev)
    out_b = torch.full((cap, H, D), float("nan"), dtype=torch.bfloat16, device=dev)
    davet.davet_view_attention(d["store"], d["store"].shape[0], torch.from_numpy(d["row0"][:-1].copy()).to(dev),
                               t32(tiles), t32(prompt), t32(resp), t32(view), B, grid, levels, *mixed, H, D, scale,
                               out_b, cu_b, cap)
    torch.cuda.synchronize()
    return out_a, cu_a, out_b, cu_b, packed


def test_view_blocks_hold_the_views_and_text(davet):
    grid, levels, H, D = 27, 4, 1, 64
    tiles, prompt, resp = [2, 1], [5, 0], [9, 3]
    mixed = (2, 3)
    d = build_both(davet, tiles, prompt, resp, grid, levels, H, D, 14, mixed)
    torch.cuda.synchronize()
    mrows = davet.davet_mixed_view_rows(grid, levels, *mixed)
    for b, t in enumerate(tiles):
        buf = bits(d["store"][int(d["row0"][b]):int(d["row0"][b + 1])])
        pyr = bits(d["pyrs"][b])
        off = davet.davet_pyramid_layout(grid, levels, t)[1]
        blk = d["blocks"][b]
        n = prompt[b] + resp[b]
        txt = bits(d["text"][int(d["text_off"][b]):int(d["text_off"][b]) + n])
        for lvl in range(levels):
            nv = off[lvl + 1] - off[lvl]
            np.testing.assert_array_equal(buf[blk[lvl]:blk[lvl] + nv], pyr[off[lvl]:off[lvl + 1]])
            np.testing.assert_array_equal(buf[blk[lvl] + nv:blk[lvl + 1]], txt)
        # the mixed view as the unfused gather forms it from the same pyramid
        # (its own parity with the oracle is held in the gather tests)
        dev = torch.device("cuda")
        i32 = lambda a: torch.tensor(a, dtype=torch.int32, device=dev)  # noqa: E731
        mv_t = torch.empty((max(t * mrows, 1), d["C"]), dtype=torch.bfloat16, device=dev)
        cu = torch.empty(2, dtype=torch.int32, device=dev)
        davet.davet_gather_view(torch.tensor([d["pyrs"][b].data_ptr()], dtype=torch.int64, device=dev), i32([t]),
                                d["text"], torch.zeros(1, dtype=torch.int64, device=dev), i32([0]), i32([0]),
                                i32([levels]), 1, grid, levels, *mixed, d["C"], mv_t, cu, max(t * mrows, 1))
        torch.cuda.synchronize()
        mv = bits(mv_t)[: t * mrows]
        np.testing.assert_array_equal(buf[blk[levels]:blk[levels] + t * mrows], mv)
        np.testing.assert_array_equal(buf[blk[levels] + t * mrows:blk[levels + 1]], txt)


@pytest.mark.parametrize("view,mixed", [([0, 3, 1], (0, 0)), ([2, 0, 3], (0, 0)), ([4, 2, 0], (2, 3)),
                                        ([4, 4, 4], (1, 1))])
def test_fused_matches_unfused_d128(davet, view, mixed):
    grid, levels, H, D = 27, 4, 2, 128
    tiles, prompt, resp = [2, 1, 3], [5, 0, 17], [9, 3, 0]
    d = build_both(davet, tiles, prompt, resp, grid, levels, H, D, 11, mixed)
    per_tile = max(729, davet.davet_mixed_view_rows(grid, levels, *mixed) if mixed[1] else 0)
    cap = sum(t * per_tile + p + r for t, p, r in zip(tiles, prompt, resp)) + 64
    davet.davet_device_status(clear=True)
    out_a, cu_a, out_b, cu_b, _ = run_both(davet, d, tiles, prompt, resp, view, grid, levels, H, D, cap, mixed)
    assert davet.davet_device_status() == (0, 0)
    assert torch.equal(cu_a, cu_b)
    n = int(cu_a[-1])
    assert np.array_equal(bits(out_a[:n]), bits(out_b[:n]))
    assert torch.isnan(out_b[n:].float()).all()  # rows past the step are not written


def test_fused_matches_unfused_d64_with_empty_request(davet):
    grid, levels, H, D = 12, 3, 4, 64
    tiles, prompt, resp = [1, 0, 2, 1], [16, 0, 3, 40], [32, 0, 1, 200]
    for view, mixed in (([0, 1, 2, 1], (0, 0)), ([3, 0, 3, 2], (2, 3))):
        d = build_both(davet, tiles, prompt, resp, grid, levels, H, D, 12, mixed)
        cap = sum(t * 144 + p + r for t, p, r in zip(tiles, prompt, resp))
        out_a, cu_a, out_b, cu_b, _ = run_both(davet, d, tiles, prompt, resp, view, grid, levels, H, D, cap, mixed)
        assert davet.davet_device_status() == (0, 0)
        assert torch.equal(cu_a, cu_b)
        n = int(cu_a[-1])
        assert np.array_equal(bits(out_a[:n]), bits(out_b[:n]))


def test_fused_capacity_overflow_is_flagged_and_clamped(davet):
    grid, levels, H, D = 27, 4, 1, 64
    tiles, prompt, resp = [1, 1], [10, 10], [10, 10]
    d = build_both(davet, tiles, prompt, resp, grid, levels, H, D, 13, (0, 0))
    davet.davet_device_status(clear=True)
    out_a, cu_a, out_b, cu_b, _ = run_both(davet, d, tiles, prompt, resp, [0, 0], grid, levels, H, D, 800, (0, 0))
    st, flags = davet.davet_device_status(clear=True)
    assert flags & 0x2 and st != 0
    assert list(cu_b.cpu().numpy()) == [0, 749, 800] == list(cu_a.cpu().numpy())
    assert np.array_equal(bits(out_a[:800]), bits(out_b[:800]))


def test_fused_view_out_of_range_is_flagged(davet):
    grid, levels, H, D = 27, 4, 1, 64
    tiles, prompt, resp = [1, 1], [10, 10], [10, 10]
    d = build_both(davet, tiles, prompt, resp, grid, levels, H, D, 15, (0, 0))
    davet.davet_device_status(clear=True)
    _, _, _, cu_b, _ = run_both(davet, d, tiles, prompt, resp, [4, 1], grid, levels, H, D, 2000, (0, 0))
    st, flags = davet.davet_device_status(clear=True)
    assert flags & 0x4
    assert list(cu_b.cpu().numpy()) == [0, 0, 196 + 20]


def test_fused_pipeline_tiny_against_oracle(davet):
    """Every step of the tiny workloads through the fused pipeline call,
    against the oracle's own pyramid (fp64 means rounded to bf16), gather and
    attention."""
    for name in ("tiny", "tiny_mixed"):
        w = workloads.make(name)
        pl = Pipeline(w, "cuda", davet, fused=True)
        feats = [workloads.features(w, b) for b in range(w.batch)]
        pl.load_inputs(feats, workloads.text_rows(w))
        pl.build_pyramids()
        torch.cuda.synchronize()
        ora_pyr = [torch.from_numpy(oracle.pyramid(feats[b], w.tiles[b], w.grid, w.n_levels, w.C)).to(torch.bfloat16)
                   for b in range(w.batch)]
        text = workloads.text_rows(w)
        if w.mixed:
            mrows = w.view_rows_per_tile(w.n_levels)
            pyrs = [np.concatenate([bits(p), oracle.mixed_view(p, w.tiles[b], w.grid, w.n_levels, *w.mixed, w.C)])
                    for b, p in enumerate(ora_pyr)]
        else:
            mrows, pyrs = 0, ora_pyr
        for t in range(w.T):
            pl.view_attention(t)
            torch.cuda.synchronize()
            assert davet.davet_device_status() == (0, 0)
            packed_ref, cu_ref = oracle.gather(pyrs, w.tiles, text, w.text_offsets(), w.prompt, w.resp, w.schedule[t],
                                               w.grid, w.n_levels, w.C, mixed_rows_per_tile=mrows)
            assert list(pl.cu.cpu().numpy()) == list(cu_ref)
            N = int(cu_ref[-1])
            ref = oracle.attention(packed_ref, cu_ref, w.H, w.D, w.scale)
            max_abs, rel = attn_errors(bf16_to_f64(pl.attn_out[:N]), ref)
            assert max_abs <= ATTN_MAX_ABS and rel <= ATTN_REL_L2, (name, t, max_abs, rel)


@pytest.mark.parametrize("name", ["single", "anyres", "highres", "ragged", "single_mixed"])
def test_fused_pipeline_full_size_matches_unfused(davet, name):
    """Full-size inputs in the benchmark's launch configuration: one step per
    distinct view schedule, fused and unfused pipelines bit-identical."""
    w = workloads.make(name)
    feats = [workloads.features(w, b) for b in range(w.batch)]
    text = workloads.text_rows(w)
    pls = []
    for fused in (False, True):
        pl = Pipeline(w, "cuda", davet, fused=fused)
        pl.load_inputs(feats, text)
        pl.build_pyramids()
        pls.append(pl)
    pu, pf = pls
    seen, steps = set(), []
    for t in range(w.T):
        key = tuple(w.schedule[t])
        if key not in seen:
            seen.add(key)
            steps.append(t)
    for t in steps[:4]:
        pu.gather(t)
        pu.attention()
        pf.view_attention(t)
        torch.cuda.synchronize()
        assert davet.davet_device_status() == (0, 0)
        assert torch.equal(pu.cu, pf.cu)
        n = int(pu.cu[-1])
        assert torch.equal(pu.attn_out[:n].view(torch.int16), pf.attn_out[:n].view(torch.int16)), (name, t)


def test_fused_matches_unfused_more_than_32_requests(davet):
    """40 requests (some empty, views mixed): the schedule lays out requests
    32 at a time and orders more than 32 with the whole CTA."""
    grid, levels, H, D = 12, 3, 2, 64
    rng = np.random.default_rng(40)
    B = 40
    tiles = [int(x) for x in rng.integers(0, 3, size=B)]
    prompt = [int(x) for x in rng.integers(0, 40, size=B)]
    resp = [int(x) for x in rng.integers(0, 90, size=B)]
    tiles[5], prompt[5], resp[5] = 0, 0, 0  # an empty request
    view = [int(x) for x in rng.integers(0, levels, size=B)]
    d = build_both(davet, tiles, prompt, resp, grid, levels, H, D, 41, (0, 0))
    cap = sum(t * 144 + p + r for t, p, r in zip(tiles, prompt, resp))
    out_a, cu_a, out_b, cu_b, _ = run_both(davet, d, tiles, prompt, resp, view, grid, levels, H, D, cap, (0, 0))
    assert davet.davet_device_status() == (0, 0)
    assert torch.equal(cu_a, cu_b)
    n = int(cu_a[-1])
    assert np.array_equal(bits(out_a[:n]), bits(out_b[:n]))
