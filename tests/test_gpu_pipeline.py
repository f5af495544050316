"""End-to-end parity of the step sequence against the oracle chain, on the
tiny workload for every step and on the 8B-class workloads for sampled
steps, through the Pipeline class the benchmark times, in both layouts:
fused (the benchmark's default: view blocks built once, then per step the
view attention, which reads each request's sequence from its view block,
and the unmasking) and unfused (pyramid once, then per step gather ->
attention -> unmask)."""
import numpy as np
import pytest
import torch

import oracle
from helpers import ATTN_MAX_ABS, ATTN_REL_L2, TOPK_REL, attn_errors, bf16_to_f64, bits, check_topk
from paper_2608_01821_gb300 import workloads
from paper_2608_01821_gb300.pipeline import Pipeline

pytestmark = pytest.mark.gpu


def make_pipeline(davet, w, fused=True):
    pl = Pipeline(w, "cuda", davet, fused=fused)
    feats = [workloads.features(w, b) for b in range(w.batch)]
    text = workloads.text_rows(w)
    pl.load_inputs(feats, text)
    pl.build_pyramids()
    torch.cuda.synchronize()
    return pl, feats, text


def oracle_pyramids(w, feats):
    out = []
    for b in range(w.batch):
        ref = oracle.pyramid(feats[b], w.tiles[b], w.grid, w.n_levels, w.C)
        out.append(torch.from_numpy(ref).float().to(torch.bfloat16))
    return out


def oracle_gather_inputs(w, pyr):
    """Per-request buffers for the oracle gather: the oracle's pyramid (fp64
    means rounded to bf16), followed by the oracle's mixed view of it when
    the workload has one."""
    if not w.mixed:
        return pyr, 0
    out = []
    for b, p in enumerate(pyr):
        mv = oracle.mixed_view(p, w.tiles[b], w.grid, w.n_levels, *w.mixed, w.C)
        out.append(np.concatenate([bits(p), mv]))
    return out, w.view_rows_per_tile(w.n_levels)


def check_packed(gpu_rows, ref_bits):
    """Packed rows against the oracle's: text rows are copies (bit-exact); a
    view row is the GPU's rounding of the same pooled value, so it may sit one
    bf16 step from the oracle's round-to-nearest (|x| < 8 here)."""
    got = gpu_rows.float().cpu().double().numpy()
    ref = torch.from_numpy(ref_bits.view(np.int16)).view(torch.bfloat16).double().numpy()
    assert np.abs(got - ref).max() <= 2.0 ** -5
    assert (bits(gpu_rows) == ref_bits).mean() > 0.999


@pytest.mark.parametrize("name,fused", [("tiny", False), ("tiny_mixed", False), ("tiny", True),
                                        ("tiny_mixed", True)])
def test_tiny_workload_every_step(davet, name, fused):
    w = workloads.make(name)
    pl, feats, text = make_pipeline(davet, w, fused)
    pyr_ref = oracle_pyramids(w, feats)
    # the GPU pyramid rounds the same values: at most one bf16 step away
    gpu_pyr = [pl.pyramid_cpu(b) for b in range(w.batch)]
    for b in range(w.batch):
        diff = (gpu_pyr[b].float() - pyr_ref[b].float()).abs()
        assert float(diff.max()) <= 2 ** -7  # at most one bf16 step on |x| < 2
    oracle_pyr, mrows = oracle_gather_inputs(w, pyr_ref)
    masked = np.ones(w.total_resp, np.uint8)
    tokens = np.full(w.total_resp, -1, np.int32)
    argmax = np.full(w.total_resp, -1, np.int32)
    cu_resp = w.cu_resp()
    for t in range(w.T):
        lg = workloads.logits(w, t)
        pl.step(t, lg.cuda())
        torch.cuda.synchronize()
        assert davet.davet_device_status() == (0, 0)
        packed_ref, cu_ref = oracle.gather(oracle_pyr, w.tiles, text, w.text_offsets(), w.prompt, w.resp,
                                           w.schedule[t], w.grid, w.n_levels, w.C, mixed_rows_per_tile=mrows)
        N = int(cu_ref[-1])
        assert list(pl.cu.cpu().numpy()) == list(cu_ref)
        if not fused:
            check_packed(pl.packed[:N], packed_ref)
        att_ref = oracle.attention(packed_ref, cu_ref, w.H, w.D, w.scale)
        max_abs, rel = attn_errors(bf16_to_f64(pl.attn_out[:N]), att_ref)
        assert max_abs <= ATTN_MAX_ABS and rel <= ATTN_REL_L2, (t, max_abs, rel)
        prev = masked.copy()
        conf_ref, com_ref, st_ref = oracle.unmask(lg, w.V, cu_resp, w.k, masked, tokens, argmax)
        picks = [int(x) for x in pl.committed[t, 0].cpu().numpy() if x >= 0]
        cref = {int(i): conf_ref[i] for i in np.nonzero(prev)[0]}
        if check_topk(picks, cref, w.k):
            masked[:] = pl.masked.cpu().numpy()
            tokens[:] = pl.tokens.cpu().numpy()
        assert np.array_equal(pl.masked.cpu().numpy(), masked)
        assert np.array_equal(pl.tokens.cpu().numpy(), tokens)
        np.testing.assert_allclose(pl.stats[t].cpu().numpy(), st_ref, rtol=TOPK_REL, atol=1e-7)
    assert masked.sum() == 0


def sampled_views(w):
    """The step views a full-size check covers: up to four distinct scheduled
    ones (per-request view vectors), then every request on the high view
    (level 0) and every request on the coarsest pooled level the schedule
    uses."""
    views, seen = [], set()
    for t in range(w.T):
        key = tuple(int(x) for x in w.schedule[t])
        if key not in seen:
            seen.add(key)
            views.append(key)
    views = views[:4]
    pooled = [int(x) for x in np.unique(w.schedule) if x < w.n_levels]
    for lvl in (0, max(pooled)):
        key = (lvl,) * w.batch
        if key not in seen:
            seen.add(key)
            views.append(key)
    return [np.array(v, np.int32) for v in views]


@pytest.mark.parametrize("fused", [True, False])
@pytest.mark.parametrize("name", ["single", "anyres", "highres", "ragged", "single_mixed"])
def test_workload_sampled_steps(davet, name, fused):
    """Full-size inputs in the benchmark's launch configuration (the fused
    layout is the benchmark's default step): for every sampled view, the
    step's cu_seqlens exactly, the packed rows bit for bit (unfused), and
    sampled (row, head) attention outputs against the oracle's attention
    over the oracle's gather of its own pyramid; the first view's commits
    exactly (near-tie rule)."""
    w = workloads.make(name)
    pl, feats, text = make_pipeline(davet, w, fused)
    gpu_pyr = [pl.pyramid_cpu(b) for b in range(w.batch)]
    oracle_pyr, mrows = oracle_gather_inputs(w, oracle_pyramids(w, feats))
    # pyramid: one request, first tile, all levels against the oracle
    side = w.level_sides()
    ref_off = oracle.level_offsets(w.grid, w.n_levels, 1)
    ref = oracle.pyramid(feats[0][0:1], 1, w.grid, w.n_levels, w.C)
    off = oracle.level_offsets(w.grid, w.n_levels, w.tiles[0])
    for lvl, g in enumerate(side):
        mine = bf16_to_f64(gpu_pyr[0][off[lvl]: off[lvl] + g * g])
        assert np.abs(mine - ref[ref_off[lvl]:ref_off[lvl + 1]]).max() <= 2 ** -6
    rng = np.random.default_rng(1)
    masked = np.ones(w.total_resp, np.uint8)
    tokens = np.full(w.total_resp, -1, np.int32)
    argmax = np.full(w.total_resp, -1, np.int32)
    lg = workloads.logits(w, 0)
    lg_dev = lg.cuda()
    for i, view in enumerate(sampled_views(w)):
        # the step runs the view vector written into schedule slot 0
        pl.schedule[0].copy_(torch.from_numpy(view))
        if fused:
            pl.view_attention(0)
        else:
            pl.gather(0)
            pl.attention()
        if i == 0:
            pl.unmask(0, lg_dev)
        torch.cuda.synchronize()
        assert davet.davet_device_status() == (0, 0)
        packed_ref, cu_ref = oracle.gather(oracle_pyr, w.tiles, text, w.text_offsets(), w.prompt, w.resp,
                                           view, w.grid, w.n_levels, w.C, mixed_rows_per_tile=mrows)
        N = int(cu_ref[-1])
        assert list(pl.cu.cpu().numpy()) == list(cu_ref), (name, list(view))
        if not fused:
            check_packed(pl.packed[:N], packed_ref)
        rows, heads = [], []
        for b in range(w.batch):
            if cu_ref[b + 1] == cu_ref[b]:
                continue
            # random rows, plus the request's first and last row (tile edges)
            rows += [cu_ref[b], cu_ref[b + 1] - 1] + list(rng.integers(cu_ref[b], cu_ref[b + 1], size=14))
            heads += list(rng.integers(0, w.H, size=16))
        rows = np.array(rows, np.int64)
        heads = np.array(heads, np.int32)
        att_ref = oracle.attention_rows(packed_ref, cu_ref, w.H, w.D, w.scale, rows, heads)
        got = bf16_to_f64(pl.attn_out[torch.as_tensor(rows, device="cuda"),
                                      torch.as_tensor(heads, device="cuda").long()])
        max_abs, rel = attn_errors(got, att_ref)
        assert max_abs <= ATTN_MAX_ABS and rel <= ATTN_REL_L2, (name, list(view), max_abs, rel)
        if i == 0:
            cu_resp = w.cu_resp()
            conf_ref, _, st_ref = oracle.unmask(lg, w.V, cu_resp, w.k, masked, tokens, argmax)
            g_com = pl.committed[0].cpu().numpy()
            for b in range(w.batch):
                cref = {int(j - cu_resp[b]): conf_ref[j] for j in range(cu_resp[b], cu_resp[b + 1])}
                check_topk([int(x) for x in g_com[b] if x >= 0], cref, w.k)
            np.testing.assert_array_equal(pl.argmax.cpu().numpy(), argmax)
