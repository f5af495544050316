"""Parity of davet_step_attention (Sec. 3.1, Eq. 1) with the fp64 oracle.

Tolerance for bf16 inputs: max |gpu - oracle| <= 1e-2 and relative L2 error
<= 5e-3 over the compared outputs.  Cases span one and many 128-row tiles,
ragged tails, empty and one-row requests, both head dimensions, garbage
(non-finite) rows past the last request, and the full packed shapes of the
8B-class workloads, checked on sampled (row, head) pairs.

Work items hold one or two 128-row query tiles; the launch picks the count
(DAVET_ATTN_QTILES forces 1 or 2); the two kinds of item take different
paths through the MMA issuer and the softmax warpgroups, so the small cases
run under each choice.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from helpers import ATTN_MAX_ABS, ATTN_REL_L2, attn_errors, bf16_to_f64
from paper_2608_01821_gb300 import workloads

pytestmark = pytest.mark.gpu

QTILES = ["auto", "1", "2"]


@pytest.fixture(params=QTILES)
def qtiles(request, monkeypatch):
    """Query tiles per work item: chosen by the launch, or forced."""
    if request.param == "auto":
        monkeypatch.delenv("DAVET_ATTN_QTILES", raising=False)
    else:
        monkeypatch.setenv("DAVET_ATTN_QTILES", request.param)
    return request.param


def run(davet, qkv_cpu, cu, H, D, max_rows=None, garbage_tail=False):
    dev = torch.device("cuda")
    N = qkv_cpu.shape[0]
    max_rows = max_rows or N
    qkv = torch.empty((max_rows, 3, H, D), dtype=torch.bfloat16, device=dev)
    qkv[:N].copy_(qkv_cpu)
    if garbage_tail and max_rows > N:
        qkv[N:].view(torch.int16).fill_(0x7FC0)  # bf16 NaN
    out = torch.full((max_rows, H, D), 3.0, dtype=torch.bfloat16, device=dev)
    cu_d = torch.tensor(cu, dtype=torch.int32, device=dev)
    davet.davet_step_attention(qkv, cu_d, len(cu) - 1, max_rows, H, D, 1.0 / math.sqrt(D), out)
    torch.cuda.synchronize()
    assert davet.davet_device_status() == (0, 0)
    return out


@pytest.mark.parametrize("lens,H,D", [
    ([192], 4, 64),            # tiny workload shape
    ([1], 2, 128),
    ([127], 2, 128),
    ([128], 2, 128),
    ([129], 2, 128),
    ([300, 0, 5, 257], 3, 128),
    ([513, 64], 2, 64),
    ([1000], 1, 128),
])
def test_dense_parity(davet, qtiles, lens, H, D):
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    N = int(cu[-1])
    qkv = workloads.qkv_rows(N, H, D, seed=sum(lens) + H + D)
    out = run(davet, qkv, cu, H, D)
    ref = oracle.attention(qkv, cu, H, D, 1.0 / math.sqrt(D))
    got = bf16_to_f64(out[:N])
    assert np.isfinite(got).all()
    max_abs, rel = attn_errors(got, ref)
    assert max_abs <= ATTN_MAX_ABS and rel <= ATTN_REL_L2, (max_abs, rel)


def test_rows_past_the_last_request_do_not_leak(davet, qtiles):
    H, D = 2, 128
    lens = [200, 77]
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    N = int(cu[-1])
    qkv = workloads.qkv_rows(N, H, D, seed=5)
    out = run(davet, qkv, cu, H, D, max_rows=N + 300, garbage_tail=True)
    ref = oracle.attention(qkv, cu, H, D, 1.0 / math.sqrt(D))
    got = bf16_to_f64(out[:N])
    assert np.isfinite(got).all()
    max_abs, rel = attn_errors(got, ref)
    assert max_abs <= ATTN_MAX_ABS and rel <= ATTN_REL_L2
    # rows past cu[batch] are not written
    assert (out[N:].float() == 3.0).all()


def test_identical_keys_give_mean_of_values(davet):
    H, D, L = 2, 128, 333
    qkv = workloads.qkv_rows(L, H, D, seed=6)
    qkv[:, 1] = qkv[0:1, 1]
    out = run(davet, qkv, [0, L], H, D)
    mean_v = bf16_to_f64(qkv[:, 2]).mean(axis=0)
    got = bf16_to_f64(out)
    assert np.abs(got - mean_v[None]).max() <= ATTN_MAX_ABS


def test_growing_scores_force_the_rescale_path(davet, qtiles):
    # key norms grow along the sequence, so later key tiles carry maxima far
    # above the first tile's (by much more than 2^8 in the log2 domain) and
    # the running max must be raised and O rescaled; values are halved to
    # keep outputs within the range where the absolute bound is meaningful
    H, D, L = 2, 64, 700
    qkv = workloads.qkv_rows(L, H, D, seed=7)
    grow = torch.linspace(0.5, 5.5, L).view(L, 1, 1)
    qkv[:, 0] = (qkv[:, 0].float() * 2).to(torch.bfloat16)
    qkv[:, 1] = (qkv[:, 1].float() * grow).to(torch.bfloat16)
    qkv[:, 2] = (qkv[:, 2].float() * 0.5).to(torch.bfloat16)
    cu = np.array([0, L], np.int32)
    out = run(davet, qkv, cu, H, D)
    ref = oracle.attention(qkv, cu, H, D, 1.0 / math.sqrt(D))
    max_abs, rel = attn_errors(bf16_to_f64(out), ref)
    assert max_abs <= ATTN_MAX_ABS and rel <= ATTN_REL_L2, (max_abs, rel)


@pytest.mark.parametrize("name", ["single", "anyres", "highres", "ragged"])
def test_full_size_sampled(davet, name):
    """The packed step shapes of each workload at level 0 (the longest
    sequences) and at its coarsest scheduled level; 64 sampled (row, head)
    outputs per request are compared with the oracle."""
    w = workloads.make(name)
    rng = np.random.default_rng(hash(name) % 1000)
    for level in sorted({0, int(w.schedule.max())}):
        lens = [w.seq_len(b, level) for b in range(w.batch)]
        cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
        N = int(cu[-1])
        qkv = workloads.qkv_rows(N, w.H, w.D, seed=w.seed * 10 + level)
        out = run(davet, qkv, cu, w.H, w.D, max_rows=w.max_total_rows())
        rows, heads = [], []
        for b in range(w.batch):
            rows += list(rng.integers(cu[b], cu[b + 1], size=64))
            heads += list(rng.integers(0, w.H, size=64))
        rows = np.array(rows, np.int64)
        heads = np.array(heads, np.int32)
        ref = oracle.attention_rows(qkv, cu, w.H, w.D, w.scale, rows, heads)
        got = bf16_to_f64(out[torch.as_tensor(rows, device="cuda"), torch.as_tensor(heads, device="cuda").long()])
        max_abs, rel = attn_errors(got, ref)
        assert max_abs <= ATTN_MAX_ABS and rel <= ATTN_REL_L2, (name, level, max_abs, rel)


@pytest.mark.parametrize("L,H,nreq", [(5120, 16, 1), (2600, 16, 2)])
def test_last_round_split_into_one_tile_items(davet, L, H, nreq):
    """Work items of two 128-row query tiles run in rounds of one item per
    SM; when the last of several rounds fills at most half of the grid its
    items run as two one-tile items (on a 152-SM GPU: 5,120 rows x 16 heads
    = 320 items, the last 16 split; 2 x 2,600 rows x 16 heads = 352 items,
    the last 48 split).  Those items are the last heads' last query blocks in the
    schedule (longest request first, head-major), so every row of the last
    head is compared with the oracle, plus sampled rows of the others."""
    lens = [L] * nreq
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    N = int(cu[-1])
    D = 128
    qkv = workloads.qkv_rows(N, H, D, seed=L + H + nreq)
    out = run(davet, qkv, cu, H, D)
    rng = np.random.default_rng(L)
    last = cu[-2]  # the last request in the schedule (equal lengths: the highest index)
    rows = np.concatenate([np.arange(last, N), rng.integers(0, N, size=256)]).astype(np.int64)
    heads = np.concatenate([np.full(N - last, H - 1), rng.integers(0, H, size=256)]).astype(np.int32)
    ref = oracle.attention_rows(qkv, cu, H, D, 1.0 / math.sqrt(D), rows, heads)
    got = bf16_to_f64(out[torch.as_tensor(rows, device="cuda"), torch.as_tensor(heads, device="cuda").long()])
    max_abs, rel = attn_errors(got, ref)
    assert max_abs <= ATTN_MAX_ABS and rel <= ATTN_REL_L2, (max_abs, rel)


@pytest.mark.parametrize("qt", ["1", "2"])
def test_many_items_per_cta(davet, monkeypatch, qt):
    """More work items than SMs, so every CTA runs several items in turn and
    its barrier phases carry over between them: 2 requests (1,900 and 731
    rows, ragged last tiles) x 40 heads; under one-tile items ~5.5 per CTA,
    under two-tile items ~3, with a one-tile item for the 1,900-row
    request's odd last tile in each head.
    Three heads are compared in full, the others on sampled rows."""
    monkeypatch.setenv("DAVET_ATTN_QTILES", qt)
    H, D = 40, 128
    lens = [1900, 731]
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    N = int(cu[-1])
    qkv = workloads.qkv_rows(N, H, D, seed=11)
    out = run(davet, qkv, cu, H, D)
    rng = np.random.default_rng(12)
    full = [0, 17, H - 1]
    rows = np.concatenate([np.tile(np.arange(N), len(full)), rng.integers(0, N, size=512)]).astype(np.int64)
    heads = np.concatenate([np.repeat(full, N), rng.integers(0, H, size=512)]).astype(np.int32)
    ref = oracle.attention_rows(qkv, cu, H, D, 1.0 / math.sqrt(D), rows, heads)
    got = bf16_to_f64(out[torch.as_tensor(rows, device="cuda"), torch.as_tensor(heads, device="cuda").long()])
    max_abs, rel = attn_errors(got, ref)
    assert max_abs <= ATTN_MAX_ABS and rel <= ATTN_REL_L2, (max_abs, rel)


def test_decreasing_boundaries_are_flagged_and_clamped(davet):
    """cu_seqlens that go backwards: the call flags an argument error and
    runs each request from the previous request's end (clamped), so
    [0, 300, 200, 500] computes the requests [0, 300), [300, 300) and
    [300, 500)."""
    H, D = 2, 64
    N = 500
    qkv = workloads.qkv_rows(N, H, D, seed=23)
    davet.davet_device_status(clear=True)
    dev = torch.device("cuda")
    qkv_d = qkv.to(dev)
    out = torch.full((N, H, D), 3.0, dtype=torch.bfloat16, device=dev)
    cu_d = torch.tensor([0, 300, 200, 500], dtype=torch.int32, device=dev)
    davet.davet_step_attention(qkv_d, cu_d, 3, N, H, D, 1.0 / math.sqrt(D), out)
    torch.cuda.synchronize()
    st, flags = davet.davet_device_status(clear=True)
    assert flags & 0x4 and st != 0
    ref = oracle.attention(qkv, np.array([0, 300, 300, 500], np.int32), H, D, 1.0 / math.sqrt(D))
    max_abs, rel = attn_errors(bf16_to_f64(out), ref)
    assert max_abs <= ATTN_MAX_ABS and rel <= ATTN_REL_L2, (max_abs, rel)


@pytest.mark.parametrize("nreq", [33, 70])
def test_more_than_32_requests(davet, nreq):
    """More than 32 requests (ragged, some empty): laid out 32 at a time and
    ordered longest first by the whole CTA."""
    H, D = 2, 64
    rng = np.random.default_rng(nreq)
    lens = [int(x) for x in rng.integers(0, 260, size=nreq)]
    lens[3] = 0
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    N = int(cu[-1])
    qkv = workloads.qkv_rows(N, H, D, seed=nreq + 1)
    out = run(davet, qkv, cu, H, D)
    ref = oracle.attention(qkv, cu, H, D, 1.0 / math.sqrt(D))
    max_abs, rel = attn_errors(bf16_to_f64(out[:N]), ref)
    assert max_abs <= ATTN_MAX_ABS and rel <= ATTN_REL_L2, (max_abs, rel)
