"""Parity of davet_gather_view (Eq. 5) with the oracle: packed rows and
cu_seqlens must be bit-exact; device-side range and capacity problems set
the device error word without writing out of bounds.  The gather copies
rows, so its per-request buffers hold seeded rows in the pyramid layout
(both sides get the same seeded values; none come from a kernel)."""
import numpy as np
import pytest
import torch

import oracle
from helpers import bits
from paper_2608_01821_gb300 import workloads

pytestmark = pytest.mark.gpu


def setup(davet, tiles, prompt, resp, grid, levels, C, seed):
    dev = torch.device("cuda")
    B = len(tiles)
    pyrs = []
    for b in range(B):
        off = oracle.level_offsets(grid, levels, tiles[b])
        pyrs.append(workloads.normal_bf16((max(off[-1], 1), C), seed * 100 + b).to(dev))
    n_text = sum(prompt) + sum(resp)
    text = workloads.normal_bf16((max(n_text, 1), C), seed * 7 + 1).to(dev)
    text_off = np.concatenate([[0], np.cumsum(np.add(prompt, resp))[:-1]]).astype(np.int64)
    d = dict(
        pyrs=pyrs,
        pyr_ptrs=torch.tensor([p.data_ptr() for p in pyrs], dtype=torch.int64, device=dev),
        tiles=torch.tensor(tiles, dtype=torch.int32, device=dev),
        text=text,
        text_off=torch.from_numpy(text_off).to(dev),
        prompt=torch.tensor(prompt, dtype=torch.int32, device=dev),
        resp=torch.tensor(resp, dtype=torch.int32, device=dev),
        text_off_np=text_off,
    )
    return d


def run(davet, d, level, grid, levels, C, cap, mixed=(0, 0)):
    dev = torch.device("cuda")
    B = len(level)
    # 64 guard rows past the capacity must stay untouched
    packed = torch.full((cap + 64, C), float("nan"), dtype=torch.bfloat16, device=dev)
    cu = torch.full((B + 1,), -5, dtype=torch.int32, device=dev)
    lv = torch.tensor(level, dtype=torch.int32, device=dev)
    davet.davet_gather_view(d["pyr_ptrs"], d["tiles"], d["text"], d["text_off"], d["prompt"], d["resp"], lv, B,
                            grid, levels, *mixed, C, packed, cu, cap)
    torch.cuda.synchronize()
    assert torch.isnan(packed[cap:].float()).all()
    return packed[:cap], cu


@pytest.mark.parametrize("level", [[0, 0, 0], [3, 1, 2], [2, 3, 0]])
def test_ragged_batch_bit_exact(davet, level):
    grid, levels, C = 27, 4, 256
    tiles, prompt, resp = [2, 1, 3], [5, 0, 17], [9, 3, 0]
    d = setup(davet, tiles, prompt, resp, grid, levels, C, 1)
    cap = sum(t * 729 + p + r for t, p, r in zip(tiles, prompt, resp))
    packed, cu = run(davet, d, level, grid, levels, C, cap)
    assert davet.davet_device_status() == (0, 0)
    ref, ref_cu = oracle.gather([p.cpu() for p in d["pyrs"]], tiles, d["text"].cpu(), d["text_off_np"], prompt,
                                resp, level, grid, levels, C)
    assert list(cu.cpu().numpy()) == list(ref_cu)
    n = int(ref_cu[-1])
    assert np.array_equal(bits(packed[:n]), ref)


def test_empty_requests_and_tiny_config(davet):
    w = workloads.make("tiny")
    grid, levels, C = w.grid, w.n_levels, w.C
    tiles, prompt, resp = [1, 0, 1], [16, 0, 0], [32, 0, 0]
    d = setup(davet, tiles, prompt, resp, grid, levels, C, 2)
    cap = 144 + 48 + 144
    packed, cu = run(davet, d, [2, 0, 1], grid, levels, C, cap)
    ref, ref_cu = oracle.gather([p.cpu() for p in d["pyrs"]], tiles, d["text"].cpu(), d["text_off_np"], prompt,
                                resp, [2, 0, 1], grid, levels, C)
    assert list(cu.cpu().numpy()) == list(ref_cu)
    assert np.array_equal(bits(packed[: int(ref_cu[-1])]), ref)


def test_capacity_overflow_is_flagged_and_clamped(davet):
    grid, levels, C = 27, 4, 64
    tiles, prompt, resp = [1, 1], [10, 10], [10, 10]
    d = setup(davet, tiles, prompt, resp, grid, levels, C, 3)
    davet.davet_device_status(clear=True)
    cap = 800  # total is 2 * 749 = 1498
    packed, cu = run(davet, d, [0, 0], grid, levels, C, cap)
    st, flags = davet.davet_device_status(clear=True)
    assert flags & 0x2 and st != 0
    assert list(cu.cpu().numpy()) == [0, 749, 800]


def test_level_out_of_range_is_flagged(davet):
    grid, levels, C = 27, 4, 64
    tiles, prompt, resp = [1, 1], [10, 10], [10, 10]
    d = setup(davet, tiles, prompt, resp, grid, levels, C, 4)
    davet.davet_device_status(clear=True)
    packed, cu = run(davet, d, [7, 1], grid, levels, C, 2000)
    st, flags = davet.davet_device_status(clear=True)
    assert flags & 0x4
    assert list(cu.cpu().numpy()) == [0, 20, 20 + 196 + 20]


def with_mixed(pyr, tiles, grid, levels, C, mixed):
    """Oracle-side buffer: the pyramid followed by its materialized mixed view."""
    p = bits(pyr)
    if tiles == 0:
        return p
    return np.concatenate([p[: oracle.level_offsets(grid, levels, tiles)[-1]],
                           oracle.mixed_view(pyr.cpu(), tiles, grid, levels, *mixed, C)])


@pytest.mark.parametrize("level,mixed", [([4, 0, 4], (2, 3)), ([1, 4, 3], (2, 3)), ([4, 4, 2], (3, 4)),
                                         ([4, 4, 4], (0, 27)), ([4, 2, 4], (1, 1))])
def test_mixed_view_bit_exact(davet, level, mixed):
    """The mixed view (Sec. 4.3) is gathered from the pyramid without being
    stored; the oracle materializes it and gathers it as one more level."""
    grid, levels, C = 27, 4, 256
    tiles, prompt, resp = [2, 1, 3], [5, 0, 17], [9, 3, 0]
    d = setup(davet, tiles, prompt, resp, grid, levels, C, 5)
    mrows = davet.davet_mixed_view_rows(grid, levels, *mixed)
    assert mrows == oracle.mixed_rows_per_tile(grid, levels, *mixed)
    cap = sum(t * max(729, mrows) + p + r for t, p, r in zip(tiles, prompt, resp))
    packed, cu = run(davet, d, level, grid, levels, C, cap, mixed)
    assert davet.davet_device_status() == (0, 0)
    pyrs = [with_mixed(p, t, grid, levels, C, mixed) for p, t in zip(d["pyrs"], tiles)]
    ref, ref_cu = oracle.gather(pyrs, tiles, d["text"].cpu(), d["text_off_np"], prompt, resp, level, grid, levels,
                                C, mixed_rows_per_tile=mrows)
    assert list(cu.cpu().numpy()) == list(ref_cu)
    assert np.array_equal(bits(packed[: int(ref_cu[-1])]), ref)


def test_mixed_view_full_width_tiny_grid(davet):
    """Odd channel tail (C/8 not a multiple of 32 lanes) on the 12x12 grid
    with coarse level 2 and stride 3: 9 + 16 rows per tile."""
    grid, levels, C = 12, 3, 768 + 8
    tiles, prompt, resp = [1, 2], [16, 3], [32, 1]
    d = setup(davet, tiles, prompt, resp, grid, levels, C, 6)
    mixed = (2, 3)
    assert davet.davet_mixed_view_rows(grid, levels, *mixed) == 25
    cap = sum(t * 144 + p + r for t, p, r in zip(tiles, prompt, resp))
    packed, cu = run(davet, d, [3, 3], grid, levels, C, cap, mixed)
    assert davet.davet_device_status() == (0, 0)
    pyrs = [with_mixed(p, t, grid, levels, C, mixed) for p, t in zip(d["pyrs"], tiles)]
    ref, ref_cu = oracle.gather(pyrs, tiles, d["text"].cpu(), d["text_off_np"], prompt, resp, [3, 3], grid, levels,
                                C, mixed_rows_per_tile=25)
    assert list(cu.cpu().numpy()) == [0, 25 + 48, 25 + 48 + 50 + 4] == list(ref_cu)
    assert np.array_equal(bits(packed[: int(ref_cu[-1])]), ref)


def test_mixed_index_without_a_mixed_view_is_flagged(davet):
    grid, levels, C = 27, 4, 64
    tiles, prompt, resp = [1, 1], [10, 10], [10, 10]
    d = setup(davet, tiles, prompt, resp, grid, levels, C, 7)
    davet.davet_device_status(clear=True)
    packed, cu = run(davet, d, [4, 2], grid, levels, C, 2000)
    st, flags = davet.davet_device_status(clear=True)
    assert flags & 0x4
    assert list(cu.cpu().numpy()) == [0, 20, 20 + 49 + 20]


def test_sync_status_reads_the_word_after_a_stream(davet):
    """davet_sync_status waits for one stream and reports the word without
    clearing it; davet_device_status then clears it."""
    grid, levels, C = 27, 4, 64
    tiles, prompt, resp = [1, 1], [10, 10], [10, 10]
    d = setup(davet, tiles, prompt, resp, grid, levels, C, 8)
    davet.davet_device_status(clear=True)
    s = torch.cuda.Stream()
    packed = torch.empty((800, C), dtype=torch.bfloat16, device="cuda")
    cu = torch.empty(3, dtype=torch.int32, device="cuda")
    lv = torch.zeros(2, dtype=torch.int32, device="cuda")
    torch.cuda.synchronize()
    davet.davet_gather_view(d["pyr_ptrs"], d["tiles"], d["text"], d["text_off"], d["prompt"], d["resp"], lv, 2,
                            grid, levels, 0, 0, C, packed, cu, 800, s)
    st, flags = davet.davet_sync_status(s)
    assert st == 5 and flags & 0x2  # DAVET_ERR_DEVICE: the capacity bit
    assert davet.davet_sync_status(s)[1] & 0x2  # not cleared
    davet.davet_device_status(clear=True)
    assert davet.davet_sync_status(s) == (0, 0)
