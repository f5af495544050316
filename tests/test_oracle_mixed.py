"""Pins for the oracle's `mixed` evidence view (Sec. 4.3: the pooled
representation augmented with a fixed subset of unpooled tokens; the subset
is read as a centred stride-s lattice of level-0 tokens) and for gathering it
as the view of a step."""
import numpy as np
import torch

import oracle


def id_pyramid(n_tiles, grid, levels, C):
    """Pyramid rows tagged (level, tile, cell mod 128, cell div 128)."""
    sides = oracle.level_sides(grid, levels)
    ids = []
    for lvl, g in enumerate(sides):
        for t in range(n_tiles):
            for cell in range(g * g):
                ids.append([lvl, t, cell % 128, cell // 128])
    a = np.zeros((len(ids), C), np.float32)
    a[:, :4] = ids
    return torch.from_numpy(a).to(torch.bfloat16)


def decode(bits):
    return torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).float().numpy()


def test_row_counts_and_ordering():
    assert oracle.mixed_rows_per_tile(27, 4, 2, 3) == 49 + 81
    assert oracle.mixed_rows_per_tile(27, 4, 3, 4) == 16 + 49
    assert oracle.mixed_rows_per_tile(12, 3, 2, 3) == 9 + 16
    # coarse < mixed < high for the paper-like three-view hierarchy
    assert 49 < oracle.mixed_rows_per_tile(27, 4, 2, 3) < 729


def test_layout_coarse_then_lattice_per_tile():
    n_tiles, grid, levels, C = 3, 27, 4, 8
    pyr = id_pyramid(n_tiles, grid, levels, C)
    out = decode(oracle.mixed_view(pyr, n_tiles, grid, levels, 2, 3, C))
    r = 0
    for t in range(n_tiles):
        for cell in range(49):
            assert list(out[r, :4]) == [2, t, cell % 128, cell // 128]
            r += 1
        for y in range(1, 27, 3):
            for x in range(1, 27, 3):
                cell = y * 27 + x
                assert list(out[r, :4]) == [0, t, cell % 128, cell // 128]
                r += 1
    assert r == out.shape[0]


def test_stride_one_keeps_every_token():
    n_tiles, grid, levels, C = 2, 5, 3, 8
    pyr = id_pyramid(n_tiles, grid, levels, C)
    out = oracle.mixed_view(pyr, n_tiles, grid, levels, 1, 1, C)
    g1 = 3
    per = g1 * g1 + 25
    pb = pyr.view(torch.int16).numpy().view(np.uint16)
    for t in range(n_tiles):
        np.testing.assert_array_equal(out[t * per + g1 * g1:(t + 1) * per], pb[t * 25:(t + 1) * 25])


def test_gather_selects_the_mixed_view_as_level_n_levels():
    n_tiles, grid, levels, C = 2, 27, 4, 8
    pyr = id_pyramid(n_tiles, grid, levels, C)
    mixed = oracle.mixed_view(pyr, n_tiles, grid, levels, 2, 3, C)
    mrows = oracle.mixed_rows_per_tile(grid, levels, 2, 3)
    full = np.concatenate([pyr.view(torch.int16).numpy().view(np.uint16), mixed])
    text = torch.zeros((7, C), dtype=torch.bfloat16)
    packed, cu = oracle.gather([full, full], [n_tiles, n_tiles], text, [0, 3], [2, 1], [1, 3], [levels, 0], grid,
                               levels, C, mixed_rows_per_tile=mrows)
    assert list(cu) == [0, n_tiles * mrows + 3, n_tiles * mrows + 3 + n_tiles * 729 + 4]
    np.testing.assert_array_equal(packed[:n_tiles * mrows], mixed)


def test_mixed_workloads_view_rows():
    from paper_2608_01821_gb300 import workloads
    for name in workloads.MIXED_NAMES:
        w = workloads.make(name)
        assert w.view_rows_per_tile(w.n_levels) == oracle.mixed_rows_per_tile(w.grid, w.n_levels, *w.mixed)
        assert set(np.unique(w.schedule)) <= set(range(w.n_views()))
    w = workloads.make("single_mixed")
    assert [w.seq_len(0, v) for v in (2, 4, 0)] == [49 + 192, 130 + 192, 729 + 192]
