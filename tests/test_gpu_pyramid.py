"""Parity of davet_build_pyramid (Sec. 4.3) with the fp64 oracle.

fp32 levels must lie within 1e-6 of the oracle relative to the window's mean
|x| (the oracle's pyramid of |x|); bf16 levels must be the round-to-nearest
of the oracle value, or a neighbour when the oracle value is that close to a
rounding midpoint; level 0 is copied bit for bit.
"""
import numpy as np
import pytest
import torch

import oracle
from helpers import POOL_REL, bf16_to_f64, bits, check_bf16_rounding
from paper_2608_01821_gb300 import workloads

pytestmark = pytest.mark.gpu


def run_case(davet, n_tiles, grid, levels, C, seed, alias):
    feat = workloads.normal_bf16((n_tiles, grid, grid, C), seed)
    side, off = davet.davet_pyramid_layout(grid, levels, n_tiles)
    rows = off[-1]
    dev = torch.device("cuda")
    pyr = torch.full((rows, C), float("nan"), dtype=torch.bfloat16, device=dev)
    p32 = torch.full((rows, C), float("nan"), dtype=torch.float32, device=dev)
    if alias:
        pyr[: off[1]].copy_(feat.reshape(-1, C))
        src = pyr
    else:
        src = feat.to(dev)
    davet.davet_build_pyramid(src, pyr, n_tiles, grid, levels, C, p32)
    torch.cuda.synchronize()
    st, flags = davet.davet_device_status()
    assert st == 0 and flags == 0
    ref = oracle.pyramid(feat, n_tiles, grid, levels, C)
    scale = oracle.pyramid_f64(np.abs(bf16_to_f64(feat)), levels)
    g32 = p32.double().cpu().numpy()
    err = np.abs(g32 - ref)
    assert np.isfinite(g32).all()
    assert (err <= POOL_REL * scale + 1e-30).all(), float((err / np.maximum(scale, 1e-30)).max())
    gb = bf16_to_f64(pyr)
    assert np.array_equal(bits(pyr[: off[1]]), bits(feat.reshape(-1, C)))
    assert check_bf16_rounding(gb, ref, scale) == 0
    return float((err / np.maximum(scale, 1e-30)).max())


@pytest.mark.parametrize("alias", [True, False])
def test_tiny_grid(davet, alias):
    run_case(davet, 1, 12, 3, 768, 11, alias)


def test_single_tile_full_channels(davet):
    worst = run_case(davet, 1, 27, 4, 12288, 12, True)
    assert worst < POOL_REL


def test_multi_tile_and_odd_grids(davet):
    run_case(davet, 5, 27, 4, 256, 13, True)
    run_case(davet, 3, 5, 5, 64, 14, False)
    run_case(davet, 2, 1, 3, 8, 15, True)
    run_case(davet, 2, 31, 5, 40, 16, False)


def test_constant_grid_is_exact(davet):
    n_tiles, grid, levels, C = 2, 27, 4, 64
    feat = torch.full((n_tiles, grid, grid, C), 0.8125, dtype=torch.bfloat16)
    side, off = davet.davet_pyramid_layout(grid, levels, n_tiles)
    pyr = torch.empty((off[-1], C), dtype=torch.bfloat16, device="cuda")
    davet.davet_build_pyramid(feat.cuda(), pyr, n_tiles, grid, levels, C)
    torch.cuda.synchronize()
    assert (pyr.float() == 0.8125).all()


def test_highres_request_sampled_tiles(davet):
    """A full 10-tile request at C = 12288; the oracle checks two tiles."""
    w = workloads.make("highres")
    feat = workloads.features(w, 0)
    side, off = davet.davet_pyramid_layout(w.grid, w.n_levels, w.tiles[0])
    pyr = torch.empty((off[-1], w.C), dtype=torch.bfloat16, device="cuda")
    pyr[: off[1]].copy_(feat.reshape(-1, w.C))
    davet.davet_build_pyramid(pyr, pyr, w.tiles[0], w.grid, w.n_levels, w.C)
    torch.cuda.synchronize()
    got = pyr.cpu()
    for t in (0, 9):
        ref = oracle.pyramid(feat[t:t + 1], 1, w.grid, w.n_levels, w.C)
        scale = oracle.pyramid_f64(np.abs(bf16_to_f64(feat[t:t + 1])), w.n_levels)
        ref_off = oracle.level_offsets(w.grid, w.n_levels, 1)
        for lvl, g in enumerate(side):
            n = g * g
            mine = bf16_to_f64(got[off[lvl] + t * n: off[lvl] + (t + 1) * n])
            assert check_bf16_rounding(mine, ref[ref_off[lvl]:ref_off[lvl + 1]],
                                       scale[ref_off[lvl]:ref_off[lvl + 1]]) == 0
