"""Pins for the oracle's evidence pyramid (Sec. 4.3, structured pooling).

Each check ties the oracle to something other than itself: a constant field,
the identity level, a closed form of the 2x2 valid-children cascade on 3x3
grids enumerated exhaustively, direct block means on even grids, PyTorch's
ceil-mode average pooling, and linearity.
"""
import itertools

import numpy as np
import pytest

import oracle


def test_level_sides():
    assert oracle.level_sides(27, 4) == [27, 14, 7, 4]
    assert oracle.level_sides(12, 3) == [12, 6, 3]
    assert oracle.level_sides(1, 3) == [1, 1, 1]
    assert oracle.level_offsets(27, 4, 5) == [0, 5 * 729, 5 * 925, 5 * 974, 5 * 990]


@pytest.mark.parametrize("grid,levels", [(27, 4), (12, 3), (5, 4), (1, 2), (2, 2)])
def test_constant_grid_pools_to_constant(grid, levels):
    rng = np.random.default_rng(grid)
    n_tiles, C = 3, 5
    consts = rng.normal(size=(n_tiles, C))
    feat = np.broadcast_to(consts[:, None, None, :], (n_tiles, grid, grid, C)).copy()
    out = oracle.pyramid_f64(feat, levels)
    off = oracle.level_offsets(grid, levels, n_tiles)
    sides = oracle.level_sides(grid, levels)
    for lvl, g in enumerate(sides):
        blk = out[off[lvl]:off[lvl + 1]].reshape(n_tiles, g * g, C)
        np.testing.assert_allclose(blk, np.broadcast_to(consts[:, None, :], blk.shape), rtol=0, atol=1e-15)


def test_level0_is_identity_bf16():
    import torch
    feat = torch.randn(2, 27, 27, 16).to(torch.bfloat16)
    out = oracle.pyramid(feat, 2, 27, 4, 16)
    np.testing.assert_array_equal(out[: 2 * 729], feat.float().double().reshape(-1, 16).numpy())


def test_3x3_exhaustive_closed_form():
    # every 3x3 grid over {-1, 0, 1}: 3^9 tiles with one channel
    grids = np.array(list(itertools.product((-1.0, 0.0, 1.0), repeat=9))).reshape(-1, 3, 3, 1)
    n = grids.shape[0]
    out = oracle.pyramid_f64(grids, 3)
    off = oracle.level_offsets(3, 3, n)
    l1 = out[off[1]:off[2], 0].reshape(n, 2, 2)
    l2 = out[off[2]:off[3], 0].reshape(n)
    x = grids[..., 0]
    # level 1: means over the in-range children of each 2x2 window
    np.testing.assert_array_equal(l1[:, 0, 0], (x[:, 0, 0] + x[:, 0, 1] + x[:, 1, 0] + x[:, 1, 1]) / 4)
    np.testing.assert_array_equal(l1[:, 0, 1], (x[:, 0, 2] + x[:, 1, 2]) / 2)
    np.testing.assert_array_equal(l1[:, 1, 0], (x[:, 2, 0] + x[:, 2, 1]) / 2)
    np.testing.assert_array_equal(l1[:, 1, 1], x[:, 2, 2])
    # level 2 of the cascade: equal weight per level-1 cell, so weights are
    # 1/16 on the full window, 1/8 on the edge pairs, 1/4 on the corner
    w = np.array([[1 / 16, 1 / 16, 1 / 8], [1 / 16, 1 / 16, 1 / 8], [1 / 8, 1 / 8, 1 / 4]])
    assert w.sum() == 1.0
    np.testing.assert_allclose(l2, np.einsum("nij,ij->n", x, w), rtol=0, atol=1e-15)


@pytest.mark.parametrize("grid,levels", [(12, 3), (16, 5), (8, 4)])
def test_even_grid_equals_direct_block_mean(grid, levels):
    rng = np.random.default_rng(7)
    n_tiles, C = 2, 3
    feat = rng.normal(size=(n_tiles, grid, grid, C))
    out = oracle.pyramid_f64(feat, levels)
    off = oracle.level_offsets(grid, levels, n_tiles)
    for lvl in range(levels):
        b = 2 ** lvl
        g = grid // b
        direct = feat.reshape(n_tiles, g, b, g, b, C).mean(axis=(2, 4))
        np.testing.assert_allclose(out[off[lvl]:off[lvl + 1]].reshape(n_tiles, g, g, C), direct,
                                   rtol=1e-13, atol=1e-14)


@pytest.mark.parametrize("grid", [27, 13, 7])
def test_odd_grid_matches_ceil_mode_avg_pool_cascade(grid):
    torch = pytest.importorskip("torch")
    F = torch.nn.functional
    rng = np.random.default_rng(grid)
    n_tiles, C, levels = 2, 4, 4
    feat = rng.normal(size=(n_tiles, grid, grid, C))
    out = oracle.pyramid_f64(feat, levels)
    off = oracle.level_offsets(grid, levels, n_tiles)
    x = torch.from_numpy(feat).permute(0, 3, 1, 2)  # N C H W, float64
    for lvl in range(levels):
        g = x.shape[-1]
        ref = x.permute(0, 2, 3, 1).reshape(n_tiles, g * g, C).numpy()
        np.testing.assert_allclose(out[off[lvl]:off[lvl + 1]].reshape(n_tiles, g * g, C), ref,
                                   rtol=1e-13, atol=1e-14)
        # ceil mode, no padding: edge windows divide by their in-range count
        x = F.avg_pool2d(x, kernel_size=2, stride=2, ceil_mode=True)


def test_linearity():
    rng = np.random.default_rng(3)
    X = rng.normal(size=(2, 27, 27, 3))
    Y = rng.normal(size=(2, 27, 27, 3))
    a, b = 0.75, -2.5
    lhs = oracle.pyramid_f64(a * X + b * Y, 4)
    rhs = a * oracle.pyramid_f64(X, 4) + b * oracle.pyramid_f64(Y, 4)
    np.testing.assert_allclose(lhs, rhs, rtol=1e-12, atol=1e-12)


def test_tiles_are_independent():
    rng = np.random.default_rng(11)
    X = rng.normal(size=(3, 27, 27, 2))
    full = oracle.pyramid_f64(X, 4)
    off3 = oracle.level_offsets(27, 4, 3)
    for t in range(3):
        one = oracle.pyramid_f64(X[t:t + 1], 4)
        off1 = oracle.level_offsets(27, 4, 1)
        for lvl in range(4):
            n = off1[lvl + 1] - off1[lvl]
            np.testing.assert_array_equal(full[off3[lvl] + t * n: off3[lvl] + (t + 1) * n],
                                          one[off1[lvl]:off1[lvl + 1]])
