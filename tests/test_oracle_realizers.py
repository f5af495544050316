"""Pins for the oracle's alternative evidence realizers (Sec. 4.3 "compatible
evidence realizers": pruning varies the retention ratio, merging the
aggregation strength; Sec. 5.3 / Table 2).

Pruning is pinned to a stable library sort; merging to closed forms
(constant tiles, a one-cell top level is the tile mean), partition and
nesting invariants, the member-mean rule in fp64, single rounds against
scipy's cosine distance, and a 4x4 example worked by hand."""
import math

import numpy as np
import pytest
import torch
from scipy.spatial.distance import cdist

import oracle


def u16(x: torch.Tensor) -> np.ndarray:
    return x.contiguous().view(torch.int16).numpy().view(np.uint16)


def f64(bits: np.ndarray) -> np.ndarray:
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).double().numpy()


def bf16_rne(x: np.ndarray) -> np.ndarray:
    return u16(torch.from_numpy(np.asarray(x, np.float64)).to(torch.bfloat16))


# ------------------------------------------------------------------ pruning
@pytest.mark.parametrize("grid,views", [(27, [729, 196, 130, 49, 16]), (12, [144, 36, 25, 9]), (5, [25, 1])])
def test_prune_matches_stable_library_sort(grid, views):
    rng = np.random.default_rng(grid)
    n_tiles = 3
    s = rng.standard_normal((n_tiles, grid * grid)).astype(np.float32)
    s[1, ::7] = s[1, 3]  # ties inside one tile
    keep = oracle.prune_keep(s, n_tiles, grid, views)
    for v, m in enumerate(views):
        for t in range(n_tiles):
            want = np.sort(np.argsort(-s[t], kind="stable")[:m])
            assert np.array_equal(keep[v][t], want)


def test_prune_nesting_identity_and_nan_rule():
    grid, n_tiles = 9, 2
    views = [81, 40, 25, 7, 1]
    rng = np.random.default_rng(7)
    s = rng.standard_normal((n_tiles, 81)).astype(np.float32)
    s[0, [4, 50, 77]] = np.nan
    s[1, :] = 0.5  # all equal: the first m tokens in raster order
    keep = oracle.prune_keep(s, n_tiles, grid, views)
    assert np.array_equal(keep[0][0], np.arange(81)) and np.array_equal(keep[0][1], np.arange(81))
    for v in range(1, len(views)):
        for t in range(n_tiles):
            assert set(keep[v][t]) <= set(keep[v - 1][t])
            assert np.all(np.diff(keep[v][t]) > 0)
        assert np.array_equal(keep[v][1], np.arange(views[v]))
    # the three NaN tokens rank last: only the 81-token view keeps them
    assert not set(keep[1][0]) & {4, 50, 77}
    assert len(set(keep[1][0]) | {4, 50, 77}) == 43


def test_prune_views_are_rows_of_the_encoding():
    grid, n_tiles, C = 6, 2, 16
    feat = torch.randn(n_tiles, grid * grid, C).to(torch.bfloat16)
    s = np.random.default_rng(3).standard_normal((n_tiles, grid * grid)).astype(np.float32)
    views = [36, 9, 4]
    rows = oracle.prune_views(feat, s, n_tiles, grid, views, C)
    keep = oracle.prune_keep(s, n_tiles, grid, views)
    fb = u16(feat)
    for v in range(3):
        want = np.concatenate([fb[t, keep[v][t]] for t in range(n_tiles)])
        assert np.array_equal(rows[v], want)


# ------------------------------------------------------------------ merging
def check_partitions(assign, sides):
    """Level l has G_l^2 non-empty tokens and coarsens level l-1."""
    L, n_tiles, n0 = assign.shape
    assert np.array_equal(assign[0], np.tile(np.arange(n0), (n_tiles, 1)))
    for l in range(1, L):
        for t in range(n_tiles):
            a = assign[l, t]
            assert np.array_equal(np.unique(a), np.arange(sides[l] ** 2))
            prev = assign[l - 1, t]
            for j in np.unique(prev):
                assert len(np.unique(a[prev == j])) == 1


def test_merge_constant_tile_is_constant_at_every_level():
    grid, levels, n_tiles, C = 12, 3, 2, 32
    v = torch.randn(C).to(torch.bfloat16)
    feat = v.expand(n_tiles, grid * grid, C).contiguous()
    lv, assign = oracle.merge_views(feat, n_tiles, grid, levels, C, 0, C)
    check_partitions(assign, oracle.level_sides(grid, levels))
    for l in range(levels):
        assert np.array_equal(lv[l], np.tile(u16(v), (lv[l].shape[0], 1)))


@pytest.mark.parametrize("grid,levels", [(8, 4), (27, 6)])
def test_merge_single_cell_top_level_is_the_tile_mean(grid, levels):
    sides = oracle.level_sides(grid, levels)
    assert sides[-1] == 1
    n_tiles, C = 2, 64
    feat = torch.randn(n_tiles, grid * grid, C).to(torch.bfloat16)
    lv, assign = oracle.merge_views(feat, n_tiles, grid, levels, C, 16, 32)
    check_partitions(assign, sides)
    mean = feat.double().mean(dim=1).numpy()
    got = f64(lv[-1])
    # binary32 sum of <= 729 terms, then one bf16 rounding
    assert np.all(np.abs(got - mean) <= np.abs(mean) * 2.0 ** -8 + 1e-5)


def test_merge_rows_are_member_means():
    grid, levels, n_tiles, C = 12, 3, 3, 48
    feat = torch.randn(n_tiles, grid * grid, C).to(torch.bfloat16)
    lv, assign = oracle.merge_views(feat, n_tiles, grid, levels, C, 8, 32)
    sides = oracle.level_sides(grid, levels)
    check_partitions(assign, sides)
    x = feat.double().numpy()
    for l in range(1, levels):
        m = sides[l] ** 2
        ref = np.stack([np.stack([x[t, assign[l, t] == j].mean(axis=0) for j in range(m)]) for t in range(n_tiles)])
        ref = ref.reshape(n_tiles * m, C)
        got = f64(lv[l])
        assert np.all(np.abs(got - ref) <= np.abs(ref) * 2.0 ** -8 + 1e-6)
        # rounding to nearest: most rows equal RNE(fp64 mean) exactly
        assert (lv[l] == bf16_rne(ref)).mean() > 0.99


@pytest.mark.parametrize("n,target", [(144, 36), (72, 36), (37, 20), (2, 1)])
def test_single_round_against_library_cosine(n, target):
    """A = even positions, B = odd positions; every member of A is matched to
    the B of highest cosine similarity (scipy's cosine distance, fp64); the r
    best-matched members of A merge; survivors keep their order."""
    rng = np.random.default_rng(n)
    C, c0, Cs = 40, 8, 24
    n0 = n
    feat = torch.from_numpy(rng.standard_normal((n0, C))).to(torch.bfloat16)
    tok = np.arange(n0, dtype=np.int32)
    nA = (n + 1) // 2
    r = min(n - target, nA)
    new, m, best, best_b = oracle.merge_round(feat, C, c0, Cs, tok, n, r)
    assert m == n - r
    X = feat.double().numpy()[:, c0:c0 + Cs]
    sim = 1.0 - cdist(X[0::2], X[1::2], metric="cosine")
    for a in range(nA):
        order = np.argsort(-sim[a], kind="stable")
        if len(order) > 1 and sim[a, order[0]] - sim[a, order[1]] < 1e-5:
            continue
        assert best_b[a] == order[0]
        assert abs(best[a] - sim[a, order[0]]) < 1e-5
    top = sim.max(axis=1)
    rank = np.argsort(-top, kind="stable")
    merged = set(rank[:r].tolist())
    if r < nA:
        assert top[rank[r - 1]] - top[rank[r]] > 1e-5  # seeded inputs have no near-tie at the cut
    # survivors keep their relative order and merged members follow their match
    surv = [p for p in range(n) if not (p % 2 == 0 and p // 2 in merged)]
    assert len(surv) == m
    for p in range(n):
        i = p  # level-0 token i sits at position i before the first round
        if p % 2 == 0 and p // 2 in merged:
            assert new[i] == surv.index(2 * int(best_b[p // 2]) + 1)
        else:
            assert new[i] == surv.index(p)


def test_worked_example_4x4_two_rounds():
    """Hand-derived: 16 unit vectors in the plane (C = Cs = 2).

    B_j (position 2j+1) points at angle beta_j; A_k (position 2k) at
    beta_sigma(k) + 5 degrees, so round 1 (n = 16 -> 4: r = min(12, 8) = 8,
    every member of A merges) sends A_k into B_sigma(k); token j of the 8
    survivors is then B_j plus one A, pointing at beta_j + 2.5 degrees.
    Round 2 (8 -> 4, r = 4): A = tokens 0, 2, 4, 6 at 2.5, 92.5, 182.5, 272.5
    degrees, B = tokens 1, 3, 5, 7 at 42.5, 132.5, 222.5, 312.5: each A is
    40 degrees from the next B and 50 from the previous one, so token 2i
    joins token 2i+1 and level 1 holds {B_2i, B_2i+1 and their A's}."""
    beta = [0, 40, 90, 130, 180, 220, 270, 310]
    sigma = [3, 0, 6, 1, 7, 2, 5, 4]
    ang = np.zeros(16)
    for j in range(8):
        ang[2 * j + 1] = beta[j]
    for k in range(8):
        ang[2 * k] = beta[sigma[k]] + 5
    x = np.stack([np.cos(np.radians(ang)), np.sin(np.radians(ang))], axis=1)
    feat = torch.from_numpy(x).to(torch.bfloat16).reshape(1, 16, 2)
    lv, assign = oracle.merge_views(feat, 1, 4, 2, 2, 0, 2)
    want = np.zeros(16, np.int32)
    for j in range(8):
        want[2 * j + 1] = j // 2
    for k in range(8):
        want[2 * k] = sigma[k] // 2
    assert np.array_equal(assign[1, 0], want)
    xb = feat.double().numpy()[0]
    for t in range(4):
        ref = xb[want == t].mean(axis=0)
        assert np.all(np.abs(f64(lv[1][t]) - ref) <= np.abs(ref) * 2.0 ** -8 + 1e-6)


def test_merge_rounds_per_level_reach_the_pooled_counts():
    """Each level holds exactly the pooled level's row count (so every view
    has the pooled hierarchy's length), and a level built from n tokens takes
    the rounds r = min(n - G_l^2, ceil(n/2)) prescribes."""
    grid, levels, C = 27, 4, 32
    feat = torch.randn(1, grid * grid, C).to(torch.bfloat16)
    lv, assign = oracle.merge_views(feat, 1, grid, levels, C, 0, 32)
    sides = oracle.level_sides(grid, levels)
    assert [x.shape[0] for x in lv] == [g * g for g in sides] == [729, 196, 49, 16]
    check_partitions(assign, sides)
    n, rounds = 729, []
    for g in sides[1:]:
        while n > g * g:
            r = min(n - g * g, math.ceil(n / 2))
            rounds.append(r)
            n -= r
    assert rounds == [365, 168, 98, 49, 25, 8]


def test_merged_mixed_view_is_merged_coarse_plus_lattice():
    """The mixed view of the merging hierarchy takes the merged coarse level
    and the same level-0 lattice as the pooled one (Sec. 4.3)."""
    grid, levels, n_tiles, C = 12, 3, 2, 16
    feat = torch.randn(n_tiles, grid * grid, C).to(torch.bfloat16)
    lv, _ = oracle.merge_views(feat, n_tiles, grid, levels, C, 0, 16)
    pyr = np.concatenate(lv)
    mixed = oracle.mixed_view(torch.from_numpy(pyr.view(np.int16)).view(torch.bfloat16), n_tiles, grid, levels,
                              2, 3, C)
    per = oracle.mixed_rows_per_tile(grid, levels, 2, 3)
    for t in range(n_tiles):
        blk = mixed[t * per:(t + 1) * per]
        assert np.array_equal(blk[:9], lv[2][t * 9:(t + 1) * 9])
        lat = [y * grid + x for y in range(1, grid, 3) for x in range(1, grid, 3)]
        assert np.array_equal(blk[9:], u16(feat)[t, lat])
