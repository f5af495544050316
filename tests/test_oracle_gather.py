"""Pins for the oracle's view gather (Sec. 3.2 / Eq. 5: the step input is the
selected view v_t followed by the query and the answer state).

Rows carry their own identity (request, level, tile, cell or text index)
encoded in bf16-exact integers, so the packed layout can be checked row by
row against an index list built independently here.
"""
import numpy as np
import torch

import oracle


def encode(ids, C):
    """Row r gets its small integer ids in the first channels (exact in bf16)."""
    ids = np.asarray(ids, dtype=np.float32).reshape(len(ids), 5)
    out = np.zeros((ids.shape[0], C), np.float32)
    out[:, : ids.shape[1]] = ids
    return torch.from_numpy(out).to(torch.bfloat16)


def build_inputs(tiles, prompt, resp, grid, levels, C):
    sides = oracle.level_sides(grid, levels)
    pyrs = []
    for b, nt in enumerate(tiles):
        ids = []
        for lvl, g in enumerate(sides):
            for t in range(nt):
                for cell in range(g * g):
                    ids.append([b, lvl, t, cell % 128, cell // 128])
        pyrs.append(encode(ids, C))
    text_ids = []
    for b in range(len(tiles)):
        for j in range(prompt[b] + resp[b]):
            text_ids.append([b, 100, j % 128, j // 128, 0])
    text = encode(text_ids, C)
    text_off = np.concatenate([[0], np.cumsum(np.add(prompt, resp))[:-1]])
    return pyrs, text, text_off, sides


def test_packed_layout_and_lengths():
    grid, levels, C = 27, 4, 8
    tiles, prompt, resp = [2, 1, 3], [5, 0, 7], [4, 3, 0]
    pyrs, text, text_off, sides = build_inputs(tiles, prompt, resp, grid, levels, C)
    level = [3, 0, 1]
    out, cu = oracle.gather(pyrs, tiles, text, text_off, prompt, resp, level, grid, levels, C)
    L = [tiles[b] * sides[level[b]] ** 2 + prompt[b] + resp[b] for b in range(3)]
    assert list(cu) == [0, L[0], L[0] + L[1], sum(L)]
    got = torch.from_numpy(out.view(np.int16)).view(torch.bfloat16).float().numpy()
    r = 0
    for b in range(3):
        g = sides[level[b]]
        for t in range(tiles[b]):
            for cell in range(g * g):
                assert list(got[r, :5]) == [b, level[b], t, cell % 128, cell // 128]
                r += 1
        for j in range(prompt[b] + resp[b]):
            assert list(got[r, :5]) == [b, 100, j % 128, j // 128, 0]
            r += 1
    assert r == out.shape[0]


def test_level0_view_is_the_encoding_and_bits_are_copied():
    grid, levels, C = 12, 3, 16
    g = torch.Generator().manual_seed(0)
    feat = torch.randn(2, grid, grid, C, generator=g).to(torch.bfloat16)
    pyr64 = oracle.pyramid(feat, 2, grid, levels, C)
    pyr = torch.from_numpy(pyr64).float().to(torch.bfloat16)
    text = torch.randn(9, C, generator=g).to(torch.bfloat16)
    out, cu = oracle.gather([pyr], [2], text, [0], [4], [5], [0], grid, levels, C)
    assert list(cu) == [0, 2 * 144 + 9]
    assert np.array_equal(out[:288], feat.reshape(288, C).view(torch.int16).numpy().view(np.uint16))
    assert np.array_equal(out[288:], text.view(torch.int16).numpy().view(np.uint16))


def test_empty_text_and_coarsest_level():
    grid, levels, C = 3, 2, 8
    pyrs, text, text_off, sides = build_inputs([1], [0], [0], grid, levels, C)
    assert sides == [3, 2]
    out, cu = oracle.gather(pyrs, [1], np.zeros((1, C), np.uint16), [0], [0], [0], [1], grid, levels, C)
    assert list(cu) == [0, 4]
