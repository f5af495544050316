"""Host-side checks of the C ABI library that need no GPU: it builds for
sm_103a, loads, exports every entry point declared in include/davet.h, and
rejects invalid arguments with a status code before touching the device."""
import ctypes
import os
import re

import pytest

import oracle

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    import paper_2608_01821_gb300 as pkg
    pkg.build()
    from paper_2608_01821_gb300 import davet
    return davet.load_cdll()


def declared_functions():
    src = open(os.path.join(ROOT, "include", "davet.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(davet_[a-z0-9_]+)\s*\(", src)))


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert "davet_build_pyramid" in names and "davet_unmask_topk" in names
    for n in names:
        assert hasattr(lib, n), n


def test_status_strings_and_version(lib):
    for code in range(6):
        assert lib.davet_status_string(code)
    assert lib.davet_status_string(99) == b"unknown status"
    assert lib.davet_version() >= 100


@pytest.mark.parametrize("grid,levels,tiles", [(27, 4, 1), (27, 4, 10), (12, 3, 1), (5, 5, 3), (1, 1, 2)])
def test_pyramid_layout_matches_oracle(lib, grid, levels, tiles):
    side = (ctypes.c_int * levels)()
    off = (ctypes.c_int64 * (levels + 1))()
    assert lib.davet_pyramid_layout(grid, levels, tiles, side, off) == 0
    assert list(side) == oracle.level_sides(grid, levels)
    assert list(off) == oracle.level_offsets(grid, levels, tiles)


@pytest.mark.parametrize("grid,levels,mixed_level,stride", [(27, 4, 2, 3), (27, 4, 3, 4), (12, 3, 2, 3), (5, 3, 1, 1),
                                                             (27, 4, 0, 27), (1, 1, 0, 1)])
def test_mixed_view_rows_matches_oracle(lib, grid, levels, mixed_level, stride):
    n = ctypes.c_int(-1)
    assert lib.davet_mixed_view_rows(grid, levels, mixed_level, stride, ctypes.byref(n)) == 0
    assert n.value == oracle.mixed_rows_per_tile(grid, levels, mixed_level, stride)


def test_mixed_view_rows_rejects_out_of_range(lib):
    n = ctypes.c_int(-1)
    for args in [(27, 4, 4, 3), (27, 4, -1, 3), (27, 4, 2, 0), (27, 4, 2, 28), (27, 6, 2, 3), (0, 4, 0, 1)]:
        assert lib.davet_mixed_view_rows(*args, ctypes.byref(n)) == 1
    assert n.value == -1


def test_invalid_arguments_are_rejected_without_a_device(lib):
    INV, UNS = 1, 2
    p = ctypes.c_void_p(1 << 20)  # never dereferenced: validation fails first
    null = None
    assert lib.davet_pyramid_layout(0, 4, 1, None, None) == INV
    assert lib.davet_pyramid_layout(27, 6, 1, None, None) == INV
    # pyramid: C not a multiple of 8, null pointers, misalignment, too many levels
    assert lib.davet_build_pyramid(p, p, 1, 27, 4, 12, null, null) == INV
    assert lib.davet_build_pyramid(null, p, 1, 27, 4, 16, null, null) == INV
    assert lib.davet_build_pyramid(ctypes.c_void_p((1 << 20) + 2), p, 1, 27, 4, 16, null, null) == INV
    assert lib.davet_build_pyramid(p, p, 1, 27, 6, 16, null, null) == UNS
    assert lib.davet_build_pyramid(p, p, 0, 27, 4, 16, null, null) == 0  # no tiles: no-op
    # attention: unsupported head dim, bad scale, null pointers
    f = ctypes.c_float
    assert lib.davet_step_attention(p, p, 1, 128, 4, 96, f(0.1), p, null) == UNS
    assert lib.davet_step_attention(p, p, 1, 128, 4, 64, f(0.0), p, null) == INV
    assert lib.davet_step_attention(null, p, 1, 128, 4, 64, f(0.1), p, null) == INV
    assert lib.davet_step_attention(p, p, 2000, 128, 4, 64, f(0.1), p, null) == UNS
    assert lib.davet_step_attention(p, p, 0, 128, 4, 64, f(0.1), p, null) == 0  # empty batch
    # fused view attention: batch above its limit, bad head dim, null store
    assert lib.davet_view_attention(p, 10, p, p, p, p, p, 300, 27, 4, 0, 0, 4, 64, f(0.1), p, p, 100, null) == UNS
    assert lib.davet_view_attention(p, 10, p, p, p, p, p, 1, 27, 4, 0, 0, 4, 96, f(0.1), p, p, 100, null) == UNS
    assert lib.davet_view_attention(null, 10, p, p, p, p, p, 1, 27, 4, 0, 0, 4, 64, f(0.1), p, p, 100, null) == INV
    assert lib.davet_view_attention(p, 10, p, p, p, p, p, 1, 27, 4, 5, 3, 4, 64, f(0.1), p, p, 100, null) == INV
    # view blocks: layout helpers against the pyramid layout plus text rows
    off = (ctypes.c_int64 * 6)()
    assert lib.davet_view_layout(27, 4, 2, 3, 2, 50, off) == 0
    assert list(off)[:6] == [0, 2 * 729 + 50, 2 * 729 + 2 * 196 + 100, 2 * (729 + 196 + 49) + 150,
                             2 * (729 + 196 + 49 + 16) + 200, 2 * (729 + 196 + 49 + 16 + 130) + 250]
    nv = ctypes.c_int(0)
    assert lib.davet_view_rows(27, 4, 0, 0, None, ctypes.byref(nv)) == 0 and nv.value == 4
    assert lib.davet_view_layout(27, 4, 5, 3, 2, 50, off) == INV
    assert lib.davet_build_views(p, p, null, 1, 27, 4, 0, 0, 5, 16, null) == INV  # text rows without text
    # realizers: pruning needs a score and cannot keep more rows than a tile has
    assert lib.davet_build_views_pruned(p, null, p, null, 1, 27, 4, 0, 0, 0, 16, null) == INV
    assert lib.davet_build_views_pruned(p, p, p, null, 1, 27, 4, 2, 1, 0, 16, null) == INV  # 49 + 729 rows
    assert lib.davet_build_views_pruned(p, p, p, null, 1, 65, 4, 0, 0, 0, 16, null) == UNS
    assert lib.davet_build_views_pruned(null, null, null, null, 0, 27, 4, 0, 0, 0, 16, null) == 0  # empty
    # merging: similarity channels, workspace size, geometry limits
    ws = ctypes.c_size_t(0)
    assert lib.davet_merge_workspace_bytes(10, 27, 4, 4096, ctypes.byref(ws)) == 0 and ws.value > 0
    ws10 = ws.value
    assert lib.davet_merge_workspace_bytes(1, 27, 4, 4096, ctypes.byref(ws)) == 0 and ws.value < ws10
    assert lib.davet_merge_workspace_bytes(1, 27, 4, 48, ctypes.byref(ws)) == INV
    assert lib.davet_merge_workspace_bytes(1, 65, 4, 64, ctypes.byref(ws)) == UNS
    mw = ctypes.c_void_p(1 << 24)
    assert lib.davet_build_views_merged(p, p, null, 1, 27, 4, 0, 0, 0, 128, 0, 48, null, mw, ws10, null) == INV
    assert lib.davet_build_views_merged(p, p, null, 1, 27, 4, 0, 0, 0, 128, 104, 32, null, mw, ws10, null) == INV
    assert lib.davet_build_views_merged(p, p, null, 1, 27, 4, 0, 0, 0, 128, 4, 32, null, mw, ws10, null) == INV
    assert lib.davet_build_views_merged(p, p, null, 10, 27, 4, 0, 0, 0, 128, 0, 32, null, mw, 1024, null) == INV
    assert lib.davet_build_views_merged(p, p, null, 10, 27, 4, 0, 0, 0, 128, 0, 32, null, null, ws10, null) == INV
    assert lib.davet_build_views_merged(null, null, null, 0, 27, 4, 0, 0, 0, 128, 0, 32, null, null, 0, null, null) == 0
    # attention scratch query: none needed
    assert lib.davet_step_attention_workspace(4, 1000, 32, 128, ctypes.byref(sz0 := ctypes.c_size_t(7))) == 0
    assert sz0.value == 0
    assert lib.davet_step_attention_workspace(4, 1000, 32, 96, ctypes.byref(sz0)) == UNS
    assert lib.davet_step_attention_workspace(-1, 1000, 32, 128, ctypes.byref(sz0)) == INV
    # full-layer kernels: GEMM shapes, epilogue codes, rotary arguments, norms, embedding
    sz = ctypes.c_size_t(0)
    no_norm = (null, 0, ctypes.c_float(0), null, null, null)  # row_ss, parts, eps, ss_out, rows_dev, stream
    assert lib.davet_linear(p, 10, 100, p, 256, p, 0, null, null, 0, 0, 128, null, 0, null, 0, *no_norm) == INV
    assert lib.davet_linear(p, 10, 128, p, 100, p, 0, null, null, 0, 0, 128, null, 0, null, 0, *no_norm) == INV
    assert lib.davet_linear(p, 10, 128, p, 256, p, 7, null, null, 0, 0, 128, null, 0, null, 0, *no_norm) == INV
    assert lib.davet_linear(p, 10, 128, p, 256, p, 1, null, null, 0, 0, 128, null, 0, null, 0, *no_norm) == INV
    assert lib.davet_linear(p, 10, 128, p, 768, p, 3, null, p, 1, 512, 96, p, 16, null, 0, *no_norm) == INV
    assert lib.davet_linear(p, 10, 128, p, 768, p, 3, null, p, 1, 300, 128, p, 16, null, 0, *no_norm) == INV
    assert lib.davet_linear(p, -1, 128, p, 256, p, 0, null, null, 0, 0, 128, null, 0, null, 0, *no_norm) == INV
    assert lib.davet_linear(null, 0, 128, null, 256, null, 0, null, null, 0, 0, 128, null, 0, null, 0, *no_norm) == 0
    # folded normalization: parts >= 1, eps >= 0; sums of squares only from store / residual epilogues
    assert lib.davet_linear(p, 10, 128, p, 256, p, 0, null, null, 0, 0, 128, null, 0, null, 0, p, 0,
                            ctypes.c_float(1e-5), null, null, null) == INV
    assert lib.davet_linear(p, 10, 128, p, 256, p, 0, null, null, 0, 0, 128, null, 0, null, 0, p, 16,
                            ctypes.c_float(-1.0), null, null, null) == INV
    assert lib.davet_linear(p, 10, 128, p, 512, p, 2, null, null, 0, 0, 128, null, 0, null, 0, null, 0,
                            ctypes.c_float(0), p, null, null) == INV
    assert lib.davet_row_sumsq(p, 10, 12, p, null, null) == INV
    assert lib.davet_row_sumsq(p, 10, 16, null, null, null) == INV
    assert lib.davet_row_sumsq(null, 0, 16, null, null, null) == 0
    assert lib.davet_linear_workspace_bytes(10, 100, 256, ctypes.byref(sz)) == INV
    assert lib.davet_rope_table(16, 96, ctypes.c_double(1e4), p, null) == INV
    assert lib.davet_rope_table(16, 128, ctypes.c_double(1.0), p, null) == INV
    assert lib.davet_rmsnorm(p, 10, 12, p, ctypes.c_float(1e-5), p, null, null, 0, null, null) == INV
    assert lib.davet_rmsnorm(p, 10, 16, p, ctypes.c_float(1e-5), p, null, p, 0, null, null) == INV
    assert lib.davet_embed_answers(p, 100, 16, p, 100, p, p, 1, 5, p, null) == INV
    assert lib.davet_embed_answers(p, 100, 16, p, 3, p, p, 1, 0, p, null) == 0
    # masked-row staging: V, null buffers, alignment; nothing to copy is fine
    assert lib.davet_stage_masked_rows(p, 12, p, 4, p, null) == INV
    assert lib.davet_stage_masked_rows(null, 16, p, 4, p, null) == INV
    assert lib.davet_stage_masked_rows(ctypes.c_void_p((1 << 20) + 2), 16, p, 4, p, null) == INV
    assert lib.davet_stage_masked_rows(null, 16, null, 0, null, null) == 0
    # gather: bad levels count, batch too large
    assert lib.davet_gather_view(p, p, p, p, p, p, p, 1, 27, 0, 0, 0, 16, p, p, 100, null) == INV
    assert lib.davet_gather_view(p, p, p, p, p, p, p, 5000, 27, 4, 0, 0, 16, p, p, 100, null) == UNS
    # gather: mixed view with a level or stride out of range
    assert lib.davet_gather_view(p, p, p, p, p, p, p, 1, 27, 4, 4, 3, 16, p, p, 100, null) == INV
    assert lib.davet_gather_view(p, p, p, p, p, p, p, 1, 27, 4, 2, 28, 16, p, p, 100, null) == INV
    assert lib.davet_gather_view(p, p, p, p, p, p, p, 1, 27, 4, 2, -1, 16, p, p, 100, null) == INV
    # unmask: k out of range, V not a multiple of 8, workspace too small
    n = ctypes.c_size_t(0)
    assert lib.davet_unmask_topk_workspace(128, 1000, 1, ctypes.byref(n)) == 0 and n.value > 0
    ws_needed = n.value
    assert lib.davet_unmask_topk(p, 1000, p, 1, 128, 0, p, p, null, null, null, null, p, ws_needed, null) == INV
    assert lib.davet_unmask_topk(p, 1001, p, 1, 128, 2, p, p, null, null, null, null, p, ws_needed, null) == INV
    assert lib.davet_unmask_topk(p, 1000, p, 1, 128, 2, p, p, null, null, null, null, p, ws_needed - 1,
                                 null) == INV
    assert lib.davet_unmask_topk(p, 1000, p, 0, 128, 2, p, p, null, null, null, null, p, ws_needed, null) == 0
    # policy: bad T, orientation, budget; step past T; missing view table
    d = ctypes.c_double
    assert lib.davet_policy_envelope(0, 0, d(0.5), d(0.2), null, 1, p, p, null) == INV
    assert lib.davet_policy_envelope(16, 2, d(0.5), d(0.2), null, 1, p, p, null) == INV
    assert lib.davet_policy_envelope(16, 0, d(1.5), d(0.2), null, 1, p, p, null) == INV
    assert lib.davet_policy_envelope(16, 0, d(0.5), d(0.2), null, 0, p, p, null) == 0
    vl = (ctypes.c_int32 * 3)(2, 1, 0)
    assert lib.davet_policy_step(16, 16, p, p, null, 1, d(0.5), vl, p, null, null) == INV
    assert lib.davet_policy_step(0, 16, p, p, null, 1, d(1.5), vl, p, null, null) == INV
    assert lib.davet_policy_step(0, 16, p, p, null, 1, d(0.5), None, p, null, null) == INV


def test_noalloc_validates_before_touching_the_device(lib):
    """davet_unmask_topk_noalloc returns its argument and size statuses
    before any device call, so they hold on a machine without a GPU.  Its
    scratch array is DAVET_NOALLOC_SCRATCH_BYTES (1 MiB); with one vocabulary
    chunk per row a row needs a 16-byte chunk record, a 4-byte confidence and
    a 4-byte index, each array starting on a 256-byte boundary.  One row more
    than that holds is rejected as unsupported; pointers are never read."""
    OK, INV, UNS = 0, 1, 2
    p = ctypes.c_void_p(1 << 20)
    scratch = 1 << 20

    def a256(x):
        return (x + 255) & ~255

    rows = scratch // 24
    while a256(16 * rows) + 2 * a256(4 * rows) > scratch:
        rows -= 1
    for V in (1024, 126464):
        assert lib.davet_unmask_topk_noalloc(p, V, p, 1, rows + 1, 2, p, p, None, None, None, None, None) == UNS
    assert lib.davet_unmask_topk_noalloc(p, 126464, p, 1, 1 << 40, 2, p, p, None, None, None, None, None) == UNS
    assert lib.davet_unmask_topk_noalloc(p, 126464, p, 70000, 100, 2, p, p, None, None, None, None, None) == UNS
    # argument errors: V not a multiple of 8, k out of range, null state,
    # logits off a 16-byte boundary, negative sizes
    assert lib.davet_unmask_topk_noalloc(p, 1001, p, 1, 10, 2, p, p, None, None, None, None, None) == INV
    assert lib.davet_unmask_topk_noalloc(p, 1024, p, 1, 10, 0, p, p, None, None, None, None, None) == INV
    assert lib.davet_unmask_topk_noalloc(p, 1024, p, 1, 10, 1025, p, p, None, None, None, None, None) == INV
    assert lib.davet_unmask_topk_noalloc(p, 1024, None, 1, 10, 2, p, p, None, None, None, None, None) == INV
    assert lib.davet_unmask_topk_noalloc(p, 1024, p, 1, 10, 2, None, p, None, None, None, None, None) == INV
    assert lib.davet_unmask_topk_noalloc(None, 1024, p, 1, 10, 2, p, p, None, None, None, None, None) == INV
    odd = ctypes.c_void_p((1 << 20) + 8)
    assert lib.davet_unmask_topk_noalloc(odd, 1024, p, 1, 10, 2, p, p, None, None, None, None, None) == INV
    assert lib.davet_unmask_topk_noalloc(p, 1024, p, 1, -1, 2, p, p, None, None, None, None, None) == INV
    assert lib.davet_unmask_topk_noalloc(p, 1024, p, -1, 10, 2, p, p, None, None, None, None, None) == INV
    # no requests: nothing to do
    assert lib.davet_unmask_topk_noalloc(p, 1024, p, 0, 0, 2, p, p, None, None, None, None, None) == OK


def test_package_fails_loudly_without_library(tmp_path):
    from paper_2608_01821_gb300 import davet
    saved = davet._lib
    davet._lib = None
    try:
        with pytest.raises(RuntimeError, match="no fallback"):
            davet.load_cdll(str(tmp_path / "missing.so"))
    finally:
        davet._lib = saved
