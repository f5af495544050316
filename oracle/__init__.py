"""Plain fp64 CPU oracle for the DAVET step-conditioning path.

TEST INFRASTRUCTURE ONLY.  The test suite, ``__graft_entry__.smoke()`` and
the CPU-baseline leg of ``bench.py`` are the only callers.  The CUDA library
never imports, links or runs anything here, and this package shares no code
with it.

The arithmetic lives in ``oracle.c`` (plain loops, double precision); this
module only compiles it with gcc, loads it with ctypes and marshals numpy
arrays.  Sections cited per function are those of the DAVET paper.

Parity status of each function (what pins it is listed in the tests under
``tests/test_oracle_*.py``):
  pyramid   pinned (constant grid, identity level, 3x3 brute force against the
            cascade closed form, even-grid block means, ceil-mode library
            pooling, linearity)
  gather    pinned (structural row-id identities)
  mixed     pinned (structural row-id identities, stride 1 = every token,
            ordered coarse < mixed < high lengths); the subset rule itself is
            a reading (a centred lattice), the paper prints none
  attention pinned (identical keys, single key, two-key sigmoid closed form,
            dominant key, permutation equivariance)
  unmask    pinned (closed-form confidences, tie rules, brute-force top-k)
  policy    pinned (Eq. 7-9 special cases, envelope mean and ordering
            invariants, Table D "High" step counts)
  prune     pinned (stable library sort, nesting, identity at full
            retention, NaN and tie rules); the score is an input (the paper
            does not define it)
  layer     pinned (rms_norm and silu against torch's library functions,
            rotary identities: position 0, pair norms, relative position,
            the first pair's angle; a zero layer is the identity, equal
            queries and keys give each request's mean value, a single-row
            request attends to itself); numpy fp64 in ``oracle/layer.py``
  merge     pinned (constant tiles, single-cell top level = tile mean,
            partition and nesting invariants, row = member mean in fp64,
            per-round greedy choices against an independent fp64 cosine,
            hand-worked 4x4 example); the matching rule is a reading
            (bipartite matching rounds), the paper prints none
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

_c_i32p = ctypes.POINTER(ctypes.c_int32)
_c_i64p = ctypes.POINTER(ctypes.c_int64)
_c_u16p = ctypes.POINTER(ctypes.c_uint16)
_c_u8p = ctypes.POINTER(ctypes.c_uint8)
_c_f64p = ctypes.POINTER(ctypes.c_double)


def build(force: bool = False) -> str:
    """Compile oracle.c into liboracle.so next to it (gcc, OpenMP)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(
            ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fPIC", "-shared", "-fopenmp", "-Wall",
             _SRC, "-o", tmp, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB)
            lib.oracle_level_sides.restype = ctypes.c_int64
            lib.oracle_mixed_view.restype = ctypes.c_int64
            lib.oracle_merge_round.restype = ctypes.c_int
            lib.oracle_policy_risk.restype = ctypes.c_double
            lib.oracle_policy_budget.restype = ctypes.c_double
            lib.oracle_policy_view.restype = ctypes.c_int
            lib.oracle_max_threads.restype = ctypes.c_int
            _lib = lib
    return _lib


def _ptr(a: np.ndarray, ctype):
    assert a.flags.c_contiguous
    return a.ctypes.data_as(ctype)


def _as_u16(x) -> np.ndarray:
    """Accept a numpy uint16 array holding bf16 bit patterns, or a torch
    bfloat16 tensor, and return a contiguous uint16 view."""
    if hasattr(x, "dtype") and str(x.dtype) == "torch.bfloat16":
        import torch
        return np.ascontiguousarray(x.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16))
    a = np.ascontiguousarray(x)
    assert a.dtype == np.uint16, a.dtype
    return a


def max_threads() -> int:
    return int(_load().oracle_max_threads())


def set_threads(n: int) -> None:
    _load().oracle_set_threads(int(n))


# ------------------------------------------------------------------ pyramid
def level_sides(grid: int, n_levels: int) -> list[int]:
    """G_0 = grid, G_l = ceil(G_{l-1}/2)."""
    side = (ctypes.c_int * n_levels)()
    _load().oracle_level_sides(grid, n_levels, side)
    return list(side)


def level_offsets(grid: int, n_levels: int, n_tiles: int) -> list[int]:
    """First row of each level in the level-major layout, plus the total."""
    off = [0]
    for g in level_sides(grid, n_levels):
        off.append(off[-1] + n_tiles * g * g)
    return off


def pyramid_f64(feat: np.ndarray, n_levels: int) -> np.ndarray:
    """feat: float64 [n_tiles, G, G, C] -> [rows, C] level-major (Sec. 4.3)."""
    feat = np.ascontiguousarray(feat, dtype=np.float64)
    n_tiles, g, g2, C = feat.shape
    assert g == g2
    rows = level_offsets(g, n_levels, n_tiles)[-1]
    out = np.empty((rows, C), dtype=np.float64)
    _load().oracle_pyramid_f64(_ptr(feat, _c_f64p), n_tiles, g, n_levels, C, _ptr(out, _c_f64p))
    return out


def pyramid(feat_bf16, n_tiles: int, grid: int, n_levels: int, C: int) -> np.ndarray:
    """bf16 bits [n_tiles*G*G*C] -> fp64 [rows, C] level-major (Sec. 4.3)."""
    f = _as_u16(feat_bf16).reshape(-1)
    assert f.size == n_tiles * grid * grid * C
    rows = level_offsets(grid, n_levels, n_tiles)[-1]
    out = np.empty((rows, C), dtype=np.float64)
    _load().oracle_pyramid_bf16(_ptr(f, _c_u16p), n_tiles, grid, n_levels, C, _ptr(out, _c_f64p))
    return out


# ------------------------------------------------------------------- gather
def mixed_rows_per_tile(grid: int, n_levels: int, coarse_level: int, stride: int) -> int:
    """Rows of the mixed view per tile: the coarse level plus the lattice."""
    g = level_sides(grid, n_levels)[coarse_level]
    n = len(range(stride // 2, grid, stride))
    return g * g + n * n


def mixed_view(pyr_bf16, n_tiles: int, grid: int, n_levels: int, coarse_level: int, stride: int, C: int):
    """The `mixed` view (Sec. 4.3) of one request's pyramid: uint16 [rows, C]."""
    p = _as_u16(pyr_bf16).reshape(-1)
    rows = n_tiles * mixed_rows_per_tile(grid, n_levels, coarse_level, stride)
    out = np.empty((rows, C), dtype=np.uint16)
    n = _load().oracle_mixed_view(_ptr(p, _c_u16p), n_tiles, grid, n_levels, coarse_level, stride, C,
                                  _ptr(out, _c_u16p))
    assert n == rows
    return out



def view_rows_per_tile(grid: int, n_levels: int, mixed=None) -> list[int]:
    """Rows per tile of every view: the pooled levels, then the mixed view."""
    rows = [g * g for g in level_sides(grid, n_levels)]
    if mixed is not None:
        rows.append(mixed_rows_per_tile(grid, n_levels, *mixed))
    return rows


# ---------------------------------------------------------------- realizers
def prune_keep(score, n_tiles: int, grid: int, rows_per_tile) -> list[np.ndarray]:
    """Nested pruning (Sec. 4.3, Sec. 5.3): per view, int32 [n_tiles, m_v] of
    the kept token indices of every tile (raster order)."""
    s = np.ascontiguousarray(np.asarray(score, dtype=np.float32).reshape(-1))
    assert s.size == n_tiles * grid * grid
    m = np.ascontiguousarray(rows_per_tile, dtype=np.int32)
    keep = np.empty(int(n_tiles * m.sum()), dtype=np.int32)
    _load().oracle_prune_keep(_ptr(s, ctypes.POINTER(ctypes.c_float)), n_tiles, grid, len(m), _ptr(m, _c_i32p),
                              _ptr(keep, _c_i32p))
    out, o = [], 0
    for mv in m:
        out.append(keep[o: o + n_tiles * mv].reshape(n_tiles, mv))
        o += n_tiles * mv
    return out


def prune_views(feat_bf16, score, n_tiles: int, grid: int, rows_per_tile, C: int) -> list[np.ndarray]:
    """Rows of every pruned view: uint16 [n_tiles * m_v, C] per view."""
    f = _as_u16(feat_bf16).reshape(n_tiles, grid * grid, C)
    return [np.concatenate([f[t, k[t]] for t in range(n_tiles)]) if n_tiles else np.empty((0, C), np.uint16)
            for k in prune_keep(score, n_tiles, grid, rows_per_tile)]


def merge_views(feat_bf16, n_tiles: int, grid: int, n_levels: int, C: int, c0: int, Cs: int):
    """Hierarchical similarity merging (Sec. 4.3, Sec. 5.3).

    Returns (levels, assign): levels[l] is uint16 [n_tiles * G_l^2, C] (level
    0 is the encoding itself) and assign is int32 [n_levels, n_tiles, grid^2],
    the level-l token each level-0 token belongs to."""
    f = _as_u16(feat_bf16).reshape(-1)
    assert f.size == n_tiles * grid * grid * C
    sides = level_sides(grid, n_levels)
    rows = sum(n_tiles * g * g for g in sides[1:])
    out = np.empty((max(rows, 1), C), dtype=np.uint16)
    assign = np.empty((n_levels, n_tiles, grid * grid), dtype=np.int32)
    _load().oracle_merge_views(_ptr(f, _c_u16p), n_tiles, grid, n_levels, C, c0, Cs, _ptr(out, _c_u16p),
                               _ptr(assign, _c_i32p))
    levels, o = [f.reshape(-1, C).copy()], 0
    for g in sides[1:]:
        levels.append(out[o: o + n_tiles * g * g])
        o += n_tiles * g * g
    return levels, assign


def merge_round(feat_bf16, C: int, c0: int, Cs: int, tok, n: int, r: int):
    """One bipartite matching round of one tile (Sec. 4.3 merging reading).

    feat: the tile's level-0 rows [n0, C]; tok: int32 [n0], the current token
    of every level-0 row.  Returns (new tok, new n, best sim [ceil(n/2)],
    matched B index [ceil(n/2)])."""
    f = _as_u16(feat_bf16).reshape(-1)
    n0 = f.size // C
    t = np.ascontiguousarray(tok, dtype=np.int32).copy()
    nA = (n + 1) // 2
    best = np.empty(max(nA, 1), dtype=np.float32)
    best_b = np.empty(max(nA, 1), dtype=np.int32)
    m = _load().oracle_merge_round(_ptr(f, _c_u16p), n0, C, c0, Cs, _ptr(t, _c_i32p), n, r,
                                   _ptr(best, ctypes.POINTER(ctypes.c_float)), _ptr(best_b, _c_i32p))
    return t, int(m), best[:nA], best_b[:nA]


def gather(pyrs, tiles, text_bf16, text_off, prompt_len, resp_len, level,
           grid: int, n_levels: int, C: int, mixed_rows_per_tile: int = 0):
    """Packed [view || prompt || response] rows per request (Eq. 5).

    pyrs: list of per-request bf16 pyramids (level-major rows x C), each
    followed by its mixed view when mixed_rows_per_tile > 0 (level index
    n_levels selects it).  Returns (packed uint16 [N, C], cu int32 [batch+1])."""
    batch = len(pyrs)
    p_arrs = [_as_u16(p).reshape(-1) for p in pyrs]
    ptrs = (_c_u16p * batch)(*[_ptr(p, _c_u16p) for p in p_arrs])
    tiles = np.ascontiguousarray(tiles, dtype=np.int32)
    text = _as_u16(text_bf16).reshape(-1)
    text_off = np.ascontiguousarray(text_off, dtype=np.int64)
    prompt_len = np.ascontiguousarray(prompt_len, dtype=np.int32)
    resp_len = np.ascontiguousarray(resp_len, dtype=np.int32)
    level = np.ascontiguousarray(level, dtype=np.int32)
    sides = level_sides(grid, n_levels) + [None]

    def vis(b):
        lv = int(level[b])
        return int(tiles[b]) * (sides[lv] ** 2 if lv < n_levels else mixed_rows_per_tile)

    total = int(sum(vis(b) + int(prompt_len[b]) + int(resp_len[b]) for b in range(batch)))
    out = np.empty((total, C), dtype=np.uint16)
    cu = np.empty(batch + 1, dtype=np.int32)
    _load().oracle_gather_mixed(ptrs, _ptr(tiles, _c_i32p), _ptr(text, _c_u16p), _ptr(text_off, _c_i64p),
                                _ptr(prompt_len, _c_i32p), _ptr(resp_len, _c_i32p), _ptr(level, _c_i32p),
                                batch, grid, n_levels, C, int(mixed_rows_per_tile), _ptr(out, _c_u16p),
                                _ptr(cu, _c_i32p))
    return out, cu


# ---------------------------------------------------------------- attention
def attention(qkv_bf16, cu, H: int, D: int, scale: float) -> np.ndarray:
    """Bidirectional attention (Eq. 1) for all rows: fp64 [N, H, D]."""
    q = _as_u16(qkv_bf16).reshape(-1)
    cu = np.ascontiguousarray(cu, dtype=np.int32)
    batch = cu.size - 1
    N = int(cu[-1])
    assert q.size >= N * 3 * H * D
    out = np.zeros((N, H, D), dtype=np.float64)
    _load().oracle_attention(_ptr(q, _c_u16p), _ptr(cu, _c_i32p), batch, H, D,
                             ctypes.c_double(scale), _ptr(out, _c_f64p))
    return out


def attention_rows(qkv_bf16, cu, H: int, D: int, scale: float, rows, heads) -> np.ndarray:
    """The same definition at sampled (row, head) pairs: fp64 [n, D]."""
    q = _as_u16(qkv_bf16).reshape(-1)
    cu = np.ascontiguousarray(cu, dtype=np.int32)
    rows = np.ascontiguousarray(rows, dtype=np.int64)
    heads = np.ascontiguousarray(heads, dtype=np.int32)
    assert rows.size == heads.size
    out = np.zeros((rows.size, D), dtype=np.float64)
    _load().oracle_attention_rows(_ptr(q, _c_u16p), _ptr(cu, _c_i32p), cu.size - 1, H, D,
                                  ctypes.c_double(scale), ctypes.c_int64(rows.size),
                                  _ptr(rows, _c_i64p), _ptr(heads, _c_i32p), _ptr(out, _c_f64p))
    return out


# ---------------------------------------------------------------- unmasking
def softmax_row(logits_bf16) -> np.ndarray:
    row = _as_u16(logits_bf16).reshape(-1)
    p = np.empty(row.size, dtype=np.float64)
    _load().oracle_softmax_row(_ptr(row, _c_u16p), row.size, _ptr(p, _c_f64p))
    return p


def unmask(logits_bf16, V: int, cu_resp, k: int, masked, tokens, argmax):
    """One confidence-ranked commitment step (Eq. 1-2).

    masked/tokens/argmax are updated in place (numpy uint8/int32/int32).
    Returns (conf fp64 [rows] (NaN where not masked), committed int32
    [batch, k], stats fp64 [batch, 2] = (mean conf, churn))."""
    lg = _as_u16(logits_bf16).reshape(-1)
    cu = np.ascontiguousarray(cu_resp, dtype=np.int32)
    batch = cu.size - 1
    rows = int(cu[-1])
    assert lg.size >= rows * V
    assert masked.dtype == np.uint8 and tokens.dtype == np.int32 and argmax.dtype == np.int32
    conf = np.full(rows, np.nan, dtype=np.float64)
    committed = np.empty((batch, k), dtype=np.int32)
    stats = np.empty((batch, 2), dtype=np.float64)
    _load().oracle_unmask(_ptr(lg, _c_u16p), V, _ptr(cu, _c_i32p), batch, k,
                          _ptr(masked, _c_u8p), _ptr(tokens, _c_i32p), _ptr(argmax, _c_i32p),
                          _ptr(conf, _c_f64p), _ptr(committed, _c_i32p), _ptr(stats, _c_f64p))
    return conf, committed, stats


# ------------------------------------------------------------------- policy
def policy_profile(T: int, orientation: str) -> np.ndarray:
    """Phase profile (Sec. 4.2): 'early' or 'late'."""
    p = np.empty(T, dtype=np.float64)
    _load().oracle_policy_profile(T, 0 if orientation == "early" else 1, _ptr(p, _c_f64p))
    return p


def policy_normalize(p, target: float) -> np.ndarray:
    p = np.ascontiguousarray(p, dtype=np.float64)
    out = np.empty_like(p)
    _load().oracle_policy_normalize(_ptr(p, _c_f64p), p.size, ctypes.c_double(target), _ptr(out, _c_f64p))
    return out


def policy_envelope(p, B: float, rho: float, demand: float):
    """Eq. 6: (lower, upper) trajectories."""
    p = np.ascontiguousarray(p, dtype=np.float64)
    lo = np.empty_like(p)
    up = np.empty_like(p)
    _load().oracle_policy_envelope(_ptr(p, _c_f64p), p.size, ctypes.c_double(B), ctypes.c_double(rho),
                                   ctypes.c_double(demand), _ptr(lo, _c_f64p), _ptr(up, _c_f64p))
    return lo, up


def policy_risk(t: int, alpha: float, cbar_prev: float, chi_prev: float) -> float:
    """Eq. 7 (t counts from 1)."""
    return float(_load().oracle_policy_risk(t, ctypes.c_double(alpha), ctypes.c_double(cbar_prev),
                                            ctypes.c_double(chi_prev)))


def policy_budget(lower_t: float, upper_t: float, r_t: float) -> float:
    """Eq. 8."""
    return float(_load().oracle_policy_budget(ctypes.c_double(lower_t), ctypes.c_double(upper_t),
                                              ctypes.c_double(r_t)))


def policy_view(b: float) -> int:
    """Eq. 9: 0 coarse, 1 mixed, 2 high."""
    return int(_load().oracle_policy_view(ctypes.c_double(b)))
