"""Thin ctypes binding of libdavet.so (C ABI in include/davet.h).

Argument marshalling only: each function takes torch tensors (or raw
integer device pointers), passes their data pointers and sizes to the C
entry point of the same name, and raises DavetError on a non-OK status.
Every step of the computation runs in the library's CUDA kernels; there is no
Python or CPU fallback, and loading fails loudly when the library is
missing.
"""
from __future__ import annotations

import ctypes
import os
import threading

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libdavet.so")

OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_CUDA, ERR_TIMEOUT, ERR_DEVICE = range(6)
DEV_TIMEOUT, DEV_CAPACITY, DEV_ARG = 0x1, 0x2, 0x4

_lock = threading.Lock()
_lib = None

_vp = ctypes.c_void_p
_i32 = ctypes.c_int32
_i64 = ctypes.c_int64
_int = ctypes.c_int
_f32 = ctypes.c_float
_sz = ctypes.c_size_t


class DavetError(RuntimeError):
    def __init__(self, fn: str, status: int, lib=None):
        msg = lib.davet_status_string(status).decode() if lib is not None else str(status)
        detail = ""
        if status == ERR_CUDA and lib is not None:
            detail = f" (cudaError {lib.davet_last_cuda_error()})"
        super().__init__(f"{fn} failed: {msg}{detail}")
        self.status = status


def _ptr(x):
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr()


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _declare(lib):
    sig = {
        "davet_version": (_int, []),
        "davet_status_string": (ctypes.c_char_p, [_int]),
        "davet_last_cuda_error": (_int, []),
        "davet_device_status": (_int, [ctypes.POINTER(ctypes.c_uint), _int]),
        "davet_sync_status": (_int, [_vp, ctypes.POINTER(ctypes.c_uint)]),
        "davet_selftest_wait_timeout": (_int, [_vp, _vp]),
        "davet_step_attention_workspace": (_int, [_int, _i64, _int, _int, ctypes.POINTER(_sz)]),
        "davet_pyramid_layout": (_int, [_int, _int, _int, ctypes.POINTER(_int), ctypes.POINTER(_i64)]),
        "davet_build_pyramid": (_int, [_vp, _vp, _int, _int, _int, _int, _vp, _vp]),
        "davet_mixed_view_rows": (_int, [_int, _int, _int, _int, ctypes.POINTER(_int)]),
        "davet_gather_view": (_int, [_vp, _vp, _vp, _vp, _vp, _vp, _vp, _int, _int, _int, _int, _int, _int, _vp,
                                     _vp, _i64, _vp]),
        "davet_step_attention": (_int, [_vp, _vp, _int, _i64, _int, _int, _f32, _vp, _vp]),
        "davet_view_rows": (_int, [_int, _int, _int, _int, ctypes.POINTER(_int), ctypes.POINTER(_int)]),
        "davet_view_layout": (_int, [_int, _int, _int, _int, _int, _int, ctypes.POINTER(_i64)]),
        "davet_build_views": (_int, [_vp, _vp, _vp, _int, _int, _int, _int, _int, _int, _int, _vp]),
        "davet_build_views_pruned": (_int, [_vp, _vp, _vp, _vp, _int, _int, _int, _int, _int, _int, _int, _vp]),
        "davet_merge_workspace_bytes": (_int, [_int, _int, _int, _int, ctypes.POINTER(_sz)]),
        "davet_build_views_merged": (_int, [_vp, _vp, _vp, _int, _int, _int, _int, _int, _int, _int, _int, _int,
                                            _vp, _vp, _sz, _vp]),
        "davet_view_attention": (_int, [_vp, _i64, _vp, _vp, _vp, _vp, _vp, _int, _int, _int, _int, _int, _int,
                                        _int, _f32, _vp, _vp, _i64, _vp]),
        "davet_unmask_topk_workspace": (_int, [_i64, _int, _int, ctypes.POINTER(_sz)]),
        "davet_unmask_topk": (_int, [_vp, _int, _vp, _int, _i64, _int, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _sz,
                                     _vp]),
        "davet_policy_envelope": (_int, [_int, _int, ctypes.c_double, ctypes.c_double, _vp, _int, _vp, _vp, _vp]),
        "davet_policy_step": (_int, [_int, _int, _vp, _vp, _vp, _int, ctypes.c_double, ctypes.POINTER(_i32), _vp,
                                     _vp, _vp]),
        "davet_linear": (_int, [_vp, _i64, _int, _vp, _int, _vp, _int, _vp, _vp, _int, _int, _int, _vp, _int, _vp,
                                _sz, _vp, _int, _f32, _vp, _vp, _vp]),
        "davet_row_sumsq": (_int, [_vp, _i64, _int, _vp, _vp, _vp]),
        "davet_linear_workspace_bytes": (_int, [_i64, _int, _int, ctypes.POINTER(_sz)]),
        "davet_rope_table": (_int, [_int, _int, ctypes.c_double, _vp, _vp]),
        "davet_stage_masked_rows": (_int, [_vp, _int, _vp, _i64, _vp, _vp]),
        "davet_rmsnorm": (_int, [_vp, _i64, _int, _vp, _f32, _vp, _vp, _vp, _int, _vp, _vp]),
        "davet_embed_answers": (_int, [_vp, _int, _int, _vp, _int, _vp, _vp, _int, _i64, _vp, _vp]),
        "davet_unmask_topk_noalloc": (_int, [_vp, _int, _vp, _int, _i64, _int, _vp, _vp, _vp, _vp, _vp, _vp,
                                             _vp]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


class Davet:
    """The loaded library; methods mirror the C entry points."""

    def __init__(self, lib):
        self.lib = lib

    def _check(self, fn, status):
        if status != OK:
            raise DavetError(fn, status, self.lib)

    # ------------------------------------------------------------ utilities
    def davet_version(self) -> int:
        return int(self.lib.davet_version())

    def davet_status_string(self, status: int) -> str:
        return self.lib.davet_status_string(status).decode()

    def davet_device_status(self, clear: bool = True) -> tuple[int, int]:
        """(status, flags) of the device error word; synchronizes the device."""
        flags = ctypes.c_uint(0)
        st = self.lib.davet_device_status(ctypes.byref(flags), 1 if clear else 0)
        return int(st), int(flags.value)

    def davet_sync_status(self, stream=None) -> tuple[int, int]:
        """(status, flags) of the device error word after the work on `stream`."""
        flags = ctypes.c_uint(0)
        st = self.lib.davet_sync_status(_stream(stream), ctypes.byref(flags))
        return int(st), int(flags.value)

    def davet_selftest_wait_timeout(self, gave_up, stream=None):
        self._check("davet_selftest_wait_timeout",
                    self.lib.davet_selftest_wait_timeout(_ptr(gave_up), _stream(stream)))

    def davet_step_attention_workspace(self, batch: int, max_total_rows: int, H: int, D: int) -> int:
        n = _sz(0)
        self._check("davet_step_attention_workspace",
                    self.lib.davet_step_attention_workspace(batch, max_total_rows, H, D, ctypes.byref(n)))
        return int(n.value)

    def davet_pyramid_layout(self, grid: int, n_levels: int, n_tiles: int):
        side = (_int * n_levels)()
        off = (_i64 * (n_levels + 1))()
        self._check("davet_pyramid_layout", self.lib.davet_pyramid_layout(grid, n_levels, n_tiles, side, off))
        return list(side), list(off)

    def davet_mixed_view_rows(self, grid: int, n_levels: int, mixed_level: int, mixed_stride: int) -> int:
        n = _int(0)
        self._check("davet_mixed_view_rows",
                    self.lib.davet_mixed_view_rows(grid, n_levels, mixed_level, mixed_stride, ctypes.byref(n)))
        return int(n.value)

    # ---------------------------------------------------------------- path
    def davet_build_pyramid(self, feat, pyr, n_tiles: int, grid: int, n_levels: int, C: int, pyr_f32=None,
                            stream=None):
        self._check("davet_build_pyramid",
                    self.lib.davet_build_pyramid(_ptr(feat), _ptr(pyr), n_tiles, grid, n_levels, C, _ptr(pyr_f32),
                                                 _stream(stream)))

    def davet_gather_view(self, pyr_ptrs, tiles, text, text_off, prompt_len, resp_len, level, batch: int,
                          grid: int, n_levels: int, mixed_level: int, mixed_stride: int, C: int, packed, cu_seqlens,
                          max_total_rows: int, stream=None):
        self._check("davet_gather_view",
                    self.lib.davet_gather_view(_ptr(pyr_ptrs), _ptr(tiles), _ptr(text), _ptr(text_off),
                                               _ptr(prompt_len), _ptr(resp_len), _ptr(level), batch, grid,
                                               n_levels, mixed_level, mixed_stride, C, _ptr(packed),
                                               _ptr(cu_seqlens), max_total_rows, _stream(stream)))

    def davet_step_attention(self, qkv, cu_seqlens, batch: int, max_total_rows: int, H: int, D: int,
                             scale: float, out, stream=None):
        self._check("davet_step_attention",
                    self.lib.davet_step_attention(_ptr(qkv), _ptr(cu_seqlens), batch, max_total_rows, H, D,
                                                  float(scale), _ptr(out), _stream(stream)))

    def davet_view_layout(self, grid: int, n_levels: int, mixed_level: int, mixed_stride: int, n_tiles: int,
                          text_rows: int) -> list[int]:
        nv = _int(0)
        self._check("davet_view_rows", self.lib.davet_view_rows(grid, n_levels, mixed_level, mixed_stride, None,
                                                                 ctypes.byref(nv)))
        off = (_i64 * (nv.value + 1))()
        self._check("davet_view_layout", self.lib.davet_view_layout(grid, n_levels, mixed_level, mixed_stride,
                                                                     n_tiles, text_rows, off))
        return list(off)

    def davet_build_views(self, feat, buf, text, n_tiles: int, grid: int, n_levels: int, mixed_level: int,
                          mixed_stride: int, text_rows: int, C: int, stream=None):
        self._check("davet_build_views",
                    self.lib.davet_build_views(_ptr(feat), _ptr(buf), _ptr(text), n_tiles, grid, n_levels,
                                               mixed_level, mixed_stride, text_rows, C, _stream(stream)))

    def davet_build_views_pruned(self, feat, score, buf, text, n_tiles: int, grid: int, n_levels: int,
                                 mixed_level: int, mixed_stride: int, text_rows: int, C: int, stream=None):
        self._check("davet_build_views_pruned",
                    self.lib.davet_build_views_pruned(_ptr(feat), _ptr(score), _ptr(buf), _ptr(text), n_tiles, grid,
                                                      n_levels, mixed_level, mixed_stride, text_rows, C,
                                                      _stream(stream)))

    def davet_merge_workspace_bytes(self, n_tiles: int, grid: int, n_levels: int, sim_C: int) -> int:
        n = _sz(0)
        self._check("davet_merge_workspace_bytes",
                    self.lib.davet_merge_workspace_bytes(n_tiles, grid, n_levels, sim_C, ctypes.byref(n)))
        return int(n.value)

    def davet_build_views_merged(self, feat, buf, text, n_tiles: int, grid: int, n_levels: int, mixed_level: int,
                                 mixed_stride: int, text_rows: int, C: int, sim_c0: int, sim_C: int, assign=None,
                                 workspace=None, workspace_bytes: int = 0, stream=None):
        if workspace is not None and not isinstance(workspace, int) and workspace_bytes == 0:
            workspace_bytes = workspace.numel() * workspace.element_size()
        self._check("davet_build_views_merged",
                    self.lib.davet_build_views_merged(_ptr(feat), _ptr(buf), _ptr(text), n_tiles, grid, n_levels,
                                                      mixed_level, mixed_stride, text_rows, C, sim_c0, sim_C,
                                                      _ptr(assign), _ptr(workspace), workspace_bytes,
                                                      _stream(stream)))

    def davet_view_attention(self, store, store_rows: int, buf_row0, tiles, prompt_len, resp_len, view, batch: int,
                             grid: int, n_levels: int, mixed_level: int, mixed_stride: int, H: int, D: int,
                             scale: float, out, cu_seqlens, max_total_rows: int, stream=None):
        self._check("davet_view_attention",
                    self.lib.davet_view_attention(_ptr(store), store_rows, _ptr(buf_row0), _ptr(tiles),
                                                  _ptr(prompt_len), _ptr(resp_len), _ptr(view), batch, grid,
                                                  n_levels, mixed_level, mixed_stride, H, D, float(scale), _ptr(out),
                                                  _ptr(cu_seqlens), max_total_rows, _stream(stream)))

    def davet_unmask_topk_workspace(self, total_rows: int, V: int, batch: int) -> int:
        n = _sz(0)
        self._check("davet_unmask_topk_workspace",
                    self.lib.davet_unmask_topk_workspace(total_rows, V, batch, ctypes.byref(n)))
        return int(n.value)

    def davet_unmask_topk(self, logits, V: int, cu_resp, batch: int, total_rows: int, k: int, masked, tokens,
                          argmax=None, conf=None, committed=None, stats=None, workspace=None,
                          workspace_bytes: int = 0, stream=None):
        if workspace is not None and not isinstance(workspace, int) and workspace_bytes == 0:
            workspace_bytes = workspace.numel() * workspace.element_size()
        self._check("davet_unmask_topk",
                    self.lib.davet_unmask_topk(_ptr(logits), V, _ptr(cu_resp), batch, total_rows, k, _ptr(masked),
                                               _ptr(tokens), _ptr(argmax), _ptr(conf), _ptr(committed),
                                               _ptr(stats), _ptr(workspace), workspace_bytes, _stream(stream)))


    EPI_STORE, EPI_RESIDUAL, EPI_SWIGLU, EPI_ROPE = 0, 1, 2, 3

    def davet_linear(self, A, M: int, K: int, W, N: int, out, epilogue: int = 0, residual=None, cu_seqlens=None,
                     batch: int = 0, rope_cols: int = 0, head_dim: int = 128, rope_table=None, max_pos: int = 0,
                     workspace=None, workspace_bytes: int = 0, row_ss=None, row_ss_parts: int = 0,
                     row_ss_eps: float = 0.0, ss_out=None, rows_dev=None, stream=None):
        if workspace is not None and not isinstance(workspace, int) and workspace_bytes == 0:
            workspace_bytes = workspace.numel() * workspace.element_size()
        self._check("davet_linear",
                    self.lib.davet_linear(_ptr(A), M, K, _ptr(W), N, _ptr(out), epilogue, _ptr(residual),
                                          _ptr(cu_seqlens), batch, rope_cols, head_dim, _ptr(rope_table), max_pos,
                                          _ptr(workspace), workspace_bytes, _ptr(row_ss), row_ss_parts,
                                          float(row_ss_eps), _ptr(ss_out), _ptr(rows_dev), _stream(stream)))

    def davet_linear_workspace_bytes(self, M: int, K: int, N: int) -> int:
        n = _sz(0)
        self._check("davet_linear_workspace_bytes", self.lib.davet_linear_workspace_bytes(M, K, N, ctypes.byref(n)))
        return int(n.value)

    def davet_rope_table(self, max_pos: int, head_dim: int, theta: float, table, stream=None):
        self._check("davet_rope_table",
                    self.lib.davet_rope_table(max_pos, head_dim, float(theta), _ptr(table), _stream(stream)))

    def davet_rmsnorm(self, x, M: int, C: int, gamma, eps: float, out, cu_seqlens=None, cu_resp=None, batch: int = 0,
                      rows_dev=None, stream=None):
        self._check("davet_rmsnorm",
                    self.lib.davet_rmsnorm(_ptr(x), M, C, _ptr(gamma), float(eps), _ptr(out), _ptr(cu_seqlens),
                                           _ptr(cu_resp), batch, _ptr(rows_dev), _stream(stream)))

    def davet_row_sumsq(self, x, M: int, C: int, ss_out, rows_dev=None, stream=None):
        self._check("davet_row_sumsq",
                    self.lib.davet_row_sumsq(_ptr(x), M, C, _ptr(ss_out), _ptr(rows_dev), _stream(stream)))

    def davet_embed_answers(self, table, V: int, C: int, tokens, mask_id: int, cu_seqlens, cu_resp, batch: int,
                            total_resp: int, x, stream=None):
        self._check("davet_embed_answers",
                    self.lib.davet_embed_answers(_ptr(table), V, C, _ptr(tokens), mask_id, _ptr(cu_seqlens),
                                                 _ptr(cu_resp), batch, total_resp, _ptr(x), _stream(stream)))

    def davet_policy_envelope(self, T: int, orientation: int, B: float, rho: float, demand, batch: int, lower,
                              upper, stream=None):
        self._check("davet_policy_envelope",
                    self.lib.davet_policy_envelope(T, orientation, float(B), float(rho), _ptr(demand), batch,
                                                   _ptr(lower), _ptr(upper), _stream(stream)))

    def davet_policy_step(self, t: int, T: int, lower, upper, stats_prev, batch: int, alpha: float, view_level,
                          level_out, budget_out=None, stream=None):
        vl = (_i32 * 3)(*[int(x) for x in view_level])
        self._check("davet_policy_step",
                    self.lib.davet_policy_step(t, T, _ptr(lower), _ptr(upper), _ptr(stats_prev), batch, float(alpha),
                                               vl, _ptr(level_out), _ptr(budget_out), _stream(stream)))

    def davet_stage_masked_rows(self, src, V: int, masked, total_rows: int, dst, stream=None):
        self._check("davet_stage_masked_rows",
                    self.lib.davet_stage_masked_rows(_ptr(src), V, _ptr(masked), total_rows, _ptr(dst),
                                                     _stream(stream)))

    def davet_unmask_topk_noalloc(self, logits, V: int, cu_resp, batch: int, total_rows: int, k: int, masked,
                                  tokens, argmax=None, conf=None, committed=None, stats=None, stream=None):
        """davet_unmask_topk for callers that cannot allocate device memory:
        the library's own fixed scratch array replaces the workspace."""
        self._check("davet_unmask_topk_noalloc",
                    self.lib.davet_unmask_topk_noalloc(_ptr(logits), V, _ptr(cu_resp), batch, total_rows, k,
                                                       _ptr(masked), _ptr(tokens), _ptr(argmax), _ptr(conf),
                                                       _ptr(committed), _ptr(stats), _stream(stream)))


_handle = None


def load_cdll(path: str = LIB_PATH):
    """Load the shared library without touching a GPU (symbol checks)."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(path):
                raise RuntimeError(f"libdavet.so not found at {path}: run paper_2608_01821_gb300.build() first "
                                   "(the CUDA library is required; there is no fallback)")
            _lib = _declare(ctypes.CDLL(path))
    return _lib


def load() -> Davet:
    global _handle
    if _handle is None:
        _handle = Davet(load_cdll())
    return _handle
