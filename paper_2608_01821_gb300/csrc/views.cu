// views.cu -- the view-block layout: every evidence view of a request (the
// pooled levels of Sec. 4.3 and, optionally, the mixed view) stored once as a
// contiguous block [view rows || the request's prompt and answer rows], so a
// step's input sequence (Eq. 5) for any view is one run of rows that the
// fused attention (davet_view_attention) reads directly.
//
// davet_build_views builds the pooled levels into their blocks (the pyramid
// kernel, writing level l at its block's start), then one copy kernel fills
// the mixed view's rows (coarse-level rows, then the level-0 lattice) and
// every block's text rows.  The copy kernel gives one warp to each 4 KB
// chunk of a destination row, eight 16-byte loads in flight per lane.
#include <algorithm>

#include "common.cuh"

namespace davet {
namespace views {

constexpr int kMaxViews = 6;  // up to five pooled levels and the mixed view
constexpr int kThreads = 256;
constexpr int kChunk = 256;  // 16-byte slices per warp task (4 KB)

struct Fill {
  uint4* buf;
  const uint4* text;
  int C8;
  int n_tiles, text_rows, n_views;
  long long block0[kMaxViews + 1];
  int rpt[kMaxViews];
  // mixed view (view index mixed_view, or -1)
  int mixed_view, coarse, stride, lat_n, mrows, g0, gc;
  long long n_mixed_rows, n_rows;  // rows the kernel writes: mixed rows, then text rows of every view
};

__device__ __forceinline__ uint4 ld_nc(const uint4* p) {
  uint4 v;
  asm volatile("ld.global.nc.v4.u32 {%0,%1,%2,%3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
  return v;
}

__global__ void __launch_bounds__(kThreads) fill_kernel(Fill f) {
  pdl_launch_dependents();
  pdl_wait();  // the pooled levels come from the pyramid kernel
  const int lane = threadIdx.x & 31;
  const long long gwarp = (static_cast<long long>(blockIdx.x) * kThreads + threadIdx.x) >> 5;
  const long long nwarps = (static_cast<long long>(gridDim.x) * kThreads) >> 5;
  const int nchunk = (f.C8 + kChunk - 1) / kChunk;
  for (long long it = gwarp; it < f.n_rows * nchunk; it += nwarps) {
    const long long k = it / nchunk;
    const int ch = static_cast<int>(it - k * nchunk);
    const uint4* src;
    long long dst_row;
    if (k < f.n_mixed_rows) {
      const long long t = k / f.mrows;
      const int r = static_cast<int>(k - t * f.mrows);
      const int gc2 = f.gc * f.gc;
      long long srow;
      if (r < gc2) {
        srow = f.block0[f.coarse] + t * gc2 + r;
      } else {
        const int i = r - gc2, iy = i / f.lat_n, ix = i - iy * f.lat_n;
        srow = f.block0[0] + t * f.g0 * f.g0 + static_cast<long long>(f.stride / 2 + iy * f.stride) * f.g0 +
               (f.stride / 2 + ix * f.stride);
      }
      src = f.buf + srow * f.C8;
      dst_row = f.block0[f.mixed_view] + k;
    } else {
      const long long q = k - f.n_mixed_rows;
      const int v = static_cast<int>(q / f.text_rows);
      const long long i = q - static_cast<long long>(v) * f.text_rows;
      src = f.text + i * f.C8;
      dst_row = f.block0[v] + static_cast<long long>(f.n_tiles) * f.rpt[v] + i;
    }
    uint4* dst = f.buf + dst_row * f.C8;
    const int c0 = ch * kChunk + lane;
    uint4 v[kChunk / 32];
#pragma unroll
    for (int u = 0; u < kChunk / 32; ++u)
      if (c0 + u * 32 < f.C8) v[u] = ld_nc(src + c0 + u * 32);
#pragma unroll
    for (int u = 0; u < kChunk / 32; ++u)
      if (c0 + u * 32 < f.C8) dst[c0 + u * 32] = v[u];
  }
}


davet_status enqueue_fill(void* buf, const void* text, int n_tiles, int grid, int n_levels, int mixed_level,
                          int mixed_stride, int text_rows, int C, bool compose_mixed, cudaStream_t st) {
  int rpt[kMaxViews];
  int nv = 0;
  const davet_status ls = davet_view_rows(grid, n_levels, mixed_level, mixed_stride, rpt, &nv);
  if (ls != DAVET_OK) return ls;
  int64_t block0[kMaxViews + 1];
  davet_view_layout(grid, n_levels, mixed_level, mixed_stride, n_tiles, text_rows, block0);
  Fill f;
  f.buf = static_cast<uint4*>(buf);
  f.text = static_cast<const uint4*>(text);
  f.C8 = C / 8;
  f.n_tiles = n_tiles;
  f.text_rows = text_rows;
  f.n_views = nv;
  for (int v = 0; v <= kMaxViews; ++v) f.block0[v] = v <= nv ? block0[v] : block0[nv];
  for (int v = 0; v < kMaxViews; ++v) f.rpt[v] = v < nv ? rpt[v] : 0;
  int side[5];
  davet_pyramid_layout(grid, n_levels, 0, side, nullptr);
  f.mixed_view = mixed_stride != 0 ? n_levels : -1;
  f.coarse = mixed_stride != 0 ? mixed_level : 0;
  f.stride = mixed_stride;
  f.lat_n = mixed_stride != 0 ? (grid - mixed_stride / 2 + mixed_stride - 1) / mixed_stride : 1;
  f.mrows = mixed_stride != 0 ? rpt[n_levels] : 1;
  f.g0 = grid;
  f.gc = side[f.coarse];
  f.n_mixed_rows = compose_mixed && mixed_stride != 0 ? static_cast<long long>(n_tiles) * f.mrows : 0;
  f.n_rows = f.n_mixed_rows + static_cast<long long>(text_rows) * nv;
  if (f.n_rows == 0) return DAVET_OK;
  const long long tasks = f.n_rows * ((f.C8 + kChunk - 1) / kChunk);
  const long long blocks = std::min<long long>((tasks + kThreads / 32 - 1) / (kThreads / 32), 152LL * 8);
  const cudaError_t e = launch(fill_kernel, dim3(static_cast<unsigned>(blocks)), dim3(kThreads), 0, st, f);
  if (e != cudaSuccess) return cuda_fail(e);
  return check_launch();
}

}  // namespace views
}  // namespace davet

extern "C" davet_status davet_view_rows(int grid, int n_levels, int mixed_level, int mixed_stride,
                                        int* rows_per_tile, int* n_views) {
  if (grid < 1 || n_levels < 1) return DAVET_ERR_INVALID_ARG;
  if (n_levels > 5 || grid > 65536) return DAVET_ERR_UNSUPPORTED;
  int side[5];
  davet_pyramid_layout(grid, n_levels, 0, side, nullptr);
  int n = n_levels;
  for (int l = 0; l < n_levels; ++l)
    if (rows_per_tile) rows_per_tile[l] = side[l] * side[l];
  if (mixed_stride != 0) {
    int m = 0;
    if (davet_mixed_view_rows(grid, n_levels, mixed_level, mixed_stride, &m) != DAVET_OK) return DAVET_ERR_INVALID_ARG;
    if (rows_per_tile) rows_per_tile[n_levels] = m;
    n = n_levels + 1;
  }
  if (n_views) *n_views = n;
  return DAVET_OK;
}

extern "C" davet_status davet_view_layout(int grid, int n_levels, int mixed_level, int mixed_stride, int n_tiles,
                                          int text_rows, int64_t* block_row0) {
  if (n_tiles < 0 || text_rows < 0) return DAVET_ERR_INVALID_ARG;
  int rpt[davet::views::kMaxViews];
  int nv = 0;
  const davet_status st = davet_view_rows(grid, n_levels, mixed_level, mixed_stride, rpt, &nv);
  if (st != DAVET_OK) return st;
  int64_t off = 0;
  for (int v = 0; v < nv; ++v) {
    if (block_row0) block_row0[v] = off;
    off += static_cast<int64_t>(n_tiles) * rpt[v] + text_rows;
  }
  if (block_row0) block_row0[nv] = off;
  return DAVET_OK;
}

extern "C" davet_status davet_build_views(const void* feat, void* buf, const void* text, int n_tiles, int grid,
                                          int n_levels, int mixed_level, int mixed_stride, int text_rows, int C,
                                          void* stream) {
  using namespace davet;
  using namespace davet::views;
  if (n_tiles < 0 || text_rows < 0 || C < 8 || C % 8 != 0) return DAVET_ERR_INVALID_ARG;
  int rpt[kMaxViews];
  int nv = 0;
  const davet_status ls = davet_view_rows(grid, n_levels, mixed_level, mixed_stride, rpt, &nv);
  if (ls != DAVET_OK) return ls;
  if (n_tiles == 0 && text_rows == 0) return DAVET_OK;  // an empty request has no blocks to fill
  if (!buf || (n_tiles > 0 && !feat) || (text_rows > 0 && !text)) return DAVET_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(feat) | reinterpret_cast<uintptr_t>(buf) | reinterpret_cast<uintptr_t>(text)) &
      15u)
    return DAVET_ERR_INVALID_ARG;
  int64_t block0[kMaxViews + 1];
  davet_view_layout(grid, n_levels, mixed_level, mixed_stride, n_tiles, text_rows, block0);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (n_tiles > 0) {
    // pooled level l at the start of block l
    const davet_status e = pyr::enqueue(feat, buf, n_tiles, grid, n_levels, C, nullptr, block0, block0[nv], st);
    if (e != DAVET_OK) return e;
  }
  return views::enqueue_fill(buf, text, n_tiles, grid, n_levels, mixed_level, mixed_stride, text_rows, C, true, st);
}
