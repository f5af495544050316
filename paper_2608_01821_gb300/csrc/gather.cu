// gather.cu -- packs the input of one denoising step (Eq. 5): for every
// request, the rows of the view its level selects followed by its prompt and
// answer rows, plus the cu_seqlens boundaries, all computed on the device so
// the call needs no host synchronization.
//
// Every block first derives the per-request lengths and their prefix sum in
// shared memory (a block-wide scan; requests are few), then copies rows with
// one warp per row: each lane moves 16-byte slices, eight loads in flight
// before the matching stores, so a warp keeps 4 KB of one row in flight.
//
// The mixed view (Sec. 4.3: pooled tokens plus a fixed subset of unpooled
// ones) is never materialized: level index n_levels selects it, and its
// source rows are computed per packed row -- per tile, the rows of the
// coarse level, then the level-0 tokens of a centred stride-s lattice
// (y, x in {s/2, s/2 + s, ...}), row-major.
#include <algorithm>

#include "common.cuh"

namespace davet {
namespace gat {

constexpr int kThreads = 256;
constexpr int kMaxBatch = 1024;
constexpr int kMaxLevels = 5;
constexpr int kChunk = 256;  // 16-byte slices per warp task (4 KB)

struct Geom {
  int side[kMaxLevels];
  int n_levels;
  int C8;
  // mixed view; stride == 0 when the caller has none
  int mixed_level;   // coarse level of the mixed view
  int mixed_stride;  // lattice stride s over the level-0 grid
  int mixed_n;       // lattice points per side
  int mixed_rows;    // rows per tile: side[mixed_level]^2 + mixed_n^2
};

struct Args {
  const uint4* const* pyr;
  const int32_t* tiles;
  const uint4* text;
  const int64_t* text_off;
  const int32_t* prompt;
  const int32_t* resp;
  const int32_t* level;
  int batch;
  uint4* packed;
  int32_t* cu_out;
  long long cap;
  unsigned* err;
};

__device__ __forceinline__ uint4 ld_nc(const uint4* p) {
  uint4 v;
  asm volatile("ld.global.nc.v4.u32 {%0,%1,%2,%3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
  return v;
}

__global__ void __launch_bounds__(kThreads) gather_kernel(Args a, Geom g) {
  extern __shared__ long long sm[];
  long long* s_cu = sm;                     // [batch+1] packed start of each request
  long long* s_len = sm + a.batch + 1;      // [batch] packed rows of each request
  long long* s_nvis = s_len + a.batch;      // [batch] visual rows
  long long* s_vis0 = s_nvis + a.batch;     // [batch] first pyramid row of the chosen level
                                            // (mixed view: of its coarse level, stored as -1 - row)
  __shared__ long long s_warp[kThreads / 32];
  __shared__ int s_bad;

  const int tid = threadIdx.x;
  if (tid == 0) s_bad = 0;
  pdl_launch_dependents();
  pdl_wait();
  __syncthreads();

  // -------- per-request lengths, then an exclusive scan into s_cu
  const int per = (a.batch + kThreads - 1) / kThreads;
  const int b0 = min(a.batch, tid * per), b1 = min(a.batch, b0 + per);
  long long local = 0;
  for (int b = b0; b < b1; ++b) {
    const int lvl = a.level[b];
    const int nt = a.tiles[b];
    const int p = a.prompt[b], r = a.resp[b];
    bool bad = false;
    long long nvis = 0, vis0 = 0;
    const bool mixed = lvl == g.n_levels && g.mixed_stride > 0;
    if (lvl < 0 || (lvl >= g.n_levels && !mixed) || nt < 0) {
      bad = true;
    } else if (mixed) {
      long long off = 0;
      for (int l = 0; l < g.mixed_level; ++l) off += static_cast<long long>(nt) * g.side[l] * g.side[l];
      vis0 = -1 - off;
      nvis = static_cast<long long>(nt) * g.mixed_rows;
    } else {
      long long off = 0;
      for (int l = 0; l < lvl; ++l) off += static_cast<long long>(nt) * g.side[l] * g.side[l];
      vis0 = off;
      nvis = static_cast<long long>(nt) * g.side[lvl] * g.side[lvl];
    }
    if (p < 0 || r < 0) bad = true;
    if (bad) s_bad = 1;
    s_nvis[b] = nvis;
    s_vis0[b] = vis0;
    const long long len = nvis + max(p, 0) + max(r, 0);
    s_len[b] = len;
    local += len;
  }
  // block-wide exclusive scan of the per-thread sums
  const int lane = tid & 31, warp = tid >> 5;
  long long incl = local;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const long long y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += y;
  }
  if (lane == 31) s_warp[warp] = incl;
  __syncthreads();
  long long run = incl - local;
  for (int w = 0; w < warp; ++w) run += s_warp[w];
  for (int b = b0; b < b1; ++b) {
    s_cu[b] = run;
    run += s_len[b];
  }
  if (b0 < b1 && b1 == a.batch) s_cu[a.batch] = run;
  if (a.batch == 0 && tid == 0) s_cu[0] = 0;
  __syncthreads();

  const long long total = s_cu[a.batch];
  const long long rows = min(total, a.cap);
  if (blockIdx.x == 0) {
    for (int b = tid; b <= a.batch; b += kThreads) a.cu_out[b] = static_cast<int32_t>(min(s_cu[b], a.cap));
    if (tid == 0) {
      if (s_bad) raise_error(a.err, DEV_ERR_ARG);
      if (total > a.cap) raise_error(a.err, DEV_ERR_CAPACITY);
    }
  }

  // -------- row copies: one warp per 4 KB chunk of a row
  const long long gwarp = (static_cast<long long>(blockIdx.x) * kThreads + tid) >> 5;
  const long long nwarps = (static_cast<long long>(gridDim.x) * kThreads) >> 5;
  const int C8 = g.C8;
  const int nchunk = (C8 + kChunk - 1) / kChunk;
  const long long items = rows * nchunk;
  for (long long it = gwarp; it < items; it += nwarps) {
    const long long row = it / nchunk;
    const int ch = static_cast<int>(it - row * nchunk);
    // request owning this row: largest b with s_cu[b] <= row
    int lo = 0, hi = a.batch - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (s_cu[mid] <= row) lo = mid; else hi = mid - 1;
    }
    const int b = lo;
    const long long j = row - s_cu[b];
    const uint4* src;
    if (j < s_nvis[b]) {
      const long long v0 = s_vis0[b];
      long long prow;
      if (v0 >= 0) {
        prow = v0 + j;
      } else {
        // mixed view: tile t, row r of the tile
        const long long t = j / g.mixed_rows;
        const int r = static_cast<int>(j - t * g.mixed_rows);
        const long long gc2 = static_cast<long long>(g.side[g.mixed_level]) * g.side[g.mixed_level];
        if (r < gc2) {
          prow = (-1 - v0) + t * gc2 + r;
        } else {
          const int i = static_cast<int>(r - gc2);
          const int iy = i / g.mixed_n, ix = i - iy * g.mixed_n;
          const int s = g.mixed_stride, G = g.side[0];
          prow = t * G * G + static_cast<long long>(s / 2 + iy * s) * G + (s / 2 + ix * s);
        }
      }
      src = a.pyr[b] + prow * C8;
    } else {
      src = a.text + (a.text_off[b] + (j - s_nvis[b])) * C8;
    }
    uint4* dst = a.packed + row * C8;
    const int c0 = ch * kChunk + lane;
    uint4 v[kChunk / 32];
#pragma unroll
    for (int u = 0; u < kChunk / 32; ++u)
      if (c0 + u * 32 < C8) v[u] = ld_nc(src + c0 + u * 32);
#pragma unroll
    for (int u = 0; u < kChunk / 32; ++u)
      if (c0 + u * 32 < C8) dst[c0 + u * 32] = v[u];
  }
}

}  // namespace gat
}  // namespace davet

extern "C" davet_status davet_gather_view(const void* const* pyr_ptrs_dev, const int32_t* tiles_dev,
                                          const void* text, const int64_t* text_off_dev,
                                          const int32_t* prompt_len_dev, const int32_t* resp_len_dev,
                                          const int32_t* level_dev, int batch, int grid, int n_levels,
                                          int mixed_level, int mixed_stride, int C, void* packed,
                                          int32_t* cu_seqlens_dev, int64_t max_total_rows, void* stream) {
  using namespace davet;
  using namespace davet::gat;
  if (batch < 0 || grid < 1 || n_levels < 1 || C < 8 || C % 8 != 0 || max_total_rows < 0)
    return DAVET_ERR_INVALID_ARG;
  if (n_levels > kMaxLevels || grid > 65536) return DAVET_ERR_UNSUPPORTED;
  int mixed_rows = 0;
  if (mixed_stride != 0 && davet_mixed_view_rows(grid, n_levels, mixed_level, mixed_stride, &mixed_rows) != DAVET_OK)
    return DAVET_ERR_INVALID_ARG;
  if (batch > kMaxBatch) return DAVET_ERR_UNSUPPORTED;
  if (max_total_rows > 0x7fffffffLL) return DAVET_ERR_UNSUPPORTED;
  if (!cu_seqlens_dev) return DAVET_ERR_INVALID_ARG;
  if (batch > 0 && (!pyr_ptrs_dev || !tiles_dev || !text || !text_off_dev || !prompt_len_dev || !resp_len_dev ||
                    !level_dev || !packed))
    return DAVET_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(text) | reinterpret_cast<uintptr_t>(packed)) & 15u) return DAVET_ERR_INVALID_ARG;

  unsigned* err = device_error_word();
  if (!err) return DAVET_ERR_CUDA;
  Geom g;
  int side[kMaxLevels];
  davet_pyramid_layout(grid, n_levels, 0, side, nullptr);
  for (int l = 0; l < kMaxLevels; ++l) g.side[l] = l < n_levels ? side[l] : 1;
  g.n_levels = n_levels;
  g.C8 = C / 8;
  g.mixed_level = mixed_stride ? mixed_level : 0;
  g.mixed_stride = mixed_stride;
  g.mixed_n = mixed_stride ? (grid - mixed_stride / 2 + mixed_stride - 1) / mixed_stride : 0;
  g.mixed_rows = mixed_rows;
  Args a;
  a.pyr = reinterpret_cast<const uint4* const*>(pyr_ptrs_dev);
  a.tiles = tiles_dev;
  a.text = static_cast<const uint4*>(text);
  a.text_off = text_off_dev;
  a.prompt = prompt_len_dev;
  a.resp = resp_len_dev;
  a.level = level_dev;
  a.batch = batch;
  a.packed = static_cast<uint4*>(packed);
  a.cu_out = cu_seqlens_dev;
  a.cap = max_total_rows;
  a.err = err;
  const size_t smem = static_cast<size_t>(4 * batch + 1) * sizeof(long long);
  // one warp per 4 KB chunk: enough blocks to cover the capacity, at most 16 blocks per SM
  const long long nchunk = (g.C8 + kChunk - 1) / kChunk;
  const long long tasks = std::max<long long>(max_total_rows * nchunk, 1);
  const long long blocks = std::min<long long>((tasks + kThreads / 32 - 1) / (kThreads / 32), 152LL * 16);
  const cudaError_t e = launch(gather_kernel, dim3(static_cast<unsigned>(std::max<long long>(blocks, 1))),
                               dim3(kThreads), smem, static_cast<cudaStream_t>(stream), a, g);
  if (e != cudaSuccess) return cuda_fail(e);
  return check_launch();
}

extern "C" davet_status davet_mixed_view_rows(int grid, int n_levels, int mixed_level, int mixed_stride,
                                              int* rows_per_tile) {
  if (grid < 1 || grid > 65536 || n_levels < 1 || n_levels > davet::gat::kMaxLevels) return DAVET_ERR_INVALID_ARG;
  if (mixed_level < 0 || mixed_level >= n_levels || mixed_stride < 1 || mixed_stride > grid)
    return DAVET_ERR_INVALID_ARG;
  int side[davet::gat::kMaxLevels];
  davet_pyramid_layout(grid, n_levels, 0, side, nullptr);
  const long long n = (grid - mixed_stride / 2 + mixed_stride - 1) / mixed_stride;
  const long long rows = static_cast<long long>(side[mixed_level]) * side[mixed_level] + n * n;
  if (rows > 0x7fffffffLL) return DAVET_ERR_UNSUPPORTED;
  if (rows_per_tile) *rows_per_tile = static_cast<int>(rows);
  return DAVET_OK;
}
