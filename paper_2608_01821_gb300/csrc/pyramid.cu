// pyramid.cu -- evidence pyramid of one request (Sec. 4.3: an ordered
// hierarchy of views built once from a single encoding by structured
// pooling; the finest view is the encoding itself).
//
// One thread owns one coarsest-level cell of one tile and one 8-channel
// (16-byte) slice of every level below it: it streams the level-0 tokens of
// that cell's quadtree once with 128-bit loads, reduces 2x2 children level by
// level in fp32 registers, and stores every level it passes through.  Each
// input byte is read once and each output byte written once; consecutive
// threads own consecutive channel slices, so every load and store of a warp
// covers 512 contiguous bytes of one token row.
#include <algorithm>

#include "common.cuh"

namespace davet {
namespace pyr {

constexpr int kMaxLevels = 5;

struct Geom {
  int side[kMaxLevels];
  long long off[kMaxLevels + 1];  // first row of each level (level-major)
  int n_tiles;
  int C8;      // 16-byte slices per row
  bool copy0;  // level 0 must be copied into the pyramid buffer
};

struct Ctx {
  const uint4* __restrict__ feat;
  uint4* __restrict__ pyr;
  float4* __restrict__ pyr32;
  int tile;
  int cv;
};

__device__ __forceinline__ uint4 ld_stream(const uint4* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ void store_row(const Ctx& c, const Geom& g, long long row, const float (&v)[8]) {
  uint4 u;
  u.x = pack_bf16x2(v[0], v[1]);
  u.y = pack_bf16x2(v[2], v[3]);
  u.z = pack_bf16x2(v[4], v[5]);
  u.w = pack_bf16x2(v[6], v[7]);
  c.pyr[row * g.C8 + c.cv] = u;
  if (c.pyr32) {
    float4* d = c.pyr32 + (row * g.C8 + c.cv) * 2;
    d[0] = make_float4(v[0], v[1], v[2], v[3]);
    d[1] = make_float4(v[4], v[5], v[6], v[7]);
  }
}

// Mean of cell (y, x) of level L (fp32), or false if the cell lies outside
// the level-L grid.  Level L >= 1 averages its in-range 2x2 children of
// level L-1 (1, 2 or 4 of them, so the scale is an exact power of two).
template <int L, int TOP>
__device__ __forceinline__ bool cell(const Ctx& c, const Geom& g, int y, int x, float (&v)[8]) {
  const int gs = g.side[L];
  if (y >= gs || x >= gs) return false;
  const long long row = g.off[L] + (static_cast<long long>(c.tile) * gs + y) * gs + x;
  if constexpr (L == 0) {
    const long long src = (static_cast<long long>(c.tile) * gs + y) * gs + x;
    const uint4 u = ld_stream(c.feat + src * g.C8 + c.cv);
    v[0] = bf16lo(u.x); v[1] = bf16hi(u.x);
    v[2] = bf16lo(u.y); v[3] = bf16hi(u.y);
    v[4] = bf16lo(u.z); v[5] = bf16hi(u.z);
    v[6] = bf16lo(u.w); v[7] = bf16hi(u.w);
    if (g.copy0) c.pyr[row * g.C8 + c.cv] = u;
    if (c.pyr32) {
      float4* d = c.pyr32 + (row * g.C8 + c.cv) * 2;
      d[0] = make_float4(v[0], v[1], v[2], v[3]);
      d[1] = make_float4(v[4], v[5], v[6], v[7]);
    }
    return true;
  } else {
    float acc[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) acc[k] = 0.f;
    int n = 0;
    if constexpr (L == TOP) {
      // the top level walks its four subtrees one after another so that
      // each subtree's loads are issued together without exhausting registers
#pragma unroll 1
      for (int q = 0; q < 4; ++q) {
        float ch[8];
        if (cell<L - 1, TOP>(c, g, 2 * y + (q >> 1), 2 * x + (q & 1), ch)) {
#pragma unroll
          for (int k = 0; k < 8; ++k) acc[k] += ch[k];
          ++n;
        }
      }
    } else {
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        float ch[8];
        if (cell<L - 1, TOP>(c, g, 2 * y + (q >> 1), 2 * x + (q & 1), ch)) {
#pragma unroll
          for (int k = 0; k < 8; ++k) acc[k] += ch[k];
          ++n;
        }
      }
    }
    const float inv = n == 4 ? 0.25f : (n == 2 ? 0.5f : 1.0f);
#pragma unroll
    for (int k = 0; k < 8; ++k) v[k] = acc[k] * inv;
    store_row(c, g, row, v);
    return true;
  }
}

// Level-DEPTH cell (y, x) from its (2^DEPTH)^2 level-0 leaves: every leaf
// load is issued before any store, so the loads are in flight together even
// when the pyramid is built in place (the output may alias the input, which
// would otherwise keep the compiler from moving later loads above earlier
// stores).  Then the levels 1..DEPTH are reduced in registers and stored.
template <int DEPTH>
__device__ __forceinline__ bool subtree(const Ctx& c, const Geom& g, int y, int x, float (&out)[8]) {
  constexpr int S = 1 << DEPTH;
  const int gd = g.side[DEPTH];
  if (y >= gd || x >= gd) return false;
  const int g0 = g.side[0];
  uint4 leaf[S * S];
#pragma unroll
  for (int i = 0; i < S; ++i)
#pragma unroll
    for (int j = 0; j < S; ++j) {
      const int ly = y * S + i, lx = x * S + j;
      if (ly < g0 && lx < g0) {
        const long long src = (static_cast<long long>(c.tile) * g0 + ly) * g0 + lx;
        leaf[i * S + j] = ld_stream(c.feat + src * g.C8 + c.cv);
      } else {
        leaf[i * S + j] = make_uint4(0, 0, 0, 0);
      }
    }
  // level 0 side effects: the copy into the pyramid and the fp32 form
  if (g.copy0 || c.pyr32) {
#pragma unroll
    for (int i = 0; i < S; ++i)
#pragma unroll
      for (int j = 0; j < S; ++j) {
        const int ly = y * S + i, lx = x * S + j;
        if (ly < g0 && lx < g0) {
          const long long row = g.off[0] + (static_cast<long long>(c.tile) * g0 + ly) * g0 + lx;
          const uint4 u = leaf[i * S + j];
          if (g.copy0) c.pyr[row * g.C8 + c.cv] = u;
          if (c.pyr32) {
            float4* d = c.pyr32 + (row * g.C8 + c.cv) * 2;
            d[0] = make_float4(bf16lo(u.x), bf16hi(u.x), bf16lo(u.y), bf16hi(u.y));
            d[1] = make_float4(bf16lo(u.z), bf16hi(u.z), bf16lo(u.w), bf16hi(u.w));
          }
        }
      }
  }
  // level 1 cells of the subtree
  float l1[(S / 2) * (S / 2)][8];
  const int g1 = g.side[1];
#pragma unroll
  for (int a = 0; a < S / 2; ++a)
#pragma unroll
    for (int b = 0; b < S / 2; ++b) {
      float acc[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) acc[k] = 0.f;
      int n = 0;
#pragma unroll
      for (int qq = 0; qq < 4; ++qq) {
        const int i = 2 * a + (qq >> 1), j = 2 * b + (qq & 1);
        if (y * S + i < g0 && x * S + j < g0) {
          // each bf16 widened exactly and added in fp32: one mixed-precision
          // add per value instead of a widening plus an add
          const uint4 u = leaf[i * S + j];
          add_bf16x2_f32(acc[0], acc[1], u.x);
          add_bf16x2_f32(acc[2], acc[3], u.y);
          add_bf16x2_f32(acc[4], acc[5], u.z);
          add_bf16x2_f32(acc[6], acc[7], u.w);
          ++n;
        }
      }
      const float inv = n == 4 ? 0.25f : (n == 2 ? 0.5f : 1.0f);
#pragma unroll
      for (int k = 0; k < 8; ++k) l1[a * (S / 2) + b][k] = acc[k] * inv;
      const int y1 = y * (S / 2) + a, x1 = x * (S / 2) + b;
      if (n > 0 && y1 < g1 && x1 < g1)
        store_row(c, g, g.off[1] + (static_cast<long long>(c.tile) * g1 + y1) * g1 + x1, l1[a * (S / 2) + b]);
    }
  if constexpr (DEPTH == 1) {
#pragma unroll
    for (int k = 0; k < 8; ++k) out[k] = l1[0][k];
    return true;
  } else {
    static_assert(DEPTH == 2, "subtree depth 1 or 2");
    // the level-2 cell from its in-range level-1 children
    float acc[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) acc[k] = 0.f;
    int n = 0;
#pragma unroll
    for (int qq = 0; qq < 4; ++qq) {
      const int y1 = 2 * y + (qq >> 1), x1 = 2 * x + (qq & 1);
      if (y1 < g1 && x1 < g1) {
#pragma unroll
        for (int k = 0; k < 8; ++k) acc[k] += l1[qq][k];
        ++n;
      }
    }
    const float inv = n == 4 ? 0.25f : (n == 2 ? 0.5f : 1.0f);
#pragma unroll
    for (int k = 0; k < 8; ++k) out[k] = acc[k] * inv;
    store_row(c, g, g.off[2] + (static_cast<long long>(c.tile) * gd + y) * gd + x, out);
    return true;
  }
}

template <int NL>
__global__ void pyramid_kernel(const uint4* __restrict__ feat, uint4* __restrict__ pyr, float4* __restrict__ pyr32,
                               Geom g) {
  constexpr int TOP = NL - 1;
  pdl_launch_dependents();
  pdl_wait();
  const int gt = g.side[TOP];
  const long long cells = static_cast<long long>(gt) * gt;
  if constexpr (NL == 1) {
    // a single level: only the copy of level 0 (and its fp32 form) remains
    const long long total = static_cast<long long>(g.n_tiles) * cells * g.C8;
    for (long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; i < total;
         i += static_cast<long long>(gridDim.x) * blockDim.x) {
      Ctx c;
      c.feat = feat;
      c.pyr = pyr;
      c.pyr32 = pyr32;
      c.cv = static_cast<int>(i % g.C8);
      const long long rest = i / g.C8;
      c.tile = static_cast<int>(rest / cells);
      const int cellid = static_cast<int>(rest % cells);
      float v[8];
      cell<0, 0>(c, g, cellid / gt, cellid % gt, v);
    }
  } else {
    // A block of 8 warps covers one top-level cell and 64 consecutive 16-byte
    // channel slices: warp w reduces child subtree q = w % 4 for slices
    // 32 * (w / 4) + lane, so every warp load reads 512 contiguous bytes of
    // one token row; the four children are then combined through shared
    // memory.
    __shared__ float s_v[4][64][9];  // [child][slice][8 values + in-range flag]
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int q = warp & 3;
    const int cv_local = (warp >> 2) * 32 + lane;
    const int chunks = (g.C8 + 63) / 64;
    const long long units = static_cast<long long>(g.n_tiles) * cells * chunks;
    for (long long u = blockIdx.x; u < units; u += gridDim.x) {
      // 32-bit divisions while the unit count fits (a 64-bit division is a
      // long subroutine)
      int chunk, cellid, tile;
      if (units <= 0xffffffffLL) {
        const unsigned u32 = static_cast<unsigned>(u);
        const unsigned rest32 = u32 / static_cast<unsigned>(chunks);
        chunk = static_cast<int>(u32 - rest32 * static_cast<unsigned>(chunks));
        cellid = static_cast<int>(rest32 % static_cast<unsigned>(cells));
        tile = static_cast<int>(rest32 / static_cast<unsigned>(cells));
      } else {
        chunk = static_cast<int>(u % chunks);
        const long long rest = u / chunks;
        cellid = static_cast<int>(rest % cells);
        tile = static_cast<int>(rest / cells);
      }
      Ctx c;
      c.feat = feat;
      c.pyr = pyr;
      c.pyr32 = pyr32;
      c.tile = tile;
      c.cv = chunk * 64 + cv_local;
      const int Y = cellid / gt, X = cellid % gt;
      float v[8];
      bool have = false;
      // each warp's child subtree issues all its leaf loads together (five
      // levels: the 64-leaf subtree walks its four quarters one at a time)
      if (c.cv < g.C8) {
        if constexpr (NL == 3 || NL == 4)
          have = subtree<TOP - 1>(c, g, 2 * Y + (q >> 1), 2 * X + (q & 1), v);
        else
          have = cell<TOP - 1, NL >= 5 ? TOP - 1 : NL>(c, g, 2 * Y + (q >> 1), 2 * X + (q & 1), v);
      }
#pragma unroll
      for (int k = 0; k < 8; ++k) s_v[q][cv_local][k] = have ? v[k] : 0.f;
      s_v[q][cv_local][8] = have ? 1.f : 0.f;
      __syncthreads();
      if (threadIdx.x < 64 && chunk * 64 + threadIdx.x < g.C8) {
        const int sl = threadIdx.x;
        float n = 0.f, acc[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) acc[k] = 0.f;
#pragma unroll
        for (int qq = 0; qq < 4; ++qq) {
          n += s_v[qq][sl][8];
#pragma unroll
          for (int k = 0; k < 8; ++k) acc[k] += s_v[qq][sl][k];
        }
        const float inv = n == 4.f ? 0.25f : (n == 2.f ? 0.5f : 1.0f);
#pragma unroll
        for (int k = 0; k < 8; ++k) acc[k] *= inv;
        Ctx ct = c;
        ct.cv = chunk * 64 + sl;
        const long long row = g.off[TOP] + (static_cast<long long>(c.tile) * gt + Y) * gt + X;
        store_row(ct, g, row, acc);
      }
      __syncthreads();
    }
  }
}

}  // namespace pyr
}  // namespace davet

extern "C" davet_status davet_pyramid_layout(int grid, int n_levels, int n_tiles, int* level_side,
                                             int64_t* level_row_offset) {
  if (grid < 1 || n_levels < 1 || n_levels > davet::pyr::kMaxLevels || n_tiles < 0) return DAVET_ERR_INVALID_ARG;
  if (grid > 65536) return DAVET_ERR_UNSUPPORTED;
  int g = grid;
  int64_t off = 0;
  for (int l = 0; l < n_levels; ++l) {
    if (level_side) level_side[l] = g;
    if (level_row_offset) level_row_offset[l] = off;
    off += static_cast<int64_t>(n_tiles) * g * g;
    g = (g + 1) / 2;
  }
  if (level_row_offset) level_row_offset[n_levels] = off;
  return DAVET_OK;
}

namespace davet {
namespace pyr {

// Enqueues the pyramid build with level l's rows starting at row off[l] of
// pyr (level 0 at off[0]; rows of a level are tile-major, row-major within a
// tile) and `extent` rows in all; arguments already checked by the caller.
davet_status enqueue(const void* feat, void* pyr, int n_tiles, int grid, int n_levels, int C, float* pyr_f32,
                     const int64_t* off, int64_t extent, cudaStream_t st) {
  Geom g;
  int side[kMaxLevels] = {};
  davet_pyramid_layout(grid, n_levels, n_tiles, side, nullptr);
  for (int l = 0; l < kMaxLevels; ++l) g.side[l] = l < n_levels ? side[l] : 1;
  for (int l = 0; l <= kMaxLevels; ++l) g.off[l] = l < n_levels ? off[l] : extent;
  g.n_tiles = n_tiles;
  g.C8 = C / 8;
  g.copy0 = feat != pyr;
  if (g.copy0) {
    // feat and the pyramid must not overlap when level 0 is copied
    const uintptr_t f0 = reinterpret_cast<uintptr_t>(feat), p0 = reinterpret_cast<uintptr_t>(pyr);
    const uintptr_t f1 = f0 + static_cast<uintptr_t>(n_tiles) * grid * grid * C * 2;
    const uintptr_t p1 = p0 + static_cast<uintptr_t>(extent) * C * 2;
    if (f0 < p1 && p0 < f1) return DAVET_ERR_INVALID_ARG;
  }

  const int gt = side[n_levels - 1];
  int threads;
  long long blocks;
  if (n_levels > 1) {
    // one block (8 warps) per (tile, top-level cell, 64-slice chunk)
    threads = 256;
    blocks = std::min<long long>(static_cast<long long>(n_tiles) * gt * gt * ((g.C8 + 63) / 64), 152LL * 64);
  } else {
    const long long total = static_cast<long long>(n_tiles) * gt * gt * g.C8;
    threads = 256;
    blocks = std::min<long long>((total + threads - 1) / threads, 152LL * 64);
  }
  const uint4* f = static_cast<const uint4*>(feat);
  uint4* p = static_cast<uint4*>(pyr);
  float4* p32 = reinterpret_cast<float4*>(pyr_f32);
  cudaError_t e;
  switch (n_levels) {
    case 1: e = launch(pyramid_kernel<1>, dim3(blocks), dim3(threads), 0, st, f, p, p32, g); break;
    case 2: e = launch(pyramid_kernel<2>, dim3(blocks), dim3(threads), 0, st, f, p, p32, g); break;
    case 3: e = launch(pyramid_kernel<3>, dim3(blocks), dim3(threads), 0, st, f, p, p32, g); break;
    case 4: e = launch(pyramid_kernel<4>, dim3(blocks), dim3(threads), 0, st, f, p, p32, g); break;
    default: e = launch(pyramid_kernel<5>, dim3(blocks), dim3(threads), 0, st, f, p, p32, g); break;
  }
  if (e != cudaSuccess) return cuda_fail(e);
  return check_launch();
}

}  // namespace pyr
}  // namespace davet

extern "C" davet_status davet_build_pyramid(const void* feat, void* pyr, int n_tiles, int grid, int n_levels, int C,
                                            float* pyr_f32, void* stream) {
  using namespace davet;
  using namespace davet::pyr;
  if (n_tiles < 0 || grid < 1 || n_levels < 1 || C < 8) return DAVET_ERR_INVALID_ARG;
  if (n_levels > kMaxLevels || grid > 65536) return DAVET_ERR_UNSUPPORTED;
  if (C % 8 != 0) return DAVET_ERR_INVALID_ARG;
  if (n_tiles == 0) return DAVET_OK;
  if (!feat || !pyr) return DAVET_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(feat) | reinterpret_cast<uintptr_t>(pyr) |
       reinterpret_cast<uintptr_t>(pyr_f32)) & 15u)
    return DAVET_ERR_INVALID_ARG;
  int64_t off[kMaxLevels + 1];
  davet_pyramid_layout(grid, n_levels, n_tiles, nullptr, off);
  return enqueue(feat, pyr, n_tiles, grid, n_levels, C, pyr_f32, off, off[n_levels], static_cast<cudaStream_t>(stream));
}
