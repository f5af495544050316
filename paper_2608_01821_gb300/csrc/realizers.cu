// realizers.cu -- the pruning and merging evidence realizers (Sec. 4.3
// "compatible evidence realizers": pruning varies the retention ratio,
// merging the aggregation strength; Sec. 5.3 / Table 2).  Both build the same
// view blocks as davet_build_views -- same views, same row counts per tile,
// same [view || text] layout -- so davet_view_attention consumes them
// unchanged; only the rows of the views differ.
//
// Pruning: one kernel.  Every CTA of a tile sorts the tile's scores in
// shared memory (bitonic, 64-bit keys: descending score, then ascending
// index), turns ranks into the kept-token list of every view (a block scan
// per view), then copies its share of the tile's view rows with one warp per
// 4 KB row chunk.  The sort is repeated by each CTA of a tile; it is a few
// microseconds, and it saves a workspace and a launch.
//
// Merging: bipartite matching rounds per level, each round three launches
// over all tiles of the request:
//   sum_kernel    feature sums S of the current tokens (members in ascending
//                 level-0 index, binary32) over the similarity channels;
//   sim_kernel    the A x B cosine block (A = even, B = odd positions): a
//                 register-blocked fp32 product over channel stages streamed
//                 into shared memory by a cp.async ring, every output
//                 accumulating its channels in ascending order with fused
//                 multiply-adds; the squared-norm chains of the staged rows
//                 run alongside (then a correctly rounded square root and
//                 division), and each A row's best match per B block is
//                 written out.  The block shape is chosen per round (64, 32
//                 or 16 rows a side) so that small late rounds still spread
//                 over the SMs;
//   select_kernel one CTA per tile: best match over the B blocks, the r
//                 best-matched members of A, the new token of every level-0
//                 token, and the member lists of the new tokens (stable).
// When a level is complete, sum_kernel writes its rows as member means (bf16).
// The merge decisions are taken in binary32 with this fixed operation order
// on purpose: the products are CUDA-core fused multiply-adds rather than
// tensor-core MMAs, whose internal accumulation order is not specified, so
// every decision is reproducible bit for bit.  The realizer runs once per
// request, before denoising.
#include <algorithm>
#include <vector>

#include "common.cuh"

namespace davet {
namespace realize {

constexpr int kMaxViews = 6;
constexpr int kThreads = 256;
constexpr int kChunk = 256;  // 16-byte slices per copy task (4 KB)

__device__ __forceinline__ uint4 ld_nc(const uint4* p) {
  uint4 v;
  asm volatile("ld.global.nc.v4.u32 {%0,%1,%2,%3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
  return v;
}

// Exclusive scan of per-thread counts over the block; returns the block total.
template <int NT>
__device__ __forceinline__ int block_exclusive_scan(int v, int* warp_tot, int& excl) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_tot[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int t = lane < NT / 32 ? warp_tot[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, t, o);
      if (lane >= o) t += y;
    }
    if (lane < NT / 32) warp_tot[lane] = t;  // inclusive
  }
  __syncthreads();
  excl = x - v + (warp > 0 ? warp_tot[warp - 1] : 0);
  const int total = warp_tot[NT / 32 - 1];
  __syncthreads();
  return total;
}

// ------------------------------------------------------------------ pruning
struct Prune {
  const uint4* feat;
  const float* score;
  uint4* buf;
  int C8, n_tok, sort_n, n_tiles, n_views, first_view;
  long long block0[kMaxViews];
  int rpt[kMaxViews];
  int rpt_off[kMaxViews + 1];  // prefix sums of rpt over the views
};

// Sort key: descending score (a NaN after every number, -0 == +0), then
// ascending token index.
__device__ __forceinline__ unsigned long long prune_key(float s, int i) {
  unsigned ord;
  if (s != s) {
    ord = 0u;
  } else {
    if (s == 0.0f) s = 0.0f;
    const unsigned u = __float_as_uint(s);
    ord = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  }
  return (static_cast<unsigned long long>(~ord) << 32) | static_cast<unsigned>(i);
}

__global__ void __launch_bounds__(kThreads) prune_kernel(Prune p) {
  extern __shared__ __align__(16) unsigned char smem[];
  unsigned long long* keys = reinterpret_cast<unsigned long long*>(smem);  // [sort_n]
  int* rank = reinterpret_cast<int*>(keys + p.sort_n);                     // [n_tok]
  int* map = rank + p.n_tok;                                               // [rpt_off[n_views]]
  __shared__ int warp_tot[kThreads / 32];
  pdl_launch_dependents();
  pdl_wait();
  const int tile = blockIdx.y;
  const float* sc = p.score + static_cast<long long>(tile) * p.n_tok;
  for (int i = threadIdx.x; i < p.sort_n; i += kThreads)
    keys[i] = i < p.n_tok ? prune_key(sc[i], i) : ~0ull;
  __syncthreads();
  for (int k = 2; k <= p.sort_n; k <<= 1) {
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int i = threadIdx.x; i < p.sort_n; i += kThreads) {
        const int ixj = i ^ j;
        if (ixj > i) {
          const unsigned long long a = keys[i], b = keys[ixj];
          if ((a > b) == ((i & k) == 0)) {
            keys[i] = b;
            keys[ixj] = a;
          }
        }
      }
      __syncthreads();
    }
  }
  for (int q = threadIdx.x; q < p.n_tok; q += kThreads) rank[static_cast<unsigned>(keys[q])] = q;
  __syncthreads();
  // kept tokens of every view in raster order: thread t scans a contiguous run
  const int per = (p.n_tok + kThreads - 1) / kThreads;
  const int i0 = min(p.n_tok, static_cast<int>(threadIdx.x) * per), i1 = min(p.n_tok, i0 + per);
  for (int v = p.first_view; v < p.n_views; ++v) {
    const int m = p.rpt[v];
    int c = 0;
    for (int i = i0; i < i1; ++i) c += rank[i] < m;
    int pos;
    block_exclusive_scan<kThreads>(c, warp_tot, pos);
    int* mv = map + p.rpt_off[v];
    for (int i = i0; i < i1; ++i)
      if (rank[i] < m) mv[pos++] = i;
  }
  __syncthreads();
  // copy: one warp per (view row, 4 KB chunk)
  const int lane = threadIdx.x & 31;
  const int nchunk = (p.C8 + kChunk - 1) / kChunk;
  const long long r0 = p.rpt_off[p.first_view];
  const long long tasks = (p.rpt_off[p.n_views] - r0) * nchunk;
  const long long nw = static_cast<long long>(gridDim.x) * (kThreads / 32);
  for (long long it = static_cast<long long>(blockIdx.x) * (kThreads / 32) + (threadIdx.x >> 5); it < tasks;
       it += nw) {
    const long long k = r0 + it / nchunk;
    const int ch = static_cast<int>(it % nchunk);
    int v = p.first_view;
    while (k >= p.rpt_off[v + 1]) ++v;
    const int pos = static_cast<int>(k - p.rpt_off[v]);
    const uint4* src = p.feat + (static_cast<long long>(tile) * p.n_tok + map[k]) * p.C8;
    uint4* dst = p.buf + (p.block0[v] + static_cast<long long>(tile) * p.rpt[v] + pos) * p.C8;
    const int c0 = ch * kChunk + lane;
    uint4 x[kChunk / 32];
#pragma unroll
    for (int u = 0; u < kChunk / 32; ++u)
      if (c0 + u * 32 < p.C8) x[u] = ld_nc(src + c0 + u * 32);
#pragma unroll
    for (int u = 0; u < kChunk / 32; ++u)
      if (c0 + u * 32 < p.C8) dst[c0 + u * 32] = x[u];
  }
}

// ------------------------------------------------------------------ merging
// Workspace of one request (every region 256-byte aligned):
//   tok     int32 [n_tiles][n0]      current token of each level-0 token
//   start   int32 [n_tiles][n0 + 1]  member-list offsets of the current tokens
//   members int32 [n_tiles][n0]      level-0 indices, ascending per token
//   best    Best  [n_tiles][bblk][nA] best match of each member of A per B block
//   S       f32   [n_tiles][n0][Cs]  similarity-channel sums of the current tokens
struct Best {
  float s;
  int b;
};

// Similarity block shapes: TM x TM members of A by B per CTA, RM x RM
// products per thread, KC channels per pipeline stage, STAGES stages.
template <int TM_, int RM_, int KC_, int STAGES_>
struct SimShape {
  static constexpr int TM = TM_, RM = RM_, KC = KC_, STAGES = STAGES_;
  static constexpr int NT = (TM / RM) * (TM / RM);
  static constexpr int PITCH = KC + 4;  // floats per staged row: 16-byte aligned, 4-bank offset per row
  static constexpr int CHUNKS = TM * KC / 4 / NT;  // 16-byte copies per operand per thread per stage
  static constexpr size_t SMEM = static_cast<size_t>(STAGES) * 2 * TM * PITCH * 4 + 2 * TM * 4;
  static_assert(NT >= 2 * TM, "the norm chains need one thread per staged row");
  static_assert(TM * KC / 4 % NT == 0, "stage copies must divide evenly");
};
using SimLarge = SimShape<64, 4, 32, 3>;
using SimMid = SimShape<32, 4, 32, 4>;
using SimSmall = SimShape<16, 2, 32, 6>;

struct Plan {
  int n0, n_levels;
  int side[5];
  std::vector<int> n, r, level;  // per round: tokens before, merged, level it builds
  int nA_max, bblk_max;
  size_t off_tok, off_start, off_members, off_best, off_S, bytes;
};

inline size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

inline Plan make_plan(int n_tiles, int grid, int n_levels, int Cs) {
  Plan P;
  P.n0 = grid * grid;
  P.n_levels = n_levels;
  davet_pyramid_layout(grid, n_levels, 0, P.side, nullptr);
  int n = P.n0;
  P.nA_max = 1;
  P.bblk_max = 1;
  for (int l = 1; l < n_levels; ++l) {
    const int target = P.side[l] * P.side[l];
    while (n > target) {
      const int nA = (n + 1) / 2, nB = n / 2;
      const int r = std::min(n - target, nA);
      P.n.push_back(n);
      P.r.push_back(r);
      P.level.push_back(l);
      P.nA_max = std::max(P.nA_max, nA);
      P.bblk_max = std::max(P.bblk_max, (nB + SimSmall::TM - 1) / SimSmall::TM);
      n -= r;
    }
  }
  const size_t T = static_cast<size_t>(n_tiles);
  size_t o = 0;
  P.off_tok = o;
  o = align256(o + T * P.n0 * 4);
  P.off_start = o;
  o = align256(o + T * (P.n0 + 1) * 4);
  P.off_members = o;
  o = align256(o + T * P.n0 * 4);
  P.off_best = o;
  o = align256(o + T * P.bblk_max * P.nA_max * sizeof(Best));
  P.off_S = o;
  o = align256(o + (P.n.empty() ? 0 : T * static_cast<size_t>(P.n0) * Cs * 4));
  P.bytes = o;
  return P;
}

struct MergeArgs {
  const uint4* feat;  // bf16 [n_tiles][n0][C]
  int C8, n0, n_tiles;
  int c0_8;  // first similarity channel / 8
  int Cs;    // similarity channels
  int32_t* tok;
  int32_t* start;
  int32_t* members;
  Best* best;
  float* S;
  int n, nA, nB, bblk, r;
};

__global__ void __launch_bounds__(kThreads) init_kernel(MergeArgs a, int32_t* assign0) {
  pdl_launch_dependents();
  pdl_wait();
  const long long total = static_cast<long long>(a.n_tiles) * (a.n0 + 1);
  for (long long q = static_cast<long long>(blockIdx.x) * kThreads + threadIdx.x; q < total;
       q += static_cast<long long>(gridDim.x) * kThreads) {
    const int t = static_cast<int>(q / (a.n0 + 1)), i = static_cast<int>(q % (a.n0 + 1));
    a.start[q] = i;
    if (i < a.n0) {
      const long long k = static_cast<long long>(t) * a.n0 + i;
      a.tok[k] = i;
      a.members[k] = i;
      if (assign0) assign0[k] = i;
    }
  }
}

__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait_group() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// One stage of the A and B rows of this CTA: TM rows x KC channels each,
// 16-byte cp.async copies (rows past the set end are zero-filled).
template <class SH>
__device__ __forceinline__ void sim_stage(const MergeArgs& a, const float* St, int a0, int b0, int k0,
                                          float* sa, float* sb) {
  constexpr int CPR = SH::KC / 4;  // 16-byte chunks per staged row
#pragma unroll
  for (int u = 0; u < SH::CHUNKS; ++u) {
    const int q = threadIdx.x + u * SH::NT;
    const int row = q / CPR, c = q % CPR;
    const bool va = a0 + row < a.nA, vb = b0 + row < a.nB;
    const float* pa = St + static_cast<long long>(va ? 2 * (a0 + row) : 0) * a.Cs + k0 + c * 4;
    const float* pb = St + static_cast<long long>(vb ? 2 * (b0 + row) + 1 : 0) * a.Cs + k0 + c * 4;
    cp_async16(smem_u32(sa + row * SH::PITCH + c * 4), pa, va ? 16 : 0);
    cp_async16(smem_u32(sb + row * SH::PITCH + c * 4), pb, vb ? 16 : 0);
  }
}

// A x B cosine block (A = even, B = odd positions) of one tile: every
// product accumulates its channels in ascending order by fused multiply-adds;
// threads 0..TM-1 (2*TM-1) also run the squared-norm chains of the staged A
// (B) rows over the same stages.  Then each A row's best match in the block.
// Thread (ty, tx) owns rows ty + i*(TM/RM) of A and tx + j*(TM/RM) of B.
template <class SH>
__global__ void __launch_bounds__(SH::NT) sim_kernel(MergeArgs a) {
  extern __shared__ __align__(16) float sm[];
  float* sA = sm;                                        // [STAGES][TM][PITCH]
  float* sB = sA + SH::STAGES * SH::TM * SH::PITCH;      // [STAGES][TM][PITCH]
  float* invA = sB + SH::STAGES * SH::TM * SH::PITCH;    // [TM]
  float* invB = invA + SH::TM;                           // [TM]
  constexpr int TD = SH::TM / SH::RM;
  pdl_launch_dependents();
  pdl_wait();
  const int t = blockIdx.z;
  const int a0 = blockIdx.x * SH::TM, b0 = blockIdx.y * SH::TM;
  const int tx = threadIdx.x % TD, ty = threadIdx.x / TD;
  const float* St = a.S + static_cast<long long>(t) * a.n0 * a.Cs;
  const int nk = a.Cs / SH::KC;
#pragma unroll
  for (int s = 0; s < SH::STAGES - 1; ++s) {
    if (s < nk) sim_stage<SH>(a, St, a0, b0, s * SH::KC, sA + s * SH::TM * SH::PITCH, sB + s * SH::TM * SH::PITCH);
    cp_async_commit();
  }
  float acc[SH::RM][SH::RM];
#pragma unroll
  for (int i = 0; i < SH::RM; ++i)
#pragma unroll
    for (int j = 0; j < SH::RM; ++j) acc[i][j] = 0.0f;
  float n2 = 0.0f;
  const bool chainA = threadIdx.x < SH::TM, chainB = !chainA && threadIdx.x < 2 * SH::TM;
  const int crow = chainA ? threadIdx.x : threadIdx.x - SH::TM;
  for (int kb = 0; kb < nk; ++kb) {
    cp_async_wait_group<SH::STAGES - 2>();
    __syncthreads();
    {  // refill the stage consumed last iteration
      const int kn = kb + SH::STAGES - 1;
      const int sn = kn % SH::STAGES;
      if (kn < nk)
        sim_stage<SH>(a, St, a0, b0, kn * SH::KC, sA + sn * SH::TM * SH::PITCH, sB + sn * SH::TM * SH::PITCH);
      cp_async_commit();
    }
    const float* A = sA + (kb % SH::STAGES) * SH::TM * SH::PITCH;
    const float* B = sB + (kb % SH::STAGES) * SH::TM * SH::PITCH;
    if (chainA || chainB) {
      const float* row = (chainA ? A : B) + crow * SH::PITCH;
#pragma unroll 4
      for (int k = 0; k < SH::KC; k += 4) {
        const float4 x = *reinterpret_cast<const float4*>(row + k);
        n2 = __fmaf_rn(x.x, x.x, n2);
        n2 = __fmaf_rn(x.y, x.y, n2);
        n2 = __fmaf_rn(x.z, x.z, n2);
        n2 = __fmaf_rn(x.w, x.w, n2);
      }
    }
#pragma unroll 1
    for (int k = 0; k < SH::KC; k += 4) {
      float4 x[SH::RM], y[SH::RM];
#pragma unroll
      for (int i = 0; i < SH::RM; ++i) x[i] = *reinterpret_cast<const float4*>(A + (ty + i * TD) * SH::PITCH + k);
#pragma unroll
      for (int j = 0; j < SH::RM; ++j) y[j] = *reinterpret_cast<const float4*>(B + (tx + j * TD) * SH::PITCH + k);
#pragma unroll
      for (int i = 0; i < SH::RM; ++i)
#pragma unroll
        for (int j = 0; j < SH::RM; ++j) {
          acc[i][j] = __fmaf_rn(x[i].x, y[j].x, acc[i][j]);
          acc[i][j] = __fmaf_rn(x[i].y, y[j].y, acc[i][j]);
          acc[i][j] = __fmaf_rn(x[i].z, y[j].z, acc[i][j]);
          acc[i][j] = __fmaf_rn(x[i].w, y[j].w, acc[i][j]);
        }
    }
  }
  cp_async_wait_group<0>();
  if (chainA || chainB) (chainA ? invA : invB)[crow] = n2 > 0.0f ? __fdiv_rn(1.0f, __fsqrt_rn(n2)) : 0.0f;
  __syncthreads();
  // best match of each owned A row among the owned B columns, then across
  // the TD threads sharing the row (ties to the smaller b)
#pragma unroll
  for (int i = 0; i < SH::RM; ++i) {
    const int ra = ty + i * TD;
    const int ai = a0 + ra;
    float bs = 0.0f;
    int bb = -1;
#pragma unroll
    for (int j = 0; j < SH::RM; ++j) {
      const int rb = tx + j * TD;
      const int bj = b0 + rb;
      if (ai < a.nA && bj < a.nB) {
        const float sc = __fmul_rn(__fmul_rn(acc[i][j], invA[ra]), invB[rb]);
        if (bb < 0 || sc > bs || (sc == bs && bj < bb)) {
          bs = sc;
          bb = bj;
        }
      }
    }
#pragma unroll
    for (int o = TD / 2; o > 0; o >>= 1) {
      const float os = __shfl_xor_sync(0xffffffffu, bs, o);
      const int ob = __shfl_xor_sync(0xffffffffu, bb, o);
      if (ob >= 0 && (bb < 0 || os > bs || (os == bs && ob < bb))) {
        bs = os;
        bb = ob;
      }
    }
    if (tx == 0 && ai < a.nA) a.best[(static_cast<long long>(t) * a.bblk + blockIdx.y) * a.nA + ai] = Best{bs, bb};
  }
}

// One CTA per tile: merge decisions of the round and the new member lists.
constexpr int kSelThreads = 512;

__global__ void __launch_bounds__(kSelThreads) select_kernel(MergeArgs a) {
  extern __shared__ __align__(16) unsigned char smem[];
  float* bs = reinterpret_cast<float*>(smem);  // [nA]
  int* bb = reinterpret_cast<int*>(bs + a.nA);  // [nA]
  int* merged = bb + a.nA;                      // [nA]
  int* newpos = merged + a.nA;                  // [n]
  int* tok = newpos + a.n;                      // [n0]
  int* cnt = tok + a.n0;                        // [n - r + 1]
  __shared__ int warp_tot[kSelThreads / 32];
  pdl_launch_dependents();
  pdl_wait();
  const int t = blockIdx.x;
  const int n1 = a.n - a.r;
  for (int x = threadIdx.x; x < a.nA; x += kSelThreads) {
    const Best* p = a.best + static_cast<long long>(t) * a.bblk * a.nA + x;
    Best b = p[0];
    for (int k = 1; k < a.bblk; ++k) {
      const Best o = p[static_cast<long long>(k) * a.nA];
      if (o.s > b.s) b = o;  // blocks ascend in b: ties keep the smaller b
    }
    bs[x] = b.s;
    bb[x] = b.b;
  }
  for (int i = threadIdx.x; i < a.n0; i += kSelThreads) tok[i] = a.tok[static_cast<long long>(t) * a.n0 + i];
  __syncthreads();
  for (int x = threadIdx.x; x < a.nA; x += kSelThreads) {
    int before = 0;
    if (a.r < a.nA) {
      const float s = bs[x];
      for (int o = 0; o < a.nA; ++o) before += (bs[o] > s) || (bs[o] == s && o < x);
    }
    merged[x] = before < a.r;
  }
  __syncthreads();
  {  // new positions of the survivors (a run of positions per thread)
    const int per = (a.n + kSelThreads - 1) / kSelThreads;
    const int p0 = min(a.n, static_cast<int>(threadIdx.x) * per), p1 = min(a.n, p0 + per);
    int c = 0;
    for (int p = p0; p < p1; ++p) c += !((p & 1) == 0 && merged[p >> 1]);
    int pos;
    block_exclusive_scan<kSelThreads>(c, warp_tot, pos);
    for (int p = p0; p < p1; ++p) newpos[p] = ((p & 1) == 0 && merged[p >> 1]) ? -1 : pos++;
  }
  for (int j = threadIdx.x; j <= n1; j += kSelThreads) cnt[j] = 0;
  __syncthreads();
  for (int i = threadIdx.x; i < a.n0; i += kSelThreads) {
    int p = tok[i];
    if ((p & 1) == 0 && merged[p >> 1]) p = 2 * bb[p >> 1] + 1;
    const int j = newpos[p];
    tok[i] = j;
    atomicAdd(&cnt[j], 1);
  }
  __syncthreads();
  {  // member-list offsets
    const int per = (n1 + 1 + kSelThreads - 1) / kSelThreads;
    const int j0 = min(n1 + 1, static_cast<int>(threadIdx.x) * per), j1 = min(n1 + 1, j0 + per);
    int c = 0;
    for (int j = j0; j < j1; ++j) c += cnt[j];
    int pos;
    block_exclusive_scan<kSelThreads>(c, warp_tot, pos);
    int32_t* st = a.start + static_cast<long long>(t) * (a.n0 + 1);
    for (int j = j0; j < j1; ++j) {
      const int k = cnt[j];
      st[j] = pos;
      cnt[j] = pos;  // becomes the fill cursor
      pos += k;
    }
  }
  __syncthreads();
  int32_t* tk = a.tok + static_cast<long long>(t) * a.n0;
  for (int i = threadIdx.x; i < a.n0; i += kSelThreads) tk[i] = tok[i];
  if (threadIdx.x < 32) {  // stable fill: members of each token in ascending level-0 index
    const int lane = threadIdx.x;
    int32_t* mem = a.members + static_cast<long long>(t) * a.n0;
    for (int base = 0; base < a.n0; base += 32) {
      const int i = base + lane;
      const unsigned act = __ballot_sync(0xffffffffu, i < a.n0);
      if (i < a.n0) {
        const int j = tok[i];
        const unsigned same = __match_any_sync(act, j);
        const int rk = __popc(same & ((1u << lane) - 1u));
        mem[cnt[j] + rk] = i;
        __syncwarp(act);
        if (rk == 0) cnt[j] += __popc(same);
      }
      __syncwarp();
    }
  }
}

// Sums of the current tokens' members (ascending level-0 index, binary32).
// ROWS == false: the similarity channels into S (4 channels per thread).
// ROWS == true : every channel, divided by the member count and rounded to
// bf16, into the level's block rows (8 channels per thread).
template <bool ROWS>
__global__ void __launch_bounds__(kThreads) sum_kernel(MergeArgs a, uint4* out, long long out_row0, int m) {
  pdl_launch_dependents();
  pdl_wait();
  const int G = ROWS ? a.C8 : a.Cs / 4;
  const long long total = static_cast<long long>(a.n_tiles) * m * G;
  for (long long q = static_cast<long long>(blockIdx.x) * kThreads + threadIdx.x; q < total;
       q += static_cast<long long>(gridDim.x) * kThreads) {
    const int g = static_cast<int>(q % G);
    const long long tj = q / G;
    const int t = static_cast<int>(tj / m), j = static_cast<int>(tj % m);
    const int32_t* st = a.start + static_cast<long long>(t) * (a.n0 + 1);
    const int32_t* mem = a.members + static_cast<long long>(t) * a.n0;
    const int m0 = st[j], m1 = st[j + 1];
    const uint4* x0 = a.feat + static_cast<long long>(t) * a.n0 * a.C8;
    if constexpr (ROWS) {
      float acc[8];
      for (int k = m0; k < m1; ++k) {
        const uint4 x = ld_nc(x0 + static_cast<long long>(mem[k]) * a.C8 + g);
        const float v[8] = {bf16lo(x.x), bf16hi(x.x), bf16lo(x.y), bf16hi(x.y),
                            bf16lo(x.z), bf16hi(x.z), bf16lo(x.w), bf16hi(x.w)};
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[e] = k == m0 ? v[e] : __fadd_rn(acc[e], v[e]);
      }
      const float cntf = static_cast<float>(m1 - m0);
      uint4 o;
      o.x = pack_bf16x2(__fdiv_rn(acc[0], cntf), __fdiv_rn(acc[1], cntf));
      o.y = pack_bf16x2(__fdiv_rn(acc[2], cntf), __fdiv_rn(acc[3], cntf));
      o.z = pack_bf16x2(__fdiv_rn(acc[4], cntf), __fdiv_rn(acc[5], cntf));
      o.w = pack_bf16x2(__fdiv_rn(acc[6], cntf), __fdiv_rn(acc[7], cntf));
      out[(out_row0 + static_cast<long long>(t) * m + j) * a.C8 + g] = o;
    } else {
      float acc[4];
      const uint2* xs = reinterpret_cast<const uint2*>(x0);
      const int C4 = a.C8 * 2;
      for (int k = m0; k < m1; ++k) {
        const uint2 x = xs[static_cast<long long>(mem[k]) * C4 + a.c0_8 * 2 + g];
        const float v[4] = {bf16lo(x.x), bf16hi(x.x), bf16lo(x.y), bf16hi(x.y)};
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[e] = k == m0 ? v[e] : __fadd_rn(acc[e], v[e]);
      }
      reinterpret_cast<float4*>(a.S + (static_cast<long long>(t) * a.n0 + j) * a.Cs)[g] =
          make_float4(acc[0], acc[1], acc[2], acc[3]);
    }
  }
}

inline davet_status ok(cudaError_t e) {
  if (e != cudaSuccess) return cuda_fail(e);
  return check_launch();
}

inline unsigned grid_for(long long work, long long per_block) {
  return static_cast<unsigned>(std::max<long long>(1, std::min<long long>((work + per_block - 1) / per_block,
                                                                          152LL * 16)));
}

inline size_t select_smem(int n0, int nA, int n, int r) {
  return static_cast<size_t>(3 * nA + n + n0 + (n - r + 1)) * 4;
}

}  // namespace realize
}  // namespace davet

using namespace davet;
using namespace davet::realize;

namespace {

davet_status check_common(const void* feat, void* buf, const void* text, int n_tiles, int grid, int n_levels,
                          int mixed_level, int mixed_stride, int text_rows, int C, int* rpt, int* nv,
                          int64_t* block0) {
  if (n_tiles < 0 || text_rows < 0 || C < 8 || C % 8 != 0) return DAVET_ERR_INVALID_ARG;
  const davet_status ls = davet_view_rows(grid, n_levels, mixed_level, mixed_stride, rpt, nv);
  if (ls != DAVET_OK) return ls;
  if (grid > 64 || n_tiles > 65535) return DAVET_ERR_UNSUPPORTED;
  if (n_tiles == 0 && text_rows == 0) return DAVET_OK;
  if (!buf || (n_tiles > 0 && !feat) || (text_rows > 0 && !text)) return DAVET_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(feat) | reinterpret_cast<uintptr_t>(buf) | reinterpret_cast<uintptr_t>(text)) &
      15u)
    return DAVET_ERR_INVALID_ARG;
  davet_view_layout(grid, n_levels, mixed_level, mixed_stride, n_tiles, text_rows, block0);
  return DAVET_OK;
}

}  // namespace

extern "C" davet_status davet_build_views_pruned(const void* feat, const float* score, void* buf, const void* text,
                                                 int n_tiles, int grid, int n_levels, int mixed_level,
                                                 int mixed_stride, int text_rows, int C, void* stream) {
  int rpt[kMaxViews];
  int nv = 0;
  int64_t block0[kMaxViews + 1];
  const davet_status cs = check_common(feat, buf, text, n_tiles, grid, n_levels, mixed_level, mixed_stride,
                                       text_rows, C, rpt, &nv, block0);
  if (cs != DAVET_OK || (n_tiles == 0 && text_rows == 0)) return cs;
  if (n_tiles > 0 && (!score || (reinterpret_cast<uintptr_t>(score) & 3u))) return DAVET_ERR_INVALID_ARG;
  for (int v = 0; v < nv; ++v)
    if (rpt[v] > grid * grid) return DAVET_ERR_INVALID_ARG;  // a view cannot keep more tokens than a tile has
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (n_tiles > 0) {
    Prune p;
    p.feat = static_cast<const uint4*>(feat);
    p.score = score;
    p.buf = static_cast<uint4*>(buf);
    p.C8 = C / 8;
    p.n_tok = grid * grid;
    p.sort_n = 1;
    while (p.sort_n < p.n_tok) p.sort_n <<= 1;
    p.n_tiles = n_tiles;
    p.n_views = nv;
    // view 0 keeps every token: skip it when the encoding is already in place
    p.first_view = feat == buf ? 1 : 0;
    p.rpt_off[0] = 0;
    for (int v = 0; v < kMaxViews; ++v) {
      p.block0[v] = v < nv ? block0[v] : 0;
      p.rpt[v] = v < nv ? rpt[v] : 0;
      p.rpt_off[v + 1] = p.rpt_off[v] + p.rpt[v];
    }
    if (p.first_view < nv) {
      const size_t smem = static_cast<size_t>(p.sort_n) * 8 + static_cast<size_t>(p.n_tok + p.rpt_off[nv]) * 4;
      const long long rows = p.rpt_off[nv] - p.rpt_off[p.first_view];
      const long long tasks = rows * ((p.C8 + kChunk - 1) / kChunk);
      // about 4 CTAs per SM over the whole request
      long long per_tile = std::max<long long>(1, (152LL * 4 + n_tiles - 1) / n_tiles);
      per_tile = std::min<long long>(per_tile, (tasks + kThreads / 32 - 1) / (kThreads / 32));
      cudaError_t e = cudaFuncSetAttribute(prune_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           static_cast<int>(smem));
      if (e != cudaSuccess) return cuda_fail(e);
      e = launch(prune_kernel, dim3(static_cast<unsigned>(per_tile), n_tiles), dim3(kThreads), smem, st, p);
      const davet_status s = ok(e);
      if (s != DAVET_OK) return s;
    }
  }
  return views::enqueue_fill(buf, text, n_tiles, grid, n_levels, mixed_level, mixed_stride, text_rows, C, false, st);
}

extern "C" davet_status davet_merge_workspace_bytes(int n_tiles, int grid, int n_levels, int sim_C, size_t* bytes) {
  if (!bytes || n_tiles < 0 || grid < 1 || n_levels < 1 || sim_C < 32 || sim_C % 32 != 0)
    return DAVET_ERR_INVALID_ARG;
  if (n_levels > 5 || grid > 64) return DAVET_ERR_UNSUPPORTED;
  *bytes = make_plan(n_tiles, grid, n_levels, sim_C).bytes;
  return DAVET_OK;
}

extern "C" davet_status davet_build_views_merged(const void* feat, void* buf, const void* text, int n_tiles, int grid,
                                                 int n_levels, int mixed_level, int mixed_stride, int text_rows, int C,
                                                 int sim_c0, int sim_C, int32_t* assign, void* workspace,
                                                 size_t workspace_bytes, void* stream) {
  int rpt[kMaxViews];
  int nv = 0;
  int64_t block0[kMaxViews + 1];
  const davet_status cs = check_common(feat, buf, text, n_tiles, grid, n_levels, mixed_level, mixed_stride,
                                       text_rows, C, rpt, &nv, block0);
  if (cs != DAVET_OK) return cs;
  if (sim_C < 32 || sim_C % 32 != 0 || sim_c0 < 0 || sim_c0 % 8 != 0 || sim_c0 + sim_C > C)
    return DAVET_ERR_INVALID_ARG;
  if (n_tiles == 0 && text_rows == 0) return DAVET_OK;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (n_tiles > 0) {
    const Plan P = make_plan(n_tiles, grid, n_levels, sim_C);
    if (!workspace || workspace_bytes < P.bytes || (reinterpret_cast<uintptr_t>(workspace) & 255u))
      return DAVET_ERR_INVALID_ARG;
    if (assign && (reinterpret_cast<uintptr_t>(assign) & 3u)) return DAVET_ERR_INVALID_ARG;
    unsigned char* ws = static_cast<unsigned char*>(workspace);
    MergeArgs a;
    a.feat = static_cast<const uint4*>(feat);
    a.C8 = C / 8;
    a.n0 = P.n0;
    a.n_tiles = n_tiles;
    a.c0_8 = sim_c0 / 8;
    a.Cs = sim_C;
    a.tok = reinterpret_cast<int32_t*>(ws + P.off_tok);
    a.start = reinterpret_cast<int32_t*>(ws + P.off_start);
    a.members = reinterpret_cast<int32_t*>(ws + P.off_members);
    a.best = reinterpret_cast<Best*>(ws + P.off_best);
    a.S = reinterpret_cast<float*>(ws + P.off_S);
    a.n = P.n0;
    a.nA = a.nB = a.bblk = a.r = 0;
    uint4* out = static_cast<uint4*>(buf);
    const size_t tile_ints = static_cast<size_t>(n_tiles) * P.n0;
    // level 0 block: the encoding itself
    if (feat != buf) {
      const cudaError_t e = cudaMemcpyAsync(buf, feat, tile_ints * C * 2, cudaMemcpyDeviceToDevice, st);
      if (e != cudaSuccess) return cuda_fail(e);
    }
    davet_status s = ok(launch(init_kernel, dim3(grid_for(static_cast<long long>(tile_ints) + n_tiles, kThreads)),
                               dim3(kThreads), 0, st, a, assign));
    if (s != DAVET_OK) return s;
    size_t max_sel = 0;
    for (size_t k = 0; k < P.n.size(); ++k)
      max_sel = std::max(max_sel, select_smem(P.n0, (P.n[k] + 1) / 2, P.n[k], P.r[k]));
    cudaError_t e = cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(std::max<size_t>(max_sel, 1024)));
    if (e != cudaSuccess) return cuda_fail(e);
    e = cudaFuncSetAttribute(sim_kernel<SimLarge>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(SimLarge::SMEM));
    if (e != cudaSuccess) return cuda_fail(e);
    for (size_t k = 0; k < P.n.size(); ++k) {
      a.n = P.n[k];
      a.r = P.r[k];
      a.nA = (a.n + 1) / 2;
      a.nB = a.n / 2;
      const long long tok_work = static_cast<long long>(n_tiles) * a.n;
      s = ok(launch(sum_kernel<false>, dim3(grid_for(tok_work * (sim_C / 4), kThreads)), dim3(kThreads), 0, st, a,
                    static_cast<uint4*>(nullptr), 0LL, a.n));
      if (s != DAVET_OK) return s;
      // the largest block shape that still gives about two CTAs per SM
      auto ctas = [&](int tm) {
        return static_cast<long long>((a.nA + tm - 1) / tm) * ((a.nB + tm - 1) / tm) * n_tiles;
      };
      if (ctas(SimLarge::TM) >= 2 * 152) {
        a.bblk = (a.nB + SimLarge::TM - 1) / SimLarge::TM;
        s = ok(launch(sim_kernel<SimLarge>, dim3((a.nA + SimLarge::TM - 1) / SimLarge::TM, a.bblk, n_tiles),
                      dim3(SimLarge::NT), SimLarge::SMEM, st, a));
      } else if (ctas(SimMid::TM) >= 2 * 152) {
        a.bblk = (a.nB + SimMid::TM - 1) / SimMid::TM;
        s = ok(launch(sim_kernel<SimMid>, dim3((a.nA + SimMid::TM - 1) / SimMid::TM, a.bblk, n_tiles),
                      dim3(SimMid::NT), SimMid::SMEM, st, a));
      } else {
        a.bblk = (a.nB + SimSmall::TM - 1) / SimSmall::TM;
        s = ok(launch(sim_kernel<SimSmall>, dim3((a.nA + SimSmall::TM - 1) / SimSmall::TM, a.bblk, n_tiles),
                      dim3(SimSmall::NT), SimSmall::SMEM, st, a));
      }
      if (s != DAVET_OK) return s;
      s = ok(launch(select_kernel, dim3(n_tiles), dim3(kSelThreads), select_smem(P.n0, a.nA, a.n, a.r), st, a));
      if (s != DAVET_OK) return s;
      const int l = P.level[k];
      if (k + 1 == P.n.size() || P.level[k + 1] != l) {  // level l complete
        const int m = P.side[l] * P.side[l];
        s = ok(launch(sum_kernel<true>, dim3(grid_for(static_cast<long long>(n_tiles) * m * a.C8, kThreads)),
                      dim3(kThreads), 0, st, a, out, static_cast<long long>(block0[l]), m));
        if (s != DAVET_OK) return s;
        if (assign) {
          e = cudaMemcpyAsync(assign + static_cast<size_t>(l) * tile_ints, a.tok, tile_ints * 4,
                              cudaMemcpyDeviceToDevice, st);
          if (e != cudaSuccess) return cuda_fail(e);
        }
      }
    }
  }
  return views::enqueue_fill(buf, text, n_tiles, grid, n_levels, mixed_level, mixed_stride, text_rows, C, true, st);
}
